"""Seeded synthetic optimizer-step inputs shaped like LLM parameter sets.

This module is the only code shared by the oracle-side tests and the CUDA-side
tests/benchmark.  It draws weights, gradients and optimizer states; it holds
none of the M+Adam arithmetic (no moment update, no rounding rule, no scale
rule).  The FP8 initial weights are produced with torch's own float8_e4m3fn
cast of a pre-scaled draw, with a per-role power-of-two exponent chosen from
the draw's standard deviation (per-tensor scaling), or per 32-element block
the power of two at or above the block's largest |w| / 448 computed with
torch in binary64 (block scaling).  NVFP4 weights take a power-of-two tensor
scale per role, per 16-element block the smallest E4M3 value whose range
covers the block (binary64), and the nearest E2M1 code (torch bucketize):
input recipes, not the optimizer's scale or rounding rules.

Stand-ins: the paper trains LLaMA-style decoders on C4/EN (Sec. 5.2, the
model-architecture table of Appendix C).  An optimizer step needs no data, so
the workloads here are parameter lists with the shapes of GPT-2 small and of
LLaMA-style 1.5B / 7B models, plus a flat tensor and a ragged stress list;
values are seeded random draws, not trained weights.

Layout: tensor k's first element has global index off[k], where off[0] = 0 and
off[k+1] is off[k] + numel[k] rounded up to a multiple of 8 (the library's
documented element-index layout).  With ``layout="flat"`` every array kind
(w, g, m, v, ve) is one allocation indexed by that global index, and tensors are
views into it; with ``layout="separate"`` each tensor is its own allocation.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace
from typing import Dict, List, Optional

import torch

ALIGN = 8  # elements; tensor starts in the global index space


@dataclass(frozen=True)
class TensorSpec:
    name: str
    numel: int
    role: str  # "matrix" | "head" | "embedding" | "bias" | "norm" | "flat"


@dataclass(frozen=True)
class Workload:
    name: str
    specs: tuple
    weight_dtype: str          # "bf16" | "e4m3" | "e4m3_b32" | "nvfp4" | "mixed_b32" | "mixed_fp4" (see format_of)
    grad_dtype: str            # "f32" | "bf16"
    moment_dtype: str          # "f32" | "bf16"
    rounding: str              # "nearest" | "stochastic"
    steps: int
    seed: int = 0
    w_std: float = 0.02
    zero_frac: float = 0.0     # fraction of weights set exactly to 0
    grad: tuple = ("normal", 1e-3)  # ("normal", s) | ("normal_logu", lo, hi) | ("student_t_logu", nu, lo, hi)
    norm_gain: float = 1.0     # initial value of norm gains
    bias_zero: bool = True     # biases start at exactly 0
    compute_copy: bool = False  # E4M3 tensors also get a BF16 compute copy
    format_list: tuple = ()    # explicit weight format per tensor (overrides weight_dtype)
    description: str = ""

    def format_of(self, spec: "TensorSpec") -> str:
        """Weight format of one tensor.  "mixed_b32" is the paper's FP8 regime
        (Sec. 5.2): linear layers block-scaled E4M3, embeddings, norms, biases
        and the LM head BF16."""
        if self.weight_dtype == "mixed_b32":
            return "e4m3_b32" if spec.role == "matrix" else "bf16"
        if self.weight_dtype == "mixed_fp4":
            return "nvfp4" if spec.role == "matrix" else "bf16"
        return self.weight_dtype

    @property
    def formats(self) -> List[str]:
        if self.format_list:
            return list(self.format_list)
        return [self.format_of(s) for s in self.specs]

    @property
    def numels(self) -> List[int]:
        return [s.numel for s in self.specs]

    @property
    def n_params(self) -> int:
        return sum(self.numels)


def global_offsets(numels) -> List[int]:
    """Start index of each tensor in the padded global element index space."""
    offs, o = [], 0
    for n in numels:
        offs.append(o)
        o = (o + int(n) + ALIGN - 1) // ALIGN * ALIGN
    return offs


def global_length(numels) -> int:
    o = 0
    for n in numels:
        o = (o + int(n) + ALIGN - 1) // ALIGN * ALIGN
    return o


# ---------------------------------------------------------------------------
# Parameter-list shapes
# ---------------------------------------------------------------------------
def gpt2_specs(layers=12, d=768, vocab=50257, ctx=1024) -> tuple:
    """GPT-2 small layout (tied LM head): wte, wpe, per-block LN/attn/MLP, ln_f."""
    s = [TensorSpec("wte", vocab * d, "embedding"), TensorSpec("wpe", ctx * d, "embedding")]
    for i in range(layers):
        p = f"h{i}."
        s += [
            TensorSpec(p + "ln_1.weight", d, "norm"), TensorSpec(p + "ln_1.bias", d, "bias"),
            TensorSpec(p + "attn.c_attn.weight", d * 3 * d, "matrix"),
            TensorSpec(p + "attn.c_attn.bias", 3 * d, "bias"),
            TensorSpec(p + "attn.c_proj.weight", d * d, "matrix"),
            TensorSpec(p + "attn.c_proj.bias", d, "bias"),
            TensorSpec(p + "ln_2.weight", d, "norm"), TensorSpec(p + "ln_2.bias", d, "bias"),
            TensorSpec(p + "mlp.c_fc.weight", d * 4 * d, "matrix"),
            TensorSpec(p + "mlp.c_fc.bias", 4 * d, "bias"),
            TensorSpec(p + "mlp.c_proj.weight", 4 * d * d, "matrix"),
            TensorSpec(p + "mlp.c_proj.bias", d, "bias"),
        ]
    s += [TensorSpec("ln_f.weight", d, "norm"), TensorSpec("ln_f.bias", d, "bias")]
    return tuple(s)


def llama_specs(layers, d, ffn, vocab) -> tuple:
    """LLaMA-style decoder: embed, per layer q/k/v/o, SwiGLU gate/up/down and two
    RMSNorm gains, final norm, untied LM head."""
    s = [TensorSpec("embed_tokens", vocab * d, "embedding")]
    for i in range(layers):
        p = f"layers.{i}."
        s += [
            TensorSpec(p + "self_attn.q_proj", d * d, "matrix"),
            TensorSpec(p + "self_attn.k_proj", d * d, "matrix"),
            TensorSpec(p + "self_attn.v_proj", d * d, "matrix"),
            TensorSpec(p + "self_attn.o_proj", d * d, "matrix"),
            TensorSpec(p + "mlp.gate_proj", d * ffn, "matrix"),
            TensorSpec(p + "mlp.up_proj", d * ffn, "matrix"),
            TensorSpec(p + "mlp.down_proj", ffn * d, "matrix"),
            TensorSpec(p + "input_layernorm", d, "norm"),
            TensorSpec(p + "post_attention_layernorm", d, "norm"),
        ]
    s += [TensorSpec("norm", d, "norm"), TensorSpec("lm_head", vocab * d, "head")]
    return tuple(s)


def ragged_specs(n_tensors, max_log2, seed) -> tuple:
    """Sizes round(exp(U[0, ln 2^max_log2])): log-uniform in [1, 2^max_log2]."""
    g = torch.Generator().manual_seed(10_000 + seed)
    u = torch.rand(n_tensors, generator=g, dtype=torch.float64)
    sizes = torch.round(torch.exp(u * (max_log2 * math.log(2.0)))).to(torch.int64).clamp_min(1)
    return tuple(TensorSpec(f"t{i}", int(n), "flat") for i, n in enumerate(sizes.tolist()))


def _flat1m():
    return Workload(
        name="flat_1m", specs=(TensorSpec("flat", 1 << 20, "flat"),),
        weight_dtype="bf16", grad_dtype="f32", moment_dtype="f32", rounding="nearest",
        steps=10, zero_frac=0.01, grad=("normal", 1e-3),
        description="single flat tensor of 1,048,576 params: bf16 w ~N(0,0.02) with 1% zeros, "
                    "fp32 g ~N(0,1e-3), fp32 moments, round-to-nearest")


def _gpt2(layers=12, d=768, vocab=50257, ctx=1024, name="gpt2_124m"):
    return Workload(
        name=name, specs=gpt2_specs(layers, d, vocab, ctx),
        weight_dtype="bf16", grad_dtype="bf16", moment_dtype="f32", rounding="stochastic",
        steps=100, grad=("normal_logu", 1e-5, 1e-2),
        description="GPT-2-small-shaped list: bf16 w ~N(0,0.02) (LN gains 1, biases 0), bf16 g "
                    "with per-tensor std log-uniform [1e-5,1e-2], fp32 moments, stochastic rounding")


def _llama15(layers=24, d=2048, ffn=5632, vocab=32000, name="llama_1p5b"):
    return Workload(
        name=name, specs=llama_specs(layers, d, ffn, vocab),
        weight_dtype="e4m3", grad_dtype="bf16", moment_dtype="f32", rounding="stochastic",
        steps=10, grad=("student_t_logu", 3.0, 1e-5, 1e-2),
        description="LLaMA-style 1.5B list (24 layers, d=2048, ffn 5632, vocab 32000): E4M3 weights "
                    "with per-tensor power-of-two scale, bf16 Student-t(3) grads scaled per tensor "
                    "(std log-uniform [1e-5,1e-2]), fp32 moments, stochastic rounding")


def _llama15_mixed(layers=24, d=2048, ffn=5632, vocab=32000, name="llama_1p5b_mixed"):
    return Workload(
        name=name, specs=llama_specs(layers, d, ffn, vocab),
        weight_dtype="mixed_b32", grad_dtype="bf16", moment_dtype="f32", rounding="stochastic",
        steps=10, grad=("student_t_logu", 3.0, 1e-5, 1e-2), compute_copy=True,
        description="LLaMA-style 1.5B list in the paper's FP8 regime: linear layers E4M3 with one "
                    "FP16 power-of-two scale per 32 weights and a BF16 compute copy written by the "
                    "step, embeddings / norms / LM head BF16; bf16 Student-t(3) grads scaled per "
                    "tensor, fp32 moments, stochastic rounding")


def _llama15_nvfp4(layers=24, d=2048, ffn=5632, vocab=32000, name="llama_1p5b_nvfp4"):
    return Workload(
        name=name, specs=llama_specs(layers, d, ffn, vocab),
        weight_dtype="mixed_fp4", grad_dtype="bf16", moment_dtype="f32", rounding="nearest",
        steps=10, grad=("student_t_logu", 3.0, 1e-5, 1e-2), compute_copy=True,
        description="LLaMA-style 1.5B list in the paper's NVFP4 regime: linear layers NVFP4 (E2M1 "
                    "codes, an E4M3 scale per 16 weights, a tensor scale) with a BF16 compute copy "
                    "written by the step, embeddings / norms / LM head BF16; bf16 Student-t(3) grads "
                    "scaled per tensor, fp32 moments, round-to-nearest (the paper trains M+Adam "
                    "without stochastic rounding)")


def _llama7(layers=32, d=4096, ffn=11008, vocab=32000, name="llama_7b"):
    return Workload(
        name=name, specs=llama_specs(layers, d, ffn, vocab),
        weight_dtype="bf16", grad_dtype="bf16", moment_dtype="bf16", rounding="stochastic",
        steps=10, grad=("normal_logu", 1e-6, 1e-2),
        description="LLaMA-style 7B list (32 layers, d=4096, ffn 11008, vocab 32000): bf16 weights, "
                    "bf16 grads with per-tensor std log-uniform [1e-6,1e-2], bf16 moments, "
                    "stochastic rounding")


def _ragged(n=20000, max_log2=22, name="ragged_20k", rounding="stochastic"):
    return Workload(
        name=name, specs=ragged_specs(n, max_log2, 0),
        weight_dtype="bf16", grad_dtype="bf16", moment_dtype="f32", rounding=rounding,
        steps=10, zero_frac=0.30, grad=("normal", 1e-3),
        description=f"ragged list of {n} tensors, sizes log-uniform [1, 2^{max_log2}], 30% zero "
                    "weights, bf16 w/g, fp32 moments")


CONFIGS: Dict[str, Workload] = {
    "flat_1m": _flat1m(),
    "gpt2_124m": _gpt2(),
    "llama_1p5b": _llama15(),
    "llama_7b": _llama7(),
    "ragged_20k": _ragged(),
    "llama_1p5b_mixed": _llama15_mixed(),
    "llama_1p5b_nvfp4": _llama15_nvfp4(),
}

# Same distributions and formats at sizes the oracle finishes in seconds,
# still spanning many 3840-element tiles and ragged tails.
SMALL: Dict[str, Workload] = {
    "flat_1m": replace(_flat1m(), specs=(TensorSpec("flat", (1 << 16) + 5, "flat"),), name="flat_small"),
    "gpt2_124m": _gpt2(layers=2, d=64, vocab=1003, ctx=64, name="gpt2_small"),
    "llama_1p5b": _llama15(layers=2, d=128, ffn=344, vocab=517, name="llama15_small"),
    "llama_7b": _llama7(layers=2, d=128, ffn=344, vocab=517, name="llama7_small"),
    "ragged_20k": _ragged(n=300, max_log2=13, name="ragged_small"),
    "llama_1p5b_mixed": _llama15_mixed(layers=2, d=128, ffn=344, vocab=517, name="llama15_mixed_small"),
    "llama_1p5b_nvfp4": _llama15_nvfp4(layers=2, d=128, ffn=344, vocab=517, name="llama15_nvfp4_small"),
}


# ---------------------------------------------------------------------------
# Materialisation
# ---------------------------------------------------------------------------
_TORCH = {"f32": torch.float32, "bf16": torch.bfloat16, "e4m3": torch.uint8, "e4m3_b32": torch.uint8,
          "nvfp4": torch.uint8}
BLOCK = 32      # elements per block scale (block-scaled E4M3)
FP4_BLOCK = 16  # elements per block scale (NVFP4)
_E2M1_MIDPOINTS = (0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0)  # between the grid values 0 .. 6


def _gen(device, seed, k, salt):
    g = torch.Generator(device=device)
    g.manual_seed((seed * 1_000_003 + k * 7919 + salt) % (2**63 - 1))
    return g


def _grad_std(wl: Workload, k: int) -> float:
    kind = wl.grad[0]
    if kind == "normal":
        return float(wl.grad[1])
    lo, hi = (wl.grad[1], wl.grad[2]) if kind == "normal_logu" else (wl.grad[2], wl.grad[3])
    u = torch.rand(1, generator=_gen("cpu", wl.seed, k, 5), dtype=torch.float64).item()
    return math.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))


def block_initial_scales(wf: torch.Tensor, default_exp: int) -> torch.Tensor:
    """Float16 power-of-two scale per 32-element block: 2^k with k the
    smallest integer such that the block's largest |w| fits under 448 * 2^k
    (evaluated in binary64 by torch), clamped to [-24, 15]; all-zero blocks
    take 2^default_exp."""
    n = wf.numel()
    nb = (n + BLOCK - 1) // BLOCK
    pad = torch.zeros(nb * BLOCK, dtype=torch.float64, device=wf.device)
    pad[:n] = wf.to(torch.float64).abs()
    amax = pad.view(nb, BLOCK).amax(dim=1)
    k = torch.ceil(torch.log2(amax / 448.0))
    k = torch.where(amax > 0, k, torch.full_like(k, float(default_exp))).clamp_(-24, 15)
    return torch.exp2(k).to(torch.float16)


def nvfp4_initial(wf: torch.Tensor, G: float):
    """Packed E2M1 codes and E4M3 block-scale codes of a draw (input recipe):
    per 16-element block the smallest positive E4M3 value v with
    6 v G >= the block's largest |w| (binary64; code 56 = 1.0 for all-zero
    blocks, 126 when none), then per element the nearest E2M1 value of
    w / (v G)."""
    dev = wf.device
    n = wf.numel()
    nb = (n + FP4_BLOCK - 1) // FP4_BLOCK
    vals = torch.arange(1, 127, dtype=torch.uint8).view(torch.float8_e4m3fn).to(torch.float64).to(dev)
    pad = torch.zeros(nb * FP4_BLOCK, dtype=torch.float64, device=dev)
    pad[:n] = wf.to(torch.float64)
    amax = pad.abs().view(nb, FP4_BLOCK).amax(dim=1)
    idx = torch.searchsorted(vals, amax / (6.0 * G)).clamp_(max=125)
    codes_s = torch.where(amax > 0, idx + 1, torch.full_like(idx, 56)).to(torch.uint8)
    d = vals[codes_s.long() - 1].repeat_interleave(FP4_BLOCK) * G
    x = pad / d
    mag = torch.bucketize(x.abs(), torch.tensor(_E2M1_MIDPOINTS, dtype=torch.float64, device=dev))
    c = (mag + 8 * (x < 0).to(mag.dtype)).to(torch.uint8)[:n]
    if n % 2:
        c = torch.cat([c, torch.zeros(1, dtype=torch.uint8, device=dev)])
    packed = (c[0::2] & 0x0F) | (c[1::2] << 4)
    return packed, codes_s


def nvfp4_tensor_scale(role: str, w_std: float, norm_gain: float) -> float:
    """Power-of-two tensor scale G putting the block scales of a draw near
    112 of E4M3's 448 (room for 4x growth): top / (6 * 112), rounded up to a
    power of two, top = 6 sigma (or the norm gain)."""
    top = norm_gain if role == "norm" else 6.0 * w_std
    return 2.0 ** math.ceil(math.log2(top / (6.0 * 112.0)))


def fp8_initial_exponent(role: str, w_std: float, norm_gain: float) -> int:
    """Power-of-two exponent the synthetic FP8 weights are first stored with:
    6 sigma (or the norm gain) fits under E4M3's largest finite value 448."""
    top = norm_gain if role == "norm" else 6.0 * w_std
    if role == "bias":
        top = 6.0 * w_std
    return int(math.ceil(math.log2(top / 448.0)))


@dataclass
class Materialized:
    workload: Workload
    offsets: List[int]
    length: int
    w: List[torch.Tensor]
    g: List[torch.Tensor]
    m: List[torch.Tensor]
    v: List[torch.Tensor]
    ve: List[torch.Tensor]
    fp8_exp: Optional[List[int]] = None
    flat: Dict[str, torch.Tensor] = field(default_factory=dict)
    formats: List[str] = field(default_factory=list)
    bscale: List[Optional[torch.Tensor]] = field(default_factory=list)  # float16 / E4M3-code block scales
    cc: List[Optional[torch.Tensor]] = field(default_factory=list)      # BF16 compute copies
    gscale: List[float] = field(default_factory=list)                   # NVFP4 tensor scales (else 0)


def _alloc(kind_dtype, numels, offsets, length, device, layout):
    if layout == "flat":
        base = torch.zeros(length, dtype=kind_dtype, device=device)
        return base, [base[o:o + n] for o, n in zip(offsets, numels)]
    return None, [torch.zeros(n, dtype=kind_dtype, device=device) for n in numels]


def materialize(wl: Workload, device="cpu", layout="separate", warm_state=False) -> Materialized:
    """Draw the workload's tensors on `device` (values depend on the device's
    generator).  warm_state=True also draws non-zero moments (as after some
    training), for checks beyond the first step."""
    numels = wl.numels
    offsets = global_offsets(numels)
    length = global_length(numels)
    formats = wl.formats
    uniform = len(set(formats)) <= 1
    wdt = _TORCH[formats[0]] if formats else torch.bfloat16
    gdt, mdt = _TORCH[wl.grad_dtype], _TORCH[wl.moment_dtype]
    flat = {}
    wbytes = [(n + 1) // 2 if f == "nvfp4" else n for n, f in zip(numels, formats)]
    if uniform and "nvfp4" not in formats:
        fw, w = _alloc(wdt, numels, offsets, length, device, layout)
    else:  # weights of different element sizes (or packed): one allocation per tensor
        fw, w = None, [torch.zeros(b, dtype=_TORCH[f], device=device) for b, f in zip(wbytes, formats)]
    fg, g = _alloc(gdt, numels, offsets, length, device, layout)
    fm, m = _alloc(mdt, numels, offsets, length, device, layout)
    fv, v = _alloc(mdt, numels, offsets, length, device, layout)
    fve, ve = _alloc(mdt, numels, offsets, length, device, layout)
    if layout == "flat":
        flat = {"g": fg, "m": fm, "v": fv, "ve": fve}
        if fw is not None:
            flat["w"] = fw
    fp8_exp = [] if "e4m3" in formats else None
    bscale = [torch.ones((n + BLOCK - 1) // BLOCK, dtype=torch.float16, device=device) if f == "e4m3_b32" else
              torch.zeros((n + FP4_BLOCK - 1) // FP4_BLOCK, dtype=torch.uint8, device=device) if f == "nvfp4" else None
              for n, f in zip(numels, formats)]
    gscale = [nvfp4_tensor_scale(s.role, wl.w_std, wl.norm_gain) if f == "nvfp4" else 0.0
              for s, f in zip(wl.specs, formats)]
    cc = [torch.zeros(n, dtype=torch.bfloat16, device=device) if wl.compute_copy and f != "bf16" else None
          for n, f in zip(numels, formats)]

    for k, spec in enumerate(wl.specs):
        n = spec.numel
        fmt = formats[k]
        if n == 0:
            if fp8_exp is not None:
                fp8_exp.append(0)
            continue
        gw = _gen(device, wl.seed, k, 1)
        # weights
        if spec.role == "norm":
            wf = torch.full((n,), wl.norm_gain, dtype=torch.float32, device=device)
        elif spec.role == "bias" and wl.bias_zero:
            wf = torch.zeros(n, dtype=torch.float32, device=device)
        else:
            wf = torch.randn(n, generator=gw, dtype=torch.float32, device=device) * wl.w_std
            if wl.zero_frac > 0:
                z = torch.rand(n, generator=gw, device=device) < wl.zero_frac
                wf[z] = 0.0
        if fp8_exp is not None:
            fp8_exp.append(fp8_initial_exponent(spec.role, wl.w_std, wl.norm_gain) if fmt == "e4m3" else 0)
        if fmt == "e4m3":
            e0 = fp8_exp[-1]
            q = (wf * (2.0 ** -e0)).clamp_(-448.0, 448.0).to(torch.float8_e4m3fn)
            w[k].copy_(q.view(torch.uint8))
        elif fmt == "nvfp4":
            packed, sc = nvfp4_initial(wf, gscale[k])
            w[k].copy_(packed)
            bscale[k].copy_(sc)
        elif fmt == "e4m3_b32":
            sc = block_initial_scales(wf, fp8_initial_exponent(spec.role, wl.w_std, wl.norm_gain))
            bscale[k].copy_(sc)
            per = sc.to(torch.float32).repeat_interleave(BLOCK)[:n]
            q = (wf / per).clamp_(-448.0, 448.0).to(torch.float8_e4m3fn)
            w[k].copy_(q.view(torch.uint8))
        else:
            w[k].copy_(wf.to(torch.bfloat16))
        # gradients
        gg = _gen(device, wl.seed, k, 2)
        sd = _grad_std(wl, k)
        if wl.grad[0] == "student_t_logu":
            nu = float(wl.grad[1])
            z = torch.randn(n, generator=gg, dtype=torch.float32, device=device)
            chi = torch.zeros(n, dtype=torch.float32, device=device)
            for _ in range(int(nu)):
                chi += torch.randn(n, generator=gg, dtype=torch.float32, device=device) ** 2
            gf = z / torch.sqrt(chi / nu) * sd
        else:
            gf = torch.randn(n, generator=gg, dtype=torch.float32, device=device) * sd
        g[k].copy_(gf.to(gdt))
        # optimizer states
        if warm_state:
            gs = _gen(device, wl.seed, k, 3)
            wabs = wf.abs() + 1e-3
            mf = 0.3 * sd * torch.randn(n, generator=gs, dtype=torch.float32, device=device)
            vf = (sd * (0.5 + torch.rand(n, generator=gs, device=device))) ** 2
            vef = (0.69314718 * sd * wabs * (0.5 + torch.rand(n, generator=gs, device=device))) ** 2
            m[k].copy_(mf.to(mdt))
            v[k].copy_(vf.to(mdt))
            ve[k].copy_(vef.to(mdt))
    return Materialized(wl, offsets, length, w, g, m, v, ve, fp8_exp, flat, formats, bscale, cc, gscale)


# ---------------------------------------------------------------------------
# The BF16-stored matrix-fitting diagnostic (the toy diagnostic of Sec. 5.1
# and its appendix): W is n x n (stored flat), five regimes
# ---------------------------------------------------------------------------
TOY_N = 4096
TOY_REGIMES = ("sign_flip", "zero_revival", "small", "large", "mixed")


@dataclass
class ToyProblem:
    regime: str
    w0: torch.Tensor       # BF16 initial weights (flat, n*n)
    wstar: torch.Tensor    # binary32 targets (flat)
    c_lo: float
    c_hi: float
    split: bool            # the two halves are separate sub-problems (mixed scales)


# Learning rates at n = 4096, B = 65536 (eta_a, eta_m; the combined rule
# shares one value across the five regimes, as in the paper's main figure).
# Chosen by a sweep over {0.01, 0.03, ..., 30} on n = 128, B = 64 (the same
# per-step hit rate B / n^2 = 1/256) for 2000 steps, scaled by the batch ratio
# 1024 (the gradient of one sample scales as 1 / B).
TOY_LR = {
    "additive": {"sign_flip": 3072.0, "zero_revival": 30720.0, "small": 10240.0, "large": 30720.0,
                 "mixed": 10240.0},
    "multiplicative": {"sign_flip": 30720.0, "zero_revival": 1024.0, "small": 1024.0, "large": 3072.0,
                       "mixed": 1024.0},
    "combined": {r: 3072.0 for r in TOY_REGIMES},
}


def toy_problem(regime: str, n: int = TOY_N, seed: int = 0, device="cpu") -> ToyProblem:
    """Targets and initial weights of one regime (the appendix's recipes):
    sign flip (w* = +-1, w0 = -w*, c = 1); zero revival (w* = +-1, w0 = 0,
    c = 1); small weights (w* = 1e-4 z, w0 = 0, c = 1e8); large weights
    (w* = 900 max(|z|, 1/900), w0 = 100, c = 1e-7); mixed scales (the first
    half small, the second half large, each with its own c)."""
    N = n * n
    g = _gen(device, seed, 0, 7000 + TOY_REGIMES.index(regime))
    if regime in ("sign_flip", "zero_revival"):
        ws = torch.randint(0, 2, (N,), generator=g, device=device).to(torch.float32) * 2 - 1
        w0 = -ws if regime == "sign_flip" else torch.zeros(N, device=device)
        return ToyProblem(regime, w0.to(torch.bfloat16), ws, 1.0, 1.0, False)
    z = torch.randn(N, generator=g, dtype=torch.float32, device=device)
    small = 1e-4 * z
    large = 900.0 * torch.clamp(z.abs(), min=1.0 / 900.0)
    if regime == "small":
        return ToyProblem(regime, torch.zeros(N, dtype=torch.bfloat16, device=device), small, 1e8, 1e8, False)
    if regime == "large":
        return ToyProblem(regime, torch.full((N,), 100.0, device=device).to(torch.bfloat16), large, 1e-7, 1e-7, False)
    half = N // 2
    ws = torch.cat([small[:half], large[half:]])
    w0 = torch.cat([torch.zeros(half, device=device), torch.full((N - half,), 100.0, device=device)])
    return ToyProblem(regime, w0.to(torch.bfloat16), ws, 1e8, 1e-7, True)


def to_numpy_bits(t: torch.Tensor):
    """Host numpy view: float32 stays float32, bfloat16 and float16 become
    uint16 bits, uint8 (E4M3 codes) stays uint8."""
    t = t.detach().to("cpu").contiguous()
    if t.dtype in (torch.bfloat16, torch.float16):
        return t.view(torch.int16).numpy().view("uint16").copy()
    return t.numpy().copy()
