"""Shared machinery of the GPU parity tests and the smoke check: run the CUDA
step (through the C ABI) and the oracle on the same seeded inputs and compare
every stored bit.

Tolerance: the library and the oracle follow the same binary32 operation
sequence, so stored weights, moments, E4M3 scale state (per-tensor rings and
FP16 block scales) and BF16 compute copies must agree bit for bit (NaN
compares equal to NaN).  That is stricter than the bar of the
method's parity contract (weights within 1 storage ulp on at most 1e-4 of
elements where rounding is stochastic, binary32 moments within relative
1e-5); `contract_ok` checks that weaker bar too, for reporting.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional

import numpy as np
import torch

import oracle
import workloads as W
from paper_2607_10611_gb300.optimizer import MPAdam

ODT = {"f32": oracle.F32, "bf16": oracle.BF16, "e4m3": oracle.E4M3, "e4m3_b32": oracle.E4M3_B32,
       "nvfp4": oracle.NVFP4}
HP_KEYS = ("lr_add", "lr_mul", "beta1", "beta2", "eps", "tau", "rmax_pos", "rmax_neg", "g_max",
           "dmult_max", "w_max", "wd_add", "bias_correction")


def oracle_hparams(wl: W.Workload, hp: Dict):
    kw = {k: v for k, v in hp.items() if k in HP_KEYS}
    return oracle.hparams(stochastic=1 if wl.rounding == "stochastic" else 0, seed=wl.seed, **kw)


def host_tensors(mt: W.Materialized) -> List[dict]:
    out = []
    for k in range(len(mt.w)):
        d = dict(w=W.to_numpy_bits(mt.w[k]), g=W.to_numpy_bits(mt.g[k]), m=W.to_numpy_bits(mt.m[k]),
                 v=W.to_numpy_bits(mt.v[k]), ve=W.to_numpy_bits(mt.ve[k]))
        if mt.bscale and mt.bscale[k] is not None:
            d["bscale"] = W.to_numpy_bits(mt.bscale[k])
        if mt.gscale and mt.gscale[k]:
            d["gscale"] = float(mt.gscale[k])
        out.append(d)
    return out


GUARD_BYTES = 64      # canary bytes before and after every separately allocated array
CANARY = 0xA5


def _guarded(t: torch.Tensor, misalign: int = 0):
    """A CUDA copy of t inside a larger buffer whose bytes before and after
    it hold a canary pattern (and, with misalign, shifted by that many
    elements); returns (view, guard record)."""
    es = t.element_size()
    g = GUARD_BYTES // es
    buf = torch.empty(t.numel() + 2 * g + misalign, dtype=t.dtype, device="cuda")
    buf.view(torch.uint8).fill_(CANARY)
    v = buf[g + misalign:g + misalign + t.numel()]
    v.copy_(t)
    return v, (buf, (g + misalign) * es, t.numel() * es)


def canary_damage(guards) -> int:
    """Bytes outside the arrays' own ranges that no longer hold the canary."""
    bad = 0
    for buf, start, nbytes in guards:
        b = buf.view(torch.uint8)
        bad += int((b[:start] != CANARY).sum()) + int((b[start + nbytes:] != CANARY).sum())
    return bad


def device_copy(mt: W.Materialized, layout: str = "separate", misalign: int = 0) -> Dict[str, list]:
    """Copy a CPU-materialised workload to cuda:0.  Separately allocated
    arrays sit between canary bytes (checked by canary_damage(out["_guards"]));
    misalign > 0 also shifts every tensor by that many elements (vector path
    off)."""
    out = {"_guards": []}
    for key in ("w", "g", "m", "v", "ve"):
        src = getattr(mt, key)
        if layout == "flat" and key in mt.flat:
            base, guard = _guarded(mt.flat[key])
            out["_guards"].append(guard)
            out[key] = [base[o:o + t.numel()] for o, t in zip(mt.offsets, src)]
        else:
            views = []
            for t in src:
                v, guard = _guarded(t, misalign)
                out["_guards"].append(guard)
                views.append(v)
            out[key] = views
    for key, src in (("bscale", mt.bscale), ("cc", mt.cc)):
        views = []
        for t in (src or [None] * len(mt.w)):
            if t is None:
                views.append(None)
            else:
                v, guard = _guarded(t, misalign)
                out["_guards"].append(guard)
                views.append(v)
        out[key] = views
    return out


def bits_equal(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """Element-wise equality of stored bit patterns, any NaN equal to any NaN."""
    eq = a.view(a.dtype) == b.view(b.dtype)
    if a.dtype == np.float32:
        ua, ub = a.view(np.uint32), b.view(np.uint32)
        eq = (ua == ub) | (np.isnan(a) & np.isnan(b))
    return eq


def mismatches(got: np.ndarray, want: np.ndarray) -> int:
    return int((~bits_equal(got, want)).sum())


def contract_ok(got_w, want_w, got_m, want_m, wdt: str) -> bool:
    """The method's parity bar (weaker than bit-exact)."""
    bad = ~bits_equal(got_w, want_w)
    if bad.any():
        if wdt == "bf16":
            d = np.abs(got_w[bad].astype(np.int64) - want_w[bad].astype(np.int64))
        else:
            d = np.abs((got_w[bad] & 0x7F).astype(np.int64) - (want_w[bad] & 0x7F).astype(np.int64))
        if d.max() > 1 or bad.mean() > 1e-4:
            return False
    if got_m.dtype == np.float32:
        with np.errstate(invalid="ignore", over="ignore"):  # inf - inf: decided by the bit comparison
            ok = bits_equal(got_m, want_m) | (np.abs(got_m - want_m) <= 1e-5 * np.abs(want_m))
        return bool(ok.all())
    return bool(bits_equal(got_m, want_m).all())


class Run:
    """A GPU optimizer and an oracle twin over the same workload."""

    def __init__(self, wl: W.Workload, *, warm: bool = False, layout: str = "separate",
                 misalign: int = 0, hp: Optional[Dict] = None, mt: Optional[W.Materialized] = None):
        self.wl = wl
        self.hp = dict(hp or {})
        self.mt = mt if mt is not None else W.materialize(wl, "cpu", layout=layout, warm_state=warm)
        self.host = host_tensors(self.mt)
        self.dev = device_copy(self.mt, layout, misalign)
        self.ohp = oracle_hparams(wl, self.hp)
        gkw = {k: v for k, v in self.hp.items() if k in HP_KEYS}
        self.formats = list(self.mt.formats) if self.mt.formats else [wl.weight_dtype] * len(self.mt.w)
        extended = wl.weight_dtype not in ("bf16", "e4m3") or bool(wl.format_list) or \
            any(x is not None for x in self.dev["cc"])
        self.opt = MPAdam(self.dev["w"], self.dev["m"], self.dev["v"], self.dev["ve"],
                          weight_dtype=self.formats if extended else wl.weight_dtype, grad_dtype=wl.grad_dtype,
                          moment_dtype=wl.moment_dtype, rounding=wl.rounding, seed=wl.seed,
                          fp8_exp=self.mt.fp8_exp,
                          block_scales=self.dev["bscale"] if extended else None,
                          compute=self.dev["cc"] if extended else None,
                          global_scales=self.mt.gscale if extended else None, **gkw)
        self.e4m3 = [k for k, f in enumerate(self.formats) if f == "e4m3"]
        self.fp8 = None
        if self.e4m3:
            self.fp8 = [None] * len(self.host)
            for k in self.e4m3:
                self.fp8[k] = oracle.fp8_init([self.host[k]], [self.mt.fp8_exp[k]])[0]
        self.wdt = [ODT[f] for f in self.formats]
        self.gdt, self.mdt = ODT[wl.grad_dtype], ODT[wl.moment_dtype]
        self.stepped = False

    def step(self, t: int):
        self.opt.step(self.dev["g"], t)
        oracle.step(self.host, wdt=self.wdt, gdt=self.gdt, mdt=self.mdt, hp=self.ohp, t=t,
                    fp8_state=self.fp8)
        torch.cuda.synchronize()
        self.stepped = True
        assert self.opt.device_status() == 0, "a bounded wait in the step kernel gave up"


    def expected_compute_copy(self, k: int) -> np.ndarray:
        """The oracle's BF16 compute copy of tensor k's current stored weights."""
        h = self.host[k]
        if self.formats[k] == "e4m3_b32":
            return oracle.dequant_bf16(h["w"], bscale=h["bscale"])
        if self.formats[k] == "nvfp4":
            return oracle.dequant_nvfp4_bf16(h["g"].size, h["w"], h["bscale"], h["gscale"])
        return oracle.dequant_bf16(h["w"], e=self.fp8[k][0])

    def compare(self, t_next: int, compute_copy: bool = True) -> Dict[str, int]:
        """Mismatch counts per array (and the E4M3 scale state read for step
        t_next); compute copies are checked when compute_copy, once a step has
        written them."""
        res = {"w": 0, "m": 0, "v": 0, "ve": 0, "bscale": 0, "cc": 0, "elements": 0, "contract_ok": True,
               "canary": canary_damage(self.dev["_guards"])}
        for k in range(len(self.host)):
            h = self.host[k]
            res["elements"] += h["g"].size
            gw = W.to_numpy_bits(self.dev["w"][k])
            gm = W.to_numpy_bits(self.dev["m"][k])
            res["w"] += mismatches(gw, h["w"])
            res["m"] += mismatches(gm, h["m"])
            res["v"] += mismatches(W.to_numpy_bits(self.dev["v"][k]), h["v"])
            res["ve"] += mismatches(W.to_numpy_bits(self.dev["ve"][k]), h["ve"])
            if "bscale" in h:
                res["bscale"] += mismatches(W.to_numpy_bits(self.dev["bscale"][k]), h["bscale"])
            if compute_copy and self.stepped and self.dev["cc"][k] is not None and h["g"].size:
                res["cc"] += mismatches(W.to_numpy_bits(self.dev["cc"][k]), self.expected_compute_copy(k))
            fmt = "bf16" if self.formats[k] == "bf16" else "e4m3"
            if self.formats[k] == "nvfp4":   # codes compared through their nibbles
                gw = oracle.nvfp4_unpack(gw, h["g"].size)
                hw = oracle.nvfp4_unpack(h["w"], h["g"].size)
                if hw.size and not contract_ok(gw, hw, gm, h["m"], "e4m3"):
                    res["contract_ok"] = False
                continue
            if h["w"].size and not contract_ok(gw, h["w"], gm, h["m"], fmt):
                res["contract_ok"] = False
        if self.fp8 is not None:
            exps = self.opt.fp8_exponents(t_next)
            amax = self.opt.fp8_amax(t_next).cpu().numpy()
            res["fp8_exp"] = sum(int(exps[k] != self.fp8[k][0]) for k in self.e4m3)
            res["fp8_amax"] = sum(int(np.float32(amax[k]).view(np.uint32) != np.float32(self.fp8[k][1]).view(np.uint32))
                                  for k in self.e4m3)
        return res

    def close(self):
        self.opt.close()


def assert_exact(res: Dict[str, int], what: str = ""):
    bad = {k: v for k, v in res.items() if k not in ("elements", "contract_ok") and v}
    assert not bad, f"{what}: mismatching elements {bad} of {res['elements']}"
