"""Writes tests/golden/step_cases.json: small hand-made cases and the oracle's
stored results after each step.  Calls only oracle/ (run from the repository
root: python tests/golden/make_golden.py).  Each case cites the passage whose
behaviour it exercises."""
import json
import math
import sys
from pathlib import Path

import numpy as np

ROOT = Path(__file__).resolve().parents[2]
sys.path.insert(0, str(ROOT))
import oracle  # noqa: E402

F32, BF16, E4M3 = oracle.F32, oracle.BF16, oracle.E4M3
NAMES = {F32: "f32", BF16: "bf16", E4M3: "e4m3"}


def bf(x):
    return oracle.bf16_rne(np.array(x, np.float32))


def f32(x):
    return np.array(x, np.float32)


CASES = [
    dict(name="hand_made_first_steps", cite="Algorithm 1; Sec. 4.1 (both branches from a zero state)",
         w=[1.0, -2.0, 0.5, 0.0, 256.0, 1e-9, -0.03, 3e-3, 1.0, -1.0, 0.02, -0.02, 7.0, -1e-4, 0.3, 0.0],
         g=[0.5, -0.5, 1e-3, -1e-3, 0.5, 1e-3, 2e-2, -1e-3, 1e-8, 3e-9, 1e-5, -1e-5, -0.25, 1e-2, 0.0, 0.0],
         hp={}, wdt=BF16, gdt=F32, mdt=F32, steps=3),
    dict(name="large_weight_stall", cite="Sec. 1, Fig. 1, Table 1 (additive steps vanish at large |w| in BF16)",
         w=[256.0, -300.0, 1024.0, 128.0, -512.0, 200.0, 300.0, -256.0],
         g=[0.5, -0.5, 0.1, -0.1, 0.3, 0.2, -0.2, 1.0],
         hp=dict(lr_add=1e-3, lr_mul=0.0), wdt=BF16, gdt=F32, mdt=F32, steps=4),
    dict(name="multiplicative_moves_large_weights", cite="Sec. 1, Fig. 1, Table 1 (non-zero update at large |w|)",
         w=[256.0, -300.0, 1024.0, 128.0, -512.0, 200.0, 300.0, -256.0],
         g=[0.5, -0.5, 0.1, -0.1, 0.3, 0.2, -0.2, 1.0],
         hp=dict(lr_add=1e-3, lr_mul=2.0), wdt=BF16, gdt=F32, mdt=F32, steps=4),
    dict(name="madam_absorbs_zero", cite="Sec. 3 (Madam cannot escape w = 0); Fig. 4(b)",
         w=[0.0, -0.0, 0.0, 1.0, -1.0, 0.0, 0.5, 0.0],
         g=[1e-2, -1e-2, 1e-3, 1e-2, 1e-2, -1e-3, 1e-3, 1e-1],
         hp=dict(lr_add=0.0, lr_mul=1e-2), wdt=BF16, gdt=F32, mdt=F32, steps=3),
    dict(name="step_cap_and_clips", cite="Algorithm 2 (g_max, the 0.75 bounds, d_mult,max, w_max, decay)",
         w=[1.0, -1.0, 0.3, 2.0, 1e-3, -5e-4, 0.06, -0.07],
         g=[1.0, 1.0, -1.0, 1e-3, 0.5, -0.5, 0.2, -0.2],
         hp=dict(lr_add=1e-2, lr_mul=0.5, g_max=0.8, dmult_max=0.1, w_max=0.05, wd_add=0.1, rmax_neg=0.6),
         wdt=BF16, gdt=F32, mdt=F32, steps=3),
    dict(name="stochastic_rounding_bf16", cite="Sec. 2 / Sec. 5.2 (stochastic rounding of BF16 weights)",
         w=[0.02 * math.sin(i) for i in range(24)], g=[1e-3 * math.cos(3 * i) for i in range(24)],
         hp=dict(stochastic=1, seed=1234), wdt=BF16, gdt=BF16, mdt=BF16, steps=3),
    dict(name="e4m3_per_tensor_scale", cite="Sec. 5.2 and the FP8-master figure (FP8 weights with scales)",
         w=[0.02 * math.sin(i) for i in range(32)], g=[1e-3 * math.cos(2 * i) for i in range(32)],
         hp=dict(stochastic=1, seed=77), wdt=E4M3, gdt=BF16, mdt=F32, steps=3, e0=-11),
    dict(name="no_bias_correction", cite="Algorithm 2 (raw moments)",
         w=[0.5, -0.25, 0.125, 0.0, 3.0, -3.0, 1e-6, -1e-6], g=[0.1, 0.1, -0.1, 0.1, 1e-4, -1e-4, 1.0, -1.0],
         hp=dict(bias_correction=0), wdt=BF16, gdt=F32, mdt=F32, steps=3),
    dict(name="non_finite_values", cite="(propagation of non-finite inputs; no step skipping)",
         w=[1.0, math.inf, math.nan, -1.0, 0.5, 0.0, 2.0, -2.0],
         g=[math.nan, 1e-3, 1e-3, math.inf, -math.inf, math.nan, 0.0, 1e-3],
         hp={}, wdt=BF16, gdt=F32, mdt=F32, steps=2),
]


def enc_w(case):
    w = f32(case["w"])
    if case["wdt"] == BF16:
        return oracle.bf16_rne(w)
    return oracle.e4m3_rne(w * np.float32(2.0 ** -case["e0"]))


def enc_g(case):
    g = f32(case["g"])
    return oracle.bf16_rne(g) if case["gdt"] == BF16 else g


def zeros_m(case, n):
    return np.zeros(n, np.uint16) if case["mdt"] == BF16 else np.zeros(n, np.float32)


def run(case):
    w = enc_w(case)
    n = w.size
    t = dict(w=w, g=enc_g(case), m=zeros_m(case, n), v=zeros_m(case, n), ve=zeros_m(case, n))
    hp = oracle.hparams(**case["hp"])
    fp8 = oracle.fp8_init([t], [case["e0"]]) if case["wdt"] == E4M3 else None
    out = []
    for step in range(1, case["steps"] + 1):
        oracle.step([t], wdt=case["wdt"], gdt=case["gdt"], mdt=case["mdt"], hp=hp, t=step, fp8_state=fp8)
        rec = {k: t[k].view(np.uint16 if t[k].dtype == np.uint16 else (np.uint8 if t[k].dtype == np.uint8 else np.uint32)).tolist()
               for k in ("w", "m", "v", "ve")}
        if fp8 is not None:
            rec["fp8_exp"] = fp8[0][0]
            rec["fp8_amax_bits"] = int(np.float32(fp8[0][1]).view(np.uint32))
        out.append(rec)
    return out


def build():
    cases = []
    for c in CASES:
        w0 = enc_w(c)
        g0 = enc_g(c)
        cases.append(dict(
            name=c["name"], cite=c["cite"], hparams=c["hp"], weight_dtype=NAMES[c["wdt"]],
            grad_dtype=NAMES[c["gdt"]], moment_dtype=NAMES[c["mdt"]], fp8_exp0=c.get("e0"),
            w0=w0.view(np.uint16 if w0.dtype == np.uint16 else np.uint8).tolist(),
            g=(g0.view(np.uint16) if g0.dtype == np.uint16 else g0.view(np.uint32)).tolist(),
            steps=run(c)))
    return cases


if __name__ == "__main__":
    out = ROOT / "tests" / "golden" / "step_cases.json"
    out.write_text(json.dumps(dict(
        note="Oracle results (written by tests/golden/make_golden.py, which calls only oracle/). "
             "Arrays hold stored bit patterns: uint16 for BF16, uint8 for E4M3, uint32 for binary32. "
             "Moments start at zero; hyper-parameters not listed take the oracle defaults.",
        cases=build()), indent=0))
    print(out)
