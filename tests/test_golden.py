"""Golden fixtures (tests/golden/step_cases.json, written by
tests/golden/make_golden.py from the oracle): the oracle must still produce
them, they must show the behaviour their cited passage describes, and the
CUDA library must reproduce every stored bit."""
import json
import math
import sys
from pathlib import Path

import numpy as np
import pytest

ROOT = Path(__file__).resolve().parents[1]
GOLDEN = json.loads((ROOT / "tests" / "golden" / "step_cases.json").read_text())
CASES = {c["name"]: c for c in GOLDEN["cases"]}


def test_oracle_still_produces_the_fixtures():
    sys.path.insert(0, str(ROOT / "tests" / "golden"))
    import make_golden
    fresh = make_golden.build()
    assert [c["name"] for c in fresh] == [c["name"] for c in GOLDEN["cases"]]
    for a, b in zip(fresh, GOLDEN["cases"]):
        assert a == b, a["name"]


def _bf16(bits):
    return (np.array(bits, np.uint32) << 16).view(np.float32)


def test_fixtures_show_the_cited_behaviour():
    stall = CASES["large_weight_stall"]
    assert stall["steps"][-1]["w"] == stall["w0"]                    # Adam stalls at large |w|
    moved = CASES["multiplicative_moves_large_weights"]
    assert all(a != b for a, b in zip(moved["steps"][-1]["w"], moved["w0"]))
    madam = CASES["madam_absorbs_zero"]
    w0, w3 = _bf16(madam["w0"]), _bf16(madam["steps"][-1]["w"])
    assert np.all(w3[w0 == 0] == 0) and np.all(np.sign(w3[w0 != 0]) == np.sign(w0[w0 != 0]))
    cap = CASES["step_cap_and_clips"]
    w = _bf16(cap["steps"][-1]["w"])
    # w_max clip in binary32, then the BF16 store rounds 0.05 to its nearest BF16 value
    assert np.all(np.abs(w) <= _bf16([0x3D4D])[0]) and _bf16([0x3D4D])[0] == np.float32(0.050048828125)
    first = CASES["hand_made_first_steps"]
    w0, w1 = _bf16(first["w0"]), _bf16(first["steps"][0]["w"])
    g = np.array(first["g"], np.uint32).view(np.float32)
    moved = (w1 != w0) & (g != 0)
    assert np.all(np.sign(w1[moved] - w0[moved]) == -np.sign(g[moved]))  # descent direction


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(CASES))
def test_library_reproduces_the_fixtures(name):
    import torch
    from paper_2607_10611_gb300 import build
    from paper_2607_10611_gb300.optimizer import MPAdam
    build()
    c = CASES[name]
    n = len(c["w0"])
    wt = {"bf16": torch.int16, "e4m3": torch.uint8}[c["weight_dtype"]]
    w = torch.tensor(np.array(c["w0"], np.int64), dtype=torch.int64).to(wt)
    w = w.view(torch.bfloat16) if c["weight_dtype"] == "bf16" else w
    g = torch.tensor(np.array(c["g"], np.int64)).to(torch.int16 if c["grad_dtype"] == "bf16" else torch.int32)
    g = g.view(torch.bfloat16 if c["grad_dtype"] == "bf16" else torch.float32)
    md = torch.bfloat16 if c["moment_dtype"] == "bf16" else torch.float32
    m, v, ve = (torch.zeros(n, dtype=md, device="cuda") for _ in range(3))
    w, g = w.cuda(), g.cuda()
    hp = dict(c["hparams"])
    rounding = "stochastic" if hp.pop("stochastic", 0) else "nearest"
    seed = hp.pop("seed", 0)
    opt = MPAdam([w], [m], [v], [ve], weight_dtype=c["weight_dtype"], grad_dtype=c["grad_dtype"],
                 moment_dtype=c["moment_dtype"], rounding=rounding, seed=seed,
                 fp8_exp=[c["fp8_exp0"]] if c["fp8_exp0"] is not None else None,
                 **{k: (math.inf if v == "inf" else v) for k, v in hp.items()})
    bits = {torch.bfloat16: torch.int16, torch.float32: torch.int32, torch.uint8: torch.uint8}
    mask = {torch.bfloat16: 0xFFFF, torch.float32: 0xFFFFFFFF, torch.uint8: 0xFF}
    for t, want in enumerate(c["steps"], start=1):
        opt.step([g], t)
        torch.cuda.synchronize()
        for key, x in (("w", w), ("m", m), ("v", v), ("ve", ve)):
            got = (x.view(bits[x.dtype]).cpu().numpy().astype(np.int64) & mask[x.dtype]).tolist()
            if x.dtype == torch.float32:   # NaN equals NaN
                a, b = np.array(got, np.uint32).view(np.float32), np.array(want[key], np.uint32).view(np.float32)
                assert np.all((a.view(np.uint32) == b.view(np.uint32)) | (np.isnan(a) & np.isnan(b))), (name, t, key)
            else:
                assert got == want[key], (name, t, key)
        if "fp8_exp" in want:
            assert opt.fp8_exponents(t + 1)[0] == want["fp8_exp"]
            assert int(opt.fp8_amax(t + 1).cpu().numpy().view(np.uint32)[0]) == want["fp8_amax_bits"]
    assert opt.device_status() == 0
    opt.close()
