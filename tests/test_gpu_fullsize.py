"""Parity at the full workload sizes, over each configuration's own step
count, in the launch configuration bench.py times (default grid and tail
pool, flat layout, inputs drawn on the GPU).

- flat_1m: every element, all 10 steps.
- gpt2_124m (100 steps), llama_7b and ragged_20k (10 steps): about a million
  sampled elements (random positions plus each tensor's first and last
  elements), stepped by the oracle one by one with their global indices.
  Every step continues from the oracle's own results of the step before
  (equal to the GPU's bit for bit, checked at every step), so no oracle input
  ever comes from the CUDA path.  The bias corrections change with t
  (Algorithm 1), so later steps are not repeats of the first.
- llama_1p5b (per-tensor E4M3): a tensor's scale depends on all of it, so
  step 1 is checked on samples of every tensor (with the amax the oracle
  computes from the stored codes), and 10 steps on whole tensors -- the
  embedding, a q projection, an FFN gate and down projection, norm gains and
  the final norm -- including the recorded scale rings at every step (their
  slots rotate with period 6).
- llama_1p5b_mixed (the FP8 regime) and llama_1p5b_nvfp4 (the NVFP4 regime,
  both roundings): 10 steps on whole sampled blocks of every low-precision
  linear (a block's scale depends on all of it) and sampled elements of every
  BF16 tensor, with block scales and compute copies.
The oracle runs on whole tensors are split across host threads (the update
is element-wise and the oracle's C calls release the GIL).
"""
import gc
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
import workloads as W

pytestmark = pytest.mark.gpu

ODT = {"f32": oracle.F32, "bf16": oracle.BF16, "e4m3": oracle.E4M3}
DEVICE = "cuda"
KEYS = ("w", "g", "m", "v", "ve")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_10611_gb300 import build
    build()


def _sync():
    if DEVICE == "cuda":
        torch.cuda.synchronize()


def _bits(t: torch.Tensor) -> np.ndarray:
    t = t.cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16).copy()
    if t.dtype == torch.float16:
        return t.view(torch.int16).numpy().view(np.uint16).copy()
    return t.numpy().copy()


def _free():
    gc.collect()
    if DEVICE == "cuda":
        torch.cuda.synchronize()
        torch.cuda.empty_cache()


def make_opt(wl, mt):
    """The CUDA optimizer as bench.py builds it."""
    from paper_2607_10611_gb300.optimizer import MPAdam
    extended = wl.weight_dtype not in ("bf16", "e4m3") or wl.compute_copy
    return MPAdam(mt.w, mt.m, mt.v, mt.ve, weight_dtype=mt.formats if extended else wl.weight_dtype,
                  grad_dtype=wl.grad_dtype, moment_dtype=wl.moment_dtype, rounding=wl.rounding, seed=wl.seed,
                  fp8_exp=mt.fp8_exp, block_scales=mt.bscale if extended else None,
                  compute=mt.cc if extended else None, global_scales=mt.gscale if extended else None)


def _setup(wl):
    mt = W.materialize(wl, DEVICE, layout="flat")
    return mt, make_opt(wl, mt)


def _pool():
    return ThreadPoolExecutor(max_workers=max(1, min(16, os.cpu_count() or 1)))


def _sample_positions(mt, n_random, seed):
    rng = np.random.default_rng(seed)
    numels = np.array([t.numel() for t in mt.g], dtype=np.int64)
    offs = np.array(mt.offsets, dtype=np.int64)
    heads = np.concatenate([offs[k] + np.arange(min(4, n)) for k, n in enumerate(numels) if n])
    tails = np.concatenate([offs[k] + np.arange(max(0, n - 4), n) for k, n in enumerate(numels) if n])
    # random elements, weighted by size, mapped into the padded global space
    cum = np.cumsum(numels)
    flat = rng.integers(0, cum[-1], n_random)
    k = np.searchsorted(cum, flat, side="right")
    within = flat - np.concatenate([[0], cum[:-1]])[k]
    pos = np.unique(np.concatenate([heads, tails, offs[k] + within]))
    tens = np.searchsorted(offs, pos, side="right") - 1
    return pos, tens


def _gather(mt, pos, keys=KEYS):
    p = torch.from_numpy(pos).to(DEVICE)
    return {key: _bits(mt.flat[key].index_select(0, p)) for key in keys}


def _assert_same(got, want, what, keys=("w", "m", "v", "ve")):
    for key in keys:
        a, b = got[key], want[key]
        eq = a.view(a.dtype) == b.view(b.dtype)
        if a.dtype == np.float32:
            eq = (a.view(np.uint32) == b.view(np.uint32)) | (np.isnan(a) & np.isnan(b))
        bad = int((~eq).sum())
        assert bad == 0, f"{what}: {bad} of {a.size} sampled {key} differ"


def _chunked_step(pool, wl, hp, t, h, gidx0, e_cur=0, e_next=0, chunk=1 << 22):
    """One oracle step over a whole tensor's host arrays, in chunks run on
    host threads; returns the largest finite |w'| over all of them."""
    n = h["g"].size
    futs = []
    for a in range(0, n, chunk):
        b = min(n, a + chunk)
        arrs = [h[key][a:b] for key in KEYS]
        futs.append(pool.submit(oracle.step_elements, hp, t, ODT[wl.weight_dtype], ODT[wl.grad_dtype],
                                ODT[wl.moment_dtype], *arrs, gidx0=gidx0 + a, e_cur=e_cur, e_next=e_next))
    return max([f.result() for f in futs], default=0.0)


def test_flat_1m_every_element_all_steps():
    wl = W.CONFIGS["flat_1m"]
    mt, opt = _setup(wl)
    hp = oracle.hparams(stochastic=0, seed=wl.seed)
    pos = np.arange(mt.g[0].numel(), dtype=np.int64)
    host = _gather(mt, pos)
    for t in range(1, wl.steps + 1):
        opt.step(mt.g, t)
        oracle.step_elements(hp, t, ODT[wl.weight_dtype], ODT[wl.grad_dtype], ODT[wl.moment_dtype],
                             *[host[k] for k in KEYS], gidx=pos)
        _assert_same(_gather(mt, pos, ("w", "m", "v", "ve")), host, f"flat_1m step {t}")
    assert opt.device_status() == 0
    opt.close()
    del mt, opt
    _free()


@pytest.mark.parametrize("name,rounding,steps", [("gpt2_124m", None, 100), ("llama_7b", None, 10),
                                                 ("ragged_20k", "nearest", 10), ("ragged_20k", "stochastic", 10)])
def test_large_bf16_lists_sampled_over_their_steps(name, rounding, steps):
    wl = W.CONFIGS[name]
    if rounding:
        wl = W.replace(wl, rounding=rounding)
    mt, opt = _setup(wl)
    hp = oracle.hparams(stochastic=1 if wl.rounding == "stochastic" else 0, seed=wl.seed)
    pos, _ = _sample_positions(mt, 1_000_000, seed=7)
    host = _gather(mt, pos)
    for t in range(1, steps + 1):
        opt.step(mt.g, t)
        oracle.step_elements(hp, t, ODT[wl.weight_dtype], ODT[wl.grad_dtype], ODT[wl.moment_dtype],
                             *[host[k] for k in KEYS], gidx=pos)
        _assert_same(_gather(mt, pos, ("w", "m", "v", "ve")), host, f"{name} step {t}")
    assert opt.device_status() == 0
    opt.close()
    del mt, opt
    _free()


def llama_whole_tensors(n_tensors, layers=24):
    """Embedding, layer 0's q projection, layer 11's FFN gate, layer 23's
    down projection, two norm gains and the final norm (list positions:
    embedding first, then 9 tensors per layer, then the final norm and the
    head)."""
    per = 9
    return [0, 1 + 0, 1 + 11 * per + 4, 1 + 23 * per + 6, 1 + 7, 1 + 12 * per + 8, n_tensors - 2]


def test_llama_1p5b_e4m3_over_ten_steps():
    wl = W.CONFIGS["llama_1p5b"]
    mt, opt = _setup(wl)
    hp = oracle.hparams(stochastic=1, seed=wl.seed)
    n = len(mt.g)
    # the oracle's own scale state before step 1: largest |decoded stored weight|
    st = [[mt.fp8_exp[k], oracle.e4m3_amax(_bits(mt.w[k]), mt.fp8_exp[k])] for k in range(n)]
    a_gpu = opt.fp8_amax(1).cpu().numpy()
    assert all(np.float32(a_gpu[k]) == np.float32(st[k][1]) for k in range(n))

    whole = llama_whole_tensors(n)
    whole_host = {k: {key: _bits(getattr(mt, key)[k]) for key in KEYS} for k in whole}
    whole_state = {k: list(st[k]) for k in whole}

    # sampled elements over every tensor, step 1
    pos, tens = _sample_positions(mt, 1_000_000, seed=11)
    host = _gather(mt, pos)
    opt.step(mt.g, 1)
    _sync()
    for k in np.unique(tens):
        sel = tens == k
        sub = {key: np.ascontiguousarray(host[key][sel]) for key in host}
        e_next = oracle.fp8_next_exponent(st[k][1], st[k][0])
        oracle.step_elements(hp, 1, oracle.E4M3, ODT[wl.grad_dtype], ODT[wl.moment_dtype],
                             *[sub[key] for key in KEYS], gidx=pos[sel], e_cur=st[k][0], e_next=e_next)
        for key in host:
            host[key][sel] = sub[key]
    _assert_same(_gather(mt, pos, ("w", "m", "v", "ve")), host, "llama_1p5b step 1 (sampled)")

    # whole tensors: steps 1 .. 10, with the recorded scale state
    with _pool() as pool:
        for t in range(1, wl.steps + 1):
            if t > 1:
                opt.step(mt.g, t)
                _sync()
            exps = opt.fp8_exponents(t + 1)
            amax = opt.fp8_amax(t + 1).cpu().numpy()
            for k in whole:
                h = whole_host[k]
                e_cur, a_cur = whole_state[k]
                e_next = oracle.fp8_next_exponent(a_cur, e_cur)
                a_next = _chunked_step(pool, wl, hp, t, h, mt.offsets[k], e_cur, e_next)
                whole_state[k] = [e_next, a_next]
                got = {key: _bits(getattr(mt, key)[k]) for key in ("w", "m", "v", "ve")}
                _assert_same(got, h, f"llama_1p5b tensor {k} step {t}")
                assert exps[k] == e_next, (k, t)
                assert np.float32(amax[k]).view(np.uint32) == np.float32(a_next).view(np.uint32), (k, t)
    assert opt.device_status() == 0
    opt.close()
    del mt, opt
    _free()


def _block_picks(wl, mt, block, n_blocks, n_elems, seed):
    """Per tensor: whole sampled blocks (block-scaled formats) or sampled
    elements (BF16), as (k, element indices, block indices or None)."""
    rng = np.random.default_rng(seed)
    picks = []
    for k, (n, f) in enumerate(zip(wl.numels, mt.formats)):
        if f in ("e4m3_b32", "nvfp4"):
            nb = (n + block - 1) // block
            blocks = np.unique(np.concatenate([[0, nb - 1], rng.integers(0, nb, n_blocks)]))
            idx = np.concatenate([np.arange(block * b, min(n, block * b + block)) for b in blocks])
            picks.append((k, idx, blocks))
        else:
            idx = np.unique(np.concatenate([[0, n - 1], rng.integers(0, n, n_elems)]))
            picks.append((k, idx, None))
    return picks


def _gather_picked(mt, k, idx, blocks, fmt):
    p = torch.from_numpy(idx).to(DEVICE)
    d = {key: _bits(getattr(mt, key)[k].index_select(0, p)) for key in KEYS if key != "w"}
    if fmt == "nvfp4":  # blocks start at even elements: whole bytes, 8 per block
        nbytes = mt.w[k].numel()
        byte_idx = np.concatenate([np.arange(8 * b, min(nbytes, 8 * b + 8)) for b in blocks])
        d["w"] = _bits(mt.w[k].index_select(0, torch.from_numpy(byte_idx).to(DEVICE)))
    else:
        d["w"] = _bits(mt.w[k].index_select(0, p))
    if blocks is not None:
        d["bscale"] = _bits(mt.bscale[k].index_select(0, torch.from_numpy(blocks).to(DEVICE)))
        d["cc"] = _bits(mt.cc[k].index_select(0, p))
    return d


@pytest.mark.parametrize("name,rounding", [("llama_1p5b_mixed", None), ("llama_1p5b_nvfp4", None),
                                           ("llama_1p5b_nvfp4", "stochastic")])
def test_paper_regimes_sampled_blocks_over_ten_steps(name, rounding):
    """The paper's FP8 regime (block-scaled E4M3 linears) and NVFP4 regime
    (NVFP4 linears) at full size, with BF16 compute copies and the rest of
    the list in BF16."""
    wl = W.CONFIGS[name]
    if rounding:
        wl = W.replace(wl, rounding=rounding)
    mt, opt = _setup(wl)
    hp = oracle.hparams(stochastic=1 if wl.rounding == "stochastic" else 0, seed=wl.seed)
    gd, md = ODT[wl.grad_dtype], ODT[wl.moment_dtype]
    fmt_lp = "nvfp4" if "nvfp4" in mt.formats else "e4m3_b32"
    block = 16 if fmt_lp == "nvfp4" else 32
    picks = _block_picks(wl, mt, block, 150, 4000, seed=17)
    host = [_gather_picked(mt, k, idx, blocks, mt.formats[k]) for k, idx, blocks in picks]
    for t in range(1, wl.steps + 1):
        opt.step(mt.g, t)
        _sync()
        for (k, idx, blocks), h in zip(picks, host):
            goff = mt.offsets[k]
            if blocks is None:
                oracle.step_elements(hp, t, oracle.BF16, gd, md, *[h[key] for key in KEYS], gidx=goff + idx)
            else:
                pos = 0
                for j, b in enumerate(blocks):
                    ln = min(block, wl.numels[k] - block * int(b))
                    sl = slice(pos, pos + ln)
                    g, m, v, ve = (h[key][sl] for key in ("g", "m", "v", "ve"))
                    bs = h["bscale"][j:j + 1]
                    if fmt_lp == "nvfp4":
                        q = h["w"][8 * j:8 * j + (ln + 1) // 2]
                        oracle.step_nvfp4(hp, t, gd, md, ln, q, bs, mt.gscale[k], g, m, v, ve,
                                          gidx0=goff + block * int(b))
                        h["cc"][sl] = oracle.dequant_nvfp4_bf16(ln, q, bs, mt.gscale[k])
                    else:
                        q = h["w"][sl]
                        oracle.step_block_e4m3(hp, t, gd, md, q, bs, g, m, v, ve, gidx0=goff + block * int(b))
                        h["cc"][sl] = oracle.dequant_bf16(q, bscale=bs)
                    pos += ln
            got = _gather_picked(mt, k, idx, blocks, mt.formats[k])
            _assert_same(got, h, f"{name} tensor {k} step {t}")
            if blocks is not None:
                assert np.array_equal(got["bscale"], h["bscale"]), f"tensor {k} step {t}: block scales"
                assert np.array_equal(got["cc"], h["cc"]), f"tensor {k} step {t}: compute copy"
    assert opt.device_status() == 0
    opt.close()
    del mt, opt
    _free()
