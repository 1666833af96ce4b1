"""The seeded input generator: shapes, counts, layout and determinism."""
import numpy as np
import torch

import workloads as W


def test_parameter_counts_of_the_named_lists():
    assert W.CONFIGS["flat_1m"].n_params == 1_048_576
    assert W.CONFIGS["gpt2_124m"].n_params == 124_439_808
    assert len(W.CONFIGS["gpt2_124m"].specs) == 148
    assert W.CONFIGS["llama_1p5b"].n_params == 1_364_297_728
    assert len(W.CONFIGS["llama_1p5b"].specs) == 219
    assert W.CONFIGS["llama_7b"].n_params == 6_738_415_616
    assert len(W.CONFIGS["llama_7b"].specs) == 291
    r = W.CONFIGS["ragged_20k"]
    assert len(r.specs) == 20000
    sizes = np.array(r.numels)
    assert sizes.min() >= 1 and sizes.max() <= 1 << 22
    assert 4.5e9 < sizes.sum() < 6.5e9


def test_offsets_are_multiples_of_8_and_cover_each_tensor():
    numels = [1, 7, 8, 9, 0, 1000, 3]
    offs = W.global_offsets(numels)
    assert offs == [0, 8, 16, 24, 40, 40, 1040]
    assert W.global_length(numels) == 1048
    assert all(o % 8 == 0 for o in offs)


def test_materialize_is_deterministic_and_formats_match():
    for name, wl in W.SMALL.items():
        a = W.materialize(wl, "cpu", warm_state=True)
        b = W.materialize(wl, "cpu", warm_state=True)
        for x, y in zip(a.w + a.g + a.ve, b.w + b.g + b.ve):
            assert torch.equal(x, y)
        assert a.w[0].dtype == (torch.uint8 if wl.weight_dtype == "e4m3" else torch.bfloat16)
        if wl.weight_dtype == "e4m3":
            assert len(a.fp8_exp) == len(wl.specs)


def test_flat_layout_views_match_offsets():
    wl = W.SMALL["ragged_20k"]
    mt = W.materialize(wl, "cpu", layout="flat")
    base = mt.flat["w"].data_ptr()
    for k, o in enumerate(mt.offsets):
        assert mt.w[k].data_ptr() == base + 2 * o
    zero_frac = float(torch.cat([x.float() for x in mt.w]).eq(0).float().mean())
    assert 0.25 < zero_frac < 0.35
