"""The step kernel's tile schedule, checked on the host (no GPU): every tile
of a launch is stepped exactly once, whichever static share, chunk length
and grid the tail pool runs with, and every run and chunk starts from the
tensor that really holds its first tile.  The schedule comes from the
library's own host code (mpadam_debug_tile_schedule), the same code that
builds the tables the kernel reads."""
import numpy as np
import pytest

from paper_2607_10611_gb300 import builder as B

TILE = 3840


@pytest.fixture(scope="module")
def N():
    B.build()
    from paper_2607_10611_gb300 import _native
    return _native


def tiles_of(n):
    return (n + TILE - 1) // TILE


def tensor_of_tile(numel):
    """Brute force: tile index -> tensor holding it."""
    owner = []
    for k, n in enumerate(numel):
        owner += [k] * tiles_of(n)
    return owner


def check(N, numel, ctas, q, chunk):
    runs, first, pool = N.mpadam_debug_tile_schedule(numel, ctas, q, chunk)
    owner = tensor_of_tile(numel)
    T = len(owner)
    seen = np.zeros(T, dtype=np.int64)
    for b in range(ctas):
        tb, ts, te = (int(x) for x in runs[b])
        assert tb == b * T // ctas and te == (b + 1) * T // ctas
        assert tb <= ts <= te
        if len(pool) and q < 1024:
            assert ts == tb + (te - tb) * q // 1024  # the kernel's split
        else:
            assert ts == te  # no pool: the whole run is static
        if tb < te:
            assert first[b] == owner[tb]
        seen[tb:ts] += 1
    last_end = -1
    for start, count, k in pool:
        start, count, k = int(start), int(count), int(k)
        assert 1 <= count <= chunk
        assert k == owner[start]
        assert start >= last_end  # claimed in tile order
        last_end = start + count
        # a chunk never leaves the tail of the run it came from
        b = next(b for b in range(ctas) if runs[b][1] <= start < runs[b][2])
        assert start + count <= runs[b][2]
        seen[start:start + count] += 1
    assert (seen == 1).all()


@pytest.mark.parametrize("q,chunk", [(1024, 4), (768, 4), (768, 1), (512, 7), (0, 1), (0, 64), (1000, 3)])
@pytest.mark.parametrize("ctas", [1, 7, 152, 1000])
def test_every_tile_once_on_a_llama_like_list(N, q, chunk, ctas):
    d, ffn, vocab = 512, 1376, 3000
    numel = [vocab * d]
    for _ in range(3):
        numel += [d, d * d, d * d, d * d, d * d, d, d * ffn, d * ffn, ffn * d]
    numel += [d, vocab * d]
    check(N, numel, ctas, q, chunk)


def test_every_tile_once_on_ragged_lists_with_empty_and_tiny_tensors(N):
    rng = np.random.default_rng(7)
    for trial in range(40):
        n = int(rng.integers(1, 60))
        numel = [int(x) for x in np.round(np.exp(rng.uniform(0, np.log(3 * TILE * 40), n)))]
        for i in rng.choice(n, size=min(n, 5), replace=False):
            numel[i] = int(rng.choice([0, 1, 7, TILE - 1, TILE, TILE + 1]))
        ctas = int(rng.choice([1, 3, 152, 500]))
        q = int(rng.choice([0, 256, 768, 1023, 1024]))
        chunk = int(rng.choice([1, 2, 4, 9]))
        check(N, numel, ctas, q, chunk)


def test_degenerate_lists(N):
    for numel in ([], [0], [0, 0, 0], [1], [TILE], [TILE + 1]):
        for ctas in (1, 152):
            for q in (0, 768, 1024):
                check(N, numel, ctas, q, 4)


def test_bad_arguments_are_refused(N):
    for args in (([10], 0, 768, 4), ([10], 4, -1, 4), ([10], 4, 1025, 4), ([10], 4, 768, 0), ([-1], 4, 768, 4)):
        with pytest.raises(N.MPAdamError) as ei:
            N.mpadam_debug_tile_schedule(*args)
        assert ei.value.status == N.MPADAM_EINVAL
