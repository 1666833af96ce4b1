"""Host-side logic of bench.py and of the product boundary, on CPU:
- the max-over-ranks timing and whole-job rate of the replicated (N > 1)
  run, with two gloo ranks;
- the reference arm (the oracle timed on the host) prints one valid line;
- the product path refuses to run without its CUDA library (no fallback);
- the hash that keys recorded DRAM traffic follows code, not comments;
- the algorithmic bytes behind the roofline, per tensor role."""
import json
import os
import subprocess
import sys
from pathlib import Path

import pytest
import torch.multiprocessing as mp

ROOT = Path(__file__).resolve().parents[1]


def _rank(rank, world, port, q):
    import torch.distributed as dist
    sys.path.insert(0, str(ROOT))
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms = [12.5, 19.25][rank]
    q.put((rank, bench.max_over_ranks(ms, "cpu")))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_with_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + os.getpid() % 1000
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert got == {0: 19.25, 1: 19.25}
    sys.path.insert(0, str(ROOT))
    import bench
    assert bench.whole_job_rate(6_738_415_616, 2, 19.25) == pytest.approx(2 * 6.738415616 / 0.01925)


def test_reference_arm_prints_one_json_line():
    r = subprocess.run([sys.executable, str(ROOT / "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "3", "--config", "gpt2_124m"], capture_output=True, text=True, timeout=600,
                       cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "Gparams/s" and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["higher_is_better"] is True and d["config"]["workload"] == "gpt2_124m"


def test_product_path_fails_loudly_without_its_library(monkeypatch, tmp_path):
    from paper_2607_10611_gb300 import _native, builder
    monkeypatch.setattr(builder, "LIB", tmp_path / "missing" / "libmpadam.so")
    monkeypatch.setattr(_native, "_LIB", None)
    with pytest.raises(RuntimeError, match="build the CUDA library"):
        _native.lib()


def test_kernel_source_hash_ignores_comments_but_not_code(tmp_path, monkeypatch):
    """The hash that keys the recorded DRAM traffic changes with the kernel's
    code, not with its comments or blank lines."""
    import shutil
    sys.path.insert(0, str(ROOT))
    import bench
    csrc = tmp_path / "paper_2607_10611_gb300" / "csrc"
    shutil.copytree(ROOT / "paper_2607_10611_gb300" / "csrc", csrc)
    monkeypatch.setattr(bench, "ROOT", tmp_path)
    h0 = bench.kernel_source_hash()
    k = csrc / "step_kernel.cuh"
    text = k.read_text()
    k.write_text("// a new comment\n\n/* and a block\n   comment */\n" + text.replace("\n", "  // note\n", 1))
    assert bench.kernel_source_hash() == h0
    k.write_text(text.replace("constexpr uint32_t kSpinLimit = 1u << 22;", "constexpr uint32_t kSpinLimit = 1u << 21;"))
    assert bench.kernel_source_hash() != h0



@pytest.mark.parametrize("name,per_matrix,per_other", [
    ("llama_7b", 18.0, 18.0),          # bf16 w read+written, bf16 g, three bf16 moments read+written
    ("llama_1p5b", 28.0, 28.0),        # E4M3 w (1+1), bf16 g, three fp32 moments (24)
    ("gpt2_124m", 30.0, 30.0),         # bf16 w (2+2), bf16 g, fp32 moments
    ("flat_1m", 32.0, 32.0),           # bf16 w, fp32 g, fp32 moments
    ("llama_1p5b_mixed", 30.125, 30.0),  # + 2-byte block scale per 32 (r+w) + 2-byte compute copy
    ("llama_1p5b_nvfp4", 29.125, 30.0),  # half-byte codes (r+w), 1-byte scale per 16 (r+w), copy
])
def test_roofline_bytes_per_element(name, per_matrix, per_other):
    """The denominator of the roofline: algorithmic bytes of one step, from
    first principles per tensor role (linears in the low-precision format,
    the rest BF16 in the mixed lists)."""
    sys.path.insert(0, str(ROOT))
    import bench
    import workloads as W
    wl = W.CONFIGS[name]
    want = sum(s.numel * (per_matrix if s.role == "matrix" else per_other) for s in wl.specs)
    assert bench.algorithmic_bytes(wl) == pytest.approx(want, rel=1e-9)
