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
    assert d["cpu_baseline"]["nproc"] == os.cpu_count()
    # the timed sample's own step time, and the sample's size, not an extrapolation
    assert d["sample_elements_per_step"] > 0
    assert d["ms_per_step"] == pytest.approx(1e3 * d["sample_elements_per_step"] / (d["value"] * 1e9), rel=0.5)
    # the same workload description as the GPU arm's line
    import bench
    import workloads as W
    wl = W.CONFIGS["gpt2_124m"]
    assert d["config"] == bench.workload_config(wl, 1, "inputs larger than L2 (no flush needed)")
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


def _fake_res(wl, ms, e2e=False):
    """What run_gpu returns, with plausible timings (full-precision floats)."""
    res = {"total_ms": ms * 20 * 1.0000123, "launch_ms": [ms * (1 + 1e-3 * i / 7) for i in range(20)],
           "wall": (0.0, 1.0), "grid": (152, 512), "launches_per_step": 1 + (wl.weight_dtype != "bf16"),
           "l2_flushed": wl.name == "flat_1m", "copy_ms": 0.0081234567 if wl.name == "flat_1m" else None,
           "one_tile_ms": 0.0082345678 if wl.name == "flat_1m" else None}
    if e2e:
        res.update(e2e_ms=101.234567, e2e_step_ms=[100.0 + 1.2345678 * i for i in range(20)],
                   h2d=13476831232, d2h=13476831232, link_ms=94.12345678, host_buffers="huge_pages",
                   host_probe_gbs={"huge_pages": 212.3, "driver": 204.9}, host_buffers_tried=2)
    return res


def test_result_line_keeps_every_secondary_list_in_the_driver_tail():
    """The driver records only the last ~1500 characters of the line: the
    secondary lists (the 1.5B target among them) must all sit there."""
    sys.path.insert(0, str(ROOT))
    import bench
    import workloads as W
    for name, w in W.CONFIGS.items():
        bench.W_DEFAULT_ROUNDING[name] = w.rounding
    wl = W.CONFIGS["llama_7b"]
    main = bench.summarize(wl, _fake_res(wl, 18.7654321, e2e=True), 1, 6783.5, "measured")
    secs = []
    for wl2 in bench.parse_secondary("llama_1p5b,llama_1p5b_mixed,llama_1p5b_nvfp4,"
                                     "llama_1p5b_nvfp4:stochastic,gpt2_124m,ragged_20k,flat_1m"):
        s2 = bench.summarize(wl2, _fake_res(wl2, 6.1234567), 1, 6783.5, "measured")
        s2["clocks"] = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 12}
        secs.append(s2)
    cpu = {"value": 0.018728084501097277, "unit": "Gparams/s", "cores": 1, "nproc": 72, "kind": "oracle",
           "sample": "one step over the first 181498738 elements of the llama_7b list (9.7 s, single thread)"}
    clocks = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 5}
    cpu_lists = {"flat_1m": {"params": 1048576, "whole_list": True, "seconds": 0.063, "ns_per_param": 60.12,
                             "gparams_per_s": 0.016634534016404936, "cores": 1},
                 "gpt2_124m": {"params": 124439808, "whole_list": True, "seconds": 7.291, "ns_per_param": 58.59,
                               "gparams_per_s": 0.017066754888876722, "cores": 1}}
    line = bench.result_line(wl, 1, 20, 5, "inputs larger than L2 (no flush needed)", main, cpu, clocks,
                             {"us_per_step": 15.51234}, "/tmp/bench_details.json", secs, 20, cpu_lists)
    text = json.dumps(line)
    assert len(text) < 3000, len(text)
    tail = text[-1400:]
    for s2 in secs:
        c = bench.compact(s2)
        assert json.dumps(c) in tail, c["workload"]
    assert '"workload": "llama_1p5b_nvfp4:stochastic"' in tail and '"workload": "llama_1p5b"' in tail
    for key in ("metric", "value", "unit", "ms_per_step", "roofline", "cpu_baseline", "e2e", "clocks"):
        assert key in line
    assert line["cpu_ns_per_param"] == {"flat_1m": 60.12, "gpt2_124m": 58.59}
    assert line["e2e"]["steps"] == 20 and line["e2e"]["ms_worst"] >= line["e2e"]["ms_median"]
    assert line["roofline"]["frac_of_nominal"] < line["roofline"]["frac"]
    # the e2e per-step times go to the details file only
    assert "step_ms" not in line["e2e"] and len(main["e2e"]["step_ms"]) == 20
    flat = [bench.compact(s2) for s2 in secs if s2["workload"] == "flat_1m"][0]
    assert flat["one_tile_ms"] == 0.0082 and flat["frac_of_copy"] > 0


def test_oracle_rate_on_a_whole_list():
    """The oracle's single-core rate is taken over one step of the whole list
    (the 1 Mi flat list here), not a sample of it."""
    sys.path.insert(0, str(ROOT))
    import bench
    r = bench.oracle_whole_lists("flat_1m")
    assert list(r) == ["flat_1m"]
    e = r["flat_1m"]
    assert e["whole_list"] and e["params"] == 1_048_576 and e["cores"] == 1
    assert e["ns_per_param"] > 0 and e["ns_per_param"] == pytest.approx(1.0 / e["gparams_per_s"], rel=1e-3)
    assert bench.oracle_whole_lists("") == {}
