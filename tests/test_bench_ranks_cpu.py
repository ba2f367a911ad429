"""Host logic of bench.py on CPU.

Multi-rank bookkeeping (gloo, world size 2): the job's time is the slowest
rank's and its throughput counts every rank's examples.  Timing rules: the
L2 flush between timed steps for inputs that L2 could keep."""

import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    local = [2.5, 4.0][rank]                      # per-rank step time (ms)
    m = bench.max_over_ranks(local, world)
    v = bench.replica_throughput(16, world, m * 1e-3)
    out[rank] = (m, v)
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_step_and_count_all_examples():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    procs = [ctx.Process(target=_worker, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for r in range(world):
        m, v = out[r]
        assert m == 4.0                          # slowest rank
        assert v == pytest.approx(2 * 16 / 4.0e-3)


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.0, 1) == 3.0
    assert bench.replica_throughput(16, 1, 2e-3) == pytest.approx(8000.0)


def test_traffic_lookup(tmp_path):
    """profiles/traffic.json entries: scaled by units of work while the
    kernel's sources hash to the recorded value, None once they change, for
    an old single-file entry, or for an incomplete one."""
    import json
    sys.path.insert(0, ROOT)
    import bench
    src = ["paper_2609_20532_gb300/csrc/k_tc_gemm.cu", "paper_2609_20532_gb300/csrc/tc_util.cuh"]
    good = {"src": src, "src_sha256_16": bench._src_sha(src), "captured_units": 100.0,
            "captured_dram_bytes": 5000.0}
    data = {"k": good, "stale": dict(good, src_sha256_16="0" * 16),
            "old": {"src": src[0], "src_sha256_16": "x", "captured_flops": 1.0,
                    "captured_dram_bytes": 1.0},
            "partial": {"src": src}}
    p = tmp_path / "traffic.json"
    p.write_text(json.dumps(data))
    assert bench._traffic("k", 250.0, str(p)) == 12500.0
    for key in ("stale", "old", "partial", "missing"):
        assert bench._traffic(key, 1.0, str(p)) is None


def test_reference_arm_line_on_cpu():
    """`bench.py --impl reference` times the oracle on the host cores and
    prints the contract's JSON line: impl, the metric and unit of our arm,
    a cpu_baseline describing the run and an e2e with no host copies."""
    import json
    import subprocess
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--workload", "single_fp32", "--steps", "3", "--warmup", "3"],
                       capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    sys.path.insert(0, ROOT)
    import bench
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["unit"] == bench.UNIT and line["higher_is_better"] is True
    assert line["steps"] == 3 and line["warmup"] == 3 and line["value"] > 0
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"]
    assert "example 0 of single_fp32" in cb["sample"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"],
                           "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_l2_flush_applies_only_to_inputs_that_l2_could_keep(monkeypatch):
    """Timed steps flush L2 (a write larger than it) when the inputs are
    below twice its size; the LLM-scale inputs (763 MB) need no flush."""
    import torch
    sys.path.insert(0, ROOT)
    import bench
    assert bench.L2_FLUSH_BYTES > bench.L2_BYTES
    monkeypatch.setattr(bench, "L2_FLUSH_BYTES", 4096)   # keep the test's buffer small
    small = bench._l2_flush_buffer(torch.device("cpu"), 3 * 10**6)
    assert small is not None and small.numel() == 4096 and small.dtype == torch.uint8
    assert bench._l2_flush_buffer(torch.device("cpu"), 2 * bench.L2_BYTES - 1) is not None
    assert bench._l2_flush_buffer(torch.device("cpu"), 2 * bench.L2_BYTES) is None
    assert bench._l2_flush_buffer(torch.device("cpu"), 763 * 10**6) is None
