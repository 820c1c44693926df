"""The benchmark's host-side contract, without a GPU: the committed ncu traffic figure is used only
for the kernel sources it was taken on, the reference arm (the oracle timed on the host cores)
prints the contract's JSON line for the same metric, and the GPU arm fails loudly instead of
falling back to the CPU."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _last_json(stdout: str) -> dict:
    lines = [ln for ln in stdout.splitlines() if ln.startswith("{")]
    assert lines, stdout[-2000:]
    return json.loads(lines[-1])


def test_traffic_figure_is_tied_to_the_kernel_sources(monkeypatch):
    traffic, src = bench.gemm_traffic(4)
    assert traffic is not None, src
    assert src == os.path.join("profiles", "dequant_gemm_gemma4b_step_traffic.md")
    # DRAM bytes of a fused-GEMM launch are at least its algorithmic bytes (each operand once)
    with open(os.path.join(ROOT, src)) as f:
        kv = dict(ln.split(": ", 1) for ln in f.read().splitlines() if ": " in ln and ln[:1].isalpha())
    assert traffic >= float(kv["algorithmic_bytes_per_launch"])
    # another workload, or any change to the kernel sources, and the figure is withheld
    assert bench.gemm_traffic(1)[0] is None
    monkeypatch.setattr(bench, "gemm_sources_sha", lambda: "0" * 64)
    t2, why = bench.gemm_traffic(4)
    assert t2 is None and "changed" in why


def test_reference_arm_prints_the_contract_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "1", "--steps", "1",
                        "--warmup", "3"], cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    d = _last_json(r.stdout)
    assert d["impl"] == "reference"
    assert d["metric"] == bench.METRIC and d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["value"] > 0 and d["steps"] == 1 and d["warmup"] >= 3
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert "qwen2.5-0.5b" in d["config"]["workload"]


def test_gpu_arm_fails_loudly_without_cuda():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present: the GPU arm is exercised by the GPU runs")
    r = subprocess.run([sys.executable, "bench.py", "--steps", "1", "--warmup", "3"], cwd=ROOT,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode != 0
    assert not any(ln.startswith("{") and '"value"' in ln for ln in r.stdout.splitlines())


def _rank_worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each rank's own time; the job's is the slowest rank's, on every rank
        t = bench.max_over_ranks(1.5 + rank, dist)
        out[rank] = (t, bench.job_tokens_per_s(16384, 20, world, t))
    finally:
        dist.destroy_process_group()


def test_two_ranks_report_the_slowest_rank_and_the_whole_job():
    """The N > 1 path's host logic over two gloo ranks: every rank gets the maximum time, and the
    value counts the tokens of both ranks over it (weak scaling: fixed work per rank)."""
    import socket

    import torch.multiprocessing as mp
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    out = mp.Manager().dict()
    mp.spawn(_rank_worker, args=(2, port, out), nprocs=2, join=True)
    assert dict(out) == {0: (2.5, 2 * 16384 * 20 / 2.5), 1: (2.5, 2 * 16384 * 20 / 2.5)}
    assert bench.max_over_ranks(3.0, None) == 3.0


def test_reference_arm_on_a_second_rank_exits_without_work():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "1", "--steps", "1",
                        "--warmup", "3"], cwd=ROOT, capture_output=True, text=True, timeout=120, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""
