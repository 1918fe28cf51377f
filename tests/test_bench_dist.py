"""The bench's multi-rank path on the host: world size 2 over gloo on CPU, with
the rendezvous on 127.0.0.1 (replicas only: the ranks share nothing but the
timing reduction; no GPU)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench

    dist, r, ws, local = bench._dist()
    assert (r, ws, local) == (rank, world, rank) and dist.get_backend() == "gloo"
    ms = bench._max_over_ranks(dist, 1.0 + rank, "cpu")  # rank 1 is the slower
    rate = bench._job_rate(1e9, ws, ms)
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump({"ms": ms, "rate": rate}, f)
    dist.destroy_process_group()


def test_timing_is_the_slowest_rank_and_value_the_whole_job(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, start_method="spawn")
    got = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    for g in got:
        assert g["ms"] == 2.0  # every rank sees the max
        assert g["rate"] == pytest.approx(1e9 * world / 2e-3)


def test_single_process_needs_no_process_group(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench

    monkeypatch.delenv("WORLD_SIZE", raising=False)
    assert bench._dist() == (None, 0, 1, 0)
    assert bench._max_over_ranks(None, 3.5, "cpu") == 3.5
    assert bench._job_rate(2e9, 1, 1.0) == pytest.approx(2e12)


def test_a_failing_section_reports_its_error_and_the_run_goes_on():
    """bench.py's sections after the headline (GEMM, configs, Q4X) each return
    their figures or an {"error": ...} of their own; the allocator's cache is
    released after each either way."""
    sys.path.insert(0, ROOT)
    import bench

    released = []

    class _Cuda:
        @staticmethod
        def empty_cache():
            released.append(1)

    class _Torch:
        cuda = _Cuda

    def boom(n):
        raise RuntimeError("device error " * n)

    assert bench._section(_Torch, lambda a, b: {"v": a + b}, 2, 3) == {"v": 5}
    out = bench._section(_Torch, boom, 100)
    assert out["error"].startswith("RuntimeError: device error") and len(out["error"]) == 300
    assert released == [1, 1]


def test_reference_arm_under_torchrun_prints_once_from_rank_0():
    """`bench.py --impl reference` launched as the driver launches N = 2: rank 0
    alone runs the oracle and prints one JSON line; rank 1 exits 0 without work."""
    env = dict(os.environ, QX_REF_BUDGET_S="3", OPENBLAS_NUM_THREADS="1")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "3", "--warmup", "3"]
    r = subprocess.run(cmd, capture_output=True, text=True, cwd=ROOT, env=env, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["steps"] == 3
    assert line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"] == {"value": line["value"], "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
