"""Multi-rank host logic of bench.py on CPU: two gloo ranks (world size 2).

The memory step runs as independent replicas, one per GPU; the only collective
is the max-over-ranks of the timings.  These tests run that reduction, the
whole-job rate and the reference arm's rank handling with the gloo backend."""
import json
import os
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, port, q):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    local_ms = [3.0, 7.5][rank]
    m = bench.max_over_ranks(local_ms, torch.device("cpu"))
    rate = bench.whole_job_rate(4680, m, world)
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, m, rate))


def _free_port():
    import socket
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def test_max_over_ranks_and_rate_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [7.5, 7.5]  # both ranks see the slowest rank's time
    assert all(abs(r[2] - 2 * 4680 / 7.5e-3) < 1e-6 for r in res)


def test_single_process_reduction_is_identity():
    import torch
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(1.25, torch.device("cpu")) == 1.25
    assert bench.whole_job_rate(4680, 1.0, 1) == 4680e3


@pytest.mark.slow
def test_reference_arm_two_ranks_rank0_prints_once():
    """torchrun-style launch of the reference arm with two gloo-free ranks: rank 0 alone
    runs the oracle sample and prints one JSON line; rank 1 exits 0 without work."""
    outs = []
    for rank in (0, 1):
        env = dict(os.environ, WORLD_SIZE="2", RANK=str(rank), LOCAL_RANK=str(rank))
        r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                            "--warmup", "3", "--ref-queries", "2"], env=env, capture_output=True, text=True,
                           timeout=900)
        assert r.returncode == 0, r.stderr[-2000:]
        outs.append(r.stdout.strip())
    assert outs[1] == ""
    line = json.loads(outs[0].splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"
    sys.path.insert(0, ROOT)
    import bench
    assert line["config"] == bench.main_config(2)  # the same config object as the GPU arm's line
    assert line["ms_per_step"] <= line["ms_per_step_extrapolated"]  # measured sample vs full-step estimate
