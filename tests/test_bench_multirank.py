"""The benchmark's multi-rank logic on CPU: two gloo ranks agree on the
slowest rank's time, pass the barrier, and only rank 0 of the reference arm
prints its line.  (The GPU arm runs one replica of the workload per rank with
no collective on the data path; what it shares with this test is the timing
and aggregation.)"""

import contextlib
import io
import json
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, _ = bench.dist_env()
        slowest = bench.max_over_ranks(10.0 + 5.0 * rank, w)
        bench.barrier(w)
        out = io.StringIO()
        with contextlib.redirect_stdout(out):
            bench.main(["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "1",
                        "--ref-units", "1"])
        bench.barrier(w)
        q.put((rank, r, w, slowest, out.getvalue()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = {}
    for _ in procs:
        rank, r, w, slowest, text = q.get(timeout=300)
        got[rank] = (r, w, slowest, text)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank in (0, 1):
        r, w, slowest, _ = got[rank]
        assert (r, w) == (rank, 2)
        assert slowest == 15.0                   # the slower rank's time on both
    line = json.loads(got[0][3].strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0
    assert got[1][3].strip() == ""              # rank 1 prints nothing


def test_job_throughput_is_weak_scaling_aggregate():
    import bench
    # 2 ranks x 1000 tokens x 4 steps in 2 s (the slowest rank) -> 4000 tokens/s
    assert bench.job_throughput(2, 1000, 4, 2000.0) == pytest.approx(4000.0)
    assert bench.job_throughput(1, 1000, 4, 2000.0) == pytest.approx(2000.0)
