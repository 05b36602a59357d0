"""Host logic of bench.py's N>1 path on CPU: two gloo ranks (replicas).

Each rank reports its own timed region and units; the whole-job value is the
sum of units over the slowest rank's time, and only rank 0 runs the
reference arm."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    ws, r, _ = bench.dist_env()
    dist = bench.init_dist(ws)
    bench.barrier(dist)
    local_ms = 100.0 * (rank + 1)      # rank 1 is the slow one
    units = 1000 * (rank + 1)
    t, value = bench.aggregate(dist, local_ms, units)
    out.put((rank, t, value))
    dist.destroy_process_group()


def test_two_rank_aggregate():
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
    for rank, t, value in res:
        assert t == pytest.approx(200.0)                  # max over ranks
        assert value == pytest.approx(3000 / 0.2)         # all units / slowest time


def test_reference_arm_nonzero_rank_does_no_work(monkeypatch):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")

    class A:
        steps, warmup, gpus = 1, 3, 2
    assert bench.run_reference(A()) == 0


def test_flop_model_matches_hand_counts():
    import bench
    f = bench.flops_per_token_head(128, 64)
    assert round(f["fwd"]) == 259413
    assert round(f["step"]) == 778240
    assert bench.decode_bytes_per_head(128) == 263180
