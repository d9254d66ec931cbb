"""The replica (N > 1) host path on CPU: two gloo ranks rendezvous on 127.0.0.1,
agree on the slowest rank's time and compute the whole-job throughput."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    from paper_2607_24841_gb300 import replicas
    w, r, lr = replicas.world_info()
    replicas.init(w, backend="gloo")
    replicas.barrier(w)
    ms = 10.0 + 2.5 * r  # rank 1 is the slower replica
    ms_max = replicas.max_over_ranks(w, ms)
    value = replicas.job_throughput(32 * 5, w, ms_max)
    replicas.barrier(w)
    replicas.finish(w)
    q.put((r, w, lr, ms_max, value))


def test_two_gloo_ranks_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs)
    out = sorted(q.get(timeout=5) for _ in range(2))
    for r, (rank, world, local, ms_max, value) in enumerate(out):
        assert (rank, world, local) == (r, 2, r)
        assert ms_max == pytest.approx(12.5)
        # 2 replicas x 5 steps x 32 tokens in the slowest replica's 12.5 ms
        assert value == pytest.approx(2 * 5 * 32 / 0.0125)


def test_single_process_defaults():
    from paper_2607_24841_gb300 import replicas
    env = {k: os.environ.pop(k) for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK") if k in os.environ}
    try:
        assert replicas.world_info() == (1, 0, 0)
        replicas.init(1)
        replicas.barrier(1)
        assert replicas.max_over_ranks(1, 3.5) == 3.5
        assert replicas.job_throughput(160, 1, 100.0) == pytest.approx(1600.0)
    finally:
        os.environ.update(env)
