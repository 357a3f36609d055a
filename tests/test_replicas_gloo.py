"""The multi-GPU path is replicas only (independent sequences per rank, no
data-path collective): two gloo ranks on the CPU run bench.py's rank setup,
barrier and max-over-ranks reduction, and get same-shaped workloads on
different seeds."""

import os
import socket

import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        r, w, local = bench.dist_env()
        bench.barrier(w)
        slowest = bench.max_over_ranks(10.0 + r, w)
        wl = bench.rank_workload(2, 0, r)
        import workloads as W
        k, _ = W.layer_kv(W.config(1, seed=wl.seed), 0, seq_range=(0, 1))
        out.put((r, w, local, slowest, wl.seed, wl.kv_tokens, wl.name, float(k[1, 0, :8].abs().sum())))
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, w0, l0, m0, s0, t0, n0, x0), (r1, w1, l1, m1, s1, t1, n1, x1) = res
    assert (r0, r1, w0, w1, l0, l1) == (0, 1, 2, 2, 0, 1)
    assert m0 == m1 == 11.0                      # the slowest rank's time, seen by both
    assert s0 != s1 and n0 == n1 and t0 == t1    # same shape, own data
    assert x0 != x1
