"""Host-side pieces of bench.py: the replica aggregation over ranks (gloo, 2 ranks on
CPU), the workload bookkeeping, and the oracle arm's bounded sample."""
import os
import socket
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    t = bench.reduce_max(10.0 + 5 * rank, torch.device("cpu"), True)
    q.put((rank, t))
    torch.distributed.destroy_process_group()


def test_reduce_max_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    assert got == [(0, 15.0), (1, 15.0)]


def test_workload_algorithmic_work_matches_sizes():
    """The long sweep: 64 problems, 301.8 GFLOP of attention (4 * heads * d * sum Nq*Nk)."""
    from oracle import ssm_oracle as O
    from paper_2608_23167_gb300 import workloads as W
    w = W.WORKLOADS["long"]
    total = 0
    for b in w.block_indices:
        r, *_ = O.select_suffix(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail)
        nq = w.block + len(r)
        total += nq * (nq + w.prompt + b * w.block)
    assert abs(4 * w.h_q * w.head_dim * total / 1e9 - 301.777) < 0.01


def test_oracle_sample_is_bounded():
    import time
    import bench
    from paper_2608_23167_gb300 import workloads as W
    t0 = time.perf_counter()
    rate, done, t_used, used = bench.oracle_sample(W.WORKLOADS["tiny"], 0.5)
    assert done >= 1 and rate > 0 and time.perf_counter() - t0 < 60
