"""World-size-2 gloo run of the multi-GPU host logic on CPU: per-rank seeds,
token shards that cover every unit exactly once, sharded reduction equal to
the unsharded one (no cross-rank dependency), and the max-over-ranks timing."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

import oracle as O
from paper_2606_26744_gb300 import dist
from paper_2606_26744_gb300 import workloads as W


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    try:
        n, m, d = 37, 4, 64
        inp = W.make_reduce_inputs(n, m, d, "f32", 0.1, seed=5)
        lo, hi = dist.shard(n, rank, world)
        H = inp["H"].double().numpy()[lo:hi]
        y, _ = O.gated_reduce(H, inp["Wf"].double().numpy(), inp["b"].double().numpy(), out_dtype="f64")
        # gather the shards on every rank
        parts = [None] * world
        torch.distributed.all_gather_object(parts, (lo, hi, y))
        t = dist.max_over_ranks([1.0 + rank, 10.0 - rank])
        q.put((rank, parts, t, dist.rank_seed(1000, rank)))
    finally:
        torch.distributed.destroy_process_group()


def test_two_rank_sharding_and_timing_reduction():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    out.sort()
    parts = out[0][1]
    covered = sorted((lo, hi) for lo, hi, _ in parts)
    assert covered[0][0] == 0 and covered[-1][1] == 37
    assert all(covered[i][1] == covered[i + 1][0] for i in range(len(covered) - 1))
    inp = W.make_reduce_inputs(37, 4, 64, "f32", 0.1, seed=5)
    full, _ = O.gated_reduce(inp["H"].double().numpy(), inp["Wf"].double().numpy(), inp["b"].double().numpy(),
                             out_dtype="f64")
    stitched = np.concatenate([y for _, _, y in sorted(parts, key=lambda x: x[0])], axis=0)
    assert np.array_equal(stitched, full)
    for rank, _, t, seed in out:
        assert t == [2.0, 10.0]
    assert out[0][3] != out[1][3]


def test_shard_edges():
    assert dist.shard(0, 0, 3) == (0, 0)
    spans = [dist.shard(10, r, 4) for r in range(4)]
    assert spans[0][0] == 0 and spans[-1][1] == 10
    assert max(h - l for l, h in spans) - min(h - l for l, h in spans) <= 1
    with pytest.raises(ValueError):
        dist.shard(5, 3, 3)
    assert dist.max_over_ranks([3.5]) == [3.5]


def _bench_worker(rank, world, port, q):
    """The bench's replica bookkeeping on one rank: its own seed and
    synthetic draft inputs, its step time reduced to the maximum over ranks,
    and the whole-job rate computed from it (the calls bench.py makes)."""
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    try:
        cfg = W.CONFIGS["tiny"]
        seed = dist.rank_seed(1000, rank)
        inp = W.make_draft_inputs(cfg, seed, device="cpu")
        ms_here = 2.0 + rank  # this rank's step time
        ms, e2e = dist.max_over_ranks([ms_here, 10.0 * (world - rank)])
        rate = dist.whole_job_rate(cfg.batch, world, ms)
        q.put((rank, float(inp["H"].double().sum()), ms, e2e, rate))
    finally:
        torch.distributed.destroy_process_group()


def test_two_rank_bench_bookkeeping():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_bench_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # distinct synthetic inputs per rank; every rank sees the slowest rank's times
    assert out[0][1] != out[1][1]
    for _, _, ms, e2e, rate in out:
        assert ms == 3.0 and e2e == 20.0
        # whole job: both ranks' blocks over the slowest rank's step
        assert rate == W.CONFIGS["tiny"].batch * world / (3.0 / 1e3)
    with pytest.raises(ValueError):
        dist.whole_job_rate(1, 0, 1.0)
