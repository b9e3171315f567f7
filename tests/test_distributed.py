"""Batch sharding across ranks (gloo, world size 2, CPU).

Each rank takes a contiguous slice of the sequences with seq_offset = its
first global index and runs the round on it alone; gathering the slices must
reproduce the unsharded round exactly (the oracle stands in for the device
path here). The benchmark's max-over-ranks timing is checked too.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2608_08721_gb300 import dist as pdist
from paper_2608_08721_gb300 import workloads


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _make_batch():
    w = workloads.WORKLOADS["ragged"].scaled(B=10, K=6, V=256)
    inp = workloads.logits(w)
    return w, {k: v.numpy() for k, v in inp.items()}


def _round(orc, w, inp, lo, hi):
    sl = {k: v[lo:hi] for k, v in inp.items()}
    q, _ = orc.confidence(sl["draft_logits"], sl["draft_tokens"], sl["temperature"])
    cost = (1.0 + 0.05 * np.arange(w.K + 1)).astype(np.float64)
    L, _ = orc.select_lengths(q, cost)
    n, bonus, _ = orc.accept(sl["target_logits"], sl["draft_logits"], sl["draft_tokens"], L, sl["temperature"],
                             seed=w.philox_seed, round_offset=2, seq_offset=lo)
    return np.stack([L, n, bonus]).astype(np.int64)


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    try:
        import oracle

        oracle.build()
        pdist.init("gloo")
        w, inp = _make_batch()
        lo, hi = pdist.shard_range(w.B, rank, world)
        mine = torch.from_numpy(_round(oracle, w, inp, lo, hi))
        sizes = [pdist.shard_range(w.B, r, world) for r in range(world)]
        parts = [torch.zeros((3, h - l), dtype=torch.int64) for l, h in sizes]
        dist.all_gather(parts, mine)
        t = pdist.max_over_ranks(1.0 + rank)
        n = pdist.sum_over_ranks(hi - lo)
        pdist.barrier()
        if rank == 0:
            q.put(("ok", torch.cat(parts, 1).numpy(), t, n))
        dist.destroy_process_group()
    except Exception as e:  # report to the parent instead of hanging it
        q.put(("err", repr(e), None, None))


def test_shard_range_partitions():
    for total in (0, 1, 7, 64):
        for world in (1, 2, 3, 8):
            rs = [pdist.shard_range(total, r, world) for r in range(world)]
            assert rs[0][0] == 0 and rs[-1][1] == total
            assert all(a[1] == b[0] for a, b in zip(rs, rs[1:]))
            sizes = [h - l for l, h in rs]
            assert max(sizes) - min(sizes) <= 1


def test_two_rank_sharded_round_equals_unsharded(orc):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    status, got, tmax, n = q.get(timeout=240)
    for p in procs:
        p.join(timeout=60)
    assert status == "ok", got
    w, inp = _make_batch()
    ref = _round(orc, w, inp, 0, w.B)
    np.testing.assert_array_equal(got, ref)
    assert tmax == 2.0 and n == w.B
