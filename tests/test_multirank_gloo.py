"""The N>1 host path on CPU: two gloo ranks each reduce a shard of a step's
requests and combine_loss reproduces the loss of the whole batch."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle as O


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _step_data(seed=3, R=9):
    rng = np.random.default_rng(seed)
    span = rng.integers(1, 7, size=R)
    cu = np.concatenate([[0], np.cumsum(span)])
    T = int(cu[-1])
    rev, fwd = rng.random(T), rng.random(T)
    n_emit = np.array([rng.integers(0, span[r] + 1) for r in range(R)])
    drv = rng.integers(0, 2, size=R)
    src = np.full(T, 255)
    for r in range(R):
        src[cu[r]:cu[r] + n_emit[r]] = drv[r]
    resp = rng.integers(0, 30, size=R)
    return rev, fwd, src, cu, n_emit, resp


def _worker(rank, world, port, agg, use_resp, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2609_36546_gb300.dist import combine_loss, shard_range
    rev, fwd, src, cu, n_emit, resp = _step_data()
    rs = shard_range(len(n_emit), rank, world)
    lo, hi = cu[rs.start], cu[rs.stop]
    sub = O.split_loss(rev[lo:hi], fwd[lo:hi], src[lo:hi], cu[rs.start:rs.stop + 1] - lo,
                       n_emit[rs.start:rs.stop], resp[rs.start:rs.stop] if use_resp else None,
                       agg_mode=agg)
    out8 = torch.tensor([sub[f] for f in O.LOSS_FIELDS])
    comb = combine_loss(out8)
    if rank == 0:
        q.put(comb.tolist())
    dist.destroy_process_group()


def test_two_rank_loss_combination_matches_whole_batch():
    ctx = mp.get_context("spawn")
    for agg in (0, 1):
        for use_resp in (False, True):
            q = ctx.Queue()
            mp.start_processes(_worker, args=(2, _free_port(), agg, use_resp, q), nprocs=2,
                               join=True, start_method="spawn")
            got = q.get(timeout=60)
            rev, fwd, src, cu, n_emit, resp = _step_data()
            ref = O.split_loss(rev, fwd, src, cu, n_emit, resp if use_resp else None, agg_mode=agg)
            np.testing.assert_allclose(got, [ref[f] for f in O.LOSS_FIELDS], rtol=1e-12, atol=1e-12)


def test_shard_ranges_partition():
    from paper_2609_36546_gb300.dist import shard_range
    for n in (0, 1, 7, 64, 1024):
        for w in (1, 2, 3, 8):
            got = [i for r in range(w) for i in shard_range(n, r, w)]
            assert got == list(range(n))
