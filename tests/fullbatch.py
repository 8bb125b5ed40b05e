"""Whole-batch comparison of a full-size verify step with the oracle (test
infrastructure).

The oracle's work is spread over a pool of host processes started with
`spawn` (the parent has already used the GPU): one task per request for the
vocabulary pass and verdict, one task per (request, attention sub-batch) for
the attention.  Payloads are produced lazily and at most `window` tasks are in
flight, so the host holds only a few requests' pages at a time.  The workers
import only numpy, the oracle and the tolerance module.
"""
from __future__ import annotations

import collections
import multiprocessing as mp
import os

import numpy as np

import oracle as O
from tests.attn_tol import attn_case_errors


def _score_job(a):
    r, t0, t1, ls, lt, toks, drv, pre, K, eos = a
    sub = O.score_span(ls, lt, toks, np.array([0, t1 - t0]), np.array([drv]), np.array([pre]),
                       K, eos)
    return r, (t0, t1, sub)


def _attn_job(a):
    return attn_case_errors(*a)


class OraclePool:
    """A spawn pool of one single-threaded process per host core (BLAS threads
    pinned to 1 in the workers)."""

    def __init__(self, cores: int | None = None):
        self.cores = max(1, min(cores or os.cpu_count() or 1, 32))

    def __enter__(self):
        self._env = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS",
                                                    "MKL_NUM_THREADS")}
        for k in self._env:
            os.environ[k] = "1"
        self.pool = mp.get_context("spawn").Pool(self.cores)
        return self

    def __exit__(self, *exc):
        self.pool.close()
        self.pool.join()
        for k, v in self._env.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v

    def imap_bounded(self, fn, payloads, window: int | None = None):
        """Results of fn over payloads, in order, with at most `window` tasks
        (and their payloads) alive at once."""
        window = window or 2 * self.cores
        pending = collections.deque()
        for p in payloads:
            pending.append(self.pool.apply_async(fn, (p,)))
            while len(pending) >= window:
                yield pending.popleft().get()
        while pending:
            yield pending.popleft().get()


def _score_payloads(step, reqs):
    from tests.parity import u16
    cu = step.cu_span.cpu().numpy()
    drv = step.driver.cpu().numpy()
    pre = step.prefix_len.cpu().numpy()
    toks = step.tokens.cpu().numpy()
    for r in reqs:
        t0, t1 = int(cu[r]), int(cu[r + 1])
        if t1 > t0:
            ls, lt = u16(step.logits_s[t0:t1]), u16(step.logits_t[t0:t1])
        else:
            ls = lt = np.zeros((0, step.V), np.uint16)
        yield (int(r), t0, t1, ls, lt, toks[t0:t1], int(drv[r]), int(pre[r]), step.K, step.eos_id)


def _attn_payloads(step, requests):
    """(q, K pages, V pages, L, scale, kernel output) per request of every
    attention sub-batch (all requests, or those in `requests`)."""
    import torch
    from tests.parity import u16
    sel = None if requests is None else set(int(r) for r in requests)
    for name, b, idx, cache in step.batches:
        q, cu_q, seq, ptab, out = b._keep
        cu = cu_q.cpu().numpy()
        seqh = seq.cpu().numpy()
        pth = ptab.cpu().numpy()
        c = step.cache_t if cache == "teacher" else step.cache_s
        for j in range(len(idx)):
            if sel is not None and int(idx[j]) not in sel:
                continue
            L = int(seqh[j])
            pages = torch.from_numpy(pth[j, :(L + 15) // 16].astype(np.int64)).to(c.k_pages.device)
            yield (u16(q[cu[j]:cu[j + 1]]), u16(c.k_pages.index_select(0, pages)),
                   u16(c.v_pages.index_select(0, pages)), L, step.scale, u16(out[cu[j]:cu[j + 1]]))


def check_step_full(step, attn_requests=None, pool: OraclePool | None = None):
    """Every request's scores and decisions, the whole batch's loss, and the
    attention of every request (or of `attn_requests`), against the oracle."""
    from tests import parity
    own = pool is None
    pool = pool or OraclePool()
    if own:
        pool.__enter__()
    try:
        orc = dict(pool.imap_bounded(_score_job, _score_payloads(step, range(step.R))))
        rep = {}
        stats = parity.new_attn_stats()
        n_ok = n_all = 0
        for e in pool.imap_bounded(_attn_job, _attn_payloads(step, attn_requests)):
            n_ok, n_all = parity.add_attn_case(stats, e, n_ok, n_all)
        rep.update(parity.finish_attn_stats(stats, n_ok, n_all))
    finally:
        if own:
            pool.__exit__(None, None, None)
    s, _ = parity.check_scores(step, None, orc=orc)
    rep.update(s)
    rep.update(parity.check_loss(step, orc))
    rep["loss_checked"] = True
    rep["attn_requests"] = "all" if attn_requests is None else len(attn_requests)
    rep["ok"] = bool(rep["attn_ok"] and rep["score_ok"] and rep["loss_ok"])
    return rep
