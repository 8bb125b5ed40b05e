"""GPU-vs-oracle comparison of one verify step (used by the -m gpu tests and
by __graft_entry__.smoke()).

Tolerances (stated once here):
* attention: every output within 2 bf16 ulp of the fp64 oracle rounded to
  bf16, the ulp taken at max(|ref|, ATTN_FLOOR * a), where a = sum_j w_j |v_jd|
  is the softmax-weighted mean magnitude of the values that output averages
  (the oracle's attention over |V|).  An fp32 evaluation of the weighted sum
  has an absolute error of a few fp32 roundings of a, whatever the size of the
  result, so a component that cancels to nearly zero cannot be held to 2 ulp
  of itself.  ATTN_FLOOR = 2^-16 is the smallest power of two under which a
  plain IEEE-fp32 evaluation (tests/attn_fp32_model.py) passes every small
  case (tests/test_attn_tolerance.py).  The strict ulp at |ref| is reported
  beside it, and at least ATTN_STRICT_FRAC of all elements must meet it.
* log-probs within 1e-3 absolute; feedback within 2e-3 (difference of two).
* KL terms within 2e-4 + 1e-4 |ref| (fp32 sums of <= 64 terms of size <= ~40).
* margin: exact (difference of two bf16 values is exact in fp32).
* decisions (covered, source, first_trans, n_emit, next_driver, new_len,
  done): bit-exact; positions with |margin| <= 1e-3 are counted separately.
* split loss: 1e-4 relative (plus 1e-6 absolute for a zero loss).
"""
from __future__ import annotations

import numpy as np
import torch

import oracle as O
from tests.attn_tol import (ATTN_FLOOR, ATTN_STRICT_FRAC, abs_bits,  # noqa: F401
                             attn_case_errors, attn_ulp_errors)

ATOL_LOGP = 1e-3
ATOL_FEEDBACK = 2e-3
KL_ATOL, KL_RTOL = 2e-4, 1e-4
LOSS_RTOL = 1e-4


def u16(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def add_attn_case(stats, e, n_strict_ok, n_all):
    """Fold one request's attn_case_errors() into the running statistics."""
    stats["attn_rows"] += e[4] // 128
    stats["attn_max_ulp"] = max(stats["attn_max_ulp"], e[0])
    stats["attn_max_ulp_strict"] = max(stats["attn_max_ulp_strict"], e[1])
    stats["attn_bad"] += e[2]
    return n_strict_ok + e[3], n_all + e[4]


def finish_attn_stats(stats, n_strict_ok, n_all):
    if n_all:
        stats["attn_frac_strict_le2"] = n_strict_ok / n_all
    stats["attn_ok"] = stats["attn_bad"] == 0 and stats["attn_frac_strict_le2"] >= ATTN_STRICT_FRAC
    return stats


def new_attn_stats():
    return dict(attn_rows=0, attn_max_ulp=0.0, attn_max_ulp_strict=0.0, attn_frac_strict_le2=1.0,
                attn_bad=0)


def check_attention(step, requests=None, max_reqs_per_batch=None, rng=None):
    """Compare every sub-batch's output for the chosen requests."""
    stats = new_attn_stats()
    n_strict_ok = n_all = 0
    for name, b, idx, cache in step.batches:
        q, cu_q, seq, ptab, out = b._keep
        cu = cu_q.cpu().numpy()
        seqh = seq.cpu().numpy()
        pth = ptab.cpu().numpy()
        pool_k, pool_v = (step.cache_t if cache == "teacher" else step.cache_s).k_pages, \
            (step.cache_t if cache == "teacher" else step.cache_s).v_pages
        local = range(len(idx))
        if requests is not None:
            sel = set(int(r) for r in requests)
            local = [j for j in range(len(idx)) if int(idx[j]) in sel]
        if max_reqs_per_batch is not None and len(local) > max_reqs_per_batch:
            local = sorted((rng or np.random.default_rng(0)).choice(list(local), max_reqs_per_batch,
                                                                   replace=False).tolist())
        for j in local:
            L = int(seqh[j])
            npg = (L + 15) // 16
            pages = torch.from_numpy(pth[j, :npg].astype(np.int64)).to(pool_k.device)
            e = attn_case_errors(u16(q[cu[j]:cu[j + 1]]), u16(pool_k.index_select(0, pages)),
                                 u16(pool_v.index_select(0, pages)), L, step.scale,
                                 u16(out[cu[j]:cu[j + 1]]))
            n_strict_ok, n_all = add_attn_case(stats, e, n_strict_ok, n_all)
    return finish_attn_stats(stats, n_strict_ok, n_all)


def oracle_scores(step, requests):
    cu = step.cu_span.cpu().numpy()
    drv = step.driver.cpu().numpy()
    pre = step.prefix_len.cpu().numpy()
    toks = step.tokens.cpu().numpy()
    res = {}
    for r in requests:
        t0, t1 = int(cu[r]), int(cu[r + 1])
        ls = u16(step.logits_s[t0:t1]) if t1 > t0 else np.zeros((0, step.V), np.uint16)
        lt = u16(step.logits_t[t0:t1]) if t1 > t0 else np.zeros((0, step.V), np.uint16)
        sub = O.score_span(ls, lt, toks[t0:t1], np.array([0, t1 - t0]), drv[r:r + 1],
                           pre[r:r + 1], step.K, step.eos_id)
        res[int(r)] = (t0, t1, sub)
    return res


def needed_positions(source, first_trans, cu_span, r):
    """For request r of a step's outputs (numpy): the mask of its emitted
    positions and of the positions up to its first transition (the ones a
    needed-rows pass defines: ipd_score_span_needed)."""
    t0, t1 = int(cu_span[r]), int(cu_span[r + 1])
    emitted = source[t0:t1] != 255
    decided = np.arange(t1 - t0) <= int(first_trans[r])
    return emitted, decided


def check_scores(step, requests=None, orc=None, needed=False):
    """Compare the scores and decisions of the chosen requests (all by
    default) with the oracle's; `orc` may hold the oracle's results already
    (request -> (t0, t1, score_span output)).  needed=True compares the
    per-token values only where a needed-rows pass defines them: log-probs,
    feedback and KL at emitted positions, coverage and margin up to the first
    transition (the decisions everywhere)."""
    R = step.R
    reqs = list(range(R)) if requests is None else [int(r) for r in requests]
    if orc is None:
        orc = oracle_scores(step, reqs)
    g = {k: v.cpu().numpy() for k, v in step.score.items()}
    st = dict(score_positions=0, max_logp_err=0.0, max_fb_err=0.0, max_kl_err=0.0,
              max_margin_err=0.0, decision_mismatch=0, near_threshold=0, near_threshold_mismatch=0,
              coverage_rate=0.0)
    ncov = 0
    for r in reqs:
        t0, t1, o = orc[r]
        sl = slice(t0, t1)
        st["score_positions"] += t1 - t0
        if t1 > t0:
            em = dec = np.ones(t1 - t0, bool)
            if needed:
                em, dec = needed_positions(o["source"], o["first_trans"], np.array([0, t1 - t0]),
                                           0)
            def err_of(name, rel=0.0):
                e = np.abs(g[name][sl] - o[name]) - rel * np.abs(o[name])
                m = dec if name == "margin" else em
                return float(e[m].max()) if m.any() else 0.0
            st["max_logp_err"] = max(st["max_logp_err"], err_of("logp_s"), err_of("logp_t"))
            st["max_fb_err"] = max(st["max_fb_err"], err_of("feedback"))
            for name in ("kl_rev", "kl_fwd"):
                st["max_kl_err"] = max(st["max_kl_err"], err_of(name, KL_RTOL))
            st["max_margin_err"] = max(st["max_margin_err"], err_of("margin"))
            near = (np.abs(o["margin"]) <= 1e-3) & dec
            cov_mis = (g["covered"][sl].astype(np.int64) != o["covered"]) & dec
            src_mis = g["source"][sl].astype(np.int64) != o["source"]
            st["near_threshold"] += int(near.sum())
            st["near_threshold_mismatch"] += int((near & cov_mis).sum())
            st["decision_mismatch"] += int(cov_mis.sum() + src_mis.sum())
            ncov += int(o["covered"].sum())
        for name in ("first_trans", "n_emit", "next_driver", "new_len", "done"):
            if int(g[name][r]) != int(o[name][0]):
                st["decision_mismatch"] += 1
    if st["score_positions"]:
        st["coverage_rate"] = ncov / st["score_positions"]
    st["score_ok"] = (st["max_logp_err"] <= ATOL_LOGP and st["max_fb_err"] <= ATOL_FEEDBACK and
                      st["max_kl_err"] <= KL_ATOL and st["max_margin_err"] <= 1e-6 and
                      st["decision_mismatch"] == 0)
    return st, orc


def check_loss(step, orc):
    """Full-batch loss check (needs the oracle scores of every request)."""
    T = step.T
    rev = np.zeros(T); fwd = np.zeros(T); src = np.zeros(T, np.int64)
    n_emit = np.zeros(step.R, np.int64)
    for r, (t0, t1, o) in orc.items():
        rev[t0:t1] = o["kl_rev"]; fwd[t0:t1] = o["kl_fwd"]; src[t0:t1] = o["source"]
        n_emit[r] = o["n_emit"][0]
    rl = None if step.resp_len is None else step.resp_len.cpu().numpy()
    ref = O.split_loss(rev, fwd, src, step.cu_span.cpu().numpy(), n_emit, rl, step.agg_mode,
                       step.dir_mode)
    got = step.out8.cpu().numpy()
    st = dict(loss_gpu=float(got[0]), loss_ref=ref["loss"], loss_rel_err=0.0)
    ok = True
    for i, name in enumerate(O.LOSS_FIELDS):
        a, b = float(got[i]), float(ref[name])
        if abs(a - b) > LOSS_RTOL * abs(b) + 1e-6:
            ok = False
        if name == "loss":
            st["loss_rel_err"] = abs(a - b) / max(abs(b), 1e-30)
    st["loss_ok"] = ok
    return st


def check_step(step, w=None, requests=None, attn_max_reqs=None, rng=None, needed=False):
    """Full comparison; requests=None checks every request and the loss.

    With a subset of requests the batch loss cannot be recomputed: the report
    then says loss_checked = False and `ok` covers attention and scores only."""
    rep = {}
    rep.update(check_attention(step, requests, attn_max_reqs, rng))
    s, orc = check_scores(step, requests, needed=needed)
    rep.update(s)
    rep["loss_checked"] = requests is None
    if requests is None:
        rep.update(check_loss(step, orc))
    ok = rep["attn_ok"] and rep["score_ok"] and (rep["loss_ok"] if requests is None else True)
    rep["ok"] = bool(ok)
    return rep
