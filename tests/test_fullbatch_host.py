"""The whole-batch checker itself, on the CPU (no GPU).

A verify step is assembled on the host and its output buffers are filled
with the oracle's own results (attention rounded to bf16, scores, decisions
and the loss), as a correct kernel would leave them.  The pooled checker must
accept that, and must reject each of a few planted mistakes: one attention
element moved by a few ulp, one flipped decision, a loss off by 1e-3.
"""
import numpy as np
import pytest
import torch

import ipd_synth as S
import oracle as O
from tests import parity
from tests.fullbatch import OraclePool, check_step_full


def _oracle_filled_step():
    from paper_2609_36546_gb300 import VerifyStep
    spec = S.small_spec(n_req=5, ctx=(20, 200), span=(1, 6), vocab=512, force="mixed")
    w = S.make_workload(spec, seed=11, device="cpu")
    step = VerifyStep.from_workload(w, device="cpu")
    for name, b, idx, cache in step.batches:
        q, cu_q, seq, ptab, out = b._keep
        c = step.cache_t if cache == "teacher" else step.cache_s
        for j in range(len(idx)):
            L = int(seq[j])
            npg = (L + 15) // 16
            pages = ptab[j, :npg].to(torch.int64)
            ref = O.paged_span_attention(parity.u16(q[int(cu_q[j]):int(cu_q[j + 1])]),
                                         parity.u16(c.k_pages.index_select(0, pages)),
                                         parity.u16(c.v_pages.index_select(0, pages)),
                                         np.arange(npg), L, step.scale)
            bits = O.f64_to_bf16(ref).view(np.int16)
            out[int(cu_q[j]):int(cu_q[j + 1])] = torch.from_numpy(bits.copy()).view(torch.bfloat16)
    orc = parity.oracle_scores(step, range(step.R))
    for r, (t0, t1, o) in orc.items():
        for k in ("logp_s", "logp_t", "feedback", "kl_rev", "kl_fwd", "margin"):
            step.score[k][t0:t1] = torch.from_numpy(np.asarray(o[k], np.float32))
        for k in ("covered", "source"):
            step.score[k][t0:t1] = torch.from_numpy(np.asarray(o[k]).astype(np.uint8))
        for k in ("first_trans", "n_emit", "new_len"):
            step.score[k][r] = int(o[k][0])
        for k in ("next_driver", "done"):
            step.score[k][r] = int(o[k][0])
    T = step.T
    rev, fwd, src = np.zeros(T), np.zeros(T), np.zeros(T, np.int64)
    n_emit = np.zeros(step.R, np.int64)
    for r, (t0, t1, o) in orc.items():
        rev[t0:t1], fwd[t0:t1], src[t0:t1] = o["kl_rev"], o["kl_fwd"], o["source"]
        n_emit[r] = o["n_emit"][0]
    loss = O.split_loss(rev, fwd, src, step.cu_span.numpy(), n_emit)
    step.out8.copy_(torch.tensor([loss[k] for k in O.LOSS_FIELDS], dtype=torch.float32))
    return step


@pytest.fixture(scope="module")
def pool():
    with OraclePool(cores=2) as p:
        yield p


def test_checker_accepts_oracle_results(pool):
    rep = check_step_full(_oracle_filled_step(), pool=pool)
    assert rep["ok"], rep
    assert rep["attn_max_ulp"] == 0.0 and rep["decision_mismatch"] == 0


def test_checker_rejects_planted_mistakes(pool):
    step = _oracle_filled_step()
    out = step.batches[0][1]._keep[4]
    v = out.view(torch.int16)
    v[0, 0, 5] += 4                      # four bf16 ulp on one element
    rep = check_step_full(step, pool=pool)
    assert not rep["attn_ok"] and rep["score_ok"] and rep["loss_ok"]

    step = _oracle_filled_step()
    r = int(step.idx_s[0])
    step.score["n_emit"][r] += 1         # one wrong decision
    rep = check_step_full(step, pool=pool)
    assert rep["attn_ok"] and not rep["score_ok"]

    step = _oracle_filled_step()
    step.out8[0] *= 1.001                # the loss 1e-3 off
    rep = check_step_full(step, pool=pool)
    assert rep["score_ok"] and not rep["loss_ok"]


def test_needed_positions_checker():
    """check_scores(needed=True) ignores the values a needed-rows pass leaves
    undefined (NaN past each transition) and still catches a wrong value at
    an emitted position or a wrong coverage up to the transition."""
    step = _oracle_filled_step()
    orc = parity.oracle_scores(step, range(step.R))
    src = step.score["source"].numpy()
    cu = step.cu_span.numpy()
    ft = step.score["first_trans"].numpy()
    em = np.zeros(step.T, bool)
    dec = np.zeros(step.T, bool)
    for r in range(step.R):
        e, d = parity.needed_positions(src, ft, cu, r)
        em[cu[r]:cu[r + 1]], dec[cu[r]:cu[r + 1]] = e, d
    assert (~dec).any() and (~em).any()  # the case has positions past transitions
    for k in ("logp_s", "logp_t", "feedback", "kl_rev", "kl_fwd"):
        step.score[k][torch.from_numpy(~em)] = float("nan")
    step.score["margin"][torch.from_numpy(~dec)] = float("nan")
    step.score["covered"][torch.from_numpy(~dec)] = 0
    st, _ = parity.check_scores(step, None, orc=orc, needed=True)
    assert st["score_ok"], st
    st, _ = parity.check_scores(step, None, orc=orc)  # the full comparison sees the NaNs
    assert not st["score_ok"]
    t = int(np.flatnonzero(em)[0])
    step.score["kl_rev"][t] += 1e-2
    st, _ = parity.check_scores(step, None, orc=orc, needed=True)
    assert not st["score_ok"] and st["max_kl_err"] > 1e-3
