"""Rule variants and vocabulary-pass by-products on the GPU vs the fp64
oracle (needs a GB300).

Tolerances: entropies within 1e-3 + 1e-4 |ref| nats (fp32 sums of
exp(l - m) and exp(l - m) l over the vocabulary, like log Z); the top-K
overlap ratio exact (it counts the same exact top-K sets as coverage);
the full-vocabulary KL within 1e-4 + 1e-3 |ref| (fp32 difference of
expectations and log-partitions of size <= ~40); decisions exact except
in requests where some position lies within 1e-3 of its rule's threshold
(counted, and required to be rare).
"""
import numpy as np
import pytest
import torch

import ipd_synth as S
import oracle as O
from tests.parity import u16

pytestmark = pytest.mark.gpu

H_ATOL, H_RTOL = 1e-3, 1e-4
FKL_ATOL, FKL_RTOL = 1e-4, 1e-3


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import ipd
    return ipd


def _step(spec, seed):
    from paper_2609_36546_gb300 import VerifyStep
    w = S.make_workload(spec, seed=seed, device="cpu")
    return w, VerifyStep.from_workload(w, device="cuda")


def _run_ext(ipd, st, take, hand, ttau, htau):
    T = st.T
    ent_s = torch.full((T,), float("nan"), device="cuda")
    ent_t = torch.full((T,), float("nan"), device="cuda")
    ovl = torch.full((T,), float("nan"), device="cuda")
    ipd.score_span_ex(st.logits_s, st.logits_t, st.tokens, st.cu_span, st.driver, st.prefix_len,
                      st.K, st.eos_id, st.score, st.ws_score, take, hand, ttau, htau, ent_s,
                      ent_t, ovl)
    torch.cuda.synchronize()
    g = {k: v.cpu().numpy() for k, v in st.score.items()}
    g["entropy_s"], g["entropy_t"], g["topk_overlap"] = (ent_s.cpu().numpy(), ent_t.cpu().numpy(),
                                                         ovl.cpu().numpy())
    return g


def _oracle(st, take, hand, ttau, htau):
    return O.score_span(u16(st.logits_s), u16(st.logits_t), st.tokens.cpu().numpy(),
                        st.cu_span.cpu().numpy(), st.driver.cpu().numpy(),
                        st.prefix_len.cpu().numpy(), st.K, st.eos_id, takeover_rule=take,
                        handback_rule=hand, takeover_tau=ttau, handback_tau=htau)


RULES = [("default", 0, 0, None, None), ("entropy-S-take/entropy-T-hand", 1, 2, "s", "t"),
         ("entropy-T-take/entropy-S-hand", 2, 1, "t", "s"), ("SKD", 0, 3, None, None),
         ("always-take/never-hand", 3, 4, None, None)]


@pytest.mark.parametrize("name,take,hand,tsrc,hsrc", RULES, ids=[r[0] for r in RULES])
def test_rules_and_byproducts_match_oracle(lib, name, take, hand, tsrc, hsrc):
    spec = S.small_spec(n_req=10, ctx=(20, 600), span=(1, 12), vocab=4096, sigma=2.5)
    w, st = _step(spec, 41)
    ls, lt = u16(st.logits_s), u16(st.logits_t)
    hs = np.array([O.entropy(O.bf16_to_f64(r)) for r in ls])
    ht = np.array([O.entropy(O.bf16_to_f64(r)) for r in lt])
    pick = {"s": hs, "t": ht, None: np.array([0.0])}
    ttau = float(np.median(pick[tsrc])) if tsrc else 0.0
    htau = float(np.median(pick[hsrc])) if hsrc else 0.0
    g = _run_ext(lib, st, take, hand, ttau, htau)
    o = _oracle(st, take, hand, ttau, htau)
    # by-products
    assert np.all(np.abs(g["entropy_s"] - o["entropy_s"]) <= H_ATOL + H_RTOL * np.abs(o["entropy_s"]))
    assert np.all(np.abs(g["entropy_t"] - o["entropy_t"]) <= H_ATOL + H_RTOL * np.abs(o["entropy_t"]))
    assert np.array_equal(g["topk_overlap"], o["topk_overlap"].astype(np.float32))
    # decisions, request by request (requests with a near-threshold position are counted)
    cu = st.cu_span.cpu().numpy()
    near_reqs = 0
    for r in range(st.R):
        sl = slice(cu[r], cu[r + 1])
        if np.any(np.abs(o["margin"][sl]) <= 1e-3):
            near_reqs += 1
            continue
        assert np.array_equal(g["covered"][sl].astype(np.int64), o["covered"][sl]), r
        assert np.array_equal(g["source"][sl].astype(np.int64), o["source"][sl]), r
        for f in ("first_trans", "n_emit", "next_driver", "new_len", "done"):
            assert int(g[f][r]) == int(o[f][r]), (r, f)
    assert near_reqs <= st.R // 5
    # the margin is the rule's signed distance from its threshold
    fin = np.isfinite(o["margin"])
    if take in (1, 2) or hand in (1, 2):
        tol = H_ATOL + H_RTOL * np.abs(o["margin"][fin]) + 1e-3
        assert np.all(np.abs(g["margin"][fin] - o["margin"][fin]) <= tol)
    assert np.array_equal(np.isposinf(g["margin"]), np.isposinf(o["margin"]))
    assert np.array_equal(np.isneginf(g["margin"]), np.isneginf(o["margin"]))


def test_default_ext_equals_plain_score_span(lib):
    spec = S.small_spec(n_req=6, ctx=(30, 500), span=(1, 9))
    w, st = _step(spec, 43)
    st.run_score()
    torch.cuda.synchronize()
    plain = {k: v.clone() for k, v in st.score.items()}
    g = _run_ext(lib, st, 0, 0, 0.0, 0.0)
    for k, v in plain.items():
        assert np.array_equal(v.cpu().numpy().view(np.uint8), g[k].view(np.uint8)), k


# positions split over clusters of 4 and 2 CTAs, and one CTA per position
@pytest.mark.parametrize("V,T", [(151936, 4), (151936, 200), (4096, 9), (4096, 700)])
def test_full_kl_matches_oracle(lib, V, T):
    g = torch.Generator().manual_seed(V + T)
    a = (torch.randn(T, V, generator=g) * 2.5).to(torch.bfloat16)
    b = (a.float() + torch.randn(T, V, generator=g)).to(torch.bfloat16)
    b[0] = a[0]  # equal rows: both KLs exactly 0
    rev = torch.empty(T, device="cuda"); fwd = torch.empty(T, device="cuda")
    lib.full_kl(a.cuda(), b.cuda(), rev, fwd)
    torch.cuda.synchronize()
    for t in range(T):
        r_ref, f_ref = O.full_kl(O.bf16_to_f64(u16(a[t])), O.bf16_to_f64(u16(b[t])))
        assert abs(rev[t].item() - r_ref) <= FKL_ATOL + FKL_RTOL * abs(r_ref), (t, rev[t].item(), r_ref)
        assert abs(fwd[t].item() - f_ref) <= FKL_ATOL + FKL_RTOL * abs(f_ref), (t, fwd[t].item(), f_ref)
    assert rev[0].item() == 0.0 and fwd[0].item() == 0.0
