"""Pins of the fp64 oracle to things other than itself (CPU only).

Each test fixes an oracle function against a library routine written by
someone else, a closed form, a hand-worked fixture from the paper's rules, a
brute force on tiny inputs, or an invariant the mathematics guarantees.  The
``test_planted_*`` tests plant a plausible mistake in a copy of the oracle's
inputs/outputs and check that the pin notices.
"""
import itertools
import math
import os

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
RNG = np.random.default_rng(1234)


def _bf16_round(x):
    return O.bf16_to_f64(O.f64_to_bf16(x))


# ---------------------------------------------------------------------------
# bf16 conversions against torch's own
# ---------------------------------------------------------------------------
def test_bf16_conversions_match_torch():
    x = np.concatenate([RNG.normal(size=4000) * 10 ** RNG.uniform(-6, 6, size=4000),
                        [0.0, -0.0, 1.0, -2.5, 1.00390625, 1.01171875]])
    ours = O.f64_to_bf16(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    back = O.bf16_to_f64(ref)
    assert np.array_equal(back, torch.from_numpy(ref.view(np.int16)).view(torch.bfloat16)
                          .to(torch.float64).numpy())


def test_bf16_ulp_is_the_spacing_of_neighbouring_bf16_values():
    """bf16_ulp sets every attention tolerance, so it is pinned to the spacing
    of adjacent bf16 numbers for every finite normal bit pattern of either
    sign: value(b + 1) - value(b) in magnitude, both values taken through
    torch's own bf16 -> fp64 conversion.  An exponent off by one anywhere
    would double or halve the spacing and fail here."""
    mags = np.arange(0x0080, 0x7f7f, dtype=np.int32)          # normal, next one still finite
    for sign in (0, 0x8000):
        b = (mags | sign).astype(np.uint16)
        nb = (mags + 1 | sign).astype(np.uint16)
        val = lambda u: torch.from_numpy(u.view(np.int16)).view(torch.bfloat16).to(
            torch.float64).numpy()
        x, xn = val(b), val(nb)
        assert np.all(np.isfinite(xn))
        assert np.array_equal(O.bf16_ulp(x), np.abs(xn - x))
    # between two bf16 values the spacing is that of the binade holding x
    assert O.bf16_ulp(1.5) == 2.0 ** -7 and O.bf16_ulp(1.999) == 2.0 ** -7
    assert O.bf16_ulp(0.75) == 2.0 ** -8 and O.bf16_ulp(-3.0e-3) == 2.0 ** -16
    assert O.bf16_ulp(float(torch.finfo(torch.bfloat16).max)) == 2.0 ** 120
    assert O.bf16_ulp(1.0) == float(torch.finfo(torch.bfloat16).eps)


# ---------------------------------------------------------------------------
# attention
# ---------------------------------------------------------------------------
def _sdpa_reference(q, k, v, scale):
    """torch's scaled_dot_product_attention in fp64 with an explicit span mask."""
    n, Hq, D = q.shape
    L, Hkv, _ = k.shape
    G = Hq // Hkv
    qt = torch.from_numpy(q).permute(1, 0, 2)                         # [Hq, n, D]
    kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(G, 0)  # [Hq, L, D]
    vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(G, 0)
    pos_q = torch.arange(n)[:, None] + (L - n)
    mask = torch.arange(L)[None, :] <= pos_q                          # [n, L]
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask, scale=scale)
    return o.permute(1, 0, 2).numpy()


@pytest.mark.parametrize("n,L,Hq,Hkv", [(1, 1, 4, 2), (1, 37, 8, 4), (4, 40, 32, 4),
                                        (7, 7, 16, 8), (16, 90, 8, 8)])
def test_attention_matches_library_sdpa(n, L, Hq, Hkv):
    q = RNG.normal(size=(n, Hq, 128))
    k = RNG.normal(size=(L, Hkv, 128))
    v = RNG.normal(size=(L, Hkv, 128))
    s = 1 / math.sqrt(128)
    np.testing.assert_allclose(O.span_attention(q, k, v, s), _sdpa_reference(q, k, v, s),
                               rtol=1e-12, atol=1e-12)


def test_attention_single_key_returns_value():
    q = RNG.normal(size=(1, 8, 128))
    k = RNG.normal(size=(1, 2, 128))
    v = RNG.normal(size=(1, 2, 128))
    o = O.span_attention(q, k, v, 0.1)
    for h in range(8):
        np.testing.assert_array_equal(o[0, h], v[0, h // 4])


def test_attention_equal_keys_average_exactly_the_visible_values():
    n, L = 5, 23
    q = RNG.normal(size=(n, 4, 128))
    k = np.repeat(RNG.normal(size=(1, 1, 128)), L, 0).repeat(2, 1)
    v = RNG.normal(size=(L, 2, 128))
    o = O.span_attention(q, k, v, 0.3)
    for i in range(n):
        vis = L - n + i + 1
        for h in range(4):
            np.testing.assert_allclose(o[i, h], v[:vis, h // 2].mean(0), rtol=1e-12, atol=1e-13)


def test_attention_gqa_head_mapping():
    L, Hq, Hkv = 9, 32, 4
    v = np.zeros((L, Hkv, 128))
    for j in range(Hkv):
        v[:, j, :] = j + 1.0
    o = O.span_attention(RNG.normal(size=(2, Hq, 128)), RNG.normal(size=(L, Hkv, 128)), v, 0.2)
    for h in range(Hq):
        np.testing.assert_allclose(o[:, h, :], h // 8 + 1.0, rtol=1e-13)


def test_attention_scale_two_keys_closed_form():
    a, scale = 3.7, 1 / math.sqrt(128)
    q = np.zeros((1, 1, 128)); q[0, 0, 0] = a
    k = np.zeros((2, 1, 128)); k[0, 0, 0] = 1.0
    v = RNG.normal(size=(2, 1, 128))
    w0 = math.exp(a * scale) / (math.exp(a * scale) + 1.0)
    np.testing.assert_allclose(O.span_attention(q, k, v, scale)[0, 0],
                               w0 * v[0, 0] + (1 - w0) * v[1, 0], rtol=1e-13)


def test_attention_is_causal_within_span():
    n, L = 6, 30
    q = RNG.normal(size=(n, 4, 128)); k = RNG.normal(size=(L, 2, 128)); v = RNG.normal(size=(L, 2, 128))
    o = O.span_attention(q, k, v, 0.09)
    k2, v2 = k.copy(), v.copy()
    k2[-2:] += 5.0; v2[-2:] -= 3.0           # perturb the last two span keys
    o2 = O.span_attention(q, k2, v2, 0.09)
    np.testing.assert_array_equal(o[:n - 2], o2[:n - 2])
    assert np.abs(o[n - 2:] - o2[n - 2:]).min() > 0


def _paged(k, v, ps=16, rng=RNG, extra_pages=5):
    L, Hkv, D = k.shape
    npg = (L + ps - 1) // ps
    pool = npg + extra_pages
    perm = rng.permutation(pool)[:npg]
    kp = rng.normal(size=(pool, Hkv, ps, D)); vp = rng.normal(size=(pool, Hkv, ps, D))
    for p in range(npg):
        seg = slice(p * ps, min(L, (p + 1) * ps))
        cnt = seg.stop - seg.start
        kp[perm[p], :, :cnt, :] = k[seg].transpose(1, 0, 2)
        vp[perm[p], :, :cnt, :] = v[seg].transpose(1, 0, 2)
    return kp, vp, perm


@pytest.mark.parametrize("L", [1, 15, 16, 17, 100])
def test_paged_equals_contiguous_and_page_permutation_is_invisible(L):
    n = min(L, 4)
    q = RNG.normal(size=(n, 8, 128)); k = RNG.normal(size=(L, 4, 128)); v = RNG.normal(size=(L, 4, 128))
    ref = O.span_attention(q, k, v, 0.088)
    for seed in (0, 1):
        kp, vp, row = _paged(k, v, rng=np.random.default_rng(seed))
        kk = O.gather_pages(kp, row, L); vv = O.gather_pages(vp, row, L)
        np.testing.assert_array_equal(kk, k)
        np.testing.assert_array_equal(O.span_attention(q, kk, vv, 0.088), ref)


# ---------------------------------------------------------------------------
# log-softmax, top-K, coverage
# ---------------------------------------------------------------------------
def test_log_partition_library_normalisation_and_shift():
    for V in (5, 4096):
        l = _bf16_round(RNG.normal(size=V) * 3)
        lz = O.log_partition(l)
        assert abs(lz - scipy.special.logsumexp(l)) < 1e-12
        assert abs(np.exp(l - lz).sum() - 1.0) < 1e-12
        assert abs(O.log_partition(l + 8.0) - (lz + 8.0)) < 1e-12


def _brute_topk(l, K):
    return [v for _, v in sorted((-l[v], v) for v in range(len(l)))][:K]


@pytest.mark.parametrize("quantum", [0.0, 0.5, 2.0])
def test_topk_matches_brute_force_sort_with_ties(quantum):
    for _ in range(20):
        V = int(RNG.integers(33, 300))
        l = RNG.normal(size=V) * 3
        if quantum:
            l = np.round(l / quantum) * quantum
        l = _bf16_round(l)
        for K in (1, 4, 16, 32):
            assert O.topk(l, K).tolist() == _brute_topk(l, K)


def test_covered_equals_rank_identity_and_margin_sign():
    for _ in range(10):
        V = int(RNG.integers(40, 120))
        l = _bf16_round(np.round(RNG.normal(size=V) * 2) / 2)
        for K in (1, 3, 16):
            top = set(O.topk(l, K).tolist())
            for x in range(V):
                rank = int(np.sum(l > l[x]) + np.sum(l[:x] == l[x]))
                cov = O.covered(l, x, K)
                assert cov == (rank < K) == (x in top)
                m = O.margin(l, x, K)
                if m > 0:
                    assert cov
                if m < 0:
                    assert not cov


# ---------------------------------------------------------------------------
# top-K KL on the union support
# ---------------------------------------------------------------------------
def test_topk_kl_matches_scipy_entropy():
    for _ in range(30):
        V, K = int(RNG.integers(20, 200)), int(RNG.choice([1, 4, 16]))
        a = _bf16_round(RNG.normal(size=V) * 2)
        b = _bf16_round(RNG.normal(size=V) * 2)
        kl_rev, kl_fwd, S = O.topk_kl(a, b, K)
        assert K <= len(S) <= 2 * K
        assert set(S) == set(_brute_topk(a, K)) | set(_brute_topk(b, K))
        pbar = scipy.special.softmax(a[S]); qbar = scipy.special.softmax(b[S])
        assert abs(kl_rev - scipy.stats.entropy(pbar, qbar)) < 1e-12
        assert abs(kl_fwd - scipy.stats.entropy(qbar, pbar)) < 1e-12


def test_topk_kl_invariants():
    for _ in range(20):
        V = 300
        a = _bf16_round(RNG.normal(size=V) * 3); b = _bf16_round(RNG.normal(size=V) * 3)
        r, f, _ = O.topk_kl(a, b, 16)
        assert r >= 0 and f >= 0
        r2, f2, _ = O.topk_kl(b, a, 16)
        assert abs(r - f2) < 1e-12 and abs(f - r2) < 1e-12
        z = O.topk_kl(a, a, 16)
        assert z[0] == 0.0 and z[1] == 0.0
        # a constant shift of one model's row leaves the renormalised KL unchanged
        s = O.topk_kl(a + 4.0, b, 16)
        assert abs(s[0] - r) < 1e-12


def test_topk_kl_K1_closed_form():
    for _ in range(50):
        a = _bf16_round(RNG.normal(size=50) * 2); b = _bf16_round(RNG.normal(size=50) * 2)
        ia, ib = int(O.topk(a, 1)[0]), int(O.topk(b, 1)[0])
        r, f, S = O.topk_kl(a, b, 1)
        if ia == ib:
            assert len(S) == 1 and r == 0.0 and f == 0.0
            continue
        lo, hi = min(ia, ib), max(ia, ib)
        p = 1 / (1 + math.exp(a[hi] - a[lo]))     # pi_bar(lo)
        s = 1 / (1 + math.exp(b[hi] - b[lo]))     # q_bar(lo)
        bern = p * math.log(p / s) + (1 - p) * math.log((1 - p) / (1 - s))
        assert abs(r - bern) < 1e-12 * max(1.0, abs(bern))


def test_sampled_token_estimator_is_unbiased_by_enumeration():
    """App. B.1: E_{x~pi}[log pi(x) - log q(x)] equals the full-vocabulary reverse
    KL.  The per-token log-probs of score_position are enumerated over every
    token of a tiny vocabulary; the feedback term is minus the estimator."""
    for _ in range(10):
        V = 7
        a = _bf16_round(RNG.normal(size=V) * 2); b = _bf16_round(RNG.normal(size=V) * 2)
        pi = scipy.special.softmax(a)
        est = 0.0
        for x in range(V):
            pos = O.score_position(a, b, x, 0, 3)
            assert abs(pos["feedback"] + (pos["logp_s"] - pos["logp_t"])) < 1e-15
            est += pi[x] * (pos["logp_s"] - pos["logp_t"])
        assert abs(est - scipy.stats.entropy(pi, scipy.special.softmax(b))) < 1e-12


# ---------------------------------------------------------------------------
# verdict
# ---------------------------------------------------------------------------
def _load_verdict_cases():
    cases = []
    for line in open(os.path.join(GOLDEN, "verdict_cases.txt")):
        line = line.split("#")[0].strip()
        if not line:
            continue
        lhs, rhs = line.split("|")
        d, cov, eos, pre = lhs.split()
        n, ft, nd, nl, done, src = rhs.split()
        cases.append((d, cov, eos, int(pre), int(n), int(ft), nd, int(nl), int(done), src))
    return cases


@pytest.mark.parametrize("case", _load_verdict_cases())
def test_verdict_hand_worked_cases(case):
    d, cov, eos, pre, n, ft, nd, nl, done, src = case
    EOS = 99
    k = len(cov)
    toks = [7] * k
    if eos != "-":
        for p in eos.split(","):
            toks[int(p)] = EOS
    v = O.verdict([c == "1" for c in cov], toks, 0 if d == "S" else 1, pre, EOS)
    assert v["n_emit"] == n and v["first_trans"] == ft and v["new_len"] == nl
    assert v["next_driver"] == (0 if nd == "S" else 1) and v["done"] == done
    code = {"S": O.SRC_STUDENT, "T": O.SRC_TEACHER, "-": O.SRC_DISCARDED}
    assert v["source"] == [code[c] for c in src]


def test_verdict_exhaustive_invariants():
    for k in range(1, 9):
        for bits in itertools.product([0, 1], repeat=k):
            for d in (0, 1):
                v = O.verdict(list(bits), [1] * k, d, 10)
                lead = next((i for i, b in enumerate(bits) if b != (1 if d == 0 else 0)), k)
                if d == 0:
                    assert v["n_emit"] == lead and v["first_trans"] == lead
                else:
                    assert v["first_trans"] == lead and v["n_emit"] == min(k, lead + 1)
                assert v["next_driver"] == (1 - d if lead < k else d)
                assert v["new_len"] == 10 + v["n_emit"] and v["done"] == 0
                assert v["source"][:v["n_emit"]] == [d] * v["n_emit"]
                assert all(s == O.SRC_DISCARDED for s in v["source"][v["n_emit"]:])


# ---------------------------------------------------------------------------
# source-split loss
# ---------------------------------------------------------------------------
_R0 = dict(src=[0, 0, 255], rev=[0.5, 0.25, 9.0], fwd=[1.0, 2.0, 9.0], n=2)
_R1 = dict(src=[1, 1, 1], rev=[3.0, 1.0, 2.0], fwd=[0.75, 0.25, 0.5], n=3)


def _golden_loss_inputs():
    src = np.array(_R0["src"] + _R1["src"])
    return (np.array(_R0["rev"] + _R1["rev"]), np.array(_R0["fwd"] + _R1["fwd"]), src,
            np.array([0, 3, 6]), np.array([_R0["n"], _R1["n"]]))


def _load_loss_cases():
    out = []
    for line in open(os.path.join(GOLDEN, "split_loss_cases.txt")):
        line = line.split("#")[0].strip()
        if line:
            lhs, rhs = line.split("|")
            dm, am, rl = lhs.split()
            out.append((int(dm), int(am), None if rl == "-" else [int(x) for x in rl.split(",")],
                        [float(x) for x in rhs.split()]))
    return out


@pytest.mark.parametrize("case", _load_loss_cases())
def test_split_loss_hand_worked(case):
    dm, am, rl, expect = case
    rev, fwd, src, cu, n = _golden_loss_inputs()
    out = O.split_loss(rev, fwd, src, cu, n, None if rl is None else np.array(rl), am, dm)
    got = [out[f] for f in O.LOSS_FIELDS[:6]]
    np.testing.assert_allclose(got, expect, rtol=0, atol=1e-15)


def _random_step(rng, R, k, driver, V=64, K=4):
    ls = rng.normal(size=(R * k, V)) * 2
    lt = rng.normal(size=(R * k, V)) * 2
    bits_s = O.f64_to_bf16(ls); bits_t = O.f64_to_bf16(lt)
    toks = rng.integers(0, V, size=R * k)
    cu = np.arange(R + 1) * k
    return bits_s, bits_t, toks, cu


def test_never_transfer_reduces_to_reverse_kl_opd():
    """Sec. 3.2.2: if control never passes to the teacher, the objective is the
    length-normalised reverse-KL on-policy distillation."""
    rng = np.random.default_rng(5)
    R, k, K = 3, 4, 4
    bs, bt, toks, cu = _random_step(rng, R, k, 0, K=K)
    # make every proposal covered: raise the teacher's logit of the proposed token
    lt = O.bf16_to_f64(bt)
    lt[np.arange(R * k), toks] = 40.0
    bt = O.f64_to_bf16(lt)
    out = O.score_span(bs, bt, toks, cu, np.zeros(R, int), np.full(R, 50), K)
    assert (out["source"] == O.SRC_STUDENT).all()
    loss = O.split_loss(out["kl_rev"], out["kl_fwd"], out["source"], cu, out["n_emit"])
    opd = np.mean([np.mean(out["kl_rev"][cu[r]:cu[r + 1]]) for r in range(R)])
    assert abs(loss["loss"] - opd) < 1e-12 and loss["intervention_ratio"] == 0.0


def test_teacher_that_never_hands_back_reduces_to_forward_kl():
    """Sec. 3.2.2: rejecting the first student token and never handing back
    gives forward-KL off-policy distillation on teacher tokens."""
    rng = np.random.default_rng(6)
    R, k, K = 3, 5, 4
    bs, bt, toks, cu = _random_step(rng, R, k, 1, K=K)
    ls = O.bf16_to_f64(bs)
    ls[np.arange(R * k), toks] = -40.0          # never covered by the student
    bs = O.f64_to_bf16(ls)
    out = O.score_span(bs, bt, toks, cu, np.ones(R, int), np.zeros(R, int), K)
    assert (out["source"] == O.SRC_TEACHER).all()
    loss = O.split_loss(out["kl_rev"], out["kl_fwd"], out["source"], cu, out["n_emit"])
    fwd = np.mean([np.mean(out["kl_fwd"][cu[r]:cu[r + 1]]) for r in range(R)])
    assert abs(loss["loss"] - fwd) < 1e-12 and loss["intervention_ratio"] == 1.0


def test_global_mean_equals_seq_mean_for_equal_lengths():
    rng = np.random.default_rng(7)
    R, k = 5, 3
    rev = rng.random(R * k); fwd = rng.random(R * k)
    src = rng.integers(0, 2, size=R * k)
    cu = np.arange(R + 1) * k
    n = np.full(R, k)
    a = O.split_loss(rev, fwd, src, cu, n, agg_mode=0)
    b = O.split_loss(rev, fwd, src, cu, n, agg_mode=1)
    assert abs(a["loss"] - b["loss"]) < 1e-12


# ---------------------------------------------------------------------------
# planted mistakes: each must be caught by a pin above
# ---------------------------------------------------------------------------
def test_planted_mistakes_are_caught():
    q = RNG.normal(size=(3, 8, 128)); k = RNG.normal(size=(20, 4, 128)); v = RNG.normal(size=(20, 4, 128))
    ref = _sdpa_reference(q, k, v, 0.1)
    # off-by-one causal window (one extra key) is caught by the library pin
    bad = np.zeros_like(ref)
    for i in range(3):
        vis = 20 - 3 + i + 2
        for h in range(8):
            kk = k[:min(vis, 20), h // 2]; s = kk @ q[i, h] * 0.1; p = np.exp(s - s.max())
            bad[i, h] = p @ v[:min(vis, 20), h // 2] / p.sum()
    assert not np.allclose(bad, ref, atol=1e-9)
    # a wrong tie-break (larger index first) is caught by the brute-force sort
    l = _bf16_round(np.array([1.0, 2.0, 2.0, 0.5, 2.0]))
    wrong = np.lexsort((-np.arange(5), -l))[:2].tolist()
    assert wrong != _brute_topk(l, 2) == O.topk(l, 2).tolist()
    # a swapped KL direction is caught by the scipy pin
    a = _bf16_round(RNG.normal(size=40)); b = _bf16_round(RNG.normal(size=40) * 3)
    r, f, S = O.topk_kl(a, b, 4)
    assert abs(f - scipy.stats.entropy(scipy.special.softmax(a[S]), scipy.special.softmax(b[S]))) > 1e-6


# ---------------------------------------------------------------------------
# vocabulary-pass by-products: entropy, top-K overlap, full-vocabulary KL
# ---------------------------------------------------------------------------
def test_entropy_against_scipy_closed_forms_and_shift():
    for V in (2, 17, 4096):
        l = _bf16_round(RNG.normal(size=V) * 3)
        ref = scipy.stats.entropy(scipy.special.softmax(l))  # library, natural log
        assert abs(O.entropy(l) - ref) < 1e-10
        assert abs(O.entropy(l + 5.0) - O.entropy(l)) < 1e-10  # shift invariance
    # uniform row: log V exactly
    assert abs(O.entropy(np.zeros(1000)) - math.log(1000)) < 1e-12
    # two-point closed form: p = sigmoid(a - b), H = -p ln p - (1-p) ln(1-p)
    a, b = 1.75, -0.5
    p = 1.0 / (1.0 + math.exp(b - a))
    assert abs(O.entropy(np.array([a, b])) - (-p * math.log(p) - (1 - p) * math.log(1 - p))) < 1e-12
    # a near-one-hot row has entropy near 0
    assert O.entropy(np.array([60.0] + [0.0] * 50)) < 1e-20


def _brute_overlap(a, b, K):
    sa = sorted(range(len(a)), key=lambda i: (-a[i], i))[:K]
    sb = sorted(range(len(b)), key=lambda i: (-b[i], i))[:K]
    return len(set(sa) & set(sb)) / K


def test_topk_overlap_brute_force_and_extremes():
    for K in (1, 4, 16):
        for quantum in (0.0, 0.5):
            a = RNG.normal(size=64) * 2; b = a + RNG.normal(size=64)
            if quantum:
                a = np.round(a / quantum) * quantum; b = np.round(b / quantum) * quantum
            a, b = _bf16_round(a), _bf16_round(b)
            assert O.topk_overlap(a, b, K) == _brute_overlap(a, b, K)
        a = _bf16_round(RNG.normal(size=64))
        assert O.topk_overlap(a, a, K) == 1.0
        assert O.topk_overlap(a, -a, K) == 0.0  # reversed order: supports disjoint (2K <= 64)


def test_full_kl_against_scipy_and_invariants():
    for V in (3, 100, 4096):
        a = _bf16_round(RNG.normal(size=V) * 2); b = _bf16_round(RNG.normal(size=V) * 2)
        pa, pb = scipy.special.softmax(a), scipy.special.softmax(b)
        rev, fwd = O.full_kl(a, b)
        assert abs(rev - scipy.special.rel_entr(pa, pb).sum()) < 1e-10
        assert abs(fwd - scipy.special.rel_entr(pb, pa).sum()) < 1e-10
        assert rev >= 0 and fwd >= 0
        assert O.full_kl(b, a) == pytest.approx((fwd, rev), abs=1e-12)
        assert O.full_kl(a, a) == (0.0, 0.0)
    # two-token closed form: KL of Bernoulli(p) against Bernoulli(q)
    p = 1 / (1 + math.exp(-1.0)); q = 1 / (1 + math.exp(-(-0.5)))
    rev, _ = O.full_kl(np.array([1.0, 0.0]), np.array([-0.5, 0.0]))
    assert abs(rev - (p * math.log(p / q) + (1 - p) * math.log((1 - p) / (1 - q)))) < 1e-12
    # the full-vocabulary KL equals the top-K KL when K = V (support = everything)
    a = _bf16_round(RNG.normal(size=12)); b = _bf16_round(RNG.normal(size=12))
    r, f, _ = O.topk_kl(a, b, 12)
    assert O.full_kl(a, b) == pytest.approx((r, f), abs=1e-12)


# ---------------------------------------------------------------------------
# takeover / handback rules
# ---------------------------------------------------------------------------
def _span(k, V=32, seed=0):
    g = np.random.default_rng(seed)
    ls = _bf16_round(g.normal(size=(k, V)) * 2)
    lt = _bf16_round(g.normal(size=(k, V)) * 2)
    toks = g.integers(0, V, size=k)
    return ls, lt, toks


def _run_rules(ls, lt, toks, driver, **kw):
    k = len(toks)
    to_bits = lambda x: O.f64_to_bf16(x)
    return O.score_span(to_bits(ls), to_bits(lt), toks, np.array([0, k]), np.array([driver]),
                        np.array([10]), 4, **kw)


def test_always_takeover_is_a_pure_student_rollout():
    # OPD as a special case: the student's span is accepted whole
    ls, lt, toks = _span(9)
    o = _run_rules(ls, lt, toks, 0, takeover_rule=O.RULE_ALWAYS)
    assert o["n_emit"][0] == 9 and o["next_driver"][0] == 0 and o["first_trans"][0] == 9
    assert (o["source"] == O.SRC_STUDENT).all()


def test_skd_handback_after_one_teacher_token():
    # SKD: top-K takeover, fixed one-token handback
    for seed in range(5):
        ls, lt, toks = _span(7, seed=seed)
        o = _run_rules(ls, lt, toks, 1, handback_rule=O.RULE_ALWAYS)
        assert o["n_emit"][0] == 1 and o["first_trans"][0] == 0 and o["next_driver"][0] == 0
        assert o["source"][0] == O.SRC_TEACHER and (o["source"][1:] == O.SRC_DISCARDED).all()
        # the takeover side is unchanged: student spans still follow top-K coverage
        a = _run_rules(ls, lt, toks, 0, handback_rule=O.RULE_ALWAYS)
        b = _run_rules(ls, lt, toks, 0)
        assert a["n_emit"][0] == b["n_emit"][0] and (a["source"] == b["source"]).all()


def test_never_handback_keeps_the_teacher_driving():
    ls, lt, toks = _span(6)
    o = _run_rules(ls, lt, toks, 1, handback_rule=O.RULE_NEVER)
    assert o["n_emit"][0] == 6 and o["next_driver"][0] == 1 and (o["source"] == O.SRC_TEACHER).all()


def test_entropy_rules_follow_the_threshold():
    ls, lt, toks = _span(8, V=64, seed=3)
    hs = [scipy.stats.entropy(scipy.special.softmax(r)) for r in ls]
    ht = [scipy.stats.entropy(scipy.special.softmax(r)) for r in lt]
    for tau in (-np.inf, float(np.median(hs)), np.inf):
        o = _run_rules(ls, lt, toks, 0, takeover_rule=O.RULE_ENTROPY_S, takeover_tau=tau)
        pred = [h <= tau for h in hs]
        n = next((i for i, c in enumerate(pred) if not c), 8)  # first uncovered = takeover
        assert o["n_emit"][0] == n and o["first_trans"][0] == n
        assert (o["covered"] == np.array(pred, dtype=np.int64)).all()
        assert np.allclose(o["margin"], tau - np.array(hs), equal_nan=True) or not np.isfinite(tau)
    tau = float(np.median(ht))
    o = _run_rules(ls, lt, toks, 1, handback_rule=O.RULE_ENTROPY_T, handback_tau=tau)
    pred = [h <= tau for h in ht]
    i = next((i for i, c in enumerate(pred) if c), None)  # first covered = handback
    assert o["n_emit"][0] == (8 if i is None else i + 1)
    assert o["next_driver"][0] == (1 if i is None else 0)
    # entropy outputs are the full-vocabulary entropies of both rows
    assert np.allclose(o["entropy_s"], hs, atol=1e-10) and np.allclose(o["entropy_t"], ht, atol=1e-10)


def test_topk_rule_is_the_default():
    ls, lt, toks = _span(7, seed=9)
    a = _run_rules(ls, lt, toks, 0)
    b = _run_rules(ls, lt, toks, 0, takeover_rule=O.RULE_TOPK, handback_rule=O.RULE_TOPK)
    for name in ("covered", "source", "n_emit", "first_trans", "next_driver"):
        assert (a[name] == b[name]).all()


def test_planted_rule_mistakes_are_caught():
    # a takeover on the teacher's entropy instead of the student's changes decisions
    ls, lt, toks = _span(8, V=64, seed=3)
    hs = [scipy.stats.entropy(scipy.special.softmax(r)) for r in ls]
    tau = float(np.median(hs))
    good = _run_rules(ls, lt, toks, 0, takeover_rule=O.RULE_ENTROPY_S, takeover_tau=tau)
    bad = _run_rules(ls, lt, toks, 0, takeover_rule=O.RULE_ENTROPY_T, takeover_tau=tau)
    assert (good["covered"] != bad["covered"]).any()
    # an entropy with the wrong sign of the mean term differs from scipy
    l = _bf16_round(RNG.normal(size=50) * 2)
    lz = O.log_partition(l); p = np.exp(l - lz)
    assert abs((lz + np.dot(p, l)) - scipy.stats.entropy(p)) > 1e-3


# ---------------------------------------------------------------------------
# gradient of the source-split objective (finite differences of the loss)
# ---------------------------------------------------------------------------
def _grad_case(seed, V=40, K=4):
    rng = np.random.default_rng(seed)
    cu = np.array([0, 3, 3, 7, 10])            # one request with an empty span
    T = int(cu[-1])
    ls = rng.normal(size=(T, V)) * 2.0          # continuous: no ties, fixed supports
    lt = rng.normal(size=(T, V)) * 2.0
    source = np.array([0, 0, 255, 1, 1, 1, 255, 0, 0, 0])
    n_emit = np.array([2, 0, 3, 3])
    resp_len = np.array([5, 0, 3, 9])
    return ls, lt, source, cu, n_emit, resp_len, K


def _loss_of_student_logits(ls, lt, source, cu, n_emit, resp_len, K, agg, dmode):
    T = ls.shape[0]
    kr = np.zeros(T); kf = np.zeros(T)
    for t in range(T):
        kr[t], kf[t], _ = O.topk_kl(ls[t], lt[t], K)
    return O.split_loss(kr, kf, source, cu, n_emit, resp_len, agg, dmode)["loss"]


@pytest.mark.parametrize("agg,dmode,use_len", [(0, 0, False), (1, 0, True), (0, 1, True),
                                                (1, 2, False), (0, 3, True)])
def test_split_loss_grad_matches_finite_differences(agg, dmode, use_len):
    ls, lt, source, cu, n_emit, resp_len, K = _grad_case(7 + dmode)
    rl = resp_len if use_len else None
    G = O.split_loss_grad(ls, lt, source, cu, n_emit, rl, K, agg, dmode, grad_scale=1.0)
    eps = 1e-6
    fd = np.zeros_like(G)
    for t in range(ls.shape[0]):
        for v in range(ls.shape[1]):
            a = ls.copy(); a[t, v] += eps
            b = ls.copy(); b[t, v] -= eps
            fd[t, v] = (_loss_of_student_logits(a, lt, source, cu, n_emit, rl, K, agg, dmode)
                        - _loss_of_student_logits(b, lt, source, cu, n_emit, rl, K, agg, dmode)) / (2 * eps)
    assert np.abs(G - fd).max() <= 1e-8 + 1e-6 * np.abs(fd).max()
    assert np.abs(G).max() > 1e-3                # the case is not trivially zero


def test_split_loss_grad_rows_are_shift_invariant_and_zero_off_the_emitted_positions():
    ls, lt, source, cu, n_emit, resp_len, K = _grad_case(3)
    G = O.split_loss_grad(ls, lt, source, cu, n_emit, None, K, 0, 0, grad_scale=2.5)
    # adding a constant to a student row leaves every KL unchanged
    assert np.abs(G.sum(axis=1)).max() < 1e-14
    for t in range(G.shape[0]):
        S = np.union1d(O.topk(ls[t], K), O.topk(lt[t], K))
        off = np.setdiff1d(np.arange(G.shape[1]), S)
        assert (G[t, off] == 0).all()
        if source[t] == O.SRC_DISCARDED:
            assert (G[t] == 0).all()
    # grad_scale is a plain factor
    G1 = O.split_loss_grad(ls, lt, source, cu, n_emit, None, K, 0, 0, grad_scale=1.0)
    assert np.allclose(G, 2.5 * G1, rtol=1e-15, atol=0)


def test_planted_gradient_mistakes_are_caught():
    ls, lt, source, cu, n_emit, resp_len, K = _grad_case(11)
    G = O.split_loss_grad(ls, lt, source, cu, n_emit, None, K, 0, 0)
    # the reverse-KL gradient without its "- KL" centring term no longer sums to 0
    t = 0
    S = np.union1d(O.topk(ls[t], K), O.topk(lt[t], K))
    lp = ls[t, S] - O.log_partition(ls[t, S]); lq = lt[t, S] - O.log_partition(lt[t, S])
    p = np.exp(lp)
    w = G[t, S][0] / (p[0] * (lp[0] - lq[0] - np.sum(p * (lp - lq))))
    bad = w * p * (lp - lq)
    assert abs(bad.sum()) > 1e-6 and abs(G[t].sum()) < 1e-14
    # the forward-KL gradient with the sign flipped disagrees with finite differences
    eps = 1e-6
    t = 3                                        # teacher-sourced: forward KL under IPD
    v = int(np.union1d(O.topk(ls[t], K), O.topk(lt[t], K))[0])
    a = ls.copy(); a[t, v] += eps
    b = ls.copy(); b[t, v] -= eps
    fd = (_loss_of_student_logits(a, lt, source, cu, n_emit, None, K, 0, 0)
          - _loss_of_student_logits(b, lt, source, cu, n_emit, None, K, 0, 0)) / (2 * eps)
    assert abs(G[t, v] - fd) < 1e-8 and abs(-G[t, v] - fd) > 1e-4


# ---------------------------------------------------------------------------
# seeded sampler: Philox known answers, lg2 accuracy, the sampled distribution
# ---------------------------------------------------------------------------
def test_philox_known_answer_vectors():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt"))
            if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for w in rows:
        v = [int(x, 16) for x in w]
        out = O.philox4x32_10(np.array([v[0:4]], dtype=np.uint32), (v[4], v[5]))[0]
        assert out.tolist() == v[6:10]


def test_lg2_against_numpy_log2():
    xs = np.concatenate([np.exp(RNG.uniform(np.log(2.0 ** -26), np.log(32.0), 200000)),
                         np.linspace(0.5, 2.0, 20001), [1 - 2.0 ** -24, 1 + 2.0 ** -23, 1.0,
                                                        2.0 ** -24, 24.0, np.sqrt(2.0)]])
    xs = xs.astype(np.float32)
    ours = O.lg2_f32(xs).astype(np.float64)
    ref = np.log2(xs.astype(np.float64))
    assert np.abs(ours - ref).max() <= 1.2e-6
    near = np.abs(xs - 1) < 0.3
    assert (np.abs(ours - ref)[near] <= 4e-7 * np.maximum(np.abs(ref[near]), 2.0 ** -24) + 1e-12).all()
    assert O.lg2_f32(np.float32(1.0)) == 0.0 and O.lg2_f32(np.float32(0.25)) == -2.0
    # the sign the Gumbel transform relies on: lg2(u) < 0 for every u < 1
    assert (O.lg2_f32(np.float32([1 - 2.0 ** -24, 0.5 + 2.0 ** -24])) < 0).all()


def test_uniforms_are_uniform_and_open():
    u = O.sample_uniforms(1 << 16, seed=12345, draw=7).astype(np.float64)
    assert u.min() > 0 and u.max() < 1
    assert scipy.stats.kstest(u, "uniform").pvalue > 1e-4
    # distinct draws give distinct streams; the same draw repeats exactly
    assert not np.array_equal(u, O.sample_uniforms(1 << 16, seed=12345, draw=8))
    assert np.array_equal(u, O.sample_uniforms(1 << 16, seed=12345, draw=7))


def _draw_counts(l_bits, n, inv_temperature=1.0, scores=None):
    V = len(l_bits)
    counts = np.zeros(V, dtype=np.int64)
    for d in range(n):
        s = O.gumbel_scores(l_bits, 99, d, inv_temperature) if scores is None else scores(d)
        counts[int(np.argmax(s))] += 1
    return counts


@pytest.mark.parametrize("inv_t", [1.0, 0.5])
def test_sampled_tokens_follow_the_softmax(inv_t):
    l = np.array([0.0, 1.0, 2.0, -1.0, 0.5, 3.0])
    bits = O.f64_to_bf16(l)
    n = 12000
    counts = _draw_counts(bits, n, inv_t)
    p = scipy.special.softmax(l * inv_t)
    assert scipy.stats.chisquare(counts, p * n).pvalue > 1e-4


def test_planted_sampler_mistakes_are_caught():
    l = np.array([0.0, 1.0, 2.0, -1.0, 0.5, 3.0])
    bits = O.f64_to_bf16(l)
    n = 12000
    p = scipy.special.softmax(l) * n
    lf = l.astype(np.float32)
    # a natural log in the outer logarithm (base mismatch) samples a tempered softmax
    nat = lambda d: lf * np.float32(1.4426950) - np.log(-O.lg2_f32(O.sample_uniforms(6, 99, d)))
    assert scipy.stats.chisquare(_draw_counts(bits, n, scores=nat), p).pvalue < 1e-6
    # dropping the log2(e) factor of the logits samples softmax(l ln 2)
    noc = lambda d: lf - O.lg2_f32(-O.lg2_f32(O.sample_uniforms(6, 99, d)))
    assert scipy.stats.chisquare(_draw_counts(bits, n, scores=noc), p).pvalue < 1e-6


def test_next_token_after_verdict_picks_the_next_drivers_row():
    V = 64
    ls = O.f64_to_bf16(RNG.normal(size=(9, V)) * 2)
    lt = O.f64_to_bf16(RNG.normal(size=(9, V)) * 2)
    cu = np.array([0, 4, 7, 9])
    prefix = np.array([10, 20, 30])
    # request 0: student span, takeover at j = 2 -> the teacher's row 2 at position 12
    # request 1: teacher span, handback at j = 0 -> the student's row 1 at position 21
    # request 2: student span, everything accepted -> no row in this step
    v = dict(n_emit=np.array([2, 1, 2]), done=np.array([0, 0, 0]),
             next_driver=np.array([1, 0, 0]))
    got = O.next_token_after_verdict(ls, lt, cu, prefix, v, seed=5, draw_base=np.array([100, 0, 0]))
    assert got[0] == O.sample_token(lt[2], 5, 100 + 12)
    assert got[1] == O.sample_token(ls[4 + 1], 5, 21)
    assert got[2] == -1
    # a request that ended (EOS) draws nothing
    v["done"] = np.array([1, 0, 0])
    assert O.next_token_after_verdict(ls, lt, cu, prefix, v, 5, np.array([100, 0, 0]))[0] == -1


# ---------------------------------------------------------------------------
# KV append: the appended paged cache attends like the concatenated sequence
# ---------------------------------------------------------------------------
def test_kv_append_then_paged_attention_equals_sdpa_on_the_concatenation():
    rng = np.random.default_rng(21)
    Hkv, D, ps = 2, 128, 16
    old_len = [5, 16, 30, 0]
    n_new = [3, 1, 0, 17]                                 # span, decode, nothing, across pages
    L = [a + b for a, b in zip(old_len, n_new)]
    max_pages = max((x + ps - 1) // ps for x in L)
    num_pages = sum((x + ps - 1) // ps for x in L) + 3
    perm = rng.permutation(num_pages)
    table = np.full((4, max_pages), -1)
    used = 0
    for r, x in enumerate(L):
        for j in range((x + ps - 1) // ps):
            table[r, j] = perm[used]; used += 1
    kp = rng.normal(size=(num_pages, Hkv, ps, D)); vp = rng.normal(size=(num_pages, Hkv, ps, D))
    old_k = [O.gather_pages(kp, table[r], old_len[r]) for r in range(4)]
    old_v = [O.gather_pages(vp, table[r], old_len[r]) for r in range(4)]
    cu = np.concatenate([[0], np.cumsum(n_new)])
    kn = rng.normal(size=(int(cu[-1]), Hkv, D)); vn = rng.normal(size=(int(cu[-1]), Hkv, D))
    k2, v2 = O.kv_append(kp, vp, kn, vn, cu, L, table)
    for r in range(4):
        if L[r] == 0:
            continue
        k_cat = np.concatenate([old_k[r], kn[cu[r]:cu[r + 1]]])
        v_cat = np.concatenate([old_v[r], vn[cu[r]:cu[r + 1]]])
        q = rng.normal(size=(max(n_new[r], 1), 4, D))
        got = O.span_attention(q, O.gather_pages(k2, table[r], L[r]),
                               O.gather_pages(v2, table[r], L[r]), 0.09)
        np.testing.assert_allclose(got, _sdpa_reference(q, k_cat, v_cat, 0.09), rtol=1e-10, atol=1e-12)
    # pages no request owns are untouched
    free = np.setdiff1d(np.arange(num_pages), table[table >= 0])
    assert np.array_equal(k2[free], kp[free]) and np.array_equal(v2[free], vp[free])
    # a position off by one is caught: the appended rows no longer form the sequence
    kb, vb = O.kv_append(kp, vp, kn, vn, cu, [x + 1 for x in L], np.pad(table, ((0, 0), (0, 1)),
                                                                       constant_values=perm[-1]))
    assert not np.array_equal(O.gather_pages(kb, table[0], L[0]), np.concatenate([old_k[0], kn[0:3]]))


@pytest.mark.parametrize("driver", [0, 1])
def test_rows_past_the_transition_do_not_change_the_verdict_or_the_loss(driver):
    """Reading R22: the verdict needs the verifier's rows up to the first
    transition, the loss the emitted positions' rows.  Replacing every row the
    reading calls unneeded (the verifier's past the transition, the proposer's
    at positions not emitted) leaves the verdict, the sources and the loss of
    the oracle unchanged."""
    for seed in range(12):
        ls, lt, toks = _span(10, V=32, seed=100 + seed)
        o = _run_rules(ls, lt, toks, driver)
        ft, n = int(o["first_trans"][0]), int(o["n_emit"][0])
        g = np.random.default_rng(seed)
        ls2, lt2 = ls.copy(), lt.copy()
        ver, prop = (lt2, ls2) if driver == 0 else (ls2, lt2)
        for i in range(10):
            if i > ft:
                ver[i] = _bf16_round(g.normal(size=32) * 2)
            if i >= n:
                prop[i] = _bf16_round(g.normal(size=32) * 2)
        o2 = _run_rules(ls2, lt2, toks, driver)
        for name in ("first_trans", "n_emit", "next_driver", "new_len", "done", "source"):
            assert np.array_equal(o[name], o2[name]), name
        em = o["source"] != O.SRC_DISCARDED
        for name in ("kl_rev", "kl_fwd", "logp_s", "logp_t"):
            assert np.array_equal(o[name][em], o2[name][em]), name
        l1 = O.split_loss(o["kl_rev"], o["kl_fwd"], o["source"], np.array([0, 10]), o["n_emit"])
        l2 = O.split_loss(o2["kl_rev"], o2["kl_fwd"], o2["source"], np.array([0, 10]),
                          o2["n_emit"])
        assert l1["loss"] == l2["loss"]
    # and a row the reading does need changes the verdict when it is replaced
    ls, lt, toks = _span(10, V=32, seed=7)
    o = _run_rules(ls, lt, toks, 0)
    ft = int(o["first_trans"][0])
    assert ft < 10  # this span has a takeover
    lt2 = lt.copy()
    lt2[ft, toks[ft]] = 50.0  # the verifier's row at the transition now covers the token
    assert _run_rules(ls, lt2, toks, 0)["first_trans"][0] != ft
