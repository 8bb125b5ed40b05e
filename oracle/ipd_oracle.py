"""Plain fp64 statement of the IPD verify step (test infrastructure only).

Every function here is the textbook definition or the paper's rule written out
in the paper's order, with no blocking, fusion or reordering.  numpy's matmul,
sort, exp and log are the only library steps.  Inputs are bf16 bit patterns
(uint16) or integers; bf16 -> fp64 conversion is exact.

Notation follows the paper: pi = student, q = teacher, K = top-K width,
S_t = union of both top-K supports (Sec. 3.1, "Sampled-Token and Top-K OPD";
Sec. 4.1 fixes the union support and K = 16), m = driver state, z = token
source (Sec. 3.2.1).
"""
from __future__ import annotations

import numpy as np

SRC_STUDENT = 0
SRC_TEACHER = 1
SRC_DISCARDED = 255


# ----------------------------------------------------------------------------
# bf16 helpers (exact conversions)
# ----------------------------------------------------------------------------
def bf16_to_f64(bits) -> np.ndarray:
    """bf16 bit patterns (uint16) -> exact fp64 values."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def f64_to_bf16(x) -> np.ndarray:
    """fp64 -> bf16 bit patterns, round to nearest even (via the exact fp32
    value when it is representable; the double rounding is avoided by rounding
    fp64 straight to 8 significant bits)."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                       # x = m * 2**e, 0.5 <= |m| < 1
    r = np.ldexp(np.round(np.ldexp(m, 8)), e - 8)   # np.round is half-to-even
    return (r.astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def bf16_ulp(x) -> np.ndarray:
    """Spacing of bf16 numbers at |x| (normal range)."""
    x = np.abs(np.asarray(x, dtype=np.float64))
    _, e = np.frexp(np.maximum(x, np.finfo(np.float32).tiny))
    return np.ldexp(1.0, e - 8)


# ----------------------------------------------------------------------------
# (a) span-verify attention and (b) proposer decode attention
# Sec. 3.2.3: the verifier evaluates the k draft tokens of a request in one
# prefill pass over its own cache (only the new tokens are computed); the
# proposer decodes one token at a time over its own cache.
# ----------------------------------------------------------------------------
def gather_pages(pages: np.ndarray, page_row: np.ndarray, L: int, page_size: int = 16):
    """Paged cache [num_pages, Hkv, page_size, D] -> contiguous [L, Hkv, D]."""
    n = (L + page_size - 1) // page_size
    blocks = [pages[int(page_row[p])] for p in range(n)]          # each [Hkv, ps, D]
    cont = np.concatenate([b.transpose(1, 0, 2) for b in blocks], axis=0) if n else \
        np.zeros((0,) + (pages.shape[1], pages.shape[3]))
    return cont[:L]


def kv_append(k_pages: np.ndarray, v_pages: np.ndarray, k_new: np.ndarray, v_new: np.ndarray,
              cu_new, seq_len, page_table, page_size: int = 16):
    """The cache after the new tokens' K/V rows are written (Sec. 3.2.3: the
    proposer's decode extends its own cache by one token, the verifier's
    prefill writes the span's k tokens into its cache, each before the
    attention that reads them).

    k_pages, v_pages: [num_pages, Hkv, page_size, D]; k_new, v_new:
    [total_new, Hkv, D].  Request r's rows cu_new[r] .. cu_new[r+1]-1 are the
    last n_r tokens of its sequence of length seq_len[r] (the length after the
    append): row i lands at position p = seq_len[r] - n_r + i, in page
    page_table[r][p // page_size], slot p % page_size.  Returns new arrays."""
    k_out, v_out = k_pages.copy(), v_pages.copy()
    for r in range(len(cu_new) - 1):
        n = int(cu_new[r + 1]) - int(cu_new[r])
        for i in range(n):
            p = int(seq_len[r]) - n + i
            page = int(page_table[r][p // page_size])
            k_out[page, :, p % page_size, :] = k_new[int(cu_new[r]) + i]
            v_out[page, :, p % page_size, :] = v_new[int(cu_new[r]) + i]
    return k_out, v_out


def span_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float) -> np.ndarray:
    """Causal attention of n span queries over a contiguous cache of L keys.

    q: [n, Hq, D]; k, v: [L, Hkv, D] (fp64).  Query i sits at absolute position
    L - n + i and sees keys 0 .. L - n + i.  Query head h reads KV head
    h // (Hq / Hkv).  Returns [n, Hq, D] fp64.  A decode query is n = 1."""
    n, Hq, D = q.shape
    L, Hkv, _ = k.shape
    G = Hq // Hkv
    out = np.zeros((n, Hq, D))
    for i in range(n):
        visible = L - n + i + 1
        for h in range(Hq):
            kh = h // G
            s = (k[:visible, kh, :] @ q[i, h, :]) * scale          # scores
            s = s - s.max()
            p = np.exp(s)
            out[i, h, :] = (p @ v[:visible, kh, :]) / p.sum()
    return out


def paged_span_attention(q_bits, k_pages_bits, v_pages_bits, page_row, L, scale):
    """span_attention on a paged cache given as bf16 bit patterns."""
    k = gather_pages(bf16_to_f64(k_pages_bits), page_row, L)
    v = gather_pages(bf16_to_f64(v_pages_bits), page_row, L)
    return span_attention(bf16_to_f64(q_bits), k, v, scale)


# ----------------------------------------------------------------------------
# (c) the vocabulary pass over both models' logits
# ----------------------------------------------------------------------------
def log_partition(l: np.ndarray) -> float:
    """log sum_v exp(l_v), with the maximum taken out first."""
    m = l.max()
    return float(m + np.log(np.exp(l - m).sum()))


def topk(l: np.ndarray, K: int) -> np.ndarray:
    """Top_K of Eq. (topk_sets): the K indices of largest probability.

    Probabilities are a monotone function of the logits at temperature 1, so the
    order is taken on the logits.  Equal logits are ordered by smaller token id
    first, which makes the set unique."""
    order = np.lexsort((np.arange(l.size), -l))
    return order[:K]


def covered(l: np.ndarray, x: int, K: int) -> bool:
    """Coverage test of Eq. (ipd_state_transition): x in Top_K(row)."""
    return bool(x in set(topk(l, K).tolist()))


def margin(l: np.ndarray, x: int, K: int) -> float:
    """l[x] minus the K-th largest logit (the coverage threshold)."""
    return float(l[x] - l[topk(l, K)[K - 1]])


def topk_kl(l_pi: np.ndarray, l_q: np.ndarray, K: int):
    """Token-level top-K KL terms on the union support.

    S_t = Top_K(pi) u Top_K(q) (Sec. 4.1 / App. A); pi and q are renormalised on
    S_t separately (Eq. topk_normalization); then
      kl_rev = KL(pi_bar || q_bar)   (Eq. topk_opd_on_sequence, l_on of Eq. ipd_off_loss)
      kl_fwd = KL(q_bar || pi_bar)   (l_off of Eq. ipd_off_loss).
    The full-vocabulary normaliser cancels in the renormalisation, so the
    restricted log-sum-exp of the raw logits is used.  Terms with zero mass
    contribute zero."""
    S = np.union1d(topk(l_pi, K), topk(l_q, K))
    a = l_pi[S]
    b = l_q[S]
    log_pi_bar = a - log_partition(a)
    log_q_bar = b - log_partition(b)
    pi_bar = np.exp(log_pi_bar)
    q_bar = np.exp(log_q_bar)
    d = log_pi_bar - log_q_bar
    kl_rev = float(np.sum(np.where(pi_bar > 0, pi_bar * d, 0.0)))
    kl_fwd = float(np.sum(np.where(q_bar > 0, q_bar * (-d), 0.0)))
    return kl_rev, kl_fwd, S


def entropy(l: np.ndarray) -> float:
    """Shannon entropy (nats) of softmax(l) over the whole vocabulary,
    log Z - sum_v p_v l_v (the per-position entropy of Sec. 3.2, Fig.
    teacher_unanchoring)."""
    lz = log_partition(l)
    p = np.exp(l - lz)
    return float(lz - np.dot(p, l))


def topk_overlap(l_pi: np.ndarray, l_q: np.ndarray, K: int) -> float:
    """Top-K overlap ratio |S^pi intersect S^q| / K (Sec. 4.2, main results)."""
    return len(set(topk(l_pi, K).tolist()) & set(topk(l_q, K).tolist())) / K


def full_kl(l_pi: np.ndarray, l_q: np.ndarray):
    """Full-vocabulary KL of Eq. (full_vocab_opd) in both directions:
    (KL(pi || q), KL(q || pi)), each sum_v p(v) (log p(v) - log p'(v))."""
    lp = l_pi - log_partition(l_pi)
    lq = l_q - log_partition(l_q)
    p, q = np.exp(lp), np.exp(lq)
    return float(np.sum(p * (lp - lq))), float(np.sum(q * (lq - lp)))


# Takeover / handback rules (Sec. 3.2.1: IPD admits other rules than top-K
# coverage, possibly different for takeover and handback; an entropy threshold
# on either model is the paper's example, and SKD is top-K takeover with a
# fixed one-token handback).  A span proposed by the student is governed by
# the takeover rule (its predicate true = accept), a span proposed by the
# teacher by the handback rule (true = hand back).
RULE_TOPK, RULE_ENTROPY_S, RULE_ENTROPY_T, RULE_ALWAYS, RULE_NEVER = 0, 1, 2, 3, 4


def rule_predicate(rule: int, tau: float, l_s: np.ndarray, l_t: np.ndarray, x: int, driver: int,
                   K: int):
    """(predicate, margin) of a rule at one position.  The margin is the signed
    distance of the decision from its threshold, >= 0 when the predicate holds
    except for exact top-K ties, which the token-id order decides."""
    if rule == RULE_TOPK:
        ver = l_t if driver == 0 else l_s  # the verifier's row
        return covered(ver, x, K), margin(ver, x, K)
    if rule in (RULE_ENTROPY_S, RULE_ENTROPY_T):
        h = entropy(l_s if rule == RULE_ENTROPY_S else l_t)
        return h <= tau, tau - h
    if rule == RULE_ALWAYS:
        return True, np.inf
    if rule == RULE_NEVER:
        return False, -np.inf
    raise ValueError(rule)


def score_position(l_s: np.ndarray, l_t: np.ndarray, x: int, driver: int, K: int,
                   rule: int = RULE_TOPK, tau: float = 0.0) -> dict:
    """All per-token quantities of one span position.

    l_s, l_t: fp64 logits of the student (pi) and teacher (q) at this position;
    x: the proposed token; driver 0 = student proposes (teacher verifies),
    1 = teacher proposes (student verifies); rule, tau: the rule governing
    the span (takeover rule for driver 0, handback rule for driver 1)."""
    logZ_s = log_partition(l_s)
    logZ_t = log_partition(l_t)
    logp_s = float(l_s[x] - logZ_s)
    logp_t = float(l_t[x] - logZ_t)
    kl_rev, kl_fwd, _ = topk_kl(l_s, l_t, K)
    cov, mar = rule_predicate(rule, tau, l_s, l_t, x, driver, K)
    return dict(
        logp_s=logp_s, logp_t=logp_t,
        # token-level teacher feedback: the per-token reward -l_hat^sample =
        # log q(x) - log pi(x) (Eq. sampled_token_opd and App. B.1)
        feedback=logp_t - logp_s,
        kl_rev=kl_rev, kl_fwd=kl_fwd,
        covered=cov, margin=mar,
        entropy_s=entropy(l_s), entropy_t=entropy(l_t),
        topk_overlap=topk_overlap(l_s, l_t, K))


def verdict(cov, tokens, driver: int, prefix_len: int, eos_id: int = -1) -> dict:
    """Apply Eq. (ipd_state_transition) token by token to one proposed span.

    Student driving (driver 0): a covered proposal is emitted with z = S; the
    first uncovered one is a takeover: it is rejected (the teacher regenerates
    that position in its next proposal), both caches roll back to the token
    before it, and the driver becomes T.  A student EOS ends the request only
    when covered.
    Teacher driving (driver 1): every proposal is emitted with z = T; the first
    covered one is the handback: it is kept, the rest of the span is dropped,
    and the driver becomes S.  A teacher EOS is accepted directly and ends the
    request.
    Both caches end at prefix_len + n_emit (Sec. 3.2.3, verdict stage)."""
    k = len(cov)
    m = driver
    n_emit = 0
    first_trans = k
    done = 0
    source = [SRC_DISCARDED] * k
    for i in range(k):
        x = int(tokens[i])
        if driver == 0:
            if cov[i]:
                source[i] = SRC_STUDENT
                n_emit = i + 1
                if eos_id >= 0 and x == eos_id:
                    done = 1
                    break
            else:
                first_trans = i
                m = 1
                break
        else:
            source[i] = SRC_TEACHER
            n_emit = i + 1
            if cov[i]:
                first_trans = i
                m = 0
            if eos_id >= 0 and x == eos_id:
                done = 1
            if cov[i] or done:
                break
    return dict(first_trans=first_trans, n_emit=n_emit, next_driver=m,
                new_len=prefix_len + n_emit, done=done, source=source)


POS_FIELDS = ("logp_s", "logp_t", "feedback", "kl_rev", "kl_fwd", "margin", "entropy_s",
              "entropy_t", "topk_overlap")


def score_span(logits_s_bits, logits_t_bits, tokens, cu_span, driver, prefix_len, K, eos_id=-1,
               requests=None, takeover_rule=RULE_TOPK, handback_rule=RULE_TOPK,
               takeover_tau=0.0, handback_tau=0.0) -> dict:
    """The whole vocabulary pass + verdict for the requests in ``requests``
    (default: all).  Per-token arrays are returned in the flat span order, with
    NaN / -1 at positions of requests that were not evaluated."""
    T = int(cu_span[-1])
    R = len(cu_span) - 1
    reqs = range(R) if requests is None else requests
    out = {name: np.full(T, np.nan) for name in POS_FIELDS}
    out["covered"] = np.full(T, -1, dtype=np.int64)
    out["source"] = np.full(T, -1, dtype=np.int64)
    for name in ("first_trans", "n_emit", "next_driver", "new_len", "done"):
        out[name] = np.full(R, -1, dtype=np.int64)
    for r in reqs:
        t0, t1 = int(cu_span[r]), int(cu_span[r + 1])
        cov = []
        d = int(driver[r])
        rule, tau = (takeover_rule, takeover_tau) if d == 0 else (handback_rule, handback_tau)
        for t in range(t0, t1):
            pos = score_position(bf16_to_f64(logits_s_bits[t]), bf16_to_f64(logits_t_bits[t]),
                                 int(tokens[t]), d, K, rule, tau)
            for name in POS_FIELDS:
                out[name][t] = pos[name]
            out["covered"][t] = int(pos["covered"])
            cov.append(pos["covered"])
        v = verdict(cov, tokens[t0:t1], int(driver[r]), int(prefix_len[r]), eos_id)
        out["source"][t0:t1] = v["source"]
        for name in ("first_trans", "n_emit", "next_driver", "new_len", "done"):
            out[name][r] = v[name]
    return out


# ----------------------------------------------------------------------------
# source-split reduction
# ----------------------------------------------------------------------------
DIR_IPD, DIR_PURE_REV, DIR_PURE_FWD, DIR_INVERSE = 0, 1, 2, 3


def split_loss(kl_rev, kl_fwd, source, cu_span, n_emit, resp_len=None, agg_mode=0,
               dir_mode=DIR_IPD) -> dict:
    """Source-split objective of Eq. (ipd_objective) for one step.

    Student-sourced positions (z = S) take l_on, teacher-sourced ones (z = T)
    take l_off (Eq. ipd_off_loss).  dir_mode selects the KL direction of each
    group as in the KL-direction ablation (Sec. 4.3): 0 IPD split (on: reverse,
    off: forward), 1 pure reverse, 2 pure forward, 3 inverse split.
    agg_mode 0 is the sequence-mean-token-mean of Eq. (ipd_objective): each
    request's sum is divided by its length |x_r| (resp_len, or the emitted
    count when resp_len is None) and requests with |x_r| = 0 are left out of
    the batch mean; agg_mode 1 is the global token mean (App. B.3).
    Returns the loss, the per-source sums and counts, the teacher intervention
    ratio (share of teacher-sourced tokens, Sec. 4.3) and the numerator /
    denominator whose ratio is the loss (so shards can be combined)."""
    on_rev = dir_mode in (DIR_IPD, DIR_PURE_REV)
    off_fwd = dir_mode in (DIR_IPD, DIR_PURE_FWD)
    R = len(cu_span) - 1
    sum_on = sum_off = 0.0
    n_on = n_off = 0
    per_req = []
    denoms = []
    for r in range(R):
        s_on = s_off = 0.0
        for t in range(int(cu_span[r]), int(cu_span[r + 1])):
            if source[t] == SRC_STUDENT:
                s_on += kl_rev[t] if on_rev else kl_fwd[t]
                n_on += 1
            elif source[t] == SRC_TEACHER:
                s_off += kl_fwd[t] if off_fwd else kl_rev[t]
                n_off += 1
        sum_on += s_on
        sum_off += s_off
        d = int(n_emit[r]) if resp_len is None else int(resp_len[r])
        per_req.append(s_on + s_off)
        denoms.append(d)
    if agg_mode == 0:
        terms = [per_req[r] / denoms[r] for r in range(R) if denoms[r] > 0]
        numer, denom = float(sum(terms)), float(len(terms))
    else:
        numer = float(sum(per_req[r] for r in range(R) if denoms[r] > 0))
        denom = float(sum(d for d in denoms if d > 0))
    loss = numer / denom if denom > 0 else 0.0
    ntot = n_on + n_off
    return dict(loss=loss, sum_on=sum_on, sum_off=sum_off, n_on=float(n_on), n_off=float(n_off),
                intervention_ratio=(n_off / ntot) if ntot else 0.0, numer=numer, denom=denom)


LOSS_FIELDS = ("loss", "sum_on", "sum_off", "n_on", "n_off", "intervention_ratio", "numer", "denom")


# ----------------------------------------------------------------------------
# gradient of the source-split objective with respect to the student's logits
# ----------------------------------------------------------------------------
def split_loss_grad(l_s, l_t, source, cu_span, n_emit, resp_len=None, K=16, agg_mode=0,
                    dir_mode=DIR_IPD, grad_scale=1.0) -> np.ndarray:
    """d(grad_scale * loss) / d l_s for the loss of ``split_loss``, as a dense
    [T, V] fp64 array.  ``l_s`` and ``l_t`` are the two models' logits as fp64
    rows (bf16 rows go through ``bf16_to_f64`` first).

    Each emitted position t contributes its token-level KL (Eq. ipd_off_loss,
    direction chosen per source as in ``split_loss``) with weight
    w_t = 1 / (R' |x_r|) under the sequence-mean-token-mean of
    Eq. (ipd_objective), or 1 / sum_r |x_r| under the global token mean.  The
    supports S_t = Top_K(pi_t) u Top_K(q_t) are piecewise constant in the
    logits and are held fixed.  With pi_bar the student's softmax restricted
    to S_t (Eq. topk_normalization; its normaliser is the only place the
    student's logits enter besides the numerator), for v in S_t:
      d KL(pi_bar || q_bar) / d l_v = pi_bar_v (log pi_bar_v - log q_bar_v - KL(pi_bar || q_bar))
      d KL(q_bar || pi_bar) / d l_v = pi_bar_v - q_bar_v
    and every logit outside S_t has gradient 0."""
    l_s = np.asarray(l_s, dtype=np.float64)
    l_t = np.asarray(l_t, dtype=np.float64)
    T, V = l_s.shape
    R = len(cu_span) - 1
    dens = [int(n_emit[r]) if resp_len is None else int(resp_len[r]) for r in range(R)]
    if agg_mode == 0:
        D = float(sum(1 for d in dens if d > 0))
    else:
        D = float(sum(d for d in dens if d > 0))
    G = np.zeros((T, V))
    for r in range(R):
        if dens[r] <= 0:
            continue
        w = grad_scale / (D * dens[r]) if agg_mode == 0 else grad_scale / D
        for t in range(int(cu_span[r]), int(cu_span[r + 1])):
            if source[t] == SRC_STUDENT:
                use_rev = dir_mode in (DIR_IPD, DIR_PURE_REV)
            elif source[t] == SRC_TEACHER:
                use_rev = dir_mode in (DIR_PURE_REV, DIR_INVERSE)
            else:
                continue
            S = np.union1d(topk(l_s[t], K), topk(l_t[t], K))
            log_pi_bar = l_s[t, S] - log_partition(l_s[t, S])
            log_q_bar = l_t[t, S] - log_partition(l_t[t, S])
            pi_bar = np.exp(log_pi_bar)
            q_bar = np.exp(log_q_bar)
            if use_rev:
                d = np.where(pi_bar > 0, log_pi_bar - log_q_bar, 0.0)
                kl = float(np.sum(pi_bar * d))
                g = pi_bar * (d - kl)
            else:
                g = pi_bar - q_bar
            G[t, S] = w * g
    return G


# ----------------------------------------------------------------------------
# seeded sampling: Gumbel-max over counter-based uniforms
# ----------------------------------------------------------------------------
# Training rollouts sample at temperature 1 with top-p 1 (App. A, training
# configuration), i.e. from the full softmax of the logits.  A draw is defined bit-exactly so that any device
# reproduces it:
#   * uniform bits: Philox4x32 with 10 rounds (Salmon, Moraes, Dror and Shaw,
#     "Parallel random numbers: as easy as 1, 2, 3", SC 2011), key = the
#     64-bit seed (low word first), counter = (v // 4, draw low word, draw high
#     word, 0); output word v % 4 belongs to token v;
#   * u_v = (2 * (bits >> 9) + 1) * 2^-24, exactly representable, in (0, 1);
#   * Gumbel-max in base 2: token = argmax_v  l_v * c - lg2(-lg2(u_v)), with
#     c = fp32(log2 e) * inv_temperature; this is argmax_v l_v / temperature +
#     G_v with G_v = -ln(-ln u_v) a standard Gumbel variable, rescaled by
#     log2 e and shifted by the constant log2(ln 2), so the token is
#     distributed as softmax(l / temperature);
#   * lg2 is a fixed fp32 procedure (below), every operation rounded to fp32
#     with no fused multiply-add; ties of the score go to the lower id.
PHILOX_M0, PHILOX_M1 = 0xD2511F53, 0xCD9E8D57     # round multipliers
PHILOX_W0, PHILOX_W1 = 0x9E3779B9, 0xBB67AE85     # key increments (Weyl sequence)
LOG2E_F32_BITS = 0x3FB8AA3B                       # fp32 nearest to log2(e)
# log2(1 + t) = t * P(t) on t in [sqrt(1/2) - 1, sqrt(2) - 1]; P's coefficients
# (lowest degree first) are a least-squares fit of log2(1 + t) / t on 4000
# Chebyshev nodes, rounded to fp32; |lg2(x) - log2(x)| <= 1.1e-6 for normal x
LG2_POLY_BITS = (0x3FB8AA3A, 0xBF38AA93, 0x3EF63BAD, 0xBEB871A3, 0x3E92FB93, 0xBE7ECB25,
                 0x3E6FD4B5, 0xBE15B661)


def _f32(bits) -> np.float32:
    return np.array([bits], dtype=np.uint32).view(np.float32)[0]


def philox4x32_10(ctr: np.ndarray, key) -> np.ndarray:
    """Philox4x32-10 of each counter row ctr[..., 0:4] (uint32) under the key
    (k0, k1): ten rounds; a round multiplies words 0 and 2 by the two
    multipliers and forms (hi(M1 c2) ^ c1 ^ k0, lo(M1 c2), hi(M0 c0) ^ c3 ^ k1,
    lo(M0 c0)); the key is bumped by the Weyl increments between rounds."""
    mask = np.uint64(0xFFFFFFFF)
    c = [np.asarray(ctr[..., i], dtype=np.uint64) for i in range(4)]
    k0, k1 = np.uint64(key[0]) & mask, np.uint64(key[1]) & mask
    for _ in range(10):
        p0 = np.uint64(PHILOX_M0) * c[0]
        p1 = np.uint64(PHILOX_M1) * c[2]
        c = [(p1 >> np.uint64(32)) ^ c[1] ^ k0, p1 & mask,
             (p0 >> np.uint64(32)) ^ c[3] ^ k1, p0 & mask]
        k0 = (k0 + np.uint64(PHILOX_W0)) & mask
        k1 = (k1 + np.uint64(PHILOX_W1)) & mask
    return np.stack(c, axis=-1).astype(np.uint32)


def lg2_f32(x) -> np.ndarray:
    """The fixed fp32 base-2 logarithm of the sampler, for positive normal x:
    x = 2^e m with m in (sqrt(1/2), sqrt(2)] (exact bit operations),
    t = m - 1 (exact), P(t) by Horner's rule, result e + t P(t); each product
    and sum rounded to fp32."""
    x = np.asarray(x, dtype=np.float32)
    b = x.view(np.uint32)
    e = ((b >> np.uint32(23)) & np.uint32(0xFF)).astype(np.int32) - 127
    mb = (b & np.uint32(0x7FFFFF)) | np.uint32(0x3F800000)
    big = mb > np.uint32(0x3FB504F3)                 # m > sqrt(2): halve it
    mb = np.where(big, mb - np.uint32(0x00800000), mb).astype(np.uint32)
    e = e + big.astype(np.int32)
    t = mb.view(np.float32) - np.float32(1.0)
    coef = [_f32(c) for c in LG2_POLY_BITS]
    p = np.full(t.shape, coef[-1], dtype=np.float32)
    for c in coef[-2::-1]:
        p = (p * t).astype(np.float32) + c
    return (e.astype(np.float32) + (t * p).astype(np.float32)).astype(np.float32)


def sample_uniforms(vocab: int, seed: int, draw: int) -> np.ndarray:
    """u_v for v in [0, vocab) of one draw (fp32)."""
    mask = 0xFFFFFFFF
    groups = (vocab + 3) // 4
    ctr = np.zeros((groups, 4), dtype=np.uint32)
    ctr[:, 0] = np.arange(groups, dtype=np.uint32)
    ctr[:, 1] = draw & mask
    ctr[:, 2] = (draw >> 32) & mask
    bits = philox4x32_10(ctr, (seed & mask, (seed >> 32) & mask)).reshape(-1)[:vocab]
    return ((bits >> np.uint32(9)).astype(np.float32) * np.float32(2.0) + np.float32(1.0)) * \
        np.float32(2.0 ** -24)


def gumbel_scores(l_bits, seed: int, draw: int, inv_temperature: float = 1.0) -> np.ndarray:
    """Per-token scores l_v c - lg2(-lg2 u_v) of one draw, fp32."""
    l = bf16_to_f64(l_bits).astype(np.float32)      # exact
    c = _f32(LOG2E_F32_BITS) * np.float32(inv_temperature)
    u = sample_uniforms(len(l), seed, draw)
    e = -lg2_f32(u)
    return (l * c).astype(np.float32) - lg2_f32(e)


def sample_token(l_bits, seed: int, draw: int, inv_temperature: float = 1.0) -> int:
    """One token drawn from softmax(l / temperature); ties to the lower id."""
    return int(np.argmax(gumbel_scores(l_bits, seed, draw, inv_temperature)))


def next_token_after_verdict(logits_s_bits, logits_t_bits, cu_span, prefix_len, verdict_out,
                             seed: int, draw_base, inv_temperature: float = 1.0) -> np.ndarray:
    """The first token of each request's next span when the verify step
    already holds the logits it is drawn from.

    After the verdict the accepted prefix ends at position P_r + n_r (n_r
    emitted tokens), and the next token is drawn by the next driver from its
    distribution at that position.  After a takeover at j (student span) the
    teacher regenerates position j, whose distribution is the teacher's row j of
    the span; after a handback at j (teacher span) the student continues at
    position j + 1, its row j + 1 -- in both cases the next driver's row
    n_r (Sec. 3.2.3, verdict stage).  With n_r = k_r (no transition) that row is not part of the step and
    with done set the request has ended: -1.  The draw number is
    draw_base[r] + P_r + n_r (the absolute position of the drawn token)."""
    R = len(cu_span) - 1
    out = np.full(R, -1, dtype=np.int64)
    for r in range(R):
        t0, t1 = int(cu_span[r]), int(cu_span[r + 1])
        n = int(verdict_out["n_emit"][r])
        if int(verdict_out["done"][r]) or n >= t1 - t0:
            continue
        rows = logits_t_bits if int(verdict_out["next_driver"][r]) == 1 else logits_s_bits
        draw = (int(draw_base[r]) + int(prefix_len[r]) + n) & 0xFFFFFFFFFFFFFFFF
        out[r] = sample_token(rows[t0 + n], seed, draw, inv_temperature)
    return out
