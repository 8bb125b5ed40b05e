"""Gradient of the source-split objective on the GPU vs the fp64 oracle
(needs a GB300).

The oracle's own verdict (source labels, emitted counts) is uploaded and fed
to both sides, so the comparison isolates the gradient.  Tolerance per
element: 3e-5 w_t + 1e-4 |ref|, with w_t the position's weight in the
objective.  The fp32 path forms log pi_bar - log q_bar - KL from values of
magnitude <= ~30 (a few ulp each, ~1e-5 absolute) and multiplies by
pi_bar <= 1, whose own relative error is ~1e-6 per unit of |log pi_bar|.
The support (ids) is exact: it is the exact top-K of both rows.  The dense
fp32 form is the sparse one scattered into zeros, bit for bit; the bf16 form
is its round-to-nearest-even.
"""
import numpy as np
import pytest
import torch

import ipd_synth as S
import oracle as O
from tests.parity import u16

pytestmark = pytest.mark.gpu

G_ATOL, G_RTOL = 3e-5, 1e-4


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import ipd
    return ipd


def _bf16_to_f32_bits(x16):
    return (x16.astype(np.uint32) << 16).view(np.float32)


def _rne_bf16(x):
    return O.bf16_to_f64(O.f64_to_bf16(np.asarray(x, dtype=np.float64)))


def _case(lib, ls, lt, tokens, cu, driver, prefix, K, agg, dmode, resp_len, scale, dense_dtypes):
    """Runs the GPU chain (score -> loss -> grad) on the oracle's verdict and
    returns the GPU outputs and the oracle's gradient."""
    dev = "cuda"
    T, V = ls.shape
    R = len(cu) - 1
    o = O.score_span(u16(ls), u16(lt), tokens, cu, driver, prefix, K)
    src = o["source"].astype(np.uint8)
    n_emit = o["n_emit"].astype(np.int32)
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(device=dev, dtype=dt)
    d_ls, d_lt = ls.to(dev), lt.to(dev)
    d_tok, d_cu = t(tokens, torch.int32), t(cu, torch.int32)
    d_drv, d_pre = t(driver, torch.uint8), t(prefix, torch.int32)
    out = lib.alloc_score_outputs(R, T, dev)
    ws = torch.empty(lib.score_workspace_size(R, T, V, K), device=dev, dtype=torch.uint8)
    tks = torch.full((T, K), -7, device=dev, dtype=torch.int32)
    tkt = torch.full((T, K), -7, device=dev, dtype=torch.int32)
    lib.score_span_ex(d_ls, d_lt, d_tok, d_cu, d_drv, d_pre, K, -1, out, ws, topk_s=tks, topk_t=tkt)
    d_src, d_ne = t(src, torch.uint8), t(n_emit, torch.int32)
    d_rl = None if resp_len is None else t(resp_len, torch.int32)
    out8 = torch.empty(8, device=dev)
    lib.split_loss(out["kl_rev"], out["kl_fwd"], d_src, d_cu, d_ne, d_rl, agg, dmode, out8)
    gi = torch.full((T, 2 * K), 123, device=dev, dtype=torch.int32)
    gv = torch.full((T, 2 * K), 9.0, device=dev)
    lib.split_loss_grad(d_ls, d_lt, tks, tkt, d_src, d_cu, d_ne, d_rl, out8, K, agg, dmode, scale,
                        gi, gv)
    dense = {}
    for dt in dense_dtypes:
        gd = torch.full((T, V), 7.0, device=dev, dtype=dt)
        gi2 = torch.empty_like(gi); gv2 = torch.empty_like(gv)
        lib.split_loss_grad(d_ls, d_lt, tks, tkt, d_src, d_cu, d_ne, d_rl, out8, K, agg, dmode,
                            scale, gi2, gv2, gd)
        dense[dt] = gd
    torch.cuda.synchronize()
    assert lib.device_error() == 0
    ref = O.split_loss_grad(O.bf16_to_f64(u16(ls)), O.bf16_to_f64(u16(lt)), src, cu, n_emit,
                            resp_len, K, agg, dmode, grad_scale=scale)
    dens = n_emit if resp_len is None else resp_len
    if agg == 0:
        D = float(sum(1 for d in dens if d > 0))
    else:
        D = float(sum(d for d in dens if d > 0))
    w = np.zeros(T)
    for r in range(R):
        if dens[r] > 0:
            w[cu[r]:cu[r + 1]] = abs(scale) / (D * dens[r] if agg == 0 else D)
    return dict(topk_s=tks.cpu().numpy(), topk_t=tkt.cpu().numpy(), gi=gi.cpu().numpy(),
                gv=gv.cpu().numpy(), dense={k: v.cpu() for k, v in dense.items()}, ref=ref,
                src=src, w=w)


def _check(g, ls, lt, K):
    T, V = ls.shape
    ref = g["ref"]
    lsf, ltf = O.bf16_to_f64(u16(ls)), O.bf16_to_f64(u16(lt))
    for t in range(T):
        es, et = O.topk(lsf[t], K), O.topk(ltf[t], K)
        assert np.array_equal(g["topk_s"][t], es), t
        assert np.array_equal(g["topk_t"][t], et), t
        emitted = g["src"][t] != O.SRC_DISCARDED and g["w"][t] > 0
        if not emitted:
            assert (g["gi"][t] == -1).all() and (g["gv"][t] == 0).all(), t
            assert (ref[t] == 0).all()
            continue
        exp_ids = np.concatenate([es, np.where(np.isin(et, es), -1, et)])
        assert np.array_equal(g["gi"][t], exp_ids), t
        on = exp_ids >= 0
        tol = G_ATOL * g["w"][t] + G_RTOL * np.abs(ref[t, exp_ids[on]])
        err = np.abs(g["gv"][t][on] - ref[t, exp_ids[on]])
        assert np.all(err <= tol), (t, err.max(), tol.min())
        assert (g["gv"][t][~on] == 0).all()
        # every nonzero of the oracle lies on the support
        assert set(np.flatnonzero(ref[t]).tolist()) <= set(exp_ids[on].tolist())
    for dt, gd in g["dense"].items():
        exp = np.zeros((T, V), dtype=np.float32)
        for t in range(T):
            on = g["gi"][t] >= 0
            exp[t, g["gi"][t][on]] = g["gv"][t][on]
        if dt == torch.float32:
            assert np.array_equal(gd.numpy().view(np.uint32), exp.view(np.uint32))
        else:
            got = _bf16_to_f32_bits(gd.view(torch.int16).numpy().view(np.uint16))
            assert np.array_equal(got, _rne_bf16(exp).astype(np.float32))


def _tokens_mixed(ls, lt, cu, driver, K):
    """Proposed tokens that the verifier covers for the first positions of
    each span and not afterwards, so that both sources get emitted."""
    T = ls.shape[0]
    tokens = np.zeros(T, dtype=np.int32)
    for t in range(T):
        r = int(np.searchsorted(cu, t, side="right") - 1)
        ver = ls[t] if driver[r] else lt[t]
        order = torch.argsort(ver.float(), descending=True, stable=True)
        i = t - int(cu[r])
        tokens[t] = int(order[(3 * i) % K]) if i < 3 else int(order[K + 50 + t])
    return tokens


MODES = [(0, 0, False, 1.0), (1, 0, True, 1.0), (0, 1, True, -2.0), (1, 2, False, 0.5),
         (0, 3, True, 1.0)]


@pytest.mark.parametrize("agg,dmode,use_len,scale", MODES)
def test_grad_matches_oracle_small(lib, agg, dmode, use_len, scale):
    spec = S.small_spec(n_req=10, ctx=(20, 600), span=(1, 12), vocab=4096, sigma=2.5)
    w = S.make_workload(spec, seed=51 + dmode, device="cpu")
    ls, lt = w.logits_s, w.logits_t
    cu = w.cu_span.numpy(); R = len(cu) - 1
    rng = np.random.default_rng(dmode)
    resp_len = rng.integers(0, 40, size=R).astype(np.int32) if use_len else None
    if resp_len is not None:
        resp_len[0] = 0                       # a request left out of the batch mean
    K = w.spec.K
    tokens = _tokens_mixed(ls, lt, cu, w.driver.numpy(), K)
    g = _case(lib, ls, lt, tokens, cu, w.driver.numpy(), w.prefix_len.numpy(), K, agg, dmode,
              resp_len, scale, (torch.float32, torch.bfloat16))
    assert (g["src"] == O.SRC_STUDENT).any() and (g["src"] == O.SRC_TEACHER).any()
    _check(g, ls, lt, K)


def test_grad_full_vocabulary_rows(lib):
    """V = 151,936 rows with mixed drivers; ragged spans; the dense forms span
    many chunks and end on a ragged one."""
    gen = torch.Generator().manual_seed(77)
    V, K = 151936, 16
    spans = [8, 3, 1, 8, 5]
    cu = np.concatenate([[0], np.cumsum(spans)]).astype(np.int32)
    T = int(cu[-1])
    lt = (torch.randn(T, V, generator=gen) * 3.0).to(torch.bfloat16)
    ls = (lt.float() * 0.8 + torch.randn(T, V, generator=gen) * 1.5).to(torch.bfloat16)
    driver = np.array([0, 1, 0, 1, 0], dtype=np.uint8)
    tokens = _tokens_mixed(ls, lt, cu, driver, K)
    g = _case(lib, ls, lt, tokens, cu, driver, np.full(5, 100, dtype=np.int32), K, 0, 0, None,
              1.0, (torch.float32, torch.bfloat16))
    assert (g["src"] == O.SRC_STUDENT).any() and (g["src"] == O.SRC_TEACHER).any()
    _check(g, ls, lt, K)
