"""Seeded sampling on the GPU vs the oracle (needs a GB300).

The draw is defined bit-exactly (Philox4x32-10 uniforms, a fixed fp32 lg2,
every operation rounded on its own), so the sampled ids must be identical.
"""
import numpy as np
import pytest
import torch

import ipd_synth as S
import oracle as O
from tests.parity import u16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import ipd
    return ipd


def _gpu_sample(lib, rows, seed, draws, inv_t):
    n, V = rows.shape
    d = rows.cuda()
    tok = torch.full((n,), -7, device="cuda", dtype=torch.int32)
    ws = torch.empty(lib.sample_workspace_size(n, V), device="cuda", dtype=torch.uint8)
    dr = torch.from_numpy(np.asarray(draws, dtype=np.uint64).view(np.int64)).cuda()
    lib.sample(d, seed, dr, tok, ws, inv_t)
    torch.cuda.synchronize()
    return tok.cpu().numpy()


@pytest.mark.parametrize("V,n,inv_t", [(4096, 40, 1.0), (4096, 16, 0.7), (151936, 6, 1.0),
                                       (8, 64, 1.0), (8200, 5, 2.0)])
def test_sample_rows_bit_exact(lib, V, n, inv_t):
    g = torch.Generator().manual_seed(V + n)
    rows = (torch.randn(n, V, generator=g) * 2.5).to(torch.bfloat16)
    rng = np.random.default_rng(V)
    draws = rng.integers(0, 2 ** 63, size=n, dtype=np.int64).astype(np.uint64) * np.uint64(2) + \
        np.uint64(1)                                    # high bits set
    seed = 0xDEADBEEF12345678
    got = _gpu_sample(lib, rows, seed, draws, inv_t)
    bits = u16(rows)
    exp = [O.sample_token(bits[i], seed, int(draws[i]), inv_t) for i in range(n)]
    assert got.tolist() == exp


def test_sample_degenerate_rows(lib):
    V = 4096
    rows = torch.zeros(4, V, dtype=torch.bfloat16)
    rows[1] = float("-inf")
    rows[1, 1234] = 0.0                                 # the only finite logit always wins
    rows[2] = float("-inf")                             # all -inf: every score ties, id 0
    rows[3, 4095] = 100.0                               # one overwhelming logit
    draws = np.arange(4, dtype=np.uint64)
    got = _gpu_sample(lib, rows, 7, draws, 1.0)
    exp = [O.sample_token(u16(rows)[i], 7, i, 1.0) for i in range(4)]
    assert got.tolist() == exp
    assert got[1] == 1234 and got[2] == 0 and got[3] == 4095


def test_sample_many_draws_of_one_row(lib):
    """Different draw numbers of one row give independent draws; the ids follow
    the oracle draw by draw."""
    V, n = 64, 512
    l = (torch.arange(V, dtype=torch.float32) / 16.0).to(torch.bfloat16)
    rows = l.unsqueeze(0).repeat(n, 1)
    draws = np.arange(1000, 1000 + n, dtype=np.uint64)
    got = _gpu_sample(lib, rows, 3, draws, 1.0)
    bits = u16(rows[0])
    assert got.tolist() == [O.sample_token(bits, 3, int(d), 1.0) for d in draws]
    assert len(set(got.tolist())) > 10


def _tokens_mixed(ls, lt, cu, driver, K):
    T = ls.shape[0]
    tokens = np.zeros(T, dtype=np.int32)
    for t in range(T):
        r = int(np.searchsorted(cu, t, side="right") - 1)
        ver = ls[t] if driver[r] else lt[t]
        order = torch.argsort(ver.float(), descending=True, stable=True)
        i = t - int(cu[r])
        tokens[t] = int(order[(3 * i) % K]) if i < 3 else int(order[K + 50 + t])
    return tokens


@pytest.mark.parametrize("V", [4096, 151936])
def test_next_token_after_verdict(lib, V):
    spec = S.small_spec(n_req=12, ctx=(20, 600), span=(1, 10), vocab=V, sigma=2.5)
    w = S.make_workload(spec, seed=61, device="cpu")
    ls, lt = w.logits_s, w.logits_t
    cu, drv, pre = w.cu_span.numpy(), w.driver.numpy(), w.prefix_len.numpy()
    R, T, K = len(cu) - 1, int(cu[-1]), w.spec.K
    tokens = _tokens_mixed(ls, lt, cu, drv, K)
    # one teacher-driven request ends on its first (emitted) token
    tdr = [r for r in range(R) if drv[r] == 1 and cu[r + 1] > cu[r]]
    eos = int(tokens[cu[tdr[0]]]) if tdr else -1
    seed = 0x0123456789ABCDEF
    base = (np.arange(R, dtype=np.uint64) << np.uint64(40)) + np.uint64(17)
    dev = "cuda"
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(device=dev, dtype=dt)
    out = lib.alloc_score_outputs(R, T, dev)
    ws = torch.empty(lib.score_workspace_size(R, T, V, K), device=dev, dtype=torch.uint8)
    nxt = torch.full((R,), -7, device=dev, dtype=torch.int32)
    lib.score_span_ex(ls.to(dev), lt.to(dev), t(tokens, torch.int32), t(cu, torch.int32),
                      t(drv, torch.uint8), t(pre, torch.int32), K, eos, out, ws,
                      next_token=nxt, draw_base=t(base.view(np.int64), torch.int64),
                      sample_seed=seed)
    torch.cuda.synchronize()
    assert lib.device_error() == 0
    o = O.score_span(u16(ls), u16(lt), tokens, cu, drv, pre, K, eos)
    exp = O.next_token_after_verdict(u16(ls), u16(lt), cu, pre, o, seed, base)
    got = nxt.cpu().numpy()
    same = [r for r in range(R) if all(int(out[f][r].item()) == int(o[f][r])
                                       for f in ("n_emit", "next_driver", "done"))]
    assert len(same) >= R - 1
    assert [int(got[r]) for r in same] == [int(exp[r]) for r in same]
    assert (exp >= 0).sum() >= 4 and (exp == -1).sum() >= 1
    if tdr:
        assert o["done"][tdr[0]] == 1 and got[tdr[0]] == -1
