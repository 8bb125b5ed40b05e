"""KV append on the GPU vs the oracle (needs a GB300): the whole page pools
after the append must be identical, bit for bit."""
import numpy as np
import pytest
import torch

import oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import ipd
    return ipd


def _case(seed, hkv, old_len, n_new, spare=5):
    rng = np.random.default_rng(seed)
    L = [a + b for a, b in zip(old_len, n_new)]
    R = len(L)
    max_pages = max(1, max((x + 15) // 16 for x in L))
    num_pages = sum((x + 15) // 16 for x in L) + spare
    perm = rng.permutation(num_pages)
    table = np.full((R, max_pages), -1, dtype=np.int32)
    used = 0
    for r, x in enumerate(L):
        for j in range((x + 15) // 16):
            table[r, j] = perm[used]; used += 1
    kp = rng.integers(0, 1 << 16, size=(num_pages, hkv, 16, 128), dtype=np.uint16)
    vp = rng.integers(0, 1 << 16, size=(num_pages, hkv, 16, 128), dtype=np.uint16)
    cu = np.concatenate([[0], np.cumsum(n_new)]).astype(np.int32)
    kn = rng.integers(0, 1 << 16, size=(int(cu[-1]), hkv, 128), dtype=np.uint16)
    vn = rng.integers(0, 1 << 16, size=(int(cu[-1]), hkv, 128), dtype=np.uint16)
    return kp, vp, kn, vn, cu, np.array(L, dtype=np.int32), table


def _t(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16) if a.dtype == np.uint16 else
                            np.ascontiguousarray(a)).cuda()


def _run(lib, kp, vp, kn, vn, cu, L, table):
    from paper_2609_36546_gb300.ipd import KVCache
    cache = KVCache(_t(kp).view(torch.bfloat16), _t(vp).view(torch.bfloat16))
    lib.kv_append(cache, _t(kn).view(torch.bfloat16), _t(vn).view(torch.bfloat16), _t(cu), _t(L),
                  _t(table))
    torch.cuda.synchronize()
    return (cache.k_pages.view(torch.int16).cpu().numpy().view(np.uint16),
            cache.v_pages.view(torch.int16).cpu().numpy().view(np.uint16))


@pytest.mark.parametrize("hkv,old_len,n_new", [
    (4, [100, 7, 0, 31, 64], [8, 8, 8, 1, 16]),            # teacher-shaped spans, page crossings
    (8, [1000, 15, 16, 300], [1, 1, 1, 1]),                # student decode appends
    (2, [3, 50, 0], [0, 17, 33]),                          # an empty request, multi-page spans
])
def test_kv_append_bit_exact(lib, hkv, old_len, n_new):
    case = _case(hkv, hkv, old_len, n_new)
    got_k, got_v = _run(lib, *case)
    assert lib.device_error() == 0
    exp_k, exp_v = O.kv_append(*case[:4], case[4], case[5], case[6])
    assert np.array_equal(got_k, exp_k) and np.array_equal(got_v, exp_v)


def test_kv_append_bad_page_is_recorded_and_skipped(lib):
    kp, vp, kn, vn, cu, L, table = _case(3, 4, [20, 40], [2, 3])
    bad = table.copy()
    bad[1, (L[1] - 1) // 16] = kp.shape[0] + 7            # outside the pool
    got_k, got_v = _run(lib, kp, vp, kn, vn, cu, L, bad)
    assert lib.device_error() == 1                         # IPD_DEVERR_PAGE_ID
    # request 0 is appended; request 1's rows that map to the bad page are skipped
    exp_k, exp_v = O.kv_append(kp, vp, kn[:2], vn[:2], cu[:2], L[:1], table[:1])
    assert np.array_equal(got_k, exp_k) and np.array_equal(got_v, exp_v)


def test_kv_append_rows_past_the_offsets_are_skipped(lib):
    """total_new counts five rows but cu_new ends at three: rows 3 and 4
    belong to no request and must not be written anywhere (recorded as
    IPD_DEVERR_SPAN); rows 0-2 land where the offsets place them."""
    kp, vp, kn, vn, cu, L, table = _case(5, 4, [20, 40], [2, 3])
    short = np.array([0, 2, 3], dtype=np.int32)     # request 1 owns only row 2
    got_k, got_v = _run(lib, kp, vp, kn, vn, short, L, table)
    assert lib.device_error() == 6                   # IPD_DEVERR_SPAN
    exp_k, exp_v = O.kv_append(kp, vp, kn[:3], vn[:3], short, L, table)
    assert np.array_equal(got_k, exp_k) and np.array_equal(got_v, exp_v)


def test_kv_append_many_equals_one_by_one_and_oracle(lib):
    """The appends of one step (span rows into two caches of different head
    counts, decode rows into both) in one launch: every pool bit-identical
    to the oracle and to the appends made one call at a time."""
    from paper_2609_36546_gb300.ipd import KVCache
    cases = [_case(11, 4, [100, 7, 0, 31], [8, 8, 8, 1]),     # teacher cache, span rows
             _case(12, 8, [1000, 15, 16, 300], [1, 1, 1, 1]),  # student cache, decode rows
             _case(13, 2, [3, 50, 0], [0, 17, 33])]            # an empty request, multi-page
    def devs():
        out = []
        for kp, vp, kn, vn, cu, L, table in cases:
            cache = KVCache(_t(kp).view(torch.bfloat16), _t(vp).view(torch.bfloat16))
            out.append((cache, _t(kn).view(torch.bfloat16), _t(vn).view(torch.bfloat16), _t(cu),
                        _t(L), _t(table)))
        return out
    many = devs()
    lib.kv_append_many(many)
    single = devs()
    for a in single:
        lib.kv_append(*a)
    torch.cuda.synchronize()
    assert lib.device_error() == 0
    for (kp, vp, kn, vn, cu, L, table), m, o in zip(cases, many, single):
        exp_k, exp_v = O.kv_append(kp, vp, kn, vn, cu, L, table)
        got_k = m[0].k_pages.view(torch.int16).cpu().numpy().view(np.uint16)
        got_v = m[0].v_pages.view(torch.int16).cpu().numpy().view(np.uint16)
        assert np.array_equal(got_k, exp_k) and np.array_equal(got_v, exp_v)
        assert torch.equal(m[0].k_pages.view(torch.int16), o[0].k_pages.view(torch.int16))
        assert torch.equal(m[0].v_pages.view(torch.int16), o[0].v_pages.view(torch.int16))
