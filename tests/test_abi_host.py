"""The C ABI on the host: the library loads, exports every function that
include/ipd.h declares, and rejects bad arguments before launching anything
(these calls never reach the GPU)."""
import ctypes
import os
import re

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ipd.h")


@pytest.fixture(scope="module")
def ipd():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import ipd as m
    return m


def _header_functions():
    src = open(os.path.join(ROOT, "include", "ipd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ipd_[a-z_0-9]+)\s*\(", src)))


def test_library_exports_every_declared_function(ipd):
    names = _header_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(ipd.lib(), n), n
    assert sorted(ipd.EXPORTS) == names


def test_status_strings_and_version(ipd):
    """Every status code the header defines has its own name."""
    with open(HEADER) as f:
        codes = dict((n, int(v)) for n, v in
                     re.findall(r"#define\s+(IPD_OK|IPD_ERR_[A-Z_]+)\s+(\d+)", f.read()))
    assert len(codes) >= 8 and codes["IPD_ERR_CAPACITY"] == 7
    for name, v in codes.items():
        assert ipd.lib().ipd_status_string(v) == name.encode(), name
        assert ipd.STATUS_CODES[name] == v
    assert ipd.lib().ipd_status_string(99) == b"IPD_ERR_UNKNOWN"
    assert ipd.lib().ipd_status_string(-1) == b"IPD_ERR_UNKNOWN"
    assert ipd.lib().ipd_version() == 100


def _fake_batch(ipd, hd=128, ps=16, hkv=4, hq=32, R=2, maxq=4, maxs=100):
    c = ipd._KVCache(16, 16, 10, ps, hkv, hd)
    b = ipd._AttnBatch(ctypes.pointer(c), hq, R, 16, 16, 16, 16, (maxs + 15) // 16, R * maxq,
                       maxq, maxs, 16)
    return c, b


def test_attn_host_validation(ipd):
    L = ipd.lib()
    c, b = _fake_batch(ipd)
    arr = (ipd._AttnBatch * 1)(b)
    assert L.ipd_attn_workspace_size(arr, 1, None, 0) > 0
    # too small a workspace is refused before any device call
    assert L.ipd_verify_attn(arr, 1, None, 0, 0.088, 256, 16, None) == ipd.STATUS_CODES["IPD_ERR_WORKSPACE"]
    for kw, code in ((dict(hd=64), "IPD_ERR_UNSUPPORTED"), (dict(ps=32), "IPD_ERR_UNSUPPORTED"),
                     (dict(hq=30), "IPD_ERR_INVALID_ARG"), (dict(maxs=2, maxq=4), "IPD_ERR_INVALID_ARG")):
        c2, b2 = _fake_batch(ipd, **kw)
        a2 = (ipd._AttnBatch * 1)(b2)
        assert L.ipd_verify_attn(a2, 1, None, 0, 0.088, 256, 1 << 30, None) == ipd.STATUS_CODES[code], kw
        assert L.ipd_attn_workspace_size(a2, 1, None, 0) == 0
    many = (ipd._AttnBatch * 9)(*([b] * 9))
    assert L.ipd_verify_attn(many, 9, None, 0, 0.088, 256, 1 << 30, None) == ipd.STATUS_CODES["IPD_ERR_INVALID_ARG"]
    assert L.ipd_verify_attn(arr, 1, None, 0, -1.0, 256, 1 << 30, None) == ipd.STATUS_CODES["IPD_ERR_INVALID_ARG"]
    # no batches at all: nothing to do
    assert L.ipd_verify_attn(None, 0, None, 0, 0.088, None, 0, None) == 0


def test_score_and_loss_host_validation(ipd):
    L = ipd.lib()
    p = [16] * 6
    outs = [16] * 13
    bad = ipd.STATUS_CODES
    args = lambda R, T, V, K: p + [R, T, V, K, -1] + outs + [16, 1 << 30, None]
    assert L.ipd_score_span(*args(2, 4, 4096, 33)) == bad["IPD_ERR_UNSUPPORTED"]
    assert L.ipd_score_span(*args(2, 4, 4096, 0)) == bad["IPD_ERR_UNSUPPORTED"]
    assert L.ipd_score_span(*args(2, 4, 4100, 16)) == bad["IPD_ERR_UNSUPPORTED"]
    assert L.ipd_score_span(*args(2, 4, 8, 16)) == bad["IPD_ERR_UNSUPPORTED"]
    assert L.ipd_score_span(*args(-1, 4, 4096, 16)) == bad["IPD_ERR_INVALID_ARG"]
    small_ws = p + [2, 4, 4096, 16, -1] + outs + [16, 8, None]
    assert L.ipd_score_span(*small_ws) == bad["IPD_ERR_WORKSPACE"]
    assert L.ipd_score_workspace_size(2, 4, 4096, 16) >= 8 * 2 * 4
    assert L.ipd_loss_workspace_size(10) == 0
    assert L.ipd_split_loss(16, 16, 16, 16, 16, None, 3, 2, 0, 16, None, 0, None) == bad["IPD_ERR_INVALID_ARG"]
    assert L.ipd_split_loss(16, 16, 16, 16, 16, None, 3, 0, 7, 16, None, 0, None) == bad["IPD_ERR_INVALID_ARG"]
    assert L.ipd_split_loss(16, 16, 16, 16, 16, None, 3, 0, 0, None, None, 0, None) == bad["IPD_ERR_INVALID_ARG"]


def test_score_ext_rejects_bad_rules_on_the_host():
    import ctypes
    from paper_2609_36546_gb300 import ipd
    for take, hand, tt in ((7, 0, 0.0), (0, -1, 0.0), (1, 0, float("nan"))):
        ext = ipd._ScoreExt(take, hand, tt, 0.0, None, None, None)
        st = ipd._lib.ipd_score_span_ex(*([None] * 6), 0, 0, 4096, 16, -1, *([None] * 13),
                                        ctypes.byref(ext), None, 0, None)
        assert st == ipd.STATUS_CODES["IPD_ERR_INVALID_ARG"]
    # full KL: host validation only
    assert ipd._lib.ipd_full_kl(None, None, 0, 4096, None, None, None) == 0
    assert ipd._lib.ipd_full_kl(None, None, 3, 4095, None, None, None) == \
        ipd.STATUS_CODES["IPD_ERR_UNSUPPORTED"]
    assert ipd._lib.ipd_full_kl(None, None, 3, 4096, None, None, None) == \
        ipd.STATUS_CODES["IPD_ERR_INVALID_ARG"]


def test_loss_grad_host_validation():
    from paper_2609_36546_gb300 import ipd
    L = ipd._lib
    bad = ipd.STATUS_CODES

    def call(R=2, T=4, V=4096, K=16, agg=0, dmode=0, scale=1.0, gi=16, gv=16, dense=None,
             dtype=0, ptr=16):
        return L.ipd_split_loss_grad(*([ptr] * 9), R, T, V, K, agg, dmode, scale, gi, gv, dense,
                                     dtype, None, 0, None)

    assert L.ipd_loss_grad_workspace_size(100, 16) == 0
    assert call(T=0, ptr=None, gi=None, gv=None) == 0           # nothing to do
    assert call(K=33) == bad["IPD_ERR_UNSUPPORTED"]
    assert call(K=0) == bad["IPD_ERR_UNSUPPORTED"]
    assert call(V=8, K=16) == bad["IPD_ERR_UNSUPPORTED"]
    assert call(agg=2) == bad["IPD_ERR_INVALID_ARG"]
    assert call(dmode=4) == bad["IPD_ERR_INVALID_ARG"]
    assert call(scale=float("nan")) == bad["IPD_ERR_INVALID_ARG"]
    assert call(scale=float("inf")) == bad["IPD_ERR_INVALID_ARG"]
    assert call(dense=32, dtype=2) == bad["IPD_ERR_INVALID_ARG"]
    assert call(dense=40) == bad["IPD_ERR_INVALID_ARG"]          # not 16-byte aligned
    assert call(gi=None) == bad["IPD_ERR_INVALID_ARG"]
    assert call(R=0) == bad["IPD_ERR_INVALID_ARG"]                # positions without requests
    assert call(R=-1) == bad["IPD_ERR_INVALID_ARG"]


def test_sample_host_validation():
    import ctypes
    from paper_2609_36546_gb300 import ipd
    L = ipd._lib
    bad = ipd.STATUS_CODES
    ws = 1 << 20
    assert L.ipd_sample_workspace_size(4, 151936) == 2 * 2048 * 8
    assert L.ipd_sample_workspace_size(3000, 4096) == 2 * 3000 * 8
    assert L.ipd_sample(None, 0, 4096, 1, None, 1.0, None, None, 0, None) == 0
    assert L.ipd_sample(16, 4, 4100, 1, None, 1.0, 16, 16, ws, None) == bad["IPD_ERR_UNSUPPORTED"]
    for it in (0.0, -1.0, float("inf"), float("nan")):
        assert L.ipd_sample(16, 4, 4096, 1, None, it, 16, 16, ws, None) == bad["IPD_ERR_INVALID_ARG"]
    assert L.ipd_sample(24, 4, 4096, 1, None, 1.0, 16, 16, ws, None) == bad["IPD_ERR_INVALID_ARG"]
    assert L.ipd_sample(16, 4, 4096, 1, None, 1.0, 16, 16, 8, None) == bad["IPD_ERR_WORKSPACE"]
    # the draw after the verdict needs a positive, finite inverse temperature
    ext = ipd._ScoreExt(0, 0, 0.0, 0.0, None, None, None, None, None, 16, None, 5, 0.0)
    st = L.ipd_score_span_ex(*([None] * 6), 0, 0, 4096, 16, -1, *([None] * 13),
                             ctypes.byref(ext), None, 0, None)
    assert st == bad["IPD_ERR_INVALID_ARG"]


def test_kv_append_host_validation():
    from paper_2609_36546_gb300 import ipd
    L = ipd._lib
    bad = ipd.STATUS_CODES
    p = 16
    ok_args = lambda **kw: [kw.get("kp", p), p, kw.get("np", 100), kw.get("hkv", 4),
                            kw.get("ps", 16), kw.get("hd", 128), kw.get("kn", p), p, p, p, p,
                            kw.get("mp", 8), kw.get("R", 2), kw.get("n", 3), None]
    assert L.ipd_kv_append(*ok_args(n=0)) == 0
    assert L.ipd_kv_append(*ok_args(ps=32)) == bad["IPD_ERR_UNSUPPORTED"]
    assert L.ipd_kv_append(*ok_args(hd=64)) == bad["IPD_ERR_UNSUPPORTED"]
    assert L.ipd_kv_append(*ok_args(hkv=0)) == bad["IPD_ERR_INVALID_ARG"]
    assert L.ipd_kv_append(*ok_args(R=0)) == bad["IPD_ERR_INVALID_ARG"]
    assert L.ipd_kv_append(*ok_args(kp=None)) == bad["IPD_ERR_INVALID_ARG"]
    assert L.ipd_kv_append(*ok_args(kn=24)) == bad["IPD_ERR_INVALID_ARG"]   # misaligned
    assert L.ipd_kv_append(*ok_args(np=-1)) == bad["IPD_ERR_INVALID_ARG"]


def test_kv_append_many_host_validation():
    """Every descriptor is checked before anything launches (no GPU: every
    case returns before a launch)."""
    import ctypes
    from paper_2609_36546_gb300 import ipd
    L = ipd._lib
    bad = ipd.STATUS_CODES
    D = ipd._KvAppendDesc
    p = 16

    def desc(**kw):
        return D(kw.get("kp", p), p, kw.get("np", 100), kw.get("hkv", 4), kw.get("ps", 16),
                 kw.get("hd", 128), p, p, p, p, p, kw.get("mp", 8), kw.get("R", 2),
                 kw.get("n", 3))

    def call(*ds, n=None):
        arr = (D * max(len(ds), 1))(*ds)
        return L.ipd_kv_append_many(arr, len(ds) if n is None else n, None)

    assert call() == 0                                     # nothing to append
    assert call(desc(n=0), desc(n=0)) == 0                 # only empty appends: no launch
    assert L.ipd_kv_append_many(None, 0, None) == 0
    assert L.ipd_kv_append_many(None, 1, None) == bad["IPD_ERR_INVALID_ARG"]
    assert call(desc(n=0), n=-1) == bad["IPD_ERR_INVALID_ARG"]
    assert call(*[desc(n=0)] * 9) == bad["IPD_ERR_INVALID_ARG"]   # more than IPD_MAX_BATCHES
    # one bad descriptor among good ones fails the call, whatever its place
    assert call(desc(n=0), desc(ps=32)) == bad["IPD_ERR_UNSUPPORTED"]
    assert call(desc(hd=64), desc(n=0)) == bad["IPD_ERR_UNSUPPORTED"]
    assert call(desc(n=0), desc(kp=None)) == bad["IPD_ERR_INVALID_ARG"]
    assert call(desc(n=0), desc(R=0)) == bad["IPD_ERR_INVALID_ARG"]
    assert call(desc(np=-1)) == bad["IPD_ERR_INVALID_ARG"]
    # the binding's struct has the C layout (plain C compile of the header)
    import os, shutil, subprocess, tempfile
    if shutil.which("gcc"):
        inc = os.path.join(ROOT, "include")
        src = ('#include <stdio.h>\n#include <stddef.h>\n#include "ipd.h"\n'
               'int main(void) { printf("%zu %zu %zu", sizeof(ipd_kv_append_desc), '
               'offsetof(ipd_kv_append_desc, k_new), offsetof(ipd_kv_append_desc, total_new)); '
               'return 0; }\n')
        with tempfile.TemporaryDirectory() as d:
            c, exe = os.path.join(d, "l.c"), os.path.join(d, "l")
            open(c, "w").write(src)
            subprocess.check_call(["gcc", "-std=c99", "-I", inc, c, "-o", exe])
            got = [int(x) for x in subprocess.check_output([exe]).split()]
        assert got == [ctypes.sizeof(D), D.k_new.offset, D.total_new.offset]


def test_attn_kernel_timing_host_side():
    import ctypes
    from paper_2609_36546_gb300 import ipd
    L = ipd._lib
    assert L.ipd_attn_kernel_time(None, None) == ipd.STATUS_CODES["IPD_ERR_INVALID_ARG"]
    assert L.ipd_set_attn_kernel_timing(1) == 0
    ms, n = ctypes.c_double(-1.0), ctypes.c_int(-1)
    assert L.ipd_attn_kernel_time(ctypes.byref(ms), ctypes.byref(n)) == 0
    assert n.value == 0 and ms.value == 0.0          # nothing launched: nothing recorded
    assert L.ipd_set_attn_kernel_timing(0) == 0
