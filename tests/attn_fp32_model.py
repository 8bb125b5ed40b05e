"""A plain IEEE-fp32 evaluation of span attention, used only to derive the
attention tolerance (test infrastructure: neither the oracle nor the CUDA
path, and shared with neither).

It computes what ``oracle.span_attention`` defines (Sec. 3.2.3: the k span
queries of a request, causal within the span, over the verifier's cache;
a decode query is k = 1) with every operation in fp32 and in key order:

* each score is a dot product of the bf16 query and key, accumulated over
  the head dimension one product at a time (bf16 x bf16 products are exact
  in fp32);
* x_j = fp32(s_j * scale * log2 e); m = max_j x_j; p_j = 2^(x_j - m) in fp32;
* the row sum l and the weighted sum o_d = sum_j p_j v_jd are accumulated in
  fp32 one key at a time, each product p_j v_jd rounded to fp32 first;
* the output o_d / l is rounded to bf16 once, by the caller.

This is the accuracy an fp32 implementation without any compensated
arithmetic reaches; the tolerance the parity tests apply is the smallest one
this model meets on every small case.
"""
from __future__ import annotations

import numpy as np

LOG2E = 1.4426950408889634


def span_attention_fp32(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float) -> np.ndarray:
    """q: [n, Hq, D]; k, v: [L, Hkv, D] (values exactly representable in bf16).
    Query i sits at position L - n + i and sees keys 0 .. L - n + i; head h reads
    KV head h // (Hq / Hkv).  Returns [n, Hq, D] fp32 (not yet rounded to bf16)."""
    n, Hq, D = q.shape
    L, Hkv, _ = k.shape
    G = Hq // Hkv
    q32, k32, v32 = (np.asarray(a, np.float32) for a in (q, k, v))
    c = np.float32(scale * LOG2E)
    out = np.zeros((n, Hq, D), np.float32)
    for i in range(n):
        vis = L - n + i + 1
        for kh in range(Hkv):
            qg = q32[i, kh * G:(kh + 1) * G]                           # [G, D]
            kk, vv = k32[:vis, kh], v32[:vis, kh]                      # [vis, D]
            prod = qg[:, None, :] * kk[None, :, :]                     # exact in fp32
            s = np.add.accumulate(prod, axis=2, dtype=np.float32)[..., -1]   # [G, vis]
            x = (s * c).astype(np.float32)
            p = np.exp2(x - x.max(axis=1, keepdims=True)).astype(np.float32)
            l = np.add.accumulate(p, axis=1, dtype=np.float32)[:, -1:]
            pv = (p[:, :, None] * vv[None, :, :]).astype(np.float32)  # [G, vis, D]
            o = np.add.accumulate(pv, axis=1, dtype=np.float32)[:, -1, :]
            out[i, kh * G:(kh + 1) * G] = (o / l).astype(np.float32)
    return out
