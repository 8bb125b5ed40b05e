"""The attention tolerance, in bf16 ulps (numpy only, so that host worker
processes can apply it without importing torch).

Every output must lie within 2 bf16 ulp of the fp64 oracle result rounded to
bf16, the ulp taken at max(|ref|, ATTN_FLOOR * a), where a = sum_j w_j |v_jd|
is the softmax-weighted mean magnitude of the values that output averages
(the oracle's attention over |V|).  An fp32 evaluation of the weighted sum has
an absolute error of a few fp32 roundings of a, whatever the size of the
result, so a component that cancels to nearly zero cannot be held to 2 ulp of
itself.  ATTN_FLOOR = 2^-16 is the smallest power of two under which a plain
IEEE-fp32 evaluation (tests/attn_fp32_model.py) passes every small case
(tests/test_attn_tolerance.py).  The strict ulp at |ref| is reported beside
it, and at least ATTN_STRICT_FRAC of all elements must meet it.
"""
from __future__ import annotations

import numpy as np

import oracle as O

ATTN_FLOOR = 2.0 ** -16
ATTN_STRICT_FRAC = 0.9999


def attn_ulp_errors(got_bits: np.ndarray, ref: np.ndarray, ref_abs: np.ndarray):
    """(error under the floor, strict error) arrays, in bf16 ulps.

    ref: the fp64 oracle output; ref_abs: the oracle's attention over |V|
    (the weighted mean magnitude a of the averaged values), same shape."""
    got = O.bf16_to_f64(got_bits)
    ref_b = O.bf16_to_f64(O.f64_to_bf16(ref))
    err = np.abs(got - ref_b)
    ulp_floor = O.bf16_ulp(np.maximum(np.abs(ref_b), ATTN_FLOOR * np.abs(ref_abs)))
    ulp_strict = O.bf16_ulp(np.maximum(np.abs(ref_b), 1e-30))
    return err / ulp_floor, err / ulp_strict


def abs_bits(bits: np.ndarray) -> np.ndarray:
    """|x| of bf16 bit patterns (the sign bit cleared: exact)."""
    return (np.asarray(bits, np.uint16) & np.uint16(0x7FFF)).astype(np.uint16)


def attn_case_errors(q, kp, vp, L, scale, got):
    """Oracle attention of one request's queries over its pages, compared with
    the kernel's output bits: (max ulp under the floor, max strict ulp, number
    of elements over 2 ulp under the floor, number within 2 strict ulp, number
    of elements)."""
    npg = kp.shape[0]
    ref = O.paged_span_attention(q, kp, vp, np.arange(npg), L, scale)
    ref_abs = O.paged_span_attention(q, kp, abs_bits(vp), np.arange(npg), L, scale)
    e_floor, e_strict = attn_ulp_errors(got, ref, ref_abs)
    return (float(e_floor.max()) if e_floor.size else 0.0,
            float(e_strict.max()) if e_strict.size else 0.0,
            int((e_floor > 2.0).sum()), int((e_strict <= 2.0).sum()), int(e_strict.size))
