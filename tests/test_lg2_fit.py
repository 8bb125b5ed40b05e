"""Where the sampler's eight lg2 coefficients come from (CPU only).

The sampler's fixed fp32 log2 (include/ipd.h at ipd_sample; the oracle's
lg2_f32 and the CUDA sampler each state the coefficients) evaluates
log2(1 + t) = t P(t) on t in [sqrt(1/2) - 1, sqrt(2) - 1] with a degree-7 P.
P is the least-squares fit of log2(1 + t) / t at 4000 Chebyshev nodes of
that interval, rounded to fp32.  This test redoes the fit with numpy and
checks the rounded coefficients against the bit patterns written in each of
the three places, so none of them can drift from the fit or from each other.
"""
import math
import os
import re

import numpy as np

import oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def fit_lg2_coefficients(n_nodes: int = 4000) -> tuple:
    """fp32 bit patterns (lowest degree first) of the least-squares degree-7
    fit of log2(1 + t) / t at n Chebyshev nodes (first kind) of
    [sqrt(1/2) - 1, sqrt(2) - 1]."""
    a, b = math.sqrt(0.5) - 1.0, math.sqrt(2.0) - 1.0
    k = np.arange(n_nodes)
    t = (a + b) / 2 + (b - a) / 2 * np.cos((2 * k + 1) * np.pi / (2 * n_nodes))
    y = np.log1p(t) / (t * math.log(2.0))
    coef = np.linalg.lstsq(np.vander(t, 8, increasing=True), y, rcond=None)[0]
    return tuple(int(w) for w in coef.astype(np.float32).view(np.uint32))


def _hex_words(text):
    return tuple(int(w, 16) for w in re.findall(r"\b(?:0x)?([0-9A-Fa-f]{8})u?\b", text))


def test_fit_reproduces_the_oracle_coefficients():
    assert fit_lg2_coefficients() == tuple(O.LG2_POLY_BITS)


def test_fit_reproduces_the_header_coefficients():
    src = open(os.path.join(ROOT, "include", "ipd.h")).read()
    line = re.search(r"lowest degree first\)\s*\n\s*\*\s*([0-9A-F ]+)\.", src).group(1)
    assert _hex_words(line) == fit_lg2_coefficients()


def test_fit_reproduces_the_cuda_coefficients():
    src = open(os.path.join(ROOT, "paper_2609_36546_gb300", "csrc", "sample.cu")).read()
    named = dict((int(i), int(h, 16)) for i, h in
                 re.findall(r"\bc([0-7]) = __uint_as_float\(0x([0-9A-Fa-f]{8})u\)", src))
    assert tuple(named[i] for i in range(8)) == fit_lg2_coefficients()


def test_the_rounded_fit_does_not_depend_on_the_node_count():
    ref = fit_lg2_coefficients()
    for n in (64, 256, 1024):
        assert fit_lg2_coefficients(n) == ref


def test_rounded_fit_is_accurate():
    """The fp32 procedure with these coefficients stays within 1.1e-6 of log2
    across both halves of the reduced range and several binades."""
    x = np.float32(2.0) ** np.linspace(-20, 20, 200001).astype(np.float32)
    err = np.abs(O.lg2_f32(x).astype(np.float64) - np.log2(x.astype(np.float64)))
    assert float(err.max()) <= 1.1e-6
