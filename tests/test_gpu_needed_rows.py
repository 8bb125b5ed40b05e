"""The needed-rows vocabulary pass (ipd_score_span_needed) on the GPU: only
the verifier's rows up to each request's first transition and the
proposer's rows of the emitted positions are defined, and must match the
fp64 oracle there; the verdict, the sources and the loss must match too."""
import numpy as np
import pytest
import torch

import ipd_synth as S
from tests import parity

pytestmark = pytest.mark.gpu

SCORE_REQ = ("first_trans", "n_emit", "next_driver", "new_len", "done")


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import ipd
    return ipd


def _step(spec, seed, rows):
    from paper_2609_36546_gb300 import VerifyStep
    w = S.make_workload(spec, seed=seed, device="cpu")
    step = VerifyStep.from_workload(w, device="cuda", rows=rows)
    step.run()
    torch.cuda.synchronize()
    return w, step


CASES = [
    ("mixed", S.small_spec(), 0),
    ("teacher-driving", S.small_spec(n_req=6, direction="T", span=(1, 16), ctx=(20, 700)), 4),
    ("ties", S.small_spec(n_req=6, vocab=4096, sigma=3.0, tie_quantum=0.5, span=(2, 6)), 5),
    ("accept-all", S.small_spec(n_req=5, force="accept", span=(3, 9)), 6),
    ("reject-all", S.small_spec(n_req=5, force="reject", span=(3, 9)), 7),
    ("mixed-eos", S.small_spec(n_req=10, force="mixed", eos_id=5, eos_prob=0.3, span=(2, 10)), 8),
    ("K1", S.small_spec(n_req=4, K=1), 9),
    ("K32", S.small_spec(n_req=4, K=32, vocab=8192), 10),
    ("wide-vocab", S.small_spec(n_req=2, vocab=151936, sigma=3.0, logits="boost", span=(4, 8),
                                ctx=(100, 400)), 12),
    # enough rows for several waves of row CTAs: later positions find their
    # request's transition already known and are skipped
    ("many-rows", S.small_spec(n_req=160, vocab=4096, span=(8, 16), ctx=(16, 64), force="mixed"),
     18),
    ("many-rows-teacher", S.small_spec(n_req=160, vocab=4096, span=(8, 16), ctx=(16, 64),
                                       direction="T"), 19),
]


@pytest.mark.parametrize("name,spec,seed", CASES, ids=[c[0] for c in CASES])
def test_needed_rows_match_oracle(lib, name, spec, seed):
    """Scores where defined, every decision, and the whole batch's loss (the
    attention of these steps is the same launch the other tests check)."""
    w, step = _step(spec, seed, "needed")
    assert lib.device_error() == 0
    rep, orc = parity.check_scores(step, None, needed=True)
    rep.update(parity.check_loss(step, orc))
    assert rep["score_ok"] and rep["loss_ok"], rep


@pytest.mark.parametrize("name,spec,seed", CASES[-2:], ids=[c[0] for c in CASES[-2:]])
def test_needed_rows_equal_all_rows_where_defined(lib, name, spec, seed):
    """Every row is read in one part by both passes here, so the values a
    needed-rows pass defines are bit-identical to the full pass's, and so are
    the decisions and the loss; rows past known transitions were skipped."""
    _, full = _step(spec, seed, "all")
    ref = {k: v.cpu() for k, v in full.score.items()}
    ref8 = full.out8.cpu()
    full.rows = "needed"
    full.run_score()
    full.run_loss()
    torch.cuda.synchronize()
    assert lib.device_error() == 0
    got = {k: v.cpu() for k, v in full.score.items()}
    for n in SCORE_REQ + ("source",):
        assert torch.equal(got[n], ref[n]), n
    assert torch.equal(full.out8.cpu(), ref8)
    cu = full.cu_span.cpu().numpy()
    src, ft = ref["source"].numpy(), ref["first_trans"].numpy()
    em = np.zeros(full.T, bool)
    dec = np.zeros(full.T, bool)
    for r in range(full.R):
        e, d = parity.needed_positions(src, ft, cu, r)
        em[cu[r]:cu[r + 1]] = e
        dec[cu[r]:cu[r + 1]] = d
    for n in ("logp_s", "logp_t", "feedback", "kl_rev", "kl_fwd"):
        assert torch.equal(got[n][em], ref[n][em]), n
    for n in ("covered", "margin"):
        assert torch.equal(got[n][dec], ref[n][dec]), n
    # positions past the transitions: some rows were not read at all
    skipped = torch.isnan(got["logp_s"][~torch.from_numpy(dec)])
    assert int(skipped.sum()) > 0


def test_span_longer_than_the_bound_is_reported(lib):
    w, step = _step(S.small_spec(n_req=4, span=(5, 9)), 21, "needed")
    assert lib.device_error() == 0
    step.max_span = int(w.span.max()) - 1
    step.run_score()
    torch.cuda.synchronize()
    assert lib.device_error() == 6  # IPD_DEVERR_SPAN


def _defined(step, score):
    """Masks of the positions a needed-rows pass defines, from its verdict."""
    cu = step.cu_span.cpu()
    lens = cu[1:] - cu[:-1]
    pos = torch.arange(step.T) - torch.repeat_interleave(cu[:-1], lens)
    dec = pos <= torch.repeat_interleave(score["first_trans"].cpu(), lens)
    return score["source"].cpu() != 255, dec


@pytest.mark.parametrize("graph", [False, True])
def test_needed_rows_from_host_equals_direct_calls(lib, graph):
    """The host-fed step (logits in request-aligned chunks, each scored as it
    lands, directly or replayed from a graph) gives the direct step's
    decisions, loss and defined values, bit for bit."""
    # chunks of more rows than one wave of row CTAs holds, so that rows are skipped
    w, step = _step(S.small_spec(n_req=400, ctx=(20, 200), span=(0, 16), vocab=4096), 45,
                    "needed")
    first = {k: v.cpu() for k, v in step.score.items()}
    o8 = step.out8.cpu()
    em, dec = _defined(step, first)
    host = step.host_inputs(3)
    results = step.host_results()
    g = step.capture_from_host(host, results) if graph else None
    for _ in range(2):
        for v in step.score.values():
            v.zero_()
        step.logits_s.zero_()
        step.logits_t.zero_()
        step.out8.zero_()
        step._in.buf.zero_()
        if g is not None:
            g.replay()
        else:
            step.run_from_host(host, results, torch.cuda.current_stream())
        torch.cuda.synchronize()
        got = {k: v.cpu() for k, v in step.score.items()}
        for n in SCORE_REQ + ("source",):
            assert torch.equal(got[n], first[n]), n
            assert torch.equal(results[n], first[n]), n
        for n in ("logp_s", "logp_t", "feedback", "kl_rev", "kl_fwd"):
            assert torch.equal(got[n][em], first[n][em]), n
        for n in ("covered", "margin"):
            assert torch.equal(got[n][dec], first[n][dec]), n
        assert torch.equal(step.out8.cpu(), o8)
        assert torch.equal(results["out8"], o8)
    assert lib.device_error() == 0


def test_host_fed_step_reading_logits_in_place(lib):
    """run_from_host(host_logits=True): the vocabulary pass reads the pinned
    host logits in place (the device copies are zeroed first, so any use of
    them would show); decisions, loss and defined values equal the
    device-resident step's, bit for bit."""
    w, step = _step(S.small_spec(n_req=400, ctx=(20, 200), span=(0, 16), vocab=4096), 47,
                    "needed")
    host = step.host_inputs(3)
    if not (lib.device_readable(host["logits_s"]) and lib.device_readable(host["logits_t"])):
        pytest.skip("pinned host memory is not mapped for the device here")
    first = {k: v.cpu() for k, v in step.score.items()}
    o8 = step.out8.cpu()
    em, dec = _defined(step, first)
    results = step.host_results()
    step.logits_s.zero_()
    step.logits_t.zero_()
    for graph in (False, True):
        for v in step.score.values():
            v.zero_()
        step.out8.zero_()
        if graph:
            step.capture_from_host(host, results, host_logits=True).replay()
        else:
            step.run_from_host(host, results, torch.cuda.current_stream(), host_logits=True)
        torch.cuda.synchronize()
        got = {k: v.cpu() for k, v in step.score.items()}
        for n in SCORE_REQ + ("source",):
            assert torch.equal(got[n], first[n]), n
            assert torch.equal(results[n], first[n]), n
        for n in ("logp_s", "logp_t", "feedback", "kl_rev", "kl_fwd"):
            assert torch.equal(got[n][em], first[n][em]), n
        for n in ("covered", "margin"):
            assert torch.equal(got[n][dec], first[n][dec]), n
        assert torch.equal(step.out8.cpu(), o8)
        assert torch.equal(results["out8"], o8)
    assert lib.device_error() == 0
    assert not lib.device_readable(torch.zeros(4))  # pageable host memory is not offered
