"""Whole full-size batches against the oracle (needs a GB300).

Each full-size workload runs once in the launch configuration the benchmark
times; then every request's scores and decisions, the whole batch's loss and
every request's attention output (span queries and decode queries, both
caches) are recomputed by the fp64 oracle on the host cores and compared at
the stated tolerances.  Batch-level identities are checked as well.
"""
import pytest
import torch

import ipd_synth as S

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import ipd
    return ipd


@pytest.fixture(scope="module")
def pool():
    from tests.fullbatch import OraclePool
    with OraclePool() as p:
        yield p


@pytest.mark.parametrize("cfg", [1, 2, 3, 4])
def test_full_batch_matches_oracle(lib, pool, cfg):
    from paper_2609_36546_gb300 import VerifyStep
    from tests.fullbatch import check_step_full
    w = S.make_workload(cfg, device="cuda")
    step = VerifyStep.from_workload(w, device="cuda")
    step.run()
    torch.cuda.synchronize()
    assert lib.device_error() == 0
    rep = check_step_full(step, pool=pool)
    print(f"{S.CONFIGS[cfg].name}:", {k: rep[k] for k in (
        "attn_rows", "attn_max_ulp", "attn_max_ulp_strict", "attn_frac_strict_le2", "max_logp_err",
        "max_kl_err", "near_threshold", "near_threshold_mismatch", "coverage_rate",
        "loss_rel_err")})
    assert rep["ok"], rep
    # identities over the whole batch
    sc = {k: v.cpu() for k, v in step.score.items()}
    o8 = step.out8.cpu()
    emitted = sc["source"] != 255
    assert int(emitted.sum()) == int(sc["n_emit"].sum())
    assert float(o8[3] + o8[4]) == float(emitted.sum())
    assert torch.all(sc["new_len"] == step.prefix_len.cpu() + sc["n_emit"])
    # the needed-rows pass on the same step: rows are read whole by both
    # passes at these sizes, so where it defines a value it is bit-identical
    o8 = step.out8.cpu()
    step.rows = "needed"
    step.run_score()
    step.run_loss()
    torch.cuda.synchronize()
    assert lib.device_error() == 0
    got = {k: v.cpu() for k, v in step.score.items()}
    for n in ("first_trans", "n_emit", "next_driver", "new_len", "done", "source"):
        assert torch.equal(got[n], sc[n]), n
    assert torch.equal(step.out8.cpu(), o8)
    cu = step.cu_span.cpu()
    pos = torch.arange(step.T) - torch.repeat_interleave(cu[:-1], cu[1:] - cu[:-1])
    first = torch.repeat_interleave(sc["first_trans"], cu[1:] - cu[:-1])
    dec = pos <= first
    for n in ("logp_s", "logp_t", "feedback", "kl_rev", "kl_fwd"):
        assert torch.equal(got[n][emitted], sc[n][emitted]), n
    for n in ("covered", "margin"):
        assert torch.equal(got[n][dec], sc[n][dec]), n
    del step, w
    torch.cuda.empty_cache()
