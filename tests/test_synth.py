"""The seeded input generator: determinism, layout, and the calibration of the
synthetic distributions (readings of the workload recipes; these are
distributions, not the method's arithmetic, so they stay parity-unpinned)."""
import numpy as np
import torch

import ipd_synth as S
import oracle as O


def test_deterministic_and_seed_dependent():
    spec = S.small_spec(n_req=5)
    a = S.make_workload(spec, seed=4)
    b = S.make_workload(spec, seed=4)
    c = S.make_workload(spec, seed=5)
    for f in ("ctx", "span", "driver", "tokens"):
        assert torch.equal(getattr(a, f), getattr(b, f))
    assert torch.equal(a.logits_s.view(torch.int16), b.logits_s.view(torch.int16))
    assert torch.equal(a.teacher.k_pages.view(torch.int16), b.teacher.k_pages.view(torch.int16))
    assert not torch.equal(a.logits_s.view(torch.int16), c.logits_s.view(torch.int16))


def test_layout_and_page_tables():
    w = S.make_workload(0)
    assert w.n_req == 4 and w.total_tokens == 16 and w.logits_s.shape == (16, 4096)
    assert sorted(w.driver.tolist()) == [0, 0, 1, 1]
    for cache, shape in ((w.teacher, S.TEACHER), (w.student, S.STUDENT)):
        assert cache.k_pages.shape[1:] == (shape.num_kv_heads, 16, 128)
        used = []
        for r in range(w.n_req):
            n = (int(w.ctx[r]) + 15) // 16
            row = cache.page_table[r]
            assert (row[:n] >= 0).all() and (row[n:] == -1).all()
            used += row[:n].tolist()
        assert len(set(used)) == len(used) and max(used) < cache.k_pages.shape[0]
    assert w.q_verify_t.shape == (8, 32, 128) and w.q_decode_s.shape == (2, 16, 128)


def test_config_metadata_ranges():
    g = torch.Generator().manual_seed(0)
    for i, spec in enumerate(S.CONFIGS):
        ctx = S._draw_ctx(spec, g)
        span = S._draw_span(spec, g)
        assert ctx.numel() == spec.n_req
        if spec.ctx[0] == "uniform":
            assert ctx.min() >= spec.ctx[1] and ctx.max() <= spec.ctx[2]
        else:
            assert ctx.min() >= spec.ctx[3] and ctx.max() <= spec.ctx[4]
            assert 2500 < float(ctx.float().median()) < 6000
        assert span.min() >= 1 and span.max() <= 16
    d = S._draw_driver(S.CONFIGS[3], g)
    assert int(d.sum()) == 256


def test_boost_recipe_acceptance_rate():
    """The verifier logit of the proposed token at 8.1 + U(0,8) lands in the
    top-16 of 151,936 N(0, 3^2) logits about 60 % of the time."""
    spec = S.small_spec(n_req=8, span=(6, 6), vocab=151936, logits="boost", sigma=3.0,
                        direction="S", ctx=(20, 40))
    w = S.make_workload(spec, seed=0)
    lt = w.logits_t.view(torch.int16).numpy().view(np.uint16)
    cov = [O.covered(O.bf16_to_f64(lt[t]), int(w.tokens[t]), 16) for t in range(w.total_tokens)]
    rate = float(np.mean(cov))
    assert 0.35 <= rate <= 0.85, rate
