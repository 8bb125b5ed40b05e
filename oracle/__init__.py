"""fp64 CPU oracle for the IPD verify step -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The product
path (``paper_2609_36546_gb300``) never imports it and shares no code with it.

Parity status per function (what pins it is listed in tests/test_oracle_pins.py):

* ``span_attention`` / ``paged_span_attention`` -- pinned (library SDPA in
  fp64, closed forms, paging invariants).
* ``kv_append`` -- pinned (the appended paged cache attends exactly like
  library SDPA over the concatenated sequence; unowned pages untouched).
* ``log_softmax_row``, ``topk``, ``covered``, ``margin`` -- pinned (scipy,
  brute-force sort, rank identity).
* ``topk_kl`` -- pinned (scipy KL on the renormalised support, K=1 closed
  form, KL >= 0 and symmetry identities).
* ``verdict`` -- pinned (hand-worked cases from the transition equation and
  the rollback rules, exhaustive invariants).
* ``split_loss`` -- pinned (hand-worked fixture, special cases that reduce to
  pure on-policy and pure off-policy distillation).
* ``split_loss_grad`` -- pinned (central finite differences of ``topk_kl`` +
  ``split_loss`` in fp64, shift invariance of every row, zero rows off the
  emitted positions).
* ``philox4x32_10`` -- pinned (the generator's published known-answer
  vectors, tests/golden/philox4x32_10_kat.txt).
* ``lg2_f32`` -- pinned (numpy log2 within 1.2e-6; exact powers of two).
* ``sample_uniforms``, ``gumbel_scores``, ``sample_token`` -- pinned
  (Kolmogorov-Smirnov uniformity; chi-square of 12000 draws against the
  softmax at two temperatures; planted base and scale mistakes rejected).
* ``next_token_after_verdict`` -- pinned (hand-worked takeover, handback,
  no-transition and EOS cases).
"""
from .ipd_oracle import *  # noqa: F401,F403
