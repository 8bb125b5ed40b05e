"""Seeded synthetic inputs for the IPD verify step.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic (no softmax, no top-K, no verdict, no loss).  Both the CUDA
path and the fp64 oracle read what it makes, so it is the one module they
share.

The workloads imitate the rollouts of the paper's experiments (Sec. 4.1 and
App. A: Qwen3 students and teachers, rollouts at temperature 1): two
co-hosted models, each with its own paged KV cache, and a span of proposed
tokens per request with both models' logits over the vocabulary.

Recipe (every number below is stated once here and nowhere else):

* Head layouts: teacher cache 32 query / 4 KV heads, student cache 16 query /
  8 KV heads, head_dim 128, page size 16 tokens.  One attention layer per model.
* Request ``r`` has a context of ``ctx[r]`` tokens in BOTH caches.  The last
  ``span[r]`` of them are the proposed span; the verified prefix is
  ``ctx[r] - span[r]``.  ``driver[r]`` is 0 when the student proposes (the
  teacher verifies, the student decodes) and 1 when the teacher proposes.
* K, V, Q ~ N(0, 1) rounded to bf16.
* Page tables: each cache's pool is a set of pages; every request takes
  ``ceil(ctx/16)`` distinct pages drawn at random from the pool (shuffled, or
  uniformly over a larger pool when ``pool_bytes`` is set).
* Logits (bf16, one row per span position per model):
    - ``normal``  : both models N(0, sigma^2).
    - ``boost``   : both models N(0, 3^2); the verifier's logit at the proposed
      token is then set to ``8.1 + U(0, 8)``.  8.1 is 3 below the expected
      16th-largest of 151,936 N(0, 3^2) draws (about 11.1), so roughly 60 % of
      proposed tokens land in the verifier's top-16.
    - ``zipf``    : l_v = -1.1 ln(rank_r(v)) + N(0, 1), one random rank
      permutation per request shared by both models, independent noise.
  The proposed token at each position is drawn from the proposer's softmax
  (Gumbel-max over its bf16 row).  Optional ``tie_quantum`` rounds logits to a
  coarse grid before bf16 so that top-K boundaries tie often; optional
  ``force`` sets the verifier's logit at the proposed token to +30 ("accept")
  or -30 ("reject"); optional ``eos_prob`` replaces proposed tokens by
  ``eos_id`` at random.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import torch

PAGE_SIZE = 16
HEAD_DIM = 128


@dataclasses.dataclass(frozen=True)
class CacheShape:
    num_q_heads: int
    num_kv_heads: int
    head_dim: int = HEAD_DIM
    page_size: int = PAGE_SIZE

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def page_bytes(self) -> int:
        """bytes of one page of K plus one page of V (all KV heads)."""
        return 2 * self.num_kv_heads * self.page_size * self.head_dim * 2


TEACHER = CacheShape(32, 4)
STUDENT = CacheShape(16, 8)


@dataclasses.dataclass(frozen=True)
class Spec:
    name: str
    n_req: int
    ctx: tuple            # ("uniform", lo, hi) | ("lognormal", median, sigma, lo, hi)
    span: tuple           # ("fixed", k) | ("uniform", lo, hi)
    direction: str        # "S" | "T" | "half" | "bernoulli"
    vocab: int
    logits: str           # "normal" | "boost" | "zipf"
    sigma: float = 3.0
    pool_bytes: Optional[int] = None   # both caches together; None = exactly what is used
    K: int = 16
    eos_id: int = -1
    eos_prob: float = 0.0
    tie_quantum: float = 0.0
    force: str = ""       # "" | "accept" | "reject" | "mixed"
    # K rows at absolute position p are scaled by 1 + key_growth * p / 128, so
    # that attention scores grow along the sequence (test workloads only)
    key_growth: float = 0.0
    # ... and by key_jump from position key_jump_at on (a step in the scores)
    key_jump_at: int = 0
    key_jump: float = 1.0


GB = 1 << 30

CONFIGS = [
    Spec("tiny verify step", 4, ("uniform", 64, 256), ("fixed", 4), "half", 4096,
         "normal", sigma=2.0),
    Spec("student-proposes/teacher-verifies, Qwen3-shaped", 64, ("uniform", 1024, 8192),
         ("fixed", 8), "S", 151936, "boost"),
    Spec("long reasoning traces", 32, ("uniform", 8192, 32768), ("fixed", 16), "S", 151936,
         "boost", pool_bytes=40 * GB),
    Spec("bidirectional high-batch mix", 512, ("uniform", 2048, 4096), ("fixed", 4), "half",
         151936, "zipf"),
    Spec("full rollout-step mix", 1024, ("lognormal", 4096, 1.0, 256, 32768), ("uniform", 1, 16),
         "bernoulli", 151936, "boost", pool_bytes=120 * GB),
]


def small_spec(n_req=6, ctx=(1, 300), span=(1, 6), direction="bernoulli", vocab=2048,
               logits="normal", sigma=2.0, **kw) -> Spec:
    """A test-sized workload; every field of Spec can be overridden."""
    return Spec("small", n_req, ("uniform", ctx[0], ctx[1]), ("uniform", span[0], span[1]),
                direction, vocab, logits, sigma=sigma, **kw)


@dataclasses.dataclass
class Cache:
    shape: CacheShape
    k_pages: torch.Tensor      # [num_pages, Hkv, 16, 128] bf16
    v_pages: torch.Tensor
    page_table: torch.Tensor   # [R, max_pages] int32, -1 where unused (host copy)


@dataclasses.dataclass
class Workload:
    spec: Spec
    seed: int
    ctx: torch.Tensor          # [R] int32 (cpu)
    span: torch.Tensor         # [R] int32 (cpu)
    driver: torch.Tensor       # [R] uint8 (cpu); 0 = student proposes, 1 = teacher proposes
    teacher: Cache
    student: Cache
    q_verify_t: torch.Tensor   # [sum span of driver==0, 32, 128] teacher-verified queries
    q_verify_s: torch.Tensor   # [sum span of driver==1, 16, 128] student-verified queries
    q_decode_s: torch.Tensor   # [#driver==0, 16, 128] student decode queries
    q_decode_t: torch.Tensor   # [#driver==1, 32, 128] teacher decode queries
    tokens: torch.Tensor       # [T_tok] int32 (device)
    logits_s: torch.Tensor     # [T_tok, V] bf16 (device)
    logits_t: torch.Tensor     # [T_tok, V] bf16 (device)

    @property
    def n_req(self) -> int:
        return int(self.ctx.numel())

    @property
    def total_tokens(self) -> int:
        return int(self.span.sum())

    @property
    def cu_span(self) -> torch.Tensor:
        out = torch.zeros(self.n_req + 1, dtype=torch.int32)
        out[1:] = torch.cumsum(self.span, 0)
        return out

    @property
    def prefix_len(self) -> torch.Tensor:
        return (self.ctx - self.span).to(torch.int32)

    def reqs(self, driver: int) -> torch.Tensor:
        return torch.nonzero(self.driver == driver).flatten()


def _draw_ctx(spec: Spec, g: torch.Generator) -> torch.Tensor:
    kind = spec.ctx[0]
    if kind == "uniform":
        lo, hi = spec.ctx[1], spec.ctx[2]
        return torch.randint(lo, hi + 1, (spec.n_req,), generator=g, dtype=torch.int64)
    if kind == "lognormal":
        median, sigma, lo, hi = spec.ctx[1:]
        z = torch.randn(spec.n_req, generator=g, dtype=torch.float64)
        v = torch.exp(math.log(median) + sigma * z).round().to(torch.int64)
        return v.clamp(lo, hi)
    raise ValueError(kind)


def _draw_span(spec: Spec, g: torch.Generator) -> torch.Tensor:
    if spec.span[0] == "fixed":
        return torch.full((spec.n_req,), spec.span[1], dtype=torch.int64)
    lo, hi = spec.span[1], spec.span[2]
    return torch.randint(lo, hi + 1, (spec.n_req,), generator=g, dtype=torch.int64)


def _draw_driver(spec: Spec, g: torch.Generator) -> torch.Tensor:
    R = spec.n_req
    if spec.direction == "S":
        return torch.zeros(R, dtype=torch.uint8)
    if spec.direction == "T":
        return torch.ones(R, dtype=torch.uint8)
    if spec.direction == "half":
        d = torch.zeros(R, dtype=torch.uint8)
        d[R // 2:] = 1
        return d[torch.randperm(R, generator=g)]
    if spec.direction == "bernoulli":
        return (torch.rand(R, generator=g) < 0.5).to(torch.uint8)
    raise ValueError(spec.direction)


def _page_table(n_pages_req: torch.Tensor, pool_pages: int, g: torch.Generator) -> torch.Tensor:
    """Distinct random pages for every request, drawn without replacement."""
    total = int(n_pages_req.sum())
    assert total <= pool_pages, (total, pool_pages)
    perm = torch.randperm(pool_pages, generator=g)[:total].to(torch.int32)
    R = n_pages_req.numel()
    maxp = max(1, int(n_pages_req.max()))
    pt = torch.full((R, maxp), -1, dtype=torch.int32)
    off = 0
    for r in range(R):
        n = int(n_pages_req[r])
        pt[r, :n] = perm[off:off + n]
        off += n
    return pt


def _fill_pages(pool: torch.Tensor, used: torch.Tensor, g: torch.Generator, chunk: int = 4096):
    """N(0,1) bf16 into the used pages of a pool (other pages are never read)."""
    for i in range(0, used.numel(), chunk):
        idx = used[i:i + chunk].to(pool.device, torch.int64)
        vals = torch.randn((idx.numel(),) + tuple(pool.shape[1:]), generator=g,
                           device=pool.device, dtype=torch.float32)
        pool.index_copy_(0, idx, vals.to(torch.bfloat16))


def _randn_bf16(shape, g, device):
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)


def make_workload(spec_or_index, seed: Optional[int] = None, device="cpu",
                  row_chunk: int = 256) -> Workload:
    """Build one verify-step workload.

    Metadata (lengths, spans, drivers, page tables) is drawn on the host from
    ``seed`` so it is the same on every device; the bulk tensors are drawn with
    a generator on ``device`` (seeded from ``seed`` too)."""
    if isinstance(spec_or_index, int):
        spec = CONFIGS[spec_or_index]
        seed = spec_or_index if seed is None else seed
    else:
        spec = spec_or_index
        seed = 0 if seed is None else seed
    device = torch.device(device)
    gh = torch.Generator(device="cpu").manual_seed(seed)
    gd = torch.Generator(device=device).manual_seed(seed + 7919)

    ctx = _draw_ctx(spec, gh)
    span = _draw_span(spec, gh)
    span = torch.minimum(span, ctx)
    driver = _draw_driver(spec, gh)
    R = spec.n_req

    n_pages = (ctx + PAGE_SIZE - 1) // PAGE_SIZE
    caches = {}
    for name, shape in (("teacher", TEACHER), ("student", STUDENT)):
        need = int(n_pages.sum())
        if spec.pool_bytes is None:
            pool_pages = need
        else:
            share = shape.page_bytes / (TEACHER.page_bytes + STUDENT.page_bytes)
            pool_pages = max(need, int(spec.pool_bytes * share) // shape.page_bytes)
        pt = _page_table(n_pages, pool_pages, gh)
        used = pt[pt >= 0]
        shp = (pool_pages, shape.num_kv_heads, PAGE_SIZE, HEAD_DIM)
        if spec.pool_bytes is None:
            k = torch.empty(shp, dtype=torch.bfloat16, device=device)
            v = torch.empty(shp, dtype=torch.bfloat16, device=device)
        else:
            k = torch.zeros(shp, dtype=torch.bfloat16, device=device) if device.type == "cpu" \
                else torch.empty(shp, dtype=torch.bfloat16, device=device)
            v = torch.zeros_like(k) if device.type == "cpu" else torch.empty_like(k)
        _fill_pages(k, used, gd)
        _fill_pages(v, used, gd)
        if spec.key_growth or spec.key_jump != 1.0:
            _grow_keys(k, pt, n_pages, spec.key_growth, spec.key_jump_at, spec.key_jump)
        caches[name] = Cache(shape, k, v, pt)

    T = int(span.sum())
    s_reqs = torch.nonzero(driver == 0).flatten()
    t_reqs = torch.nonzero(driver == 1).flatten()
    n_qt = int(span[s_reqs].sum())
    n_qs = int(span[t_reqs].sum())
    q_verify_t = _randn_bf16((n_qt, TEACHER.num_q_heads, HEAD_DIM), gd, device)
    q_verify_s = _randn_bf16((n_qs, STUDENT.num_q_heads, HEAD_DIM), gd, device)
    q_decode_s = _randn_bf16((s_reqs.numel(), STUDENT.num_q_heads, HEAD_DIM), gd, device)
    q_decode_t = _randn_bf16((t_reqs.numel(), TEACHER.num_q_heads, HEAD_DIM), gd, device)

    tokens, ls, lt = _make_logits(spec, span, driver, gh, gd, device, row_chunk)
    return Workload(spec, seed, ctx.to(torch.int32), span.to(torch.int32), driver,
                    caches["teacher"], caches["student"], q_verify_t, q_verify_s,
                    q_decode_s, q_decode_t, tokens, ls, lt)


def _grow_keys(k, page_table, n_pages, growth: float, jump_at: int = 0, jump: float = 1.0):
    """Scales the K row at absolute position p of every request by
    1 + growth * p / 128, times `jump` from position jump_at on (rounded to
    bf16)."""
    pos = torch.arange(PAGE_SIZE, dtype=torch.float32)
    for r in range(page_table.shape[0]):
        for j in range(int(n_pages[r])):
            p = 16 * j + pos
            f = (1.0 + growth * p / 128.0) * torch.where(p >= jump_at, jump, 1.0) \
                if jump_at else (1.0 + growth * p / 128.0)
            f = f.to(k.device)
            page = int(page_table[r, j])
            k[page] = (k[page].float() * f[None, :, None]).to(torch.bfloat16)


def _make_logits(spec: Spec, span, driver, gh, gd, device, row_chunk):
    R, V = spec.n_req, spec.vocab
    T = int(span.sum())
    req_of_tok = torch.repeat_interleave(torch.arange(R), span)
    drv_tok = driver[req_of_tok].to(device)
    tokens = torch.empty(T, dtype=torch.int32, device=device)
    ls = torch.empty((T, V), dtype=torch.bfloat16, device=device)
    lt = torch.empty((T, V), dtype=torch.bfloat16, device=device)
    perms = None
    if spec.logits == "zipf":
        perms = {}
    for t0 in range(0, T, row_chunk):
        t1 = min(T, t0 + row_chunk)
        n = t1 - t0
        if spec.logits in ("normal", "boost"):
            a = torch.randn((n, V), generator=gd, device=device) * spec.sigma
            b = torch.randn((n, V), generator=gd, device=device) * spec.sigma
        elif spec.logits == "zipf":
            rows_req = req_of_tok[t0:t1]
            base = torch.empty((n, V), device=device)
            for r in torch.unique(rows_req).tolist():
                if r not in perms:
                    perms[r] = torch.randperm(V, generator=gd, device=device)
                rank = perms[r].to(torch.float32) + 1.0
                base[rows_req == r] = -1.1 * torch.log(rank)
            a = base + torch.randn((n, V), generator=gd, device=device)
            b = base + torch.randn((n, V), generator=gd, device=device)
        else:
            raise ValueError(spec.logits)
        if spec.tie_quantum > 0:
            a = torch.round(a / spec.tie_quantum) * spec.tie_quantum
            b = torch.round(b / spec.tie_quantum) * spec.tie_quantum
        a = a.to(torch.bfloat16)
        b = b.to(torch.bfloat16)
        d = drv_tok[t0:t1]
        # proposer row: the student's (a) when driver == 0, the teacher's (b) otherwise
        prop = torch.where((d == 0)[:, None], a, b).float()
        u = torch.rand((n, V), generator=gd, device=device).clamp_min(1e-30)
        gumbel = -torch.log(-torch.log(u))
        tok = torch.argmax(prop + gumbel, dim=1)
        if spec.eos_prob > 0 and spec.eos_id >= 0:
            e = torch.rand(n, generator=gd, device=device) < spec.eos_prob
            tok = torch.where(e, torch.full_like(tok, spec.eos_id), tok)
        rows = torch.arange(n, device=device)
        ver_is_teacher = d == 0
        if spec.logits == "boost" or spec.force:
            if spec.force == "accept":
                val = torch.full((n,), 30.0, device=device)
            elif spec.force == "reject":
                val = torch.full((n,), -30.0, device=device)
            elif spec.force == "mixed":
                coin = torch.rand(n, generator=gd, device=device) < 0.7
                val = torch.where(coin, torch.full((n,), 30.0, device=device),
                                  torch.full((n,), -30.0, device=device))
            else:
                val = 8.1 + 8.0 * torch.rand(n, generator=gd, device=device)
            val = val.to(torch.bfloat16)
            bt = b[rows, tok].clone()
            at = a[rows, tok].clone()
            b[rows, tok] = torch.where(ver_is_teacher, val, bt)
            a[rows, tok] = torch.where(ver_is_teacher, at, val)
        tokens[t0:t1] = tok.to(torch.int32)
        ls[t0:t1] = a
        lt[t0:t1] = b
    return tokens, ls, lt
