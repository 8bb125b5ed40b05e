"""One verify step of the fused engine, assembled from plain tensors.

Host glue only: it groups requests by verifier (Sec. 3.2.3: requests are
grouped by their verifier for the verification stage and by their driver for
the proposal stage), allocates the device buffers, and issues the three C-ABI
calls on one stream:

  ipd_verify_attn  teacher-verify + student-verify span attention and the
                   student / teacher decode attention, one launch
  ipd_score_span   vocabulary pass, verdict and cache bookkeeping
  ipd_split_loss   source-split objective
"""
from __future__ import annotations

import math
from typing import Optional

import torch

from . import ipd

SCALE = 1.0 / math.sqrt(128.0)


def _cu(lengths: torch.Tensor) -> torch.Tensor:
    out = torch.zeros(lengths.numel() + 1, dtype=torch.int32)
    out[1:] = torch.cumsum(lengths.to(torch.int64), 0).to(torch.int32)
    return out


# Names of the score outputs a host-fed step copies back, besides "out8".
RESULT_NAMES = ("first_trans", "n_emit", "next_driver", "new_len", "done", "source")


def chunk_plan(cu_span: torch.Tensor, n_chunks: int):
    """Request-aligned chunks of a step's span positions for a host-fed step.

    Chunk c covers requests [r0, r1) and positions [t0, t1) = [cu[r0], cu[r1]),
    about T / n_chunks positions each (a chunk may hold no request, except
    the last).  Returns the list of (r0, r1, t0, t1) and the chunks' span
    offsets, each rebased to its t0 and concatenated (R + #chunks entries)."""
    cu = cu_span.to(torch.int64).cpu()
    R, T = cu.numel() - 1, int(cu[-1])
    bounds, r0 = [], 0
    for c in range(1, n_chunks + 1):
        target = T * c // n_chunks
        r1 = R if c == n_chunks else max(r0, int(torch.searchsorted(cu, target, right=True)) - 1)
        if r1 > r0 or c == n_chunks:
            bounds.append((r0, r1, int(cu[r0]), int(cu[r1])))
        r0 = r1
    cu_chunk = torch.cat([(cu[a:b + 1] - cu[a]).to(torch.int32) for a, b, _, _ in bounds])
    return bounds, cu_chunk


class _Packed:
    """Named tensors laid out in one byte buffer (256-byte aligned slots), so
    that a host<->device transfer of all of them is one copy: many small
    copies each pay a fixed cost that dwarfs their bytes."""

    def __init__(self, named, device, pin: bool = False):
        self.layout, off = [], 0
        for name, t in named:
            nb = t.numel() * t.element_size()
            self.layout.append((name, off, nb, t.dtype, tuple(t.shape)))
            off = (off + nb + 255) // 256 * 256
        self.buf = torch.empty(max(off, 256), dtype=torch.uint8, device=device, pin_memory=pin)
        self.views = {name: self._view(o, nb, dt, sh) for name, o, nb, dt, sh in self.layout}
        for name, t in named:
            self.views[name].copy_(t)

    def _view(self, off, nb, dtype, shape):
        return self.buf[off:off + nb].view(dtype).view(shape)

    def mirror(self, device, pin: bool = False) -> "_Packed":
        """The same layout in a new buffer, holding a copy of this one."""
        m = _Packed.__new__(_Packed)
        m.layout = self.layout
        m.buf = torch.empty(self.buf.numel(), dtype=torch.uint8, device=device, pin_memory=pin)
        m.buf.copy_(self.buf)
        m.views = {name: m._view(o, nb, dt, sh) for name, o, nb, dt, sh in self.layout}
        return m


class VerifyStep:
    """Device buffers and calls of one verify step.

    Host inputs (cpu tensors): ctx [R] (KV length of both caches, span
    included), span [R], driver [R] (0: the student proposed), page tables
    [R, max_pages] for the teacher and the student cache.  Device inputs:
    the four paged pools, the span queries for each verifier, the decode
    queries for each proposer, the proposed tokens and both models' logits.

    The pools and the logits are used in place.  The queries, tokens and
    request metadata are copied, at construction, into one device buffer
    owned by the step (attributes ``tokens``, ``cu_span``, ``driver``,
    ``prefix_len`` and each batch's tensors are views into it), so that a
    host-fed step moves them with one copy.
    """

    def __init__(self, teacher_k, teacher_v, student_k, student_v, ctx, span, driver,
                 pt_teacher, pt_student, q_verify_t, q_verify_s, q_decode_s, q_decode_t, tokens,
                 logits_s, logits_t, K: int = 16, eos_id: int = -1, resp_len=None,
                 agg_mode: int = ipd.AGG_SEQ_MEAN_TOKEN_MEAN, dir_mode: int = ipd.DIR_SPLIT,
                 scale: float = SCALE, device="cuda", rows: str = "all"):
        dev = torch.device(device)
        self.device = dev
        # "all": the vocabulary pass reads every logits row (ipd_score_span);
        # "needed": only the rows the verdict and the emitted positions need
        # (ipd_score_span_needed); the verdict, sources and loss are the same
        if rows not in ("all", "needed"):
            raise ValueError(f"rows must be 'all' or 'needed', not {rows!r}")
        self.rows = rows
        self.K, self.eos_id, self.agg_mode, self.dir_mode, self.scale = K, eos_id, agg_mode, \
            dir_mode, scale
        ctx = ctx.to(torch.int32).cpu()
        span = span.to(torch.int32).cpu()
        driver = driver.to(torch.uint8).cpu()
        self.R = int(ctx.numel())
        self.T = int(span.sum())
        self.max_span = max(1, int(span.max())) if span.numel() else 1
        self.cache_t = ipd.KVCache(teacher_k, teacher_v)
        self.cache_s = ipd.KVCache(student_k, student_v)
        idx_s = torch.nonzero(driver == 0).flatten()   # student proposes, teacher verifies
        idx_t = torch.nonzero(driver == 1).flatten()
        self.idx_s, self.idx_t = idx_s, idx_t

        one = lambda idx: torch.ones(idx.numel(), dtype=torch.int32)
        # (name, cache, queries, request indices, query lengths, page table, cache name)
        subs = [s for s in (
            ("verify_teacher", self.cache_t, q_verify_t, idx_s, span[idx_s], pt_teacher, "teacher"),
            ("verify_student", self.cache_s, q_verify_s, idx_t, span[idx_t], pt_student, "student"),
            ("decode_student", self.cache_s, q_decode_s, idx_s, one(idx_s), pt_student, "student"),
            ("decode_teacher", self.cache_t, q_decode_t, idx_t, one(idx_t), pt_teacher, "teacher"))
            if s[3].numel() > 0]
        # Every per-step input but the logits (queries, query offsets, lengths,
        # page tables, tokens, request metadata, and room for the chunk
        # offsets of a host-fed step) lives in one device buffer.
        named = []
        for n, _, q, idx, q_len, pt, _ in subs:
            named += [(n + ".q", q), (n + ".cu_q", _cu(q_len)), (n + ".seq", ctx[idx].contiguous()),
                      (n + ".ptab", pt[idx].contiguous())]
        named += [("tokens", tokens), ("cu_span", _cu(span)), ("driver", driver),
                  ("prefix_len", (ctx - span).to(torch.int32)),
                  ("cu_chunk", torch.zeros(2 * self.R + 2, dtype=torch.int32))]
        self._in = _Packed(named, dev)
        v = self._in.views
        # (name, batch, request indices, cache name) for every non-empty sub-batch
        self.batches = []
        for n, cache, _, idx, q_len, _, cname in subs:
            q = v[n + ".q"]
            b = ipd.AttnBatch(cache, q, v[n + ".cu_q"], v[n + ".seq"], v[n + ".ptab"],
                              torch.empty_like(q), int(q_len.max()), int(ctx[idx].max()))
            self.batches.append((n, b, idx, cname))
        self.verify = [b for n, b, _, _ in self.batches if n.startswith("verify")]
        self.decode = [b for n, b, _, _ in self.batches if n.startswith("decode")]
        self.ws_attn = torch.empty(max(256, ipd.attn_workspace_size(self.verify, self.decode)),
                                   dtype=torch.uint8, device=dev)
        # scoring
        self.logits_s, self.logits_t = logits_s, logits_t
        self.tokens, self.cu_span, self.driver, self.prefix_len = (
            v["tokens"], v["cu_span"], v["driver"], v["prefix_len"])
        self.V = int(logits_s.shape[1])
        self.resp_len = None if resp_len is None else resp_len.to(torch.int32).to(dev)
        self.score = ipd.alloc_score_outputs(self.R, self.T, dev)
        # the results a host-fed step reads back, in one buffer as well
        self._res = _Packed([(n, self.score[n]) for n in RESULT_NAMES] +
                            [("out8", torch.zeros(8, dtype=torch.float32))], dev)
        self.score.update({n: self._res.views[n] for n in RESULT_NAMES})
        self.out8 = self._res.views["out8"]
        self.ws_score = torch.empty(max(256, ipd.score_workspace_size(self.R, self.T, self.V, K)),
                                    dtype=torch.uint8, device=dev)

    @classmethod
    def from_workload(cls, w, device="cuda", **kw):
        """Build from an object with the attributes of a synthetic workload."""
        dev = torch.device(device)
        mv = lambda t: t.to(dev)
        kw.setdefault("K", w.spec.K)
        kw.setdefault("eos_id", w.spec.eos_id)
        return cls(mv(w.teacher.k_pages), mv(w.teacher.v_pages), mv(w.student.k_pages),
                   mv(w.student.v_pages), w.ctx, w.span, w.driver, w.teacher.page_table,
                   w.student.page_table, mv(w.q_verify_t), mv(w.q_verify_s), mv(w.q_decode_s),
                   mv(w.q_decode_t), mv(w.tokens), mv(w.logits_s), mv(w.logits_t), device=dev,
                   **kw)

    # -- the three calls ------------------------------------------------------
    def run_attention(self, stream=None):
        ipd.verify_attn(self.verify, self.decode, self.scale, self.ws_attn, stream)

    def _score_call(self, ls, lt, tokens, cu_span, driver, prefix_len, out, stream):
        if self.rows == "needed":
            ipd.score_span_needed(ls, lt, tokens, cu_span, driver, prefix_len, self.K,
                                  self.eos_id, self.max_span, out, self.ws_score, stream)
        else:
            ipd.score_span(ls, lt, tokens, cu_span, driver, prefix_len, self.K, self.eos_id, out,
                           self.ws_score, stream)

    def run_score(self, stream=None):
        self._score_call(self.logits_s, self.logits_t, self.tokens, self.cu_span, self.driver,
                         self.prefix_len, self.score, stream)

    def run_loss(self, stream=None):
        s = self.score
        ipd.split_loss(s["kl_rev"], s["kl_fwd"], s["source"], self.cu_span, s["n_emit"],
                       self.resp_len, self.agg_mode, self.dir_mode, self.out8, stream)

    def run(self, stream=None, overlap: bool = False):
        """The step's three calls.  The vocabulary pass and the loss read only
        the step's inputs (logits, tokens, request metadata) and each other,
        never the attention outputs, so with overlap=True they run on a side
        stream forked from `stream` and joined at the end: the row pass takes
        the SMs while the attention's planner runs, and the epilogue and the
        loss take the SMs that the first attention CTAs to finish leave
        free, inside the attention's tail."""
        if not overlap:
            self.run_attention(stream)
            self.run_score(stream)
            self.run_loss(stream)
            return
        main = stream if stream is not None else torch.cuda.current_stream(self.device)
        if getattr(self, "_side", None) is None:
            self._side = torch.cuda.Stream(device=self.device)
        side = self._side
        side.wait_stream(main)
        self.run_attention(main)
        self.run_score(side)
        self.run_loss(side)
        main.wait_stream(side)

    def capture(self, warmup: int = 2, overlap: bool = False) -> "torch.cuda.CUDAGraph":
        """Record one step (the three calls, five kernels) as a CUDA graph.

        The calls allocate nothing and never synchronise, so the whole step
        captures; each replay re-runs the step on the current contents of
        this object's buffers (same shapes and addresses), without the host
        work and launch gaps of issuing the calls one by one."""
        side = torch.cuda.Stream(device=self.device)
        side.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(side):
            for _ in range(warmup):
                self.run(overlap=overlap)
        torch.cuda.current_stream(self.device).wait_stream(side)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            self.run(overlap=overlap)
        return graph

    # -- one step end to end from host memory ---------------------------------
    def host_inputs(self, n_chunks: int = 4) -> dict:
        """Pinned host copies of every per-step input (each batch's queries and
        metadata, tokens, request metadata, both models' logits), plus the
        request-aligned chunk plan that run_from_host uses for the logits.
        Everything but the logits sits in one pinned buffer ("_arena") laid out
        like the step's device buffer; the other keys are views into it."""
        arena = self._in.mirror("cpu", pin=True)
        h = dict(arena.views)
        h["_arena"] = arena.buf
        h["logits_s"] = self.logits_s.cpu().pin_memory()
        h["logits_t"] = self.logits_t.cpu().pin_memory()
        bounds, cu_chunk = chunk_plan(h["cu_span"], n_chunks)
        h["cu_chunk"][:cu_chunk.numel()] = cu_chunk  # at most 2R + 1 entries
        h["_chunks"] = bounds
        return h

    def host_results(self) -> dict:
        """Pinned host buffers for the results of a host-fed step: the names of
        RESULT_NAMES plus "out8", views into one pinned buffer ("_arena") that
        run_from_host fills with one copy."""
        arena = self._res.mirror("cpu", pin=True)
        out = dict(arena.views)
        out["_arena"] = arena.buf
        return out

    def run_from_host(self, host: dict, results: dict, stream=None, host_logits: bool = False):
        """One step whose inputs sit in pinned host memory (``host_inputs``)
        and whose results (verdict per request, source per token, loss
        record) are copied back into ``results``: ``host_results()``, read
        back with one copy, or any dict of pinned tensors named like the
        score outputs plus "out8".  The caller synchronises ``stream``.

        The queries and metadata go first, in one copy, and the attention
        starts as soon as they land; the logits, most of the bytes, follow on
        a copy stream in request-aligned chunks, and each chunk is scored as
        soon as it lands, so that only the last chunk's scoring and the loss
        follow the transfer.  Every kernel sees the same data as in run(), so
        the results are bit-identical.

        host_logits=True (needed-rows steps only, with pinned logits the
        device can read in place): the logits are not copied at all; the
        vocabulary pass reads its rows from host memory, so only the rows the
        verdict and the emitted positions need cross the host link."""
        if host_logits:
            if self.rows != "needed":
                raise ValueError("host_logits needs a step with rows='needed'")
            if not (ipd.device_readable(host["logits_s"]) and
                    ipd.device_readable(host["logits_t"])):
                raise ValueError("the host logits are not readable by the device in place")
            return self._run_from_host_logits(host, results, stream)
        main = stream if stream is not None else torch.cuda.current_stream(self.device)
        if getattr(self, "_copy", None) is None:
            self._copy = torch.cuda.Stream(device=self.device)
            self._scorer = torch.cuda.Stream(device=self.device)
        cp, sc = self._copy, self._scorer
        # the previous step's kernels are done with every buffer written here
        cp.wait_stream(main)
        sc.wait_stream(main)
        with torch.cuda.stream(main):
            self._in.buf.copy_(host["_arena"], non_blocking=True)
        meta = torch.cuda.Event()
        meta.record(main)
        self.run_attention(main)
        landed = []
        with torch.cuda.stream(cp):
            for r0, r1, t0, t1 in host["_chunks"]:
                if t1 > t0:
                    self.logits_s[t0:t1].copy_(host["logits_s"][t0:t1], non_blocking=True)
                    self.logits_t[t0:t1].copy_(host["logits_t"][t0:t1], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(cp)
                landed.append(ev)
        sc.wait_event(meta)
        cu_chunk = self._in.views["cu_chunk"]
        off = 0
        for (r0, r1, t0, t1), ev in zip(host["_chunks"], landed):
            sc.wait_event(ev)
            out = {n: self.score[n][t0:t1] for n, _ in ipd.SCORE_TOKEN_OUTPUTS}
            out.update({n: self.score[n][r0:r1] for n, _ in ipd.SCORE_REQ_OUTPUTS})
            self._score_call(self.logits_s[t0:t1], self.logits_t[t0:t1], self.tokens[t0:t1],
                             cu_chunk[off:off + r1 - r0 + 1], self.driver[r0:r1],
                             self.prefix_len[r0:r1], out, sc)
            off += r1 - r0 + 1
        main.wait_stream(sc)
        main.wait_stream(cp)
        self.run_loss(main)
        with torch.cuda.stream(main):
            if "_arena" in results:
                results["_arena"].copy_(self._res.buf, non_blocking=True)
            else:
                for name, t in results.items():
                    t.copy_(self.out8 if name == "out8" else self.score[name], non_blocking=True)

    def _run_from_host_logits(self, host: dict, results: dict, stream=None):
        main = stream if stream is not None else torch.cuda.current_stream(self.device)
        if getattr(self, "_scorer", None) is None:
            self._copy = torch.cuda.Stream(device=self.device)
            self._scorer = torch.cuda.Stream(device=self.device)
        sc = self._scorer
        sc.wait_stream(main)
        with torch.cuda.stream(main):
            self._in.buf.copy_(host["_arena"], non_blocking=True)
        meta = torch.cuda.Event()
        meta.record(main)
        self.run_attention(main)
        sc.wait_event(meta)
        self._score_call(host["logits_s"], host["logits_t"], self.tokens, self.cu_span,
                         self.driver, self.prefix_len, self.score, sc)
        main.wait_stream(sc)
        self.run_loss(main)
        with torch.cuda.stream(main):
            if "_arena" in results:
                results["_arena"].copy_(self._res.buf, non_blocking=True)
            else:
                for name, t in results.items():
                    t.copy_(self.out8 if name == "out8" else self.score[name], non_blocking=True)

    def capture_from_host(self, host: dict, results: dict, warmup: int = 2,
                          host_logits: bool = False) -> "torch.cuda.CUDAGraph":
        """run_from_host recorded as one CUDA graph: every copy and kernel of
        the step, with the same pinned host buffers and device buffers at
        each replay, without the per-call host work of issuing them."""
        side = torch.cuda.Stream(device=self.device)
        side.wait_stream(torch.cuda.current_stream(self.device))
        for _ in range(warmup):
            self.run_from_host(host, results, side, host_logits=host_logits)
        side.synchronize()
        torch.cuda.current_stream(self.device).wait_stream(side)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            self.run_from_host(host, results, torch.cuda.current_stream(self.device),
                               host_logits=host_logits)
        return graph

    # -- bytes the step must move (algorithmic) --------------------------------
    def attn_bytes(self, ctx: torch.Tensor) -> int:
        """KV pages read (exact lengths) + Q read + O written, both caches."""
        total = 0
        for b in self.verify + self.decode:
            hkv = b.cache.num_kv_heads
            seq = b._keep[2].cpu().to(torch.int64)
            total += int(seq.sum()) * hkv * 128 * 2 * 2          # K and V, bf16
            q = b._keep[0]
            total += 2 * q.numel() * q.element_size()              # Q in, O out
        return total

    def logits_bytes_full(self) -> int:
        return 2 * self.T * self.V * 2

    def logits_bytes_alg(self) -> int:
        """Verifier rows for positions 0..first_trans (clipped to the span) and
        proposer rows for the emitted positions (needs the step's outputs)."""
        cu = self.cu_span.cpu()
        ft = self.score["first_trans"].cpu()
        ne = self.score["n_emit"].cpu()
        rows = 0
        for r in range(self.R):
            k = int(cu[r + 1] - cu[r])
            rows += min(k, int(ft[r]) + 1) + int(ne[r])
        return rows * self.V * 2

    def vocab_rows_bytes(self) -> int:
        return self.logits_bytes_full()
