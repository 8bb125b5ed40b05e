"""Verify-step benchmark: verified tokens/s on one GB300 (and N replicas).

One step = the whole hot path on one batch: ipd_verify_attn (span-verify
attention on the verifier's cache co-launched with the proposer's decode
attention), the vocabulary pass + verdict (ipd_score_span_needed: the logits
rows the verdict and the emitted positions need; --rows all: ipd_score_span,
every row) and ipd_split_loss.
Inputs are synthetic, seeded, resident in HBM and larger than L2, so every
step streams its KV pages and logits from DRAM.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config I] [--impl reference]
  python bench.py --next-rows [--config I] [--steps K]
  python bench.py --attn-only [--config I] [--requests R] [--direction S|T] [--span LO HI]
  python bench.py --score-only [--config I] [--requests R] [--rows needed|all]

The headline workload is the full rollout-step mix (1024 requests, lognormal
contexts up to 32K, spans of 1-16 tokens, both directions, 120 GB of KV
pools), the largest that fits one GPU; the other full-size workloads follow
in a `per_config` record (device-timed the same way, fewer steps).
Prints one JSON line (rank 0).  ``--impl reference`` times the fp64 CPU
oracle (the only reference that exists for this path) on a bounded sample of
the same workload.
"""
from __future__ import annotations

import argparse
import json
import math
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# kernels one step launches: ipd_verify_attn (planner, attention; split tasks
# are merged inside the attention kernel), ipd_score_span (row pass,
# epilogue), ipd_split_loss (one)
LAUNCHES_PER_STEP = 5
METRIC = "verified tokens/s on 1 GB300; achieved HBM GB/s as % of peak"
UNIT = "tokens/s"
HBM_FALLBACK_GBS = 6800.0


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return HBM_FALLBACK_GBS, "fallback"


ATTN_SRC = os.path.join(ROOT, "paper_2609_36546_gb300", "csrc", "attn.cu")


def attn_code_key(src: str = ATTN_SRC) -> str:
    """Names the attention kernel's code: the first 16 hex digits of the
    SHA-256 of csrc/attn.cu with its // comments and blank lines removed, so
    that a comment edit does not retire an ncu record of the same code."""
    import hashlib
    lines = []
    for line in open(src, encoding="utf-8"):
        code = line.split("//", 1)[0].rstrip()
        if code:
            lines.append(code)
    return hashlib.sha256("\n".join(lines).encode()).hexdigest()[:16]


def _committed_traffic(cfg: int, attn_bytes: int, profiles: str = os.path.join(ROOT, "profiles"),
                       src: str = ATTN_SRC):
    """DRAM bytes per attention launch from the committed ncu record of this
    workload, or None when the kernel's code has changed since it was taken.
    The record is a capture of a smaller case of the same shape; its ratio of
    DRAM bytes to algorithmic bytes scales to this launch's bytes."""
    path = os.path.join(profiles, f"attn_traffic_cfg{cfg}.json")
    try:
        rec = json.load(open(path))
        if rec.get("attn_code_key") != attn_code_key(src):
            return None
        return int(round(rec["traffic_over_algorithmic"] * attn_bytes))
    except Exception:
        return None


def _workload_name(cfg: int) -> str:
    import ipd_synth as S
    s = S.CONFIGS[cfg]
    return (f"{s.name}: {s.n_req} requests, ctx {s.ctx}, span {s.span}, "
            f"direction {s.direction}, teacher 32Q/4KV + student 16Q/8KV heads, head_dim 128, "
            f"page 16, vocab {s.vocab}, logits '{s.logits}', K={s.K}, one attention layer per model")


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(index)], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "samples": len(sm), "reasons": sorted(reasons)}


def _smi_index(local_rank: int) -> int:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    ids = [v for v in vis.split(",") if v.strip()]
    if ids and all(v.strip().isdigit() for v in ids) and local_rank < len(ids):
        return int(ids[local_rank])
    try:
        n = len(subprocess.run(["nvidia-smi", "-L"], capture_output=True, text=True,
                               timeout=10).stdout.strip().splitlines())
        if n == 1:
            return 0
    except Exception:
        pass
    return local_rank


# ---------------------------------------------------------------------------
# oracle timing (cpu_baseline and --impl reference)
# ---------------------------------------------------------------------------
def _oracle_request(payload):
    """The oracle's full path for one request: verify + decode attention,
    the vocabulary pass of every span position, the verdict and the loss."""
    import numpy as np
    import oracle as O
    t0 = time.perf_counter()
    for q, kp, vp, L in payload["attn"]:
        O.paged_span_attention(q, kp, vp, np.arange(kp.shape[0]), L, payload["scale"])
    k = payload["ls"].shape[0]
    out = O.score_span(payload["ls"], payload["lt"], payload["tokens"], np.array([0, k]),
                       np.array([payload["driver"]]), np.array([payload["prefix"]]),
                       payload["K"], payload["eos"])
    O.split_loss(out["kl_rev"], out["kl_fwd"], out["source"], np.array([0, k]), out["n_emit"])
    return k, time.perf_counter() - t0


def _request_payload(step, w, r):
    import numpy as np
    import torch
    from tests.parity import u16
    pay = {"attn": [], "scale": step.scale, "K": step.K, "eos": step.eos_id,
           "driver": int(w.driver[r]), "prefix": int(w.ctx[r] - w.span[r])}
    for name, b, idx, cache in step.batches:
        pos = (idx == r).nonzero().flatten()
        if pos.numel() == 0:
            continue
        j = int(pos[0])
        q, cu_q, seq, ptab, _ = b._keep
        cu = cu_q.cpu()
        L = int(seq[j])
        npg = (L + 15) // 16
        pages = ptab[j, :npg].to(torch.int64)
        c = step.cache_t if cache == "teacher" else step.cache_s
        pay["attn"].append((u16(q[int(cu[j]):int(cu[j + 1])]), u16(c.k_pages.index_select(0, pages)),
                            u16(c.v_pages.index_select(0, pages)), L))
    t0, t1 = int(step.cu_span[r]), int(step.cu_span[r + 1])
    pay["ls"] = u16(step.logits_s[t0:t1])
    pay["lt"] = u16(step.logits_t[t0:t1])
    pay["tokens"] = step.tokens[t0:t1].cpu().numpy()
    return pay


def cpu_baseline(step, w, budget_s: float = 25.0) -> dict:
    """The oracle on the host cores (a spawn pool, one request per task) on a
    bounded sample of the same workload: whole requests, taken in order."""
    cores = max(1, min(os.cpu_count() or 1, 32))
    ctx = mp.get_context("spawn")
    env_keep = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS",
                                               "MKL_NUM_THREADS")}
    for k in env_keep:
        os.environ[k] = "1"
    try:
        with ctx.Pool(cores) as pool:
            # one request alone first, to size the sample to the budget
            first = _request_payload(step, w, 0)
            k0, t_one = pool.apply(_oracle_request, (first,))
            n_req = max(1, min(step.R, int(budget_s / max(t_one, 1e-3) * cores * 0.8)))
            n_req = max(cores, n_req) if step.R >= cores else step.R
            n_req = min(n_req, step.R)
            payloads = [_request_payload(step, w, r) for r in range(n_req)]
            t0 = time.perf_counter()
            res = pool.map(_oracle_request, payloads, chunksize=1)
            wall = time.perf_counter() - t0
    finally:
        for k, v in env_keep.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    toks = sum(k for k, _ in res)
    return {"value": toks / wall, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"first {n_req} of {step.R} requests ({toks} span tokens), whole oracle path "
                      f"per request (attention of both caches, vocabulary pass, verdict, loss), "
                      f"numpy fp64, one process per core, BLAS single-threaded; wall {wall:.1f} s"}


# ---------------------------------------------------------------------------
def _init_dist(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("nccl", rank=rank, world_size=world,
                                device_id=torch.device("cuda", local))
    return world, rank, local


def _barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def _max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _sum_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda")
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def run_reference(args):
    """--impl reference: the fp64 oracle on the host, one verified token per
    step (its verifier attention query, the request's decode query, the
    vocabulary pass of its two logits rows, verdict and loss)."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import numpy as np
    import ipd_synth as S
    import oracle as O
    # a small resident sample of the workload, generated on the host
    spec = S.CONFIGS[args.config]
    n_req = 2
    sample_spec = S.Spec(spec.name + " (sample)", n_req, spec.ctx, spec.span, "S" if spec.direction
                         in ("S", "half", "bernoulli") else "T", spec.vocab, spec.logits,
                         sigma=spec.sigma, K=spec.K)
    w = S.make_workload(sample_spec, seed=args.config, device="cpu")
    from tests.parity import u16
    scale = 1.0 / math.sqrt(128.0)
    toks = w.tokens.numpy()
    cu = w.cu_span.numpy()
    ls, lt = u16(w.logits_s), u16(w.logits_t)

    def one_token(i):
        r = i % n_req
        t = int(cu[r]) + (i // n_req) % int(w.span[r])
        pos = t - int(cu[r])
        L = int(w.ctx[r])
        npg = (L + 15) // 16
        ver, prop = (w.teacher, w.student) if int(w.driver[r]) == 0 else (w.student, w.teacher)
        qv = w.q_verify_t if int(w.driver[r]) == 0 else w.q_verify_s
        qd = w.q_decode_s if int(w.driver[r]) == 0 else w.q_decode_t
        rows = ver.page_table[r, :npg].long()
        prow = prop.page_table[r, :npg].long()
        qi = u16(qv[t:t + 1])
        O.paged_span_attention(qi, u16(ver.k_pages[rows]), u16(ver.v_pages[rows]),
                               np.arange(npg), L - int(w.span[r]) + pos + 1, scale)
        O.paged_span_attention(u16(qd[r:r + 1]), u16(prop.k_pages[prow]), u16(prop.v_pages[prow]),
                               np.arange(npg), L, scale)
        out = O.score_span(ls[t:t + 1], lt[t:t + 1], toks[t:t + 1], np.array([0, 1]),
                           w.driver[r:r + 1].numpy(), np.array([L - 1]), w.spec.K, -1)
        O.split_loss(out["kl_rev"], out["kl_fwd"], out["source"], np.array([0, 1]), out["n_emit"])

    for i in range(args.warmup):
        one_token(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        one_token(args.warmup + i)
    el = time.perf_counter() - t0
    value = args.steps / el
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * el / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": _workload_name(args.config)},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": "one verified token per step (its verify query over the "
                                       "verifier cache, the request's decode query, both logits "
                                       "rows, verdict, loss), 2 host-generated requests of the "
                                       "workload's shape, cycled"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def measure_config(cfg, K, W, world, rank, stream, sampler=None, rows="needed"):
    """Device-timed steps of one workload: per-call events, the attention
    kernel's own events, and the step replayed from CUDA graphs.  Returns the
    step, the workload and a dict of figures (max over ranks)."""
    import torch
    import ipd_synth as S
    from paper_2609_36546_gb300 import VerifyStep, ipd

    w = S.make_workload(cfg, seed=cfg + 1000 * rank, device="cuda")
    step = VerifyStep.from_workload(w, device="cuda", rows=rows)
    T_tok = step.T
    # warm-up (also yields the verdict used for the algorithmic byte count)
    for _ in range(W):
        step.run(stream)
    torch.cuda.synchronize()
    if ipd.device_error() != 0:
        raise RuntimeError("device-side check failed during warm-up")
    attn_bytes = step.attn_bytes(w.ctx)
    logits_alg = step.logits_bytes_alg()
    logits_full = step.logits_bytes_full()
    # coverage among the positions up to each request's first transition (the
    # ones both vocabulary passes decide; the needed-rows pass leaves later
    # positions unread)
    if T_tok:
        cu = step.cu_span.cpu()
        lens = cu[1:] - cu[:-1]
        pos = torch.arange(T_tok) - torch.repeat_interleave(cu[:-1], lens)
        dec = pos <= torch.repeat_interleave(step.score["first_trans"].cpu(), lens)
        accept_rate = float(step.score["covered"].cpu()[dec].float().mean())
    else:
        accept_rate = 0.0
    emitted = int(step.score["n_emit"].sum())

    # ---- K steps call by call, per-call events on the launching stream ----
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    _barrier(world)
    torch.cuda.synchronize()
    # the library also records events around the attention kernel alone
    # (without its planner launch), on the same stream
    ipd.set_attn_kernel_timing(True)
    t_start.record(stream)
    for i in range(K):
        e = ev[i]
        e[0].record(stream)
        step.run_attention(stream)
        e[1].record(stream)
        step.run_score(stream)
        e[2].record(stream)
        step.run_loss(stream)
        e[3].record(stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    _barrier(world)
    el_direct_ms = t_start.elapsed_time(t_end)
    k_total_ms, k_launches = ipd.attn_kernel_time()
    ipd.set_attn_kernel_timing(False)
    attn_kernel_ms = k_total_ms / max(k_launches, 1)
    attn_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in ev)
    score_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in ev)
    loss_ms = statistics.mean(e[2].elapsed_time(e[3]) for e in ev)

    # ---- the same K steps replayed from a CUDA graph of one step (same
    # kernels and buffers, no per-call host work): the step time ----
    graph = step.capture(overlap=True)
    torch.cuda.synchronize()
    g_start = torch.cuda.Event(enable_timing=True)
    g_end = torch.cuda.Event(enable_timing=True)
    _barrier(world)
    torch.cuda.synchronize()
    g_start.record(stream)
    for i in range(K):
        graph.replay()
    g_end.record(stream)
    torch.cuda.synchronize()
    _barrier(world)
    clocks = sampler.stop() if sampler else None
    if ipd.device_error() != 0:
        raise RuntimeError("device-side check failed during the timed steps")
    el_ms = g_start.elapsed_time(g_end)
    # the same graph with every call on one stream (no overlap), for reference
    graph1 = step.capture(overlap=False)
    torch.cuda.synchronize()
    g_start.record(stream)
    for i in range(K):
        graph1.replay()
    g_end.record(stream)
    torch.cuda.synchronize()
    del graph, graph1
    ms_step_one_stream = _max_over_ranks(g_start.elapsed_time(g_end), world) / K
    el_max = _max_over_ranks(el_ms, world)
    tokens_all = _sum_over_ranks(float(T_tok * K), world)
    ms_step = el_max / K
    peak, peak_kind = _peaks()
    achieved = attn_bytes / (attn_kernel_ms / 1e3) / 1e9
    achieved_call = attn_bytes / (attn_ms / 1e3) / 1e9
    step_alg = attn_bytes + logits_alg
    step_full = attn_bytes + logits_full
    fig = {
        "value": tokens_all / (el_max / 1e3), "ms_per_step": ms_step, "tokens_per_step": T_tok,
        "requests": step.R, "clocks": clocks,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": _committed_traffic(cfg, attn_bytes),
                     "peak_kind": peak_kind,
                     "kernel": "attn_kernel (the attention launch of ipd_verify_attn; split "
                               "tasks merge inside it)",
                     "bytes_per_launch": attn_bytes, "ms_per_launch": attn_kernel_ms,
                     "launches_timed": k_launches,
                     "call": {"what": "ipd_verify_attn: planner launch + attention launch",
                              "ms": attn_ms, "achieved": achieved_call,
                              "frac": achieved_call / peak}},
        "step_hbm": {"bytes_alg": step_alg, "bytes_full": step_full,
                     "gbs_alg": step_alg / (ms_step / 1e3) / 1e9,
                     "gbs_full": step_full / (ms_step / 1e3) / 1e9,
                     "frac_alg_of_measured": step_alg / (ms_step / 1e3) / 1e9 / peak,
                     "frac_full_of_nominal_8tbs": step_full / (ms_step / 1e3) / 1e9 / 8000.0},
        "calls_ms": {"verify_attn": attn_ms, "score_span": score_ms, "split_loss": loss_ms},
        "ms_per_step_one_stream_graph": ms_step_one_stream,
        "ms_per_step_direct_calls": _max_over_ranks(el_direct_ms, world) / K,
        "acceptance": {"coverage_rate_to_transition": accept_rate,
                       "emitted_tokens_per_step": emitted},
    }
    return step, w, fig


def run_gpu(args):
    import torch
    world, rank, local = _init_dist(args)
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()

    cfg = args.config
    stream = torch.cuda.current_stream()
    K = args.steps
    sampler = ClockSampler(_smi_index(local)) if rank == 0 else None
    time.sleep(0.3 if sampler else 0.0)
    step, w, fig = measure_config(cfg, K, max(3, args.warmup), world, rank, stream, sampler,
                                  rows=args.rows)

    # ---- end to end through host buffers ----
    e2e = run_e2e(step, w, min(K, args.e2e_steps), stream, world)
    cpu = cpu_baseline(step, w) if (world == 1 and rank == 0 and not args.no_cpu_baseline) \
        else None
    del step, w
    torch.cuda.empty_cache()

    # ---- the other full-size workloads, device-timed the same way (fewer
    # steps, no end-to-end leg), one at a time ----
    per_config = {}
    if world == 1 and not args.no_per_config:
        import ipd_synth as S
        for c in range(1, len(S.CONFIGS)):
            if c == cfg:
                continue
            st, wc, f = measure_config(c, min(K, args.per_config_steps), max(3, args.warmup),
                                       world, rank, stream, rows=args.rows)
            per_config[S.CONFIGS[c].name] = {
                "workload": _workload_name(c), "value": f["value"], "unit": UNIT,
                "ms_per_step": f["ms_per_step"],
                "roofline_frac": f["roofline"]["frac"],
                "attn_kernel_ms": f["roofline"]["ms_per_launch"],
                "attn_call_frac": f["roofline"]["call"]["frac"],
                "step_hbm_frac_alg_of_measured": f["step_hbm"]["frac_alg_of_measured"],
                "traffic": f["roofline"]["traffic"]}
            del st, wc
            torch.cuda.empty_cache()
    if rank != 0:
        return
    line = {
        "metric": METRIC, "value": fig["value"], "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": max(3, args.warmup), "ms_per_step": fig["ms_per_step"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": _workload_name(cfg), "seed": cfg,
                   "tokens_per_step": fig["tokens_per_step"], "requests": fig["requests"],
                   "l2": "inputs larger than L2 (no flush needed)",
                   "vocab_pass": ("logits rows the verdict and the emitted positions need "
                                  "(ipd_score_span_needed)" if args.rows == "needed" else
                                  "every logits row (ipd_score_span)"),
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "roofline": fig["roofline"], "step_hbm": fig["step_hbm"], "calls_ms": fig["calls_ms"],
        "ms_per_step_one_stream_graph": fig["ms_per_step_one_stream_graph"],
        "ms_per_step_direct_calls": fig["ms_per_step_direct_calls"],
        "timing": "value: K steps replayed from a CUDA graph of one step (the vocabulary pass "
                  "and the loss on a forked stream, joined at the end); calls_ms and the "
                  "roofline: the same K steps issued call by call on one stream, CUDA events "
                  "around each call, and around each attention kernel launch (recorded by the "
                  "library on the call's stream)",
        "acceptance": fig["acceptance"],
        "e2e": e2e, "clocks": fig["clocks"],
        "gpu_launches": LAUNCHES_PER_STEP * K,
    }
    if cpu is not None:
        line["cpu_baseline"] = cpu
    if per_config:
        line["per_config"] = per_config
    print(json.dumps(line), flush=True)


def run_e2e(step, w, K, stream, world):
    """The same step through host buffers, via VerifyStep.run_from_host: the
    per-step inputs (queries and their metadata, both models' logits, tokens,
    request metadata) come from pinned host memory, the step runs, and its
    results (per-request verdict, per-token sources, loss record) are copied
    back and read before the next step; the KV pools stay resident (they are
    the cache state, not step inputs).  Queries and metadata go in one copy
    and the attention starts when they land.  With the needed-rows
    vocabulary pass and logits the device can read in place, the pass reads
    its rows straight from host memory, so only the rows it needs cross the
    link (counted from the row records' "not read" flags); otherwise the
    logits are copied in four chunks, each scored as it lands.  The step, its
    copies included, is replayed from one CUDA graph
    (VerifyStep.capture_from_host)."""
    import torch
    from paper_2609_36546_gb300 import ipd
    host = step.host_inputs(n_chunks=4)
    results = step.host_results()
    d2h = results["_arena"].numel()
    in_place = step.rows == "needed" and ipd.device_readable(host["logits_s"]) and \
        ipd.device_readable(host["logits_t"])

    def timed(host_logits):
        graph = step.capture_from_host(host, results, host_logits=host_logits)
        for _ in range(2):
            graph.replay()
            stream.synchronize()
        _barrier(world)
        t0 = time.perf_counter()
        for _ in range(K):
            graph.replay()                # inputs in, the step, results out
            stream.synchronize()          # the engine reads the verdict before the next step
        el = _max_over_ranks(time.perf_counter() - t0, world)
        del graph
        return _sum_over_ranks(float(step.T * K), world) / el

    row_bytes = step.V * 2
    all_rows = 2 * step.T * row_bytes
    copy_all = timed(False)
    out = {"unit": UNIT, "d2h_bytes_per_step": d2h, "steps": K,
           "copy_all_logits": {"value": copy_all,
                               "h2d_bytes_per_step": host["_arena"].numel() + all_rows}}
    if in_place:
        value = timed(True)
        # rows one more such step reads: the row records' flags (byte 12 of
        # each 272-byte record), preset to 2; the pass sets 0 (read) or 1 (not
        # read), or leaves them when it read every row in one wave
        n = 2 * step.T
        flags = step.ws_score[:n * 272].view(n, 272)[:, 12:16]
        flags.copy_(torch.tensor([2, 0, 0, 0], dtype=torch.uint8, device=flags.device)
                    .expand_as(flags))
        step.run_from_host(host, results, stream, host_logits=True)
        stream.synchronize()
        f = flags.contiguous().view(torch.int32).flatten()
        read = n if bool((f == 2).all()) else int((f == 0).sum())
        out.update({"value": value, "h2d_bytes_per_step": host["_arena"].numel() + read * row_bytes,
                    "logits_rows_read_last_step": read, "logits_rows": n,
                    "note": "pinned host inputs: queries, tokens and metadata in one copy; the "
                            "vocabulary pass reads the logits rows it needs from pinned host "
                            "memory in place (the rest never cross the link); results back in "
                            "one copy; synchronised per step; KV pools resident; the step "
                            "replayed from one CUDA graph. copy_all_logits: the same step "
                            "copying both models' logits in four chunks first"})
    else:
        out.update({"value": copy_all, "h2d_bytes_per_step": host["_arena"].numel() + all_rows,
                    "note": "pinned host -> device inputs (Q, tokens and metadata in one copy, "
                            "the logits in 4 chunks) and device -> host results (one copy) each "
                            "step, synchronised per step; KV pools resident; the attention "
                            "overlaps the logits transfer, and each chunk is scored as it lands; "
                            "the step with its copies replayed from one CUDA graph"})
    return out


# ---------------------------------------------------------------------------
# --next-rows: the calls beyond the step (rules and by-products, full KL, the
# loss gradient), each timed alone from a CUDA graph of one call, with its
# algorithmic bytes and the oracle timed on a sample beside it
# ---------------------------------------------------------------------------
def _graph_ms(fn, reps: int) -> float:
    import torch
    cur = torch.cuda.current_stream()
    side = torch.cuda.Stream()
    side.wait_stream(cur)
    with torch.cuda.stream(side):
        for _ in range(3):
            fn()
    cur.wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    for _ in range(3):
        g.replay()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record(cur)
    for _ in range(reps):
        g.replay()
    b.record(cur)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def _oracle_ms(fn, n: int) -> float:
    t0 = time.perf_counter()
    fn()
    return (time.perf_counter() - t0) * 1e3 / max(n, 1)


def run_next_rows(args):
    import numpy as np
    import torch
    import __graft_entry__
    __graft_entry__.build()
    import ipd_synth as S
    import oracle as O
    from paper_2609_36546_gb300 import VerifyStep, ipd
    from tests.parity import u16

    cfg = args.config
    w = S.make_workload(cfg, seed=cfg, device="cuda")
    st = VerifyStep.from_workload(w, device="cuda")
    T, V, K, R = st.T, st.V, st.K, st.R
    reps = max(5, min(args.steps, 200))
    peak, peak_kind = _peaks()
    dev = "cuda"
    ent_s = torch.empty(T, device=dev)
    ent_t = torch.empty(T, device=dev)
    ovl = torch.empty(T, device=dev)
    tks = torch.empty(T, K, device=dev, dtype=torch.int32)
    tkt = torch.empty_like(tks)
    rev = torch.empty(T, device=dev)
    fwd = torch.empty(T, device=dev)
    gi = torch.empty(T, 2 * K, device=dev, dtype=torch.int32)
    gv = torch.empty(T, 2 * K, device=dev)
    dense32 = torch.empty(T, V, device=dev, dtype=torch.float32)
    dense16 = torch.empty(T, V, device=dev, dtype=torch.bfloat16)
    tau = 3.0

    def score_ex():
        ipd.score_span_ex(st.logits_s, st.logits_t, st.tokens, st.cu_span, st.driver,
                          st.prefix_len, K, st.eos_id, st.score, st.ws_score,
                          ipd.RULE_ENTROPY_S, ipd.RULE_ALWAYS, tau, 0.0, ent_s, ent_t, ovl, tks, tkt)

    nxt = torch.empty(R, device=dev, dtype=torch.int32)
    seed = 0x5EED

    def score_draw():
        ipd.score_span_ex(st.logits_s, st.logits_t, st.tokens, st.cu_span, st.driver,
                          st.prefix_len, K, st.eos_id, st.score, st.ws_score, next_token=nxt,
                          sample_seed=seed)

    # standalone draws: one row per request (the proposers' decode rows stand-in)
    dec_rows = st.logits_s[:R] if T >= R else st.logits_s
    n_dec = dec_rows.shape[0]
    draw_ids = torch.arange(n_dec, device=dev, dtype=torch.int64)
    dec_tok = torch.empty(n_dec, device=dev, dtype=torch.int32)
    ws_s = torch.empty(max(8, ipd.sample_workspace_size(n_dec, V)), device=dev, dtype=torch.uint8)
    # KV appends of the step: every batch's new rows (span rows for the verifiers,
    # one row per request for the proposers) at the last positions of each sequence
    appends = []
    kv_bytes = 0
    for name, b, idx, cname in st.batches:
        q, cu_q, seq, ptab = b._keep[0], b._keep[1], b._keep[2], b._keep[3]
        cache = st.cache_t if cname == "teacher" else st.cache_s
        hkv = cache.k_pages.shape[1]
        nrow = int(q.shape[0])
        kn = torch.randn(nrow, hkv, 128, device=dev).to(torch.bfloat16)
        vn = torch.randn(nrow, hkv, 128, device=dev).to(torch.bfloat16)
        appends.append((cache, kn, vn, cu_q, seq, ptab))
        kv_bytes += 2 * 2 * nrow * hkv * 128 * 2       # K and V rows, read and written

    def kv_all():  # the step's appends in one launch
        ipd.kv_append_many(appends)

    def kv_each():  # one call (one launch) per append
        for cache, kn, vn, cu_q, seq, ptab in appends:
            ipd.kv_append(cache, kn, vn, cu_q, seq, ptab)

    score_ex()
    st.run_loss()
    grad_args = (st.logits_s, st.logits_t, tks, tkt, st.score["source"], st.cu_span,
                 st.score["n_emit"], st.resp_len, st.out8, K, st.agg_mode, st.dir_mode, 1.0, gi, gv)
    sampler = ClockSampler(_smi_index(0))
    time.sleep(0.3)
    rows_bytes = 2 * T * V * 2
    t_plain = _graph_ms(st.run_score, reps)
    t_ex = _graph_ms(score_ex, reps)
    t_kl = _graph_ms(lambda: ipd.full_kl(st.logits_s, st.logits_t, rev, fwd), reps)
    t_gs = _graph_ms(lambda: ipd.split_loss_grad(*grad_args), reps)
    t_g32 = _graph_ms(lambda: ipd.split_loss_grad(*grad_args, dense32), reps)
    t_g16 = _graph_ms(lambda: ipd.split_loss_grad(*grad_args, dense16), reps)
    t_draw = _graph_ms(score_draw, reps)
    t_samp = _graph_ms(lambda: ipd.sample(dec_rows, seed, draw_ids, dec_tok, ws_s), reps)
    t_kv = _graph_ms(kv_all, reps)
    t_kv_each = _graph_ms(kv_each, reps)
    clocks = sampler.stop()
    torch.cuda.synchronize()
    if ipd.device_error() != 0:
        raise RuntimeError("device-side check failed")
    n_emitted = int((st.score["source"] != 255).sum())

    # the oracle on a sample of the same inputs
    n_s = min(4, T)
    ls_h, lt_h = u16(st.logits_s[:n_s]), u16(st.logits_t[:n_s])
    ls64, lt64 = O.bf16_to_f64(ls_h), O.bf16_to_f64(lt_h)
    o_kl = _oracle_ms(lambda: [O.full_kl(ls64[i], lt64[i]) for i in range(n_s)], n_s)
    r_s = 0
    cu_h = st.cu_span.cpu().numpy()
    while r_s < R and cu_h[r_s + 1] == 0:
        r_s += 1
    t0, t1 = int(cu_h[r_s]), int(cu_h[r_s + 1])
    sub_cu = np.array([0, t1 - t0])
    sub = lambda x: x[t0:t1]
    ls_r, lt_r = u16(sub(st.logits_s)), u16(sub(st.logits_t))
    o_ex = _oracle_ms(lambda: O.score_span(
        ls_r, lt_r, sub(st.tokens).cpu().numpy(), sub_cu, st.driver[r_s:r_s + 1].cpu().numpy(),
        st.prefix_len[r_s:r_s + 1].cpu().numpy(), K, st.eos_id, takeover_rule=O.RULE_ENTROPY_S,
        handback_rule=O.RULE_ALWAYS, takeover_tau=tau), t1 - t0)
    src_r = sub(st.score["source"]).cpu().numpy()
    ne_r = st.score["n_emit"][r_s:r_s + 1].cpu().numpy()
    o_g = _oracle_ms(lambda: O.split_loss_grad(O.bf16_to_f64(ls_r), O.bf16_to_f64(lt_r), src_r,
                                               sub_cu, ne_r, None, K), t1 - t0)
    dec_h = u16(dec_rows[:n_s])
    o_samp = _oracle_ms(lambda: [O.sample_token(dec_h[i], seed, i) for i in range(n_s)], n_s)
    # the oracle's append of one request's span rows, on a pool of that request's pages
    cache0, kn0, vn0, cu0, seq0, pt0 = appends[0]
    cu0h, seq0h, pt0h = cu0.cpu().numpy(), seq0.cpu().numpy(), pt0.cpu().numpy()
    n0 = int(cu0h[1] - cu0h[0])
    pg = [int(x) for x in pt0h[0, :(int(seq0h[0]) + 15) // 16]]
    kp0 = u16(cache0.k_pages[pg]); vp0 = u16(cache0.v_pages[pg])
    o_kv = _oracle_ms(lambda: O.kv_append(kp0, vp0, u16(kn0[:n0]), u16(vn0[:n0]), np.array([0, n0]),
                                          seq0h[:1], np.arange(len(pg))[None, :]), n0)

    def row(ms, nbytes, oracle_ms_pos, note):
        gbs = nbytes / (ms / 1e3) / 1e9
        return {"ms": ms, "us_per_position": ms * 1e3 / max(T, 1), "bytes": nbytes, "gbs": gbs,
                "frac": gbs / peak, "oracle_ms_per_position": oracle_ms_pos, "note": note}

    sparse_bytes = T * 2 * K * 4 * 2 + T * 2 * K * 2 * 2 + n_emitted * 2 * K * 8
    line = {
        "mode": "next_rows", "config": {"workload": _workload_name(cfg), "seed": cfg,
                                         "tokens": T, "requests": R, "vocab": V, "K": K},
        "peak": peak, "peak_kind": peak_kind, "reps": reps,
        "timing": "each call alone, replayed from a CUDA graph of one call; CUDA events "
                  "around the replays; inputs larger than L2",
        "rows": {
            "score_span (default step call, for comparison)": row(
                t_plain, rows_bytes, None, "full rows of both models read once"),
            "score_span_ex (entropy-S takeover, always handback, entropies, overlap, "
            "top-K lists)": row(t_ex, rows_bytes, o_ex, "full rows of both models read once"),
            "full_kl": row(t_kl, rows_bytes, o_kl, "full rows of both models read once"),
            "split_loss_grad sparse": row(t_gs, sparse_bytes, o_g,
                                          "top-K lists + 4K gathered logits + 2K (id, value)"),
            "split_loss_grad sparse + dense fp32": row(t_g32, T * V * 4 + sparse_bytes, None,
                                                       "dense [T, V] fp32 written"),
            "split_loss_grad sparse + dense bf16": row(t_g16, T * V * 2 + sparse_bytes, None,
                                                       "dense [T, V] bf16 written"),
            "score_span_ex + next-token draw": row(
                t_draw, rows_bytes + R * V * 2, None,
                "score pass, then one row per request re-read for the draw"),
            "sample (one row per request)": dict(row(
                t_samp, n_dec * V * 2, o_samp, "ALU-bound: Philox + two lg2 per entry"),
                rows=n_dec, us_per_row=t_samp * 1e3 / max(n_dec, 1),
                oracle_ms_per_row=o_samp),
            "kv_append (all span and decode rows of the step)": dict(row(
                t_kv, kv_bytes, o_kv, "latency-bound: ~1-4 MB per step"),
                oracle_ms_per_row=o_kv, appends=len(appends), launches=1,
                ms_one_call_per_append=t_kv_each),
        },
        "oracle_sample": f"full_kl and sample: {n_s} rows; score_span_ex and split_loss_grad: "
                         f"request {r_s} ({t1 - t0} positions); kv_append: one request's "
                         f"{n0} rows; numpy, one core",
        "clocks": clocks,
    }
    print(json.dumps(line), flush=True)


def _reduced_workload(args):
    """The workload of configuration --config with the --requests,
    --direction and --span changes (pools then hold only the pages used)."""
    import dataclasses
    import ipd_synth as S
    spec = S.CONFIGS[args.config]
    changes = {}
    if args.requests:
        changes.update(n_req=args.requests, pool_bytes=None)
    if args.direction:
        changes.update(direction=args.direction)
    if args.span:
        changes.update(span=("uniform", args.span[0], args.span[1]))
    if changes:
        spec = dataclasses.replace(spec, name=spec.name + " (shape kept, " +
                                   ", ".join(f"{k}={v}" for k, v in changes.items()) + ")",
                                   **changes)
    return spec, S.make_workload(spec, seed=args.config, device="cuda")


def run_score_only(args):
    """--score-only: only the vocabulary pass and verdict of a workload shaped
    like configuration --config (same changes as --attn-only), in the mode
    --rows names; the case an ncu capture of the row kernel runs.  Prints one
    JSON line: the rows read, the bytes they hold, and the mean call time."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import VerifyStep, ipd
    spec, w = _reduced_workload(args)
    step = VerifyStep.from_workload(w, device="cuda", rows=args.rows)
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        step.run_score(stream)
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step.run_score(stream)
    t1.record(stream)
    torch.cuda.synchronize()
    if ipd.device_error() != 0:
        raise RuntimeError("device-side check failed")
    ms = t0.elapsed_time(t1) / max(args.steps, 1)
    row_bytes = step.V * 2
    # rows one more call reads: the row records' "not read" flags (one record
    # of 272 bytes per row, the flag at byte 12), preset to 2.  A needed-rows
    # pass over several waves writes every flag (0 read, 1 skipped); a call
    # that leaves them at 2 took the full pass and read every row.
    n_rows = 2 * step.T
    read = n_rows
    if args.rows == "needed" and n_rows:
        flags = step.ws_score[:n_rows * 272].view(n_rows, 272)[:, 12:16]
        flags.copy_(torch.tensor([2, 0, 0, 0], dtype=torch.uint8, device=flags.device)
                    .expand_as(flags))
        step.run_score(stream)
        torch.cuda.synchronize()
        f = flags.contiguous().view(torch.int32).flatten()
        if not bool((f == 2).all()):
            read = int((f == 0).sum())
    print(json.dumps({"workload": spec.name, "requests": spec.n_req, "rows": args.rows,
                      "logits_rows": n_rows, "rows_read": read, "bytes_read": read * row_bytes,
                      "emitted": int(step.score["n_emit"].sum()), "ms_per_call": ms,
                      "calls": args.steps}), flush=True)


def run_attn_only(args):
    """--attn-only: only the attention call (planner + attention launch) of a
    workload shaped like configuration --config, optionally with fewer
    requests (--requests; pools then hold only the pages used), one direction
    (--direction S|T) or other span lengths (--span LO HI).  A small case of
    this kind is what an ncu capture runs; it prints one JSON line with the
    algorithmic bytes and the mean time of the attention launch."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_36546_gb300 import VerifyStep, ipd
    spec, w = _reduced_workload(args)
    step = VerifyStep.from_workload(w, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        step.run_attention(stream)
    torch.cuda.synchronize()
    ipd.set_attn_kernel_timing(True)
    for _ in range(args.steps):
        step.run_attention(stream)
    ms, n = ipd.attn_kernel_time()
    ipd.set_attn_kernel_timing(False)
    if ipd.device_error() != 0:
        raise RuntimeError("device-side check failed")
    nbytes = step.attn_bytes(w.ctx)
    ms /= max(n, 1)
    peak, kind = _peaks()
    print(json.dumps({"workload": spec.name, "requests": spec.n_req, "launches": n,
                      "bytes_per_launch": nbytes, "ms_per_launch": ms,
                      "gbs": nbytes / ms / 1e6, "frac": nbytes / ms / 1e6 / peak,
                      "peak_kind": kind}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    # the largest single-GPU workload: the full rollout-step mix
    ap.add_argument("--config", type=int, default=4)
    ap.add_argument("--impl", default="ipd", choices=["ipd", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=200)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-per-config", action="store_true",
                    help="skip the device-timed figures of the other workloads")
    ap.add_argument("--per-config-steps", type=int, default=100)
    ap.add_argument("--rows", choices=["needed", "all"], default="needed",
                    help="vocabulary pass of the step: only the logits rows the verdict and "
                         "the emitted positions need, or every row")
    ap.add_argument("--next-rows", action="store_true",
                    help="time the calls beyond the step instead (one GPU)")
    ap.add_argument("--attn-only", action="store_true",
                    help="time only the attention call (profiling cases; one GPU)")
    ap.add_argument("--score-only", action="store_true",
                    help="time only the vocabulary pass and verdict (profiling cases; one GPU)")
    ap.add_argument("--requests", type=int, default=0,
                    help="--attn-only / --score-only: requests of the workload (pools sized "
                         "to them)")
    ap.add_argument("--direction", choices=["S", "T", "half", "bernoulli"], default=None,
                    help="--attn-only / --score-only: which model proposes")
    ap.add_argument("--span", type=int, nargs=2, default=None,
                    help="--attn-only / --score-only: span lengths drawn uniformly in [LO, HI]")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    if args.next_rows:
        run_next_rows(args)
    elif args.attn_only:
        run_attn_only(args)
    elif args.score_only:
        run_score_only(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
