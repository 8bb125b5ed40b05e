"""ctypes binding of libipd.so: argument marshalling only.

Every function here forwards torch tensors (device memory) as raw pointers to
the C ABI declared in include/ipd.h and raises IpdError on a non-zero status.
No step of the computation runs in Python, and there is no fallback: if the
shared library cannot be loaded, importing the binding fails.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libipd.so")

IPD_OK = 0
STATUS = {0: "IPD_OK", 1: "IPD_ERR_INVALID_ARG", 2: "IPD_ERR_UNSUPPORTED", 3: "IPD_ERR_WORKSPACE",
          4: "IPD_ERR_CUDA", 5: "IPD_ERR_TIMEOUT", 6: "IPD_ERR_DEVICE", 7: "IPD_ERR_CAPACITY"}
STATUS_CODES = {v: k for k, v in STATUS.items()}
DEVERR = {0: "none", 1: "page id", 2: "seq len", 3: "token id", 4: "plan overflow", 5: "wait",
          6: "span offsets"}

DIR_SPLIT, DIR_REVERSE, DIR_FORWARD, DIR_INVERSE = 0, 1, 2, 3
AGG_SEQ_MEAN_TOKEN_MEAN, AGG_GLOBAL_TOKEN_MEAN = 0, 1
LOSS_FIELDS = ("loss", "sum_on", "sum_off", "n_on", "n_off", "intervention_ratio", "numer", "denom")

# Exported symbols of include/ipd.h (checked by the CPU test suite).
EXPORTS = ("ipd_attn_workspace_size", "ipd_verify_attn", "ipd_decode_attn",
           "ipd_score_workspace_size", "ipd_score_span", "ipd_loss_workspace_size",
           "ipd_split_loss", "ipd_get_device_error", "ipd_status_string", "ipd_version",
           "ipd_score_span_static", "ipd_score_span_ex", "ipd_score_span_needed", "ipd_full_kl",
           "ipd_loss_grad_workspace_size", "ipd_split_loss_grad", "ipd_sample_workspace_size",
           "ipd_sample", "ipd_kv_append", "ipd_kv_append_many", "ipd_set_attn_kernel_timing",
           "ipd_attn_kernel_time", "ipd_device_readable")
# takeover / handback rules (IPD_RULE_*)
RULE_TOPK, RULE_ENTROPY_S, RULE_ENTROPY_T, RULE_ALWAYS, RULE_NEVER = 0, 1, 2, 3, 4
# element type of the dense gradient (IPD_DTYPE_*)
DTYPE_F32, DTYPE_BF16 = 0, 1
STATIC_MAX_TOKENS = 4096  # IPD_STATIC_MAX_TOKENS


class IpdError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {STATUS.get(status, status)}")
        self.status = status


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libipd.so not built ({LIB_PATH}); run __graft_entry__.build()")
    return ctypes.CDLL(LIB_PATH)


_lib = _load()

c_p = ctypes.c_void_p
c_i = ctypes.c_int
c_sz = ctypes.c_size_t


class _KVCache(ctypes.Structure):
    _fields_ = [("k_pages", c_p), ("v_pages", c_p), ("num_pages", ctypes.c_int64),
                ("page_size", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32)]


class _ScoreExt(ctypes.Structure):
    _fields_ = [("takeover_rule", ctypes.c_int32), ("handback_rule", ctypes.c_int32),
                ("takeover_tau", ctypes.c_float), ("handback_tau", ctypes.c_float),
                ("entropy_s", c_p), ("entropy_t", c_p), ("topk_overlap", c_p),
                ("topk_s", c_p), ("topk_t", c_p), ("next_token", c_p), ("draw_base", c_p),
                ("sample_seed", ctypes.c_uint64), ("inv_temperature", ctypes.c_float)]


class _KvAppendDesc(ctypes.Structure):
    _fields_ = [("k_pages", c_p), ("v_pages", c_p), ("num_pages", ctypes.c_int64),
                ("num_kv_heads", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("k_new", c_p), ("v_new", c_p), ("cu_new", c_p),
                ("seq_len", c_p), ("page_table", c_p), ("max_pages", ctypes.c_int32),
                ("num_reqs", ctypes.c_int32), ("total_new", ctypes.c_int32)]


class _AttnBatch(ctypes.Structure):
    _fields_ = [("cache", ctypes.POINTER(_KVCache)), ("num_q_heads", ctypes.c_int32),
                ("num_reqs", ctypes.c_int32), ("q", c_p), ("cu_q", c_p), ("seq_len", c_p),
                ("page_table", c_p), ("max_pages", ctypes.c_int32), ("total_q", ctypes.c_int32),
                ("max_q_len", ctypes.c_int32), ("max_seq_len", ctypes.c_int32), ("out", c_p)]


_lib.ipd_attn_workspace_size.restype = c_sz
_lib.ipd_attn_workspace_size.argtypes = [ctypes.POINTER(_AttnBatch), c_i,
                                         ctypes.POINTER(_AttnBatch), c_i]
_lib.ipd_verify_attn.restype = c_i
_lib.ipd_verify_attn.argtypes = [ctypes.POINTER(_AttnBatch), c_i, ctypes.POINTER(_AttnBatch), c_i,
                                 ctypes.c_float, c_p, c_sz, c_p]
_lib.ipd_decode_attn.restype = c_i
_lib.ipd_decode_attn.argtypes = [ctypes.POINTER(_AttnBatch), c_i, ctypes.c_float, c_p, c_sz, c_p]
_lib.ipd_score_workspace_size.restype = c_sz
_lib.ipd_score_workspace_size.argtypes = [c_i, c_i, c_i, c_i]
_lib.ipd_score_span.restype = c_i
_lib.ipd_score_span.argtypes = [c_p] * 6 + [c_i] * 5 + [c_p] * 13 + [c_p, c_sz, c_p]
_lib.ipd_device_readable.restype = c_i
_lib.ipd_device_readable.argtypes = [c_p, ctypes.POINTER(c_i)]
_lib.ipd_score_span_needed.restype = c_i
_lib.ipd_score_span_needed.argtypes = [c_p] * 6 + [c_i] * 6 + [c_p] * 13 + [c_p, c_sz, c_p]
_lib.ipd_score_span_ex.restype = c_i
_lib.ipd_score_span_ex.argtypes = ([c_p] * 6 + [c_i] * 5 + [c_p] * 13 +
                                   [ctypes.POINTER(_ScoreExt), c_p, c_sz, c_p])
_lib.ipd_full_kl.restype = c_i
_lib.ipd_full_kl.argtypes = [c_p, c_p, c_i, c_i, c_p, c_p, c_p]
_lib.ipd_score_span_static.restype = c_i
_lib.ipd_score_span_static.argtypes = [c_p] * 6 + [c_i] * 5 + [c_p] * 13 + [c_p]
_lib.ipd_loss_workspace_size.restype = c_sz
_lib.ipd_loss_workspace_size.argtypes = [c_i]
_lib.ipd_split_loss.restype = c_i
_lib.ipd_split_loss.argtypes = [c_p] * 6 + [c_i, c_i, c_i, c_p, c_p, c_sz, c_p]
_lib.ipd_loss_grad_workspace_size.restype = c_sz
_lib.ipd_loss_grad_workspace_size.argtypes = [c_i, c_i]
_lib.ipd_split_loss_grad.restype = c_i
_lib.ipd_split_loss_grad.argtypes = ([c_p] * 9 + [c_i] * 6 + [ctypes.c_float, c_p, c_p, c_p, c_i,
                                      c_p, c_sz, c_p])
_lib.ipd_sample_workspace_size.restype = c_sz
_lib.ipd_sample_workspace_size.argtypes = [c_i, c_i]
_lib.ipd_sample.restype = c_i
_lib.ipd_sample.argtypes = [c_p, c_i, c_i, ctypes.c_uint64, c_p, ctypes.c_float, c_p, c_p, c_sz,
                            c_p]
_lib.ipd_kv_append.restype = c_i
_lib.ipd_kv_append.argtypes = [c_p, c_p, ctypes.c_int64, c_i, c_i, c_i, c_p, c_p, c_p, c_p, c_p,
                               c_i, c_i, c_i, c_p]
_lib.ipd_kv_append_many.restype = c_i
_lib.ipd_kv_append_many.argtypes = [ctypes.POINTER(_KvAppendDesc), c_i, c_p]
_lib.ipd_set_attn_kernel_timing.restype = c_i
_lib.ipd_set_attn_kernel_timing.argtypes = [c_i]
_lib.ipd_attn_kernel_time.restype = c_i
_lib.ipd_attn_kernel_time.argtypes = [ctypes.POINTER(ctypes.c_double), ctypes.POINTER(c_i)]
_lib.ipd_get_device_error.restype = c_i
_lib.ipd_get_device_error.argtypes = [ctypes.POINTER(ctypes.c_uint32)]
_lib.ipd_status_string.restype = ctypes.c_char_p
_lib.ipd_status_string.argtypes = [c_i]
_lib.ipd_version.restype = c_i


def lib() -> ctypes.CDLL:
    return _lib


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else None
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _check(st: int, what: str):
    if st != IPD_OK:
        raise IpdError(st, what)


class KVCache:
    """A paged KV cache: k_pages / v_pages are [num_pages, Hkv, 16, 128] bf16."""

    def __init__(self, k_pages: torch.Tensor, v_pages: torch.Tensor):
        assert k_pages.shape == v_pages.shape and k_pages.dim() == 4
        self.k_pages, self.v_pages = k_pages, v_pages
        self.c = _KVCache(_ptr(k_pages), _ptr(v_pages), k_pages.shape[0], k_pages.shape[2],
                          k_pages.shape[1], k_pages.shape[3])

    @property
    def num_kv_heads(self) -> int:
        return self.k_pages.shape[1]


class AttnBatch:
    """One sub-batch of requests attending one cache (see ipd_attn_batch).

    q [total_q, Hq, 128] bf16, cu_q [R+1] int32, seq_len [R] int32,
    page_table [R, max_pages] int32, out [total_q, Hq, 128] bf16 (all device);
    max_q_len / max_seq_len are host-known bounds."""

    def __init__(self, cache: KVCache, q, cu_q, seq_len, page_table, out, max_q_len: int,
                 max_seq_len: int):
        self.cache = cache
        self._keep = (q, cu_q, seq_len, page_table, out)
        R = seq_len.numel()
        self.c = _AttnBatch(ctypes.pointer(cache.c), q.shape[1], R, _ptr(q), _ptr(cu_q),
                            _ptr(seq_len), _ptr(page_table), page_table.shape[1], q.shape[0],
                            max_q_len, max_seq_len, _ptr(out))
        self.out = out


def _arr(batches: Sequence[AttnBatch]):
    n = len(batches)
    if n == 0:
        return None, 0
    a = (_AttnBatch * n)(*[b.c for b in batches])
    return a, n


def attn_workspace_size(verify: Sequence[AttnBatch], decode: Sequence[AttnBatch] = ()) -> int:
    va, nv = _arr(verify)
    da, nd = _arr(decode)
    return int(_lib.ipd_attn_workspace_size(va, nv, da, nd))


def verify_attn(verify: Sequence[AttnBatch], decode: Sequence[AttnBatch], softmax_scale: float,
                workspace: torch.Tensor, stream=None):
    va, nv = _arr(verify)
    da, nd = _arr(decode)
    _check(_lib.ipd_verify_attn(va, nv, da, nd, softmax_scale, _ptr(workspace),
                                workspace.numel() * workspace.element_size(), _stream(stream)),
           "ipd_verify_attn")


def decode_attn(decode: Sequence[AttnBatch], softmax_scale: float, workspace: torch.Tensor,
                stream=None):
    da, nd = _arr(decode)
    _check(_lib.ipd_decode_attn(da, nd, softmax_scale, _ptr(workspace),
                                workspace.numel() * workspace.element_size(), _stream(stream)),
           "ipd_decode_attn")


def score_workspace_size(num_reqs: int, total_tokens: int, vocab: int, K: int) -> int:
    return int(_lib.ipd_score_workspace_size(num_reqs, total_tokens, vocab, K))


SCORE_TOKEN_OUTPUTS = (("logp_s", torch.float32), ("logp_t", torch.float32),
                       ("feedback", torch.float32), ("kl_rev", torch.float32),
                       ("kl_fwd", torch.float32), ("covered", torch.uint8),
                       ("margin", torch.float32), ("source", torch.uint8))
SCORE_REQ_OUTPUTS = (("first_trans", torch.int32), ("n_emit", torch.int32),
                     ("next_driver", torch.uint8), ("new_len", torch.int32), ("done", torch.uint8))


def alloc_score_outputs(num_reqs: int, total_tokens: int, device) -> dict:
    out = {n: torch.empty(total_tokens, dtype=dt, device=device) for n, dt in SCORE_TOKEN_OUTPUTS}
    out.update({n: torch.empty(num_reqs, dtype=dt, device=device) for n, dt in SCORE_REQ_OUTPUTS})
    return out


def score_span(logits_student, logits_teacher, tokens, cu_span, driver, prefix_len, K: int,
               eos_id: int, out: dict, workspace: torch.Tensor, stream=None):
    R = driver.numel()
    T, V = logits_student.shape
    _check(_lib.ipd_score_span(
        _ptr(logits_student), _ptr(logits_teacher), _ptr(tokens), _ptr(cu_span), _ptr(driver),
        _ptr(prefix_len), R, T, V, K, eos_id,
        *[_ptr(out[n]) for n, _ in SCORE_TOKEN_OUTPUTS],
        *[_ptr(out[n]) for n, _ in SCORE_REQ_OUTPUTS],
        _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)),
        "ipd_score_span")


def device_readable(t: torch.Tensor) -> bool:
    """Whether the library's kernels can read tensor t where it lives (device
    memory, or pinned host memory mapped into the device's address space)."""
    r = c_i(0)
    _check(_lib.ipd_device_readable(_ptr(t), ctypes.byref(r)), "ipd_device_readable")
    return bool(r.value)


def score_span_needed(logits_student, logits_teacher, tokens, cu_span, driver, prefix_len,
                      K: int, eos_id: int, max_span: int, out: dict, workspace: torch.Tensor,
                      stream=None):
    """ipd_score_span reading only the rows the verdict and the emitted
    positions need; ``max_span`` bounds every request's span length."""
    R = driver.numel()
    T, V = logits_student.shape
    _check(_lib.ipd_score_span_needed(
        _ptr(logits_student), _ptr(logits_teacher), _ptr(tokens), _ptr(cu_span), _ptr(driver),
        _ptr(prefix_len), R, T, V, K, eos_id, max_span,
        *[_ptr(out[n]) for n, _ in SCORE_TOKEN_OUTPUTS],
        *[_ptr(out[n]) for n, _ in SCORE_REQ_OUTPUTS],
        _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)),
        "ipd_score_span_needed")


def score_span_ex(logits_student, logits_teacher, tokens, cu_span, driver, prefix_len, K: int,
                  eos_id: int, out: dict, workspace: torch.Tensor, takeover_rule: int = RULE_TOPK,
                  handback_rule: int = RULE_TOPK, takeover_tau: float = 0.0,
                  handback_tau: float = 0.0, entropy_s: Optional[torch.Tensor] = None,
                  entropy_t: Optional[torch.Tensor] = None,
                  topk_overlap: Optional[torch.Tensor] = None,
                  topk_s: Optional[torch.Tensor] = None, topk_t: Optional[torch.Tensor] = None,
                  next_token: Optional[torch.Tensor] = None,
                  draw_base: Optional[torch.Tensor] = None, sample_seed: int = 0,
                  inv_temperature: float = 1.0, stream=None):
    """ipd_score_span with selectable takeover / handback rules and the
    optional per-token entropies and top-K overlap ratio (fp32 [T] tensors),
    top-K id lists (int32 [T, K]) and the next span's first token per request
    (int32 [R]; draw numbers from ``draw_base``, uint64 as int64 [R])."""
    R = driver.numel()
    T, V = logits_student.shape
    ext = _ScoreExt(takeover_rule, handback_rule, takeover_tau, handback_tau,
                    _ptr(entropy_s), _ptr(entropy_t), _ptr(topk_overlap), _ptr(topk_s),
                    _ptr(topk_t), _ptr(next_token), _ptr(draw_base),
                    sample_seed & 0xFFFFFFFFFFFFFFFF, inv_temperature)
    _check(_lib.ipd_score_span_ex(
        _ptr(logits_student), _ptr(logits_teacher), _ptr(tokens), _ptr(cu_span), _ptr(driver),
        _ptr(prefix_len), R, T, V, K, eos_id,
        *[_ptr(out[n]) for n, _ in SCORE_TOKEN_OUTPUTS],
        *[_ptr(out[n]) for n, _ in SCORE_REQ_OUTPUTS],
        ctypes.byref(ext), _ptr(workspace), workspace.numel() * workspace.element_size(),
        _stream(stream)), "ipd_score_span_ex")


def full_kl(logits_student, logits_teacher, kl_rev_full: torch.Tensor, kl_fwd_full: torch.Tensor,
            stream=None):
    """Full-vocabulary KL in both directions at every span position."""
    T, V = logits_student.shape
    _check(_lib.ipd_full_kl(_ptr(logits_student), _ptr(logits_teacher), T, V, _ptr(kl_rev_full),
                            _ptr(kl_fwd_full), _stream(stream)), "ipd_full_kl")


def score_span_static(logits_student, logits_teacher, tokens, cu_span, driver, prefix_len,
                      K: int, eos_id: int, out: dict, stream=None):
    """ipd_score_span without a workspace: for callers that cannot allocate
    device memory (the scratch is the library's static device array, at most
    STATIC_MAX_TOKENS span positions; overlapping calls race on it)."""
    R = driver.numel()
    T, V = logits_student.shape
    _check(_lib.ipd_score_span_static(
        _ptr(logits_student), _ptr(logits_teacher), _ptr(tokens), _ptr(cu_span), _ptr(driver),
        _ptr(prefix_len), R, T, V, K, eos_id,
        *[_ptr(out[n]) for n, _ in SCORE_TOKEN_OUTPUTS],
        *[_ptr(out[n]) for n, _ in SCORE_REQ_OUTPUTS],
        _stream(stream)), "ipd_score_span_static")


def split_loss(kl_rev, kl_fwd, source, cu_span, n_emit, resp_len, agg_mode: int, dir_mode: int,
               out8: torch.Tensor, stream=None):
    R = cu_span.numel() - 1
    _check(_lib.ipd_split_loss(_ptr(kl_rev), _ptr(kl_fwd), _ptr(source), _ptr(cu_span),
                               _ptr(n_emit), _ptr(resp_len), R, agg_mode, dir_mode, _ptr(out8),
                               None, 0, _stream(stream)), "ipd_split_loss")


def kv_append(cache: "KVCache", k_new, v_new, cu_new, seq_len, page_table, stream=None):
    """Writes the new tokens' K/V rows ([n, Hkv, 128] bf16) into the cache's
    pages at the last positions of each request's sequence (``seq_len`` is
    the length after the append)."""
    R = cu_new.numel() - 1
    _check(_lib.ipd_kv_append(_ptr(cache.k_pages), _ptr(cache.v_pages), cache.k_pages.shape[0],
                              cache.k_pages.shape[1], 16, 128, _ptr(k_new), _ptr(v_new),
                              _ptr(cu_new), _ptr(seq_len), _ptr(page_table),
                              page_table.shape[1], R, k_new.shape[0], _stream(stream)),
           "ipd_kv_append")


def kv_append_many(appends, stream=None):
    """Several appends in one launch: ``appends`` is a sequence of (cache,
    k_new, v_new, cu_new, seq_len, page_table) tuples, each as in kv_append."""
    n = len(appends)
    arr = (_KvAppendDesc * max(n, 1))()
    for i, (cache, k_new, v_new, cu_new, seq_len, page_table) in enumerate(appends):
        arr[i] = _KvAppendDesc(_ptr(cache.k_pages), _ptr(cache.v_pages), cache.k_pages.shape[0],
                               cache.k_pages.shape[1], 16, 128, _ptr(k_new), _ptr(v_new),
                               _ptr(cu_new), _ptr(seq_len), _ptr(page_table),
                               page_table.shape[1], cu_new.numel() - 1, k_new.shape[0])
    _check(_lib.ipd_kv_append_many(arr, n, _stream(stream)), "ipd_kv_append_many")


def sample_workspace_size(n_rows: int, vocab: int) -> int:
    return int(_lib.ipd_sample_workspace_size(n_rows, vocab))


def sample(logits, seed: int, draw_id: Optional[torch.Tensor], tokens: torch.Tensor,
           workspace: torch.Tensor, inv_temperature: float = 1.0, stream=None):
    """One seeded draw per row of ``logits`` ([n, V] bf16) into ``tokens``
    (int32 [n]); ``draw_id`` holds the rows' uint64 draw numbers (as int64)."""
    n, V = logits.shape
    _check(_lib.ipd_sample(_ptr(logits), n, V, seed & 0xFFFFFFFFFFFFFFFF, _ptr(draw_id),
                           inv_temperature, _ptr(tokens), _ptr(workspace),
                           workspace.numel() * workspace.element_size(), _stream(stream)),
           "ipd_sample")


def split_loss_grad(logits_student, logits_teacher, topk_s, topk_t, source, cu_span, n_emit,
                    resp_len, loss_out8, K: int, agg_mode: int, dir_mode: int, grad_scale: float,
                    grad_idx: torch.Tensor, grad_val: torch.Tensor,
                    grad_dense: Optional[torch.Tensor] = None, stream=None):
    """Gradient of grad_scale * loss with respect to the student's logits:
    sparse [T, 2K] ids / values, and the dense [T, V] form when ``grad_dense``
    (fp32 or bf16) is given."""
    R = cu_span.numel() - 1
    T, V = logits_student.shape
    dtype = DTYPE_F32
    if grad_dense is not None:
        if grad_dense.dtype == torch.bfloat16:
            dtype = DTYPE_BF16
        elif grad_dense.dtype != torch.float32:
            raise IpdError(STATUS_CODES["IPD_ERR_INVALID_ARG"], "ipd_split_loss_grad: dense dtype")
    _check(_lib.ipd_split_loss_grad(
        _ptr(logits_student), _ptr(logits_teacher), _ptr(topk_s), _ptr(topk_t), _ptr(source),
        _ptr(cu_span), _ptr(n_emit), _ptr(resp_len), _ptr(loss_out8), R, T, V, K, agg_mode,
        dir_mode, grad_scale, _ptr(grad_idx), _ptr(grad_val), _ptr(grad_dense), dtype, None, 0,
        _stream(stream)), "ipd_split_loss_grad")


def set_attn_kernel_timing(on: bool):
    _check(_lib.ipd_set_attn_kernel_timing(1 if on else 0), "ipd_set_attn_kernel_timing")


def attn_kernel_time():
    """(summed ms, launches) of the attention kernels timed since timing was
    switched on or last read (synchronises)."""
    ms = ctypes.c_double(0.0)
    n = c_i(0)
    _check(_lib.ipd_attn_kernel_time(ctypes.byref(ms), ctypes.byref(n)), "ipd_attn_kernel_time")
    return float(ms.value), int(n.value)


def device_error() -> int:
    """Reads and clears the device-side error word (synchronises)."""
    v = ctypes.c_uint32(0)
    _check(_lib.ipd_get_device_error(ctypes.byref(v)), "ipd_get_device_error")
    return int(v.value)
