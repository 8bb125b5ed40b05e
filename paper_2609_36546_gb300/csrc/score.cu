// The vocabulary pass of the verify step (Sec. 3.1 top-K supports, Sec. 3.2.1
// coverage rules, Sec. 3.2.2 source-split KL terms, Sec. 3.2.3 verdict).
//
// Kernel 1 (row pass), one CTA per logits row (2 rows per span position: the
// student's and the teacher's), one read of the row from HBM:
//   - log Z = log sum exp(l) with a per-thread online maximum (fp32),
//   - the exact top-K (K <= 32) under the order (logit desc, token id asc).
//     Every warp keeps its best 32 keys sorted across its lanes; a 64-bit key
//     (bf16 order code << 32 | ~token id) makes keys distinct and the order
//     total.  A warp-uniform threshold filters candidates with one compare
//     per 8 logits, and warps share their thresholds through shared memory.
//   - the logit of the proposed token.
// Kernel 2 (epilogue), one CTA per request: union support, renormalised KL in
// both directions, log-probs and feedback, coverage and margin, then the
// verdict of the request's span.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "common.cuh"

IPD_DECLARE_ERROR_WORD(g_score_err);

namespace {

constexpr int kRowThreads = 256;
constexpr int kRowWarps = kRowThreads / 32;
constexpr int kEpiThreads = 256;

struct RowOut {
  float logz;     // log sum_v exp(l_v)
  float lx;       // logit of the proposed token (NaN if the token id is invalid)
  int pad[2];
  unsigned long long keys[IPD_MAX_K];  // best first
};

// Order code of a bf16 value: monotone in the value, -0 folded onto +0.
__device__ __forceinline__ uint32_t ord16(uint32_t b) {
  b &= 0xffffu;
  if (b == 0x8000u) b = 0;
  return (b & 0x8000u) ? (~b & 0xffffu) : (b | 0x8000u);
}
__device__ __forceinline__ float ord16_to_float(uint32_t o) {
  uint32_t b = (o & 0x8000u) ? (o & 0x7fffu) : (~o & 0xffffu);
  return __uint_as_float(b << 16);
}
__device__ __forceinline__ unsigned long long make_key(uint32_t bits16, uint32_t idx) {
  return ((unsigned long long)ord16(bits16) << 32) | (unsigned long long)(0xffffffffu - idx);
}
__device__ __forceinline__ uint32_t key_idx(unsigned long long k) {
  return 0xffffffffu - (uint32_t)k;
}
__device__ __forceinline__ float key_val(unsigned long long k) {
  return ord16_to_float((uint32_t)(k >> 32));
}

// bf16 bits of element e (0..7) of an 8-element vector.
__device__ __forceinline__ uint32_t elem_bits(const uint4 &r, int e) {
  const uint32_t w = (e < 4) ? ((e < 2) ? r.x : r.y) : ((e < 6) ? r.z : r.w);
  return (e & 1) ? (w >> 16) : (w & 0xffffu);
}

// Maximum of 8 bf16 values (one 16-byte vector) as fp32, via packed bf16x2 max.
__device__ __forceinline__ float bf16x8_max(const uint4 &r) {
  uint32_t a, b, c;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(r.x), "r"(r.y));
  asm("max.bf16x2 %0, %1, %2;" : "=r"(b) : "r"(r.z), "r"(r.w));
  asm("max.bf16x2 %0, %1, %2;" : "=r"(c) : "r"(a), "r"(b));
  return fmaxf(bf16lo(c), bf16hi(c));
}

__device__ __forceinline__ unsigned long long shfl_u64(unsigned long long v, int src) {
  return __shfl_sync(0xffffffffu, v, src);
}

// Insert key c into the warp's descending list (lane i holds the i-th best).
__device__ __forceinline__ void list_insert(unsigned long long &L, unsigned long long c, int lane) {
  const int pos = __popc(__ballot_sync(0xffffffffu, L > c));
  const unsigned long long up = __shfl_up_sync(0xffffffffu, L, 1);
  if (lane == pos) L = c;
  else if (lane > pos) L = up;
}

// Bitonic sort of one key per lane, descending over lanes.
__device__ __forceinline__ unsigned long long warp_sort_desc(unsigned long long k, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int j = size >> 1; j > 0; j >>= 1) {
      const unsigned long long o = __shfl_xor_sync(0xffffffffu, k, j);
      const bool lower = (lane & j) == 0;
      const bool desc = (lane & size) == 0;
      const unsigned long long hi = k > o ? k : o, lo = k > o ? o : k;
      k = (lower == desc) ? hi : lo;
    }
  }
  return k;
}

__global__ void __launch_bounds__(kRowThreads, 4) score_rows_kernel(
    const uint16_t *__restrict__ ls, const uint16_t *__restrict__ lt,
    const int32_t *__restrict__ tokens, int vocab, int K, RowOut *__restrict__ out) {
  __shared__ unsigned long long s_theta;
  __shared__ unsigned long long s_lists[kRowWarps][32];
  __shared__ float s_m[kRowWarps], s_s[kRowWarps];

  const int t = blockIdx.x >> 1, model = blockIdx.x & 1;
  const uint16_t *row = (model ? lt : ls) + (size_t)t * vocab;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) s_theta = 0ull;
  __syncthreads();

  const int nvec = vocab >> 3;
  float m = -INFINITY, s = 0.f;
  unsigned long long L = 0ull, theta = 0ull;

  // Block-wide warm-up.  Every thread takes the best key among its first
  // U vectors (8*U logits); the 17th largest of those 256 lane maxima starts
  // the shared threshold.  At least 16 logits of the row are strictly above
  // it, so no member of the row's top-K (K <= 16 here; larger K lowers it to
  // the (K+1)-th) is ever filtered out, and only ~0.3 % of N(0,1)-like logits
  // pass it from the start.
  constexpr int U = 4;
  uint4 pre[U];
  unsigned long long lane_best = 0ull;
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int v0 = u * kRowThreads + (int)threadIdx.x;
    pre[u] = make_uint4(0xff80ff80u, 0xff80ff80u, 0xff80ff80u, 0xff80ff80u);  // -inf
    if (v0 < nvec) pre[u] = ldg_stream(row + (size_t)v0 * 8);
  }
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int v0 = u * kRowThreads + (int)threadIdx.x;
    if (v0 < nvec) {
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const unsigned long long k = make_key(elem_bits(pre[u], e), (uint32_t)v0 * 8u + e);
        lane_best = k > lane_best ? k : lane_best;
      }
    }
  }
  s_lists[warp][lane] = warp_sort_desc(lane_best, lane);
  __syncthreads();
  {
    const unsigned long long c = s_lists[warp][lane];
    int rank = 0;
#pragma unroll 1
    for (int w2 = 0; w2 < kRowWarps; ++w2) {
      int lo = 0, hi = 32;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (s_lists[w2][mid] > c) lo = mid + 1;
        else hi = mid;
      }
      rank += lo;
    }
    if (c != 0ull && rank == (K > 16 ? K : 16)) s_theta = c;  // the (max(K,16)+1)-th largest
  }
  __syncthreads();
  L = 0ull;
  theta = 0ull;

  // Four independent 16-byte loads per thread are in flight per iteration.
  // Per 8 logits: the maximum on the packed bf16 words (3 max instructions),
  // then unpack, one fused multiply-add and one hardware 2^x each for the sum.
  // The candidate filter compares the vector maximum with the threshold's
  // value; only vectors reaching it build 64-bit keys.
  // The trip count is the same for every thread (warp-wide ballots below).
  for (int base = 0; base < nvec; base += kRowThreads * U) {
    uint4 raw[U];
    int vv[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      vv[u] = base + u * kRowThreads + (int)threadIdx.x;
      raw[u] = make_uint4(0xff80ff80u, 0xff80ff80u, 0xff80ff80u, 0xff80ff80u);  // -inf
      if (base == 0) raw[u] = pre[u];
      else if (vv[u] < nvec) raw[u] = ldg_stream(row + (size_t)vv[u] * 8);
    }
    float vmx[U];
#pragma unroll
    for (int u = 0; u < U; ++u) vmx[u] = bf16x8_max(raw[u]);
    const float bmax = fmaxf(fmaxf(vmx[0], vmx[1]), fmaxf(vmx[2], vmx[3]));
    if (bmax > m) {
      s *= ex2_approx((m - bmax) * kLog2e);
      m = bmax;
    }
    if (m != -INFINITY) {
      const float ml = -m * kLog2e;
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t w[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          s += ex2_approx(fmaf(bf16lo(w[q]), kLog2e, ml));
          s += ex2_approx(fmaf(bf16hi(w[q]), kLog2e, ml));
        }
      }
    }
    // candidate filter against the warp / block threshold
    const unsigned long long sth = s_theta;
    const unsigned long long th = theta > sth ? theta : sth;
    const float thf = key_val(th);  // threshold value (keys equal in value go to the full test)
    uint32_t pending = 0;           // bit 8u + e: element e of vector u
    if (th == 0ull || bmax >= thf) {
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (vv[u] < nvec && (th == 0ull || vmx[u] >= thf)) {
#pragma unroll
          for (int e = 0; e < 8; ++e)
            if (make_key(elem_bits(raw[u], e), (uint32_t)vv[u] * 8u + e) > th)
              pending |= 1u << (8 * u + e);
        }
    }
    unsigned any = __ballot_sync(0xffffffffu, pending != 0);
    if (any) {
      while (any) {
        const int leader = __ffs(any) - 1;
        unsigned long long c = 0ull;
        if (lane == leader) {
          const int bit = __ffs(pending) - 1;
          pending &= pending - 1;
          const int u = bit >> 3, e = bit & 7;
          const uint4 r = u == 0 ? raw[0] : (u == 1 ? raw[1] : (u == 2 ? raw[2] : raw[3]));
          const int vsel = u == 0 ? vv[0] : (u == 1 ? vv[1] : (u == 2 ? vv[2] : vv[3]));
          c = make_key(elem_bits(r, e), (uint32_t)vsel * 8u + e);
        }
        c = shfl_u64(c, leader);
        if (c > theta) {
          list_insert(L, c, lane);
          theta = shfl_u64(L, K - 1);
        }
        any = __ballot_sync(0xffffffffu, pending != 0);
      }
      if (lane == 0 && theta > s_theta) atomicMax(&s_theta, theta);
    }
  }
  // Every logit of the row went through the filter exactly once, so each
  // reached at most one warp list and the keys in the lists are distinct.

  // block merge of the log-sum-exp
  float wm = warp_max(m);
  float ws = (m == -INFINITY) ? 0.f : s * exp2f((m - wm) * kLog2e);
  if (wm == -INFINITY) ws = 0.f;
  ws = warp_sum(ws);
  s_lists[warp][lane] = L;
  if (lane == 0) {
    s_m[warp] = wm;
    s_s[warp] = ws;
  }
  __syncthreads();
  if (warp == 0) {
    float bm = lane < kRowWarps ? s_m[lane] : -INFINITY;
    const float gm = warp_max(bm);
    float bs = (lane < kRowWarps && bm != -INFINITY) ? s_s[lane] * exp2f((bm - gm) * kLog2e) : 0.f;
    bs = warp_sum(bs);
    // merge of the warp lists: the rank of a key in the union is the number of
    // larger keys in every list (binary search in each sorted list)
    if (lane == 0) {
      out[blockIdx.x].logz = gm + logf(bs);
      const int x = tokens[t];
      float lx = __int_as_float(0x7fc00000);
      if (x >= 0 && x < vocab) lx = bf16f(row[x]);
      out[blockIdx.x].lx = lx;
    }
  }
  // every thread ranks one candidate key (kRowWarps * 32 == kRowThreads)
  {
    const unsigned long long c = s_lists[warp][lane];
    int rank = 0;
#pragma unroll 1
    for (int w2 = 0; w2 < kRowWarps; ++w2) {
      // number of keys > c in list w2 (descending): binary search
      int lo = 0, hi = 32;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (s_lists[w2][mid] > c) lo = mid + 1;
        else hi = mid;
      }
      rank += lo;
    }
    if (c != 0ull && rank < K) out[blockIdx.x].keys[rank] = c;
  }
}

__global__ void __launch_bounds__(kEpiThreads) score_epilogue_kernel(
    const uint16_t *__restrict__ ls, const uint16_t *__restrict__ lt,
    const int32_t *__restrict__ tokens, const int32_t *__restrict__ cu_span,
    const uint8_t *__restrict__ driver, const int32_t *__restrict__ prefix_len, int vocab, int K,
    int eos_id, const RowOut *__restrict__ rows, float *logp_s, float *logp_t, float *feedback,
    float *kl_rev, float *kl_fwd, uint8_t *covered, float *margin, uint8_t *source,
    int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver, int32_t *new_len, uint8_t *done,
    int total_tokens) {
  __shared__ uint8_t s_cov[1024];
  const int r = blockIdx.x;
  const int t0 = cu_span[r], t1 = cu_span[r + 1];
  const int drv = driver[r] ? 1 : 0;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (t0 < 0 || t1 < t0 || t1 > total_tokens) {
    if (threadIdx.x == 0) ipd_set_error(&g_score_err, IPD_DEVERR_SPAN);
    return;
  }
  const int k = t1 - t0;

  for (int t = t0 + warp; t < t1; t += kEpiThreads / 32) {
    const RowOut &rs = rows[2 * t], &rq = rows[2 * t + 1];
    const int x = tokens[t];
    const bool xok = x >= 0 && x < vocab;
    if (!xok && lane == 0) ipd_set_error(&g_score_err, IPD_DEVERR_TOKEN);
    const uint16_t *rowS = ls + (size_t)t * vocab, *rowT = lt + (size_t)t * vocab;
    // union support S = Top_K(pi) u Top_K(q)
    unsigned long long kS = 0ull, kT = 0ull;
    uint32_t iS = 0, iT = 0;
    if (lane < K) {
      kS = rs.keys[lane];
      kT = rq.keys[lane];
      iS = key_idx(kS);
      iT = key_idx(kT);
      if (iS >= (uint32_t)vocab) iS = 0;  // never taken: K <= vocab fills every slot
      if (iT >= (uint32_t)vocab) iT = 0;
    }
    bool dupT = false;
    for (int j = 0; j < K; ++j) {
      const uint32_t o = __shfl_sync(0xffffffffu, iS, j);
      dupT |= (o == iT);
    }
    const bool hasS = lane < K, hasT = lane < K && !dupT;
    // a = student logit, b = teacher logit, for the two union elements of this lane
    float aS = 0.f, bS = 0.f, aT = 0.f, bT = 0.f;
    if (hasS) {
      aS = key_val(kS);
      bS = bf16f(rowT[iS]);
    }
    if (hasT) {
      bT = key_val(kT);
      aT = bf16f(rowS[iT]);
    }
    const float ma = warp_max(fmaxf(hasS ? aS : -INFINITY, hasT ? aT : -INFINITY));
    const float mb = warp_max(fmaxf(hasS ? bS : -INFINITY, hasT ? bT : -INFINITY));
    float sa = (hasS ? expf(aS - ma) : 0.f) + (hasT ? expf(aT - ma) : 0.f);
    float sb = (hasS ? expf(bS - mb) : 0.f) + (hasT ? expf(bT - mb) : 0.f);
    sa = warp_sum(sa);
    sb = warp_sum(sb);
    const float lza = ma + logf(sa), lzb = mb + logf(sb);
    float kr = 0.f, kf = 0.f;
    if (hasS) {
      const float la = aS - lza, lb = bS - lzb;
      const float pa = expf(la), pb = expf(lb);
      if (pa > 0.f) kr += pa * (la - lb);
      if (pb > 0.f) kf += pb * (lb - la);
    }
    if (hasT) {
      const float la = aT - lza, lb = bT - lzb;
      const float pa = expf(la), pb = expf(lb);
      if (pa > 0.f) kr += pa * (la - lb);
      if (pb > 0.f) kf += pb * (lb - la);
    }
    kr = warp_sum(kr);
    kf = warp_sum(kf);
    // coverage by the verifier's Top_K: the teacher's row when the student drives
    const unsigned long long kv = drv ? kS : kT;
    const bool hit = xok && lane < K && key_idx(kv) == (uint32_t)x;
    const bool cov = __ballot_sync(0xffffffffu, hit) != 0;
    const unsigned long long kth = shfl_u64(kv, K - 1);
    if (lane == 0) {
      const RowOut &rv = drv ? rs : rq;
      const float lps = rs.lx - rs.logz, lpt = rq.lx - rq.logz;
      logp_s[t] = lps;
      logp_t[t] = lpt;
      feedback[t] = lpt - lps;
      kl_rev[t] = kr;
      kl_fwd[t] = kf;
      covered[t] = cov ? 1 : 0;
      margin[t] = rv.lx - key_val(kth);
      if (t - t0 < 1024) s_cov[t - t0] = cov ? 1 : 0;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // Eq. (ipd_state_transition) applied position by position until the first
    // state change or an accepted EOS; rollback rules of the verdict stage.
    int n = 0, ft = k, nd = drv, dn = 0;
    for (int i = 0; i < k; ++i) {
      const int c = (i < 1024) ? s_cov[i] : covered[t0 + i];
      const bool eos = eos_id >= 0 && tokens[t0 + i] == eos_id;
      if (drv == 0) {
        if (!c) {  // takeover: the student token is rejected, not emitted
          ft = i;
          nd = 1;
          break;
        }
        n = i + 1;
        if (eos) {
          dn = 1;
          break;
        }
      } else {
        n = i + 1;  // a teacher token is always kept
        if (c) {    // handback
          ft = i;
          nd = 0;
        }
        if (eos) dn = 1;
        if (c || eos) break;
      }
    }
    for (int i = 0; i < k; ++i) source[t0 + i] = i < n ? (uint8_t)drv : (uint8_t)255;
    first_trans[r] = ft;
    n_emit[r] = n;
    next_driver[r] = (uint8_t)nd;
    new_len[r] = prefix_len[r] + n;
    done[r] = (uint8_t)dn;
  }
}

}  // namespace

extern "C" __attribute__((visibility("hidden"))) unsigned int ipd_internal_take_score_error() {
  unsigned int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_score_err, sizeof(v)) != cudaSuccess) return 0xffffffffu;
  if (cudaMemcpyToSymbol(g_score_err, &z, sizeof(z)) != cudaSuccess) return 0xffffffffu;
  return v;
}

extern "C" size_t ipd_score_workspace_size(int num_reqs, int total_tokens, int vocab, int K) {
  if (num_reqs < 0 || total_tokens < 0 || vocab < 1 || K < 1) return 0;
  return (size_t)total_tokens * 2 * sizeof(RowOut) + 256;
}

extern "C" int ipd_score_span(const uint16_t *logits_student, const uint16_t *logits_teacher,
                              const int32_t *tokens, const int32_t *cu_span,
                              const uint8_t *driver, const int32_t *prefix_len, int num_reqs,
                              int total_tokens, int vocab, int K, int eos_id, float *logp_s,
                              float *logp_t, float *feedback, float *kl_rev, float *kl_fwd,
                              uint8_t *covered, float *margin, uint8_t *source,
                              int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver,
                              int32_t *new_len, uint8_t *done, void *workspace,
                              size_t workspace_bytes, ipd_stream_t stream) {
  if (num_reqs < 0 || total_tokens < 0) return IPD_ERR_INVALID_ARG;
  if (K < 1 || K > IPD_MAX_K) return IPD_ERR_UNSUPPORTED;
  if (vocab < 8 || vocab % 8 || K > vocab) return IPD_ERR_UNSUPPORTED;
  if (num_reqs == 0) return IPD_OK;
  if (!cu_span || !driver || !prefix_len || !first_trans || !n_emit || !next_driver || !new_len ||
      !done)
    return IPD_ERR_INVALID_ARG;
  if (total_tokens > 0 &&
      (!logits_student || !logits_teacher || !tokens || !logp_s || !logp_t || !feedback ||
       !kl_rev || !kl_fwd || !covered || !margin || !source))
    return IPD_ERR_INVALID_ARG;
  if (((uintptr_t)logits_student | (uintptr_t)logits_teacher) & 15) return IPD_ERR_INVALID_ARG;
  const size_t need = ipd_score_workspace_size(num_reqs, total_tokens, vocab, K);
  if (total_tokens > 0 && (!workspace || workspace_bytes < need || ((uintptr_t)workspace & 15)))
    return IPD_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  RowOut *rows = static_cast<RowOut *>(workspace);
  if (total_tokens > 0) {
    score_rows_kernel<<<2 * total_tokens, kRowThreads, 0, st>>>(logits_student, logits_teacher,
                                                                tokens, vocab, K, rows);
    if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  }
  score_epilogue_kernel<<<num_reqs, kEpiThreads, 0, st>>>(
      logits_student, logits_teacher, tokens, cu_span, driver, prefix_len, vocab, K, eos_id, rows,
      logp_s, logp_t, feedback, kl_rev, kl_fwd, covered, margin, source, first_trans, n_emit,
      next_driver, new_len, done, total_tokens);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}

// ---------------------------------------------------------------------------
// ipd_score_span_static: the same computation for callers that cannot
// allocate device memory.  The per-row scratch that ipd_score_span takes from
// the caller's workspace lives here in one file-scope device array, sized for
// IPD_STATIC_MAX_TOKENS span positions.  Every GPU that loads the library
// holds this array (about 2.1 MiB) until the process exits.
// ---------------------------------------------------------------------------
static __device__ __align__(256) RowOut g_static_rows[2 * IPD_STATIC_MAX_TOKENS];

namespace {
std::mutex g_static_mu;
RowOut *g_static_ptr[64] = {};  // device address of g_static_rows, per device

// In host code g_static_rows names a host-side stand-in, not device memory:
// the device address is looked up once per device, with that device current.
int static_rows(RowOut **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return IPD_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (!g_static_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_rows) != cudaSuccess || !p) return IPD_ERR_CUDA;
    g_static_ptr[dev] = static_cast<RowOut *>(p);
  }
  *out = g_static_ptr[dev];
  return IPD_OK;
}
}  // namespace

extern "C" int ipd_score_span_static(const uint16_t *logits_student,
                                     const uint16_t *logits_teacher, const int32_t *tokens,
                                     const int32_t *cu_span, const uint8_t *driver,
                                     const int32_t *prefix_len, int num_reqs, int total_tokens,
                                     int vocab, int K, int eos_id, float *logp_s, float *logp_t,
                                     float *feedback, float *kl_rev, float *kl_fwd,
                                     uint8_t *covered, float *margin, uint8_t *source,
                                     int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver,
                                     int32_t *new_len, uint8_t *done, ipd_stream_t stream) {
  if (num_reqs < 0 || total_tokens < 0) return IPD_ERR_INVALID_ARG;
  if (K < 1 || K > IPD_MAX_K) return IPD_ERR_UNSUPPORTED;
  if (vocab < 8 || vocab % 8 || K > vocab) return IPD_ERR_UNSUPPORTED;
  if (total_tokens > IPD_STATIC_MAX_TOKENS) return IPD_ERR_CAPACITY;
  if (num_reqs == 0) return IPD_OK;
  if (!cu_span || !driver || !prefix_len || !first_trans || !n_emit || !next_driver || !new_len ||
      !done)
    return IPD_ERR_INVALID_ARG;
  if (total_tokens > 0 &&
      (!logits_student || !logits_teacher || !tokens || !logp_s || !logp_t || !feedback ||
       !kl_rev || !kl_fwd || !covered || !margin || !source))
    return IPD_ERR_INVALID_ARG;
  if (((uintptr_t)logits_student | (uintptr_t)logits_teacher) & 15) return IPD_ERR_INVALID_ARG;
  RowOut *rows = nullptr;
  const int st = static_rows(&rows);
  if (st != IPD_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // Every RowOut the epilogue reads is written by the row kernel of the same
  // call first, so nothing in the array has to start at zero.
  if (total_tokens > 0) {
    score_rows_kernel<<<2 * total_tokens, kRowThreads, 0, s>>>(logits_student, logits_teacher,
                                                               tokens, vocab, K, rows);
    if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  }
  score_epilogue_kernel<<<num_reqs, kEpiThreads, 0, s>>>(
      logits_student, logits_teacher, tokens, cu_span, driver, prefix_len, vocab, K, eos_id, rows,
      logp_s, logp_t, feedback, kl_rev, kl_fwd, covered, margin, source, first_trans, n_emit,
      next_driver, new_len, done, total_tokens);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}
