// Source-split objective of one verify step (Sec. 3.2.2, Eq. ipd_off_loss and
// Eq. ipd_objective; global token mean of App. B.3; KL-direction variants of
// the ablation in Sec. 4.3).  One CTA; every thread reduces a fixed set of
// requests in position order and a fixed-shape tree combines the threads, so
// the result is bitwise reproducible.
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

IPD_DECLARE_ERROR_WORD(g_loss_err);

namespace {

constexpr int kLossThreads = 256;
constexpr int kLossWarps = kLossThreads / 32;

// Fixed-shape butterfly sum over a warp (the same order on every run).
__device__ __forceinline__ float warp_tree_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Eight warps; thread i reduces requests i, i + 256, ... in position order,
// each warp sums its lanes by a fixed butterfly, and warp 0 adds the eight
// warp sums in warp order.  192 bytes of shared memory.
__global__ void __launch_bounds__(kLossThreads) split_loss_kernel(
    const float *__restrict__ kl_rev, const float *__restrict__ kl_fwd,
    const uint8_t *__restrict__ source, const int32_t *__restrict__ cu_span,
    const int32_t *__restrict__ n_emit, const int32_t *__restrict__ resp_len, int num_reqs,
    int agg_mode, int dir_mode, float *__restrict__ out8) {
  __shared__ float sh[6][kLossWarps];
  const bool on_rev = dir_mode == IPD_DIR_SPLIT || dir_mode == IPD_DIR_REVERSE;
  const bool off_fwd = dir_mode == IPD_DIR_SPLIT || dir_mode == IPD_DIR_FORWARD;
  float sum_on = 0.f, sum_off = 0.f, numer = 0.f, denom = 0.f;
  int n_on = 0, n_off = 0;
  for (int r = threadIdx.x; r < num_reqs; r += kLossThreads) {
    float s_on = 0.f, s_off = 0.f;
    const int t0 = cu_span[r], t1 = cu_span[r + 1];
    if (t0 < 0 || t1 < t0) continue;  // offsets already reported by ipd_score_span
    for (int t = t0; t < t1; ++t) {
      const uint8_t z = source[t];
      if (z == 0) {
        s_on += on_rev ? kl_rev[t] : kl_fwd[t];
        ++n_on;
      } else if (z == 1) {
        s_off += off_fwd ? kl_fwd[t] : kl_rev[t];
        ++n_off;
      }
    }
    sum_on += s_on;
    sum_off += s_off;
    const int d = resp_len ? resp_len[r] : n_emit[r];
    if (d > 0) {
      if (agg_mode == IPD_AGG_SEQ_MEAN_TOKEN_MEAN) {
        numer += (s_on + s_off) / (float)d;
        denom += 1.f;
      } else {
        numer += s_on + s_off;
        denom += (float)d;
      }
    }
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float v[6] = {sum_on, sum_off, (float)n_on, (float)n_off, numer, denom};
#pragma unroll
  for (int q = 0; q < 6; ++q) {
    const float w = warp_tree_sum(v[q]);
    if (lane == 0) sh[q][warp] = w;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float a[6];
#pragma unroll
    for (int q = 0; q < 6; ++q) {
      a[q] = 0.f;
#pragma unroll
      for (int w = 0; w < kLossWarps; ++w) a[q] += sh[q][w];
    }
    const float nt = a[2] + a[3];
    out8[0] = a[5] > 0.f ? a[4] / a[5] : 0.f;
    out8[1] = a[0];
    out8[2] = a[1];
    out8[3] = a[2];
    out8[4] = a[3];
    out8[5] = nt > 0.f ? a[3] / nt : 0.f;
    out8[6] = a[4];
    out8[7] = a[5];
  }
}

}  // namespace

// The loss needs no scratch: one CTA reduces the step in shared memory.
extern "C" size_t ipd_loss_workspace_size(int /*num_reqs*/) { return 0; }

extern "C" int ipd_split_loss(const float *kl_rev, const float *kl_fwd, const uint8_t *source,
                              const int32_t *cu_span, const int32_t *n_emit,
                              const int32_t *resp_len, int num_reqs, int agg_mode, int dir_mode,
                              float *out8, void *workspace, size_t workspace_bytes,
                              ipd_stream_t stream) {
  (void)workspace;
  (void)workspace_bytes;
  if (num_reqs < 0 || !out8) return IPD_ERR_INVALID_ARG;
  if (agg_mode != IPD_AGG_SEQ_MEAN_TOKEN_MEAN && agg_mode != IPD_AGG_GLOBAL_TOKEN_MEAN)
    return IPD_ERR_INVALID_ARG;
  if (dir_mode < IPD_DIR_SPLIT || dir_mode > IPD_DIR_INVERSE) return IPD_ERR_INVALID_ARG;
  if (num_reqs > 0 && (!kl_rev || !kl_fwd || !source || !cu_span || (!n_emit && !resp_len)))
    return IPD_ERR_INVALID_ARG;
  split_loss_kernel<<<1, kLossThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      kl_rev, kl_fwd, source, cu_span, n_emit, resp_len, num_reqs, agg_mode, dir_mode, out8);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}

// ---------------------------------------------------------------------------
// Gradient of the objective with respect to the student's logits.
//
// loss_grad_sparse_kernel: one warp per span position.  Lane j < K holds the
// student's j-th top-K id and the teacher's j-th; a teacher id already in the
// student's list is dropped, so the warp holds S_t = Top_K(pi) u Top_K(q)
// once.  It gathers both models' logits at S_t, renormalises each on S_t
// (Eq. topk_normalization) and writes w_t times the derivative of the
// position's KL (Eq. ipd_off_loss) with the support held fixed:
//   reverse KL(pi_bar || q_bar): pi_bar_v (log pi_bar_v - log q_bar_v - KL)
//   forward KL(q_bar || pi_bar): pi_bar_v - q_bar_v.
// w_t is the position's weight in Eq. (ipd_objective): 1 / (D |x_r|) for the
// sequence-mean-token-mean, 1 / D for the global token mean (App. B.3), with D
// the denominator ipd_split_loss reported.
//
// loss_grad_dense_kernel: the vocabulary-wide form.  Each CTA takes chunks of
// the flat [T][V] array, writes zeros over its chunk with 16-byte stores, and
// after a CTA barrier stores the sparse entries that fall inside the chunk.
// ---------------------------------------------------------------------------
namespace {

constexpr int kGradThreads = 256;
constexpr int kGradWarps = kGradThreads / 32;
constexpr int kDenseThreads = 256;
constexpr long long kDenseChunk = 8192;  // elements per CTA step (multiple of 8)

__global__ void __launch_bounds__(kGradThreads) loss_grad_sparse_kernel(
    const uint16_t *__restrict__ ls, const uint16_t *__restrict__ lt,
    const int32_t *__restrict__ topk_s, const int32_t *__restrict__ topk_t,
    const uint8_t *__restrict__ source, const int32_t *__restrict__ cu_span,
    const int32_t *__restrict__ n_emit, const int32_t *__restrict__ resp_len,
    const float *__restrict__ out8, int num_reqs, int total_tokens, int vocab, int K,
    int agg_mode, int dir_mode, float grad_scale, int32_t *__restrict__ grad_idx,
    float *__restrict__ grad_val) {
  const int lane = threadIdx.x & 31;
  const int t = blockIdx.x * kGradWarps + (threadIdx.x >> 5);
  if (t >= total_tokens) return;
  const int slots = 2 * K;
  int32_t *gi = grad_idx + (size_t)t * slots;
  float *gv = grad_val + (size_t)t * slots;
  // the request holding position t: the last r with cu_span[r] <= t
  int lo = 0, hi = num_reqs - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (cu_span[mid] <= t) lo = mid;
    else hi = mid - 1;
  }
  const int d = resp_len ? resp_len[lo] : n_emit[lo];
  const float D = out8[7];
  const uint8_t z = source[t];
  float w = 0.f;
  if ((z == 0 || z == 1) && d > 0 && D > 0.f)
    w = agg_mode == IPD_AGG_SEQ_MEAN_TOKEN_MEAN ? grad_scale / (D * (float)d) : grad_scale / D;
  int iS = 0, iT = 0;
  bool bad = false;
  if (w != 0.f && lane < K) {
    iS = topk_s[(size_t)t * K + lane];
    iT = topk_t[(size_t)t * K + lane];
    bad = iS < 0 || iS >= vocab || iT < 0 || iT >= vocab;
  }
  if (__any_sync(0xffffffffu, bad)) {
    if (lane == 0) ipd_set_error(&g_loss_err, IPD_DEVERR_TOKEN);
    w = 0.f;
  }
  if (w == 0.f) {
    for (int j = lane; j < slots; j += 32) {
      gi[j] = -1;
      gv[j] = 0.f;
    }
    return;
  }
  bool dupT = false;
  for (int j = 0; j < K; ++j) dupT |= (__shfl_sync(0xffffffffu, iS, j) == iT);
  const bool hasS = lane < K, hasT = lane < K && !dupT;
  const uint16_t *rowS = ls + (size_t)t * vocab, *rowT = lt + (size_t)t * vocab;
  float aS = 0.f, bS = 0.f, aT = 0.f, bT = 0.f;
  if (hasS) {
    aS = bf16f(rowS[iS]);
    bS = bf16f(rowT[iS]);
  }
  if (hasT) {
    aT = bf16f(rowS[iT]);
    bT = bf16f(rowT[iT]);
  }
  const float ma = warp_max(fmaxf(hasS ? aS : -INFINITY, hasT ? aT : -INFINITY));
  const float mb = warp_max(fmaxf(hasS ? bS : -INFINITY, hasT ? bT : -INFINITY));
  const float sa = warp_sum((hasS ? expf(aS - ma) : 0.f) + (hasT ? expf(aT - ma) : 0.f));
  const float sb = warp_sum((hasS ? expf(bS - mb) : 0.f) + (hasT ? expf(bT - mb) : 0.f));
  const float lza = ma + logf(sa), lzb = mb + logf(sb);
  const float laS = aS - lza, lbS = bS - lzb, laT = aT - lza, lbT = bT - lzb;
  const float paS = hasS ? expf(laS) : 0.f, pbS = hasS ? expf(lbS) : 0.f;
  const float paT = hasT ? expf(laT) : 0.f, pbT = hasT ? expf(lbT) : 0.f;
  const bool use_rev = z == 0 ? (dir_mode == IPD_DIR_SPLIT || dir_mode == IPD_DIR_REVERSE)
                              : (dir_mode == IPD_DIR_REVERSE || dir_mode == IPD_DIR_INVERSE);
  float gS, gT;
  if (use_rev) {
    const float kr = warp_sum((paS > 0.f ? paS * (laS - lbS) : 0.f) +
                              (paT > 0.f ? paT * (laT - lbT) : 0.f));
    gS = paS > 0.f ? paS * (laS - lbS - kr) : 0.f;
    gT = paT > 0.f ? paT * (laT - lbT - kr) : 0.f;
  } else {
    gS = paS - pbS;
    gT = paT - pbT;
  }
  if (lane < K) {
    gi[lane] = iS;
    gv[lane] = w * gS;
    gi[K + lane] = hasT ? iT : -1;
    gv[K + lane] = hasT ? w * gT : 0.f;
  }
}

__device__ __forceinline__ void store_grad(float *p, float v) { *p = v; }
__device__ __forceinline__ void store_grad(uint16_t *p, float v) { *p = f2bf16(v); }

template <typename OutT>
__global__ void __launch_bounds__(kDenseThreads) loss_grad_dense_kernel(
    const int32_t *__restrict__ grad_idx, const float *__restrict__ grad_val, long long total,
    int vocab, int slots, OutT *__restrict__ dense) {
  constexpr int kPerVec = 16 / sizeof(OutT);
  const long long n_chunks = (total + kDenseChunk - 1) / kDenseChunk;
  for (long long c = blockIdx.x; c < n_chunks; c += gridDim.x) {
    const long long a = c * kDenseChunk;
    const long long b = a + kDenseChunk < total ? a + kDenseChunk : total;
    const long long va = a / kPerVec, vb = b / kPerVec;
    uint4 *dv = reinterpret_cast<uint4 *>(dense);
    for (long long i = va + threadIdx.x; i < vb; i += kDenseThreads) dv[i] = make_uint4(0, 0, 0, 0);
    for (long long e = vb * kPerVec + threadIdx.x; e < b; e += kDenseThreads) store_grad(dense + e, 0.f);
    __syncthreads();
    const long long r0 = a / vocab, r1 = (b - 1) / vocab;
    for (long long row = r0; row <= r1; ++row) {
      for (int j = threadIdx.x; j < slots; j += kDenseThreads) {
        const int idx = grad_idx[row * slots + j];
        if (idx < 0 || idx >= vocab) continue;
        const long long pos = row * vocab + idx;
        if (pos >= a && pos < b) store_grad(dense + pos, grad_val[row * slots + j]);
      }
    }
  }
}

}  // namespace

extern "C" __attribute__((visibility("hidden"))) unsigned int ipd_internal_take_loss_error() {
  unsigned int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_loss_err, sizeof(v)) != cudaSuccess) return 0xffffffffu;
  if (cudaMemcpyToSymbol(g_loss_err, &z, sizeof(z)) != cudaSuccess) return 0xffffffffu;
  return v;
}

extern "C" size_t ipd_loss_grad_workspace_size(int total_tokens, int K) {
  return (total_tokens < 0 || K < 0) ? 0 : 0;
}

extern "C" int ipd_split_loss_grad(const uint16_t *logits_student, const uint16_t *logits_teacher,
                                   const int32_t *topk_s, const int32_t *topk_t,
                                   const uint8_t *source, const int32_t *cu_span,
                                   const int32_t *n_emit, const int32_t *resp_len,
                                   const float *loss_out8, int num_reqs, int total_tokens,
                                   int vocab, int K, int agg_mode, int dir_mode, float grad_scale,
                                   int32_t *grad_idx, float *grad_val, void *grad_dense,
                                   int dense_dtype, void *workspace, size_t workspace_bytes,
                                   ipd_stream_t stream) {
  (void)workspace;
  (void)workspace_bytes;
  if (num_reqs < 0 || total_tokens < 0 || vocab < 1) return IPD_ERR_INVALID_ARG;
  if (K < 1 || K > IPD_MAX_K || K > vocab) return IPD_ERR_UNSUPPORTED;
  if (agg_mode != IPD_AGG_SEQ_MEAN_TOKEN_MEAN && agg_mode != IPD_AGG_GLOBAL_TOKEN_MEAN)
    return IPD_ERR_INVALID_ARG;
  if (dir_mode < IPD_DIR_SPLIT || dir_mode > IPD_DIR_INVERSE) return IPD_ERR_INVALID_ARG;
  if (!(grad_scale - grad_scale == 0.f)) return IPD_ERR_INVALID_ARG;  // NaN or infinite
  if (grad_dense && dense_dtype != IPD_DTYPE_F32 && dense_dtype != IPD_DTYPE_BF16)
    return IPD_ERR_INVALID_ARG;
  if (grad_dense && (reinterpret_cast<uintptr_t>(grad_dense) & 15u)) return IPD_ERR_INVALID_ARG;
  if (total_tokens == 0) return IPD_OK;
  if (num_reqs == 0 || !logits_student || !logits_teacher || !topk_s || !topk_t || !source ||
      !cu_span || (!n_emit && !resp_len) || !loss_out8 || !grad_idx || !grad_val)
    return IPD_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int blocks = (total_tokens + kGradWarps - 1) / kGradWarps;
  loss_grad_sparse_kernel<<<blocks, kGradThreads, 0, st>>>(
      logits_student, logits_teacher, topk_s, topk_t, source, cu_span, n_emit, resp_len,
      loss_out8, num_reqs, total_tokens, vocab, K, agg_mode, dir_mode, grad_scale, grad_idx,
      grad_val);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  if (grad_dense) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return IPD_ERR_CUDA;
    const long long total = (long long)total_tokens * vocab;
    const long long n_chunks = (total + kDenseChunk - 1) / kDenseChunk;
    const long long cap = (long long)sms * 8;
    const int grid = (int)(n_chunks < cap ? n_chunks : cap);
    if (dense_dtype == IPD_DTYPE_F32)
      loss_grad_dense_kernel<float><<<grid, kDenseThreads, 0, st>>>(
          grad_idx, grad_val, total, vocab, 2 * K, static_cast<float *>(grad_dense));
    else
      loss_grad_dense_kernel<uint16_t><<<grid, kDenseThreads, 0, st>>>(
          grad_idx, grad_val, total, vocab, 2 * K, static_cast<uint16_t *>(grad_dense));
    if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  }
  return IPD_OK;
}
