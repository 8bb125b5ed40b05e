// Source-split objective of one verify step (Sec. 3.2.2, Eq. ipd_off_loss and
// Eq. ipd_objective; global token mean of App. B.3; KL-direction variants of
// the ablation in Sec. 4.3).  One CTA; every thread reduces a fixed set of
// requests in position order and a fixed-shape tree combines the threads, so
// the result is bitwise reproducible.
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace {

constexpr int kLossThreads = 512;

__global__ void __launch_bounds__(kLossThreads) split_loss_kernel(
    const float *__restrict__ kl_rev, const float *__restrict__ kl_fwd,
    const uint8_t *__restrict__ source, const int32_t *__restrict__ cu_span,
    const int32_t *__restrict__ n_emit, const int32_t *__restrict__ resp_len, int num_reqs,
    int agg_mode, int dir_mode, float *__restrict__ out8) {
  __shared__ float sh[6][kLossThreads];
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
  const int tid = threadIdx.x;
  sh[0][tid] = sum_on;
  sh[1][tid] = sum_off;
  sh[2][tid] = (float)n_on;
  sh[3][tid] = (float)n_off;
  sh[4][tid] = numer;
  sh[5][tid] = denom;
  __syncthreads();
  for (int stride = kLossThreads / 2; stride > 0; stride >>= 1) {
    if (tid < stride) {
#pragma unroll
      for (int q = 0; q < 6; ++q) sh[q][tid] += sh[q][tid + stride];
    }
    __syncthreads();
  }
  if (tid == 0) {
    const float nt = sh[2][0] + sh[3][0];
    out8[0] = sh[5][0] > 0.f ? sh[4][0] / sh[5][0] : 0.f;
    out8[1] = sh[0][0];
    out8[2] = sh[1][0];
    out8[3] = sh[2][0];
    out8[4] = sh[3][0];
    out8[5] = nt > 0.f ? sh[3][0] / nt : 0.f;
    out8[6] = sh[4][0];
    out8[7] = sh[5][0];
  }
}

}  // namespace

extern "C" size_t ipd_loss_workspace_size(int num_reqs) { return num_reqs < 0 ? 0 : 0; }

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
