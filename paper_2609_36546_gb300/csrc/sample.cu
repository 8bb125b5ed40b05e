// Seeded sampling from the full softmax at a given temperature (training
// rollouts sample at temperature 1, top-p 1: App. A, training configuration).
//
// A draw is a deterministic function of (logits row, seed, draw number,
// inverse temperature), defined bit-exactly so that any device reproduces it:
//   bits_v  = word v % 4 of Philox4x32-10(counter = (v / 4, draw_lo, draw_hi, 0),
//             key = (seed_lo, seed_hi))   (Salmon et al., SC 2011)
//   u_v     = (2 (bits_v >> 9) + 1) 2^-24                       in (0, 1), exact
//   s_v     = fl(l_v c) - lg2(-lg2(u_v)),   c = fl(fp32(log2 e) * inv_temperature)
//   token   = argmax_v s_v, ties to the lower id
// with lg2 the fixed fp32 procedure below and every product and sum rounded
// to fp32 on its own (no fused multiply-add).  This is the Gumbel-max trick in
// base 2: l c - lg2(-lg2 u) = log2(e) (l / T - ln(-ln u)) - log2(ln 2).
//
// Kernels: the vocabulary of each sampled row is cut into chunks of 8192
// entries, one CTA per (row, chunk).  A thread takes 8 consecutive entries at
// a time (one 16-byte load, two Philox blocks) and keeps the largest
// (score, -id) key; a CTA reduces its keys and stores one partial per chunk;
// a second kernel reduces the chunks of each row (max is order-free, so the
// result does not depend on the schedule).
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace {

constexpr uint32_t kPhiloxM0 = 0xD2511F53u, kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u, kPhiloxW1 = 0xBB67AE85u;
constexpr uint32_t kLog2eBits = 0x3FB8AA3Bu;
constexpr int kSampleThreads = 256;
constexpr int kSampleChunk = 8192;  // vocabulary entries per CTA (multiple of 8)

// log2(1 + t) = t P(t) on [sqrt(1/2) - 1, sqrt(2) - 1]: least-squares fit of
// log2(1 + t) / t on Chebyshev nodes, coefficients rounded to fp32 (lowest
// degree first); |lg2(x) - log2(x)| <= 1.1e-6 for normal x.
__device__ __forceinline__ float lg2_fixed(float x) {
  const uint32_t b = __float_as_uint(x);
  int e = (int)((b >> 23) & 0xffu) - 127;
  uint32_t mb = (b & 0x7fffffu) | 0x3f800000u;
  if (mb > 0x3fb504f3u) {  // m > sqrt(2): halve it
    mb -= 0x00800000u;
    e += 1;
  }
  const float t = __fsub_rn(__uint_as_float(mb), 1.0f);
  float p = __uint_as_float(0xBE15B661u);
  p = __fadd_rn(__fmul_rn(p, t), __uint_as_float(0x3E6FD4B5u));
  p = __fadd_rn(__fmul_rn(p, t), __uint_as_float(0xBE7ECB25u));
  p = __fadd_rn(__fmul_rn(p, t), __uint_as_float(0x3E92FB93u));
  p = __fadd_rn(__fmul_rn(p, t), __uint_as_float(0xBEB871A3u));
  p = __fadd_rn(__fmul_rn(p, t), __uint_as_float(0x3EF63BADu));
  p = __fadd_rn(__fmul_rn(p, t), __uint_as_float(0xBF38AA93u));
  p = __fadd_rn(__fmul_rn(p, t), __uint_as_float(0x3FB8AA3Au));
  return __fadd_rn((float)e, __fmul_rn(t, p));
}

// Philox4x32 with 10 rounds.
__device__ __forceinline__ uint4 philox10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    const uint32_t lo0 = kPhiloxM0 * c.x, hi0 = __umulhi(kPhiloxM0, c.x);
    const uint32_t lo1 = kPhiloxM1 * c.z, hi1 = __umulhi(kPhiloxM1, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    k0 += kPhiloxW0;
    k1 += kPhiloxW1;
  }
  return c;
}

// (score, -id) as one ordered 64-bit key; -0 is folded onto +0
__device__ __forceinline__ unsigned long long score_key(float s, uint32_t v) {
  uint32_t b = __float_as_uint(s);
  if (b == 0x80000000u) b = 0u;
  const uint32_t o = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return ((unsigned long long)o << 32) | (unsigned long long)(0xffffffffu - v);
}

__device__ __forceinline__ unsigned long long max_u64(unsigned long long a, unsigned long long b) {
  return a > b ? a : b;
}

__device__ __forceinline__ float sample_score(uint32_t lbits16, uint32_t rbits, float c) {
  const float l = __uint_as_float(lbits16 << 16);
  const float u = __fmul_rn((float)((rbits >> 9) * 2u + 1u), 5.9604644775390625e-08f);  // 2^-24
  const float e = -lg2_fixed(u);
  return __fsub_rn(__fmul_rn(l, c), lg2_fixed(e));
}

// mode 0: row r of `rows0` with draw draw_id[r].  mode 1 (after a verdict):
// request r draws the first token of its next span from the next driver's
// row n_emit[r] of its span (rows0 = student, rows1 = teacher) with draw
// draw_id[r] + prefix_len[r] + n_emit[r]; no draw when the request ended or
// every span token was emitted.
__global__ void __launch_bounds__(kSampleThreads) sample_partial_kernel(
    int mode, const uint16_t *__restrict__ rows0, const uint16_t *__restrict__ rows1, int vocab,
    int n_chunks, uint32_t seed_lo, uint32_t seed_hi, const uint64_t *__restrict__ draw_id,
    float inv_temperature, const int32_t *__restrict__ cu_span,
    const int32_t *__restrict__ prefix_len, const int32_t *__restrict__ n_emit,
    const uint8_t *__restrict__ next_driver, const uint8_t *__restrict__ done,
    unsigned long long *__restrict__ partial) {
  __shared__ unsigned long long s_best[kSampleThreads / 32];
  const int r = blockIdx.x / n_chunks, chunk = blockIdx.x % n_chunks;
  const uint16_t *row;
  uint64_t draw = draw_id ? draw_id[r] : 0ull;
  if (mode == 1) {
    const int t0 = cu_span[r], t1 = cu_span[r + 1], n = n_emit[r];
    if (done[r] || t0 < 0 || n < 0 || n >= t1 - t0) {
      if (threadIdx.x == 0) partial[blockIdx.x] = 0ull;
      return;
    }
    row = (next_driver[r] ? rows1 : rows0) + (size_t)(t0 + n) * vocab;
    draw += (uint64_t)(int64_t)(prefix_len[r] + n);
  } else {
    row = rows0 + (size_t)r * vocab;
  }
  const uint32_t dlo = (uint32_t)draw, dhi = (uint32_t)(draw >> 32);
  const float c = __fmul_rn(__uint_as_float(kLog2eBits), inv_temperature);
  const int end = min((chunk + 1) * kSampleChunk, vocab);
  unsigned long long best = 0ull;
  for (int v0 = chunk * kSampleChunk + threadIdx.x * 8; v0 < end; v0 += kSampleThreads * 8) {
    const uint4 raw = __ldg(reinterpret_cast<const uint4 *>(row + v0));
    const uint32_t g = (uint32_t)v0 >> 2;
    const uint4 ra = philox10(make_uint4(g, dlo, dhi, 0u), seed_lo, seed_hi);
    const uint4 rb = philox10(make_uint4(g + 1u, dlo, dhi, 0u), seed_lo, seed_hi);
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
    const uint32_t rr[8] = {ra.x, ra.y, ra.z, ra.w, rb.x, rb.y, rb.z, rb.w};
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const uint32_t lb = (e & 1) ? (w[e >> 1] >> 16) : (w[e >> 1] & 0xffffu);
      best = max_u64(best, score_key(sample_score(lb, rr[e], c), (uint32_t)(v0 + e)));
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) best = max_u64(best, __shfl_xor_sync(0xffffffffu, best, o));
  if ((threadIdx.x & 31) == 0) s_best[threadIdx.x >> 5] = best;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long b = s_best[0];
#pragma unroll
    for (int i = 1; i < kSampleThreads / 32; ++i) b = max_u64(b, s_best[i]);
    partial[blockIdx.x] = b;
  }
}

// one warp per row: the best of the row's chunk keys -> token id (-1: none)
__global__ void __launch_bounds__(256) sample_finalize_kernel(
    const unsigned long long *__restrict__ partial, int n_rows, int n_chunks,
    int32_t *__restrict__ tokens) {
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= n_rows) return;
  unsigned long long b = 0ull;
  if (partial)
    for (int c = lane; c < n_chunks; c += 32) b = max_u64(b, partial[(size_t)r * n_chunks + c]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) b = max_u64(b, __shfl_xor_sync(0xffffffffu, b, o));
  if (lane == 0) tokens[r] = b ? (int32_t)(0xffffffffu - (uint32_t)b) : -1;
}

int n_chunks_for(int vocab) { return (vocab + kSampleChunk - 1) / kSampleChunk; }

}  // namespace

extern "C" __attribute__((visibility("hidden"))) size_t ipd_internal_sample_ws(int n_rows,
                                                                              int vocab) {
  return (size_t)n_rows * n_chunks_for(vocab) * sizeof(unsigned long long);
}

// The draw after a verdict, launched by ipd_score_span_ex (ws: ipd_internal_sample_ws bytes,
// or NULL when the step has no span tokens).
extern "C" __attribute__((visibility("hidden"))) int ipd_internal_sample_after_verdict(
    const uint16_t *ls, const uint16_t *lt, int num_reqs, int total_tokens, int vocab,
    uint64_t seed, const uint64_t *draw_base, float inv_temperature, const int32_t *cu_span,
    const int32_t *prefix_len, const int32_t *n_emit, const uint8_t *next_driver,
    const uint8_t *done, int32_t *next_token, void *ws, cudaStream_t st) {
  const int nc = n_chunks_for(vocab);
  unsigned long long *partial = nullptr;
  if (total_tokens > 0) {
    partial = static_cast<unsigned long long *>(ws);
    sample_partial_kernel<<<num_reqs * nc, kSampleThreads, 0, st>>>(
        1, ls, lt, vocab, nc, (uint32_t)seed, (uint32_t)(seed >> 32), draw_base, inv_temperature,
        cu_span, prefix_len, n_emit, next_driver, done, partial);
    if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  }
  sample_finalize_kernel<<<(num_reqs + 7) / 8, 256, 0, st>>>(partial, num_reqs, nc, next_token);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}

extern "C" size_t ipd_sample_workspace_size(int n_rows, int vocab) {
  if (n_rows < 0 || vocab < 1) return 0;
  return ipd_internal_sample_ws(n_rows, vocab);
}

extern "C" int ipd_sample(const uint16_t *logits, int n_rows, int vocab, uint64_t seed,
                          const uint64_t *draw_id, float inv_temperature, int32_t *tokens,
                          void *workspace, size_t workspace_bytes, ipd_stream_t stream) {
  if (n_rows < 0) return IPD_ERR_INVALID_ARG;
  if (vocab < 8 || vocab % 8) return IPD_ERR_UNSUPPORTED;
  if (!(inv_temperature > 0.f) || !(inv_temperature - inv_temperature == 0.f))
    return IPD_ERR_INVALID_ARG;  // not positive and finite
  if (n_rows == 0) return IPD_OK;
  if (!logits || !tokens || ((uintptr_t)logits & 15)) return IPD_ERR_INVALID_ARG;
  const int nc = n_chunks_for(vocab);
  if ((long long)n_rows * nc > 0x7fffffffLL) return IPD_ERR_UNSUPPORTED;
  if (!workspace || workspace_bytes < ipd_internal_sample_ws(n_rows, vocab) ||
      ((uintptr_t)workspace & 7))
    return IPD_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  unsigned long long *partial = static_cast<unsigned long long *>(workspace);
  sample_partial_kernel<<<n_rows * nc, kSampleThreads, 0, st>>>(
      0, logits, nullptr, vocab, nc, (uint32_t)seed, (uint32_t)(seed >> 32), draw_id,
      inv_temperature, nullptr, nullptr, nullptr, nullptr, nullptr, partial);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  sample_finalize_kernel<<<(n_rows + 7) / 8, 256, 0, st>>>(partial, n_rows, nc, tokens);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}
