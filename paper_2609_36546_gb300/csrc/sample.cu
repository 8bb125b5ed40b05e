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
constexpr int kSampleGridCap = 2048;  // CTAs of one launch when the rows are fewer

// The ten round keys of one seed (key + i * Weyl increment), passed by value
// so that the rounds read them from the kernel's parameter bank.
struct PhiloxKeys {
  uint32_t k0[10], k1[10];
};

PhiloxKeys philox_keys(uint64_t seed) {
  PhiloxKeys k;
  uint32_t a = (uint32_t)seed, b = (uint32_t)(seed >> 32);
  for (int i = 0; i < 10; ++i) {
    k.k0[i] = a;
    k.k1[i] = b;
    a += kPhiloxW0;
    b += kPhiloxW1;
  }
  return k;
}

// Philox4x32 with 10 rounds.
__device__ __forceinline__ uint4 philox10(uint4 c, const PhiloxKeys &key) {
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    const uint32_t lo0 = kPhiloxM0 * c.x, hi0 = __umulhi(kPhiloxM0, c.x);
    const uint32_t lo1 = kPhiloxM1 * c.z, hi1 = __umulhi(kPhiloxM1, c.z);
    c = make_uint4(hi1 ^ c.y ^ key.k0[i], lo1, hi0 ^ c.w ^ key.k1[i], lo0);
  }
  return c;
}

// (score, -id) as one ordered 64-bit key; -0 is folded onto +0; 0 = no entry
__device__ __forceinline__ unsigned long long score_key(float s, int v) {
  if (v < 0) return 0ull;
  uint32_t b = __float_as_uint(s);
  if (b == 0x80000000u) b = 0u;
  const uint32_t o = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return ((unsigned long long)o << 32) | (unsigned long long)(0xffffffffu - (uint32_t)v);
}

__device__ __forceinline__ unsigned long long max_u64(unsigned long long a, unsigned long long b) {
  return a > b ? a : b;
}

IPD_DEVINL unsigned long long f2_mul(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// The fixed lg2 of the sampler, of two positive values at once: for x =
// 2^e m with m in (sqrt(1/2), sqrt(2)], lg2(x) = e + t P(t) with t = m - 1
// and P by Horner's rule; P's coefficients are a least-squares fit of
// log2(1 + t) / t on Chebyshev nodes of [sqrt(1/2) - 1, sqrt(2) - 1], rounded
// to fp32 (|lg2(x) - log2(x)| <= 1.1e-6 for normal x).  The integer steps run
// per lane, the fp32 steps on packed pairs (each lane rounded exactly like the
// scalar operation, no fused multiply-add).  The reduction to m in (sqrt(1/2), sqrt(2)] subtracts the bit
// pattern just above sqrt(1/2) and shifts arithmetically: e = floor((b -
// bits(sqrt(1/2))^+) / 2^23), m = b - e 2^23 -- the same (m, e) as halving m
// when it exceeds sqrt(2); e enters as (1.5 2^23 + e) - 1.5 2^23, exact.
__device__ __forceinline__ unsigned long long lg2_x2(unsigned long long x2) {
  float x0, x1;
  f2_unpack(x2, x0, x1);
  const uint32_t b0 = __float_as_uint(x0), b1 = __float_as_uint(x1);
  const int e0 = (int)(b0 - 0x3f3504f4u) >> 23, e1 = (int)(b1 - 0x3f3504f4u) >> 23;
  const uint32_t m0 = b0 - ((uint32_t)e0 << 23), m1 = b1 - ((uint32_t)e1 << 23);
  const unsigned long long ef = f2_sub(
      f2_pack(__uint_as_float(0x4b400000u + (uint32_t)e0), __uint_as_float(0x4b400000u + (uint32_t)e1)),
      f2_pack(12582912.0f, 12582912.0f));
  const unsigned long long t =
      f2_sub(f2_pack(__uint_as_float(m0), __uint_as_float(m1)), f2_pack(1.0f, 1.0f));
  const float c7 = __uint_as_float(0xBE15B661u), c6 = __uint_as_float(0x3E6FD4B5u),
              c5 = __uint_as_float(0xBE7ECB25u), c4 = __uint_as_float(0x3E92FB93u),
              c3 = __uint_as_float(0xBEB871A3u), c2 = __uint_as_float(0x3EF63BADu),
              c1 = __uint_as_float(0xBF38AA93u), c0 = __uint_as_float(0x3FB8AA3Au);
  unsigned long long p = f2_pack(c7, c7);
  p = f2_add(f2_mul(p, t), f2_pack(c6, c6));
  p = f2_add(f2_mul(p, t), f2_pack(c5, c5));
  p = f2_add(f2_mul(p, t), f2_pack(c4, c4));
  p = f2_add(f2_mul(p, t), f2_pack(c3, c3));
  p = f2_add(f2_mul(p, t), f2_pack(c2, c2));
  p = f2_add(f2_mul(p, t), f2_pack(c1, c1));
  p = f2_add(f2_mul(p, t), f2_pack(c0, c0));
  return f2_add(ef, f2_mul(t, p));
}

// scores of two entries: u = (2 (bits >> 9) + 1) 2^-24, formed exactly as
// (1 + (bits >> 9) 2^-23) - (1 - 2^-24); s = l c - lg2(-lg2 u)
__device__ __forceinline__ void score_x2(uint32_t lbits2, uint32_t r0, uint32_t r1,
                                         unsigned long long c2, float &s0, float &s1) {
  const unsigned long long u = f2_sub(
      f2_pack(__uint_as_float(0x3f800000u | (r0 >> 9)), __uint_as_float(0x3f800000u | (r1 >> 9))),
      f2_pack(__uint_as_float(0x3f7fffffu), __uint_as_float(0x3f7fffffu)));
  const unsigned long long e = f2_mul(lg2_x2(u), f2_pack(-1.0f, -1.0f));  // -lg2 u > 0
  const unsigned long long g = lg2_x2(e);                                    // lg2(-lg2 u)
  const unsigned long long l = f2_pack(bf16lo(lbits2), bf16hi(lbits2));
  f2_unpack(f2_sub(f2_mul(l, c2), g), s0, s1);
}

// One draw per row of a list of rows.  mode 0: row r is row r of `rows0`
// with draw number draw_id[r].  mode 1 (after a verdict): request r draws the
// first token of its next span from the next driver's row n_emit[r] of its
// span (rows0 = student, rows1 = teacher) with draw number draw_id[r] +
// prefix_len[r] + n_emit[r]; a request that ended or emitted every span token
// draws nothing.
//
// Work split: the rows' 8-entry vectors form one flat range that is cut into
// gridDim.x equal pieces, one per CTA (grid >= rows, so a piece meets at most
// two rows).  Each CTA stores its best key for the first and the second row
// it meets (0 where it meets none).
__global__ void __launch_bounds__(kSampleThreads, 5) sample_partial_kernel(
    int mode, const uint16_t *__restrict__ rows0, const uint16_t *__restrict__ rows1, int vocab,
    int n_rows, const PhiloxKeys key, const uint64_t *__restrict__ draw_id,
    float inv_temperature, const int32_t *__restrict__ cu_span,
    const int32_t *__restrict__ prefix_len, const int32_t *__restrict__ n_emit,
    const uint8_t *__restrict__ next_driver, const uint8_t *__restrict__ done,
    unsigned long long *__restrict__ partial) {
  __shared__ unsigned long long s_best[2][kSampleThreads / 32];
  __shared__ const uint16_t *s_row[2];
  __shared__ uint32_t s_draw[2][2];
  const long long nv = vocab >> 3;  // vectors per row
  const long long total = nv * n_rows;
  const long long lo = total * blockIdx.x / gridDim.x, hi = total * (blockIdx.x + 1) / gridDim.x;
  const int row_lo = (int)(lo / nv);
  const long long boundary = (long long)(row_lo + 1) * nv;
  if (threadIdx.x < 2) {
    const int r = row_lo + (int)threadIdx.x;
    const uint16_t *row = nullptr;
    uint64_t draw = 0ull;
    if (r < n_rows) {
      draw = draw_id ? draw_id[r] : 0ull;
      if (mode == 1) {
        const int t0 = cu_span[r], t1 = cu_span[r + 1], n = n_emit[r];
        if (!(done[r] || t0 < 0 || n < 0 || n >= t1 - t0)) {
          row = (next_driver[r] ? rows1 : rows0) + (size_t)(t0 + n) * vocab;
          draw += (uint64_t)(int64_t)(prefix_len[r] + n);
        }
      } else {
        row = rows0 + (size_t)r * vocab;
      }
    }
    s_row[threadIdx.x] = row;
    s_draw[threadIdx.x][0] = (uint32_t)draw;
    s_draw[threadIdx.x][1] = (uint32_t)(draw >> 32);
  }
  __syncthreads();
  const float cf = __fmul_rn(__uint_as_float(kLog2eBits), inv_temperature);
  const unsigned long long c2 = f2_pack(cf, cf);
  // per thread and row: the best score and its id; entries come in increasing
  // id, so a strict comparison keeps the lower id of equal scores (-0 == +0
  // too), and a row whose entries all score -inf keeps its first id
  float bs0 = -INFINITY, bs1 = -INFINITY;
  int bv0 = -1, bv1 = -1;
  for (long long vec = lo + threadIdx.x; vec < hi; vec += kSampleThreads) {
    const int k = vec >= boundary ? 1 : 0;
    const uint16_t *row = s_row[k];
    if (row == nullptr) continue;
    const int v0 = (int)(vec - (long long)(row_lo + k) * nv) * 8;
    float cbs = k ? bs1 : bs0;
    int cbv = k ? bv1 : bv0;
    if (cbv < 0) cbv = v0;
    const uint4 raw = __ldg(reinterpret_cast<const uint4 *>(row + v0));
    const uint32_t g = (uint32_t)v0 >> 2;
    const uint4 ra = philox10(make_uint4(g, s_draw[k][0], s_draw[k][1], 0u), key);
    const uint4 rb = philox10(make_uint4(g + 1u, s_draw[k][0], s_draw[k][1], 0u), key);
    float sc[8];
    score_x2(raw.x, ra.x, ra.y, c2, sc[0], sc[1]);
    score_x2(raw.y, ra.z, ra.w, c2, sc[2], sc[3]);
    score_x2(raw.z, rb.x, rb.y, c2, sc[4], sc[5]);
    score_x2(raw.w, rb.z, rb.w, c2, sc[6], sc[7]);
    // the vector's best; a new record (rare after the first vectors) looks up
    // its first entry
    const float m8 = fmaxf(fmaxf(fmaxf(sc[0], sc[1]), fmaxf(sc[2], sc[3])),
                           fmaxf(fmaxf(sc[4], sc[5]), fmaxf(sc[6], sc[7])));
    if (m8 > cbs) {
      int e = 0;
#pragma unroll
      for (int j = 7; j >= 0; --j)
        if (sc[j] == m8) e = j;
      cbs = m8;
      cbv = v0 + e;
    }
    if (k) {
      bs1 = cbs;
      bv1 = cbv;
    } else {
      bs0 = cbs;
      bv0 = cbv;
    }
  }
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    unsigned long long b = k ? score_key(bs1, bv1) : score_key(bs0, bv0);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) b = max_u64(b, __shfl_xor_sync(0xffffffffu, b, o));
    if ((threadIdx.x & 31) == 0) s_best[k][threadIdx.x >> 5] = b;
  }
  __syncthreads();
  if (threadIdx.x < 2) {
    unsigned long long b = 0ull;
#pragma unroll
    for (int i = 0; i < kSampleThreads / 32; ++i) b = max_u64(b, s_best[threadIdx.x][i]);
    partial[2 * (size_t)blockIdx.x + threadIdx.x] = b;
  }
}

// one warp per row: the best key over the CTAs whose piece meets the row ->
// token id (-1: none)
__global__ void __launch_bounds__(256) sample_finalize_kernel(
    const unsigned long long *__restrict__ partial, int n_rows, int vocab, int grid,
    int32_t *__restrict__ tokens) {
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= n_rows) return;
  unsigned long long b = 0ull;
  if (partial) {
    const long long nv = vocab >> 3, total = nv * n_rows;
    // CTA i covers [floor(i total / grid), floor((i + 1) total / grid)); the
    // CTA holding vector x is the largest i with floor(i total / grid) <= x
    auto cta_of = [&](long long x) { return (int)(((x + 1) * grid + total - 1) / total) - 1; };
    const int i0 = cta_of((long long)r * nv), i1 = cta_of((long long)(r + 1) * nv - 1);
    for (int i = i0 + lane; i <= i1; i += 32) {
      const int first_row = (int)((total * i / grid) / nv);
      b = max_u64(b, partial[2 * (size_t)i + (first_row == r ? 0 : 1)]);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) b = max_u64(b, __shfl_xor_sync(0xffffffffu, b, o));
  if (lane == 0) tokens[r] = b ? (int32_t)(0xffffffffu - (uint32_t)b) : -1;
}

// CTAs of one launch: every resident slot of the GPU once (so the equal
// pieces run as one wave), at least one per row
int sample_grid(int n_rows) {
  static int cap[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return -1;
  if (cap[dev] == 0) {
    int sms = 0, per_sm = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, sample_partial_kernel,
                                                      kSampleThreads, 0) != cudaSuccess)
      return -1;
    const int c = sms * (per_sm > 0 ? per_sm : 1);
    cap[dev] = c < kSampleGridCap ? c : kSampleGridCap;
  }
  return n_rows > cap[dev] ? n_rows : cap[dev];
}

}  // namespace

extern "C" __attribute__((visibility("hidden"))) size_t ipd_internal_sample_ws(int n_rows,
                                                                              int vocab) {
  (void)vocab;
  const size_t g = n_rows > kSampleGridCap ? (size_t)n_rows : (size_t)kSampleGridCap;
  return 2 * g * sizeof(unsigned long long);
}

// The draw after a verdict, launched by ipd_score_span_ex (ws: ipd_internal_sample_ws bytes,
// or NULL when the step has no span tokens).
extern "C" __attribute__((visibility("hidden"))) int ipd_internal_sample_after_verdict(
    const uint16_t *ls, const uint16_t *lt, int num_reqs, int total_tokens, int vocab,
    uint64_t seed, const uint64_t *draw_base, float inv_temperature, const int32_t *cu_span,
    const int32_t *prefix_len, const int32_t *n_emit, const uint8_t *next_driver,
    const uint8_t *done, int32_t *next_token, void *ws, cudaStream_t st) {
  unsigned long long *partial = nullptr;
  int grid = 1;
  if (total_tokens > 0) {
    grid = sample_grid(num_reqs);
    if (grid < 0) return IPD_ERR_CUDA;
    partial = static_cast<unsigned long long *>(ws);
    sample_partial_kernel<<<grid, kSampleThreads, 0, st>>>(
        1, ls, lt, vocab, num_reqs, philox_keys(seed), draw_base,
        inv_temperature, cu_span, prefix_len, n_emit, next_driver, done, partial);
    if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  }
  sample_finalize_kernel<<<(num_reqs + 7) / 8, 256, 0, st>>>(partial, num_reqs, vocab, grid,
                                                              next_token);
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
  if ((long long)n_rows * (vocab >> 3) > 0x3fffffffffffLL) return IPD_ERR_UNSUPPORTED;
  if (!workspace || workspace_bytes < ipd_internal_sample_ws(n_rows, vocab) ||
      ((uintptr_t)workspace & 7))
    return IPD_ERR_WORKSPACE;
  const int grid = sample_grid(n_rows);
  if (grid < 0) return IPD_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  unsigned long long *partial = static_cast<unsigned long long *>(workspace);
  sample_partial_kernel<<<grid, kSampleThreads, 0, st>>>(
      0, logits, nullptr, vocab, n_rows, philox_keys(seed), draw_id,
      inv_temperature, nullptr, nullptr, nullptr, nullptr, nullptr, partial);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  sample_finalize_kernel<<<(n_rows + 7) / 8, 256, 0, st>>>(partial, n_rows, vocab, grid, tokens);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}
