// The vocabulary pass of the verify step (Sec. 3.1 top-K supports, Sec. 3.2.1
// coverage rules, Sec. 3.2.2 source-split KL terms, Sec. 3.2.3 verdict).
//
// Kernel 1 (row pass), one CTA per part of a logits row (2 rows per span
// position: the student's and the teacher's), one read of the row from HBM:
//   - the part's log-sum-exp (maximum and scaled sum, fp32),
//   - the part's exact top-K (K <= 32) under the order (logit desc, token id
//     asc), through a threshold filter, a per-warp queue of vectors that pass
//     it and a per-warp candidate buffer.
// Kernel 2 (epilogue), one CTA per request: each row's log Z and top-K from
// its parts, union support, renormalised KL in both directions, log-probs
// and feedback, coverage and margin, then the verdict of the request's span.
#include <algorithm>
#include <cooperative_groups.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "common.cuh"

IPD_DECLARE_ERROR_WORD(g_score_err);

namespace {

constexpr int kRowThreads = 128;  // eight row CTAs per SM: every row of a step in flight at once
constexpr int kRowWarps = kRowThreads / 32;
constexpr int kEpiThreads = 256;
constexpr int kMaxParts = 4;  // a logits row is split into up to this many parts, one CTA each
constexpr int kRowCtasPerSm = 8;  // resident row CTAs per SM (the kernel's launch bounds)
constexpr int kMaxGroups = 32;    // group maxima a row thread keeps
constexpr int kMaxGroupVecs = 8;  // vectors a lane puts on its warp's list per round
constexpr int kBuf = 64;     // per-warp candidate buffer: up to 32 kept keys + one round of 32

// One part of one logits row.
struct RowOut {
  float m;  // maximum logit of the part (-inf if the part is empty)
  float s;  // sum over the part of exp(l - m)
  float u;  // sum over the part of exp(l - m) * l (entropy; 0 unless it was asked for)
  int skipped;  // needed-rows pass only: 1 if the row was not read (not needed)
  unsigned long long keys[IPD_MAX_K];  // the part's best keys, best first, 0 past the end
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

// Bitonic sort of one float per lane, descending over lanes.
__device__ __forceinline__ float warp_sort_desc_f(float k, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int j = size >> 1; j > 0; j >>= 1) {
      const float o = __shfl_xor_sync(0xffffffffu, k, j);
      const bool lower = (lane & j) == 0;
      const bool desc = (lane & size) == 0;
      k = (lower == desc) ? fmaxf(k, o) : fminf(k, o);
    }
  }
  return k;
}

// Top 32 of two descending lists of 32 (one entry per lane), descending:
// max(a[l], b[31 - l]) is a bitonic sequence holding the 32 largest entries,
// which a bitonic merge (five compare-exchange steps) sorts.
__device__ __forceinline__ float warp_top32_f(float a, float b, int lane) {
  float c = fmaxf(a, __shfl_sync(0xffffffffu, b, 31 - lane));
#pragma unroll
  for (int j = 16; j > 0; j >>= 1) {
    const float o = __shfl_xor_sync(0xffffffffu, c, j);
    c = (lane & j) ? fminf(c, o) : fmaxf(c, o);
  }
  return c;
}
__device__ __forceinline__ unsigned long long warp_top32_u64(unsigned long long a,
                                                             unsigned long long b, int lane) {
  const unsigned long long br = shfl_u64(b, 31 - lane);
  unsigned long long c = a > br ? a : br;
#pragma unroll
  for (int j = 16; j > 0; j >>= 1) {
    const unsigned long long o = __shfl_xor_sync(0xffffffffu, c, j);
    c = (lane & j) ? (c < o ? c : o) : (c > o ? c : o);
  }
  return c;
}

// Row pass over one part of one logits row (Sec. 3.1, Sec. 3.2.1):
//   - the part's log-sum-exp as (m, s) with a per-thread online maximum;
//   - the part's exact top-K (K <= 32) under the order (logit desc, token id
//     asc), a 64-bit key (bf16 order code << 32 | ~token id) making keys
//     distinct and the order total.
// The stream does only the log-sum-exp and, per thread, notes the largest
// logit of every group of its vectors (two iterations, 64 logits: one
// shared-memory store).  Afterwards tau = the K-th largest of the threads'
// maxima: K distinct logits are >= tau, so every top-K logit is >= tau and
// lies in a group whose maximum is >= tau -- about K groups of the part.
// Those groups are read again (from L2), their keys >= (tau, largest id) go
// to the warp's buffer, which is cut back to its best K (by rank) when it
// fills, and the warps' lists are merged by rank.
// The needed-rows pass (kNeeded) reads only the rows that the verdict and the
// emitted positions need (Sec. 3.2.3: the tokens after a request's first
// state change are discarded; the loss sums over emitted tokens).  Its grid is (2 R, max span): block (r, i) takes
// the verifier's row of request r's span position i and block (R + r, i) the
// proposer's, so the blocks of position 0 of every request are dispatched
// first (the verifiers' rows before the proposers'), then position 1, and
// so on.  A verifier row whose token decides the verdict (not covered under a
// student-driven span, covered under a teacher-driven one) lowers the
// request's transition bound trans[r]; a block whose position lies past the
// bound it reads skips its row: the verifier's rows are needed up to the
// first transition, the proposer's at the emitted positions before it (and
// at it, for a handback).  The bound only ever falls towards the true first
// transition, so no needed row is skipped.
struct NeededRows {
  const int32_t *tokens, *cu_span;
  const uint8_t *driver;
  int *trans;  // [R] lowest transition position seen so far (starts high)
  int total_tokens;
};

template <bool kEntropy,  // also accumulate sum exp(l - m) l (entropies / entropy rules)
          bool kNeeded>   // the needed-rows pass (one part per row)
__global__ void __launch_bounds__(kRowThreads, kRowCtasPerSm) score_rows_kernel(
    const uint16_t *__restrict__ ls, const uint16_t *__restrict__ lt, int vocab, int K, int parts,
    RowOut *__restrict__ out, const NeededRows nr) {
  constexpr int U = 4;  // vectors per thread and iteration
  __shared__ uint16_t s_gmax[kMaxGroups][kRowThreads];  // group maxima (order codes, 0: none)
  __shared__ float s_sorted[kRowWarps][32];
  __shared__ float s_tau;
  static_assert(IPD_MAX_K == 32, "one key per lane");
  __shared__ unsigned long long s_lists[kRowWarps][32];
  __shared__ unsigned long long s_buf[kRowWarps][kBuf];
  __shared__ int s_cand[kRowWarps][32 * kMaxGroupVecs];  // a round's candidate vectors
  __shared__ float s_m[kRowWarps], s_s[kRowWarps], s_u[kRowWarps];

  int row_id = blockIdx.x / parts, part = blockIdx.x % parts, oi = blockIdx.x;
  int r = 0, pos = 0, drv = 0, ver = 0;
  if (kNeeded) {
    // blocks 0 .. R-1 of a position take the verifiers' rows, R .. 2R-1 the
    // proposers', so a proposer's row starts after its verifier's when the
    // position spans more than one wave
    const int R = gridDim.x >> 1;
    const bool is_ver = (int)blockIdx.x < R;
    r = is_ver ? blockIdx.x : blockIdx.x - R;
    pos = blockIdx.y;
    const int t0 = nr.cu_span[r], k = nr.cu_span[r + 1] - t0;
    // no such position (or offsets the epilogue reports as broken)
    if (pos >= k || t0 < 0 || t0 + k > nr.total_tokens) return;
    drv = nr.driver[r] ? 1 : 0;
    ver = drv ? 0 : 1;  // the verifier's row: the teacher's when the student drives
    row_id = 2 * (t0 + pos) + (is_ver ? ver : 1 - ver);
    part = 0;
    oi = row_id;
    const int tr = *reinterpret_cast<volatile const int *>(nr.trans + r);
    const bool need = (row_id & 1) == ver ? pos <= tr : (drv ? pos <= tr : pos < tr);
    if (!need) {
      if (threadIdx.x == 0) out[oi].skipped = 1;
      return;
    }
  }
  const int t = row_id >> 1, model = row_id & 1;
  const uint16_t *row = (model ? lt : ls) + (size_t)t * vocab;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, tid = threadIdx.x;
  const int nvec = vocab >> 3;
  const int per = (nvec + parts - 1) / parts;
  const int v_lo = min(nvec, part * per), v_hi = min(nvec, v_lo + per);
  const int n_iter = (v_hi - v_lo + kRowThreads * U - 1) / (kRowThreads * U);
  // iterations per group: two, or more so that a thread has at most kMaxGroups
  const int ipg = max(2, (n_iter + kMaxGroups - 1) / kMaxGroups);
  const int n_groups = (n_iter + ipg - 1) / ipg;
  unsigned long long *buf = s_buf[warp];

  float m = -INFINITY;
  unsigned long long s2 = 0ull;  // running sum of exp(l - m), as a packed pair
  unsigned long long u2 = 0ull;  // running sum of exp(l - m) * l, as a packed pair

  // ---- stream: log-sum-exp and group maxima ----
  // Each iteration takes four 16-byte vectors per thread and issues the loads
  // of the next iteration's four before it works on them, so eight loads per
  // thread are in flight.  Per 8 logits: the maximum on the packed bf16
  // words, then unpack, one fused multiply-add and one hardware 2^x each for
  // the sum.
  uint4 nxt[U];
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int v0 = v_lo + u * kRowThreads + tid;
    nxt[u] = make_uint4(0xff80ff80u, 0xff80ff80u, 0xff80ff80u, 0xff80ff80u);  // -inf
    if (v0 < v_hi) nxt[u] = ldg_stream(row + (size_t)v0 * 8);
  }
  float gmax = -INFINITY;
  for (int it = 0; it < n_iter; ++it) {
    const int base = v_lo + it * kRowThreads * U;
    uint4 raw[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      raw[u] = nxt[u];
      const int vn = base + (U + u) * kRowThreads + tid;
      nxt[u] = make_uint4(0xff80ff80u, 0xff80ff80u, 0xff80ff80u, 0xff80ff80u);  // -inf
      if (vn < v_hi) nxt[u] = ldg_stream(row + (size_t)vn * 8);
    }
    float vmx[U];
#pragma unroll
    for (int u = 0; u < U; ++u) vmx[u] = bf16x8_max(raw[u]);
    const float bmax = fmaxf(fmaxf(vmx[0], vmx[1]), fmaxf(vmx[2], vmx[3]));
    gmax = fmaxf(gmax, bmax);
    if (it % ipg == ipg - 1 || it == n_iter - 1) {
      // vectors past the part read as -inf; a group with none of the part's
      // vectors keeps code 0 (a real logit, -inf included, has a code >= 1)
      const bool real = v_lo + (it / ipg) * ipg * kRowThreads * U + tid < v_hi;
      s_gmax[it / ipg][tid] = real ? (uint16_t)ord16(__float_as_uint(gmax) >> 16) : (uint16_t)0;
      gmax = -INFINITY;
    }
    if (bmax > m) {
      const float f = ex2_approx((m - bmax) * kLog2e);
      float s0, s1, u0, u1;
      f2_unpack(s2, s0, s1);
      f2_unpack(u2, u0, u1);
      s2 = f2_pack(s0 * f, s1 * f);
      if (kEntropy) u2 = f2_pack(u0 * f, u1 * f);
      m = bmax;
    }
    if (m != -INFINITY) {
      // the two halves of each bf16 pair run as one packed fp32 pair
      const unsigned long long l2e = f2_pack(kLog2e, kLog2e);
      const unsigned long long ml = f2_pack(-m * kLog2e, -m * kLog2e);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t w[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float x0, x1;
          const unsigned long long ll = f2_pack(bf16lo(w[q]), bf16hi(w[q]));
          f2_unpack(f2_fma(ll, l2e, ml), x0, x1);
          const unsigned long long pp = f2_pack(ex2_approx(x0), ex2_approx(x1));
          s2 = f2_add(s2, pp);
          if (kEntropy) u2 = f2_fma(pp, ll, u2);
        }
      }
    }
  }

  // ---- tau: the K-th largest of the threads' maxima ----
  // A thread that read no logit of the part holds -inf and is not counted;
  // with fewer than K counted maxima every group of the part qualifies.
  {
    const bool real = v_lo + tid < v_hi;
    s_sorted[warp][lane] = warp_sort_desc_f(real ? m : -INFINITY, lane);
    __syncthreads();
    if (warp == 0) {  // the top 32 of the four sorted lists, then its K-th entry
      static_assert(kRowWarps == 4, "two rounds of pairwise merges");
      const float a = warp_top32_f(s_sorted[0][lane], s_sorted[1][lane], lane);
      const float b = warp_top32_f(s_sorted[2][lane], s_sorted[3][lane], lane);
      const float c = warp_top32_f(a, b, lane);
      if (lane == K - 1) s_tau = c;  // -inf when fewer than K logits were read
    }
    __syncthreads();
  }
  const float tau = s_tau;
  const uint32_t g_code = tau == -INFINITY ? 1u : ord16(__float_as_uint(tau) >> 16);

  // ---- examine the groups that reach tau ----
  // Keys > (tau, largest id) are the candidates: every logit >= tau.  A lane
  // loads four of a qualifying group's vectors at once, then the warp
  // examines them vector by vector.
  const unsigned long long th = tau == -INFINITY ? 0ull : (unsigned long long)g_code << 32;
  unsigned long long theta = 0ull;  // K-th best key this warp holds (0: fewer than K)
  int nb = 0;
  auto compact = [&]() {
    __syncwarp();
    const unsigned long long a = lane < nb ? buf[lane] : 0ull;
    const unsigned long long b = lane + 32 < nb ? buf[lane + 32] : 0ull;
    int ra = 0, rb = 0;
    for (int j = 0; j < nb; ++j) {
      const unsigned long long x = buf[j];
      ra += x > a;
      rb += x > b;
    }
    __syncwarp();
    if (lane < nb && ra < K) buf[ra] = a;
    if (lane + 32 < nb && rb < K) buf[rb] = b;
    __syncwarp();
    nb = nb < K ? nb : K;
    if (nb == K) theta = buf[K - 1];
  };
  // Rounds: every lane takes up to kMaxGroupVecs vectors of its next
  // qualifying group; the warp lists them (a prefix sum over lanes) and
  // examines the list one vector per lane, loading 32 at a time.  Usually a
  // single round.
  int j_next = 0, q_next = 0;  // this lane's next group, and next vector in it
  while (true) {
    while (j_next < n_groups && s_gmax[j_next][tid] < g_code) ++j_next;
    const bool have = j_next < n_groups;
    if (!__any_sync(0xffffffffu, have)) break;
    const int it0 = j_next * ipg;
    const int g_n = have ? (min(it0 + ipg, n_iter) - it0) * U : 0;  // the group's vectors
    const int n_lane = min(kMaxGroupVecs, g_n - q_next);
    int off = n_lane;  // inclusive prefix sum over lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, off, o);
      if (lane >= o) off += y;
    }
    const int total = __shfl_sync(0xffffffffu, off, 31);
    off -= n_lane;
    int *cand = s_cand[warp];
    for (int q = 0; q < n_lane; ++q) {
      const int qq = q_next + q;
      cand[off + q] = v_lo + (it0 + qq / U) * kRowThreads * U + (qq % U) * kRowThreads + tid;
    }
    __syncwarp();
    for (int b0 = 0; b0 < total; b0 += 32) {
      const int v = b0 + lane < total ? cand[b0 + lane] : -1;
      const bool ok = v >= 0 && v < v_hi;
      uint4 r = make_uint4(0xff80ff80u, 0xff80ff80u, 0xff80ff80u, 0xff80ff80u);  // -inf
      if (ok) r = __ldg(reinterpret_cast<const uint4 *>(row + (size_t)v * 8));
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const uint32_t bits = elem_bits(r, e);
        // a logit below tau's value cannot pass; the rest take the key test
        const bool maybe = ok && ord16(bits) >= g_code;
        if (__any_sync(0xffffffffu, maybe)) {
          const unsigned long long th_now = theta > th ? theta : th;
          const unsigned long long key = make_key(bits, (uint32_t)v * 8u + e);
          const bool c = maybe && key > th_now;
          const unsigned bal = __ballot_sync(0xffffffffu, c);
          if (bal) {
            if (nb + 32 > kBuf) compact();
            if (c) buf[nb + __popc(bal & ((1u << lane) - 1u))] = key;
            nb += __popc(bal);
          }
        }
      }
    }
    __syncwarp();
    if (have) {
      q_next += n_lane;
      if (q_next >= g_n) {
        ++j_next;
        q_next = 0;
      }
    }
  }
  if (nb > 0) compact();

  // block merge of the log-sum-exp (and of the entropy's weighted sum)
  float s, u;
  {
    float s0, s1, u0, u1;
    f2_unpack(s2, s0, s1);
    f2_unpack(u2, u0, u1);
    s = s0 + s1;
    u = u0 + u1;
  }
  float wm = warp_max(m);
  const float wf = (m == -INFINITY || wm == -INFINITY) ? 0.f : exp2f((m - wm) * kLog2e);
  float ws = warp_sum(s * wf);
  float wu = warp_sum(u * wf);
  s_lists[warp][lane] = lane < nb ? buf[lane] : 0ull;
  if (lane == 0) {
    s_m[warp] = wm;
    s_s[warp] = ws;
    s_u[warp] = wu;
  }
  __syncthreads();
  if (warp == 0) {
    float bm = lane < kRowWarps ? s_m[lane] : -INFINITY;
    const float gm = warp_max(bm);
    const float bf = (lane < kRowWarps && bm != -INFINITY) ? exp2f((bm - gm) * kLog2e) : 0.f;
    const float bs = warp_sum(lane < kRowWarps ? s_s[lane] * bf : 0.f);
    const float bu = warp_sum(lane < kRowWarps ? s_u[lane] * bf : 0.f);
    if (lane == 0) {
      out[oi].m = gm;
      out[oi].s = bs;
      out[oi].u = bu;
      if (kNeeded) out[oi].skipped = 0;
    }
    // the warps' lists (each sorted, 0 past its end) merged to the part's top K
    const unsigned long long a = warp_top32_u64(s_lists[0][lane], s_lists[1][lane], lane);
    const unsigned long long b = warp_top32_u64(s_lists[2][lane], s_lists[3][lane], lane);
    const unsigned long long c = warp_top32_u64(a, b, lane);
    out[oi].keys[lane] = lane < K ? c : 0ull;
    if (kNeeded && model == ver) {
      // coverage of the proposed token by this verifier row's Top_K
      const int x = nr.tokens[t];
      const bool hit = lane < K && x >= 0 && x < vocab && key_idx(c) == (uint32_t)x;
      const bool cov = __ballot_sync(0xffffffffu, hit) != 0;
      if (lane == 0 && (drv ? cov : !cov)) atomicMin(nr.trans + r, pos);
    }
  }
}

// Rules and optional outputs of the epilogue (ipd_score_ext on the device).
struct EpiOpts {
  int take_rule, hand_rule;
  float take_tau, hand_tau;
  float *entropy_s, *entropy_t, *topk_overlap;
  int32_t *topk_s, *topk_t;
};

__global__ void __launch_bounds__(kEpiThreads) score_epilogue_kernel(
    const uint16_t *__restrict__ ls, const uint16_t *__restrict__ lt,
    const int32_t *__restrict__ tokens, const int32_t *__restrict__ cu_span,
    const uint8_t *__restrict__ driver, const int32_t *__restrict__ prefix_len, int vocab, int K,
    int eos_id, const RowOut *__restrict__ rows, int parts, float *logp_s, float *logp_t,
    float *feedback,
    float *kl_rev, float *kl_fwd, uint8_t *covered, float *margin, uint8_t *source,
    int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver, int32_t *new_len, uint8_t *done,
    int total_tokens, const EpiOpts opt, int max_span = 0, bool needed_rows = false) {
  // No shared memory.  In a step that forks the vocabulary pass onto its
  // own stream, this kernel's CTAs take the SMs that the first attention
  // CTAs to finish leave free, so it runs inside the attention's tail.
  const int r = blockIdx.x;
  const int t0 = cu_span[r], t1 = cu_span[r + 1];
  const int drv = driver[r] ? 1 : 0;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (t0 < 0 || t1 < t0 || t1 > total_tokens) {
    if (threadIdx.x == 0) ipd_set_error(&g_score_err, IPD_DEVERR_SPAN);
    return;
  }
  const int k = t1 - t0;
  // a span longer than the bound a needed-rows call was given (max_span > 0)
  // would have been read only in part
  if (max_span > 0 && k > max_span) {
    if (threadIdx.x == 0) ipd_set_error(&g_score_err, IPD_DEVERR_SPAN);
    return;
  }

  for (int t = t0 + warp; t < t1; t += kEpiThreads / 32) {
    const int x = tokens[t];
    const bool xok = x >= 0 && x < vocab;
    if (!xok && lane == 0) ipd_set_error(&g_score_err, IPD_DEVERR_TOKEN);
    const uint16_t *rowS = ls + (size_t)t * vocab, *rowT = lt + (size_t)t * vocab;
    // each row's records, one per part: log Z = m + log s, the entropy
    // log Z - u / s, and the top-K keys, best first (lane j holds the j-th).
    // The parts' sums combine against their common maximum, and their
    // sorted key lists merge into the row's (the top K of the union of the
    // parts' top K is the row's top K).
    float logz[2], ent[2];
    unsigned long long key2[2];
#pragma unroll
    for (int mdl = 0; mdl < 2; ++mdl) {
      const RowOut *pr = rows + (size_t)(2 * t + mdl) * parts;
      float M = pr->m, S = pr->s, Uw = pr->u;
      unsigned long long kk = pr->keys[lane];  // 0 past the part's K keys
      for (int q = 1; q < parts; ++q) {
        const float mq = pr[q].m, sq = pr[q].s, uq = pr[q].u;
        const float mn = fmaxf(M, mq);
        if (mn != -INFINITY) {
          const float a = M == -INFINITY ? 0.f : exp2f((M - mn) * kLog2e);
          const float b = mq == -INFINITY ? 0.f : exp2f((mq - mn) * kLog2e);
          S = S * a + sq * b;
          Uw = Uw * a + uq * b;
          M = mn;
        }
        kk = warp_top32_u64(kk, pr[q].keys[lane], lane);
      }
      logz[mdl] = M + logf(S);
      ent[mdl] = logz[mdl] - Uw / S;  // H = log Z - E[l]
      key2[mdl] = lane < K ? kk : 0ull;
    }
    const float nan = __int_as_float(0x7fc00000);
    const float lxS = xok ? bf16f(rowS[x]) : nan, lxT = xok ? bf16f(rowT[x]) : nan;
    // union support S = Top_K(pi) u Top_K(q)
    unsigned long long kS = 0ull, kT = 0ull;
    uint32_t iS = 0, iT = 0;
    if (lane < K) {
      kS = key2[0];
      kT = key2[1];
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
    const unsigned long long kth = shfl_u64(kv, K - 1);
    // the predicate of the rule governing this span (Sec. 3.2.1)
    const int rule = drv ? opt.hand_rule : opt.take_rule;
    const float tau = drv ? opt.hand_tau : opt.take_tau;
    bool cov;
    float mar;
    if (rule == IPD_RULE_TOPK) {
      cov = __ballot_sync(0xffffffffu, hit) != 0;
      mar = (drv ? lxS : lxT) - key_val(kth);
    } else if (rule == IPD_RULE_ENTROPY_S || rule == IPD_RULE_ENTROPY_T) {
      const float h = rule == IPD_RULE_ENTROPY_S ? ent[0] : ent[1];
      cov = h <= tau;
      mar = tau - h;
    } else {
      cov = rule == IPD_RULE_ALWAYS;
      mar = cov ? INFINITY : -INFINITY;
    }
    if (lane < K) {
      if (opt.topk_s) opt.topk_s[(size_t)t * K + lane] = (int32_t)iS;
      if (opt.topk_t) opt.topk_t[(size_t)t * K + lane] = (int32_t)iT;
    }
    // |Top_K(pi) n Top_K(q)|: teacher keys also in the student's list
    const int n_common = __popc(__ballot_sync(0xffffffffu, lane < K && dupT));
    // a needed-rows pass leaves the rows past the transition unread: the
    // values that would come from them are NaN (coverage 0)
    const bool skip_s = needed_rows && rows[(size_t)2 * t * parts].skipped;
    const bool skip_t = needed_rows && rows[(size_t)(2 * t + 1) * parts].skipped;
    const bool skip_ver = drv ? skip_s : skip_t;
    if (lane == 0) {
      const float lps = lxS - logz[0], lpt = lxT - logz[1];
      const bool both = !skip_s && !skip_t;
      logp_s[t] = both ? lps : nan;
      logp_t[t] = both ? lpt : nan;
      feedback[t] = both ? lpt - lps : nan;
      kl_rev[t] = both ? kr : nan;
      kl_fwd[t] = both ? kf : nan;
      covered[t] = cov && !skip_ver ? 1 : 0;
      margin[t] = skip_ver ? nan : mar;
      if (opt.entropy_s) opt.entropy_s[t] = ent[0];
      if (opt.entropy_t) opt.entropy_t[t] = ent[1];
      if (opt.topk_overlap) opt.topk_overlap[t] = (float)n_common / (float)K;
    }
  }
  __syncthreads();  // the block's writes of `covered` are visible to thread 0
  if (threadIdx.x == 0) {
    // Eq. (ipd_state_transition) applied position by position until the first
    // state change or an accepted EOS; rollback rules of the verdict stage.
    int n = 0, ft = k, nd = drv, dn = 0;
    for (int i = 0; i < k; ++i) {
      const int c = covered[t0 + i];
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

extern "C" __attribute__((visibility("hidden"))) size_t ipd_internal_sample_ws(int n_rows,
                                                                              int vocab);
extern "C" __attribute__((visibility("hidden"))) int ipd_internal_sample_after_verdict(
    const uint16_t *ls, const uint16_t *lt, int num_reqs, int total_tokens, int vocab,
    uint64_t seed, const uint64_t *draw_base, float inv_temperature, const int32_t *cu_span,
    const int32_t *prefix_len, const int32_t *n_emit, const uint8_t *next_driver,
    const uint8_t *done, int32_t *next_token, void *ws, cudaStream_t st);

namespace {
// workspace: the row records (room for kMaxParts per row), then (256-byte
// aligned) the sampler's partials
size_t rows_region(int total_tokens) {
  return ((size_t)total_tokens * 2 * kMaxParts * sizeof(RowOut) + 255) & ~(size_t)255;
}

int g_sms[64] = {};  // SM count per device, read once

// Parts per logits row: as many (up to kMaxParts) as keep every row CTA of
// the call in one wave, so a pass over few rows is not held to one CTA's
// streaming rate per row.  A part keeps at least four loads per thread.
int row_parts(int total_tokens, int vocab, int max_parts) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  if (!g_sms[dev] &&
      cudaDeviceGetAttribute(&g_sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 1;
  const long long slots = (long long)kRowCtasPerSm * g_sms[dev];
  for (int q = max_parts; q > 1; q >>= 1)
    if (2LL * total_tokens * q <= slots && vocab / 8 / q >= kRowThreads * 4) return q;
  return 1;
}

// the needed-rows pass's transition bounds, after the row records and the
// sampler's partials
size_t trans_offset(int num_reqs, int total_tokens, int vocab) {
  return (rows_region(total_tokens) + ipd_internal_sample_ws(num_reqs, vocab) + 255) &
         ~(size_t)255;
}
}  // namespace

extern "C" size_t ipd_score_workspace_size(int num_reqs, int total_tokens, int vocab, int K) {
  if (num_reqs < 0 || total_tokens < 0 || vocab < 1 || K < 1) return 0;
  return trans_offset(num_reqs, total_tokens, vocab) + (size_t)num_reqs * sizeof(int) + 256;
}

namespace {
// host form of the options; false on an invalid rule or threshold
bool epi_opts(const ipd_score_ext *ext, EpiOpts *o) {
  *o = EpiOpts{IPD_RULE_TOPK, IPD_RULE_TOPK, 0.f, 0.f, nullptr, nullptr, nullptr, nullptr,
               nullptr};
  if (!ext) return true;
  auto ok_rule = [](int r) { return r >= IPD_RULE_TOPK && r <= IPD_RULE_NEVER; };
  if (!ok_rule(ext->takeover_rule) || !ok_rule(ext->handback_rule)) return false;
  if (ext->takeover_tau != ext->takeover_tau || ext->handback_tau != ext->handback_tau)
    return false;
  *o = EpiOpts{ext->takeover_rule, ext->handback_rule, ext->takeover_tau, ext->handback_tau,
               ext->entropy_s, ext->entropy_t, ext->topk_overlap, ext->topk_s, ext->topk_t};
  if (ext->next_token && !(ext->inv_temperature > 0.f &&
                           ext->inv_temperature - ext->inv_temperature == 0.f))
    return false;  // the draw needs a positive, finite inverse temperature
  return true;
}
}  // namespace

extern "C" int ipd_score_span_ex(const uint16_t *logits_student, const uint16_t *logits_teacher,
                                 const int32_t *tokens, const int32_t *cu_span,
                                 const uint8_t *driver, const int32_t *prefix_len, int num_reqs,
                                 int total_tokens, int vocab, int K, int eos_id, float *logp_s,
                                 float *logp_t, float *feedback, float *kl_rev, float *kl_fwd,
                                 uint8_t *covered, float *margin, uint8_t *source,
                                 int32_t *first_trans, int32_t *n_emit, uint8_t *next_driver,
                                 int32_t *new_len, uint8_t *done, const ipd_score_ext *ext,
                                 void *workspace, size_t workspace_bytes, ipd_stream_t stream) {
  if (num_reqs < 0 || total_tokens < 0) return IPD_ERR_INVALID_ARG;
  if (K < 1 || K > IPD_MAX_K) return IPD_ERR_UNSUPPORTED;
  if (vocab < 8 || vocab % 8 || K > vocab) return IPD_ERR_UNSUPPORTED;
  EpiOpts opt;
  if (!epi_opts(ext, &opt)) return IPD_ERR_INVALID_ARG;
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
  const int parts = row_parts(total_tokens, vocab, kMaxParts);
  if (total_tokens > 0) {
    const bool need_h = opt.entropy_s || opt.entropy_t || opt.take_rule == IPD_RULE_ENTROPY_S ||
                        opt.take_rule == IPD_RULE_ENTROPY_T || opt.hand_rule == IPD_RULE_ENTROPY_S ||
                        opt.hand_rule == IPD_RULE_ENTROPY_T;
    if (need_h)
      score_rows_kernel<true, false><<<2 * parts * total_tokens, kRowThreads, 0, st>>>(
          logits_student, logits_teacher, vocab, K, parts, rows, NeededRows{});
    else
      score_rows_kernel<false, false><<<2 * parts * total_tokens, kRowThreads, 0, st>>>(
          logits_student, logits_teacher, vocab, K, parts, rows, NeededRows{});
    if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  }
  score_epilogue_kernel<<<num_reqs, kEpiThreads, 0, st>>>(
      logits_student, logits_teacher, tokens, cu_span, driver, prefix_len, vocab, K, eos_id, rows,
      parts, logp_s, logp_t, feedback, kl_rev, kl_fwd, covered, margin, source, first_trans,
      n_emit, next_driver, new_len, done, total_tokens, opt);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  if (ext && ext->next_token)
    return ipd_internal_sample_after_verdict(
        logits_student, logits_teacher, num_reqs, total_tokens, vocab, ext->sample_seed,
        ext->draw_base, ext->inv_temperature, cu_span, prefix_len, n_emit, next_driver, done,
        ext->next_token, static_cast<char *>(workspace) + rows_region(total_tokens), st);
  return IPD_OK;
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
  return ipd_score_span_ex(logits_student, logits_teacher, tokens, cu_span, driver, prefix_len,
                           num_reqs, total_tokens, vocab, K, eos_id, logp_s, logp_t, feedback,
                           kl_rev, kl_fwd, covered, margin, source, first_trans, n_emit,
                           next_driver, new_len, done, nullptr, workspace, workspace_bytes,
                           stream);
}

extern "C" int ipd_score_span_needed(const uint16_t *logits_student,
                                     const uint16_t *logits_teacher, const int32_t *tokens,
                                     const int32_t *cu_span, const uint8_t *driver,
                                     const int32_t *prefix_len, int num_reqs, int total_tokens,
                                     int vocab, int K, int eos_id, int max_span, float *logp_s,
                                     float *logp_t, float *feedback, float *kl_rev,
                                     float *kl_fwd, uint8_t *covered, float *margin,
                                     uint8_t *source, int32_t *first_trans, int32_t *n_emit,
                                     uint8_t *next_driver, int32_t *new_len, uint8_t *done,
                                     void *workspace, size_t workspace_bytes,
                                     ipd_stream_t stream) {
  if (num_reqs < 0 || total_tokens < 0) return IPD_ERR_INVALID_ARG;
  if (K < 1 || K > IPD_MAX_K) return IPD_ERR_UNSUPPORTED;
  if (vocab < 8 || vocab % 8 || K > vocab) return IPD_ERR_UNSUPPORTED;
  if (num_reqs == 0) return IPD_OK;
  if (max_span < 1 || max_span > 65535) return IPD_ERR_INVALID_ARG;
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
  int *trans = reinterpret_cast<int *>(static_cast<char *>(workspace) +
                                       trans_offset(num_reqs, total_tokens, vocab));
  // When every row CTA fits one wave, every row starts before any transition
  // is known: the full pass (rows in up to four parts) is then as fast or
  // faster, and defines every position.
  const int parts = row_parts(total_tokens, vocab, kMaxParts);
  int dev = 0;
  const bool one_wave = cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64 &&
                        g_sms[dev] > 0 &&
                        2LL * total_tokens <= (long long)kRowCtasPerSm * g_sms[dev];
  if (one_wave) {
    if (total_tokens > 0) {
      score_rows_kernel<false, false><<<2 * parts * total_tokens, kRowThreads, 0, st>>>(
          logits_student, logits_teacher, vocab, K, parts, rows, NeededRows{});
      if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
    }
    score_epilogue_kernel<<<num_reqs, kEpiThreads, 0, st>>>(
        logits_student, logits_teacher, tokens, cu_span, driver, prefix_len, vocab, K, eos_id,
        rows, parts, logp_s, logp_t, feedback, kl_rev, kl_fwd, covered, margin, source,
        first_trans, n_emit, next_driver, new_len, done, total_tokens,
        EpiOpts{IPD_RULE_TOPK, IPD_RULE_TOPK, 0.f, 0.f, nullptr, nullptr, nullptr, nullptr,
                nullptr},
        max_span, false);
    return cudaGetLastError() == cudaSuccess ? IPD_OK : IPD_ERR_CUDA;
  }
  if (total_tokens > 0) {
    // every bound starts above any position (0x7f7f7f7f)
    if (cudaMemsetAsync(trans, 0x7f, (size_t)num_reqs * sizeof(int), st) != cudaSuccess)
      return IPD_ERR_CUDA;
    score_rows_kernel<false, true><<<dim3(2 * num_reqs, max_span), kRowThreads, 0, st>>>(
        logits_student, logits_teacher, vocab, K, 1, rows,
        NeededRows{tokens, cu_span, driver, trans, total_tokens});
    if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  }
  score_epilogue_kernel<<<num_reqs, kEpiThreads, 0, st>>>(
      logits_student, logits_teacher, tokens, cu_span, driver, prefix_len, vocab, K, eos_id, rows,
      1, logp_s, logp_t, feedback, kl_rev, kl_fwd, covered, margin, source, first_trans, n_emit,
      next_driver, new_len, done, total_tokens,
      EpiOpts{IPD_RULE_TOPK, IPD_RULE_TOPK, 0.f, 0.f, nullptr, nullptr, nullptr, nullptr, nullptr},
      max_span, true);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}

// ---------------------------------------------------------------------------
// Full-vocabulary KL (Eq. full_vocab_opd), both directions, reading the
// student's and the teacher's row of a span position together.  Per thread
// and row: a running maximum m, s = sum exp(l - m); per thread: a = sum
// exp(l_s - m_s) (l_s - l_t) and b = sum exp(l_t - m_t) (l_t - l_s), each
// rescaled with its row's maximum.  Then KL(pi || q) = a / s_s - log Z_s +
// log Z_t and KL(q || pi) = b / s_t - log Z_t + log Z_s.
// A position is one cluster of P CTAs (P = 1, 2 or 4), CTA r taking part r
// of both rows; the parts' six sums meet in CTA 0's shared memory (the
// cluster's distributed shared memory), so a call over few positions still
// fills the GPU in one wave without a scratch buffer or a second launch.
// ---------------------------------------------------------------------------
namespace {
constexpr int kKlThreads = 256;
constexpr int kKlCtasPerSm = 4;  // the kernel's launch bounds

template <int P>
__global__ void __launch_bounds__(kKlThreads, kKlCtasPerSm) full_kl_kernel(
    const uint16_t *__restrict__ ls, const uint16_t *__restrict__ lt, int vocab,
    float *__restrict__ kl_rev, float *__restrict__ kl_fwd) {
  __shared__ float sh[kKlThreads / 32][6];
  __shared__ float s_part[6];  // this CTA's part: ms, s_s, a, mt, s_t, -b
  const int t = blockIdx.x / P, part = blockIdx.x % P;  // part = rank in the cluster
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint4 *rs = reinterpret_cast<const uint4 *>(ls + (size_t)t * vocab);
  const uint4 *rt = reinterpret_cast<const uint4 *>(lt + (size_t)t * vocab);
  const int nvec_all = vocab >> 3;
  const int per = (nvec_all + P - 1) / P;
  const int v_lo = min(nvec_all, part * per), nvec = min(nvec_all, v_lo + per);
  float ms = -INFINITY, mt = -INFINITY;
  unsigned long long ss = 0ull, st = 0ull, aa = 0ull, bb = 0ull;  // packed pairs
  const unsigned long long l2e = f2_pack(kLog2e, kLog2e);
  constexpr int U = 2;
  for (int base = v_lo; base < nvec; base += kKlThreads * U) {
    uint4 xs[U], xt[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int v = base + u * kKlThreads + (int)threadIdx.x;
      ok[u] = v < nvec;
      xs[u] = ok[u] ? ldg_stream(rs + v) : make_uint4(0xff80ff80u, 0xff80ff80u, 0xff80ff80u, 0xff80ff80u);
      xt[u] = ok[u] ? ldg_stream(rt + v) : make_uint4(0xff80ff80u, 0xff80ff80u, 0xff80ff80u, 0xff80ff80u);
    }
    float bs = -INFINITY, bt = -INFINITY;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      bs = fmaxf(bs, bf16x8_max(xs[u]));
      bt = fmaxf(bt, bf16x8_max(xt[u]));
    }
    if (bs > ms) {  // rescale the student-weighted sums
      const float f = ex2_approx((ms - bs) * kLog2e);
      const unsigned long long ff = f2_pack(f, f), z = 0ull;
      ss = f2_fma(ss, ff, z);
      aa = f2_fma(aa, ff, z);
      ms = bs;
    }
    if (bt > mt) {
      const float f = ex2_approx((mt - bt) * kLog2e);
      const unsigned long long ff = f2_pack(f, f), z = 0ull;
      st = f2_fma(st, ff, z);
      bb = f2_fma(bb, ff, z);
      mt = bt;
    }
    const unsigned long long mls = f2_pack(-ms * kLog2e, -ms * kLog2e);
    const unsigned long long mlt = f2_pack(-mt * kLog2e, -mt * kLog2e);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (!ok[u]) continue;
      const uint32_t ws[4] = {xs[u].x, xs[u].y, xs[u].z, xs[u].w};
      const uint32_t wt[4] = {xt[u].x, xt[u].y, xt[u].z, xt[u].w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const unsigned long long vs = f2_pack(bf16lo(ws[q]), bf16hi(ws[q]));
        const unsigned long long vt = f2_pack(bf16lo(wt[q]), bf16hi(wt[q]));
        float e0, e1, g0, g1;
        f2_unpack(f2_fma(vs, l2e, mls), e0, e1);
        f2_unpack(f2_fma(vt, l2e, mlt), g0, g1);
        const unsigned long long p = f2_pack(ex2_approx(e0), ex2_approx(e1));
        const unsigned long long qq = f2_pack(ex2_approx(g0), ex2_approx(g1));
        const unsigned long long d = f2_sub(vs, vt);  // l_s - l_t
        ss = f2_add(ss, p);
        st = f2_add(st, qq);
        aa = f2_fma(p, d, aa);
        bb = f2_fma(qq, d, bb);  // sum q (l_s - l_t) = -b
      }
    }
  }
  float v[6];  // ms, s_s, a, mt, s_t, -b (per thread)
  {
    float x0, x1;
    v[0] = ms;
    f2_unpack(ss, x0, x1); v[1] = x0 + x1;
    f2_unpack(aa, x0, x1); v[2] = x0 + x1;
    v[3] = mt;
    f2_unpack(st, x0, x1); v[4] = x0 + x1;
    f2_unpack(bb, x0, x1); v[5] = x0 + x1;
  }
  // warp then block merge: rescale each thread's sums to the common maxima
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const float M = warp_max(v[3 * r]);
    const float f = (v[3 * r] == -INFINITY) ? 0.f : exp2f((v[3 * r] - M) * kLog2e);
    v[3 * r] = M;
    v[3 * r + 1] = warp_sum(v[3 * r + 1] * f);
    v[3 * r + 2] = warp_sum(v[3 * r + 2] * f);
  }
  if (lane == 0)
#pragma unroll
    for (int i = 0; i < 6; ++i) sh[warp][i] = v[i];
  __syncthreads();
  if (warp == 0) {
    float w[6];
#pragma unroll
    for (int i = 0; i < 6; ++i) w[i] = lane < kKlThreads / 32 ? sh[lane][i] : (i % 3 == 0 ? -INFINITY : 0.f);
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const float M = warp_max(w[3 * r]);
      const float f = (w[3 * r] == -INFINITY) ? 0.f : exp2f((w[3 * r] - M) * kLog2e);
      w[3 * r] = M;
      w[3 * r + 1] = warp_sum(w[3 * r + 1] * f);
      w[3 * r + 2] = warp_sum(w[3 * r + 2] * f);
    }
    if (P == 1) {
      if (lane == 0) {
        const float lzs = w[0] + logf(w[1]), lzt = w[3] + logf(w[4]);
        kl_rev[t] = w[2] / w[1] - lzs + lzt;
        kl_fwd[t] = -w[5] / w[4] - lzt + lzs;
      }
    } else if (lane == 0) {
#pragma unroll
      for (int i = 0; i < 6; ++i) s_part[i] = w[i];
    }
  }
  if constexpr (P > 1) {
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    cluster.sync();  // every part's sums are in its CTA's shared memory
    if (part == 0 && warp == 0) {
      // lane q < P holds part q's sums; then the same max-rescaled merge
      float w[6];
      const float *src = lane < P ? cluster.map_shared_rank(s_part, lane) : nullptr;
#pragma unroll
      for (int i = 0; i < 6; ++i) w[i] = src ? src[i] : (i % 3 == 0 ? -INFINITY : 0.f);
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const float M = warp_max(w[3 * r]);
        const float f = (w[3 * r] == -INFINITY) ? 0.f : exp2f((w[3 * r] - M) * kLog2e);
        w[3 * r] = M;
        w[3 * r + 1] = warp_sum(w[3 * r + 1] * f);
        w[3 * r + 2] = warp_sum(w[3 * r + 2] * f);
      }
      if (lane == 0) {
        const float lzs = w[0] + logf(w[1]), lzt = w[3] + logf(w[4]);
        kl_rev[t] = w[2] / w[1] - lzs + lzt;
        kl_fwd[t] = -w[5] / w[4] - lzt + lzs;
      }
    }
    cluster.sync();  // CTA 0 has read every part before any CTA exits
  }
}

int g_kl_sms[64] = {};  // SM count per device, read once

template <int P>
cudaError_t launch_full_kl(const uint16_t *ls, const uint16_t *lt, int T, int vocab, float *rev,
                           float *fwd, cudaStream_t st) {
  if (P == 1) {
    full_kl_kernel<1><<<T, kKlThreads, 0, st>>>(ls, lt, vocab, rev, fwd);
    return cudaGetLastError();
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)T * P);
  cfg.blockDim = dim3(kKlThreads);
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = P;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, full_kl_kernel<P>, ls, lt, vocab, rev, fwd);
}
}  // namespace

extern "C" int ipd_full_kl(const uint16_t *logits_student, const uint16_t *logits_teacher,
                           int total_tokens, int vocab, float *kl_rev_full, float *kl_fwd_full,
                           ipd_stream_t stream) {
  if (total_tokens < 0) return IPD_ERR_INVALID_ARG;
  if (vocab < 8 || vocab % 8) return IPD_ERR_UNSUPPORTED;
  if (total_tokens == 0) return IPD_OK;
  if (!logits_student || !logits_teacher || !kl_rev_full || !kl_fwd_full)
    return IPD_ERR_INVALID_ARG;
  if (((uintptr_t)logits_student | (uintptr_t)logits_teacher) & 15) return IPD_ERR_INVALID_ARG;
  // parts per position: as many as keep every CTA of the call in one wave,
  // with at least two loads per thread and row in a part
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return IPD_ERR_CUDA;
  if (!g_kl_sms[dev] &&
      cudaDeviceGetAttribute(&g_kl_sms[dev], cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return IPD_ERR_CUDA;
  const long long slots = (long long)kKlCtasPerSm * g_kl_sms[dev];
  int P = 1;
  for (int q = 4; q > 1; q >>= 1)
    if ((long long)total_tokens * q <= slots && vocab / 8 / q >= kKlThreads * 2) {
      P = q;
      break;
    }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const cudaError_t e =
      P == 4 ? launch_full_kl<4>(logits_student, logits_teacher, total_tokens, vocab, kl_rev_full,
                                 kl_fwd_full, st)
      : P == 2 ? launch_full_kl<2>(logits_student, logits_teacher, total_tokens, vocab,
                                   kl_rev_full, kl_fwd_full, st)
               : launch_full_kl<1>(logits_student, logits_teacher, total_tokens, vocab,
                                   kl_rev_full, kl_fwd_full, st);
  if (e != cudaSuccess || cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
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
  // call first, so nothing in the array has to start at zero.  The array
  // holds 2 IPD_STATIC_MAX_TOKENS records: parts * total_tokens stays within.
  const int parts = row_parts(
      total_tokens, vocab,
      total_tokens > 0 ? std::min(kMaxParts, IPD_STATIC_MAX_TOKENS / total_tokens) : 1);
  if (total_tokens > 0) {
    score_rows_kernel<false, false><<<2 * parts * total_tokens, kRowThreads, 0, s>>>(
        logits_student, logits_teacher, vocab, K, parts, rows, NeededRows{});
    if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  }
  score_epilogue_kernel<<<num_reqs, kEpiThreads, 0, s>>>(
      logits_student, logits_teacher, tokens, cu_span, driver, prefix_len, vocab, K, eos_id, rows,
      parts, logp_s, logp_t, feedback, kl_rev, kl_fwd, covered, margin, source, first_trans,
      n_emit, next_driver, new_len, done, total_tokens,
      EpiOpts{IPD_RULE_TOPK, IPD_RULE_TOPK, 0.f, 0.f, nullptr, nullptr, nullptr});
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}
