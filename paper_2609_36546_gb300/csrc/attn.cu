// Paged span-verify attention and proposer decode attention, co-launched.
//
// Sec. 3.2.3 (verification stage): each verifier evaluates the k_r unverified
// draft tokens of a request in one prefill pass over its own cache; only the
// new tokens are computed (their K/V are already in the cache).  Proposal
// stage: the proposer decodes one token over its own cache.  Both run here as
// one persistent launch over both caches, whose GQA shapes differ.
//
// Work decomposition (device side, no host round trip):
//   task  = (batch, request, kv head, row block); a row is one (span query,
//           query head) pair, row = i * G + j for query i and head kvh*G + j.
//   item  = (task, KV chunk); tasks longer than about a quarter of an SM's
//           share are split, items are claimed longest first, and the CTA
//           that finishes a split task's last item merges its partials.
// KV pages stream through a 3-stage ring of 128-key stages (64 KB), one
// 4 KB 4-D TMA box per page and tensor.
// Two compute paths, chosen per task by its row count:
//   tensor path (rows >= kTcMinRows): a 128-lane tile.  S = Q K^T (Q from
//     TMEM, K from shared memory, N = 128 keys) and P V run on tcgen05 with
//     fp32 accumulators in TMEM.  P is passed as three bf16 terms (its upper
//     16 bits, the truncated residual and what is left of it, rounded), so
//     P V sees each probability to within 2^-25 of itself.  Each chunk's P V
//     starts a fresh accumulator, and the chunks are summed in fp32
//     registers with round-to-nearest adds: the tensor core's own
//     accumulation does not round to nearest, and summed over a whole long
//     context its error reaches several bf16 ulp of the result.
//     All eight compute warps work on a tile, two threads per TMEM lane, each
//     taking part of a chunk's keys and half of the output dimensions.  A
//     tile of at most 32 (64) rows is repeated 4 (2) times over the lanes,
//     the copies splitting each chunk's keys, and its P terms are stacked in
//     the 128 rows of one shared-memory operand (three terms of 32 rows, or
//     two of 64 with the third in TMEM), so P V costs 8 (16) MMAs per chunk
//     instead of 24: those tiles would otherwise be bound by the tensor pipe.
//     S is double-buffered, so the softmax of chunk j overlaps Q K^T of j+1
//     and P V of j-1.
//   CUDA-core path (fewer rows: the GQA-2 decode and one-token spans, two
//     rows): fp32 FMA on the first four compute warps, two pages of 16 keys
//     per warp and stage, two lanes per key.  From four rows up the tensor
//     path is faster even with most of its tile empty: at 4-6 rows the
//     CUDA-core FMAs limit the stream.
// Warp roles: warps 0-7 compute, warp 8 streams the K pages of each stage and
// warp 11 its V pages, warp 9 issues Q K^T and warp 10 P V.  One thread issuing
// a burst of MMAs stalls about 100 cycles per instruction, more than an MMA
// takes to run, so the two products of a chunk are issued by two warps; a
// warp issuing a stage's 16 TMA boxes took about 2000 cycles, two thirds of
// the stage's time at the HBM rate, so K and V boxes come from two warps.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>

#include "common.cuh"

IPD_DECLARE_ERROR_WORD(g_attn_err);

namespace {

constexpr int kPage = 16;
constexpr int kD = 128;
constexpr int kStagePages = 8;                    // 128 keys per stage
constexpr int kStageKeys = kStagePages * kPage;
constexpr int kStages = 3;
// A stage holds the K pages then the V pages.  One page (16 keys x 128 dims
// of one kv head) is one 4 KB TMA box laid out as two 8-key groups of 2 KB,
// each group as its 64-dim halves, each half one 128-byte-swizzled 1 KB atom
// (8 rows x 128 B).  Key row R, half h of a tensor sits at
// (R / 8) * 2048 + h * 1024 + (R % 8) * 128: a K-major operand with 8-row
// groups 2048 B apart, or an MN-major one with halves 1024 B apart.
constexpr int kPageBytes = kPage * kD * 2;        // 4 KB
constexpr int kGroupBytes = 2048;                 // 8 keys, both halves
constexpr int kAtomBytes = 1024;                  // 8 keys, one 64-dim half
constexpr int kTensorBytes = kStagePages * kPageBytes;  // 32 KB of K (or V) per stage
constexpr int kStageBytes = 2 * kTensorBytes;     // 64 KB
constexpr int kTcRows = 128;                      // TMEM lanes of a tensor-core tile (M)
// Tasks with at least this many rows use the tensor path.  The library is
// built with 4; the build accepts another value (IPD_TC_MIN_ROWS) only to
// measure the crossover between the two paths.
#ifndef IPD_TC_MIN_ROWS
#define IPD_TC_MIN_ROWS 4
#endif
constexpr int kTcMinRows = IPD_TC_MIN_ROWS;
static_assert(kTcMinRows >= 3 && kTcMinRows <= 8, "CUDA-core tasks have 2 to 7 rows");
constexpr int kCcRows = kTcMinRows - 1;           // CUDA-core tasks have fewer rows
constexpr int kCW = 8;                            // compute warps (two per TMEM lane block)
constexpr int kCcW = 4;                           // of them, the CUDA-core path's warps
constexpr int kProducerWarp = kCW;
constexpr int kMmaWarp = kCW + 1;                 // issues Q K^T (and owns the TMEM allocation)
constexpr int kPvWarp = kCW + 2;                  // issues P V
constexpr int kVLoadWarp = kCW + 3;               // issues the V boxes of each stage
constexpr int kThreads = (kCW + 4) * 32;           // three warpgroups; warps 10 and 11 exit early
// Register split: the block is launched with 168 registers a thread (three
// warps share each SM sub-partition's 16K registers); the third warpgroup
// (producer, MMA issuer and two idle warps) gives registers back so that the
// compute warpgroups can hold their per-lane output sums.
constexpr int kRegsLaunch = 168, kRegsAux = 56, kRegsCompute = 224;
static_assert(2 * 128 * kRegsCompute + 128 * kRegsAux <= kThreads * kRegsLaunch,
              "the register split must fit the registers the block was launched with");
constexpr int kTargetItemsPerSm = 4;               // items of about a quarter of an SM's share
constexpr int kSizesPerBatch = 32;                // claim order: batch by batch, and within a
constexpr int kSizeBuckets = IPD_MAX_BATCHES * kSizesPerBatch;  // batch the longest items first
static_assert(kSizeBuckets % 32 == 0, "bucket prefix: whole lanes");
constexpr int kMaxTargetItems = 4096;            // bound used for workspace sizing
constexpr int kMinChunkPages = 16;
constexpr int kSplitMax = 16;
constexpr int kPStride = 132;                     // floats per partial row: o[128], m, l, pad
constexpr uint32_t kTmemCols = 512;
// TMEM columns: the S double buffer at 0 and 128 (fp32, one column per key)
// and the O product of one chunk at 256.  Columns 384..511 hold, for tiles of
// up to 64 rows, the Q tile at 384 (64 columns of bf16 pairs) and the third
// term of P at 448 (64 columns of bf16 pairs; one buffer, written only after
// the previous chunk's P V has completed); for 128-row tiles, whose Q tile
// sits in shared memory, the third term of P at 384 + 64 b for S buffer b.
// In 128-row tiles a consumed S buffer is overwritten with the first two
// terms of P as bf16 pairs: for keys 16kk .. 16kk + 15, columns 16kk ..
// 16kk + 7 hold the first and 16kk + 8 .. 16kk + 15 the second (p_col), in
// place of the S values of the same keys, so that each thread writes only
// columns it has itself just read.
__device__ __forceinline__ uint32_t col_s(uint32_t b) { return b * 128u; }
constexpr uint32_t kColO = 256;
constexpr uint32_t kColQ = 384;
constexpr uint32_t kColT3 = 448;
// column (relative to an S buffer) of keys 16 kk .. 16 kk + 15 of term 1 or
// term 2 of P
__host__ __device__ constexpr uint32_t p_col(int kk, int term) {
  return 16u * (uint32_t)kk + 8u * (uint32_t)(term - 1);
}
// column of keys 16 kk .. 16 kk + 15 of the third term of P (tiles of up to
// 64 rows), and for S buffer b of a 128-row tile
__host__ __device__ constexpr uint32_t t3_col(int kk) { return kColT3 + 8u * (uint32_t)kk; }
__host__ __device__ constexpr uint32_t t3_col_full(uint32_t b, int kk) {
  return kColQ + 64u * b + 8u * (uint32_t)kk;
}
// item paths: CUDA cores, or a tensor tile repeated 4, 2 or 1 times over the
// 128 TMEM lanes (at most 32, at most 64, or up to 128 rows)
constexpr int kPathCc = 0, kPathTc4 = 1, kPathTc2 = 2, kPathTc1 = 3;
__host__ __device__ constexpr int tc_path(int rows) {
  return rows <= kTcRows / 4 ? kPathTc4 : rows <= kTcRows / 2 ? kPathTc2 : kPathTc1;
}

struct BatchDev {
  const uint16_t *q;
  uint16_t *out;
  const int *cu_q;
  const int *seq_len;
  const int *page_table;
  long long num_pages;
  int num_reqs, hq, hkv, group, max_pages, max_q_len, total_q, cache;
};

struct __align__(16) Item {
  int b, r, kvh, rb;
  int split, n_split, page_lo, page_hi;
  int task, pbase, rows, path;  // path: kPathCc or kPathTc4 / 2 / 1
};
static_assert(sizeof(Item) == 48, "items are written as three 16-byte vectors");

struct AttnParams {
  CUtensorMap tmap[2 * IPD_MAX_BATCHES];  // K and V map of every distinct cache
  BatchDev b[IPD_MAX_BATCHES];
  int req_base[IPD_MAX_BATCHES + 1];
  int n_batches;
  int total_reqs;
  float scale_log2;
  int *ctrl;       // [0] n_items, [1] dynamic item counter, [2] n_tasks, [3] partial rows,
                   // [4] 1 if some task is split (claim the next item late)
  int4 *reqinfo;   // per flattened request: (unused), task offset, partial offset, n_split
  Item *items;
  int *split_done; // per task: split items finished (the planner zeroes those of split tasks)
  int2 *reqslot;   // per flattened request: slot offsets of its full-size and last splits
  float *partials;
  int item_cap, task_cap;
  long long prow_cap;
  int target_items;  // work-list size the planner aims for (a multiple of the SM count)
  int n_sms;
};

struct StageMeta {
  int item;
  int page0;
  int npages;
  int flags;        // 1 = first stage of its item, 2 = last stage
  uint32_t invalid; // pages of the stage whose id failed validation
  int path;
  int pad[2];
};

// --------------------------------------------------------------------------
// host-side sizes
// --------------------------------------------------------------------------
struct WsLayout {
  size_t off_ctrl, off_reqinfo, off_reqslot, off_items, off_done, off_partials, total;
  int item_cap, task_cap, total_reqs;
  long long prow_cap;
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int validate_batch(const ipd_attn_batch *b) {
  if (!b || !b->cache) return IPD_ERR_INVALID_ARG;
  const ipd_kv_cache *c = b->cache;
  if (c->page_size != kPage || c->head_dim != kD) return IPD_ERR_UNSUPPORTED;
  if (c->num_kv_heads < 1 || c->num_kv_heads > 64) return IPD_ERR_UNSUPPORTED;
  if (b->num_q_heads < 1 || b->num_q_heads % c->num_kv_heads) return IPD_ERR_INVALID_ARG;
  if (b->num_q_heads / c->num_kv_heads > kTcRows) return IPD_ERR_UNSUPPORTED;
  if (b->num_reqs < 0 || b->total_q < 0 || b->max_q_len < 0 || b->max_seq_len < 0)
    return IPD_ERR_INVALID_ARG;
  if (b->num_reqs == 0) return IPD_OK;
  if (b->max_q_len < 1 || b->max_seq_len < b->max_q_len) return IPD_ERR_INVALID_ARG;
  if ((long long)b->max_pages * kPage < b->max_seq_len) return IPD_ERR_INVALID_ARG;
  if (c->num_pages < 1) return IPD_ERR_INVALID_ARG;
  if (c->num_pages * c->num_kv_heads * (long long)kPage >= (1LL << 31)) return IPD_ERR_UNSUPPORTED;
  if (!b->q || !b->out || !b->cu_q || !b->seq_len || !b->page_table || !c->k_pages ||
      !c->v_pages)
    return IPD_ERR_INVALID_ARG;
  if (((uintptr_t)b->q | (uintptr_t)b->out | (uintptr_t)c->k_pages | (uintptr_t)c->v_pages) & 15)
    return IPD_ERR_INVALID_ARG;
  if (b->total_q > (long long)b->num_reqs * b->max_q_len) return IPD_ERR_INVALID_ARG;
  return IPD_OK;
}

int collect(const ipd_attn_batch *verify, int nv, const ipd_attn_batch *decode, int nd,
            const ipd_attn_batch **out) {
  if (nv < 0 || nd < 0 || nv + nd > IPD_MAX_BATCHES) return IPD_ERR_INVALID_ARG;
  if ((nv && !verify) || (nd && !decode)) return IPD_ERR_INVALID_ARG;
  int n = 0;
  for (int i = 0; i < nv; ++i) out[n++] = &verify[i];
  for (int i = 0; i < nd; ++i) out[n++] = &decode[i];
  for (int i = 0; i < n; ++i) {
    const int st = validate_batch(out[i]);
    if (st != IPD_OK) return st;
  }
  return IPD_OK;
}

// rows per row block of a task with `rows` rows
__host__ __device__ inline int rows_per_block(int rows) {
  return rows >= kTcMinRows ? kTcRows : kCcRows;
}

WsLayout layout(const ipd_attn_batch *const *bs, int n) {
  WsLayout L{};
  long long task_cap = 0, rows_all = 0;
  int reqs = 0;
  for (int i = 0; i < n; ++i) {
    const ipd_attn_batch *b = bs[i];
    const int G = b->num_q_heads / b->cache->num_kv_heads;
    // a task with r rows has ceil(r / rows_per_block(r)) row blocks; the
    // largest r = max_q_len * G bounds every request of the batch
    const long long rmax = (long long)b->max_q_len * G;
    const long long nrb = rmax >= kTcMinRows ? (rmax + kTcRows - 1) / kTcRows : 1;
    task_cap += (long long)b->num_reqs * b->cache->num_kv_heads * nrb;
    rows_all += (long long)b->total_q * b->num_q_heads;
    reqs += b->num_reqs;
  }
  const long long item_cap = task_cap + 2LL * kMaxTargetItems;
  const long long prow_cap =
      std::min<long long>(2LL * kMaxTargetItems * kTcRows, (long long)kSplitMax * rows_all);
  L.item_cap = (int)std::min<long long>(item_cap, 1LL << 30);
  L.task_cap = (int)std::min<long long>(task_cap, 1LL << 30);
  L.prow_cap = prow_cap;
  L.total_reqs = reqs;
  size_t off = 0;
  L.off_ctrl = off;
  off = align_up(off + 64, 256);
  L.off_reqinfo = off;
  off = align_up(off + (size_t)reqs * sizeof(int4), 256);
  L.off_reqslot = off;
  off = align_up(off + (size_t)reqs * sizeof(int2), 256);
  L.off_items = off;
  off = align_up(off + (size_t)L.item_cap * sizeof(Item), 256);
  L.off_done = off;
  off = align_up(off + (size_t)L.task_cap * sizeof(int), 256);
  L.off_partials = off;
  off = align_up(off + (size_t)prow_cap * kPStride * sizeof(float), 256);
  L.total = off;
  return L;
}

// --------------------------------------------------------------------------
// planner: one block builds the work list from the device-resident lengths
// --------------------------------------------------------------------------
__device__ __forceinline__ int find_batch(const AttnParams &p, int gi) {
  int b = 0;
  while (b + 1 < p.n_batches && gi >= p.req_base[b + 1]) ++b;
  return b;
}

struct ReqShape {
  int ql, L, pages, rows, nrb, rpb, ok;
};

__device__ ReqShape req_shape(const AttnParams &p, int b, int r) {
  const BatchDev &B = p.b[b];
  ReqShape s{};
  const int c0 = B.cu_q[r], c1 = B.cu_q[r + 1];
  s.ql = c1 - c0;
  s.L = B.seq_len[r];
  s.ok = 1;
  if (s.ql < 0 || c0 < 0 || c1 > B.total_q) {
    ipd_set_error(&g_attn_err, IPD_DEVERR_SPAN);
    s.ok = 0;
  } else if (s.ql > B.max_q_len || s.L < s.ql || s.L > B.max_pages * kPage) {
    ipd_set_error(&g_attn_err, IPD_DEVERR_SEQ_LEN);
    s.ok = 0;
  }
  if (!s.ok || s.ql == 0) {
    s.ql = 0; s.L = 0; s.pages = 0; s.rows = 0; s.nrb = 0; s.rpb = 1;
    return s;
  }
  s.pages = (s.L + kPage - 1) / kPage;
  s.rows = s.ql * B.group;
  s.rpb = rows_per_block(s.rows);
  s.nrb = (s.rows + s.rpb - 1) / s.rpb;
  return s;
}

template <typename T>
__device__ T block_sum(T v, T *red) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  T t = 0;
  for (int i = 0; i < nw; ++i) t += red[i];
  __syncthreads();
  return t;
}

// maximum of one int per thread across the block (red: one slot per warp)
__device__ int block_max_int(int v, long long *red) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  int t = 0;
  for (int i = 0; i < nw; ++i) t = max(t, (int)red[i]);
  __syncthreads();
  return t;
}

// exclusive scan of four ints across the block; returns totals in tot
__device__ void block_scan4(int4 v, int4 &excl, int4 &tot, int4 *sh) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int4 inc = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int x = __shfl_up_sync(0xffffffffu, inc.x, o);
    const int y = __shfl_up_sync(0xffffffffu, inc.y, o);
    const int z = __shfl_up_sync(0xffffffffu, inc.z, o);
    const int q = __shfl_up_sync(0xffffffffu, inc.w, o);
    if (lane >= o) { inc.x += x; inc.y += y; inc.z += z; inc.w += q; }
  }
  __syncthreads();
  if (lane == 31) sh[w] = inc;
  __syncthreads();
  int4 base = make_int4(0, 0, 0, 0);
  tot = make_int4(0, 0, 0, 0);
  for (int i = 0; i < nw; ++i) {
    if (i < w) { base.x += sh[i].x; base.y += sh[i].y; base.z += sh[i].z; base.w += sh[i].w; }
    tot.x += sh[i].x; tot.y += sh[i].y; tot.z += sh[i].z; tot.w += sh[i].w;
  }
  excl = make_int4(base.x + inc.x - v.x, base.y + inc.y - v.y, base.z + inc.z - v.z,
                   base.w + inc.w - v.w);
  __syncthreads();
}

// Pages per split of a request with `pages` pages, for a target chunk size:
// a whole number of stages, so only a request's last split ends mid-stage.
__device__ __forceinline__ int split_pages(int pages, int chunk) {
  int ns = (int)(((unsigned)pages + (unsigned)chunk - 1u) / (unsigned)chunk);
  if (ns > kSplitMax) ns = kSplitMax;
  const int per = (int)(((unsigned)pages + (unsigned)ns - 1u) / (unsigned)ns);
  return (per + kStagePages - 1) / kStagePages * kStagePages;
}
__device__ __forceinline__ int split_count(int pages, int chunk) {
  const int per = split_pages(pages, chunk);
  return (pages + per - 1) / per;
}

// Claim-order bucket of an item of batch `b` with `n` pages; higher buckets
// are claimed first.  Streaming one cache at a time measured faster than
// interleaving both (every CTA streams more slowly when the two pools are
// read at once), and longest-first within a batch keeps the tail short.
__device__ __forceinline__ int size_bucket(int b, int n_batches, int n, int chunk) {
  const unsigned top = (unsigned)((chunk + kStagePages - 1) / kStagePages * kStagePages);  // usual largest
  unsigned k = (unsigned)n * (unsigned)(kSizesPerBatch - 1) / top;  // n < 2^27: no overflow
  if (k > (unsigned)(kSizesPerBatch - 1)) k = kSizesPerBatch - 1;
  return (n_batches - 1 - b) * kSizesPerBatch + (int)k;
}

// Reserve n consecutive slots of bucket `bucket` (< 0: none) for every lane;
// lanes asking for the same bucket share one shared-memory atomic.  All 32
// lanes call it.  Returns the lane's first slot, relative to the bucket.
__device__ __forceinline__ int warp_reserve(int *slots, int bucket, int n) {
  const int lane = threadIdx.x & 31;
  const unsigned grp = __match_any_sync(0xffffffffu, bucket);
  const unsigned same_n = __match_any_sync(0xffffffffu, n);
  int excl = 0, total = 0;
  if ((grp & same_n) == grp) {  // one count for the whole group (the usual case)
    excl = n * __popc(grp & ((1u << lane) - 1u));
    total = n * __popc(grp);
  } else {
    for (unsigned m = grp; m; m &= m - 1) {
      const int l = __ffs(m) - 1;
      const int v = __shfl_sync(grp, n, l);
      if (l < lane) excl += v;
      total += v;
    }
  }
  const int leader = __ffs(grp) - 1;
  int base = 0;
  if (lane == leader && bucket >= 0 && total > 0) base = atomicAdd(&slots[bucket], total);
  base = __shfl_sync(grp, base, leader);
  return base + excl;
}

// One block of kT threads (256 for up to 1024 requests, else 1024).  Each
// thread owns requests tid, tid + kT, ...; the first kPlanCache of them keep
// their shape (two loads each) in registers across the three passes: total
// work, per-request counts with their block scan, and the items.  The
// 256-thread block needs a quarter of an SM's registers, so it starts beside
// row-pass CTAs already resident there; a 1024-thread block needs a whole
// SM's registers and would wait for the row pass to drain an SM.
constexpr int kPlanThreads = 1024;  // the planner block for more than 256 * kPlanCache requests
constexpr int kPlanCache = 4;

template <int kT>
__global__ void __launch_bounds__(kT) attn_plan_kernel(const __grid_constant__ AttnParams p) {
  __shared__ long long red[32];
  __shared__ int4 sh4[32];
  __shared__ int s_fail;
  __shared__ int s_slot[kSizeBuckets];  // items per size bucket, then each bucket's next slot
  const int tid = threadIdx.x;
  if (tid == 0) s_fail = 0;
  for (int i = tid; i < kSizeBuckets; i += kT) s_slot[i] = 0;

  ReqShape cs[kPlanCache];
  int cbat[kPlanCache];
#pragma unroll
  for (int k = 0; k < kPlanCache; ++k) {
    const int gi = tid + k * kT;
    cbat[k] = 0;
    cs[k] = ReqShape{};
    if (gi < p.total_reqs) {
      cbat[k] = find_batch(p, gi);
      cs[k] = req_shape(p, cbat[k], gi - p.req_base[cbat[k]]);
    }
  }
  // the k-th request of this thread (k < kPlanCache from registers)
  auto shape_of = [&](int k, int gi, int &b) -> ReqShape {
#pragma unroll
    for (int j = 0; j < kPlanCache; ++j)
      if (k == j) {
        b = cbat[j];
        return cs[j];
      }
    b = find_batch(p, gi);
    return req_shape(p, b, gi - p.req_base[b]);
  };
  const int n_rounds = (p.total_reqs + kT - 1) / kT;

  long long w = 0;
  int pmax = 0;
  for (int k = 0; k < n_rounds; ++k) {
    const int gi = tid + k * kT;
    if (gi < p.total_reqs) {
      int b;
      const ReqShape s = shape_of(k, gi, b);
      w += (long long)s.pages * p.b[b].hkv * s.nrb;
      pmax = max(pmax, s.pages);
    }
  }
  const long long W = block_sum<long long>(w, red);
  const int P_max = block_max_int(pmax, red);
  // chunks of a quarter of an SM's share split the long tasks for balance;
  // when no task reaches half a share, tasks stay whole (splitting them only
  // adds item boundaries and merges: measured 3 % on 768 tasks of <= 512
  // pages over 152 SMs)
  long long chunk_ll = (W + p.target_items - 1) / p.target_items;
  if ((long long)P_max <= 2 * chunk_ll) chunk_ll = P_max > chunk_ll ? P_max : chunk_ll;
  if (chunk_ll < kMinChunkPages) chunk_ll = kMinChunkPages;
  if (chunk_ll > (1LL << 30)) chunk_ll = 1LL << 30;
  const int chunk = (int)chunk_ll;

  // per request: split count, task and partial-row offsets (exclusive
  // scans), and the size histogram of its items
  int4 carry = make_int4(0, 0, 0, 0);  // (unused), tasks, partial rows, items
  for (int k = 0; k < n_rounds; ++k) {
    const int gi = tid + k * kT;
    int4 cnt = make_int4(0, 0, 0, 0);
    int nsplit = 1;
    // splits 0 .. ns-2 have `per` pages (one bucket), the last split the rest
    int bk_main = -1, n_main = 0, bk_last = -1, n_last = 0;
    if (gi < p.total_reqs) {
      int b;
      const ReqShape s = shape_of(k, gi, b);
      if (s.pages > 0) {
        nsplit = split_count(s.pages, chunk);
        const int per = split_pages(s.pages, chunk);
        const int hkv = p.b[b].hkv;
        const int tasks = hkv * s.nrb;
        cnt = make_int4(0, tasks, nsplit > 1 ? nsplit * hkv * s.rows : 0, tasks * nsplit);
        if (nsplit > 1) {
          bk_main = size_bucket(b, p.n_batches, per, chunk);
          n_main = (nsplit - 1) * tasks;
        }
        bk_last = size_bucket(b, p.n_batches, s.pages - (nsplit - 1) * per, chunk);
        n_last = tasks;
      }
    }
    const int off_main = warp_reserve(s_slot, bk_main, n_main);
    const int off_last = warp_reserve(s_slot, bk_last, n_last);
    if (gi < p.total_reqs) p.reqslot[gi] = make_int2(off_main, off_last);
    int4 ex, tot;
    block_scan4(cnt, ex, tot, sh4);
    if (gi < p.total_reqs)
      p.reqinfo[gi] = make_int4(carry.x + ex.x, carry.y + ex.y, carry.z + ex.z, nsplit);
    carry.x += tot.x; carry.y += tot.y; carry.z += tot.z; carry.w += tot.w;
  }
  __syncthreads();
  if (tid < 32) {
    // bucket start slots, largest bucket first: lane l sums buckets
    // kSizeBuckets-1-8l .. -7 (descending), then an exclusive warp scan
    constexpr int kPer = kSizeBuckets / 32;
    int v[kPer], sum = 0;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      v[i] = s_slot[kSizeBuckets - 1 - (tid * kPer + i)];
      sum += v[i];
    }
    int inc = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, inc, o);
      if (tid >= o) inc += y;
    }
    int off = inc - sum;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      s_slot[kSizeBuckets - 1 - (tid * kPer + i)] = off;
      off += v[i];
    }
  }
  if (tid == 0) {
    if (carry.w > p.item_cap || carry.y > p.task_cap || carry.z > p.prow_cap) {
      ipd_set_error(&g_attn_err, IPD_DEVERR_PLAN);
      s_fail = 1;
    }
    p.ctrl[0] = s_fail ? 0 : carry.w;
    p.ctrl[1] = 0;
    p.ctrl[2] = carry.y;
    p.ctrl[3] = carry.z;
    p.ctrl[4] = chunk < P_max ? 1 : 0;
  }
  __syncthreads();
  if (s_fail) return;

  for (int k = 0; k < n_rounds; ++k) {
    const int gi = tid + k * kT;
    if (gi >= p.total_reqs) continue;
    int b;
    const ReqShape s = shape_of(k, gi, b);
    if (s.pages == 0) continue;
    const int r = gi - p.req_base[b];
    const int4 info = p.reqinfo[gi];
    const int task = info.y;
    const int ns = info.w;
    const int per = split_pages(s.pages, chunk);
    const int hkv = p.b[b].hkv;
    const int tasks = hkv * s.nrb;
    const int2 rs = p.reqslot[gi];
    const int base_main = ns > 1 ? s_slot[size_bucket(b, p.n_batches, per, chunk)] + rs.x : 0;
    const int base_last =
        s_slot[size_bucket(b, p.n_batches, s.pages - (ns - 1) * per, chunk)] + rs.y;
    const int path = s.rows < kTcMinRows ? kPathCc : -1;
    for (int sp = 0; sp < ns; ++sp) {
      const int lo = sp * per, hi = min(s.pages, (sp + 1) * per);
      int slot = sp < ns - 1 ? base_main + sp * tasks : base_last;
      int task_t = task;
      for (int kvh = 0; kvh < hkv; ++kvh) {
        for (int rb = 0; rb < s.nrb; ++rb) {
          const int rows = min(s.rpb, s.rows - rb * s.rpb);
          const int pbase = ns > 1 ? info.z + ns * (kvh * s.rows + rb * s.rpb) : -1;
          const int pth = path >= 0 ? path : tc_path(rows);
          int4 *dst = reinterpret_cast<int4 *>(p.items + slot);
          dst[0] = make_int4(b, r, kvh, rb);
          dst[1] = make_int4(sp, ns, lo, hi);
          if (ns > 1 && sp == 0) p.split_done[task_t] = 0;
          dst[2] = make_int4(task_t++, pbase, rows, pth);
          ++slot;
        }
      }
    }
  }
}

// Split-KV merge of one output row of a task split over several items: the
// splits' partial rows (unnormalised O, maximum m, sum l, all in log2 units)
// combine into the output row; lane = 4 dims, every split's loads in flight
// at once.
__device__ void merge_split_row(const AttnParams &p, const Item &I, int r, int lane) {
  const BatchDev &Bt = p.b[I.b];
  const int q0 = Bt.cu_q[I.r], G = Bt.group;
  const int rpb = I.path != kPathCc ? kTcRows : kCcRows;
  const int ns = I.n_split;
  const size_t sstr = (size_t)I.rows * kPStride;
  const float *base = p.partials + (size_t)(I.pbase + r) * kPStride;
  const float mv = lane < ns ? __ldcg(base + lane * sstr + 128) : -INFINITY;
  const float lv = lane < ns ? __ldcg(base + lane * sstr + 129) : 0.f;
  float4 ov[kSplitMax];
#pragma unroll
  for (int sp = 0; sp < kSplitMax; ++sp)
    if (sp < ns) ov[sp] = __ldcg(reinterpret_cast<const float4 *>(base + sp * sstr) + lane);
  const float Mx = warp_max(mv);
  const float f = mv == -INFINITY ? 0.f : ex2_approx(mv - Mx);
  const float Ls = warp_sum(lv * f);
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int sp = 0; sp < kSplitMax; ++sp) {
    if (sp < ns) {
      const float fs = __shfl_sync(0xffffffffu, f, sp);
      acc.x = fmaf(ov[sp].x, fs, acc.x);
      acc.y = fmaf(ov[sp].y, fs, acc.y);
      acc.z = fmaf(ov[sp].z, fs, acc.z);
      acc.w = fmaf(ov[sp].w, fs, acc.w);
    }
  }
  const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
  const int grow = I.rb * rpb + r;
  const int qi = grow / G, j = grow % G;
  uint2 pk;
  pk.x = pack_bf16x2(acc.x * inv, acc.y * inv);
  pk.y = pack_bf16x2(acc.z * inv, acc.w * inv);
  *reinterpret_cast<uint2 *>(Bt.out + ((size_t)(q0 + qi) * Bt.hq + I.kvh * G + j) * kD +
                             lane * 4) = pk;
}

// --------------------------------------------------------------------------
// the attention kernel
// --------------------------------------------------------------------------
// V jobs handed from the K producer to the V producer.  The K producer
// writes job i + kVJobs after the K slot of stage use i + kVJobs - kStages
// is released, which the compute warps do only once they have finished use
// i + kVJobs - kStages - 1; finishing a use means the V of the use before it
// was issued (its P V, or the CUDA-core path's own wait, saw it land), so
// job i + kVJobs - kStages - 2 >= i, and job i, have been read by then.
constexpr int kVJobs = 2 * kStages;

struct Smem {
  static constexpr int off_stage = 0;                              // 3 x 64 KB, 1024-aligned
  // the P operand of a stacked tile, or the Q tile of a 128-row tile: two
  // halves (64 keys, or 64 dims) of 128 rows x 128 B, 128-byte swizzled (a
  // K-major A operand); also the finalize's exchange area and the CUDA-core
  // path's scratch
  static constexpr int off_p = off_stage + kStages * kStageBytes;
  static constexpr int kPHalf = kTcRows * 128;                     // 16 KB
  static constexpr int off_x = off_p + 2 * kPHalf;                 // row-max / row-sum exchange [2][256]
  static constexpr int off_meta = off_x + 2 * 256 * 4;
  static constexpr int off_bar = off_meta + kStages * (int)sizeof(StageMeta);
  static constexpr int n_bars = 4 * kStages + 6 + kVJobs;
  static constexpr int off_misc = off_bar + n_bars * 8;
  // per stage use (a ring of kVJobs), the V boxes' coordinates for the
  // second producer warp: eight page slots and the V tensor map's index
  // (-1: stop)
  static constexpr int off_vjob = off_misc + 64;
  static constexpr int total = off_vjob + kVJobs * 16 * 4;
  // CUDA-core path scratch (inside the P region, unused by that path)
  static constexpr int off_ccq = off_p;                              // fp32 [7][128]
  static constexpr int off_merge = off_ccq + kCcRows * kD * 4;       // fp32 [4][8][132]
  static constexpr int off_ps = off_merge + kCcW * 8 * kPStride * 4;  // fp32 [4][8][16] / [4][32][2]
};
static_assert(Smem::off_ps + kCcW * 8 * 16 * 4 <= Smem::off_x, "CUDA-core scratch overflow");
static_assert(kTcRows / 2 * kD * 4 <= 2 * Smem::kPHalf, "O exchange overflow");
static_assert(Smem::off_p % 1024 == 0, "swizzle atoms of the P tile");
static_assert(Smem::off_bar % 8 == 0, "mbarrier alignment");
static_assert(Smem::total <= 227 * 1024, "shared memory");

struct Bars {
  // KV ring: full = the stage's K (and its metadata) landed, vfull = its V
  // landed; empty = its K slot free, vempty = its V slot free.  In tiles of
  // up to 64 rows K is released once Q K^T has read it and V after P V, so
  // K is refilled a chunk earlier; other stages are released whole.
  uint64_t *full, *empty, *vfull, *vempty;
  uint64_t *q_ready;       // Q tile written to TMEM (one phase per tensor item)
  uint64_t *s_full;        // S = Q K^T landed, per S buffer (one phase per use)
  uint64_t *p_full;        // P of a chunk written (one phase per chunk)
  uint64_t *p_free;        // P V product of a chunk done: P read, O written (one phase per chunk)
  uint64_t *s_free;        // P V of a chunk done, per S buffer: the buffer may take the next Q K^T
  uint64_t *v_go;          // per V job slot: the job is written (one phase per use of the slot)
};

__device__ __forceinline__ Bars bars(uint8_t *smem) {
  uint64_t *b = reinterpret_cast<uint64_t *>(smem + Smem::off_bar);
  Bars r;
  r.full = b;
  r.empty = b + kStages;
  r.vfull = b + 2 * kStages;
  r.vempty = b + 3 * kStages;
  r.q_ready = b + 4 * kStages;
  r.s_full = r.q_ready + 1;
  r.p_full = r.s_full + 2;
  r.p_free = r.p_full + 1;
  r.s_free = r.p_free + 1;
  r.v_go = r.s_free + 2;
  return r;
}

// byte offset of 16-byte chunk c (0..7) of row `row` in a 128-byte-swizzled
// block of 128-byte rows (the layout TMA writes with SWIZZLE_128B)
__device__ __forceinline__ uint32_t sw128(int row, int c) {
  return (uint32_t)(row * 128 + ((c ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint8_t *stage_k(uint8_t *smem, int s) {
  return smem + Smem::off_stage + s * kStageBytes;
}
__device__ __forceinline__ uint8_t *stage_v(uint8_t *smem, int s) {
  return stage_k(smem, s) + kTensorBytes;
}
// row R (key of the stage), 64-dim half h of a staged K or V tensor; its
// 16-byte chunk c sits at ((c ^ (R & 7)) << 4)
__device__ __forceinline__ const uint8_t *kv_row(const uint8_t *t, int R, int h) {
  return t + (R >> 3) * kGroupBytes + h * kAtomBytes + (R & 7) * 128;
}

// fp32 Q layout of the CUDA-core path: dim d = half*64 + c*8 + sub*4 + e is
// stored at half*64 + sub*32 + c*4 + e (conflict-free float4 reads below).
__device__ __forceinline__ int q_slot(int d) {
  const int half = d >> 6, c = (d >> 3) & 7, sub = (d >> 2) & 1, e = d & 3;
  return half * 64 + sub * 32 + c * 4 + e;
}


struct CompCtx {
  uint8_t *smem;
  Bars B;
  StageMeta *meta;
  uint32_t *misc;  // [0] TMEM base, [1] abort flag
  uint32_t tmem;
  int warp, lane, ctid;
};

__device__ __forceinline__ bool wait_or_abort(const CompCtx &X, uint64_t *bar, uint32_t par) {
  if (mbar_wait_bounded(bar, par)) return true;
  ipd_set_error(&g_attn_err, IPD_DEVERR_WAIT);
  atomicExch(&X.misc[1], 1u);
  return false;
}

struct ItemGeom {
  const BatchDev *Bt;
  int q0, ql, L, G, hq;
};

__device__ __forceinline__ ItemGeom item_geom(const AttnParams &p, const Item &I) {
  ItemGeom g;
  g.Bt = &p.b[I.b];
  g.q0 = g.Bt->cu_q[I.r];
  g.ql = g.Bt->cu_q[I.r + 1] - g.q0;
  g.L = g.Bt->seq_len[I.r];
  g.G = g.Bt->group;
  g.hq = g.Bt->hq;
  return g;
}

// query / output row of task row `grow` (query grow / G, head kvh * G + grow % G)
__device__ __forceinline__ size_t row_off(const ItemGeom &g, const Item &I, int grow) {
  const int qi = grow / g.G, j = grow % g.G;
  return ((size_t)(g.q0 + qi) * g.hq + I.kvh * g.G + j) * kD;
}
__device__ __forceinline__ uint16_t *out_row(const ItemGeom &g, const Item &I, int grow) {
  return g.Bt->out + row_off(g, I, grow);
}
__device__ __forceinline__ const uint16_t *q_row(const ItemGeom &g, const Item &I, int grow) {
  return g.Bt->q + row_off(g, I, grow);
}

// Zero the V rows of stage s at or past the end of the sequence: unwritten
// cache slots may hold non-finite bits, and a zero probability times NaN is NaN.
// Waits for the stage's V first (false on a time-out); V of a stage without
// a tail is never touched by the compute warps.
__device__ __forceinline__ bool zero_tail(const CompCtx &X, int s, uint32_t par, int page0, int L,
                                          int nthreads, int bar) {
  const int tail0 = max(L - page0 * kPage, 0);  // first key slot at or past L
  if (tail0 >= kStageKeys) return true;
  if (!wait_or_abort(X, &bars(X.smem).vfull[s], par)) return false;
  uint8_t *vb = stage_v(X.smem, s);
  for (int e = X.ctid; e < (kStageKeys - tail0) * 16; e += nthreads) {
    const int row = tail0 + e / 16, cpart = e % 16;
    *reinterpret_cast<uint4 *>(const_cast<uint8_t *>(kv_row(vb, row, cpart >> 3)) + (cpart & 7) * 16) =
        make_uint4(0, 0, 0, 0);
  }
  fence_proxy_async_smem();
  named_bar_sync(bar, nthreads);
  return true;
}

// ============================ tensor-core path ============================
// One 128-lane tile over the item's KV chunks of 128 keys, worked on by all
// eight compute warps.  Warps w and w + 4 reach the same TMEM lanes
// 32 (w % 4) .. 32 (w % 4) + 31, so every lane has two threads.
// A tile of at most 128 / F rows (F = 4, 2 or 1) is repeated F times over the
// lanes (its Q is written F times): lane t holds row t mod (128 / F) and owns
// keys [128 k / F, 128 (k + 1) / F) of every chunk, k = t / (128 / F), which
// its two threads split.  Every SM sub-partition thus has softmax work
// however few rows the tile has, and a thread's share of a chunk is 64 / F
// keys.
// P reaches the tensor cores as three bf16 terms (its upper 16 bits, the
// truncated residual and what is left of it, rounded), so P V sees each
// probability to within 2^-25 of itself.  Where the terms go:
//   F = 4: all three to the shared-memory P operand, term j of row r in
//     operand row 32 j + r (rows 96..127 are not used): one MMA per 16 keys
//     leaves the three terms' products in O lanes r, 32 + r and 64 + r;
//   F = 2: terms 1 and 2 to operand rows r and 64 + r, the third to the
//     lane's TMEM columns at kColT3 (the other copy's keys there are zeros,
//     written once per item): two MMAs per 16 keys, O lanes r and 64 + r;
//   F = 1: terms 1 and 2 overwrite the chunk's own S columns, the third goes
//     to the columns of the S buffer's parity at 384: three MMAs per 16 keys,
//     every A operand read from TMEM.  Its Q tile is in shared memory.
// Terms bound for the P operand or kColT3 are written only once the previous
// chunk's P V, their last reader, has completed: the first 16-key step's
// terms wait in registers for it, later steps are stored as they are made.
// Every chunk's P V lands in a fresh O (its first MMA overwrites O), and each
// thread adds its 64 output dimensions of it into fp32 registers with
// round-to-nearest adds.  The tensor core's accumulator does not round to
// nearest, and its error grows with the number of products summed into one
// accumulator (measured: 6 to 25 bf16 ulp of the tolerance floor after 8K to
// 32K keys); within one 128-key chunk it stays far below the floor.
// The row maximum is exchanged among the row's threads through shared memory
// and rescales the register sums only when it grows by more than 2^8.
// Returns false on a wait time-out.  `it` (stage counter) and `c` (chunk
// counter) advance.
template <int F>
__device__ __forceinline__ bool tc_item(const AttnParams &p, const CompCtx &X, const Item &I,
                                        uint32_t &it, uint32_t &c) {
  constexpr int kRep = kTcRows / F;                 // rows of one copy (>= 32: a copy is warp-uniform)
  constexpr int kKT = 64 / F;                       // keys of a chunk per thread
  constexpr int kSteps = kKT / 16;                  // 16-key steps per thread
  constexpr int kExpUnroll = F == 1 ? 1 : kSteps;  // exponential-pass steps unrolled
  const ItemGeom g = item_geom(p, I);
  const Bars &B = X.B;
  const int lb = X.warp & 3;                        // lane block of this warp
  const int second = X.warp >> 2;                   // which of the lane's two threads
  const int t = lb * 32 + X.lane;                   // TMEM lane
  const int copy = t / kRep;
  const int row = t % kRep;                         // tile row
  const int kown = copy * (kStageKeys / F);         // first key the lane owns
  const int k0 = kown + second * kKT;               // first key of this thread
  const bool real = row < I.rows;
  // F = 4 leaves O lanes 96..127 unused (the P operand's rows 96..127 are
  // not written); their threads take no O.
  const bool takes_o = F != 4 || t < 3 * kRep;
  const uint32_t tl = X.tmem + ((uint32_t)(lb * 32) << 16);
  const int lim = g.L - g.ql + (I.rb * kTcRows + row) / g.G;  // last key this row sees
  const int lim_all = g.L - g.ql;                             // every row sees up to here
  const float sl2 = p.scale_log2;
  float *xbuf = reinterpret_cast<float *>(X.smem + Smem::off_x);  // [2][2][128]
  uint8_t *ps = X.smem + Smem::off_p;
  float m_used = -INFINITY;  // maximum the exponentials are taken against (log2 units)
  float l_run = 0.f;         // this thread's share of the row sum (in the scale of m_used)
  float alpha_pend = 1.f;    // rescale still owed by the product in O (see below)
  float acc[64];             // output dims 64 second .. of this lane's O, summed over chunks
#pragma unroll
  for (int e = 0; e < 64; ++e) acc[e] = 0.f;
  // "P V of chunk k has landed in O" is completion k of p_free.  Chunk k waits
  // for completion k - 1 before its threads arrive on p_full, so the barrier
  // is never more than one phase behind a wait and the parity cannot alias.
  auto wait_pv_done = [&](uint32_t k) -> bool { return wait_or_abort(X, B.p_free, k & 1); };
  // acc = (acc + this thread's dims of O) * alpha
  auto take_o = [&](float alpha) {
    if (!takes_o) return;
    const bool scaled = __any_sync(0xffffffffu, alpha != 1.f);
    uint32_t r[2][32];
    tc_ld_32x32b_x32(tl + kColO + 64 * second, r[0]);
    tc_ld_32x32b_x32(tl + kColO + 64 * second + 32, r[1]);
    tc_wait_ld();
    if (scaled) {
#pragma unroll
      for (int e = 0; e < 64; ++e) acc[e] = (acc[e] + __uint_as_float(r[e >> 5][e & 31])) * alpha;
    } else {
#pragma unroll
      for (int e = 0; e < 64; ++e) acc[e] += __uint_as_float(r[e >> 5][e & 31]);
    }
  };
  // 16 keys (8 bf16 pairs) of one term into P operand row `ar`, from key kb
  auto store_p = [&](int ar, int kb, const uint32_t (&v)[8]) {
    uint8_t *h = ps + (kb >> 6) * Smem::kPHalf;
    const int j = (kb & 63) >> 3;
    *reinterpret_cast<uint4 *>(h + sw128(ar, j)) = make_uint4(v[0], v[1], v[2], v[3]);
    *reinterpret_cast<uint4 *>(h + sw128(ar, j + 1)) = make_uint4(v[4], v[5], v[6], v[7]);
  };

  for (bool first = true;; first = false) {
    const int s = it % kStages;
    if (!wait_or_abort(X, &B.full[s], (it / kStages) & 1)) return false;
    const StageMeta M = X.meta[s];
    if (!zero_tail(X, s, (it / kStages) & 1, M.page0, g.L, kCW * 32, 1)) return false;
    if (first) {
      const uint4 *src =
          reinterpret_cast<const uint4 *>(q_row(g, I, I.rb * kTcRows + row) + 64 * second);
      if (F == 1) {
        // The shared-memory region is the CUDA-core path's scratch: after a
        // CUDA-core item, warps kCcW.. get here while the first warps may
        // still be using it.
        named_bar_sync(1, kCW * 32);
        // Q: this thread's half of the lane's row (dims 64 second ..) into
        // operand row t of the swizzled Q tile
        uint8_t *qh = ps + second * Smem::kPHalf;
#pragma unroll
        for (int j = 0; j < 8; ++j)
          *reinterpret_cast<uint4 *>(qh + sw128(t, j)) = real ? __ldg(src + j) : make_uint4(0, 0, 0, 0);
        fence_proxy_async_smem();
      } else {
        // Q: this thread's half of the lane's row (dims 64 second ..) as 32
        // TMEM columns of bf16 pairs (zeros past the rows)
        uint32_t qw[32];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          uint4 v = make_uint4(0, 0, 0, 0);
          if (real) v = __ldg(src + j);
          qw[4 * j + 0] = v.x;
          qw[4 * j + 1] = v.y;
          qw[4 * j + 2] = v.z;
          qw[4 * j + 3] = v.w;
        }
        tc_st_32x32b_x32(tl + kColQ + 32 * second, qw);
        if (F == 2 && second == 0) {
          // zeros in the third-term columns of the other copy's keys
          const uint32_t z[32] = {};
          tc_st_32x32b_x32(tl + t3_col(copy == 0 ? 4 : 0), z);
        }
        tc_wait_st();
        tc_fence_before();
      }
      __syncwarp();
      if (X.lane == 0) mbar_arrive(B.q_ready);
    }
    // This warp is done with the stage's metadata and, unless the tile is a
    // 128-row one (whose S may be recomputed from the stage's K below: its
    // stage is released by its P V, which follows), with its K.
    __syncwarp();
    if (X.lane == 0) mbar_arrive(&B.empty[s]);

    const uint32_t b = c & 1;
    if (!wait_or_abort(X, &B.s_full[b], (c >> 1) & 1)) return false;
    tc_fence_after();
    const int kp0 = M.page0 * kPage;
    const bool full_vis =
        M.npages == kStagePages && M.invalid == 0 && kp0 + kStageKeys - 1 <= lim_all;
    // -inf for the keys of the stage this row does not see
    auto mask = [&](auto &v, int col0) {
      if (!full_vis) {
#pragma unroll
        for (int e = 0; e < (int)(sizeof(v) / sizeof(v[0])); ++e) {
          const int col = col0 + e;
          const bool vis = (col >> 4) < M.npages && !((M.invalid >> (col >> 4)) & 1u) &&
                           kp0 + col <= lim;
          if (!vis) v[e] = 0xff800000u;
        }
      }
    };
    // This thread's S values: tiles repeated over the lanes keep theirs (16
    // or 32) in registers, loaded at once; 128-row tiles read theirs 16 at a
    // time from TMEM.
    constexpr int kKeep = F == 1 ? 1 : kSteps;
    uint32_t sv[kKeep][16];
    if (F != 1) {
#pragma unroll
      for (int q = 0; q < kKeep; ++q) tc_ld_32x32b_x16(tl + col_s(b) + k0 + 16 * q, sv[q]);
      tc_wait_ld();
#pragma unroll
      for (int q = 0; q < kKeep; ++q) mask(sv[q], k0 + 16 * q);
    }
    // the maximum of 16 values (three-operand maxima: 8 instructions)
    auto max16 = [](const uint32_t (&v)[16], float m) {
      float m5[5];
#pragma unroll
      for (int e = 0; e < 5; ++e)
        m5[e] = fmax3(__uint_as_float(v[3 * e]), __uint_as_float(v[3 * e + 1]),
                      __uint_as_float(v[3 * e + 2]));
      return fmax3(m, fmax3(m5[0], m5[1], m5[2]), fmax3(m5[3], m5[4], __uint_as_float(v[15])));
    };
    // a 128-row tile's S values of keys k0 + 16 q .. on CUDA cores, from its Q
    // tile in shared memory and the stage's K (only after a jump of the
    // maximum has made the tensor core's values unusable: see below)
    auto recompute_s = [&](int q, uint32_t (&v)[16]) {
      const uint8_t *kst = stage_k(X.smem, s);
      float a[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) a[e] = 0.f;
      for (int h = 0; h < 2; ++h) {
        for (int j = 0; j < 8; ++j) {
          const uint4 qv = *reinterpret_cast<const uint4 *>(ps + h * Smem::kPHalf + sw128(t, j));
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int R = k0 + 16 * q + e;
            const uint4 kv =
                *reinterpret_cast<const uint4 *>(kv_row(kst, R, h) + ((j ^ (R & 7)) << 4));
            float x = a[e];
            x = fmaf(bf16lo(qv.x), bf16lo(kv.x), x);
            x = fmaf(bf16hi(qv.x), bf16hi(kv.x), x);
            x = fmaf(bf16lo(qv.y), bf16lo(kv.y), x);
            x = fmaf(bf16hi(qv.y), bf16hi(kv.y), x);
            x = fmaf(bf16lo(qv.z), bf16lo(kv.z), x);
            x = fmaf(bf16hi(qv.z), bf16hi(kv.z), x);
            x = fmaf(bf16lo(qv.w), bf16lo(kv.w), x);
            a[e] = fmaf(bf16hi(qv.w), bf16hi(kv.w), x);
          }
        }
      }
#pragma unroll
      for (int e = 0; e < 16; ++e) v[e] = __float_as_uint(a[e]);
      mask(v, k0 + 16 * q);
    };

    // p = 2^(s*scale - m) as three bf16 terms, each the residual of the ones
    // before rounded to nearest: hi = bf16(p), lo = bf16(p - hi), lo2 =
    // bf16(p - hi - lo).  Both subtractions are exact (a residual has at most
    // 16 significant bits), so |p - hi - lo - lo2| <= 2^-27 p.  One conversion
    // packs a pair of keys' terms; the scaling, residuals and row sum run on
    // packed fp32 pairs.
    // the previous chunk's P V has read the P operand and the third-term
    // columns once this returns
    auto wait_prev = [&]() -> bool {
      if (!wait_pv_done(c - 1)) return false;
      tc_fence_after();
      return true;
    };
    // source 0: S from registers (repeated tiles) or TMEM (128-row tiles);
    // source 1: recomputed on CUDA cores (128-row tiles).  Adds the thread's
    // chunk maximum into *lm when given.
    auto exp_pass = [&](float moff, int source, unsigned long long &lsum2, float *lm) -> bool {
      const unsigned long long sl2x2 = f2_pack(sl2, sl2), moffx2 = f2_pack(moff, moff);
      // the two bf16 halves of a packed pair as fp32 values
      auto lo_f = [](uint32_t w) { return __uint_as_float(w << 16); };
      auto hi_f = [](uint32_t w) { return __uint_as_float(w & 0xffff0000u); };
      // (a 128-row tile's four steps stay a loop: its hot code then fits the
      // instruction cache)
#pragma unroll kExpUnroll
      for (int q = 0; q < kSteps; ++q) {
        uint32_t(&sr)[16] = sv[F == 1 ? 0 : q];
        if (F == 1) {
          if (source == 0) {
            tc_ld_32x32b_x16(tl + col_s(b) + k0 + 16 * q, sr);
            tc_wait_ld();
            mask(sr, k0 + 16 * q);
          } else {
            recompute_s(q, sr);
          }
        }
        if (lm) *lm = max16(sr, *lm);
        uint32_t th[8], tlo[8], t3[8];
#pragma unroll
        for (int e = 0; e < 16; e += 2) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[e]), __uint_as_float(sr[e + 1])), sl2x2,
                           moffx2),
                    x0, x1);
          const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
          const unsigned long long pp = f2_pack(p0, p1);
          const uint32_t w1 = pack_bf16x2(p0, p1);
          const unsigned long long l2 = f2_sub(pp, f2_pack(lo_f(w1), hi_f(w1)));
          float l0, l1, r0, r1;
          f2_unpack(l2, l0, l1);
          const uint32_t w2 = pack_bf16x2(l0, l1);
          f2_unpack(f2_sub(l2, f2_pack(lo_f(w2), hi_f(w2))), r0, r1);
          th[e >> 1] = w1;
          tlo[e >> 1] = w2;
          t3[e >> 1] = pack_bf16x2(r0, r1);
          lsum2 = f2_add(lsum2, pp);
        }
        const int kb = k0 + 16 * q;
        if (F == 1) {
          // the first two terms overwrite the S columns of these 16 keys,
          // which this thread has just read (and no other thread reads); the
          // third goes to the columns of this S buffer's parity, last read
          // by the P V of chunk c - 2
          tc_st_32x32b_x8(tl + col_s(b) + p_col(kb >> 4, 1), th);
          tc_st_32x32b_x8(tl + col_s(b) + p_col(kb >> 4, 2), tlo);
          tc_st_32x32b_x8(tl + t3_col_full(b, kb >> 4), t3);
        } else {
          if (q == 0 && !wait_prev()) return false;
          store_p(row, kb, th);
          store_p(kRep + row, kb, tlo);
          if (F == 4) store_p(2 * kRep + row, kb, t3);
          else tc_st_32x32b_x8(tl + t3_col(kb >> 4), t3);
        }
      }
      return true;
    };
    // the row's chunk maximum (log2 units) from the threads' entries
    float *xm = xbuf + (c & 1) * (2 * kTcRows);
    auto row_max = [&](float lm) {
      xm[second * kTcRows + t] = lm;
      // only the warps holding copies of the thread's row meet: a 128-row
      // tile's row lives in one lane block, a 64-row tile's in two
      if (F == 1) named_bar_sync(4 + lb, 64);
      else if (F == 2) named_bar_sync(8 + (lb & 1), 128);  // lane blocks lb and lb ^ 2
      else named_bar_sync(1, kCW * 32);
      float mx = lm;
#pragma unroll
      for (int j = 0; j < F; ++j)
        mx = fmaxf(mx, fmaxf(xm[row + j * kRep], xm[kTcRows + row + j * kRep]));
      return mx * sl2;
    };

    // The first chunk of an item (and every chunk of a repeated tile) takes
    // its row maximum first and the exponentials against it, the running
    // maximum moving up (and the sums rescaled) when the chunk's is 2^8
    // larger.  Later chunks of 128-row tiles take the exponentials against
    // the running maximum m_used in the same pass as the chunk's own maximum
    // (one pass over S, one exchange after it):
    //  - if the chunk's maximum exceeds m_used by more than 2^8, the running
    //    maximum moves up after the chunk: its P and row sum are in the old
    //    scale, so the rescale alpha_next is applied with its product, at the
    //    next chunk;
    //  - if it exceeds m_used by more than 2^64 (p could overflow), the
    //    chunk's exponentials are taken again against its own maximum, from
    //    S kept in registers or, in 128-row tiles, recomputed on CUDA cores.
    unsigned long long lsum2 = 0ull;  // {0.f, 0.f}
    float alpha_now = 1.f;   // rescale of acc and l_run before this chunk is added
    float alpha_next = 1.f;  // rescale after this chunk (applied with its product)
    float m_next = m_used;
    if (first || F != 1) {
      // (repeated tiles keep their S in registers: their maximum costs no
      // second read, and the one-pass form measured slower for them)
      float lm = -INFINITY;
#pragma unroll
      for (int q = 0; q < kSteps; ++q) {
        uint32_t(&sr)[16] = sv[F == 1 ? 0 : q];
        if (F == 1) {
          tc_ld_32x32b_x16(tl + col_s(b) + k0 + 16 * q, sr);
          tc_wait_ld();
          mask(sr, k0 + 16 * q);
        }
        lm = max16(sr, lm);
      }
      const float mcs = row_max(lm);
      if (real && mcs != -INFINITY) {
        // the lazy rescale: keep the old maximum unless the chunk's is 2^8 larger
        if (m_used == -INFINITY) {
          m_used = m_next = mcs;
        } else if (mcs > m_used + 8.f) {
          alpha_now = ex2_approx(m_used - mcs);
          m_used = m_next = mcs;
        }
      }
      const float moff = (!real || m_used == -INFINITY) ? -INFINITY : -m_used;
      if (!exp_pass(moff, 0, lsum2, nullptr)) return false;
    } else {
      float lm = -INFINITY;
      float moff = (!real || m_used == -INFINITY) ? -INFINITY : -m_used;
      if (!exp_pass(moff, 0, lsum2, &lm)) return false;
      const float mcs = row_max(lm);
      bool redo = false;
      if (real && mcs != -INFINITY) {
        if (m_used == -INFINITY || mcs > m_used + 64.f) {
          alpha_now = m_used == -INFINITY ? 0.f : ex2_approx(m_used - mcs);
          m_used = m_next = mcs;
          moff = -mcs;
          redo = true;
        } else if (mcs > m_used + 8.f) {
          alpha_next = ex2_approx(m_used - mcs);
          m_next = mcs;
        }
      }
      // TMEM loads and stores are warp-wide: the whole warp takes the second
      // pass when one of its rows needs it (its other rows recompute their
      // exponentials against their unchanged maximum)
      if (__any_sync(0xffffffffu, redo)) {
        lsum2 = 0ull;
        if (!exp_pass(moff, F == 1 ? 1 : 0, lsum2, nullptr)) return false;
      }
    }
    // then the previous chunk's product into the registers (before this
    // chunk's product overwrites O), with the rescales decided since
    if (F == 1 && !wait_prev()) return false;
    if (F != 1) fence_proxy_async_smem();
    if (!first) take_o(alpha_pend * alpha_now);
    {
      float a0, a1;
      f2_unpack(lsum2, a0, a1);
      if (real) l_run = (l_run * alpha_now + (a0 + a1)) * alpha_next;
    }
    alpha_pend = alpha_next;
    m_used = m_next;
    tc_wait_st();
    tc_fence_before();
    __syncwarp();
    if (X.lane == 0) mbar_arrive(B.p_full);
    ++it;
    ++c;
    if (M.flags & 2) break;
  }

  // ---- the last chunk's product, then the copies' sums into the first copy ----
  if (!wait_pv_done(c - 1)) return false;
  tc_fence_after();
  take_o(alpha_pend);
  // the other parity of the maximum exchange: its last readers (chunk c - 2)
  // have all passed chunk c - 1's barrier
  float *xl = xbuf + (c & 1) * (2 * kTcRows);
  xl[second * kTcRows + t] = l_run;
  // O sums travel through the P region (free: the item's last P V has
  // completed); 16-byte chunk j of exchange row r sits at chunk j ^ (r & 7)
  float *ox = reinterpret_cast<float *>(ps);  // [64][128] fp32
  auto ox_at = [&](int r, int j) { return reinterpret_cast<float4 *>(ox + r * kD) + (j ^ (r & 7)); };
#pragma unroll
  for (int step = kTcRows / 2; step >= kRep; step >>= 1) {
    if (t >= step && t < 2 * step) {
#pragma unroll
      for (int c4 = 0; c4 < 16; ++c4)
        *ox_at(t - step, 16 * second + c4) =
            make_float4(acc[4 * c4], acc[4 * c4 + 1], acc[4 * c4 + 2], acc[4 * c4 + 3]);
    }
    named_bar_sync(1, kCW * 32);
    if (t < step) {
#pragma unroll
      for (int c4 = 0; c4 < 16; ++c4) {
        const float4 v = *ox_at(t, 16 * second + c4);
        acc[4 * c4] += v.x;
        acc[4 * c4 + 1] += v.y;
        acc[4 * c4 + 2] += v.z;
        acc[4 * c4 + 3] += v.w;
      }
    }
    named_bar_sync(1, kCW * 32);
  }
  if (F == 1) named_bar_sync(1, kCW * 32);  // the row sums are visible
  if (t < kRep && real) {
    float l_tot = 0.f;
#pragma unroll
    for (int j = 0; j < F; ++j) l_tot += xl[row + j * kRep] + xl[kTcRows + row + j * kRep];
    if (I.n_split == 1) {
      const float inv = l_tot > 0.f ? 1.f / l_tot : 0.f;
      uint4 *orow = reinterpret_cast<uint4 *>(out_row(g, I, I.rb * kTcRows + row) + 64 * second);
#pragma unroll
      for (int c8 = 0; c8 < 8; ++c8) {
        uint4 v;
        v.x = pack_bf16x2(acc[8 * c8 + 0] * inv, acc[8 * c8 + 1] * inv);
        v.y = pack_bf16x2(acc[8 * c8 + 2] * inv, acc[8 * c8 + 3] * inv);
        v.z = pack_bf16x2(acc[8 * c8 + 4] * inv, acc[8 * c8 + 5] * inv);
        v.w = pack_bf16x2(acc[8 * c8 + 6] * inv, acc[8 * c8 + 7] * inv);
        orow[c8] = v;
      }
    } else {
      float *prow = p.partials + ((size_t)I.pbase + (size_t)I.split * I.rows + row) * kPStride;
#pragma unroll
      for (int c4 = 0; c4 < 16; ++c4)
        __stcg(reinterpret_cast<float4 *>(prow + 64 * second) + c4,
               make_float4(acc[4 * c4], acc[4 * c4 + 1], acc[4 * c4 + 2], acc[4 * c4 + 3]));
      if (second == 0) {
        __stcg(prow + 128, m_used);
        __stcg(prow + 129, l_tot);
      }
    }
  }
  // TMEM O and the exchange areas are free again once every thread is here
  tc_fence_before();
  named_bar_sync(1, kCW * 32);
  return true;
}

// ============================ CUDA-core path ============================
// Fewer than kTcMinRows rows; warp w takes pages w and w + 4 of every stage,
// lanes split a page's 16 keys in halves of the head dimension.
template <int NR>
__device__ __forceinline__ bool cc_item(const AttnParams &p, const CompCtx &X, const Item &I,
                                        uint32_t &it) {
  const ItemGeom g = item_geom(p, I);
  const Bars &B = X.B;
  const int warp = X.warp, lane = X.lane;
  float *qs = reinterpret_cast<float *>(X.smem + Smem::off_ccq);
  float *mg = reinterpret_cast<float *>(X.smem + Smem::off_merge);
  float *ps = reinterpret_cast<float *>(X.smem + Smem::off_ps);
  // NR rows known at compile time, or up to NR with run-time guards when NR == kCcRows
  const int nrow = NR < kCcRows ? NR : I.rows;
  float cm[NR], cl[NR], co[NR][4];

  for (bool first = true;; first = false) {
    const int s = it % kStages;
    if (!wait_or_abort(X, &B.full[s], (it / kStages) & 1)) return false;
    if (!wait_or_abort(X, &B.vfull[s], (it / kStages) & 1)) return false;
    const StageMeta M = X.meta[s];
    zero_tail(X, s, (it / kStages) & 1, M.page0, g.L, kCcW * 32, 3);
    if (first) {
      for (int e = X.ctid; e < nrow * (kD / 8); e += kCcW * 32) {
        const int rho = e / (kD / 8), c8 = e % (kD / 8);
        const int grow = I.rb * kCcRows + rho;
        const int qi = grow / g.G, j = grow % g.G;
        const uint4 raw = *reinterpret_cast<const uint4 *>(
            g.Bt->q + ((size_t)(g.q0 + qi) * g.hq + I.kvh * g.G + j) * kD + c8 * 8);
        float *dst = qs + rho * kD;
        const int d0 = c8 * 8;
        dst[q_slot(d0 + 0)] = bf16lo(raw.x);
        dst[q_slot(d0 + 1)] = bf16hi(raw.x);
        dst[q_slot(d0 + 2)] = bf16lo(raw.y);
        dst[q_slot(d0 + 3)] = bf16hi(raw.y);
        dst[q_slot(d0 + 4)] = bf16lo(raw.z);
        dst[q_slot(d0 + 5)] = bf16hi(raw.z);
        dst[q_slot(d0 + 6)] = bf16lo(raw.w);
        dst[q_slot(d0 + 7)] = bf16hi(raw.w);
      }
#pragma unroll
      for (int r = 0; r < NR; ++r) {
        cm[r] = -INFINITY;
        cl[r] = 0.f;
        co[r][0] = co[r][1] = co[r][2] = co[r][3] = 0.f;
      }
      named_bar_sync(3, kCcW * 32);
    }
#pragma unroll 1
    for (int jp = 0; jp < kStagePages / kCcW; ++jp) {
      const int pg = warp + kCcW * jp;  // pages warp, warp + 4 of the stage
      if (pg < M.npages) {
        const int key = lane >> 1, half = lane & 1;
        const int R = pg * kPage + key;  // key row within the stage
        const uint8_t *kb = kv_row(stage_k(X.smem, s), R, half);
        const uint8_t *vb = stage_v(X.smem, s);
        const int kpos = (M.page0 + pg) * kPage + key;
        const bool page_ok = !((M.invalid >> pg) & 1u);
        uint4 kr[8];
#pragma unroll
        for (int cc = 0; cc < 8; ++cc) {
          const int lc = (cc + 4 * half) & 7;  // logical chunk, rotated per half
          kr[cc] = *reinterpret_cast<const uint4 *>(kb + ((lc ^ (R & 7)) << 4));
        }
#pragma unroll
        for (int r = 0; r < NR; ++r) {
          if (r < nrow) {
            const float *qrow = qs + r * kD + half * 64;
            float pa[4] = {0.f, 0.f, 0.f, 0.f};  // four independent partial sums
#pragma unroll
            for (int cc = 0; cc < 8; ++cc) {
              const int lc = (cc + 4 * half) & 7;
              const float4 a = *reinterpret_cast<const float4 *>(qrow + lc * 4);
              const float4 b2 = *reinterpret_cast<const float4 *>(qrow + 32 + lc * 4);
              float &acc = pa[cc & 3];
              acc = fmaf(bf16lo(kr[cc].x), a.x, acc);
              acc = fmaf(bf16hi(kr[cc].x), a.y, acc);
              acc = fmaf(bf16lo(kr[cc].y), a.z, acc);
              acc = fmaf(bf16hi(kr[cc].y), a.w, acc);
              acc = fmaf(bf16lo(kr[cc].z), b2.x, acc);
              acc = fmaf(bf16hi(kr[cc].z), b2.y, acc);
              acc = fmaf(bf16lo(kr[cc].w), b2.z, acc);
              acc = fmaf(bf16hi(kr[cc].w), b2.w, acc);
            }
            float acc = (pa[0] + pa[1]) + (pa[2] + pa[3]);
            acc += __shfl_xor_sync(0xffffffffu, acc, 1);
            const int qi = (I.rb * kCcRows + r) / g.G;
            const bool vis = page_ok && kpos < g.L && kpos <= g.L - g.ql + qi;
            const float sc = vis ? acc * p.scale_log2 : -INFINITY;
            float mx = sc;
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
            const float mnew = fmaxf(cm[r], mx);
            float alpha = 1.f, pr = 0.f;
            if (mnew != -INFINITY) {
              alpha = exp2f(cm[r] - mnew);
              pr = exp2f(sc - mnew);
            }
            cl[r] = cl[r] * alpha + (half == 0 ? pr : 0.f);
            co[r][0] *= alpha;
            co[r][1] *= alpha;
            co[r][2] *= alpha;
            co[r][3] *= alpha;
            cm[r] = mnew;
            if (half == 0) ps[(warp * 8 + r) * 16 + key] = pr;
          }
        }
        __syncwarp();
        // P V: lane owns dims 4*lane .. 4*lane+3
        const int vhalf = lane >> 4, vc = (lane & 15) >> 1, vsub = (lane & 1) * 8;
#pragma unroll
        for (int jk = 0; jk < kPage; ++jk) {
          const int Rv = pg * kPage + jk;
          const uint2 vv = *reinterpret_cast<const uint2 *>(kv_row(vb, Rv, vhalf) +
                                                            ((vc ^ (Rv & 7)) << 4) + vsub);
          const float v0 = bf16lo(vv.x), v1 = bf16hi(vv.x), v2 = bf16lo(vv.y), v3 = bf16hi(vv.y);
#pragma unroll
          for (int r = 0; r < NR; ++r) {
            if (r < nrow) {
              const float pj = ps[(warp * 8 + r) * 16 + jk];
              co[r][0] = fmaf(pj, v0, co[r][0]);
              co[r][1] = fmaf(pj, v1, co[r][1]);
              co[r][2] = fmaf(pj, v2, co[r][2]);
              co[r][3] = fmaf(pj, v3, co[r][3]);
            }
          }
        }
      }
      __syncwarp();  // ps is rewritten by the next page
    }
    if (lane == 0) mbar_arrive(&B.empty[s]);
    ++it;
    if (M.flags & 2) break;
  }

  // ---- finalize: merge the four warps' page subsets ----
#pragma unroll
  for (int r = 0; r < NR; ++r)
    if (r < nrow) cl[r] = warp_sum(cl[r]);
#pragma unroll
  for (int r = 0; r < NR; ++r) {
    if (r < nrow) {
      float *dst = mg + (warp * 8 + r) * kPStride;
      *reinterpret_cast<float4 *>(dst + lane * 4) = make_float4(co[r][0], co[r][1], co[r][2], co[r][3]);
      if (lane == 0) {
        dst[128] = cm[r];
        dst[129] = cl[r];
      }
    }
  }
  named_bar_sync(3, kCcW * 32);
  if (warp == 0) {
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      if (r < nrow) {
        float Mx = -INFINITY;
        for (int w2 = 0; w2 < kCcW; ++w2) Mx = fmaxf(Mx, mg[(w2 * 8 + r) * kPStride + 128]);
        float Ls = 0.f, O0 = 0.f, O1 = 0.f, O2 = 0.f, O3 = 0.f;
        for (int w2 = 0; w2 < kCcW; ++w2) {
          const float *src = mg + (w2 * 8 + r) * kPStride;
          const float sc = (src[128] == -INFINITY) ? 0.f : exp2f(src[128] - Mx);
          const float4 ov = *reinterpret_cast<const float4 *>(src + lane * 4);
          Ls += src[129] * sc;
          O0 += ov.x * sc;
          O1 += ov.y * sc;
          O2 += ov.z * sc;
          O3 += ov.w * sc;
        }
        const int grow = I.rb * kCcRows + r;
        const int qi = grow / g.G, j = grow % g.G;
        if (I.n_split == 1) {
          const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
          uint2 pk;
          pk.x = (uint32_t)f2bf16(O0 * inv) | ((uint32_t)f2bf16(O1 * inv) << 16);
          pk.y = (uint32_t)f2bf16(O2 * inv) | ((uint32_t)f2bf16(O3 * inv) << 16);
          *reinterpret_cast<uint2 *>(g.Bt->out + ((size_t)(g.q0 + qi) * g.hq + I.kvh * g.G + j) * kD +
                                     lane * 4) = pk;
        } else {
          float *dst = p.partials + ((size_t)I.pbase + (size_t)I.split * I.rows + r) * kPStride;
          __stcg(reinterpret_cast<float4 *>(dst + lane * 4), make_float4(O0, O1, O2, O3));
          if (lane == 0) {
            __stcg(dst + 128, Mx);
            __stcg(dst + 129, Ls);
          }
        }
      }
    }
  }
  named_bar_sync(3, kCcW * 32);
  return true;
}

// Two-row tasks (GQA group 2 decode), the bulk of the CUDA-core work.  Warp
// w takes pages w and w + 4 of every stage (32 keys); lane = (k, q) with
// k = lane / 4 and q = lane % 4.
//   Q K^T: the lane holds dims 32q .. 32q + 31 of both query rows in fp32
//     registers and takes them against keys g * 8 + k, g = 0..3 (all K loads
//     in flight together); a butterfly over the four quarter lanes leaves lane
//     (k, q) with both rows' scores of key q * 8 + k (six shuffles).
//   P V: lane owns output dims 4 lane .. 4 lane + 3 of both rows; the
//     probabilities come back from shared memory as broadcasts.
// The warps' partial (m, l, O) are merged at the end of the item.
__device__ __forceinline__ bool cc2_item(const AttnParams &p, const CompCtx &X, const Item &I,
                                         uint32_t &it) {
  constexpr int NR = 2;
  const ItemGeom g = item_geom(p, I);
  const Bars &B = X.B;
  const int warp = X.warp, lane = X.lane;
  const int kq = lane >> 2, qq = lane & 3;
  float *mg = reinterpret_cast<float *>(X.smem + Smem::off_merge);
  float *pw = reinterpret_cast<float *>(X.smem + Smem::off_ps) + warp * 32 * NR;  // [32 keys][2]
  float qv[NR][32];
  int lim[NR];
#pragma unroll
  for (int r = 0; r < NR; ++r) {
    const int grow = I.rb * kCcRows + r;
    lim[r] = g.L - g.ql + grow / g.G;
    const uint4 *src = reinterpret_cast<const uint4 *>(q_row(g, I, grow) + qq * 32);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint4 v = __ldg(src + j);
      qv[r][8 * j + 0] = bf16lo(v.x);
      qv[r][8 * j + 1] = bf16hi(v.x);
      qv[r][8 * j + 2] = bf16lo(v.y);
      qv[r][8 * j + 3] = bf16hi(v.y);
      qv[r][8 * j + 4] = bf16lo(v.z);
      qv[r][8 * j + 5] = bf16hi(v.z);
      qv[r][8 * j + 6] = bf16lo(v.w);
      qv[r][8 * j + 7] = bf16hi(v.w);
    }
  }
  float cm[NR], cl[NR], co[NR][4];
#pragma unroll
  for (int r = 0; r < NR; ++r) {
    cm[r] = -INFINITY;
    cl[r] = 0.f;
    co[r][0] = co[r][1] = co[r][2] = co[r][3] = 0.f;
  }
  const int vhalf = lane >> 4, vc = (lane & 15) >> 1, vsub = (lane & 1) * 8;

  for (;;) {
    const int s = it % kStages;
    if (!wait_or_abort(X, &B.full[s], (it / kStages) & 1)) return false;
    if (!wait_or_abort(X, &B.vfull[s], (it / kStages) & 1)) return false;
    const StageMeta M = X.meta[s];
    zero_tail(X, s, (it / kStages) & 1, M.page0, g.L, kCcW * 32, 3);
    const uint8_t *kst = stage_k(X.smem, s);
    const uint8_t *vb = stage_v(X.smem, s);
    // ---- partial dot products of this lane's quarter for keys g * 8 + k ----
    float part[4][NR];
#pragma unroll
    for (int gg = 0; gg < 4; ++gg) {
      const int R = (warp + kCcW * (gg >> 1)) * kPage + (gg & 1) * 8 + kq;
      const uint8_t *kb = kv_row(kst, R, qq >> 1);
      uint4 kr[4];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        kr[j] = *reinterpret_cast<const uint4 *>(kb + (((4 * (qq & 1) + j) ^ (R & 7)) << 4));
#pragma unroll
      for (int r = 0; r < NR; ++r) {
        float a0 = 0.f, a1 = 0.f;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          a0 = fmaf(bf16lo(kr[j].x), qv[r][8 * j + 0], a0);
          a1 = fmaf(bf16hi(kr[j].x), qv[r][8 * j + 1], a1);
          a0 = fmaf(bf16lo(kr[j].y), qv[r][8 * j + 2], a0);
          a1 = fmaf(bf16hi(kr[j].y), qv[r][8 * j + 3], a1);
          a0 = fmaf(bf16lo(kr[j].z), qv[r][8 * j + 4], a0);
          a1 = fmaf(bf16hi(kr[j].z), qv[r][8 * j + 5], a1);
          a0 = fmaf(bf16lo(kr[j].w), qv[r][8 * j + 6], a0);
          a1 = fmaf(bf16hi(kr[j].w), qv[r][8 * j + 7], a1);
        }
        part[gg][r] = a0 + a1;
      }
    }
    // ---- butterfly over the quarters: lane keeps group qq ----
    const bool odd = qq & 1, up = qq >> 1;
    float half_sum[2][NR];
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int r = 0; r < NR; ++r) {
        const float send = odd ? part[2 * i][r] : part[2 * i + 1][r];
        const float keep = odd ? part[2 * i + 1][r] : part[2 * i][r];
        half_sum[i][r] = keep + __shfl_xor_sync(0xffffffffu, send, 1);
      }
    float sc[NR];
    const int pg = warp + kCcW * up;
    const int kpos = (M.page0 + pg) * kPage + (int)odd * 8 + kq;
    const bool page_ok = pg < M.npages && !((M.invalid >> pg) & 1u);
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      const float send = up ? half_sum[0][r] : half_sum[1][r];
      const float keep = up ? half_sum[1][r] : half_sum[0][r];
      const float tot = keep + __shfl_xor_sync(0xffffffffu, send, 2);
      sc[r] = (page_ok && kpos <= lim[r]) ? tot * p.scale_log2 : -INFINITY;
    }
    // ---- online softmax over the warp's 32 keys ----
    float pr[NR];
#pragma unroll
    for (int r = 0; r < NR; ++r) {
      const float mnew = fmaxf(cm[r], warp_max(sc[r]));
      const float alpha = mnew == -INFINITY ? 1.f : ex2_approx(cm[r] - mnew);
      pr[r] = mnew == -INFINITY ? 0.f : ex2_approx(sc[r] - mnew);
      cl[r] = fmaf(cl[r], alpha, pr[r]);
      co[r][0] *= alpha;
      co[r][1] *= alpha;
      co[r][2] *= alpha;
      co[r][3] *= alpha;
      cm[r] = mnew;
    }
    *reinterpret_cast<float2 *>(pw + (qq * 8 + kq) * NR) = make_float2(pr[0], pr[1]);
    __syncwarp();
    // ---- P V: 32 keys into this lane's 4 dims of both rows ----
#pragma unroll 8
    for (int key = 0; key < 32; ++key) {
      const int R = (warp + kCcW * (key >> 4)) * kPage + (key & 15);
      const uint2 vv = *reinterpret_cast<const uint2 *>(kv_row(vb, R, vhalf) +
                                                        ((vc ^ (R & 7)) << 4) + vsub);
      const float2 pk = *reinterpret_cast<const float2 *>(pw + key * NR);
      const float v0 = bf16lo(vv.x), v1 = bf16hi(vv.x), v2 = bf16lo(vv.y), v3 = bf16hi(vv.y);
      co[0][0] = fmaf(pk.x, v0, co[0][0]);
      co[0][1] = fmaf(pk.x, v1, co[0][1]);
      co[0][2] = fmaf(pk.x, v2, co[0][2]);
      co[0][3] = fmaf(pk.x, v3, co[0][3]);
      co[1][0] = fmaf(pk.y, v0, co[1][0]);
      co[1][1] = fmaf(pk.y, v1, co[1][1]);
      co[1][2] = fmaf(pk.y, v2, co[1][2]);
      co[1][3] = fmaf(pk.y, v3, co[1][3]);
    }
    __syncwarp();  // pw is rewritten at the next stage
    if (lane == 0) mbar_arrive(&B.empty[s]);
    ++it;
    if (M.flags & 2) break;
  }

  // ---- finalize: merge the four warps' partial results ----
#pragma unroll
  for (int r = 0; r < NR; ++r) cl[r] = warp_sum(cl[r]);
#pragma unroll
  for (int r = 0; r < NR; ++r) {
    float *dst = mg + (warp * 8 + r) * kPStride;
    *reinterpret_cast<float4 *>(dst + lane * 4) = make_float4(co[r][0], co[r][1], co[r][2], co[r][3]);
    if (lane == 0) {
      dst[128] = cm[r];
      dst[129] = cl[r];
    }
  }
  named_bar_sync(3, kCcW * 32);
  if (warp < NR) {  // warp r merges row r
    const int r = warp;
    float Mx = -INFINITY;
#pragma unroll
    for (int w2 = 0; w2 < kCcW; ++w2) Mx = fmaxf(Mx, mg[(w2 * 8 + r) * kPStride + 128]);
    float Ls = 0.f, O0 = 0.f, O1 = 0.f, O2 = 0.f, O3 = 0.f;
#pragma unroll
    for (int w2 = 0; w2 < kCcW; ++w2) {
      const float *src = mg + (w2 * 8 + r) * kPStride;
      const float sc = (src[128] == -INFINITY) ? 0.f : ex2_approx(src[128] - Mx);
      const float4 ov = *reinterpret_cast<const float4 *>(src + lane * 4);
      Ls = fmaf(src[129], sc, Ls);
      O0 = fmaf(ov.x, sc, O0);
      O1 = fmaf(ov.y, sc, O1);
      O2 = fmaf(ov.z, sc, O2);
      O3 = fmaf(ov.w, sc, O3);
    }
    const int grow = I.rb * kCcRows + r;
    if (I.n_split == 1) {
      const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
      uint2 pk;
      pk.x = pack_bf16x2(O0 * inv, O1 * inv);
      pk.y = pack_bf16x2(O2 * inv, O3 * inv);
      *reinterpret_cast<uint2 *>(out_row(g, I, grow) + lane * 4) = pk;
    } else {
      float *dst = p.partials + ((size_t)I.pbase + (size_t)I.split * I.rows + r) * kPStride;
      __stcg(reinterpret_cast<float4 *>(dst + lane * 4), make_float4(O0, O1, O2, O3));
      if (lane == 0) {
        __stcg(dst + 128, Mx);
        __stcg(dst + 129, Ls);
      }
    }
  }
  named_bar_sync(3, kCcW * 32);
  return true;
}

// A CUDA-core item runs on the first kCcW compute warps; the others release
// each of its stages (the stage's empty barrier counts every compute warp).
__device__ __forceinline__ bool pass_item(const CompCtx &X, uint32_t &it) {
  for (;;) {
    const int s = it % kStages;
    if (!wait_or_abort(X, &X.B.full[s], (it / kStages) & 1)) return false;
    const int flags = X.meta[s].flags;
    __syncwarp();
    if (X.lane == 0) mbar_arrive(&X.B.empty[s]);
    ++it;
    if (flags & 2) return true;
  }
}

__global__ void __launch_bounds__(kThreads, 1) attn_kernel(const __grid_constant__ AttnParams p) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const Bars B = bars(smem);
  StageMeta *meta = reinterpret_cast<StageMeta *>(smem + Smem::off_meta);
  // misc[0] TMEM base, [1] abort flag
  uint32_t *misc = reinterpret_cast<uint32_t *>(smem + Smem::off_misc);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the 128-byte swizzle atoms of TMA and tcgen05 assume 1024-byte alignment
  if (smem_u32(smem) & 1023u) {
    if (threadIdx.x == 0) ipd_set_error(&g_attn_err, IPD_DEVERR_PLAN);
    return;
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&B.full[s], 1);
      mbar_init(&B.vfull[s], 1);
      mbar_init(&B.empty[s], 2 + kCW);  // both MMA issuers and every compute warp
      // the P V of a tile of up to 64 rows, else the K producer (below)
      mbar_init(&B.vempty[s], 1);
    }
    mbar_init(B.q_ready, kCW);
    for (int i = 0; i < 2; ++i) mbar_init(&B.s_full[i], 1);
    mbar_init(B.p_full, kCW);
    mbar_init(B.p_free, 1);
    for (int i = 0; i < 2; ++i) mbar_init(&B.s_free[i], 1);
    for (int j = 0; j < kVJobs; ++j) mbar_init(&B.v_go[j], 1);
    misc[1] = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tc_alloc(&misc[0], kTmemCols);
    tc_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = misc[0];
  const int n_items = p.ctrl[0];

  if (warp >= kCW) {
  // the third warpgroup: producer, MMA issuer, and two warps that only take
  // part in the register split
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegsAux));
  if (warp == kProducerWarp) {
    // ------------------------------ producer ------------------------------
    // Page ids are read 32 at a time (one coalesced load per warp), one batch
    // ahead of use, and the next item's descriptor is fetched while the
    // current one streams, so no TMA issue waits on a global load.
    // When the planner split tasks into chunks of about equal size, the next
    // item is claimed four stages before the current one ends, so that the
    // CTA that frees up first takes it (2 % off a launch whose tasks split).
    // With whole tasks of very different sizes, claiming it as the current
    // one starts measured as good or better.
    const uint64_t policy = l2_policy_evict_first();
    uint32_t it = 0;
    bool aborted = false;
    // bit s: stage s's current use belongs to a 128-row tile or a CUDA-core
    // item.  Such a stage is released whole (a 128-row tile's by its P V: an
    // earlier refill of its K measured slower for these compute-bound tiles;
    // a CUDA-core item's by the compute warps, which read V themselves), and
    // this warp passes the V half of that release on to the V producer.
    uint32_t joint = 0;
    int *vjob = reinterpret_cast<int *>(smem + Smem::off_vjob);  // [kVJobs][16]
    // the next item's index: the atomic is issued at one stage and its value
    // taken at a later one, so that the producer does not wait for it
    int claim_v = 0;
    auto claim_issue = [&]() {
      if (lane == 0) claim_v = atomicAdd(&p.ctrl[1], 1);
    };
    auto claim_take = [&]() -> int { return __shfl_sync(0xffffffffu, claim_v, 0); };
    auto claim = [&]() -> int {
      claim_issue();
      return claim_take();
    };
    // hands stage use `i`'s V boxes (or a stop, tm < 0) to the V producer warp
    auto post_v = [&](uint32_t i, int w, int tm) {
      const int j = i % kVJobs;
      if (lane < kStagePages) vjob[16 * j + lane] = w;
      if (lane == 0) vjob[16 * j + 8] = tm;
      __syncwarp();
      if (lane == 0) mbar_arrive(&B.v_go[j]);
    };
    // page id of page `page_lo + 32 * batch + lane`, or -1 past the item
    auto load_ids = [&](const Item &I, int batch) -> int {
      const int pg = I.page_lo + 32 * batch + lane;
      if (pg >= I.page_hi) return -1;
      const BatchDev &Bp = p.b[I.b];
      return __ldg(Bp.page_table + (long long)I.r * Bp.max_pages + pg);
    };
    int idx = claim();
    Item I{};
    int ids = -1;
    if (idx < n_items) {
      I = p.items[idx];
      ids = load_ids(I, 0);
    }
    const bool late_claim = p.ctrl[4] != 0;
    while (idx < n_items) {
      int nxt = n_items;
      Item In = I;
      const BatchDev &Bt = p.b[I.b];
      const void *tk = &p.tmap[2 * Bt.cache];
      const int oob_w = (int)(Bt.num_pages * Bt.hkv * 2);  // a box here reads zeros
      const int npages = I.page_hi - I.page_lo;
      const int nst = (npages + kStagePages - 1) / kStagePages;
      int ids_next = (npages > 32) ? load_ids(I, 1) : -1;
      int ids_item_next = -1;
      const int st_claim = late_claim ? max(0, nst - 4) : 0;
      const int st_take = min(nst - 1, st_claim + 1);
      for (int st = 0; st < nst; ++st) {
        if (st == st_claim) claim_issue();
        if (st == st_take) {
          nxt = claim_take();
          if (nxt < n_items) In = p.items[nxt];  // consumed at the next item
        }
        if (st == max(st_take, nst - 2) && nxt < n_items) ids_item_next = load_ids(In, 0);
        const int rel = st * kStagePages;  // first page of the stage, relative to page_lo
        if (rel > 0 && (rel & 31) == 0) {   // move to the next batch of 32 ids
          ids = ids_next;
          ids_next = (rel + 32 < npages) ? load_ids(I, (rel >> 5) + 1) : -1;
        }
        const int page = I.page_lo + rel;
        const int np = min(kStagePages, npages - rel);
        const int s = it % kStages;
        const uint32_t ph = (it / kStages) & 1;
        const int pid = __shfl_sync(0xffffffffu, ids, (rel & 31) + (lane & (kStagePages - 1)));
        if (!mbar_wait_bounded(&B.empty[s], ph ^ 1)) {
          ipd_set_error(&g_attn_err, IPD_DEVERR_WAIT);
          aborted = true;
          break;
        }
        if (lane == 0 && ((joint >> s) & 1)) mbar_arrive(&B.vempty[s]);
        joint = (joint & ~(1u << s)) |
                ((I.path == kPathTc1 || I.path == kPathCc ? 1u : 0u) << s);
        int w = oob_w;
        bool ok = false;
        if (lane < np) {
          ok = pid >= 0 && (long long)pid < Bt.num_pages;
          if (!ok) ipd_set_error(&g_attn_err, IPD_DEVERR_PAGE_ID);
          else w = (pid * Bt.hkv + I.kvh) * 2;
        }
        const uint32_t okmask = __ballot_sync(0xffffffffu, ok);
        if (lane == 0) {
          StageMeta m;
          m.item = idx;
          m.page0 = page;
          m.npages = np;
          m.flags = (st == 0 ? 1 : 0) | (st == nst - 1 ? 2 : 0);
          m.invalid = (~okmask) & ((1u << np) - 1u);
          m.path = I.path;
          meta[s] = m;
          mbar_arrive_expect_tx(&B.full[s], kTensorBytes);
        }
        post_v(it, w, 2 * Bt.cache + 1);
        if (lane < kStagePages)  // every page slot is written (zeros past the item)
          tma_load_4d(stage_k(smem, s) + lane * kPageBytes, tk, 0, 0, 0, w, &B.full[s], policy);
        ++it;
      }
      if (nst == 0 && !aborted) {  // (the planner emits no empty item)
        nxt = claim();
        if (nxt < n_items) {
          In = p.items[nxt];
          ids_item_next = load_ids(In, 0);
        }
      }
      if (aborted) break;
      idx = nxt;
      if (idx < n_items) {
        I = In;
        ids = ids_item_next;
      }
    }
    if (!aborted) {
      const int s = it % kStages;
      const uint32_t ph = (it / kStages) & 1;
      if (mbar_wait_bounded(&B.empty[s], ph ^ 1)) {
        post_v(it, 0, -1);
        if (lane == 0) {
          meta[s].item = -1;
          mbar_arrive(&B.full[s]);
        }
      } else {
        ipd_set_error(&g_attn_err, IPD_DEVERR_WAIT);
        aborted = true;
      }
    }
    // (stage use `it` has not been handed over: its v_go phase is free)
    if (aborted) post_v(it, 0, -1);
    if (aborted) {
      // the consumers stopped: let this CTA's copies land before exiting
      if (lane == 0) atomicExch(&misc[1], 1u);
      for (uint32_t k = (it > (uint32_t)kStages ? it - kStages : 0); k < it; ++k)
        (void)mbar_wait_bounded(&B.full[k % kStages], (k / kStages) & 1);
    }
    return;
  }

  if (warp == kVLoadWarp) {
    // ---------------------------- V producer -------------------------------
    // Issues each stage's V boxes as the K producer hands them over, once the
    // stage's V slot is free (its previous P V done).
    const uint64_t policy = l2_policy_evict_first();
    const int *vjob = reinterpret_cast<const int *>(smem + Smem::off_vjob);
    uint32_t it = 0;
    bool aborted = false;
    for (;; ++it) {
      const int s = it % kStages, j = it % kVJobs;
      if (!mbar_wait_bounded(&B.v_go[j], (it / kVJobs) & 1)) {
        aborted = true;
        break;
      }
      const int tm = vjob[16 * j + 8];
      if (tm < 0) break;
      if (!mbar_wait_bounded(&B.vempty[s], ((it / kStages) & 1) ^ 1)) {
        aborted = true;
        break;
      }
      if (lane == 0) mbar_arrive_expect_tx(&B.vfull[s], kTensorBytes);
      __syncwarp();
      if (lane < kStagePages)
        tma_load_4d(stage_v(smem, s) + lane * kPageBytes, &p.tmap[tm], 0, 0, 0,
                    vjob[16 * j + lane], &B.vfull[s], policy);
    }
    if (aborted) {
      ipd_set_error(&g_attn_err, IPD_DEVERR_WAIT);
      if (lane == 0) atomicExch(&misc[1], 1u);
    }
    if (aborted || *(volatile uint32_t *)&misc[1]) {
      // the consumers stopped: let this CTA's copies land before exiting
      for (uint32_t k = (it > (uint32_t)kStages ? it - kStages : 0); k < it; ++k)
        (void)mbar_wait_bounded(&B.vfull[k % kStages], (k / kStages) & 1);
    }
    return;
  }

  if (warp == kMmaWarp || warp == kPvWarp) {
    // ----------------------------- MMA issuers ------------------------------
    // Both issuers walk the same stages.  Warp kMmaWarp issues Q K^T of
    // tensor chunk j into S buffer j & 1 as soon as its stage has landed (and
    // the buffer's previous chunk, j - 2, has had its P V); warp kPvWarp
    // issues P V of chunk j once its P is written and its V has landed, and
    // releases the stage's V (a 128-row tile's whole stage).
    constexpr uint32_t idesc_s = idesc_bf16_f32(kTcRows, kStageKeys, 0);
    constexpr uint32_t idesc_o = idesc_bf16_f32(kTcRows, kD, 1);
    const uint32_t pa = smem_u32(smem + Smem::off_p);
    const bool is_qk = warp == kMmaWarp;
    uint32_t it = 0, c = 0, nq = 0;
    bool ok = true;
    auto mwait = [&](uint64_t *bar, uint32_t par) -> bool {
      if (mbar_wait_bounded(bar, par)) return true;
      ok = false;
      return false;
    };
    for (;;) {
      const int s = it % kStages;
      if (!mwait(&B.full[s], (it / kStages) & 1)) break;
      int item = 0, flags = 0, path = 0;
      if (lane == 0) {
        item = meta[s].item;
        flags = meta[s].flags;
        path = meta[s].path;
      }
      item = __shfl_sync(0xffffffffu, item, 0);
      flags = __shfl_sync(0xffffffffu, flags, 0);
      path = __shfl_sync(0xffffffffu, path, 0);
      if (item < 0 || *(volatile uint32_t *)&misc[1]) break;
      // the P V issuer has read the stage's metadata (the K producer may
      // rewrite it once the K slot is free)
      if (!is_qk && lane == 0 && path != kPathTc1) mbar_arrive(&B.empty[s]);
      if (path == kPathCc) {
        if (is_qk && lane == 0) mbar_arrive(&B.empty[s]);
        __syncwarp();
        ++it;
        continue;
      }
      if (is_qk) {
        if (flags & 1) {  // a new tensor item: its Q tile must be written
          if (!mwait(B.q_ready, nq & 1)) break;
          ++nq;
        }
        // the S buffer's previous chunk has had its P V (which for 128-row
        // tiles reads two terms of P from it)
        if (c >= 2 && !mwait(&B.s_free[c & 1], ((c >> 1) - 1) & 1)) break;
        tc_fence_after();
        if (lane == 0) {
          // K dims 16kk.. (K-major: 64-dim halves 1 KB apart, 8-key groups 2 KB)
          const uint64_t bd0 = sdesc_sw128(smem_u32(stage_k(smem, s)), 16, kGroupBytes);
          const uint32_t sd = tmem + col_s(c & 1);
          if (path == kPathTc1) {
            // Q dims 16kk.. in shared memory (K-major: 64-dim halves 16 KB
            // apart, 8-row groups 1 KB)
            const uint64_t ad0 = sdesc_sw128(pa, 16, 1024);
#pragma unroll
            for (int kk = 0; kk < kD / 16; ++kk) {
              const uint64_t bd = bd0 + (uint64_t)(((kk >> 2) * kAtomBytes + (kk & 3) * 32) >> 4);
              const uint64_t ad = sdesc_advance(ad0, (kk >> 2) * Smem::kPHalf + (kk & 3) * 32);
              tc_mma_bf16(sd, ad, bd, idesc_s, kk > 0);
            }
          } else {
            // Q dims 16kk.. are TMEM columns 8kk.. of the Q tile
#pragma unroll
            for (int kk = 0; kk < kD / 16; ++kk) {
              const uint64_t bd = bd0 + (uint64_t)(((kk >> 2) * kAtomBytes + (kk & 3) * 32) >> 4);
              tc_mma_bf16_ta(sd, tmem + kColQ + 8 * kk, bd, idesc_s, kk > 0);
            }
          }
          tc_commit(&B.s_full[c & 1]);
          if (path != kPathTc1) tc_commit(&B.empty[s]);  // Q K^T has read the stage's K
          else mbar_arrive(&B.empty[s]);
        }
        __syncwarp();
      } else {
        if (!mwait(B.p_full, c & 1)) break;
        if (!mwait(&B.vfull[s], (it / kStages) & 1)) break;
        tc_fence_after();
        if (lane == 0) {
          // V keys 16kk.. as an MN-major operand: 64-dim halves 1 KB apart,
          // 8-key groups 2 KB; the descriptor of step kk + 1 is that of kk with
          // its start address 4 KB further
          uint64_t bd = sdesc_sw128(smem_u32(stage_v(smem, s)), kAtomBytes, kGroupBytes);
          constexpr uint64_t kVStep = (2 * kGroupBytes) >> 4;
          if (path == kPathTc1) {
            // the three terms of P: two in the chunk's S buffer, the third in
            // the columns of its parity
            const uint32_t pt = tmem + col_s(c & 1), p3 = tmem + t3_col_full(c & 1, 0);
#pragma unroll
            for (int kk = 0; kk < kStageKeys / 16; ++kk, bd += kVStep) {
              tc_mma_bf16_ta(tmem + kColO, pt + p_col(kk, 1), bd, idesc_o, kk == 0 ? 0u : 1u);
              tc_mma_bf16_ta(tmem + kColO, pt + p_col(kk, 2), bd, idesc_o, 1u);
              tc_mma_bf16_ta(tmem + kColO, p3 + 8 * kk, bd, idesc_o, 1u);
            }
          } else {
            // the stacked terms in the shared-memory P operand (K-major:
            // 64-key halves 16 KB apart, 8-row groups 1 KB), and for tiles of
            // up to 64 rows the third term from TMEM
            const uint64_t ad0 = sdesc_sw128(pa, 16, 1024);
            const bool t3 = path == kPathTc2;
#pragma unroll
            for (int kk = 0; kk < kStageKeys / 16; ++kk, bd += kVStep) {
              const uint64_t ad = sdesc_advance(ad0, (kk >> 2) * Smem::kPHalf + (kk & 3) * 32);
              tc_mma_bf16(tmem + kColO, ad, bd, idesc_o, kk == 0 ? 0u : 1u);
              if (t3) tc_mma_bf16_ta(tmem + kColO, tmem + t3_col(kk), bd, idesc_o, 1u);
            }
          }
          tc_commit(B.p_free);
          tc_commit(&B.s_free[c & 1]);
          tc_commit(path == kPathTc1 ? &B.empty[s] : &B.vempty[s]);
        }
        __syncwarp();
      }
      ++c;
      ++it;
    }
    if (!ok) {
      ipd_set_error(&g_attn_err, IPD_DEVERR_WAIT);
      atomicExch(&misc[1], 1u);
    }
    // every tensor-core op and TMEM access is finished before TMEM is released
    tc_fence_before();
    named_bar_sync(2, (kCW + 2) * 32);
    tc_fence_after();
    if (is_qk) tc_dealloc(tmem, kTmemCols);
    return;
  }

  return;
  }

  // -------------------------------- compute warps --------------------------------
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(kRegsCompute));
  const CompCtx X{smem, B, meta, misc, tmem, warp, lane, (int)threadIdx.x};
  uint32_t it = 0, c = 0;
  for (;;) {
    const int s = it % kStages;
    if (!wait_or_abort(X, &B.full[s], (it / kStages) & 1)) break;
    const StageMeta M = meta[s];
    if (M.item < 0 || *(volatile uint32_t *)&misc[1]) break;
    const Item I = p.items[M.item];
    bool ok;
    if (I.path != kPathCc) {
      // copies of the tile's rows over the 128 lanes: 4 (<= 32 rows), 2 (<= 64) or 1
      if (I.path == kPathTc4) ok = tc_item<4>(p, X, I, it, c);
      else if (I.path == kPathTc2) ok = tc_item<2>(p, X, I, it, c);
      else ok = tc_item<1>(p, X, I, it, c);
    } else if (warp < kCcW) {
      // GQA-2 decode (two rows) has its own layout; other sizes take the
      // guarded loop
      if (I.rows == 2) ok = cc2_item(p, X, I, it);
      else ok = cc_item<kCcRows>(p, X, I, it);
    } else {
      ok = pass_item(X, it);  // the other warps only release the item's stages
    }
    if (!ok) break;
    if (I.n_split > 1) {
      // The last of a split task's items to finish merges the task's
      // partials.  Every thread's partial rows are made visible device-wide
      // before one thread counts the item; the CTA that completes the count
      // reads every split's rows (its own and other CTAs') from L2.
      __threadfence();
      named_bar_sync(1, kCW * 32);
      if (threadIdx.x == 0)
        misc[2] = atomicAdd(&p.split_done[I.task], 1) == I.n_split - 1 ? 1u : 0u;
      named_bar_sync(1, kCW * 32);
      if (*(volatile uint32_t *)&misc[2]) {
        __threadfence();
        for (int r = warp; r < I.rows; r += kCW) merge_split_row(p, I, r, lane);
      }
      named_bar_sync(1, kCW * 32);  // misc[2] is read before the next split item rewrites it
    }
  }
  tc_fence_before();
  named_bar_sync(2, (kCW + 2) * 32);
}

// --------------------------------------------------------------------------
// host launch
// --------------------------------------------------------------------------
struct DevInfo {
  int sms = 0;
  bool attr_set = false;
};
DevInfo g_dev[64];

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int get_encoder() {
  if (g_encode) return IPD_OK;
  void *fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                       &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || !fn)
    return IPD_ERR_CUDA;
  g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  return IPD_OK;
}

// A pool [num_pages][Hkv][16][128] bf16 seen as a 4-D tensor (x: 64 dims,
// y: 8 rows 256 B apart, z: 2 halves 128 B apart, w: 8-row groups 2 KB
// apart), 128-byte swizzle; a box (64, 8, 2, 2) is one page of one kv head
// in the stage layout (two groups, each as its two halves).
int encode_pool(CUtensorMap *m, const void *base, long long rows) {
  cuuint64_t dims[4] = {64, 8, 2, (cuuint64_t)(rows / 8)};
  cuuint64_t strides[3] = {(cuuint64_t)kD * 2, 128, (cuuint64_t)kGroupBytes};
  cuuint32_t box[4] = {64, 8, 2, 2};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  const CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base),
                              dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? IPD_OK : IPD_ERR_CUDA;
}

// Optional timing of the attention kernel alone (a measurement aid): CUDA
// events recorded on the call's stream around each attn_kernel launch.
struct KernelTiming {
  bool on = false;
  int n = 0;
  cudaEvent_t ev[2 * 4096] = {};
};
KernelTiming g_timing;

int launch(const ipd_attn_batch *const *bs, int n, float scale, void *ws, size_t ws_bytes,
           cudaStream_t stream) {
  if (!(scale > 0.f) || scale != scale) return IPD_ERR_INVALID_ARG;
  const WsLayout W = layout(bs, n);
  if (W.total_reqs == 0) return IPD_OK;
  if (!ws || ws_bytes < W.total || ((uintptr_t)ws & 255)) return IPD_ERR_WORKSPACE;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return IPD_ERR_CUDA;
  DevInfo &D = g_dev[dev];
  if (!D.attr_set) {
    if (cudaDeviceGetAttribute(&D.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return IPD_ERR_CUDA;
    if (cudaFuncSetAttribute(attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             Smem::total) != cudaSuccess)
      return IPD_ERR_CUDA;
    D.attr_set = true;
  }
  if (get_encoder() != IPD_OK) return IPD_ERR_CUDA;
  AttnParams P;
  memset(&P, 0, sizeof(P));
  P.n_batches = n;
  const ipd_kv_cache *caches[IPD_MAX_BATCHES];
  int n_caches = 0;
  int base = 0;
  for (int i = 0; i < n; ++i) {
    const ipd_attn_batch *b = bs[i];
    int ci = 0;
    while (ci < n_caches && !(caches[ci]->k_pages == b->cache->k_pages &&
                              caches[ci]->v_pages == b->cache->v_pages &&
                              caches[ci]->num_pages == b->cache->num_pages &&
                              caches[ci]->num_kv_heads == b->cache->num_kv_heads))
      ++ci;
    if (ci == n_caches) {
      caches[n_caches++] = b->cache;
      const long long rows = b->cache->num_pages * b->cache->num_kv_heads * kPage;
      if (encode_pool(&P.tmap[2 * ci], b->cache->k_pages, rows) != IPD_OK ||
          encode_pool(&P.tmap[2 * ci + 1], b->cache->v_pages, rows) != IPD_OK)
        return IPD_ERR_CUDA;
    }
    BatchDev &Bd = P.b[i];
    Bd.q = b->q;
    Bd.out = b->out;
    Bd.cu_q = b->cu_q;
    Bd.seq_len = b->seq_len;
    Bd.page_table = b->page_table;
    Bd.num_pages = b->cache->num_pages;
    Bd.num_reqs = b->num_reqs;
    Bd.hq = b->num_q_heads;
    Bd.hkv = b->cache->num_kv_heads;
    Bd.group = Bd.hq / Bd.hkv;
    Bd.max_pages = b->max_pages;
    Bd.max_q_len = b->max_q_len;
    Bd.total_q = b->total_q;
    Bd.cache = ci;
    P.req_base[i] = base;
    base += b->num_reqs;
  }
  P.req_base[n] = base;
  P.total_reqs = base;
  P.scale_log2 = scale * kLog2e;
  uint8_t *w = static_cast<uint8_t *>(ws);
  P.ctrl = reinterpret_cast<int *>(w + W.off_ctrl);
  P.reqinfo = reinterpret_cast<int4 *>(w + W.off_reqinfo);
  P.items = reinterpret_cast<Item *>(w + W.off_items);
  P.reqslot = reinterpret_cast<int2 *>(w + W.off_reqslot);
  P.split_done = reinterpret_cast<int *>(w + W.off_done);
  P.partials = reinterpret_cast<float *>(w + W.off_partials);
  P.item_cap = W.item_cap;
  P.task_cap = W.task_cap;
  P.prow_cap = W.prow_cap;
  P.target_items = std::min(kMaxTargetItems, kTargetItemsPerSm * D.sms);
  P.n_sms = D.sms;

  // a small planner block fits beside row-pass CTAs already on an SM, so a
  // step that runs both at once does not hold the attention back
  if (W.total_reqs <= 256 * kPlanCache)
    attn_plan_kernel<256><<<1, 256, 0, stream>>>(P);
  else
    attn_plan_kernel<kPlanThreads><<<1, kPlanThreads, 0, stream>>>(P);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  const int grid = std::max(1, std::min(D.sms, W.item_cap));
  const bool timed = g_timing.on && g_timing.n < 4096;
  if (timed) {
    cudaEvent_t *e = &g_timing.ev[2 * g_timing.n];
    if ((!e[0] && cudaEventCreate(&e[0]) != cudaSuccess) ||
        (!e[1] && cudaEventCreate(&e[1]) != cudaSuccess) ||
        cudaEventRecord(e[0], stream) != cudaSuccess)
      return IPD_ERR_CUDA;
  }
  attn_kernel<<<grid, kThreads, Smem::total, stream>>>(P);
  if (timed) {
    if (cudaEventRecord(g_timing.ev[2 * g_timing.n + 1], stream) != cudaSuccess)
      return IPD_ERR_CUDA;
    ++g_timing.n;
  }
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}

}  // namespace

extern "C" __attribute__((visibility("hidden"))) unsigned int ipd_internal_take_attn_error() {
  unsigned int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_attn_err, sizeof(v)) != cudaSuccess) return 0xffffffffu;
  if (cudaMemcpyToSymbol(g_attn_err, &z, sizeof(z)) != cudaSuccess) return 0xffffffffu;
  return v;
}

extern "C" size_t ipd_attn_workspace_size(const ipd_attn_batch *verify, int n_verify,
                                          const ipd_attn_batch *decode, int n_decode) {
  const ipd_attn_batch *bs[IPD_MAX_BATCHES];
  if (collect(verify, n_verify, decode, n_decode, bs) != IPD_OK) return 0;
  return layout(bs, n_verify + n_decode).total;
}

extern "C" int ipd_verify_attn(const ipd_attn_batch *verify, int n_verify,
                               const ipd_attn_batch *decode, int n_decode, float softmax_scale,
                               void *workspace, size_t workspace_bytes, ipd_stream_t stream) {
  const ipd_attn_batch *bs[IPD_MAX_BATCHES];
  const int st = collect(verify, n_verify, decode, n_decode, bs);
  if (st != IPD_OK) return st;
  return launch(bs, n_verify + n_decode, softmax_scale, workspace, workspace_bytes,
                reinterpret_cast<cudaStream_t>(stream));
}

extern "C" int ipd_decode_attn(const ipd_attn_batch *decode, int n_decode, float softmax_scale,
                               void *workspace, size_t workspace_bytes, ipd_stream_t stream) {
  return ipd_verify_attn(nullptr, 0, decode, n_decode, softmax_scale, workspace, workspace_bytes,
                         stream);
}

extern "C" int ipd_set_attn_kernel_timing(int on) {
  g_timing.on = on != 0;
  g_timing.n = 0;
  return IPD_OK;
}

extern "C" int ipd_attn_kernel_time(double *total_ms, int *launches) {
  if (!total_ms || !launches) return IPD_ERR_INVALID_ARG;
  double sum = 0.0;
  for (int i = 0; i < g_timing.n; ++i) {
    float ms = 0.f;
    if (cudaEventSynchronize(g_timing.ev[2 * i + 1]) != cudaSuccess ||
        cudaEventElapsedTime(&ms, g_timing.ev[2 * i], g_timing.ev[2 * i + 1]) != cudaSuccess)
      return IPD_ERR_CUDA;
    sum += ms;
  }
  *total_ms = sum;
  *launches = g_timing.n;
  g_timing.n = 0;
  return IPD_OK;
}
