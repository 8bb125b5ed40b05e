// Paged span-verify attention and proposer decode attention, co-launched.
//
// Sec. 3.2.3 (verification stage): each verifier evaluates the k_r unverified
// draft tokens of a request in one prefill pass over its own cache; only the
// new tokens are computed (their K/V are already in the cache).  Proposal
// stage: the proposer decodes one token over its own cache.  Both run here as
// one persistent launch over both caches, whose GQA shapes differ.
//
// Work decomposition (device side, no host round trip):
//   task  = (batch, request, kv head, row block of <= kRowsCuda query rows)
//   item  = (task, KV chunk); long tasks are split into chunks so that the
//           work list has about kTargetItems items, and split partials are
//           merged by the last CTA to finish a task (atomic ticket, no wait).
// A row is one (query, query head) pair of a task: row = i * G + j for span
// query i and head kvh * G + j.
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>

#include <algorithm>

#include "common.cuh"

IPD_DECLARE_ERROR_WORD(g_attn_err);

namespace {

constexpr int kPage = 16;
constexpr int kD = 128;
constexpr int kTileBytes = kPage * kD * 2;  // one page of one KV head: 4 KB
constexpr int kRowsCuda = 64;               // rows per item
constexpr int kPPS = 8;                     // pages per pipeline stage
constexpr int kStages = 2;
constexpr int kCW = 8;                      // consumer warps
constexpr int kThreads = (kCW + 1) * 32;    // + one producer warp
constexpr int kTargetItems = 2048;
constexpr int kMinChunkPages = 16;
constexpr int kSplitMax = 16;
constexpr int kPStride = 132;               // floats per partial row: o[128], m, l, pad

struct BatchDev {
  const uint16_t *q;
  uint16_t *out;
  const int *cu_q;
  const int *seq_len;
  const int *page_table;
  const uint16_t *k_pages;
  const uint16_t *v_pages;
  long long num_pages;
  int num_reqs, hq, hkv, group, max_pages, max_q_len, total_q;
};

struct Item {
  int b, r, kvh, rb;
  int split, n_split, page_lo, page_hi;
  int task, pbase, rows, pad;
};

struct AttnParams {
  BatchDev b[IPD_MAX_BATCHES];
  int req_base[IPD_MAX_BATCHES + 1];
  int n_batches;
  int total_reqs;
  float scale_log2;
  int *ctrl;       // [0] n_items, [1] dynamic item counter, [2] n_tasks, [3] partial rows
  int4 *reqinfo;   // per flattened request: item offset, task offset, partial offset, n_split
  Item *items;
  int *tickets;
  float *partials;
  int item_cap, task_cap;
  long long prow_cap;
};

struct StageMeta {
  int item;
  int page0;
  int npages;
  int flags;        // 1 = first stage of its item, 2 = last stage
  uint32_t invalid; // pages of the stage whose id failed validation
  int pad[3];
};

// --------------------------------------------------------------------------
// host-side sizes
// --------------------------------------------------------------------------
struct WsLayout {
  size_t off_ctrl, off_reqinfo, off_items, off_tickets, off_partials, total;
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
  if (b->num_q_heads / c->num_kv_heads > kRowsCuda) return IPD_ERR_UNSUPPORTED;
  if (b->num_reqs < 0 || b->total_q < 0 || b->max_q_len < 0 || b->max_seq_len < 0)
    return IPD_ERR_INVALID_ARG;
  if (b->num_reqs == 0) return IPD_OK;
  if (b->max_q_len < 1 || b->max_seq_len < b->max_q_len) return IPD_ERR_INVALID_ARG;
  if ((long long)b->max_pages * kPage < b->max_seq_len) return IPD_ERR_INVALID_ARG;
  if (c->num_pages < 1) return IPD_ERR_INVALID_ARG;
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
    int st = validate_batch(out[i]);
    if (st != IPD_OK) return st;
  }
  return IPD_OK;
}

WsLayout layout(const ipd_attn_batch *const *bs, int n) {
  WsLayout L{};
  long long task_cap = 0, rows_all = 0;
  int reqs = 0;
  for (int i = 0; i < n; ++i) {
    const ipd_attn_batch *b = bs[i];
    int G = b->num_q_heads / b->cache->num_kv_heads;
    long long nrb = ((long long)b->max_q_len * G + kRowsCuda - 1) / kRowsCuda;
    task_cap += (long long)b->num_reqs * b->cache->num_kv_heads * nrb;
    rows_all += (long long)b->total_q * b->num_q_heads;
    reqs += b->num_reqs;
  }
  long long item_cap = task_cap + 2LL * kTargetItems;
  long long prow_cap = std::min<long long>(2LL * kTargetItems * kRowsCuda, kSplitMax * rows_all);
  L.item_cap = (int)std::min<long long>(item_cap, 1LL << 30);
  L.task_cap = (int)std::min<long long>(task_cap, 1LL << 30);
  L.prow_cap = prow_cap;
  L.total_reqs = reqs;
  size_t off = 0;
  L.off_ctrl = off;
  off = align_up(off + 64, 256);
  L.off_reqinfo = off;
  off = align_up(off + (size_t)reqs * sizeof(int4), 256);
  L.off_items = off;
  off = align_up(off + (size_t)L.item_cap * sizeof(Item), 256);
  L.off_tickets = off;
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
  int ql, L, pages, rows, nrb, ok;
};

__device__ ReqShape req_shape(const AttnParams &p, int b, int r) {
  const BatchDev &B = p.b[b];
  ReqShape s{};
  int c0 = B.cu_q[r], c1 = B.cu_q[r + 1];
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
    s.ql = 0; s.L = 0; s.pages = 0; s.rows = 0; s.nrb = 0;
    return s;
  }
  s.pages = (s.L + kPage - 1) / kPage;
  s.rows = s.ql * B.group;
  s.nrb = (s.rows + kRowsCuda - 1) / kRowsCuda;
  return s;
}

template <typename T>
__device__ T block_sum(T v, T *red) {
  int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
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

// exclusive scan of three ints across the block; returns totals in tot
__device__ void block_scan3(int3 v, int3 &excl, int3 &tot, int3 *sh) {
  int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int3 inc = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int x = __shfl_up_sync(0xffffffffu, inc.x, o);
    int y = __shfl_up_sync(0xffffffffu, inc.y, o);
    int z = __shfl_up_sync(0xffffffffu, inc.z, o);
    if (lane >= o) { inc.x += x; inc.y += y; inc.z += z; }
  }
  __syncthreads();
  if (lane == 31) sh[w] = inc;
  __syncthreads();
  int3 base = make_int3(0, 0, 0);
  tot = make_int3(0, 0, 0);
  for (int i = 0; i < nw; ++i) {
    if (i < w) { base.x += sh[i].x; base.y += sh[i].y; base.z += sh[i].z; }
    tot.x += sh[i].x; tot.y += sh[i].y; tot.z += sh[i].z;
  }
  excl = make_int3(base.x + inc.x - v.x, base.y + inc.y - v.y, base.z + inc.z - v.z);
  __syncthreads();
}

__global__ void __launch_bounds__(1024) attn_plan_kernel(const __grid_constant__ AttnParams p) {
  __shared__ long long red[32];
  __shared__ int3 sh3[32];
  __shared__ int s_fail;
  const int tid = threadIdx.x;
  if (tid == 0) s_fail = 0;

  long long w = 0;
  for (int gi = tid; gi < p.total_reqs; gi += blockDim.x) {
    int b = find_batch(p, gi);
    ReqShape s = req_shape(p, b, gi - p.req_base[b]);
    w += (long long)s.pages * p.b[b].hkv * s.nrb;
  }
  long long W = block_sum<long long>(w, red);
  long long chunk = (W + kTargetItems - 1) / kTargetItems;
  if (chunk < kMinChunkPages) chunk = kMinChunkPages;

  int3 carry = make_int3(0, 0, 0);
  for (int base = 0; base < p.total_reqs; base += blockDim.x) {
    int gi = base + tid;
    int3 cnt = make_int3(0, 0, 0);
    int nsplit = 1;
    if (gi < p.total_reqs) {
      int b = find_batch(p, gi);
      ReqShape s = req_shape(p, b, gi - p.req_base[b]);
      if (s.pages > 0) {
        long long ns = (s.pages + chunk - 1) / chunk;
        nsplit = (int)(ns < kSplitMax ? ns : kSplitMax);
        int tasks = p.b[b].hkv * s.nrb;
        cnt = make_int3(tasks * nsplit, tasks, nsplit > 1 ? nsplit * p.b[b].hkv * s.rows : 0);
      }
    }
    int3 ex, tot;
    block_scan3(cnt, ex, tot, sh3);
    if (gi < p.total_reqs)
      p.reqinfo[gi] = make_int4(carry.x + ex.x, carry.y + ex.y, carry.z + ex.z, nsplit);
    carry.x += tot.x; carry.y += tot.y; carry.z += tot.z;
  }
  if (tid == 0) {
    if (carry.x > p.item_cap || carry.y > p.task_cap || carry.z > p.prow_cap) {
      ipd_set_error(&g_attn_err, IPD_DEVERR_PLAN);
      s_fail = 1;
    }
    p.ctrl[0] = s_fail ? 0 : carry.x;
    p.ctrl[1] = 0;
    p.ctrl[2] = carry.y;
    p.ctrl[3] = carry.z;
  }
  __syncthreads();
  if (s_fail) return;

  for (int gi = tid; gi < p.total_reqs; gi += blockDim.x) {
    int b = find_batch(p, gi);
    int r = gi - p.req_base[b];
    ReqShape s = req_shape(p, b, r);
    if (s.pages == 0) continue;
    int4 info = p.reqinfo[gi];
    int item = info.x, task = info.y, ns = info.w;
    int per = (s.pages + ns - 1) / ns;
    for (int kvh = 0; kvh < p.b[b].hkv; ++kvh) {
      for (int rb = 0; rb < s.nrb; ++rb) {
        int rows = min(kRowsCuda, s.rows - rb * kRowsCuda);
        int pbase = ns > 1 ? info.z + ns * (kvh * s.rows + rb * kRowsCuda) : -1;
        p.tickets[task] = 0;
        for (int sp = 0; sp < ns; ++sp) {
          Item it;
          it.b = b; it.r = r; it.kvh = kvh; it.rb = rb;
          it.split = sp; it.n_split = ns;
          it.page_lo = sp * per;
          it.page_hi = min(s.pages, (sp + 1) * per);
          it.task = task; it.pbase = pbase; it.rows = rows; it.pad = 0;
          if (it.page_lo >= it.page_hi) {  // cannot happen with per = ceil(pages/ns); kept safe
            it.page_lo = it.page_hi = 0;
          }
          p.items[item++] = it;
        }
        ++task;
      }
    }
  }
}

// --------------------------------------------------------------------------
// attention kernel (CUDA cores)
// --------------------------------------------------------------------------
struct SmemLayout {
  static constexpr int kStageBytes = kPPS * 2 * kTileBytes;             // 64 KB
  static constexpr int off_stage = 0;
  static constexpr int off_q = off_stage + kStages * kStageBytes;       // fp32 [64][128]
  static constexpr int off_p = off_q + kRowsCuda * kD * 4;              // fp32 [8 warps][8][16]
  static constexpr int off_merge = off_p + kCW * 8 * 16 * 4;            // fp32 [8][8][132]
  static constexpr int off_meta = off_merge + kCW * 8 * kPStride * 4;
  static constexpr int off_bar = off_meta + kStages * (int)sizeof(StageMeta);
  static constexpr int off_misc = off_bar + 2 * kStages * 8;
  static constexpr int total = off_misc + 64;
};

__device__ __forceinline__ uint8_t *stage_tile(uint8_t *smem, int s, int page, int kv) {
  return smem + SmemLayout::off_stage + s * SmemLayout::kStageBytes + (page * 2 + kv) * kTileBytes;
}

// fp32 Q layout in shared memory: for a row, dim d = half*64 + c*8 + sub*4 + e is
// stored at half*64 + sub*32 + c*4 + e, so that eight lanes reading chunk
// (c + lane) & 7 of the same row touch eight different bank groups.
__device__ __forceinline__ int q_slot(int d) {
  int half = d >> 6, c = (d >> 3) & 7, sub = (d >> 2) & 1, e = d & 3;
  return half * 64 + sub * 32 + c * 4 + e;
}

__global__ void __launch_bounds__(kThreads, 1) attn_kernel(const __grid_constant__ AttnParams p) {
  extern __shared__ __align__(1024) uint8_t smem[];
  float *qs = reinterpret_cast<float *>(smem + SmemLayout::off_q);
  float *ps = reinterpret_cast<float *>(smem + SmemLayout::off_p);
  float *mg = reinterpret_cast<float *>(smem + SmemLayout::off_merge);
  StageMeta *meta = reinterpret_cast<StageMeta *>(smem + SmemLayout::off_meta);
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + SmemLayout::off_bar);
  uint64_t *empty = full + kStages;
  int *misc = reinterpret_cast<int *>(smem + SmemLayout::off_misc);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCW);
    }
    misc[0] = 0;  // abort flag
    fence_mbar_init();
  }
  __syncthreads();
  const int n_items = p.ctrl[0];

  if (warp == kCW) {
    // ------------------------------ producer ------------------------------
    const uint64_t policy = l2_policy_evict_first();
    uint32_t it = 0;
    bool aborted = false;
    for (;;) {
      int idx = 0;
      if (lane == 0) idx = atomicAdd(&p.ctrl[1], 1);
      idx = __shfl_sync(0xffffffffu, idx, 0);
      if (idx >= n_items) break;
      const Item I = p.items[idx];
      const BatchDev &B = p.b[I.b];
      const int *prow = B.page_table + (long long)I.r * B.max_pages;
      for (int page = I.page_lo; page < I.page_hi && !aborted; page += kPPS) {
        const int np = min(kPPS, I.page_hi - page);
        const int s = it % kStages;
        const uint32_t ph = (it / kStages) & 1;
        if (!mbar_wait_bounded(&empty[s], ph ^ 1)) {
          ipd_set_error(&g_attn_err, IPD_DEVERR_WAIT);
          aborted = true;
          break;
        }
        int pid = -1;
        bool ok = false;
        if (lane < np) {
          pid = prow[page + lane];
          ok = pid >= 0 && (long long)pid < B.num_pages;
          if (!ok) ipd_set_error(&g_attn_err, IPD_DEVERR_PAGE_ID);
        }
        const uint32_t okmask = __ballot_sync(0xffffffffu, ok);
        if (lane == 0) {
          StageMeta m;
          m.item = idx;
          m.page0 = page;
          m.npages = np;
          m.flags = (page == I.page_lo ? 1 : 0) | (page + np >= I.page_hi ? 2 : 0);
          m.invalid = (~okmask) & ((1u << np) - 1u);
          meta[s] = m;
          mbar_arrive_expect_tx(&full[s], (uint32_t)__popc(okmask) * 2u * kTileBytes);
        }
        __syncwarp();
        if (ok) {
          const size_t off = ((size_t)pid * B.hkv + I.kvh) * (size_t)(kPage * kD);
          bulk_g2s_evict_first(stage_tile(smem, s, lane, 0), B.k_pages + off, kTileBytes, &full[s],
                               policy);
          bulk_g2s_evict_first(stage_tile(smem, s, lane, 1), B.v_pages + off, kTileBytes, &full[s],
                               policy);
        }
        ++it;
      }
      if (aborted) break;
    }
    if (!aborted) {
      // end-of-work marker in the next slot, once the consumers have freed it
      const int s = it % kStages;
      const uint32_t ph = (it / kStages) & 1;
      if (mbar_wait_bounded(&empty[s], ph ^ 1)) {
        if (lane == 0) {
          meta[s].item = -1;
          mbar_arrive(&full[s]);
        }
        return;  // the consumers wait for every copy still in flight
      }
      ipd_set_error(&g_attn_err, IPD_DEVERR_WAIT);
    }
    // time-out path: the consumers stopped; make sure no copy issued by this
    // CTA is still landing in shared memory before the CTA exits.  No slot
    // was reused after stage it-1, so the parities below are unambiguous.
    if (lane == 0) atomicExch(&misc[0], 1);
    for (uint32_t k = (it > (uint32_t)kStages ? it - kStages : 0); k < it; ++k)
      (void)mbar_wait_bounded(&full[k % kStages], (k / kStages) & 1);
    return;
  }

  // -------------------------------- consumers --------------------------------
  const int ctid = threadIdx.x;  // 0 .. 255
  uint32_t it = 0;
  // item context (warp-uniform)
  Item I{};
  int ql = 0, L = 0, G = 1, hq = 1, q0 = 0, rows = 0;
  int n_rg = 1, pw_count = 1, rg = 0, pw = 0, nrow_g = 0;
  bool active = false;
  float m[8], l[8], o[8][4];

  for (;;) {
    const int s = it % kStages;
    const uint32_t ph = (it / kStages) & 1;
    if (!mbar_wait_bounded(&full[s], ph)) {
      ipd_set_error(&g_attn_err, IPD_DEVERR_WAIT);
      atomicExch(&misc[0], 1);
      break;
    }
    const StageMeta M = meta[s];
    if (M.item < 0 || *(volatile int *)&misc[0]) break;
    if (M.flags & 1) {
      I = p.items[M.item];
      const BatchDev &B = p.b[I.b];
      q0 = B.cu_q[I.r];
      ql = B.cu_q[I.r + 1] - q0;
      L = B.seq_len[I.r];
      G = B.group;
      hq = B.hq;
      rows = I.rows;
      n_rg = (rows + 7) >> 3;
      pw_count = kCW / n_rg;
      rg = warp % n_rg;
      pw = warp / n_rg;
      active = pw < pw_count;
      nrow_g = active ? min(8, rows - rg * 8) : 0;
      // stage the item's query rows (fp32) into shared memory
      for (int e = ctid; e < rows * (kD / 8); e += kCW * 32) {
        const int rho = e / (kD / 8), c8 = e % (kD / 8);
        const int grow = I.rb * kRowsCuda + rho;
        const int qi = grow / G, j = grow % G;
        const uint4 raw = *reinterpret_cast<const uint4 *>(
            B.q + ((size_t)(q0 + qi) * hq + I.kvh * G + j) * kD + c8 * 8);
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
      for (int g = 0; g < 8; ++g) {
        m[g] = -INFINITY;
        l[g] = 0.f;
        o[g][0] = o[g][1] = o[g][2] = o[g][3] = 0.f;
      }
      named_bar_sync(1, kCW * 32);
    }

    if (active) {
      const int key = lane >> 1, half = lane & 1;
      for (int pg = pw; pg < M.npages; pg += pw_count) {
        const uint8_t *Kp = stage_tile(smem, s, pg, 0);
        const uint8_t *Vp = stage_tile(smem, s, pg, 1);
        const int kpos = (M.page0 + pg) * kPage + key;
        const bool page_ok = !((M.invalid >> pg) & 1u);
        uint4 kr[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const int cc = (c + lane) & 7;
          kr[c] = *reinterpret_cast<const uint4 *>(Kp + key * 256 + half * 128 + cc * 16);
        }
#pragma unroll
        for (int g = 0; g < 8; ++g) {
          if (g < nrow_g) {
            const int rho = rg * 8 + g;
            const float *qrow = qs + rho * kD + half * 64;
            float acc = 0.f;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
              const int cc = (c + lane) & 7;
              const float4 a = *reinterpret_cast<const float4 *>(qrow + cc * 4);
              const float4 b2 = *reinterpret_cast<const float4 *>(qrow + 32 + cc * 4);
              acc = fmaf(bf16lo(kr[c].x), a.x, acc);
              acc = fmaf(bf16hi(kr[c].x), a.y, acc);
              acc = fmaf(bf16lo(kr[c].y), a.z, acc);
              acc = fmaf(bf16hi(kr[c].y), a.w, acc);
              acc = fmaf(bf16lo(kr[c].z), b2.x, acc);
              acc = fmaf(bf16hi(kr[c].z), b2.y, acc);
              acc = fmaf(bf16lo(kr[c].w), b2.z, acc);
              acc = fmaf(bf16hi(kr[c].w), b2.w, acc);
            }
            acc += __shfl_xor_sync(0xffffffffu, acc, 1);
            const int qi = (I.rb * kRowsCuda + rho) / G;
            const bool vis = page_ok && kpos < L && kpos <= L - ql + qi;
            const float sc = vis ? acc * p.scale_log2 : -INFINITY;
            float mx = sc;
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
            const float mnew = fmaxf(m[g], mx);
            float alpha = 1.f, pr = 0.f;
            if (mnew != -INFINITY) {
              alpha = exp2f(m[g] - mnew);
              pr = exp2f(sc - mnew);
            }
            l[g] = l[g] * alpha + (half == 0 ? pr : 0.f);
            o[g][0] *= alpha;
            o[g][1] *= alpha;
            o[g][2] *= alpha;
            o[g][3] *= alpha;
            m[g] = mnew;
            if (half == 0) ps[(warp * 8 + g) * 16 + key] = pr;
          }
        }
        __syncwarp();
#pragma unroll 4
        for (int jk = 0; jk < 16; ++jk) {
          const uint2 vv = *reinterpret_cast<const uint2 *>(Vp + jk * 256 + lane * 8);
          const float v0 = bf16lo(vv.x), v1 = bf16hi(vv.x), v2 = bf16lo(vv.y), v3 = bf16hi(vv.y);
#pragma unroll
          for (int g = 0; g < 8; ++g) {
            if (g < nrow_g) {
              const float pj = ps[(warp * 8 + g) * 16 + jk];
              o[g][0] = fmaf(pj, v0, o[g][0]);
              o[g][1] = fmaf(pj, v1, o[g][1]);
              o[g][2] = fmaf(pj, v2, o[g][2]);
              o[g][3] = fmaf(pj, v3, o[g][3]);
            }
          }
        }
        __syncwarp();
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);

    if (M.flags & 2) {
      // ------------------------------ finalize ------------------------------
      const BatchDev &B = p.b[I.b];
#pragma unroll
      for (int g = 0; g < 8; ++g)
        if (g < nrow_g) l[g] = warp_sum(l[g]);
      if (pw_count > 1) {
        if (active) {
#pragma unroll
          for (int g = 0; g < 8; ++g) {
            if (g < nrow_g) {
              float *dst = mg + (warp * 8 + g) * kPStride;
              *reinterpret_cast<float4 *>(dst + lane * 4) =
                  make_float4(o[g][0], o[g][1], o[g][2], o[g][3]);
              if (lane == 0) {
                dst[128] = m[g];
                dst[129] = l[g];
              }
            }
          }
        }
        named_bar_sync(1, kCW * 32);
        if (active && pw == 0) {
#pragma unroll
          for (int g = 0; g < 8; ++g) {
            if (g < nrow_g) {
              float Mx = -INFINITY;
              for (int w2 = 0; w2 < pw_count; ++w2)
                Mx = fmaxf(Mx, mg[((rg + w2 * n_rg) * 8 + g) * kPStride + 128]);
              float Ls = 0.f, O0 = 0.f, O1 = 0.f, O2 = 0.f, O3 = 0.f;
              for (int w2 = 0; w2 < pw_count; ++w2) {
                const float *src = mg + ((rg + w2 * n_rg) * 8 + g) * kPStride;
                const float sc = (src[128] == -INFINITY) ? 0.f : exp2f(src[128] - Mx);
                const float4 ov = *reinterpret_cast<const float4 *>(src + lane * 4);
                Ls += src[129] * sc;
                O0 += ov.x * sc;
                O1 += ov.y * sc;
                O2 += ov.z * sc;
                O3 += ov.w * sc;
              }
              m[g] = Mx;
              l[g] = Ls;
              o[g][0] = O0; o[g][1] = O1; o[g][2] = O2; o[g][3] = O3;
            }
          }
        }
      }
      const bool owner = active && pw == 0;
      if (I.n_split == 1) {
        if (owner) {
#pragma unroll
          for (int g = 0; g < 8; ++g) {
            if (g < nrow_g) {
              const int grow = I.rb * kRowsCuda + rg * 8 + g;
              const int qi = grow / G, j = grow % G;
              const float inv = l[g] > 0.f ? 1.f / l[g] : 0.f;
              uint2 pk;
              pk.x = (uint32_t)f2bf16(o[g][0] * inv) | ((uint32_t)f2bf16(o[g][1] * inv) << 16);
              pk.y = (uint32_t)f2bf16(o[g][2] * inv) | ((uint32_t)f2bf16(o[g][3] * inv) << 16);
              *reinterpret_cast<uint2 *>(B.out + ((size_t)(q0 + qi) * hq + I.kvh * G + j) * kD +
                                         lane * 4) = pk;
            }
          }
        }
      } else {
        if (owner) {
#pragma unroll
          for (int g = 0; g < 8; ++g) {
            if (g < nrow_g) {
              float *dst = p.partials +
                           ((size_t)I.pbase + (size_t)I.split * rows + rg * 8 + g) * kPStride;
              __stcg(reinterpret_cast<float4 *>(dst + lane * 4),
                     make_float4(o[g][0], o[g][1], o[g][2], o[g][3]));
              if (lane == 0) {
                __stcg(dst + 128, m[g]);
                __stcg(dst + 129, l[g]);
              }
            }
          }
        }
        __threadfence();
        named_bar_sync(1, kCW * 32);
        if (ctid == 0) misc[1] = (atomicAdd(&p.tickets[I.task], 1) == I.n_split - 1);
        named_bar_sync(1, kCW * 32);
        if (misc[1]) {
          __threadfence();
          for (int rho = warp; rho < rows; rho += kCW) {
            float Mx = -INFINITY;
            for (int sp = 0; sp < I.n_split; ++sp)
              Mx = fmaxf(Mx, __ldcg(p.partials + ((size_t)I.pbase + (size_t)sp * rows + rho) *
                                                     kPStride + 128));
            float Ls = 0.f, O0 = 0.f, O1 = 0.f, O2 = 0.f, O3 = 0.f;
            for (int sp = 0; sp < I.n_split; ++sp) {
              const float *src = p.partials + ((size_t)I.pbase + (size_t)sp * rows + rho) * kPStride;
              const float mm = __ldcg(src + 128);
              const float sc = (mm == -INFINITY) ? 0.f : exp2f(mm - Mx);
              const float4 ov = __ldcg(reinterpret_cast<const float4 *>(src + lane * 4));
              Ls += __ldcg(src + 129) * sc;
              O0 += ov.x * sc;
              O1 += ov.y * sc;
              O2 += ov.z * sc;
              O3 += ov.w * sc;
            }
            const int grow = I.rb * kRowsCuda + rho;
            const int qi = grow / G, j = grow % G;
            const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
            uint2 pk;
            pk.x = (uint32_t)f2bf16(O0 * inv) | ((uint32_t)f2bf16(O1 * inv) << 16);
            pk.y = (uint32_t)f2bf16(O2 * inv) | ((uint32_t)f2bf16(O3 * inv) << 16);
            *reinterpret_cast<uint2 *>(B.out + ((size_t)(q0 + qi) * hq + I.kvh * G + j) * kD +
                                       lane * 4) = pk;
          }
        }
      }
      named_bar_sync(1, kCW * 32);
    }
    ++it;
  }
}

// --------------------------------------------------------------------------
// host launch
// --------------------------------------------------------------------------
struct DevInfo {
  int sms = 0;
  bool attr_set = false;
};
DevInfo g_dev[64];

int launch(const ipd_attn_batch *const *bs, int n, float scale, void *ws, size_t ws_bytes,
           cudaStream_t stream) {
  if (!(scale > 0.f) || scale != scale) return IPD_ERR_INVALID_ARG;
  WsLayout W = layout(bs, n);
  if (W.total_reqs == 0) return IPD_OK;
  if (!ws || ws_bytes < W.total || ((uintptr_t)ws & 255)) return IPD_ERR_WORKSPACE;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return IPD_ERR_CUDA;
  DevInfo &D = g_dev[dev];
  if (!D.attr_set) {
    if (cudaDeviceGetAttribute(&D.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return IPD_ERR_CUDA;
    if (cudaFuncSetAttribute(attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SmemLayout::total) != cudaSuccess)
      return IPD_ERR_CUDA;
    D.attr_set = true;
  }
  AttnParams P{};
  P.n_batches = n;
  int base = 0;
  for (int i = 0; i < n; ++i) {
    const ipd_attn_batch *b = bs[i];
    BatchDev &B = P.b[i];
    B.q = b->q;
    B.out = b->out;
    B.cu_q = b->cu_q;
    B.seq_len = b->seq_len;
    B.page_table = b->page_table;
    B.k_pages = b->cache->k_pages;
    B.v_pages = b->cache->v_pages;
    B.num_pages = b->cache->num_pages;
    B.num_reqs = b->num_reqs;
    B.hq = b->num_q_heads;
    B.hkv = b->cache->num_kv_heads;
    B.group = B.hq / B.hkv;
    B.max_pages = b->max_pages;
    B.max_q_len = b->max_q_len;
    B.total_q = b->total_q;
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
  P.tickets = reinterpret_cast<int *>(w + W.off_tickets);
  P.partials = reinterpret_cast<float *>(w + W.off_partials);
  P.item_cap = W.item_cap;
  P.task_cap = W.task_cap;
  P.prow_cap = W.prow_cap;

  attn_plan_kernel<<<1, 1024, 0, stream>>>(P);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  const int grid = std::max(1, std::min(D.sms, W.item_cap));
  attn_kernel<<<grid, kThreads, SmemLayout::total, stream>>>(P);
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
  int st = collect(verify, n_verify, decode, n_decode, bs);
  if (st != IPD_OK) return st;
  return launch(bs, n_verify + n_decode, softmax_scale, workspace, workspace_bytes,
                reinterpret_cast<cudaStream_t>(stream));
}

extern "C" int ipd_decode_attn(const ipd_attn_batch *decode, int n_decode, float softmax_scale,
                               void *workspace, size_t workspace_bytes, ipd_stream_t stream) {
  return ipd_verify_attn(nullptr, 0, decode, n_decode, softmax_scale, workspace, workspace_bytes,
                         stream);
}
