// Append of newly computed tokens' K/V rows into a paged cache (Sec. 3.2.3:
// the proposer's decode extends its own cache by one token per step, the
// verifier's prefill writes the span's tokens into its cache; each happens
// before the attention that reads them).
//
// One thread per 16-byte piece of a row (a 128-wide bf16 head row is 16
// pieces): consecutive threads cover one head row, then the next head, then
// the next token, so both the reads of the new rows and the writes into a
// page slot are contiguous 256-byte runs.  Every write is bounds-checked
// against the request offsets, the sequence length, the page table and the
// pool; a bad entry is recorded in the device error word and skipped.  One launch takes up to IPD_MAX_BATCHES appends
// (caches and request batches), so a step's appends cost one launch.
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include "common.cuh"

IPD_DECLARE_ERROR_WORD(g_kv_err);

namespace {

constexpr int kPieces = 16;  // 16-byte pieces per 128-wide bf16 row
constexpr int kAppendThreads = 256;

// One append (one cache, one batch of requests) of a launch.
struct AppendDev {
  uint16_t *k_pages, *v_pages;
  const uint16_t *k_new, *v_new;
  const int32_t *cu_new, *seq_len, *page_table;
  long long num_pages;
  long long n_units;  // total_new * hkv * kPieces pieces of K (as many of V)
  int hkv, max_pages, num_reqs, pad;
};

struct AppendParams {
  AppendDev d[IPD_MAX_BATCHES];
  long long end[IPD_MAX_BATCHES];  // exclusive prefix of 2 n_units over the appends
  int n;
};

__global__ void __launch_bounds__(kAppendThreads) kv_append_kernel(
    const __grid_constant__ AppendParams P) {
  const long long total = P.end[P.n - 1];
  for (long long u0 = (long long)blockIdx.x * kAppendThreads + threadIdx.x; u0 < total;
       u0 += (long long)gridDim.x * kAppendThreads) {
    int di = 0;
    while (di + 1 < P.n && u0 >= P.end[di]) ++di;
    const AppendDev &D = P.d[di];
    const long long u = u0 - (di > 0 ? P.end[di - 1] : 0);
    const bool is_v = u >= D.n_units;
    const long long w = is_v ? u - D.n_units : u;
    const long long per_tok = (long long)D.hkv * kPieces;
    const int tok = (int)(w / per_tok);
    const int rem = (int)(w % per_tok);
    const int h = rem / kPieces, c = rem % kPieces;
    // a row that no request's offsets cover is not written
    if (tok < D.cu_new[0] || tok >= D.cu_new[D.num_reqs]) {
      ipd_set_error(&g_kv_err, IPD_DEVERR_SPAN);
      continue;
    }
    // the request holding new row `tok`: the last r with cu_new[r] <= tok
    int lo = 0, hi = D.num_reqs - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (D.cu_new[mid] <= tok) lo = mid;
      else hi = mid - 1;
    }
    const int n = D.cu_new[lo + 1] - D.cu_new[lo];
    const int p = D.seq_len[lo] - n + (tok - D.cu_new[lo]);  // absolute position of the row
    if (p < 0 || p >= D.seq_len[lo] || (p >> 4) >= D.max_pages) {
      ipd_set_error(&g_kv_err, IPD_DEVERR_SEQ_LEN);
      continue;
    }
    const int page = D.page_table[(size_t)lo * D.max_pages + (p >> 4)];
    if (page < 0 || page >= D.num_pages) {
      ipd_set_error(&g_kv_err, IPD_DEVERR_PAGE_ID);
      continue;
    }
    const uint4 *src = reinterpret_cast<const uint4 *>(is_v ? D.v_new : D.k_new);
    uint4 *dst = reinterpret_cast<uint4 *>(is_v ? D.v_pages : D.k_pages);
    dst[(((size_t)page * D.hkv + h) * 16 + (p & 15)) * kPieces + c] =
        src[((size_t)tok * D.hkv + h) * kPieces + c];
  }
}

// Host validation of one append; fills its device descriptor.  IPD_OK with
// n_units == 0 for an append with no rows.
int check_append(const ipd_kv_append_desc &a, AppendDev *d) {
  if (a.num_reqs < 0 || a.total_new < 0 || a.num_pages < 0 || a.num_kv_heads < 1 ||
      a.max_pages < 1)
    return IPD_ERR_INVALID_ARG;
  if (a.page_size != 16 || a.head_dim != 128) return IPD_ERR_UNSUPPORTED;
  *d = AppendDev{};
  if (a.total_new == 0) return IPD_OK;
  if (a.num_reqs == 0 || !a.k_pages || !a.v_pages || !a.k_new || !a.v_new || !a.cu_new ||
      !a.seq_len || !a.page_table)
    return IPD_ERR_INVALID_ARG;
  if (((uintptr_t)a.k_pages | (uintptr_t)a.v_pages | (uintptr_t)a.k_new | (uintptr_t)a.v_new) &
      15)
    return IPD_ERR_INVALID_ARG;
  *d = AppendDev{a.k_pages, a.v_pages, a.k_new, a.v_new, a.cu_new, a.seq_len, a.page_table,
                 a.num_pages, (long long)a.total_new * a.num_kv_heads * kPieces,
                 a.num_kv_heads, a.max_pages, a.num_reqs, 0};
  return IPD_OK;
}

int launch_appends(const ipd_kv_append_desc *descs, int n, ipd_stream_t stream) {
  if (n < 0 || n > IPD_MAX_BATCHES || (n > 0 && !descs)) return IPD_ERR_INVALID_ARG;
  AppendParams P;
  memset(&P, 0, sizeof(P));
  long long total = 0;
  for (int i = 0; i < n; ++i) {
    AppendDev d;
    const int st = check_append(descs[i], &d);
    if (st != IPD_OK) return st;
    if (d.n_units == 0) continue;  // nothing to write: not part of the launch
    P.d[P.n] = d;
    total += 2 * d.n_units;
    P.end[P.n] = total;
    ++P.n;
  }
  if (P.n == 0) return IPD_OK;
  const long long blocks = (total + kAppendThreads - 1) / kAppendThreads;
  const int grid = (int)(blocks < 8192 ? blocks : 8192);
  kv_append_kernel<<<grid, kAppendThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(P);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}

}  // namespace

extern "C" __attribute__((visibility("hidden"))) unsigned int ipd_internal_take_kv_error() {
  unsigned int v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_kv_err, sizeof(v)) != cudaSuccess) return 0xffffffffu;
  if (cudaMemcpyToSymbol(g_kv_err, &z, sizeof(z)) != cudaSuccess) return 0xffffffffu;
  return v;
}

extern "C" int ipd_kv_append(uint16_t *k_pages, uint16_t *v_pages, int64_t num_pages,
                             int num_kv_heads, int page_size, int head_dim,
                             const uint16_t *k_new, const uint16_t *v_new, const int32_t *cu_new,
                             const int32_t *seq_len, const int32_t *page_table, int max_pages,
                             int num_reqs, int total_new, ipd_stream_t stream) {
  const ipd_kv_append_desc a{k_pages, v_pages, num_pages, num_kv_heads, page_size, head_dim,
                             k_new,   v_new,   cu_new,    seq_len,      page_table, max_pages,
                             num_reqs, total_new};
  return launch_appends(&a, 1, stream);
}

extern "C" int ipd_kv_append_many(const ipd_kv_append_desc *appends, int n,
                                  ipd_stream_t stream) {
  return launch_appends(appends, n, stream);
}
