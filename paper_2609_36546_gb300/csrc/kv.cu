// Append of newly computed tokens' K/V rows into a paged cache (Sec. 3.2.3:
// the proposer's decode extends its own cache by one token per step, the
// verifier's prefill writes the span's tokens into its cache; each happens
// before the attention that reads them).
//
// One thread per 16-byte piece of a row (a 128-wide bf16 head row is 16
// pieces): consecutive threads cover one head row, then the next head, then
// the next token, so both the reads of the new rows and the writes into a
// page slot are contiguous 256-byte runs.  Every write is bounds-checked
// against the page table and the pool; a bad entry is recorded in the device
// error word and skipped.
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

IPD_DECLARE_ERROR_WORD(g_kv_err);

namespace {

constexpr int kPieces = 16;  // 16-byte pieces per 128-wide bf16 row
constexpr int kAppendThreads = 256;

__global__ void __launch_bounds__(kAppendThreads) kv_append_kernel(
    uint16_t *__restrict__ k_pages, uint16_t *__restrict__ v_pages, long long num_pages, int hkv,
    const uint16_t *__restrict__ k_new, const uint16_t *__restrict__ v_new,
    const int32_t *__restrict__ cu_new, const int32_t *__restrict__ seq_len,
    const int32_t *__restrict__ page_table, int max_pages, int num_reqs, long long n_units) {
  const long long per_tok = (long long)hkv * kPieces;
  for (long long u = (long long)blockIdx.x * kAppendThreads + threadIdx.x; u < 2 * n_units;
       u += (long long)gridDim.x * kAppendThreads) {
    const bool is_v = u >= n_units;
    const long long w = is_v ? u - n_units : u;
    const int tok = (int)(w / per_tok);
    const int rem = (int)(w % per_tok);
    const int h = rem / kPieces, c = rem % kPieces;
    // the request holding new row `tok`: the last r with cu_new[r] <= tok
    int lo = 0, hi = num_reqs - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (cu_new[mid] <= tok) lo = mid;
      else hi = mid - 1;
    }
    const int n = cu_new[lo + 1] - cu_new[lo];
    const int p = seq_len[lo] - n + (tok - cu_new[lo]);  // absolute position of the row
    if (p < 0 || (p >> 4) >= max_pages) {
      ipd_set_error(&g_kv_err, IPD_DEVERR_SEQ_LEN);
      continue;
    }
    const int page = page_table[(size_t)lo * max_pages + (p >> 4)];
    if (page < 0 || page >= num_pages) {
      ipd_set_error(&g_kv_err, IPD_DEVERR_PAGE_ID);
      continue;
    }
    const uint4 *src = reinterpret_cast<const uint4 *>(is_v ? v_new : k_new);
    uint4 *dst = reinterpret_cast<uint4 *>(is_v ? v_pages : k_pages);
    dst[(((size_t)page * hkv + h) * 16 + (p & 15)) * kPieces + c] =
        src[((size_t)tok * hkv + h) * kPieces + c];
  }
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
  if (num_reqs < 0 || total_new < 0 || num_pages < 0 || num_kv_heads < 1 || max_pages < 1)
    return IPD_ERR_INVALID_ARG;
  if (page_size != 16 || head_dim != 128) return IPD_ERR_UNSUPPORTED;
  if (total_new == 0) return IPD_OK;
  if (num_reqs == 0 || !k_pages || !v_pages || !k_new || !v_new || !cu_new || !seq_len ||
      !page_table)
    return IPD_ERR_INVALID_ARG;
  if (((uintptr_t)k_pages | (uintptr_t)v_pages | (uintptr_t)k_new | (uintptr_t)v_new) & 15)
    return IPD_ERR_INVALID_ARG;
  const long long n_units = (long long)total_new * num_kv_heads * kPieces;
  const long long blocks = (2 * n_units + kAppendThreads - 1) / kAppendThreads;
  const int grid = (int)(blocks < 8192 ? blocks : 8192);
  kv_append_kernel<<<grid, kAppendThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      k_pages, v_pages, num_pages, num_kv_heads, k_new, v_new, cu_new, seq_len, page_table,
      max_pages, num_reqs, n_units);
  if (cudaGetLastError() != cudaSuccess) return IPD_ERR_CUDA;
  return IPD_OK;
}
