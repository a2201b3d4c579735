// kv_commit.cu -- the context update of Algorithm 1 (m <- m + a + 1) applied to
// the KV cache: the accepted prefix of the verify block stays, the rejected
// draft slots are cleared, ctx_lens advances by a + 1.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace spade {
namespace commit {

// One CTA per sequence: every thread reads ctx_lens[b] before any thread
// writes it, so the in-place update cannot race.
// Paged caches: block_table [B, max_pages] names the page of every page_size
// slots; block_table == nullptr means dense caches [B, Hkv, cap, D].
__global__ void __launch_bounds__(256) kv_commit_kernel(uint4 *k_cache, uint4 *v_cache,
                                                       int32_t *ctx_lens, const int32_t *accepted,
                                                       const int32_t *n_draft, int Hkv, int D,
                                                       int cap, int32_t *status,
                                                       const int32_t *block_table, int page_size,
                                                       int max_pages, int num_pages) {
  const int b = blockIdx.x;
  const int ctx = ctx_lens[b];
  const int a = accepted[b];
  const int k = n_draft[b];
  int bad = 0;
  if (ctx < 0 || k < 0 || a < 0 || a > k) bad = SPADE_DEV_BAD_INDEX;
  else if (static_cast<int64_t>(ctx) + k + 1 > cap) bad = SPADE_DEV_CAPACITY;
  __syncthreads();
  if (bad) {
    if (threadIdx.x == 0) atomicOr(status, bad);
    return;
  }
  const int lo = ctx + a + 1;        // first rejected slot
  const int n_slots = k - a;         // slots lo .. ctx + k
  const int vec = D / 8;             // 16-byte vectors per slot
  if (block_table) {
    // Every page the rejected slots use must exist before anything is cleared.
    int bad_page = 0;
    for (int s = threadIdx.x; s < n_slots; s += blockDim.x) {
      const int pg = block_table[static_cast<int64_t>(b) * max_pages + (lo + s) / page_size];
      if (pg < 0 || pg >= num_pages) bad_page = 1;
    }
    if (__syncthreads_or(bad_page)) {
      if (threadIdx.x == 0) atomicOr(status, SPADE_DEV_BAD_INDEX);
      return;
    }
  }
  const int per_head = n_slots * vec;
  const int total = Hkv * per_head;
  const uint4 z = make_uint4(0, 0, 0, 0);
  for (int e = threadIdx.x; e < total; e += blockDim.x) {
    const int h = e / per_head;
    const int r = e - h * per_head;
    const int slot = lo + r / vec;
    size_t off;
    if (block_table) {
      const int pg = block_table[static_cast<int64_t>(b) * max_pages + slot / page_size];
      off = ((static_cast<size_t>(pg) * Hkv + h) * page_size + slot % page_size) * vec + r % vec;
    } else {
      off = ((static_cast<size_t>(b) * Hkv + h) * cap + lo) * vec + r;
    }
    k_cache[off] = z;
    v_cache[off] = z;
  }
  __syncthreads();
  if (threadIdx.x == 0) ctx_lens[b] = lo;
}

}  // namespace commit
}  // namespace spade

using namespace spade;

extern "C" spade_status spade_kv_commit(void *k_cache, void *v_cache, int32_t *ctx_lens,
                                        const int32_t *accepted_len, const int32_t *n_draft,
                                        int32_t B, int32_t Hkv, int32_t D, int32_t cap,
                                        int32_t *status, spade_stream_t stream) {
  if (!k_cache || !v_cache || !ctx_lens || !accepted_len || !n_draft || !status)
    return fail(SPADE_ERR_INVALID_ARG, "spade_kv_commit: null pointer argument");
  if (B <= 0 || Hkv <= 0 || cap <= 0 || D <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_kv_commit: non-positive size");
  if (D % 8) return fail(SPADE_ERR_SHAPE, "spade_kv_commit: D = %d must be a multiple of 8", D);
  if (!aligned(k_cache, 16) || !aligned(v_cache, 16))
    return fail(SPADE_ERR_INVALID_ARG, "spade_kv_commit: caches must be 16-byte aligned");
  spade_status st = device_info(nullptr, nullptr);
  if (st != SPADE_OK) return st;
  commit::kv_commit_kernel<<<B, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      static_cast<uint4 *>(k_cache), static_cast<uint4 *>(v_cache), ctx_lens, accepted_len,
      n_draft, Hkv, D, cap, status, nullptr, 0, 0, 0);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "kv_commit launch");
  return SPADE_OK;
}

extern "C" spade_status spade_kv_commit_paged(void *k_pool, void *v_pool, const int32_t *block_table,
                                              int32_t *ctx_lens, const int32_t *accepted_len,
                                              const int32_t *n_draft, int32_t B, int32_t Hkv, int32_t D,
                                              int32_t page_size, int32_t num_pages, int32_t max_pages,
                                              int32_t *status, spade_stream_t stream) {
  if (!k_pool || !v_pool || !block_table || !ctx_lens || !accepted_len || !n_draft || !status)
    return fail(SPADE_ERR_INVALID_ARG, "spade_kv_commit_paged: null pointer argument");
  if (B <= 0 || Hkv <= 0 || D <= 0 || page_size <= 0 || num_pages <= 0 || max_pages <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_kv_commit_paged: non-positive size");
  if (D % 8) return fail(SPADE_ERR_SHAPE, "spade_kv_commit_paged: D = %d must be a multiple of 8", D);
  if (static_cast<int64_t>(max_pages) * page_size >= (int64_t(1) << 31))
    return fail(SPADE_ERR_CAPACITY, "max_pages * page_size exceeds 2^31");
  if (!aligned(k_pool, 16) || !aligned(v_pool, 16))
    return fail(SPADE_ERR_INVALID_ARG, "spade_kv_commit_paged: pools must be 16-byte aligned");
  spade_status st = device_info(nullptr, nullptr);
  if (st != SPADE_OK) return st;
  commit::kv_commit_kernel<<<B, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      static_cast<uint4 *>(k_pool), static_cast<uint4 *>(v_pool), ctx_lens, accepted_len, n_draft, Hkv,
      D, max_pages * page_size, status, block_table, page_size, max_pages, num_pages);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "kv_commit_paged launch");
  return SPADE_OK;
}
