// verify_attention.cu -- attention of the k+1 verify positions of every sequence
// against its bf16 KV cache (the verifier's single forward pass over the draft
// block: Sec. III-B "Verification Stage", Algorithm 1 cloud step).  This file
// holds the C-ABI entry points: argument checks, the workspace (merge counters
// and split partials), the tensor maps, and the launch of the tensor-memory
// kernel in verify_attention_tc.cu (head dims 64 and 128).  The schedule
// (stream-K over 64-key slices, GQA row blocks as units) and the log-sum-exp
// merge of split units are in attn_common.cuh.
#include <mutex>

#include "attn_common.cuh"

namespace spade {
namespace attn {

static int row_blocks(int G, int max_k) { return (G * (max_k + 1) + kRowBlock - 1) / kRowBlock; }

}  // namespace attn
}  // namespace spade

using namespace spade;

extern "C" size_t spade_attn_workspace_size(int32_t B, int32_t Hq, int32_t Hkv, int32_t D,
                                            int32_t cap, int32_t max_k) {
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv || (D != 64 && D != 128) || cap <= 0 || max_k < 0)
    return 0;
  int sms = 0;
  if (device_info(&sms, nullptr) != SPADE_OK) return 0;
  const int RB = attn::row_blocks(Hq / Hkv, max_k);
  const size_t units = static_cast<size_t>(B) * Hkv * RB;
  const size_t counters = round_up(units * 4, 256);
  return counters + (units + sms) * attn::slot_floats(D) * sizeof(float);
}

namespace spade {
namespace attn {
// Page geometry of a paged cache (see Params).
struct Paging {
  const int32_t *block_table;
  int page_size, max_pages, num_pages;
};
}  // namespace attn
}  // namespace spade

static spade_status verify_attention_impl(
    const void *q, const void *k_cache, const void *v_cache, const int32_t *ctx_lens,
    const int32_t *n_draft, const int32_t *cu_q, void *out, float *lse, int32_t B, int32_t Hq,
    int32_t Hkv, int32_t D, int32_t cap, int32_t max_k, int32_t R, void *workspace,
    size_t workspace_bytes, int32_t *status, spade_stream_t stream, const attn::Paging *pg) {
  if (!q || !k_cache || !v_cache || !ctx_lens || !n_draft || !cu_q || !out || !status)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention: null pointer argument");
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0 || max_k < 0 || R <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention: non-positive size");
  if (Hq % Hkv) return fail(SPADE_ERR_SHAPE, "Hq (%d) must be a multiple of Hkv (%d)", Hq, Hkv);
  if (D != 64 && D != 128) return fail(SPADE_ERR_SHAPE, "head dim %d not supported (64 or 128)", D);
  if (B > attn::kMaxB) return fail(SPADE_ERR_SHAPE, "B = %d exceeds %d sequences per call", B, attn::kMaxB);
  if (R < B) return fail(SPADE_ERR_INVALID_ARG, "R = %d < B = %d", R, B);
  const int64_t cache_rows = pg ? static_cast<int64_t>(pg->num_pages) * Hkv * pg->page_size
                                : static_cast<int64_t>(B) * Hkv * cap;
  if (cache_rows >= (int64_t(1) << 31))
    return fail(SPADE_ERR_CAPACITY, "KV cache rows (B or pages) * Hkv * slots exceed 2^31");
  if (!aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(q, 16) || !aligned(out, 16))
    return fail(SPADE_ERR_INVALID_ARG, "q, caches and out must be 16-byte aligned");
  int sms = 0;
  spade_status st = device_info(&sms, nullptr);
  if (st != SPADE_OK) return st;
  const int G = Hq / Hkv;
  const int RB = attn::row_blocks(G, max_k);
  const size_t need = spade_attn_workspace_size(B, Hq, Hkv, D, cap, max_k);
  if (!workspace || workspace_bytes < need || !aligned(workspace, 256))
    return fail(SPADE_ERR_WORKSPACE, "attention workspace needs %zu bytes, 256-byte aligned (got %zu)",
                need, workspace_bytes);
  const int units = B * Hkv * RB;

  attn::Params p;
  p.q = static_cast<const __nv_bfloat16 *>(q);
  p.out = static_cast<__nv_bfloat16 *>(out);
  p.lse = lse;
  p.ctx_lens = ctx_lens;
  p.n_draft = n_draft;
  p.cu_q = cu_q;
  p.counters = static_cast<int32_t *>(workspace);
  p.partials = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) +
                                         round_up(static_cast<size_t>(units) * 4, 256));
  p.status = status;
  p.B = B; p.Hq = Hq; p.Hkv = Hkv; p.G = G; p.cap = cap; p.max_k = max_k; p.R = R; p.RB = RB;
  p.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(D));
  p.block_table = pg ? pg->block_table : nullptr;
  p.page_size = pg ? pg->page_size : 0;
  p.max_pages = pg ? pg->max_pages : 0;
  p.num_pages = pg ? pg->num_pages : 0;
  // The tensor-memory kernel charges each unit's epilogue and pipeline restart
  // to the CTA that starts it; a 64-dim slice moves half the bytes of a
  // 128-dim one, so the same restart costs twice the slices.
  p.unit_cost = (D == 128) ? attn::kUnitCostTc : 2 * attn::kUnitCostTc;
  // One CTA per SM, never more CTAs than key chunks could exist.
  const int64_t max_chunks = static_cast<int64_t>(units) * ((cap + attn::kChunk - 1) / attn::kChunk);
  p.num_ctas = static_cast<int>(max_chunks < sms ? max_chunks : sms);

  const uint64_t rows = static_cast<uint64_t>(cache_rows);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  {
    // Tensor-memory kernel: 128-key boxes of every 64-dim slab, and 64-key
    // boxes of one slab for a segment's last odd slice.
    CUtensorMap k2, v2, k1, v1;
    if (!encode_tmap_rows_by_slab(&k2, k_cache, rows, D, 128) ||
        !encode_tmap_rows_by_slab(&v2, v_cache, rows, D, 128) ||
        !encode_tmap_rows_by_slab(&k1, k_cache, rows, D, attn::kChunk, 1) ||
        !encode_tmap_rows_by_slab(&v1, v_cache, rows, D, attn::kChunk, 1))
      return SPADE_ERR_CUDA;
    const int rows_max = G * (max_k + 1) < attn::kRowBlock ? G * (max_k + 1) : attn::kRowBlock;
    e = attn::launch_tc(p, k2, v2, k1, v1, (rows_max + 15) / 16 * 16, D, s);
  }
  if (e != cudaSuccess) return cuda_fail(e, "verify_attention launch");
  return SPADE_OK;
}

extern "C" spade_status spade_verify_attention(
    const void *q, const void *k_cache, const void *v_cache, const int32_t *ctx_lens,
    const int32_t *n_draft, const int32_t *cu_q, void *out, float *lse, int32_t B, int32_t Hq,
    int32_t Hkv, int32_t D, int32_t cap, int32_t max_k, int32_t R, void *workspace,
    size_t workspace_bytes, int32_t *status, spade_stream_t stream) {
  return verify_attention_impl(q, k_cache, v_cache, ctx_lens, n_draft, cu_q, out, lse, B, Hq, Hkv, D,
                               cap, max_k, R, workspace, workspace_bytes, status, stream, nullptr);
}

extern "C" spade_status spade_verify_attention_paged(
    const void *q, const void *k_pool, const void *v_pool, const int32_t *block_table,
    const int32_t *ctx_lens, const int32_t *n_draft, const int32_t *cu_q, void *out, float *lse,
    int32_t B, int32_t Hq, int32_t Hkv, int32_t D, int32_t page_size, int32_t num_pages,
    int32_t max_pages, int32_t max_k, int32_t R, void *workspace, size_t workspace_bytes,
    int32_t *status, spade_stream_t stream) {
  if (!block_table) return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention_paged: null block_table");
  if (page_size <= 0 || num_pages <= 0 || max_pages <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention_paged: non-positive page geometry");
  if (page_size % attn::kChunk)
    return fail(SPADE_ERR_SHAPE, "page size %d must be a multiple of %d", page_size, attn::kChunk);
  if (static_cast<int64_t>(max_pages) * page_size >= (int64_t(1) << 31))
    return fail(SPADE_ERR_CAPACITY, "max_pages * page_size exceeds 2^31");
  const attn::Paging pg{block_table, page_size, max_pages, num_pages};
  return verify_attention_impl(q, k_pool, v_pool, ctx_lens, n_draft, cu_q, out, lse, B, Hq, Hkv, D,
                               max_pages * page_size, max_k, R, workspace, workspace_bytes, status,
                               stream, &pg);
}

// ---------------------------------------------------------------------------
// Allocation-free variant.  Some callers cannot allocate device memory at all:
// plugin hosts that hand a kernel only its input and output buffers, or
// serving loops that freeze their memory pool after start-up.  For them the
// attention's scratch (merge counters and split partials) lives in a
// file-scope device array instead of a caller-provided workspace.  The array
// is reserved on every GPU that loads this library, until the process exits.
namespace spade {
namespace attn_noalloc {

constexpr size_t kScratchBytes = size_t(32) << 20;  // 32 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) uint8_t g_scratch[kScratchBytes];

static std::mutex g_mu;
static void *g_ptr[kMaxDevices];  // device address of g_scratch, per device

// Host code must not pass `g_scratch` itself to a kernel: on the host that
// name is a stand-in, not a device address.  Resolve it once per device.
static spade_status scratch_address(int dev, void **out) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_ptr[dev]) {
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(attention scratch)");
    g_ptr[dev] = p;
  }
  *out = g_ptr[dev];
  return SPADE_OK;
}

}  // namespace attn_noalloc
}  // namespace spade

extern "C" spade_status spade_verify_attention_noalloc(
    const void *q, const void *k_cache, const void *v_cache, const int32_t *ctx_lens,
    const int32_t *n_draft, const int32_t *cu_q, void *out, float *lse, int32_t B, int32_t Hq,
    int32_t Hkv, int32_t D, int32_t cap, int32_t max_k, int32_t R, int32_t *status,
    spade_stream_t stream) {
  using namespace attn_noalloc;
  // The same size checks, in the same order and with the same codes, as
  // spade_verify_attention.
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0 || max_k < 0 || R <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention_noalloc: non-positive size");
  if (Hq % Hkv) return fail(SPADE_ERR_SHAPE, "Hq (%d) must be a multiple of Hkv (%d)", Hq, Hkv);
  if (D != 64 && D != 128) return fail(SPADE_ERR_SHAPE, "head dim %d not supported (64 or 128)", D);
  int dev = 0;
  spade_status st = device_info(nullptr, &dev);
  if (st != SPADE_OK) return st;
  if (dev >= kMaxDevices) return fail(SPADE_ERR_UNSUPPORTED_DEVICE, "device %d", dev);
  const size_t need = spade_attn_workspace_size(B, Hq, Hkv, D, cap, max_k);
  if (need == 0) return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention_noalloc: bad sizes");
  if (need > kScratchBytes)
    return fail(SPADE_ERR_CAPACITY,
                "spade_verify_attention_noalloc: these sizes need %zu bytes of scratch; the static "
                "scratch holds %zu bytes (use spade_verify_attention with a workspace)",
                need, kScratchBytes);
  void *scratch = nullptr;
  st = scratch_address(dev, &scratch);
  if (st != SPADE_OK) return st;
  // The merge counters must start at zero; the array keeps whatever the last
  // call (possibly an interrupted one) left there.
  const size_t units = static_cast<size_t>(B) * Hkv * attn::row_blocks(Hq / Hkv, max_k);
  const cudaError_t e = cudaMemsetAsync(scratch, 0, round_up(units * 4, 256),
                                        reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync(attention scratch counters)");
  return spade_verify_attention(q, k_cache, v_cache, ctx_lens, n_draft, cu_q, out, lse, B, Hq, Hkv,
                                D, cap, max_k, R, scratch, kScratchBytes, status, stream);
}
