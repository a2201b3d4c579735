// qkv_rope.cu -- the verifier's projection of the verify block into queries,
// keys and values, with rotary position embedding, writing the block's keys
// and values straight into its KV-cache slots.  This is the attention input
// side of f_l in x_{l+1} = x_l + f_l(x_l) (Sec. III-A) for the d+1 positions
// the verifier scores in a single forward pass (Sec. III-B, Algorithm 1 cloud
// step); the verify attention that follows reads those slots.
//
// Design (GB300):
//  * y = x W^T is a dense contraction, so it runs on the tensor cores:
//    tcgen05.mma kind::f16 (bf16 in, fp32 in tensor memory) with W's output
//    rows on the MMA M side (128-row tiles: one head of dimension 128, or two
//    of dimension 64, per tile) and the R verify rows on N.  At R = 72 the
//    work is bound by streaming W from HBM (50 MB for the Llama-3-8B layer),
//    so the grid is filled by splitting K: the `splits` CTAs of one tile form
//    a thread-block cluster, each accumulates its share of the k-chunks, and
//    the partial sums meet through distributed shared memory -- no workspace,
//    no second launch.
//  * Warp roles: warp 0 streams W and x tiles with TMA into a ring of stages;
//    warp 1 issues the MMAs (one elected thread) and owns the tensor memory;
//    warps 2-5 move the accumulator to shared memory and, after the cluster
//    barrier, sum the partials of their share of (row, dimension pair) items,
//    rotate query and key pairs (dimension j with j + D/2, angle pos *
//    theta^(-2j/D), pos = ctx_b + i) and store bf16: queries to q_out, keys and
//    values to cache slot ctx_b + i of their sequence.
//  * Programmatic dependent launch: barriers, tensor memory and tensor-map
//    prefetch come before the wait on the previous kernel; the attention that
//    follows may be scheduled while this kernel finishes.
#include <cuda_bf16.h>

#include <cstdint>

#include "internal.h"
#include "ptx.cuh"

namespace spade {
namespace qkv {

constexpr int kTileM = 128;                     // W rows per tile (MMA M)
constexpr int kKChunk = 64;                     // k elements per 128-byte swizzled row
constexpr int kWBytes = kTileM * kKChunk * 2;   // 16 KB: one W tile x one k-chunk
constexpr int kMaxR = 512;                      // verify rows per call
constexpr int kMaxSplits = 8;                   // portable cluster size
constexpr int kEpiWarps = 4;
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr int kRedCols = 256;                   // accumulator columns reduced per round
constexpr int kSmemBudget = 220 * 1024;
constexpr int kMaxStages = 8;

struct Params {
  const int32_t *ctx_lens;
  const int32_t *n_draft;
  const int32_t *cu_q;
  __nv_bfloat16 *q_out;    // [R, Hq, D]
  __nv_bfloat16 *k_cache;  // [B, Hkv, cap, D]
  __nv_bfloat16 *v_cache;  // [B, Hkv, cap, D]
  int32_t *status;
  int B, R, H, Hq, Hkv, D, cap, max_k;
  int splits;   // CTAs per tile (cluster size), each with a contiguous share of the k-chunks
  int KC;       // k-chunks (ceil(H / 64))
  int Ncols;    // R rounded up to 16: MMA N (two MMAs of <= 256 when above 256)
  int stages;   // ring depth
  uint32_t tmem_cols;
  float inv_freq[64];  // theta^(-2j/D), j < D/2, rounded from double on the host
  // Paged caches (block_table null: dense [B, Hkv, cap, D]): pools
  // [num_pages, Hkv, page_size, D], block_table [B, max_pages].
  const int32_t *block_table;
  int page_size, max_pages, num_pages;
};

// Shared-memory plan (offsets from a 1024-byte aligned base).
struct Layout {
  int stage_bytes, ring, rseq, rpos, bars, misc, total;
};
__host__ __device__ inline Layout layout(int Ncols, int stages) {
  Layout L;
  L.stage_bytes = kWBytes + Ncols * 128;
  L.ring = 0;
  L.rseq = stages * L.stage_bytes;   // int32 [kMaxR]: sequence of each row (-1: skip)
  L.rpos = L.rseq + kMaxR * 4;       // int32 [kMaxR]: position of each row
  L.bars = L.rpos + kMaxR * 4;       // full[stages], empty[stages], acc
  L.misc = L.bars + (2 * kMaxStages + 2) * 8;  // tmem base, abort flag
  L.total = L.misc + 64 + 1024;      // + slack for the 1024-byte alignment
  return L;
}

__global__ void __launch_bounds__(kThreads, 1)
    qkv_rope_kernel(const __grid_constant__ Params p, const __grid_constant__ CUtensorMap tm_w,
                    const __grid_constant__ CUtensorMap tm_x0, const __grid_constant__ CUtensorMap tm_x1) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const Layout L = layout(p.Ncols, p.stages);
  int32_t *s_rseq = reinterpret_cast<int32_t *>(smem + L.rseq);
  int32_t *s_rpos = reinterpret_cast<int32_t *>(smem + L.rpos);
  uint64_t *bar_full = reinterpret_cast<uint64_t *>(smem + L.bars);
  uint64_t *bar_empty = bar_full + kMaxStages;
  uint64_t *bar_acc = bar_empty + kMaxStages;
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + L.misc);
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + L.misc + 8);

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int S = p.splits;
  const int rank = static_cast<int>(blockIdx.x) % S;  // == %cluster_ctarank (clusters along x)
  const int tile = static_cast<int>(blockIdx.x) / S;
  const int kc0 = p.KC * rank / S, kc1 = p.KC * (rank + 1) / S;
  const int nk = kc1 - kc0;

  // ---- set-up that reads no input -----------------------------------------
  if (tid == 0) *s_abort = 0;
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_w);
    tma_prefetch_desc(&tm_x0);
    if (p.Ncols > 256) tma_prefetch_desc(&tm_x1);
  } else if (warp == 1) {
    if (lane == 0) {
      for (int s = 0; s < p.stages; ++s) {
        mbar_init(&bar_full[s], 1);
        mbar_init(&bar_empty[s], 1);
      }
      mbar_init(bar_acc, 1);
      fence_mbar_init();
    }
    __syncwarp();
    tmem_alloc(s_tmem, p.tmem_cols);
    tmem_relinquish();
  }
  griddep_wait();
  griddep_launch_dependents();
  // ---- row table: sequence and position of every verify row ---------------
  for (int r = tid; r < p.R; r += kThreads) s_rseq[r] = -1;
  __syncthreads();
  for (int b = tid; b < p.B; b += kThreads) {
    const int c = p.ctx_lens[b], k = p.n_draft[b];
    const int q0 = p.cu_q[b], q1 = p.cu_q[b + 1];
    int bad = 0;
    if (c < 0 || k < 0 || k > p.max_k || q0 < 0 || q1 > p.R || q1 - q0 != k + 1) bad = SPADE_DEV_BAD_INDEX;
    else if (static_cast<int64_t>(c) + k + 1 > p.cap) bad = SPADE_DEV_CAPACITY;
    if (bad) {
      if (blockIdx.x == 0) atomicOr(p.status, bad);
      continue;
    }
    if (p.block_table) {
      // Every page the block writes must exist.
      for (int i = 0; i <= k; ++i) {
        const int pg = p.block_table[static_cast<int64_t>(b) * p.max_pages + (c + i) / p.page_size];
        if (pg < 0 || pg >= p.num_pages) bad = SPADE_DEV_BAD_INDEX;
      }
      if (bad) {
        if (blockIdx.x == 0) atomicOr(p.status, bad);
        continue;
      }
    }
    for (int i = 0; i <= k; ++i) {
      s_rseq[q0 + i] = b;
      s_rpos[q0 + i] = c + i;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  const uint32_t smem_base = smem_u32(smem);
  const int n0 = p.Ncols > 256 ? 256 : p.Ncols;  // first MMA N-chunk (and x box rows)
  const int n1 = p.Ncols - n0;                   // second N-chunk, 0 if none

  if (warp == 0) {
    // ============================ producer: TMA ============================
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first();  // W streams once
      const uint64_t pol_x = l2_policy_evict_last();   // x is re-read by every tile
      const uint32_t bytes = kWBytes + p.Ncols * 128;
      bool expired = false;
      int issued = 0;
      for (int i = 0; i < nk; ++i) {
        const int st = i % p.stages;
        const uint32_t ph = (i / p.stages) & 1;
        if (!mbar_wait(&bar_empty[st], ph ^ 1, s_abort)) expired = true;
        if (*s_abort) break;
        issued = i + 1;
        uint8_t *stage = smem + L.ring + st * L.stage_bytes;
        const int kx = (kc0 + i) * kKChunk;
        mbar_arrive_expect_tx(&bar_full[st], bytes);
        tma_load_2d(stage, &tm_w, kx, tile * kTileM, &bar_full[st], pol_w);
        tma_load_2d(stage + kWBytes, &tm_x0, kx, 0, &bar_full[st], pol_x);
        if (n1) tma_load_2d(stage + kWBytes + n0 * 128, &tm_x1, kx, n0, &bar_full[st], pol_x);
      }
      if (expired || *s_abort) {
        atomicOr(p.status, SPADE_DEV_TIMEOUT);
        // Drain: every copy issued must land before shared memory goes away.
        for (int i = (issued > p.stages ? issued - p.stages : 0); i < issued; ++i)
          mbar_wait_unabortable(&bar_full[i % p.stages], (i / p.stages) & 1);
      }
    }
  } else if (warp == 1) {
    // ============================ MMA issuer ===============================
    if (lane == 0) {
      const uint32_t idesc0 = idesc_bf16_f32(kTileM, n0);
      const uint32_t idesc1 = idesc_bf16_f32(kTileM, n1 ? n1 : 16);
      bool expired = false;
      for (int i = 0; i < nk; ++i) {
        const int st = i % p.stages;
        const uint32_t ph = (i / p.stages) & 1;
        if (!mbar_wait(&bar_full[st], ph, s_abort)) expired = true;
        tc_fence_after();
        if (!*s_abort) {
          const uint32_t a = smem_base + L.ring + st * L.stage_bytes;
          const uint32_t b = a + kWBytes;
#pragma unroll
          for (int kk = 0; kk < kKChunk / 16; ++kk) {
            const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
            tc_mma_f16(tmem, smem_desc_sw128(a + kk * 32), smem_desc_sw128(b + kk * 32), idesc0, acc);
            if (n1)
              tc_mma_f16(tmem + 256, smem_desc_sw128(a + kk * 32), smem_desc_sw128(b + n0 * 128 + kk * 32),
                         idesc1, acc);
          }
        }
        tc_commit(&bar_empty[st]);
      }
      tc_commit(bar_acc);  // arrives once every MMA above is done (at once if none)
      if (expired) atomicOr(p.status, SPADE_DEV_TIMEOUT);
    }
  }


  // ======================= epilogue (every thread) =========================
  // Rounds of up to 256 accumulator columns: warps 2-5 move their tensor-memory
  // lane quadrant to shared memory (the ring is free once the MMAs are done),
  // the cluster barrier makes every CTA's partial visible, then the cluster's
  // CTAs share the round's (row, dimension pair) items: each sums the partials
  // of the split-K CTAs from distributed shared memory, rotates query and key
  // pairs and stores bf16; a second barrier keeps every CTA's partial alive
  // until all have read it.
  float *red = reinterpret_cast<float *>(smem + L.ring);  // [kRedCols][128]
  uint32_t red_rank[kMaxSplits];
#pragma unroll
  for (int s = 0; s < kMaxSplits; ++s) red_rank[s] = s < S ? cluster_map(red, s) : 0u;
  const int hpt = kTileM / p.D;  // heads per tile
  const int half = p.D / 2;
  bool acc_ready = false;
  for (int c0 = 0; c0 < p.Ncols; c0 += kRedCols) {
    const int nc = min(kRedCols, p.Ncols - c0);
    if (warp >= 2) {
      const int q4 = warp & 3;  // tensor-memory lane quadrant this warp may access
      if (!acc_ready) {
        if (!mbar_wait(bar_acc, 0, s_abort)) atomicOr(p.status, SPADE_DEV_TIMEOUT);
        tc_fence_after();
        acc_ready = true;
      }
      const uint32_t tl = tmem + (static_cast<uint32_t>(q4 * 32) << 16) + static_cast<uint32_t>(c0);
      for (int c = 0; c < nc; c += 8) {
        uint32_t v[8];
        tmem_ld8(tl + c, v);
        tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < 8; ++e) red[(c + e) * kTileM + q4 * 32 + lane] = __uint_as_float(v[e]);
      }
    }
    __syncwarp();
    cluster_sync();
    // Items are (row, 4 consecutive dimension pairs of one head): two float4
    // loads per split CTA, all issued before any is used.
    constexpr int kQuads = kTileM / 8;  // quads of pairs per accumulator column
    const int items = nc * kQuads;
    const int i0 = items * rank / S, i1 = items * (rank + 1) / S;
    for (int it = i0 + tid; it < i1; it += kThreads) {
      const int col = it / kQuads, qd = it % kQuads;
      const int r = c0 + col;
      if (r >= p.R) continue;
      const int b = s_rseq[r];
      if (b < 0) continue;
      const int pp = qd * 4;  // first pair of the quad
      const int hloc = pp / half, j0 = pp % half;
      const int d1 = hloc * p.D + j0;
      const uint32_t off1 = static_cast<uint32_t>((col * kTileM + d1) * 4);
      const uint32_t off2 = off1 + static_cast<uint32_t>(half * 4);
      float4 a[kMaxSplits], c[kMaxSplits];
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s) {
        if (s < S) {
          a[s] = ld_dsmem_f32x4(red_rank[s] + off1);
          c[s] = ld_dsmem_f32x4(red_rank[s] + off2);
        }
      }
      float y1[4] = {0.f, 0.f, 0.f, 0.f}, y2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int s = 0; s < kMaxSplits; ++s) {
        if (s < S) {
          y1[0] += a[s].x; y1[1] += a[s].y; y1[2] += a[s].z; y1[3] += a[s].w;
          y2[0] += c[s].x; y2[1] += c[s].y; y2[2] += c[s].z; y2[3] += c[s].w;
        }
      }
      const int hg = tile * hpt + hloc;  // head among the Hq + 2 Hkv of the projection
      const int pos = s_rpos[r];
      if (hg < p.Hq + p.Hkv) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float sn, cs;
          sincosf(static_cast<float>(pos) * p.inv_freq[j0 + e], &sn, &cs);
          const float o1 = y1[e] * cs - y2[e] * sn, o2 = y2[e] * cs + y1[e] * sn;
          y1[e] = o1;
          y2[e] = o2;
        }
      }
      __nv_bfloat16 *dst;
      if (hg < p.Hq) {
        dst = p.q_out + (static_cast<size_t>(r) * p.Hq + hg) * p.D;
      } else {
        const int hk = hg < p.Hq + p.Hkv ? hg - p.Hq : hg - p.Hq - p.Hkv;
        __nv_bfloat16 *cache = hg < p.Hq + p.Hkv ? p.k_cache : p.v_cache;
        if (p.block_table) {
          const int pg = p.block_table[static_cast<int64_t>(b) * p.max_pages + pos / p.page_size];
          dst = cache + ((static_cast<size_t>(pg) * p.Hkv + hk) * p.page_size + pos % p.page_size) * p.D;
        } else {
          dst = cache + ((static_cast<size_t>(b) * p.Hkv + hk) * p.cap + pos) * p.D;
        }
      }
      // 4 bf16 = 8 bytes at each half (j0 is a multiple of 4, rows 16-byte aligned).
      *reinterpret_cast<uint2 *>(dst + j0) = make_uint2(pack_bf16(y1[0], y1[1]), pack_bf16(y1[2], y1[3]));
      *reinterpret_cast<uint2 *>(dst + j0 + half) = make_uint2(pack_bf16(y2[0], y2[1]), pack_bf16(y2[2], y2[3]));
    }
    __syncwarp();
    cluster_sync();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, p.tmem_cols);
  }
}

}  // namespace qkv
}  // namespace spade

namespace spade {
namespace qkv {

// Clusters of `splits` CTAs (with `smem` bytes each) that the device can hold
// at once; 0 if the query fails.
static int max_active_clusters(int splits, int smem) {
  static int cache[kMaxSplits + 1][2] = {};
  static int cached_smem[kMaxSplits + 1] = {};
  if (cached_smem[splits] == smem && cache[splits][0]) return cache[splits][1];
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(splits);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, qkv_rope_kernel, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  cache[splits][0] = 1;
  cache[splits][1] = n;
  cached_smem[splits] = smem;
  return n;
}

}  // namespace qkv
}  // namespace spade

using namespace spade;

namespace spade {
namespace qkv {
struct Paging {
  const int32_t *block_table;
  int page_size, max_pages, num_pages;
};
}  // namespace qkv
}  // namespace spade

static spade_status qkv_rope_impl(const void *x, const void *w_qkv, const int32_t *ctx_lens,
                                  const int32_t *n_draft, const int32_t *cu_q, void *q_out, void *k_cache,
                                  void *v_cache, int32_t B, int32_t R, int32_t H, int32_t Hq, int32_t Hkv,
                                  int32_t D, int32_t cap, int32_t max_k, float rope_theta, int32_t *status,
                                  spade_stream_t stream, const qkv::Paging *pg) {
  using namespace qkv;
  if (!x || !w_qkv || !ctx_lens || !n_draft || !cu_q || !q_out || !k_cache || !v_cache || !status)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_qkv_rope: null pointer argument");
  if (B <= 0 || R < B || H <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0 || max_k < 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_qkv_rope: bad sizes B=%d R=%d H=%d Hq=%d Hkv=%d cap=%d",
                B, R, H, Hq, Hkv, cap);
  if (!(rope_theta > 1.f) || rope_theta != rope_theta || rope_theta > 3.0e38f)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_qkv_rope: rope_theta must be finite and > 1");
  if (Hq % Hkv) return fail(SPADE_ERR_SHAPE, "Hq (%d) must be a multiple of Hkv (%d)", Hq, Hkv);
  if (D != 64 && D != 128) return fail(SPADE_ERR_SHAPE, "head dim %d not supported (64 or 128)", D);
  if ((Hq + 2 * Hkv) * D % kTileM)
    return fail(SPADE_ERR_SHAPE, "(Hq + 2 Hkv) * D = %d must be a multiple of %d", (Hq + 2 * Hkv) * D, kTileM);
  if (H % 8) return fail(SPADE_ERR_SHAPE, "hidden size %d must be a multiple of 8", H);
  if (R > kMaxR) return fail(SPADE_ERR_SHAPE, "R = %d verify rows exceed %d per call", R, kMaxR);
  if (!aligned(x, 16) || !aligned(w_qkv, 16) || !aligned(q_out, 16) || !aligned(k_cache, 16) ||
      !aligned(v_cache, 16))
    return fail(SPADE_ERR_INVALID_ARG, "x, w_qkv, q_out and the caches must be 16-byte aligned");
  int sms = 0;
  spade_status st = device_info(&sms, nullptr);
  if (st != SPADE_OK) return st;

  Params p{};
  p.ctx_lens = ctx_lens;
  p.n_draft = n_draft;
  p.cu_q = cu_q;
  p.q_out = static_cast<__nv_bfloat16 *>(q_out);
  p.k_cache = static_cast<__nv_bfloat16 *>(k_cache);
  p.v_cache = static_cast<__nv_bfloat16 *>(v_cache);
  p.status = status;
  p.B = B; p.R = R; p.H = H; p.Hq = Hq; p.Hkv = Hkv; p.D = D; p.cap = cap; p.max_k = max_k;
  p.block_table = pg ? pg->block_table : nullptr;
  p.page_size = pg ? pg->page_size : 0;
  p.max_pages = pg ? pg->max_pages : 0;
  p.num_pages = pg ? pg->num_pages : 0;
  p.KC = (H + kKChunk - 1) / kKChunk;
  p.Ncols = (R + 15) / 16 * 16;
  p.tmem_cols = 32;
  while (p.tmem_cols < static_cast<uint32_t>(p.Ncols)) p.tmem_cols *= 2;
  for (int j = 0; j < D / 2; ++j) p.inv_freq[j] = static_cast<float>(pow(static_cast<double>(rope_theta), -2.0 * j / D));
  const int tiles = (Hq + 2 * Hkv) * D / kTileM;
  // Ring: as many stages as fit, at least two, holding at least one round of
  // the reduction buffer (256 columns x 128 rows of fp32) once the MMAs are done.
  const int stage = kWBytes + p.Ncols * 128;
  const int fixed = layout(p.Ncols, 0).total;
  p.stages = (kSmemBudget - fixed) / stage;
  if (p.stages > kMaxStages) p.stages = kMaxStages;
  const int red = (p.Ncols < kRedCols ? p.Ncols : kRedCols) * kTileM * 4;
  if (p.stages < 2 || p.stages * stage < red)
    return fail(SPADE_ERR_SHAPE, "shared memory too small for R = %d", R);
  const int smem = layout(p.Ncols, p.stages).total;
  static bool configured = false;
  if (!configured) {
    // The plan above never exceeds kSmemBudget (alignment slack included).
    cudaError_t e = cudaFuncSetAttribute(qkv_rope_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemBudget);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(qkv_rope)");
    configured = true;
  }
  // Split K over a cluster of CTAs per tile so the grid fills the SMs, as
  // long as every cluster of the grid fits on the device at once.
  int S = sms / tiles;
  if (S > kMaxSplits) S = kMaxSplits;
  if (S > p.KC) S = p.KC;
  if (S < 1) S = 1;
  while (S > 1 && max_active_clusters(S, smem) < tiles) --S;
  p.splits = S;

  CUtensorMap tw, tx0, tx1;
  const int n0 = p.Ncols > 256 ? 256 : p.Ncols;
  const int n1 = p.Ncols - n0;
  if (!encode_tmap_bf16_sw128(&tw, w_qkv, H, static_cast<uint64_t>(Hq + 2 * Hkv) * D, static_cast<uint64_t>(H) * 2,
                              kKChunk, kTileM) ||
      !encode_tmap_bf16_sw128(&tx0, x, H, R, static_cast<uint64_t>(H) * 2, kKChunk, n0) ||
      !encode_tmap_bf16_sw128(&tx1, x, H, R, static_cast<uint64_t>(H) * 2, kKChunk, n1 ? n1 : 16))
    return SPADE_ERR_CUDA;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(tiles * S);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = reinterpret_cast<cudaStream_t>(stream);
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, qkv_rope_kernel, p, tw, tx0, tx1);
  if (e != cudaSuccess) return cuda_fail(e, "qkv_rope launch");
  return SPADE_OK;
}

extern "C" spade_status spade_verify_qkv_rope(const void *x, const void *w_qkv, const int32_t *ctx_lens,
                                              const int32_t *n_draft, const int32_t *cu_q, void *q_out,
                                              void *k_cache, void *v_cache, int32_t B, int32_t R,
                                              int32_t H, int32_t Hq, int32_t Hkv, int32_t D, int32_t cap,
                                              int32_t max_k, float rope_theta, int32_t *status,
                                              spade_stream_t stream) {
  return qkv_rope_impl(x, w_qkv, ctx_lens, n_draft, cu_q, q_out, k_cache, v_cache, B, R, H, Hq, Hkv, D, cap,
                       max_k, rope_theta, status, stream, nullptr);
}

extern "C" spade_status spade_verify_qkv_rope_paged(const void *x, const void *w_qkv,
                                                    const int32_t *block_table, const int32_t *ctx_lens,
                                                    const int32_t *n_draft, const int32_t *cu_q, void *q_out,
                                                    void *k_pool, void *v_pool, int32_t B, int32_t R,
                                                    int32_t H, int32_t Hq, int32_t Hkv, int32_t D,
                                                    int32_t page_size, int32_t num_pages, int32_t max_pages,
                                                    int32_t max_k, float rope_theta, int32_t *status,
                                                    spade_stream_t stream) {
  if (!block_table) return fail(SPADE_ERR_INVALID_ARG, "spade_verify_qkv_rope_paged: null block_table");
  if (page_size <= 0 || num_pages <= 0 || max_pages <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_qkv_rope_paged: non-positive page geometry");
  if (static_cast<int64_t>(max_pages) * page_size >= (int64_t(1) << 31))
    return fail(SPADE_ERR_CAPACITY, "max_pages * page_size exceeds 2^31");
  const qkv::Paging pg{block_table, page_size, max_pages, num_pages};
  return qkv_rope_impl(x, w_qkv, ctx_lens, n_draft, cu_q, q_out, k_pool, v_pool, B, R, H, Hq, Hkv, D,
                       max_pages * page_size, max_k, rope_theta, status, stream, &pg);
}
