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
//    work is bound by streaming W from HBM (50 MB for the Llama-3-8B layer).
//  * Stream-K over (tile, k-chunk of 64) units: the units are laid end to end
//    and cut into one equal range per SM, so every SM streams the same share
//    of W whatever the tile count.  A ring stage holds up to KG = 2 chunks of
//    one tile (two consecutive chunks of the range in the same tile arrive as
//    one 3-D box of 128 rows x 256 contiguous bytes; KG = 1 when H is not a
//    multiple of 64).  A CTA's range covers pieces of one to three
//    tiles ("segments"); each segment accumulates in one of two tensor-memory
//    buffers (the next segment's MMAs start while the last one is drained),
//    and its fp32 partial goes to the CTA's own workspace slot.  A tile
//    computed by one CTA is finished by that CTA.  A tile split over several
//    CTAs is finished by the CTA whose part arrives last, or, when the grid
//    has CTAs to spare (two or more per tile), after every CTA's stream in
//    row slabs spread over the whole grid (the launch is cooperative, so
//    every CTA is resident and a slab's CTA may wait for the tile's parts).
//    Either way the parts are summed in CTA order -- the same order every
//    call, so results do not depend on arrival order -- and the finisher rotates
//    query and key pairs (dimension j with j + D/2, angle pos *
//    theta^(-2j/D), pos = ctx_b + i) and stores bf16: queries to q_out, keys
//    and values to cache slot ctx_b + i of their sequence (or, for a paged
//    cache, where the block table puts that slot).
//  * Warp roles: warp 0 streams W and x tiles with TMA into a ring of stages;
//    warp 1 issues the MMAs (one elected thread) and owns the tensor memory;
//    warps 2-5 drain accumulators, publish partials and run the reduction.
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
constexpr int kEpiWarps = 4;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr int kSmemBudget = 220 * 1024;
constexpr int kMaxStages = 8;


struct Params {
  const int32_t *ctx_lens;
  const int32_t *n_draft;
  const int32_t *cu_q;
  __nv_bfloat16 *q_out;    // [R, Hq, D]
  __nv_bfloat16 *k_cache;  // [B, Hkv, cap, D] (or a pool, see block_table)
  __nv_bfloat16 *v_cache;
  int32_t *status;
  float *partials;         // [num_ctas + tiles slots][Ncols][128] fp32 (workspace)
  int32_t *counters;       // [2][tiles]: parts published, slabs done; zero between calls (workspace)
  int B, R, H, Hq, Hkv, D, cap, max_k;
  int tiles;    // (Hq + 2 Hkv) D / 128
  int KC;       // k-chunks (ceil(H / 64))
  int KG;       // k-chunks per ring stage at most (1 or 2; 2 only when H is a multiple of 64)
  int units;    // tiles * KC
  int num_ctas;
  int Ncols;    // R rounded up to 16: MMA N (two MMAs of <= 256 when above 256)
  int stages;   // ring depth
  int nbuf;     // accumulator buffers (2 when two fit in tensor memory)
  int slabs;    // row slabs per split tile in the final reduction
  uint32_t buf_cols, tmem_cols;
  float inv_freq[64];  // theta^(-2j/D), j < D/2, rounded from double on the host
  // Paged caches (block_table null: dense [B, Hkv, cap, D]): pools
  // [num_pages, Hkv, page_size, D], block_table [B, max_pages].
  const int32_t *block_table;
  int page_size, max_pages, num_pages;
};

// Shared-memory plan (offsets from a 1024-byte aligned base).
struct Layout {
  int stage_bytes, ring, rseq, rpos, bars, misc, freq, total;
};
__host__ __device__ inline Layout layout(int Ncols, int stages, int KG) {
  Layout L;
  L.stage_bytes = KG * (kWBytes + Ncols * 128);  // KG W chunks, then KG x chunks
  L.ring = 0;
  L.rseq = stages * L.stage_bytes;   // int32 [kMaxR]: sequence of each row (-1: skip)
  L.rpos = L.rseq + kMaxR * 4;       // int32 [kMaxR]: position of each row
  L.bars = L.rpos + kMaxR * 4;       // full[stages], empty[stages], acc_full[2], acc_empty[2]
  L.misc = L.bars + (2 * kMaxStages + 4) * 8;  // tmem base, abort flag, last-arrival flag
  L.freq = L.misc + 64;              // float [64]: rotary frequencies (per-thread indices
                                     // into the parameter array would serialise)
  L.total = L.freq + 64 * 4 + 1024;  // + slack for the 1024-byte alignment
  return L;
}

// Unit range [u0, u1) of CTA i, and the CTA whose range holds unit u.
__host__ __device__ inline int range_lo(int units, int n, int i) {
  return static_cast<int>(static_cast<int64_t>(units) * i / n);
}
__device__ inline int unit_owner(int units, int n, int u) {
  return static_cast<int>((static_cast<int64_t>(u + 1) * n + units - 1) / units - 1);
}

// Publication of one partial at its tile's counter (one thread, after a
// barrier that orders the partial's stores before it).
__device__ __forceinline__ void publish_part(int32_t *counter) {
  asm volatile("red.release.gpu.global.add.s32 [%0], 1;" ::"l"(counter) : "memory");
}
__device__ __forceinline__ int load_acquire(const int32_t *a) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(a) : "memory");
  return v;
}
__device__ __forceinline__ int add_acq_rel(int32_t *a, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(a), "r"(v) : "memory");
  return old;
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory"); }


// Sine and cosine of pos * f: the product as an exact pair (a + e == pos * f),
// reduced to [-pi, pi] with 2 pi split in two parts (Cody and Waite's method),
// then the SFU's sine and cosine (accurate to a few 1e-7 on that interval).
__device__ __forceinline__ void rope_angle(int pos, float f, float *sn, float *cs) {
  const float x = static_cast<float>(pos);  // exact: positions are below 2^24
  const float a = x * f;
  const float e = fmaf(x, f, -a);
  const float k = rintf(a * 0.15915494309189535f);           // 1 / (2 pi)
  float r = fmaf(-k, 6.28318548202514648f, a);               // 2 pi rounded to float
  r = fmaf(-k, -1.7484555314695172e-07f, r);                 // 2 pi minus that
  __sincosf(r + e, sn, cs);
}

// The reduction of verify rows [r0, r1) of tile t once every part has been
// published: for each row and each 4 consecutive dimension pairs of a head
// (thread th of nth takes items th, th + nth, ...), the sum of the partials
// of CTAs c_first .. c_first + nparts - 1 in that order, the rotation of
// query and key pairs and the bf16 stores (q_out, or the cache slot ctx_b + i
// of the row's sequence).  Each thread takes kIB items at a time and issues
// the loads of every item and kPB parts before using any (the reduction is
// bound by L2 latency, so the rounds of loads are what it costs).
template <int kIB, int kPB>
__device__ __noinline__ void reduce_tile(const Params &p, const int32_t *s_rseq, const int32_t *s_rpos,
                                         const float *s_freq, int t, int c_first, int nparts, int r0,
                                         int r1, int th, int nth) {
  // Every field used below in a local: the stores through dst could alias
  // the parameter block as far as the compiler knows, and it would reload them.
  const int D = p.D, Hq = p.Hq, Hkv = p.Hkv, cap = p.cap, Ncols = p.Ncols;
  const int max_pages = p.max_pages, page_size = p.page_size;
  const int32_t *block_table = p.block_table;
  __nv_bfloat16 *q_out = p.q_out, *k_cache = p.k_cache, *v_cache = p.v_cache;
  const float *partials = p.partials;
  const int half = D / 2;
  const int hpt = kTileM / D;  // heads per tile
  // Items: (row, 4 consecutive dimension pairs of one head); partials summed
  // in CTA order c_first .. c_last, every load of an item issued first.
  constexpr int kQuads = kTileM / 8;
  const float *base = partials + static_cast<size_t>(c_first + t) * Ncols * kTileM;
  const size_t slot = static_cast<size_t>(Ncols) * kTileM;
  const int nitems = (r1 - r0) * kQuads;
  for (int it0 = th; it0 < nitems; it0 += nth * kIB) {
    int rr[kIB], d1[kIB], hl[kIB], jj[kIB], bb[kIB];
    float y1[kIB][4], y2[kIB][4];
#pragma unroll
    for (int i = 0; i < kIB; ++i) {
      const int it = it0 + i * nth;
      rr[i] = it < nitems ? r0 + it / kQuads : 0;
      const int pp = (it % kQuads) * 4;
      hl[i] = pp / half;
      jj[i] = pp % half;
      d1[i] = hl[i] * D + jj[i];
      bb[i] = it < nitems ? s_rseq[rr[i]] : -1;
#pragma unroll
      for (int e = 0; e < 4; ++e) y1[i][e] = y2[i][e] = 0.f;
    }
    for (int s0 = 0; s0 < nparts; s0 += kPB) {
      float4 a[kIB][kPB], c[kIB][kPB];
#pragma unroll
      for (int i = 0; i < kIB; ++i)
#pragma unroll
        for (int s = 0; s < kPB; ++s)
          if (bb[i] >= 0 && s0 + s < nparts) {
            const float *ps = base + (s0 + s) * slot + rr[i] * kTileM + d1[i];
            a[i][s] = __ldcg(reinterpret_cast<const float4 *>(ps));
            c[i][s] = __ldcg(reinterpret_cast<const float4 *>(ps + half));
          }
#pragma unroll
      for (int i = 0; i < kIB; ++i)
#pragma unroll
        for (int s = 0; s < kPB; ++s)
          if (bb[i] >= 0 && s0 + s < nparts) {
            y1[i][0] += a[i][s].x; y1[i][1] += a[i][s].y; y1[i][2] += a[i][s].z; y1[i][3] += a[i][s].w;
            y2[i][0] += c[i][s].x; y2[i][1] += c[i][s].y; y2[i][2] += c[i][s].z; y2[i][3] += c[i][s].w;
          }
    }
#pragma unroll
    for (int i = 0; i < kIB; ++i) {
      const int b = bb[i];
      if (b < 0) continue;
      const int r = rr[i], j0 = jj[i];
      const int hg = t * hpt + hl[i];  // head among the Hq + 2 Hkv of the projection
      const int pos = s_rpos[r];
      if (hg < Hq + Hkv) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float sn, cs;
          rope_angle(pos, s_freq[j0 + e], &sn, &cs);
          const float o1 = y1[i][e] * cs - y2[i][e] * sn, o2 = y2[i][e] * cs + y1[i][e] * sn;
          y1[i][e] = o1;
          y2[i][e] = o2;
        }
      }
      __nv_bfloat16 *dst;
      if (hg < Hq) {
        dst = q_out + (static_cast<size_t>(r) * Hq + hg) * D;
      } else {
        const int hk = hg < Hq + Hkv ? hg - Hq : hg - Hq - Hkv;
        __nv_bfloat16 *cache = hg < Hq + Hkv ? k_cache : v_cache;
        if (block_table) {
          const int pg = block_table[static_cast<int64_t>(b) * max_pages + pos / page_size];
          dst = cache + ((static_cast<size_t>(pg) * Hkv + hk) * page_size + pos % page_size) * D;
        } else {
          dst = cache + ((static_cast<size_t>(b) * Hkv + hk) * cap + pos) * D;
        }
      }
      // 4 bf16 = 8 bytes at each half (j0 a multiple of 4, rows 16-byte aligned).
      *reinterpret_cast<uint2 *>(dst + j0) =
          make_uint2(pack_bf16(y1[i][0], y1[i][1]), pack_bf16(y1[i][2], y1[i][3]));
      *reinterpret_cast<uint2 *>(dst + j0 + half) =
          make_uint2(pack_bf16(y2[i][0], y2[i][1]), pack_bf16(y2[i][2], y2[i][3]));
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    qkv_rope_kernel(const __grid_constant__ Params p, const __grid_constant__ CUtensorMap tm_w,
                    const __grid_constant__ CUtensorMap tm_x0, const __grid_constant__ CUtensorMap tm_x1,
                    const __grid_constant__ CUtensorMap tm_w3) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const Layout L = layout(p.Ncols, p.stages, p.KG);
  int32_t *s_rseq = reinterpret_cast<int32_t *>(smem + L.rseq);
  int32_t *s_rpos = reinterpret_cast<int32_t *>(smem + L.rpos);
  uint64_t *bar_full = reinterpret_cast<uint64_t *>(smem + L.bars);
  uint64_t *bar_empty = bar_full + kMaxStages;
  uint64_t *acc_full = bar_empty + kMaxStages;  // [2]
  uint64_t *acc_empty = acc_full + 2;           // [2]
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + L.misc);
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + L.misc + 8);
  float *s_freq = reinterpret_cast<float *>(smem + L.freq);
  volatile int *s_last = reinterpret_cast<volatile int *>(smem + L.misc + 16);
  volatile int *s_fin = reinterpret_cast<volatile int *>(smem + L.misc + 32);  // last tile, c_first, nparts; slab flag

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int u0 = range_lo(p.units, p.num_ctas, blockIdx.x);
  const int u1 = range_lo(p.units, p.num_ctas, blockIdx.x + 1);

  // ---- set-up that reads no input -----------------------------------------
  if (tid == 0) { *s_abort = 0; s_fin[0] = -1; }
  for (int j = tid; j < 64; j += kThreads) s_freq[j] = p.inv_freq[j];
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(p.KG > 1 ? &tm_w3 : &tm_w);
    tma_prefetch_desc(&tm_x0);
    if (p.Ncols > 256) tma_prefetch_desc(&tm_x1);
  } else if (warp == 1) {
    if (lane == 0) {
      for (int s = 0; s < p.stages; ++s) {
        mbar_init(&bar_full[s], 1);
        mbar_init(&bar_empty[s], 1);
      }
      for (int b = 0; b < 2; ++b) {
        mbar_init(&acc_full[b], 1);
        mbar_init(&acc_empty[b], kEpiWarps);
      }
      fence_mbar_init();
    }
    __syncwarp();
    tmem_alloc(s_tmem, p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();  // barriers and the tensor-memory allocation
  tc_fence_after();
  // Inputs written by earlier kernels in the stream are visible from here on.
  griddep_wait();
  griddep_launch_dependents();
  const uint32_t tmem = *s_tmem;
  const uint32_t smem_base = smem_u32(smem);
  const int n0 = p.Ncols > 256 ? 256 : p.Ncols;  // first MMA N-chunk (and x box rows)
  const int n1 = p.Ncols - n0;                   // second N-chunk, 0 if none

  if (warp == 0) {
    // ============================ producer: TMA ============================
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first();  // W streams once
      const uint64_t pol_x = l2_policy_evict_last();   // x is re-read for every unit
      const uint32_t xbytes = p.Ncols * 128;  // x rows of one k-chunk
      bool expired = false;
      int issued = 0;
      for (int u = u0, i = 0; u < u1; ++i) {
        const int st = i % p.stages;
        const uint32_t ph = (i / p.stages) & 1;
        if (!mbar_wait(&bar_empty[st], ph ^ 1, s_abort)) expired = true;
        if (*s_abort) break;
        issued = i + 1;
        uint8_t *stage = smem + L.ring + st * L.stage_bytes;
        const int t = u / p.KC, c0 = u - t * p.KC;
        const int nch = min(p.KG, min(u1, (t + 1) * p.KC) - u);  // chunks of one tile and this range
        mbar_arrive_expect_tx(&bar_full[st], nch * (kWBytes + xbytes));
        if (nch > 1)
          tma_load_3d(stage, &tm_w3, 0, t * kTileM, c0, &bar_full[st], pol_w);  // nch chunks, 16 KB apart
        else
          tma_load_2d(stage, &tm_w, c0 * kKChunk, t * kTileM, &bar_full[st], pol_w);
        uint8_t *xs = stage + p.KG * kWBytes;
        for (int j = 0; j < nch; ++j) {
          tma_load_2d(xs + j * xbytes, &tm_x0, (c0 + j) * kKChunk, 0, &bar_full[st], pol_x);
          if (n1) tma_load_2d(xs + j * xbytes + n0 * 128, &tm_x1, (c0 + j) * kKChunk, n0, &bar_full[st], pol_x);
        }
        u += nch;
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
      int i = 0, seg = 0;
      for (int u = u0; u < u1; ++seg) {
        const int t = u / p.KC;
        const int se = min(u1, (t + 1) * p.KC);
        const int buf = seg % p.nbuf, use = seg / p.nbuf;
        // The buffer's previous segment has been drained by the epilogue warps.
        if (use > 0 && !mbar_wait(&acc_empty[buf], (use - 1) & 1, s_abort)) expired = true;
        tc_fence_after();
        const uint32_t acc_addr = tmem + static_cast<uint32_t>(buf) * p.buf_cols;
        for (const int us = u; u < se; ++i) {
          const int st = i % p.stages;
          const uint32_t ph = (i / p.stages) & 1;
          const int nch = min(p.KG, se - u);  // as the producer cut the stage
          if (!mbar_wait(&bar_full[st], ph, s_abort)) expired = true;
          tc_fence_after();
          if (!*s_abort) {
            const uint32_t a0 = smem_base + L.ring + st * L.stage_bytes;
            for (int j = 0; j < nch; ++j) {
              const uint32_t a = a0 + j * kWBytes;
              const uint32_t b = a0 + p.KG * kWBytes + j * p.Ncols * 128;
#pragma unroll
              for (int kk = 0; kk < kKChunk / 16; ++kk) {
                const uint32_t acc = (u > us || j > 0 || kk > 0) ? 1u : 0u;
                tc_mma_f16(acc_addr, smem_desc_sw128(a + kk * 32), smem_desc_sw128(b + kk * 32), idesc0, acc);
                if (n1)
                  tc_mma_f16(acc_addr + 256, smem_desc_sw128(a + kk * 32),
                             smem_desc_sw128(b + n0 * 128 + kk * 32), idesc1, acc);
              }
            }
          }
          tc_commit(&bar_empty[st]);
          u += nch;
        }
        tc_commit(&acc_full[buf]);
      }
      if (expired) atomicOr(p.status, SPADE_DEV_TIMEOUT);
    }
  } else {
    // ===================== epilogue warps: drain, publish, reduce ==========
    const int et = tid - 64;         // 0..127
    const int q4 = warp & 3;         // tensor-memory lane quadrant this warp may access
    // Row table: sequence and position of every verify row.  Only the tile
    // reductions read it, so it is built here while the producer and the MMA
    // warp already stream the first units.
    for (int r = et; r < p.R; r += kEpiThreads) s_rseq[r] = -1;
    epi_bar();
    for (int b = et; b < p.B; b += kEpiThreads) {
      const int c = p.ctx_lens[b], k = p.n_draft[b];
      const int q0 = p.cu_q[b], q1 = p.cu_q[b + 1];
      int bad = 0;
      if (c < 0 || k < 0 || k > p.max_k || q0 < 0 || q1 > p.R || q1 - q0 != k + 1) bad = SPADE_DEV_BAD_INDEX;
      else if (static_cast<int64_t>(c) + k + 1 > p.cap) bad = SPADE_DEV_CAPACITY;
      if (!bad && p.block_table) {
        // Every page the block writes must exist.
        for (int i = 0; i <= k; ++i) {
          const int pg = p.block_table[static_cast<int64_t>(b) * p.max_pages + (c + i) / p.page_size];
          if (pg < 0 || pg >= p.num_pages) bad = SPADE_DEV_BAD_INDEX;
        }
      }
      if (bad) {
        if (blockIdx.x == 0) atomicOr(p.status, bad);
        continue;
      }
      for (int i = 0; i <= k; ++i) {
        s_rseq[q0 + i] = b;
        s_rpos[q0 + i] = c + i;
      }
    }
    epi_bar();
    bool expired = false;
    int seg = 0;
    for (int u = u0; u < u1; ++seg) {
      const int t = u / p.KC;
      const int se = min(u1, (t + 1) * p.KC);
      const int buf = seg % p.nbuf, use = seg / p.nbuf;
      if (!mbar_wait(&acc_full[buf], use & 1, s_abort)) expired = true;
      tc_fence_after();
      // Accumulator -> this CTA's slot [Ncols][128] of the tile's partials.
      float *part = p.partials + static_cast<size_t>(blockIdx.x + t) * p.Ncols * kTileM;
      const uint32_t tl = tmem + (static_cast<uint32_t>(q4 * 32) << 16) + static_cast<uint32_t>(buf) * p.buf_cols;
      for (int c = 0; c < p.Ncols; c += 8) {
        uint32_t v[8];
        tmem_ld8(tl + c, v);
        tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < 8; ++e) __stcg(part + (c + e) * kTileM + q4 * 32 + lane, __uint_as_float(v[e]));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[buf]);
      // Publish the part.  With slabs, a split tile is finished after the
      // stream; otherwise the CTA whose part completes the tile (every
      // CTA of a whole tile) finishes it here, or, for the CTA's last tile,
      // below with every thread of the CTA.
      const int c_first = unit_owner(p.units, p.num_ctas, t * p.KC);
      const int nparts = unit_owner(p.units, p.num_ctas, (t + 1) * p.KC - 1) - c_first + 1;
      epi_bar();
      if (nparts > 1 && p.slabs > 1) {
        if (et == 0) publish_part(&p.counters[t]);
      } else {
        // Release publishes this part; for the last one, acquire makes the others visible.
        if (et == 0) *s_last = nparts == 1 || add_acq_rel(&p.counters[t], 1) == nparts - 1;
        epi_bar();
        if (*s_last) {
          if (se == u1) {
            if (et == 0) { s_fin[0] = t; s_fin[1] = c_first; s_fin[2] = nparts; }
          } else {
            if (nparts == 1)
              reduce_tile<6, 1>(p, s_rseq, s_rpos, s_freq, t, c_first, 1, 0, p.R, et, kEpiThreads);
            else
              reduce_tile<3, 3>(p, s_rseq, s_rpos, s_freq, t, c_first, nparts, 0, p.R, et, kEpiThreads);
            if (et == 0 && nparts > 1) p.counters[t] = 0;  // every part has arrived: reset for the next call
          }
        }
      }
      u = se;
    }
    if (expired) atomicOr(p.status, SPADE_DEV_TIMEOUT);
  }
  // The CTA's last tile, if this CTA finishes it, with every thread.
  __syncwarp();
  __syncthreads();
  if (s_fin[0] >= 0) {
    const int t = s_fin[0], c_first = s_fin[1], nparts = s_fin[2];
    if (nparts == 1)
      reduce_tile<6, 1>(p, s_rseq, s_rpos, s_freq, t, c_first, 1, 0, p.R, tid, kThreads);
    else
      reduce_tile<3, 3>(p, s_rseq, s_rpos, s_freq, t, c_first, nparts, 0, p.R, tid, kThreads);
    if (tid == 0 && nparts > 1) p.counters[t] = 0;  // every part has arrived: reset for the next call
  }
  // Row slabs of the split tiles (slabs > 1): item i = t * slabs + s goes to
  // CTA i mod num_ctas.  The slab waits until all of the tile's parts are
  // published (acquire, bounded), and the tile's last slab to finish resets
  // both counters for the next call.
  int32_t *published = p.counters, *slabs_done = p.counters + p.tiles;
  for (int item = blockIdx.x; p.slabs > 1 && item < p.tiles * p.slabs; item += p.num_ctas) {
    const int t = item / p.slabs, sl = item - t * p.slabs;
    const int c_first = unit_owner(p.units, p.num_ctas, t * p.KC);
    const int nparts = unit_owner(p.units, p.num_ctas, (t + 1) * p.KC - 1) - c_first + 1;
    if (nparts == 1) continue;  // a whole tile: finished by its CTA
    if (tid == 0) {
      s_fin[3] = 1;
      if (load_acquire(&published[t]) != nparts) {
        const uint64_t t0 = globaltimer();
        while (load_acquire(&published[t]) != nparts) {
          if (globaltimer() - t0 > kWaitLimitNs) {
            atomicOr(p.status, SPADE_DEV_TIMEOUT);
            s_fin[3] = 0;
            break;
          }
        }
      }
    }
    __syncthreads();
    const int ok = s_fin[3];
    if (ok) {
      const int r0 = static_cast<int>(static_cast<int64_t>(p.R) * sl / p.slabs);
      const int r1 = static_cast<int>(static_cast<int64_t>(p.R) * (sl + 1) / p.slabs);
      reduce_tile<2, 6>(p, s_rseq, s_rpos, s_freq, t, c_first, nparts, r0, r1, tid, kThreads);
    }
    __syncthreads();  // every load of the parts is done
    if (tid == 0 && ok && add_acq_rel(&slabs_done[t], 1) == p.slabs - 1) {
      published[t] = 0;
      slabs_done[t] = 0;
    }
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
struct Paging {
  const int32_t *block_table;
  int page_size, max_pages, num_pages;
};
static size_t counter_bytes(int tiles) { return round_up(static_cast<size_t>(tiles) * 8, 256); }
static size_t workspace_bytes_for(int R, int tiles, int sms) {
  const size_t ncols = static_cast<size_t>((R + 15) / 16 * 16);
  return counter_bytes(tiles) + static_cast<size_t>(sms + tiles) * ncols * kTileM * 4;
}
}  // namespace qkv
}  // namespace spade

using namespace spade;

extern "C" size_t spade_qkv_workspace_size(int32_t R, int32_t Hq, int32_t Hkv, int32_t D) {
  if (R <= 0 || R > qkv::kMaxR || Hq <= 0 || Hkv <= 0 || (D != 64 && D != 128) || (Hq + 2 * Hkv) * D % qkv::kTileM)
    return 0;
  int sms = 0;
  if (device_info(&sms, nullptr) != SPADE_OK) return 0;
  return qkv::workspace_bytes_for(R, (Hq + 2 * Hkv) * D / qkv::kTileM, sms);
}

static spade_status qkv_rope_impl(const void *x, const void *w_qkv, const int32_t *ctx_lens,
                                  const int32_t *n_draft, const int32_t *cu_q, void *q_out, void *k_cache,
                                  void *v_cache, int32_t B, int32_t R, int32_t H, int32_t Hq, int32_t Hkv,
                                  int32_t D, int32_t cap, int32_t max_k, float rope_theta, void *workspace,
                                  size_t workspace_bytes, int32_t *status, spade_stream_t stream,
                                  const qkv::Paging *pg) {
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
  const int tiles = (Hq + 2 * Hkv) * D / kTileM;
  const size_t need = workspace_bytes_for(R, tiles, sms);
  if (!workspace || workspace_bytes < need || !aligned(workspace, 256))
    return fail(SPADE_ERR_WORKSPACE, "qkv workspace needs %zu bytes, 256-byte aligned (got %zu)", need,
                workspace_bytes);

  Params p{};
  p.ctx_lens = ctx_lens;
  p.n_draft = n_draft;
  p.cu_q = cu_q;
  p.q_out = static_cast<__nv_bfloat16 *>(q_out);
  p.k_cache = static_cast<__nv_bfloat16 *>(k_cache);
  p.v_cache = static_cast<__nv_bfloat16 *>(v_cache);
  p.status = status;
  p.counters = static_cast<int32_t *>(workspace);
  p.partials = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + counter_bytes(tiles));
  p.B = B; p.R = R; p.H = H; p.Hq = Hq; p.Hkv = Hkv; p.D = D; p.cap = cap; p.max_k = max_k;
  p.block_table = pg ? pg->block_table : nullptr;
  p.page_size = pg ? pg->page_size : 0;
  p.max_pages = pg ? pg->max_pages : 0;
  p.num_pages = pg ? pg->num_pages : 0;
  p.tiles = tiles;
  p.KC = (H + kKChunk - 1) / kKChunk;
  p.Ncols = (R + 15) / 16 * 16;
  p.buf_cols = 32;
  while (p.buf_cols < static_cast<uint32_t>(p.Ncols)) p.buf_cols *= 2;
  p.nbuf = p.buf_cols * 2 <= 512 ? 2 : 1;
  p.tmem_cols = p.buf_cols * p.nbuf;
  for (int j = 0; j < D / 2; ++j) p.inv_freq[j] = static_cast<float>(pow(static_cast<double>(rope_theta), -2.0 * j / D));
  // Stages of up to two k-chunks when H allows the 3-D view and the ring
  // still holds three of them; otherwise one chunk per stage.
  p.KG = 1;
  if (H % kKChunk == 0 && (kSmemBudget - layout(p.Ncols, 0, 2).total) / layout(p.Ncols, 0, 2).stage_bytes >= 3)
    p.KG = 2;
  p.units = tiles * p.KC;
  p.num_ctas = p.units < sms ? p.units : sms;
  // Slabs: as many as keep every CTA busy in the final reduction, of at
  // least 8 rows each (one: split tiles are finished by their last part's CTA).
  p.slabs = p.num_ctas / tiles;
  if (p.slabs > R / 8) p.slabs = R / 8;
  if (p.slabs < 1) p.slabs = 1;
  p.stages = (kSmemBudget - layout(p.Ncols, 0, p.KG).total) / layout(p.Ncols, 0, p.KG).stage_bytes;
  if (p.stages > kMaxStages) p.stages = kMaxStages;
  if (p.stages < 2) return fail(SPADE_ERR_SHAPE, "shared memory too small for R = %d", R);
  const int smem = layout(p.Ncols, p.stages, p.KG).total;
  static bool configured = false;
  if (!configured) {
    // The plan above never exceeds kSmemBudget (alignment slack included).
    cudaError_t e = cudaFuncSetAttribute(qkv_rope_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(qkv_rope)");
    configured = true;
  }
  CUtensorMap tw, tx0, tx1, tw3;
  const int n0 = p.Ncols > 256 ? 256 : p.Ncols;
  const int n1 = p.Ncols - n0;
  const uint64_t wrows = static_cast<uint64_t>(Hq + 2 * Hkv) * D;
  if (!encode_tmap_bf16_sw128(&tw, w_qkv, H, wrows, static_cast<uint64_t>(H) * 2, kKChunk, kTileM) ||
      !encode_tmap_bf16_sw128(&tx0, x, H, R, static_cast<uint64_t>(H) * 2, kKChunk, n0) ||
      !encode_tmap_bf16_sw128(&tx1, x, H, R, static_cast<uint64_t>(H) * 2, kKChunk, n1 ? n1 : 16))
    return SPADE_ERR_CUDA;
  if (p.KG > 1) {
    if (!encode_tmap_rows_by_slab(&tw3, w_qkv, wrows, static_cast<uint32_t>(H), kTileM, static_cast<uint32_t>(p.KG)))
      return SPADE_ERR_CUDA;
  } else {
    tw3 = tw;  // unused
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.num_ctas);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = reinterpret_cast<cudaStream_t>(stream);
  // Cooperative: the final reduction's slabs wait for other CTAs' partials,
  // so every CTA must be resident (one per SM at most).
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeCooperative;
  attr[1].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, qkv_rope_kernel, p, tw, tx0, tx1, tw3);
  if (e != cudaSuccess) return cuda_fail(e, "qkv_rope launch");
  return SPADE_OK;
}

extern "C" spade_status spade_verify_qkv_rope(const void *x, const void *w_qkv, const int32_t *ctx_lens,
                                              const int32_t *n_draft, const int32_t *cu_q, void *q_out,
                                              void *k_cache, void *v_cache, int32_t B, int32_t R,
                                              int32_t H, int32_t Hq, int32_t Hkv, int32_t D, int32_t cap,
                                              int32_t max_k, float rope_theta, void *workspace,
                                              size_t workspace_bytes, int32_t *status, spade_stream_t stream) {
  return qkv_rope_impl(x, w_qkv, ctx_lens, n_draft, cu_q, q_out, k_cache, v_cache, B, R, H, Hq, Hkv, D, cap,
                       max_k, rope_theta, workspace, workspace_bytes, status, stream, nullptr);
}

extern "C" spade_status spade_verify_qkv_rope_paged(const void *x, const void *w_qkv,
                                                    const int32_t *block_table, const int32_t *ctx_lens,
                                                    const int32_t *n_draft, const int32_t *cu_q, void *q_out,
                                                    void *k_pool, void *v_pool, int32_t B, int32_t R,
                                                    int32_t H, int32_t Hq, int32_t Hkv, int32_t D,
                                                    int32_t page_size, int32_t num_pages, int32_t max_pages,
                                                    int32_t max_k, float rope_theta, void *workspace,
                                                    size_t workspace_bytes, int32_t *status,
                                                    spade_stream_t stream) {
  if (!block_table) return fail(SPADE_ERR_INVALID_ARG, "spade_verify_qkv_rope_paged: null block_table");
  if (page_size <= 0 || num_pages <= 0 || max_pages <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_qkv_rope_paged: non-positive page geometry");
  if (static_cast<int64_t>(max_pages) * page_size >= (int64_t(1) << 31))
    return fail(SPADE_ERR_CAPACITY, "max_pages * page_size exceeds 2^31");
  const qkv::Paging pg{block_table, page_size, max_pages, num_pages};
  return qkv_rope_impl(x, w_qkv, ctx_lens, n_draft, cu_q, q_out, k_pool, v_pool, B, R, H, Hq, Hkv, D,
                       max_pages * page_size, max_k, rope_theta, workspace, workspace_bytes, status, stream, &pg);
}
