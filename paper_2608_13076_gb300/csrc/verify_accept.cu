// verify_accept.cu -- LM head o = g(x_L) and softmax (Sec. III-A) fused with the
// accept test alpha(x) = min(1, p(x)/q(x)) and the residual sampling from
// p'(x) = norm(max(0, p(x) - q(x))) (Sec. III-C), i.e. the verify / accept /
// correct steps of Algorithm 1 for every sequence of the batch.
//
// Design (GB300):
//  * The contraction logits[r, x] = hidden[r, :] . W[x, :] runs on the 5th-gen
//    tensor cores (tcgen05.mma kind::f16, bf16 in, fp32 accumulators in TMEM).
//    The vocabulary is the M side of the MMA (128 vocab rows per tile) and the
//    R verify rows are the N side, so W -- the only large operand -- streams
//    from HBM exactly once while the few hidden rows are re-read from L2.
//  * One CTA per SM (cooperative launch) owns a contiguous vocabulary slice.
//    All its tiles' logits stay resident in TMEM (512 columns x 128 lanes);
//    when the padded MMA width does not leave room for every tile, finished
//    tiles are compacted to the exact row count and the next round of tiles
//    accumulates in the freed columns.  Logits never reach HBM.
//  * Warp roles: warp 0 issues TMA loads of W and hidden chunks (128-byte
//    swizzle) into mbarrier rings, warp 1 owns TMEM and issues the MMAs from a
//    single thread, warps 2-5 read accumulators back (tcgen05.ld) and reduce
//    per-row max / sum-exp / argmax across the vocabulary with warp shuffles.
//  * Two bounded device-wide barriers: after the first every CTA merges the
//    per-slice statistics into p(d) and argmax for every row and takes the
//    accept decisions; after the second the slice masses of the distribution
//    to sample (residual or p, fp64) are known, and the CTA whose slice holds
//    the point u*Z scans its resident logits in vocabulary order to pick the
//    token.
#include <cuda_bf16.h>

#include <cfloat>

#include "internal.h"
#include "ptx.cuh"

namespace spade {
namespace accept {

constexpr int kTileV = 128;    // vocab rows per tile (MMA M)
constexpr int kKChunk = 64;    // K elements per TMA box row (128 bytes)
constexpr int kEpiWarps = 4;
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr int kMaxR = 256;     // verify rows per call on the resident path (MMA N <= 256)
constexpr int kMaxRounds = 8;
constexpr int kTmemCols = 512;
constexpr int kSmemBudget = 216 * 1024;
constexpr int kWSlotBytes = kTileV * kKChunk * 2;  // 16 KB

struct Params {
  const int32_t *draft_tokens;
  const float *draft_probs;
  const float *uniforms;
  const int32_t *mode;
  const int32_t *cu_q;
  const int32_t *n_draft;
  int32_t *accepted_len;
  int32_t *next_token;
  int32_t *status;
  unsigned *bar;     // [2]: arrival count, generation
  float4 *pstat;     // [NC][R]: slice max, slice sum-exp, slice argmax (bits), -
  float *ldraft;     // [R]: logit of the row's draft token
  double2 *zpart;    // [NC][B]: slice mass of the distribution to sample, of p
  int B, R, H, V, T, NC, Ncols, Rs, KC, nrounds;
  int round_tiles[kMaxRounds];
  int HS, WS;        // hidden / W ring slots
  uint32_t idesc;
  uint32_t tmem_cols;
};

struct Smem {
  int off_h, off_bar, off_misc, off_draft, off_wst, total;
};

__host__ __device__ inline Smem smem_layout(const Params &p) {
  Smem s;
  s.off_h = p.WS * kWSlotBytes;
  s.off_bar = s.off_h + p.HS * p.Ncols * 128;
  s.off_misc = s.off_bar + (2 * p.WS + 2 * p.HS + 2) * 8;
  s.off_draft = s.off_misc + 64;
  s.off_wst = s.off_draft + kMaxR * 4;
  s.total = s.off_wst + kEpiWarps * kMaxR * 16 + 1024;
  return s;
}

__device__ __forceinline__ void named_bar(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

__device__ __forceinline__ unsigned ld_acquire(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Device-wide barrier among the NC co-resident CTAs (cooperative launch).  The
// last CTA to arrive resets the count and bumps the generation; the others
// poll the generation with a time limit.  Returns false if the wait expired.
__device__ bool grid_barrier(unsigned *bar, int nctas) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    s_ok = 1;
    const unsigned gen = ld_acquire(bar + 1);
    __threadfence();
    const unsigned arrived = atomicAdd(bar, 1u);
    if (arrived == static_cast<unsigned>(nctas) - 1) {
      atomicExch(bar, 0u);
      __threadfence();
      atomicAdd(bar + 1, 1u);
    } else {
      const uint64_t t0 = globaltimer();
      while (ld_acquire(bar + 1) == gen) {
        if (globaltimer() - t0 > kWaitLimitNs) { s_ok = 0; break; }
      }
    }
    __threadfence();
  }
  __syncthreads();
  return s_ok != 0;
}

// (max, argmax) merge with the lowest index winning ties.
__device__ __forceinline__ void argmax_merge(float &m, int &i, float om, int oi) {
  if (om > m || (om == m && oi < i)) { m = om; i = oi; }
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__global__ void __launch_bounds__(kThreads, 1) verify_accept_kernel(
    const __grid_constant__ Params p, const __grid_constant__ CUtensorMap tm_w,
    const __grid_constant__ CUtensorMap tm_h) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const Smem L = smem_layout(p);
  uint8_t *w_ring = smem;
  uint8_t *h_ring = smem + L.off_h;
  uint64_t *w_full = reinterpret_cast<uint64_t *>(smem + L.off_bar);
  uint64_t *w_empty = w_full + p.WS;
  uint64_t *h_full = w_empty + p.WS;
  uint64_t *h_empty = h_full + p.HS;
  uint64_t *acc_full = h_empty + p.HS;
  uint64_t *acc_empty = acc_full + 1;
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + L.off_misc);
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + L.off_misc + 8);
  int *s_any_stoch = reinterpret_cast<int *>(smem + L.off_misc + 16);
  int32_t *s_draft = reinterpret_cast<int32_t *>(smem + L.off_draft);
  float4 *s_wst = reinterpret_cast<float4 *>(smem + L.off_wst);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c = blockIdx.x;
  const int t_lo = static_cast<int>(static_cast<int64_t>(c) * p.T / p.NC);
  const int t_hi = static_cast<int>(static_cast<int64_t>(c + 1) * p.T / p.NC);
  const int ntiles = t_hi - t_lo;

  // ---- set-up: barriers, TMEM, per-row draft tokens ------------------------
  if (tid == 0) {
    *s_abort = 0;
    *s_any_stoch = 0;
    for (int s = 0; s < p.WS; ++s) { mbar_init(&w_full[s], 1); mbar_init(&w_empty[s], 1); }
    for (int s = 0; s < p.HS; ++s) { mbar_init(&h_full[s], 1); mbar_init(&h_empty[s], 1); }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, kEpiWarps);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(s_tmem, p.tmem_cols);
    tmem_relinquish();
  }
  for (int n = tid; n < kMaxR; n += kThreads) s_draft[n] = -1;
  __syncthreads();
  // Row n = cu_q[b] + i holds draft i of sequence b for i < k_b.
  for (int b = tid; b < p.B; b += kThreads) {
    const int r0 = p.cu_q[b], k = p.n_draft[b], r1 = p.cu_q[b + 1];
    if (r0 < 0 || k < 0 || r1 - r0 != k + 1 || r1 > p.R) {
      atomicOr(p.status, SPADE_DEV_BAD_INDEX);
      continue;
    }
    for (int i = 0; i < k; ++i) s_draft[r0 + i] = p.draft_tokens[r0 - b + i];
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  int rounds_issued = 0;  // MMA thread: accumulator rounds committed

  // ======================= phase A: logits + slice statistics =============
  if (warp == 0) {
    if (lane == 0 && ntiles > 0) {
      tma_prefetch_desc(&tm_w);
      tma_prefetch_desc(&tm_h);
      const uint64_t pol_w = l2_policy_evict_first();
      const uint64_t pol_h = l2_policy_evict_last();
      uint32_t wi = 0, hi = 0, w_issued = 0, h_issued = 0;
      int tdone = 0;
      for (int r = 0; r < p.nrounds && tdone < ntiles; ++r) {
        const int nt = min(p.round_tiles[r], ntiles - tdone);
        for (int kc = 0; kc < p.KC; ++kc) {
          {
            const int s = hi % p.HS;
            mbar_wait(&h_empty[s], ((hi / p.HS) & 1) ^ 1, s_abort);
            if (!*s_abort) {
              mbar_arrive_expect_tx(&h_full[s], p.Ncols * 128);
              tma_load_2d(h_ring + s * p.Ncols * 128, &tm_h, kc * kKChunk, 0, &h_full[s], pol_h);
              h_issued = hi + 1;
            }
            ++hi;
          }
          for (int j = 0; j < nt; ++j) {
            const int s = wi % p.WS;
            mbar_wait(&w_empty[s], ((wi / p.WS) & 1) ^ 1, s_abort);
            if (!*s_abort) {
              mbar_arrive_expect_tx(&w_full[s], kWSlotBytes);
              tma_load_2d(w_ring + s * kWSlotBytes, &tm_w, kc * kKChunk,
                          (t_lo + tdone + j) * kTileV, &w_full[s], pol_w);
              w_issued = wi + 1;
            }
            ++wi;
          }
        }
        tdone += nt;
      }
      if (*s_abort) {
        // Every copy issued must land before the CTA's shared memory goes away.
        for (uint32_t j = (w_issued > (uint32_t)p.WS ? w_issued - p.WS : 0); j < w_issued; ++j)
          mbar_wait_unabortable(&w_full[j % p.WS], (j / p.WS) & 1);
        for (uint32_t j = (h_issued > (uint32_t)p.HS ? h_issued - p.HS : 0); j < h_issued; ++j)
          mbar_wait_unabortable(&h_full[j % p.HS], (j / p.HS) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && ntiles > 0) {
      uint32_t wi = 0, hi = 0;
      int tdone = 0, used = 0;
      rounds_issued = 0;
      for (int r = 0; r < p.nrounds && tdone < ntiles; ++r) {
        const int nt = min(p.round_tiles[r], ntiles - tdone);
        if (r > 0) mbar_wait(acc_empty, (r - 1) & 1, s_abort);
        tc_fence_after();
        for (int kc = 0; kc < p.KC; ++kc) {
          const int hs = hi % p.HS;
          mbar_wait(&h_full[hs], (hi / p.HS) & 1, s_abort);
          tc_fence_after();
          const uint32_t h_addr = smem_u32(h_ring + hs * p.Ncols * 128);
          for (int j = 0; j < nt; ++j) {
            const int ws = wi % p.WS;
            mbar_wait(&w_full[ws], (wi / p.WS) & 1, s_abort);
            tc_fence_after();
            const uint32_t w_addr = smem_u32(w_ring + ws * kWSlotBytes);
            const uint32_t d_tmem = tmem + static_cast<uint32_t>(used + j * p.Ncols);
#pragma unroll
            for (int k16 = 0; k16 < kKChunk / 16; ++k16) {
              tc_mma_f16(d_tmem, smem_desc_sw128(w_addr + 32 * k16),
                         smem_desc_sw128(h_addr + 32 * k16), p.idesc, (kc | k16) != 0);
            }
            tc_commit(&w_empty[ws]);
            ++wi;
          }
          tc_commit(&h_empty[hs]);
          ++hi;
        }
        tc_commit(acc_full);
        ++rounds_issued;
        used += nt * p.Rs;
        tdone += nt;
      }
    }
  } else {
    // ---- epilogue warps: slice statistics per row, compaction -----------
    const int ew = warp - 2;             // 0..3
    const int q4 = warp & 3;             // TMEM lane quarter this warp may access
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    float4 *wst = s_wst + ew * kMaxR;    // this warp's running stats per row
    for (int n = lane; n < p.R; n += 32) wst[n] = make_float4(-INFINITY, 0.f, __int_as_float(INT_MAX), 0.f);
    __syncwarp();
    int tdone = 0, used = 0;
    for (int r = 0; r < p.nrounds && tdone < ntiles; ++r) {
      const int nt = min(p.round_tiles[r], ntiles - tdone);
      if (!mbar_wait(acc_full, r & 1, s_abort)) atomicOr(p.status, SPADE_DEV_TIMEOUT);
      tc_fence_after();
      for (int j = 0; j < nt; ++j) {
        const int v = (t_lo + tdone + j) * kTileV + q4 * 32 + lane;
        const bool valid = v < p.V;
        const uint32_t col0 = tmem + lane_base + static_cast<uint32_t>(used + j * p.Ncols);
        for (int c8 = 0; c8 * 8 < p.R; ++c8) {
          uint32_t raw[8];
          tmem_ld8(col0 + c8 * 8, raw);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int n = c8 * 8 + e;
            if (n < p.R) {
              const float x = valid ? __uint_as_float(raw[e]) : -INFINITY;
              if (valid && s_draft[n] == v) p.ldraft[n] = x;
              float mv = x;
              int mi = v;
#pragma unroll
              for (int o = 16; o > 0; o >>= 1)
                argmax_merge(mv, mi, __shfl_xor_sync(0xffffffffu, mv, o),
                             __shfl_xor_sync(0xffffffffu, mi, o));
              float ev = (x == -INFINITY) ? 0.f : ex2((x - mv) * 1.4426950408889634f);
#pragma unroll
              for (int o = 16; o > 0; o >>= 1) ev += __shfl_xor_sync(0xffffffffu, ev, o);
              if (lane == (n & 31)) {
                float4 st = wst[n];
                const float M = fmaxf(st.x, mv);
                if (M != -INFINITY) {
                  st.y = st.y * ex2((st.x - M) * 1.4426950408889634f) +
                         ev * ex2((mv - M) * 1.4426950408889634f);
                }
                int si = __float_as_int(st.z);
                argmax_merge(st.x, si, mv, mi);
                st.x = M;
                st.z = __int_as_float(si);
                wst[n] = st;
              }
            }
          }
        }
      }
      // Compaction: move this round's tiles from stride Ncols to stride Rs.
      if (p.Ncols != p.Rs) {
        for (int j = 0; j < nt; ++j) {
          const uint32_t src = tmem + lane_base + static_cast<uint32_t>(used + j * p.Ncols);
          const uint32_t dst = tmem + lane_base + static_cast<uint32_t>(used + j * p.Rs);
          if (src == dst) continue;
          for (int c8 = 0; c8 < p.Rs / 8; ++c8) {
            uint32_t raw[8];
            tmem_ld8(src + c8 * 8, raw);
            tmem_wait_ld();
            tmem_st8(dst + c8 * 8, raw);
          }
        }
        tmem_wait_st();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty);
      used += nt * p.Rs;
      tdone += nt;
    }
    // Merge the four warps' statistics and publish this CTA's slice partials.
    named_bar(1, kEpiWarps * 32);
    for (int n = tid - 64; n < p.R; n += kEpiWarps * 32) {
      float m = -INFINITY, s = 0.f;
      int idx = INT_MAX;
      for (int w = 0; w < kEpiWarps; ++w) {
        const float4 st = s_wst[w * kMaxR + n];
        const float M = fmaxf(m, st.x);
        if (M != -INFINITY)
          s = s * ex2((m - M) * 1.4426950408889634f) + st.y * ex2((st.x - M) * 1.4426950408889634f);
        int i2 = idx;
        argmax_merge(m, i2, st.x, __float_as_int(st.z));
        m = M;
        idx = i2;
      }
      __stcg(&p.pstat[static_cast<size_t>(c) * p.R + n], make_float4(m, s, __int_as_float(idx), 0.f));
    }
  }
  if (*s_abort) atomicOr(p.status, SPADE_DEV_TIMEOUT);

  // ======================= phase B: global row statistics, decisions =======
  if (!grid_barrier(p.bar, p.NC)) {
    atomicOr(p.status, SPADE_DEV_TIMEOUT);
    *s_abort = 1;
  }
  // Phase-A buffers are idle now: reuse the W ring for per-row / per-seq data.
  float *g_m = reinterpret_cast<float *>(w_ring);           // [R]
  float *g_s = g_m + kMaxR;                                 // [R]
  int *g_arg = reinterpret_cast<int *>(g_s + kMaxR);        // [R]
  int *s_acc = g_arg + kMaxR;                               // [B]
  int *s_rstar = s_acc + kMaxR;                             // [B]
  int *s_owner = s_rstar + kMaxR;                           // [B]
  int *s_usep = s_owner + kMaxR;                            // [B]
  double *s_T = reinterpret_cast<double *>(s_usep + kMaxR); // [B]
  double *s_red = s_T + kMaxR;                              // [kEpiWarps * 2]
  for (int n = warp; n < p.R; n += kThreads / 32) {
    float m = -INFINITY, s = 0.f;
    int idx = INT_MAX;
    for (int cc = lane; cc < p.NC; cc += 32) {
      const float4 st = __ldcg(&p.pstat[static_cast<size_t>(cc) * p.R + n]);
      const float M = fmaxf(m, st.x);
      if (M != -INFINITY) s = s * expf(m - M) + st.y * expf(st.x - M);
      int i2 = idx;
      argmax_merge(m, i2, st.x, __float_as_int(st.z));
      m = M;
      idx = i2;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float om = __shfl_xor_sync(0xffffffffu, m, o);
      const float os = __shfl_xor_sync(0xffffffffu, s, o);
      const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
      const float M = fmaxf(m, om);
      if (M != -INFINITY) s = s * expf(m - M) + os * expf(om - M);
      int i2 = idx;
      argmax_merge(m, i2, om, oi);
      m = M;
      idx = i2;
    }
    if (lane == 0) { g_m[n] = m; g_s[n] = s; g_arg[n] = idx; }
  }
  __syncthreads();
  for (int b = tid; b < p.B; b += kThreads) {
    const int r0 = p.cu_q[b], k = p.n_draft[b];
    const int md = p.mode[b];
    if (md != 0 && md != 1 && c == 0) atomicOr(p.status, SPADE_DEV_BAD_INDEX);
    const bool stoch = (md == 1) && p.draft_probs != nullptr;
    int a = 0;
    if (r0 >= 0 && k >= 0 && p.cu_q[b + 1] - r0 == k + 1 && p.cu_q[b + 1] <= p.R) {
      for (; a < k; ++a) {
        const int n = r0 + a;
        const int d = p.draft_tokens[r0 - b + a];
        bool ok;
        if (d < 0 || d >= p.V) {
          if (c == 0) atomicOr(p.status, SPADE_DEV_BAD_INDEX);
          ok = false;
        } else if (!stoch) {
          ok = (d == g_arg[n]);
        } else {
          const float pd = expf(__ldcg(&p.ldraft[n]) - g_m[n]) / g_s[n];
          const float qd = p.draft_probs[static_cast<size_t>(r0 - b + a) * p.V + d];
          ok = (qd > 0.f) ? (p.uniforms[n] < pd / qd) : (pd > 0.f);
        }
        if (!ok) break;
      }
    } else {
      a = -1;
    }
    s_acc[b] = a;
    s_rstar[b] = (a >= 0) ? r0 + a : -1;
    if (a >= 0 && stoch) atomicOr(s_any_stoch, 1);
    if (c == 0) {
      p.accepted_len[b] = a < 0 ? 0 : a;
      if (a < 0) p.next_token[b] = -1;
      else if (!stoch) p.next_token[b] = g_arg[r0 + a];
    }
  }
  __syncthreads();

  if (*s_any_stoch) {
    // =================== phase C: slice masses of the sampled distribution ==
    for (int b = 0; b < p.B; ++b) {
      const bool stoch = (p.mode[b] == 1) && p.draft_probs != nullptr && s_acc[b] >= 0;
      if (!stoch) continue;
      if (warp >= 2) {
        const int ew = warp - 2, q4 = warp & 3;
        const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
        const int n = s_rstar[b];
        const int a = s_acc[b], k = p.n_draft[b];
        const float *qrow = (a < k) ? p.draft_probs + static_cast<size_t>(p.cu_q[b] - b + a) * p.V : nullptr;
        const float M = g_m[n], invS = 1.f / g_s[n];
        double z = 0.0, zp = 0.0;
        for (int j = 0; j < ntiles; ++j) {
          const int v = (t_lo + j) * kTileV + q4 * 32 + lane;
          uint32_t raw;
          tmem_ld1(tmem + lane_base + static_cast<uint32_t>(j * p.Rs + n), raw);
          tmem_wait_ld();
          if (v < p.V) {
            const double pv = static_cast<double>(expf(__uint_as_float(raw) - M) * invS);
            zp += pv;
            z += qrow ? fmax(0.0, pv - static_cast<double>(qrow[v])) : pv;
          }
        }
        z = warp_sum_d(z);
        zp = warp_sum_d(zp);
        if (lane == 0) { s_red[ew * 2] = z; s_red[ew * 2 + 1] = zp; }
        named_bar(1, kEpiWarps * 32);
        if (ew == 0 && lane == 0) {
          double zs = 0.0, zps = 0.0;
          for (int w = 0; w < kEpiWarps; ++w) { zs += s_red[w * 2]; zps += s_red[w * 2 + 1]; }
          __stcg(&p.zpart[static_cast<size_t>(c) * p.B + b], make_double2(zs, zps));
        }
        named_bar(1, kEpiWarps * 32);
      }
    }
    if (!grid_barrier(p.bar, p.NC)) {
      atomicOr(p.status, SPADE_DEV_TIMEOUT);
      *s_abort = 1;
    }
    // =================== phase D: owner slice of u*Z, in-slice scan =========
    for (int b = warp; b < p.B; b += kThreads / 32) {
      const bool stoch = (p.mode[b] == 1) && p.draft_probs != nullptr && s_acc[b] >= 0;
      if (!stoch) { if (lane == 0) s_owner[b] = -1; continue; }
      double tot = 0.0, totp = 0.0;
      for (int cc = lane; cc < p.NC; cc += 32) {
        const double2 z = __ldcg(&p.zpart[static_cast<size_t>(cc) * p.B + b]);
        tot += z.x;
        totp += z.y;
      }
      tot = warp_sum_d(tot);
      totp = warp_sum_d(totp);
      const bool usep = !(tot > 0.0 && isfinite(tot));
      const double Z = usep ? totp : tot;
      const int rk = p.cu_q[b] + p.n_draft[b];
      const double Tgt = static_cast<double>(p.uniforms[rk]) * Z;
      // First slice whose cumulative mass exceeds Tgt; else the last slice with mass.
      double base = 0.0;
      int owner = -1, last_pos = -1;
      double base_last = 0.0, base_owner = 0.0;
      for (int c0 = 0; c0 < p.NC && owner < 0; c0 += 32) {
        const int cc = c0 + lane;
        double z = 0.0;
        if (cc < p.NC) {
          const double2 zz = __ldcg(&p.zpart[static_cast<size_t>(cc) * p.B + b]);
          z = usep ? zz.y : zz.x;
        }
        double incl = z;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const double t = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += t;
        }
        const unsigned hit = __ballot_sync(0xffffffffu, cc < p.NC && base + incl > Tgt);
        const unsigned pos = __ballot_sync(0xffffffffu, cc < p.NC && z > 0.0);
        if (hit) {
          const int l = __ffs(hit) - 1;
          owner = c0 + l;
          base_owner = base + __shfl_sync(0xffffffffu, incl - z, l);
        }
        if (pos) {
          const int l = 31 - __clz(pos);
          last_pos = c0 + l;
          base_last = base + __shfl_sync(0xffffffffu, incl - z, l);
        }
        base += __shfl_sync(0xffffffffu, incl, 31);
      }
      if (lane == 0) {
        if (usep && c == 0) atomicOr(p.status, SPADE_DEV_FALLBACK);
        if (owner >= 0) {
          s_owner[b] = owner;
          s_T[b] = Tgt - base_owner;
        } else {
          s_owner[b] = last_pos;
          s_T[b] = Tgt - base_last;  // beyond the slice total: the scan clamps
        }
        s_usep[b] = usep;
      }
    }
    __syncthreads();
    if (warp >= 2) {
      const int ew = warp - 2, q4 = warp & 3;
      const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
      for (int b = 0; b < p.B; ++b) {
        if (s_owner[b] != c) continue;
        const int n = s_rstar[b];
        const int a = s_acc[b], k = p.n_draft[b];
        const bool usep = s_usep[b] != 0;
        const float *qrow = (a < k && !usep)
                                ? p.draft_probs + static_cast<size_t>(p.cu_q[b] - b + a) * p.V
                                : nullptr;
        const float M = g_m[n], invS = 1.f / g_s[n];
        const double Tgt = s_T[b];
        double run = 0.0;
        int found = -1, last_pos = -1;
        for (int j = 0; j < ntiles && found < 0; ++j) {
          const int v = (t_lo + j) * kTileV + q4 * 32 + lane;
          uint32_t raw;
          tmem_ld1(tmem + lane_base + static_cast<uint32_t>(j * p.Rs + n), raw);
          tmem_wait_ld();
          double rv = 0.0;
          if (v < p.V) {
            const double pv = static_cast<double>(expf(__uint_as_float(raw) - M) * invS);
            rv = qrow ? fmax(0.0, pv - static_cast<double>(qrow[v])) : pv;
          }
          double incl = rv;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const double t = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += t;
          }
          const double wsum = __shfl_sync(0xffffffffu, incl, 31);
          if (lane == 0) s_red[ew * 2] = wsum;
          named_bar(1, kEpiWarps * 32);
          double before = run;  // mass of this slice before this warp's 32 entries
          for (int w = 0; w < q4; ++w) before += s_red[((w + 2) & 3) * 2];
          double tile_tot = 0.0;
          for (int w = 0; w < kEpiWarps; ++w) tile_tot += s_red[w * 2];
          const unsigned hit = __ballot_sync(0xffffffffu, before + incl > Tgt && rv > 0.0);
          const unsigned pos = __ballot_sync(0xffffffffu, rv > 0.0);
          int my_found = hit ? v - lane + (__ffs(hit) - 1) : -1;
          int my_last = pos ? v - lane + (31 - __clz(pos)) : -1;
          named_bar(1, kEpiWarps * 32);
          if (lane == 0) {
            reinterpret_cast<int *>(s_red)[2 * kEpiWarps * 2 + q4] = my_found;
            reinterpret_cast<int *>(s_red)[2 * kEpiWarps * 2 + 4 + q4] = my_last;
          }
          named_bar(1, kEpiWarps * 32);
          const int *res = reinterpret_cast<const int *>(s_red) + 2 * kEpiWarps * 2;
          for (int w = 0; w < 4 && found < 0; ++w) found = res[w];
          for (int w = 0; w < 4; ++w) last_pos = res[4 + w] >= 0 ? res[4 + w] : last_pos;
          run += tile_tot;
          named_bar(1, kEpiWarps * 32);
        }
        if (ew == 0 && lane == 0) p.next_token[b] = found >= 0 ? found : last_pos;
      }
    }
  }

  // ---- teardown: every TMEM access above has completed --------------------
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    // No MMA may still write TMEM when it is released (matters only after an
    // expired wait; otherwise the epilogue already consumed the last round).
    if (lane == 0 && rounds_issued > 0) mbar_wait_unabortable(acc_full, (rounds_issued - 1) & 1);
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, p.tmem_cols);
  }
}

// Plans the TMEM residency rounds of one CTA's `tiles` vocab tiles: tiles of a
// round accumulate at stride Ncols; finished rounds are compacted to stride Rs.
static bool plan_rounds(int tiles, int Ncols, int Rs, int *round_tiles, int *nrounds) {
  int used = 0, done = 0, r = 0;
  while (done < tiles) {
    if (r == kMaxRounds) return false;
    const int fit = (kTmemCols - used) / Ncols;
    if (fit <= 0) return false;
    const int n = fit < tiles - done ? fit : tiles - done;
    round_tiles[r++] = n;
    used += n * Rs;
    done += n;
  }
  *nrounds = r;
  return used <= kTmemCols;
}

struct Plan {
  int T, NC, Ncols, Rs;
};

static Plan make_plan(int R, int V, int sms) {
  Plan pl;
  pl.T = (V + kTileV - 1) / kTileV;
  pl.NC = pl.T < sms ? pl.T : sms;
  pl.Ncols = (R + 15) / 16 * 16;
  pl.Rs = (R + 7) / 8 * 8;
  return pl;
}

static size_t workspace_bytes_for(int B, int R, int NC) {
  size_t off = 256;                                     // barrier words
  off += round_up(static_cast<size_t>(NC) * R * 16, 256);  // pstat
  off += round_up(static_cast<size_t>(R) * 4, 256);       // ldraft
  off += round_up(static_cast<size_t>(NC) * B * 16, 256); // zpart
  return off;
}

}  // namespace accept
}  // namespace spade

using namespace spade;

extern "C" size_t spade_accept_workspace_size(int32_t B, int32_t R, int32_t H, int32_t V) {
  if (B <= 0 || R < B || H <= 0 || V <= 0) return 0;
  int sms = 0;
  if (device_info(&sms, nullptr) != SPADE_OK) return 0;
  const accept::Plan pl = accept::make_plan(R, V, sms);
  return accept::workspace_bytes_for(B, R, pl.NC);
}

extern "C" spade_status spade_verify_accept(const void *hidden, const void *w_lm,
                                            const int32_t *draft_tokens, const float *draft_probs,
                                            const float *uniforms, const int32_t *mode,
                                            const int32_t *cu_q, const int32_t *n_draft,
                                            int32_t *accepted_len, int32_t *next_token, int32_t B,
                                            int32_t R, int32_t H, int32_t V, void *workspace,
                                            size_t workspace_bytes, int32_t *status,
                                            spade_stream_t stream) {
  using namespace accept;
  if (!hidden || !w_lm || !uniforms || !mode || !cu_q || !n_draft || !accepted_len ||
      !next_token || !status || (R > B && !draft_tokens))
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept: null pointer argument");
  if (B <= 0 || R < B || H <= 0 || V <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept: bad sizes B=%d R=%d H=%d V=%d", B, R, H, V);
  if (H % 8) return fail(SPADE_ERR_SHAPE, "hidden size %d must be a multiple of 8", H);
  if (R > kMaxR) return fail(SPADE_ERR_SHAPE, "R = %d verify rows exceed %d per call", R, kMaxR);
  if (!aligned(hidden, 16) || !aligned(w_lm, 16))
    return fail(SPADE_ERR_INVALID_ARG, "hidden and w_lm must be 16-byte aligned");
  int sms = 0;
  spade_status st = device_info(&sms, nullptr);
  if (st != SPADE_OK) return st;

  const Plan pl = make_plan(R, V, sms);
  Params p{};
  p.draft_tokens = draft_tokens;
  p.draft_probs = draft_probs;
  p.uniforms = uniforms;
  p.mode = mode;
  p.cu_q = cu_q;
  p.n_draft = n_draft;
  p.accepted_len = accepted_len;
  p.next_token = next_token;
  p.status = status;
  p.B = B; p.R = R; p.H = H; p.V = V;
  p.T = pl.T; p.NC = pl.NC; p.Ncols = pl.Ncols; p.Rs = pl.Rs;
  p.KC = (H + kKChunk - 1) / kKChunk;
  const int tiles_max = (pl.T + pl.NC - 1) / pl.NC;
  if (!plan_rounds(tiles_max, pl.Ncols, pl.Rs, p.round_tiles, &p.nrounds))
    return fail(SPADE_ERR_SHAPE,
                "logits of %d rows x %d vocab do not fit on chip (%d tiles per SM, %d TMEM columns each)",
                R, V, tiles_max, pl.Rs);
  p.idesc = idesc_bf16_f32(kTileV, pl.Ncols);
  p.tmem_cols = kTmemCols;
  p.HS = 3;
  p.WS = 2;
  {
    Params probe = p;
    probe.WS = 0;
    const int fixed = smem_layout(probe).total;
    p.WS = (kSmemBudget - fixed) / kWSlotBytes;
    if (p.WS > 12) p.WS = 12;
    if (p.WS < 2) return fail(SPADE_ERR_SHAPE, "shared memory too small for R = %d", R);
  }
  const size_t need = workspace_bytes_for(B, R, pl.NC);
  if (!workspace || workspace_bytes < need || !aligned(workspace, 256))
    return fail(SPADE_ERR_WORKSPACE, "accept workspace needs %zu bytes, 256-byte aligned (got %zu)",
                need, workspace_bytes);
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  p.bar = reinterpret_cast<unsigned *>(ws);
  size_t off = 256;
  p.pstat = reinterpret_cast<float4 *>(ws + off);
  off += round_up(static_cast<size_t>(pl.NC) * R * 16, 256);
  p.ldraft = reinterpret_cast<float *>(ws + off);
  off += round_up(static_cast<size_t>(R) * 4, 256);
  p.zpart = reinterpret_cast<double2 *>(ws + off);

  CUtensorMap tw, th;
  if (!encode_tmap_bf16_sw128(&tw, w_lm, H, V, static_cast<uint64_t>(H) * 2, kKChunk, kTileV) ||
      !encode_tmap_bf16_sw128(&th, hidden, H, R, static_cast<uint64_t>(H) * 2, kKChunk, pl.Ncols))
    return SPADE_ERR_CUDA;

  const int smem = smem_layout(p).total;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(verify_accept_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBudget + 2048);
    if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(verify_accept)");
    configured = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(pl.NC);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = reinterpret_cast<cudaStream_t>(stream);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, verify_accept_kernel, p, tw, th);
  if (e != cudaSuccess) return cuda_fail(e, "verify_accept cooperative launch");
  return SPADE_OK;
}
