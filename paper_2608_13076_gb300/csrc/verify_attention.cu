// verify_attention.cu -- attention of the k+1 verify positions of every sequence
// against its bf16 KV cache (the verifier's single forward pass over the draft
// block: Sec. III-B "Verification Stage", Algorithm 1 cloud step).  This file
// holds the C-ABI entry points (head dim 128 dispatches to the tensor-memory
// kernel in verify_attention_tc.cu) and the warp-MMA kernel used for head dim 64.
//
// Warp-MMA kernel design (GB300):
//  * Work unit = (sequence b, KV head, block of <= 64 query rows).  The G query
//    heads of a KV head times the k_b+1 positions form the rows, so every K/V
//    tile fetched from HBM is used by all of them (GQA grouping).
//  * Split-KV as a stream-K schedule: the key chunks (64 keys) of all units are
//    laid end to end and cut into one equal range per CTA (grid = SM count), so
//    ragged batches stay balanced.  A unit cut between CTAs leaves fp32
//    partials (O, running max, running sum) in the workspace; the CTA that
//    finishes a unit last (atomic counter) merges them by log-sum-exp.
//  * One producer warp streams K/V chunks with TMA (128B-swizzled boxes) into a
//    multi-stage ring guarded by mbarriers; consumer warps run the QK^T and PV
//    products on bf16 warp MMAs with fp32 accumulators and an online softmax
//    whose row statistics are merged with warp shuffles.
//  * The causal mask is applied only to chunks that reach past ctx_b, i.e.
//    inside the draft block; cache slots beyond ctx_b + k_b are zeroed in the
//    value fragments so whatever they hold cannot reach the result.
#include <mutex>

#include "attn_common.cuh"

namespace spade {
namespace attn {

constexpr int kSmemBudget = 220 * 1024;

template <int D, int MT>
struct Layout {
  static constexpr int KS = (MT == 1) ? 4 : 2;  // key slices per stage
  static constexpr int NW = MT * KS;            // consumer warps
  static constexpr int THREADS = 32 * (NW + 1);
  static constexpr int KW = kChunk / KS;  // keys per consumer warp per stage
  static constexpr int BOXES = D / 64;    // 128-byte swizzle boxes per tile row
  static constexpr int TILE_BYTES = kChunk * D * 2;
  static constexpr int STAGE_BYTES = 2 * TILE_BYTES;
  static constexpr int Q_BYTES = kRowBlock * D * 2;
  static constexpr int MERGE_BYTES = (KS > 1) ? NW * 16 * D * 4 : 0;
  static constexpr int ML_BYTES = NW * 32 * 4;
  static constexpr int SCHED_BYTES = kMaxB * 8 + (kMaxB + 1) * 8;
  static constexpr int FIXED = Q_BYTES + MERGE_BYTES + ML_BYTES + SCHED_BYTES + 512;
  static constexpr int STAGES_RAW = (kSmemBudget - FIXED - 1024) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_RAW > 8 ? 8 : STAGES_RAW;
  static_assert(STAGES >= 2, "pipeline needs two stages");
  static constexpr int OFF_Q = STAGES * STAGE_BYTES;
  static constexpr int OFF_MERGE = OFF_Q + Q_BYTES;
  static constexpr int OFF_ML = OFF_MERGE + MERGE_BYTES;
  static constexpr int OFF_PREF = OFF_ML + ML_BYTES;          // int64 [kMaxB + 1]
  static constexpr int OFF_CTX = OFF_PREF + (kMaxB + 1) * 8;  // int32 [kMaxB]
  static constexpr int OFF_K = OFF_CTX + kMaxB * 4;           // int32 [kMaxB]
  static constexpr int OFF_BAR = round_up_c(OFF_K + kMaxB * 4, 8);
  static constexpr int OFF_MISC = OFF_BAR + 2 * STAGES * 8;
  static constexpr int SMEM = OFF_MISC + 64 + 1024;  // + slack for 1024-byte alignment
};

// Byte offset of 16-byte chunk `c` (0..D/8-1) of row `r` inside a K/V stage
// tile written by TMA with 128-byte swizzle (box = 64 rows x 128 bytes).
__device__ __forceinline__ uint32_t sw128_off(int r, int c) {
  return (c >> 3) * (kChunk * 128) + r * 128 + (((c & 7) ^ (r & 7)) << 4);
}

template <int D, int MT>
__global__ void __launch_bounds__(Layout<D, MT>::THREADS, 1)
    verify_attention_kernel(const __grid_constant__ Params p,
                            const __grid_constant__ CUtensorMap tm_k,
                            const __grid_constant__ CUtensorMap tm_v) {
  using L = Layout<D, MT>;
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, derived by pointer arithmetic so that the compiler
  // keeps the shared state space (plain ld/st.shared, not generic accesses).
  uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  int64_t *s_pref = reinterpret_cast<int64_t *>(smem + L::OFF_PREF);
  int32_t *s_ctx = reinterpret_cast<int32_t *>(smem + L::OFF_CTX);
  int32_t *s_kd = reinterpret_cast<int32_t *>(smem + L::OFF_K);
  uint64_t *full_bar = reinterpret_cast<uint64_t *>(smem + L::OFF_BAR);
  uint64_t *empty_bar = full_bar + L::STAGES;
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + L::OFF_MISC);
  volatile int *s_last = s_abort + 1;

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;

  // ---- per-sequence validation and chunk counts ---------------------------
  if (tid == 0) { *s_abort = 0; *s_last = 0; }
  sched_validate(p, s_ctx, s_kd, tid, blockDim.x);
  block_sync();
  Sched sc;
  sc.pref = s_pref; sc.ctx = s_ctx; sc.kd = s_kd;
  sc.B = p.B; sc.Hkv = p.Hkv; sc.G = p.G; sc.RB = p.RB; sc.E = p.unit_cost; sc.num_ctas = p.num_ctas;
  if (warp == 0) {
    sched_scan(p, sc, s_pref, lane);
  } else if (warp == 1 && lane == 0) {
    for (int s = 0; s < L::STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], L::NW);
    }
    fence_mbar_init();
  }
  block_sync();
  sc.total = s_pref[p.B];
  if (sc.total == 0) return;
  // Never more CTAs than chunks: every CTA kept has a non-empty range, so the
  // CTAs between a unit's first and last owner all contribute a partial.
  sc.num_ctas = static_cast<int>(sc.total < p.num_ctas ? sc.total : p.num_ctas);
  if (static_cast<int>(blockIdx.x) >= sc.num_ctas) return;
  const int64_t x_begin = static_cast<int64_t>(blockIdx.x) * sc.total / sc.num_ctas;
  const int64_t x_end = static_cast<int64_t>(blockIdx.x + 1) * sc.total / sc.num_ctas;

  if (warp == 0) {
    // ======================= producer: TMA K/V chunks =======================
    if (lane == 0) {
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      const uint64_t pol = l2_policy_evict_first();
      uint32_t it = 0, issued = 0;
      bool expired = false;
      for (int64_t x = x_begin; x < x_end;) {
        const Seg g = locate(sc, x);
        const int64_t seg_end = min(x_end, g.ust + g.nch);
        const int row0 = (g.b * p.Hkv + g.kvh) * p.cap;
        for (int ci = g.ci; x < seg_end; ++ci, ++x, ++it) {
          const int s = it % L::STAGES;
          const uint32_t ph = (it / L::STAGES) & 1;
          if (!mbar_wait(&empty_bar[s], ph ^ 1, s_abort)) expired = true;
          if (*s_abort) continue;  // no new copies once any wait has expired
          uint8_t *kt = smem + s * L::STAGE_BYTES;
          uint8_t *vt = kt + L::TILE_BYTES;
          mbar_arrive_expect_tx(&full_bar[s], L::STAGE_BYTES);
          // One box per tile: 64 keys x all of D, landing as [D/64][64 keys][64].
          tma_load_3d(kt, &tm_k, 0, row0 + ci * kChunk, 0, &full_bar[s], pol);
          tma_load_3d(vt, &tm_v, 0, row0 + ci * kChunk, 0, &full_bar[s], pol);
          issued = it + 1;
        }
      }
      if (expired || *s_abort) {
        atomicOr(p.status, SPADE_DEV_TIMEOUT);
        // Drain: every copy issued must land before the CTA's smem goes away.
        for (uint32_t j = (issued > L::STAGES ? issued - L::STAGES : 0); j < issued; ++j) {
          const int s = j % L::STAGES;
          const uint32_t ph = (j / L::STAGES) & 1;
          const uint64_t t0 = globaltimer();
          while (!mbar_try_wait(&full_bar[s], ph) && globaltimer() - t0 < kWaitLimitNs) {}
        }
      }
    }
    return;
  }

  // ========================= consumers =======================================
  const int cw = warp - 1;       // consumer warp index
  const int mt = cw % MT;        // m16 tile of the row block
  const int ks = cw / MT;        // key slice of each stage
  const int NT = L::NW * 32;
  const int ctid = tid - 32;
  uint8_t *s_q = smem + L::OFF_Q;
  float *s_merge = reinterpret_cast<float *>(smem + L::OFF_MERGE);
  float *s_ml = reinterpret_cast<float *>(smem + L::OFF_ML);
  const uint32_t s_q_u32 = smem_u32(s_q);
  bool expired = false;
  uint32_t it = 0;

  for (int64_t x = x_begin; x < x_end;) {
    const Seg g = locate(sc, x);
    const int64_t seg_end = min(x_end, g.ust + g.nch);
    const int n_here = static_cast<int>(seg_end - x);
    const int ctx = s_ctx[g.b];
    const int kd = s_kd[g.b];
    const int Mb = p.G * (kd + 1);
    const int nrow = min(kRowBlock, Mb - kRowBlock * g.rb);
    const int Lkeys = ctx + kd + 1;
    const int q_row0 = p.cu_q[g.b];
    const bool active = mt * 16 < nrow;

    // ---- stage Q of this unit into smem (swizzled 16-byte chunks) ----------
    named_bar(1, NT);
    for (int e = ctid; e < kRowBlock * (D / 8); e += NT) {
      const int r = e / (D / 8), c = e % (D / 8);
      uint4 v = make_uint4(0, 0, 0, 0);
      if (r < nrow) {
        const int row = kRowBlock * g.rb + r;
        const int i = row / p.G, gh = row % p.G;
        const size_t off = (static_cast<size_t>(q_row0 + i) * p.Hq + g.kvh * p.G + gh) * D + c * 8;
        v = *reinterpret_cast<const uint4 *>(p.q + off);
      }
      const int pc = (c & ~7) | ((c & 7) ^ (r & 7));
      *reinterpret_cast<uint4 *>(s_q + r * (D * 2) + pc * 16) = v;
    }
    named_bar(1, NT);

    // A fragments of this warp's 16 query rows, all of D.
    uint32_t qa[D / 16][4];
    if (active) {
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const int r = mt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int c = kk * 2 + (lane >> 4);
        const int pc = (c & ~7) | ((c & 7) ^ (r & 7));
        ldmatrix_x4(s_q_u32 + r * (D * 2) + pc * 16, qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3]);
      }
    }
    // Row limits: row -> position i = row / G sees keys [0, ctx + i].
    const int rloc0 = mt * 16 + (lane >> 2);
    const int rg0 = kRowBlock * g.rb + rloc0, rg1 = rg0 + 8;
    const int lim0 = ctx + (rg0 < Mb ? rg0 / p.G : kd);
    const int lim1 = ctx + (rg1 < Mb ? rg1 / p.G : kd);

    float o[D / 8][4];
#pragma unroll
    for (int j = 0; j < D / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

    for (int ci = g.ci; ci < g.ci + n_here; ++ci, ++it) {
      const int s = it % L::STAGES;
      const uint32_t ph = (it / L::STAGES) & 1;
      if (!mbar_wait(&full_bar[s], ph, s_abort)) expired = true;
      if (active) {
        const uint32_t kt = smem_u32(smem + s * L::STAGE_BYTES);
        const uint32_t vt = kt + L::TILE_BYTES;
        const int key_w = ks * L::KW;  // first key of this warp inside the chunk
        // ---- S = Q K^T (16 rows x KW keys) ----
        float sacc[L::KW / 8][4];
#pragma unroll
        for (int j = 0; j < L::KW / 8; ++j) sacc[j][0] = sacc[j][1] = sacc[j][2] = sacc[j][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
#pragma unroll
          for (int n2 = 0; n2 < L::KW / 16; ++n2) {
            const int key = key_w + n2 * 16 + (lane & 7) + (lane >> 4) * 8;
            const int c = kk * 2 + ((lane >> 3) & 1);
            uint32_t b0, b1, b2, b3;
            ldmatrix_x4(kt + sw128_off(key, c), b0, b1, b2, b3);
            mma_bf16_16816(sacc[2 * n2], qa[kk], b0, b1);
            mma_bf16_16816(sacc[2 * n2 + 1], qa[kk], b2, b3);
          }
        }
        // ---- scale, causal mask inside the draft block, online softmax ----
        const int key_base = ci * kChunk + key_w + 2 * (lane & 3);
        const bool need_mask = ci * kChunk + kChunk - 1 > ctx;
        float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
        for (int j = 0; j < L::KW / 8; ++j) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            float t0 = sacc[j][e] * p.scale_log2;
            float t1 = sacc[j][2 + e] * p.scale_log2;
            if (need_mask) {
              const int key = key_base + j * 8 + e;
              if (key > lim0) t0 = -INFINITY;
              if (key > lim1) t1 = -INFINITY;
            }
            sacc[j][e] = t0;
            sacc[j][2 + e] = t1;
            mx0 = fmaxf(mx0, t0);
            mx1 = fmaxf(mx1, t1);
          }
        }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        const float mu0 = (mn0 == -INFINITY) ? 0.f : mn0;
        const float mu1 = (mn1 == -INFINITY) ? 0.f : mn1;
        const float a0 = ex2(m0 - mu0), a1 = ex2(m1 - mu1);
        m0 = mn0;
        m1 = mn1;
        float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
        for (int j = 0; j < L::KW / 8; ++j) {
          sacc[j][0] = ex2(sacc[j][0] - mu0);
          sacc[j][1] = ex2(sacc[j][1] - mu0);
          sacc[j][2] = ex2(sacc[j][2] - mu1);
          sacc[j][3] = ex2(sacc[j][3] - mu1);
          rs0 += sacc[j][0] + sacc[j][1];
          rs1 += sacc[j][2] + sacc[j][3];
        }
        l0 = l0 * a0 + rs0;
        l1 = l1 * a1 + rs1;
#pragma unroll
        for (int j = 0; j < D / 8; ++j) {
          o[j][0] *= a0; o[j][1] *= a0;
          o[j][2] *= a1; o[j][3] *= a1;
        }
        // ---- O += P V ----
        const bool tail = ci * kChunk + kChunk > Lkeys;
#pragma unroll
        for (int k2 = 0; k2 < L::KW / 16; ++k2) {
          uint32_t pa[4];
          pa[0] = pack_bf16(sacc[2 * k2][0], sacc[2 * k2][1]);
          pa[1] = pack_bf16(sacc[2 * k2][2], sacc[2 * k2][3]);
          pa[2] = pack_bf16(sacc[2 * k2 + 1][0], sacc[2 * k2 + 1][1]);
          pa[3] = pack_bf16(sacc[2 * k2 + 1][2], sacc[2 * k2 + 1][3]);
          // Keys of this thread's value-fragment halves (for the tail zeroing).
          const int kb = ci * kChunk + key_w + k2 * 16 + 2 * (lane & 3);
          uint32_t vmask0 = 0xffffffffu, vmask1 = 0xffffffffu;
          if (tail) {
            vmask0 = (kb < Lkeys ? 0x0000ffffu : 0u) | (kb + 1 < Lkeys ? 0xffff0000u : 0u);
            vmask1 = (kb + 8 < Lkeys ? 0x0000ffffu : 0u) | (kb + 9 < Lkeys ? 0xffff0000u : 0u);
          }
#pragma unroll
          for (int dn = 0; dn < D / 16; ++dn) {
            const int key = key_w + k2 * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
            const int c = dn * 2 + (lane >> 4);
            uint32_t b0, b1, b2, b3;
            ldmatrix_x4_trans(vt + sw128_off(key, c), b0, b1, b2, b3);
            mma_bf16_16816(o[2 * dn], pa, b0 & vmask0, b1 & vmask1);
            mma_bf16_16816(o[2 * dn + 1], pa, b2 & vmask0, b3 & vmask1);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[s]);
    }
    if (expired) {
      atomicOr(p.status, SPADE_DEV_TIMEOUT);
      expired = false;
    }
    x = seg_end;

    // ---- merge the key slices of this CTA --------------------------------
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    if constexpr (L::KS > 1) {
      float *mo = s_merge + cw * 16 * D;
      if ((lane & 3) == 0) {
        s_ml[cw * 32 + (lane >> 2)] = m0;
        s_ml[cw * 32 + (lane >> 2) + 8] = m1;
        s_ml[cw * 32 + 16 + (lane >> 2)] = l0;
        s_ml[cw * 32 + 16 + (lane >> 2) + 8] = l1;
      }
#pragma unroll
      for (int j = 0; j < D / 8; ++j) {
        const int d = j * 8 + 2 * (lane & 3);
        *reinterpret_cast<float2 *>(mo + (lane >> 2) * D + d) = make_float2(o[j][0], o[j][1]);
        *reinterpret_cast<float2 *>(mo + ((lane >> 2) + 8) * D + d) = make_float2(o[j][2], o[j][3]);
      }
      named_bar(1, NT);
      if (ks == 0) {
        float M0 = -INFINITY, M1 = -INFINITY;
#pragma unroll
        for (int s2 = 0; s2 < L::KS; ++s2) {
          M0 = fmaxf(M0, s_ml[(mt + s2 * MT) * 32 + (lane >> 2)]);
          M1 = fmaxf(M1, s_ml[(mt + s2 * MT) * 32 + (lane >> 2) + 8]);
        }
        const float U0 = (M0 == -INFINITY) ? 0.f : M0, U1 = (M1 == -INFINITY) ? 0.f : M1;
        float w0[L::KS], w1[L::KS];
        float L0 = 0.f, L1 = 0.f;
#pragma unroll
        for (int s2 = 0; s2 < L::KS; ++s2) {
          const int w = mt + s2 * MT;
          w0[s2] = ex2(s_ml[w * 32 + (lane >> 2)] - U0);
          w1[s2] = ex2(s_ml[w * 32 + (lane >> 2) + 8] - U1);
          L0 += w0[s2] * s_ml[w * 32 + 16 + (lane >> 2)];
          L1 += w1[s2] * s_ml[w * 32 + 16 + (lane >> 2) + 8];
        }
#pragma unroll
        for (int j = 0; j < D / 8; ++j) {
          const int d = j * 8 + 2 * (lane & 3);
          float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
          for (int s2 = 0; s2 < L::KS; ++s2) {
            const float *mw = s_merge + (mt + s2 * MT) * 16 * D;
            const float2 v0 = *reinterpret_cast<const float2 *>(mw + (lane >> 2) * D + d);
            const float2 v1 = *reinterpret_cast<const float2 *>(mw + ((lane >> 2) + 8) * D + d);
            acc0.x += w0[s2] * v0.x; acc0.y += w0[s2] * v0.y;
            acc1.x += w1[s2] * v1.x; acc1.y += w1[s2] * v1.y;
          }
          o[j][0] = acc0.x; o[j][1] = acc0.y; o[j][2] = acc1.x; o[j][3] = acc1.y;
        }
        m0 = M0; m1 = M1; l0 = L0; l1 = L1;
      }
    }

    // ---- emit: final output, or a partial for the cross-CTA merge ---------
    const int unit = (g.b * p.Hkv + g.kvh) * p.RB + g.rb;
    const int64_t c_first = sc.owner(g.ust + sc.E);
    const int64_t c_last = sc.owner(g.ust + sc.E + g.nch - 1);
    const int nparts = static_cast<int>(c_last - c_first + 1);
    const bool writer = (ks == 0) && active;
    if (nparts == 1) {
      if (writer) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int rl = rloc0 + 8 * h;
          if (rl < nrow) {
            const int row = kRowBlock * g.rb + rl;
            const int i = row / p.G, gh = row % p.G;
            const size_t orow = static_cast<size_t>(q_row0 + i) * p.Hq + g.kvh * p.G + gh;
            const float inv = 1.f / (h ? l1 : l0);
#pragma unroll
            for (int j = 0; j < D / 8; ++j) {
              const int d = j * 8 + 2 * (lane & 3);
              *reinterpret_cast<uint32_t *>(p.out + orow * D + d) =
                  pack_bf16(o[j][2 * h] * inv, o[j][2 * h + 1] * inv);
            }
            if (p.lse && (lane & 3) == 0)
              p.lse[orow] = ((h ? m1 : m0) + log2f(h ? l1 : l0)) * 0.69314718055994531f;
          }
        }
      }
    } else {
      const int64_t slot = blockIdx.x + unit;
      float *part = p.partials + slot * slot_floats(D);
      if (writer) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int rl = rloc0 + 8 * h;
#pragma unroll
          for (int j = 0; j < D / 8; ++j) {
            const int d = j * 8 + 2 * (lane & 3);
            __stcg(reinterpret_cast<float2 *>(part + rl * D + d), make_float2(o[j][2 * h], o[j][2 * h + 1]));
          }
          if ((lane & 3) == 0) {
            __stcg(part + kRowBlock * D + rl, h ? m1 : m0);
            __stcg(part + kRowBlock * D + kRowBlock + rl, h ? l1 : l0);
          }
        }
      }
      named_bar(1, NT);
      if (ctid == 0) *s_last = arrive_part(&p.counters[unit], nparts);
      named_bar(1, NT);
      if (*s_last) {
        // This CTA finished the unit last: merge every partial by log-sum-exp.
        merge_partials<D>(p, c_first + unit, nparts, nrow, g.rb, g.kvh, q_row0, cw, L::NW, lane);
        if (ctid == 0) p.counters[unit] = 0;  // every part has arrived: reset for the next call
      }
    }
  }
}

template <int D, int MT>
static cudaError_t launch(const Params &p, const CUtensorMap &tk, const CUtensorMap &tv,
                          cudaStream_t stream) {
  using L = Layout<D, MT>;
  auto kern = verify_attention_kernel<D, MT>;
  static bool configured = false;  // per template instance; the attribute is per function
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  kern<<<p.num_ctas, L::THREADS, L::SMEM, stream>>>(p, tk, tv);
  return cudaGetLastError();
}

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

extern "C" spade_status spade_verify_attention(
    const void *q, const void *k_cache, const void *v_cache, const int32_t *ctx_lens,
    const int32_t *n_draft, const int32_t *cu_q, void *out, float *lse, int32_t B, int32_t Hq,
    int32_t Hkv, int32_t D, int32_t cap, int32_t max_k, int32_t R, void *workspace,
    size_t workspace_bytes, int32_t *status, spade_stream_t stream) {
  if (!q || !k_cache || !v_cache || !ctx_lens || !n_draft || !cu_q || !out || !status)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention: null pointer argument");
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0 || max_k < 0 || R <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention: non-positive size");
  if (Hq % Hkv) return fail(SPADE_ERR_SHAPE, "Hq (%d) must be a multiple of Hkv (%d)", Hq, Hkv);
  if (D != 64 && D != 128) return fail(SPADE_ERR_SHAPE, "head dim %d not supported (64 or 128)", D);
  if (B > attn::kMaxB) return fail(SPADE_ERR_SHAPE, "B = %d exceeds %d sequences per call", B, attn::kMaxB);
  if (R < B) return fail(SPADE_ERR_INVALID_ARG, "R = %d < B = %d", R, B);
  if (static_cast<int64_t>(B) * Hkv * cap >= (int64_t(1) << 31))
    return fail(SPADE_ERR_CAPACITY, "KV cache rows B*Hkv*cap exceed 2^31");
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
  // The tensor-memory kernel charges each unit's epilogue and pipeline restart
  // to the CTA that starts it (about five slices' worth); the warp-MMA kernel
  // keeps the plain split.
  p.unit_cost = (D == 128) ? attn::kUnitCostTc : 0;
  // One CTA per SM, never more CTAs than key chunks could exist.
  const int64_t max_chunks = static_cast<int64_t>(units) * ((cap + attn::kChunk - 1) / attn::kChunk);
  p.num_ctas = static_cast<int>(max_chunks < sms ? max_chunks : sms);

  const uint64_t rows = static_cast<uint64_t>(B) * Hkv * cap;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (D == 128) {
    // Tensor-memory kernel: 128-key boxes of both 64-dim slabs, and 64-key
    // boxes of one slab for a segment's last odd slice.
    CUtensorMap k2, v2, k1, v1;
    if (!encode_tmap_rows_by_slab(&k2, k_cache, rows, D, 128) ||
        !encode_tmap_rows_by_slab(&v2, v_cache, rows, D, 128) ||
        !encode_tmap_rows_by_slab(&k1, k_cache, rows, D, attn::kChunk, 1) ||
        !encode_tmap_rows_by_slab(&v1, v_cache, rows, D, attn::kChunk, 1))
      return SPADE_ERR_CUDA;
    const int rows_max = G * (max_k + 1) < attn::kRowBlock ? G * (max_k + 1) : attn::kRowBlock;
    e = attn::launch_tc(p, k2, v2, k1, v1, (rows_max + 15) / 16 * 16, s);
  } else {
    CUtensorMap tk, tv;
    if (!encode_tmap_rows_by_slab(&tk, k_cache, rows, D, attn::kChunk) ||
        !encode_tmap_rows_by_slab(&tv, v_cache, rows, D, attn::kChunk))
      return SPADE_ERR_CUDA;
    const int mt = (G * (max_k + 1) >= attn::kRowBlock) ? 4 : (G * (max_k + 1) + 15) / 16;
    switch (mt) {
      case 1: e = attn::launch<64, 1>(p, tk, tv, s); break;
      case 2: e = attn::launch<64, 2>(p, tk, tv, s); break;
      case 3: e = attn::launch<64, 3>(p, tk, tv, s); break;
      default: e = attn::launch<64, 4>(p, tk, tv, s); break;
    }
  }
  if (e != cudaSuccess) return cuda_fail(e, "verify_attention launch");
  return SPADE_OK;
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
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || cap <= 0 || max_k < 0 || R <= 0 || Hq % Hkv ||
      (D != 64 && D != 128))
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_attention_noalloc: bad sizes");
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
