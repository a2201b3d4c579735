// attn_common.cuh -- pieces of the verify-attention kernel (tensor memory,
// head dims 64 and 128) shared with its host entry points: parameters, the
// stream-K schedule over key chunks, and the log-sum-exp merge of split
// partials (Sec. III-B "Verification Stage": the verifier's attention of the
// k+1 draft positions against the cached context).
#pragma once
#include <cuda_bf16.h>

#include <cfloat>
#include <cstdint>

#include "internal.h"
#include "ptx.cuh"

namespace spade {
namespace attn {

constexpr int kChunk = 64;     // keys per schedule slice (two per MMA chunk)
constexpr int kRowBlock = 64;  // query rows per work unit
constexpr int kMaxB = 512;     // sequences per call (per-CTA schedule lives in smem)
constexpr int kUnitCostTc = 11; // virtual slices per unit in the tensor-memory kernel's schedule

struct Params {
  const __nv_bfloat16 *q;
  __nv_bfloat16 *out;
  float *lse;
  const int32_t *ctx_lens;
  const int32_t *n_draft;
  const int32_t *cu_q;
  int32_t *counters;  // [units], zero between calls
  float *partials;    // [(num_ctas + units) slots][kRowBlock * D + 2 * kRowBlock]
  int32_t *status;
  int B, Hq, Hkv, G, cap, max_k, R, RB, num_ctas;
  int unit_cost;     // virtual slices charged at each unit's start (the schedule's cost model)
  float scale_log2;  // log2(e) / sqrt(D)
  // Paged cache (block_table null: dense [B, Hkv, cap, D] caches).  The pools
  // are [num_pages, Hkv, page_size, D]; block_table[b * max_pages + j] is the
  // page of sequence b's slots [j * page_size, (j + 1) * page_size).
  const int32_t *block_table;
  int page_size, max_pages, num_pages;
};

// Pool row of the 64-key slice starting at key `key` of (b, kvh) in a paged
// cache.  An out-of-range page id is reported and mapped past the last row,
// where the tensor copy reads zeros.
__device__ __forceinline__ int paged_row(const Params &p, int b, int kvh, int key) {
  const int page = __ldg(p.block_table + static_cast<int64_t>(b) * p.max_pages + key / p.page_size);
  const int64_t rows = static_cast<int64_t>(p.num_pages) * p.Hkv * p.page_size;
  if (page < 0 || page >= p.num_pages) {
    atomicOr(p.status, SPADE_DEV_BAD_INDEX);
    return static_cast<int>(rows);
  }
  return static_cast<int>((static_cast<int64_t>(page) * p.Hkv + kvh) * p.page_size + key % p.page_size);
}

constexpr int round_up_c(int x, int a) { return (x + a - 1) / a * a; }

// n / d for n >= 0, d > 0: a 32-bit division whenever both fit (every schedule
// of practical size), else the 64-bit one.  A 64-bit division is a long
// software sequence, and the schedule sits on the path to the first copy.
__device__ __forceinline__ int64_t div_nn(int64_t n, int64_t d) {
  if (((n | d) >> 31) == 0)
    return static_cast<int64_t>(static_cast<uint32_t>(n) / static_cast<uint32_t>(d));
  return n / d;
}

__host__ __device__ constexpr int slot_floats(int D) { return kRowBlock * D + 2 * kRowBlock; }

// Per-CTA view of the schedule.  The units' key slices are laid end to end in
// a cost space where every unit also carries E virtual slices at its start
// (its epilogue and pipeline restart), and the cost space is cut into one equal
// range per CTA; E = 0 is the plain stream-K split over slices.
struct Sched {
  const int64_t *pref;  // [B+1] cost prefix over sequences
  const int32_t *ctx;   // [B]
  const int32_t *kd;    // [B]  (-1 marks an invalid sequence: no work)
  int B, Hkv, G, RB, E;
  int64_t total;
  int num_ctas;

  __device__ int rows_of(int b) const { return G * (kd[b] + 1); }
  __device__ int rb_count(int b) const {
    return kd[b] < 0 ? 0 : (rows_of(b) + kRowBlock - 1) / kRowBlock;
  }
  __device__ int chunks(int b, int rb) const {
    const int m = rows_of(b);
    const int last_row = min(kRowBlock * (rb + 1), m) - 1;
    const int i_hi = last_row / G;
    return (ctx[b] + i_hi + 1 + kChunk - 1) / kChunk;
  }
  __device__ int cost(int b, int rb) const { return chunks(b, rb) + E; }
  // CTA whose range holds cost position x.
  __device__ int64_t owner(int64_t x) const {
    return div_nn((x + 1) * num_ctas + total - 1, total) - 1;
  }
};

struct Seg {
  int b, kvh, rb;
  int ci;        // cost offset of the position within the unit (0 .. E + nch - 1)
  int nch;       // key slices of the unit
  int64_t ust;   // cost position of the unit's start (its first real slice is at ust + E)
};

// The unit and cost offset of position x inside sequence b's cost range.
__device__ __forceinline__ Seg locate_in(const Sched &s, int b, int64_t x) {
  const int lo = b;
  Seg g;
  g.b = lo;
  g.nch = 0;
  const int nrb = s.rb_count(lo);
  int span = 0;
  for (int rb = 0; rb < nrb; ++rb) span += s.cost(lo, rb);
  int64_t o = x - s.pref[lo];
  g.kvh = static_cast<int>(div_nn(o, span));
  int o2 = static_cast<int>(o - static_cast<int64_t>(g.kvh) * span);
  int cum = 0;
  g.rb = 0;
  for (int rb = 0; rb < nrb; ++rb) {
    const int c = s.cost(lo, rb);
    if (o2 < cum + c) { g.rb = rb; g.nch = c - s.E; break; }
    cum += c;
  }
  g.ci = o2 - cum;
  g.ust = s.pref[lo] + static_cast<int64_t>(g.kvh) * span + cum;
  return g;
}

// Position x of the cost space (one thread): the sequence by binary search.
__device__ __forceinline__ Seg locate(const Sched &s, int64_t x) {
  int lo = 0, hi = s.B - 1;  // largest b with pref[b] <= x
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s.pref[mid] <= x) lo = mid; else hi = mid - 1;
  }
  return locate_in(s, lo, x);
}

// The same for a whole warp (all lanes get the result): lane l tests whether
// sequence b0 + l holds x, so 32 sequences take one vote instead of a chain of
// dependent shared-memory loads.
__device__ __forceinline__ Seg locate_warp(const Sched &s, int64_t x, int lane) {
  int b = 0;
  for (int b0 = 0; b0 < s.B; b0 += 32) {
    const int bb = b0 + lane;
    const bool hit = bb < s.B && s.pref[bb] <= x && x < s.pref[bb + 1];
    const unsigned m = __ballot_sync(0xffffffffu, hit);
    if (m) {
      b = b0 + __ffs(m) - 1;
      break;
    }
  }
  return locate_in(s, b, x);
}

// A CTA's range [x_begin, x_end) of the cost space and the schedule totals,
// computed once by the set-up warp and read by every role.
struct CtaRange {
  int64_t x_begin, x_end, total;
  int num_ctas;
  int active;  // 0: this CTA has no work
};

// bar.sync is the aligned form: every lane of a warp must arrive together.
// Lanes that ran ahead of a divergent lane (a lane-0-only loop) reconverge
// first, so no warp reaches the barrier before all of its lanes do.
__device__ __forceinline__ void named_bar(int id, int threads) {
  __syncwarp();
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}
__device__ __forceinline__ void block_sync() {
  __syncwarp();
  __syncthreads();
}

// Per-sequence validation (all threads of the CTA): invalid sequences get
// kd = -1 (no work) and CTA 0 records why in the status word.
__device__ __forceinline__ void sched_validate(const Params &p, int32_t *s_ctx, int32_t *s_kd,
                                               int tid, int nthreads) {
  for (int b = tid; b < p.B; b += nthreads) {
    const int c = p.ctx_lens[b], k = p.n_draft[b];
    const int q0 = p.cu_q[b], q1 = p.cu_q[b + 1];
    int bad = 0;
    if (c < 0 || k < 0 || k > p.max_k || q0 < 0 || q1 > p.R || q1 - q0 != k + 1) bad = SPADE_DEV_BAD_INDEX;
    else if (static_cast<int64_t>(c) + k + 1 > p.cap) bad = SPADE_DEV_CAPACITY;
    if (bad && blockIdx.x == 0) atomicOr(p.status, bad);
    s_ctx[b] = c;
    s_kd[b] = bad ? -1 : k;
  }
}

// Exclusive prefix over sequences of their costs (one warp):
// W_b = Hkv * sum over row blocks of (chunks(b, rb) + E).
__device__ __forceinline__ void sched_scan(const Params &p, const Sched &sc, int64_t *s_pref,
                                           int lane) {
  int64_t carry = 0;
  for (int b0 = 0; b0 < p.B; b0 += 32) {
    const int b = b0 + lane;
    int64_t w = 0;
    if (b < p.B) {
      const int nrb = sc.rb_count(b);
      int span = 0;
      for (int rb = 0; rb < nrb; ++rb) span += sc.cost(b, rb);
      w = static_cast<int64_t>(p.Hkv) * span;
    }
    int64_t incl = w;
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (b < p.B) s_pref[b] = carry + incl - w;
    carry += __shfl_sync(0xffffffffu, incl, 31);
  }
  if (lane == 0) s_pref[p.B] = carry;
}

// Output row of unit-local row `rl` of row block `rb`: rows are ordered
// (draft position i, query head of the group gh).
__device__ __forceinline__ size_t out_row(const Params &p, int q_row0, int kvh, int rb, int rl) {
  const int row = kRowBlock * rb + rl;
  const int i = row / p.G, gh = row % p.G;
  return static_cast<size_t>(q_row0 + i) * p.Hq + kvh * p.G + gh;
}

// Log-sum-exp merge of the nparts partials (slots slot0 ..) of one unit into
// the bf16 output and the lse, run by warps cw = 0..nw-1 of the CTA that
// finished the unit last.  Online merge over batches of kBatch partials; each
// warp step takes RPW rows, so RPW * kBatch partial rows per lane are in
// flight together.
template <int D, int RPW = 2>
__device__ void merge_partials(const Params &p, int64_t slot0, int nparts, int nrow, int rb,
                               int kvh, int q_row0, int cw, int nw, int lane) {
  constexpr int PER = D / 32;
  constexpr int kBatch = 4;
  for (int rl0 = RPW * cw; rl0 < nrow; rl0 += RPW * nw) {
    float M[RPW], Lsum[RPW], acc[RPW][PER];
#pragma unroll
    for (int h = 0; h < RPW; ++h) {
      M[h] = -INFINITY;
      Lsum[h] = 0.f;
#pragma unroll
      for (int e = 0; e < PER; ++e) acc[h][e] = 0.f;
    }
    for (int s0 = 0; s0 < nparts; s0 += kBatch) {
      float mv[RPW][kBatch], lv[RPW][kBatch], ov[RPW][kBatch][PER];
#pragma unroll
      for (int h = 0; h < RPW; ++h) {
        const int rl = min(rl0 + h, nrow - 1);
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
          if (s0 + j < nparts) {
            const float *ps = p.partials + (slot0 + s0 + j) * slot_floats(D);
            mv[h][j] = __ldcg(ps + kRowBlock * D + rl);
            lv[h][j] = __ldcg(ps + kRowBlock * D + kRowBlock + rl);
            if constexpr (PER == 4) {
              const float4 v = __ldcg(reinterpret_cast<const float4 *>(ps + rl * D + lane * 4));
              ov[h][j][0] = v.x; ov[h][j][1] = v.y; ov[h][j][2] = v.z; ov[h][j][3] = v.w;
            } else {
              const float2 v = __ldcg(reinterpret_cast<const float2 *>(ps + rl * D + lane * 2));
              ov[h][j][0] = v.x; ov[h][j][1] = v.y;
            }
          } else {
            mv[h][j] = -INFINITY;
            lv[h][j] = 0.f;
#pragma unroll
            for (int e = 0; e < PER; ++e) ov[h][j][e] = 0.f;
          }
        }
      }
#pragma unroll
      for (int h = 0; h < RPW; ++h) {
        float Mn = M[h];
#pragma unroll
        for (int j = 0; j < kBatch; ++j) Mn = fmaxf(Mn, mv[h][j]);
        const float U = (Mn == -INFINITY) ? 0.f : Mn;
        const float f = ex2(M[h] - U);
        Lsum[h] *= f;
#pragma unroll
        for (int e = 0; e < PER; ++e) acc[h][e] *= f;
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
          const float w = ex2(mv[h][j] - U);
          Lsum[h] += w * lv[h][j];
#pragma unroll
          for (int e = 0; e < PER; ++e) acc[h][e] += w * ov[h][j][e];
        }
        M[h] = Mn;
      }
    }
#pragma unroll
    for (int h = 0; h < RPW; ++h) {
      const int rl = rl0 + h;
      if (rl < nrow) {
        const size_t orow = out_row(p, q_row0, kvh, rb, rl);
        const float inv = 1.f / Lsum[h];
        if constexpr (PER == 4) {
          uint2 v;
          v.x = pack_bf16(acc[h][0] * inv, acc[h][1] * inv);
          v.y = pack_bf16(acc[h][2] * inv, acc[h][3] * inv);
          *reinterpret_cast<uint2 *>(p.out + orow * D + lane * 4) = v;
        } else {
          *reinterpret_cast<uint32_t *>(p.out + orow * D + lane * 2) =
              pack_bf16(acc[h][0] * inv, acc[h][1] * inv);
        }
        if (p.lse && lane == 0) p.lse[orow] = (M[h] + log2f(Lsum[h])) * 0.69314718055994531f;
      }
    }
  }
}

// Arrival of one split part at its unit's counter (one thread, after a CTA
// barrier that orders every partial store of the CTA before it): the
// acquire-release atomic publishes this CTA's partial and, for the last part,
// makes every other part visible.  Returns true for the last part.
__device__ __forceinline__ bool arrive_part(int32_t *counter, int nparts) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;" : "=r"(old) : "l"(counter) : "memory");
  return old == nparts - 1;
}

// Tensor-memory kernel for head dims 64 and 128 (verify_attention_tc.cu).  The
// four tensor maps view the K and V caches as [rows][64] slabs: `k2`/`v2`
// fetch 128 keys x every slab per box, `k1`/`v1` 64 keys x one slab.
cudaError_t launch_tc(const Params &p, const CUtensorMap &k2, const CUtensorMap &v2,
                      const CUtensorMap &k1, const CUtensorMap &v1, int nr, int d, cudaStream_t stream);

}  // namespace attn
}  // namespace spade
