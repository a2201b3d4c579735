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
//  * W and hidden arrive by TMA in 32 KB boxes: a 3-D view of the row-major
//    matrix fetches 128 rows x 2 k-chunks at once and lands them as two
//    canonical 128B-swizzled K-major tiles (a 2-D view covers a ragged tail).
//  * One CTA per SM (cooperative launch) owns a contiguous vocabulary slice.
//    All its tiles' logits stay resident in TMEM (512 columns x 128 lanes);
//    finished tiles are compacted from the padded MMA width to the row count,
//    which frees columns for the next round of tiles.  Logits never reach HBM.
//  * Warp roles: warp 0 issues TMA loads, warp 1 owns TMEM and issues the
//    MMAs from a single thread, warps 2-5 read accumulators back (tcgen05.ld)
//    and reduce per-row max / sum-exp / argmax across the vocabulary (an
//    8-row shared-memory transpose, then a 4-lane shuffle merge).
//  * Bounded device-wide barriers separate the phases: after the first, CTA c
//    merges the slice statistics of rows c, c + NC, ...; after the second every
//    CTA holds max, sum-exp and argmax of every row and takes the accept
//    decisions; after the third (only with stochastic sequences) the slice
//    masses of the distribution to sample (residual or p, float-float sums)
//    are known, and the CTA whose slice holds the point u*Z locates its
//    32-entry segment and scans it in vocabulary order to pick the token.
//  * More verify rows than TMEM keeps resident: two launches.  The first keeps
//    only the row statistics and takes the decisions; with an even grid it
//    runs on CTA pairs (clusters of two, tcgen05 cta_group::2): one MMA of
//    M = 256 takes A rows 0-127 from the even CTA's shared memory and
//    128-255 from the odd one's, and splits each N-chunk's hidden rows
//    between them, so an SM receives half the hidden bytes per k-chunk.  The
//    second launch recomputes only the rows to sample.
#include <cuda_bf16.h>

#include <cfloat>

#include "internal.h"
#include "ptx.cuh"

namespace spade {
namespace accept {

constexpr int kTileV = 128;    // vocab rows per tile (MMA M)
constexpr int kKChunk = 64;    // K elements per 128-byte swizzle row
constexpr int kEpiWarps = 4;
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr int kMaxRes = 256;   // rows kept resident in TMEM (MMA N <= 256)
constexpr int kMaxR = 512;     // verify rows per call (two-pass path above kMaxRes)
constexpr int kMaxB = 256;
constexpr int kMaxRounds = 32;
// Kernel kinds.  kResident: the whole step in one launch, logits resident in
// TMEM.  kStatsOnly: first pass for more rows than TMEM holds -- statistics and
// accept decisions only; the rows to sample are gathered into the workspace.
// kPresampled: second pass, resident, on the gathered rows with the decisions
// already taken.
constexpr int kResident = 0, kStatsOnly = 1, kPresampled = 2;
constexpr int kMaxTilesPerCta = 32;
constexpr int kMaxPairSlots = 16;  // W-ring slots of the short last tile's own round
constexpr int kMaxNC = 256;  // CTAs (vocabulary slices) per launch

// Residual masses through shared memory (phase C): groups of kFG sampled rows
// are staged as p and q slices, then every thread sums 32-entry segments
// serially; slices of at most kFastSlice vocab rows, at most kFastSeqs sampled
// rows (else the register path below).
constexpr int kFG = 8;
static_assert(kFG <= 32, "one lane prepares each staged row");
constexpr int kFastSlice = 1024;
constexpr int kFastSegs = kFastSlice / 32;
constexpr int kFastSeqs = 64;
constexpr int kQStride = kFastSlice + 4;  // floats per staged q row (16-byte multiple)
constexpr int kSegPad = 33;               // floats per staged 32-entry segment (bank skew)
constexpr int kTmemCols = 512;
constexpr int kSmemBudget = 220 * 1024;
constexpr int kSmemMax = 225 * 1024;  // opt-in limit (227 KB) minus static shared memory
constexpr int kWChunkBytes = kTileV * kKChunk * 2;  // 16 KB: one tile x one k-chunk
static_assert(kEpiWarps * kMaxR * 16 <= 2 * kWChunkBytes, "per-warp row statistics fit two W slots");
constexpr float kLog2e = 1.4426950408889634f;

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
  unsigned *bar;     // [0]: arrival count, [kGenWord * (1 + r)]: generation copy r
  float4 *pstat;     // [NC][R]: slice max, slice sum-exp, slice argmax (bits), -
  float *ldraft;     // [R]: logit of the row's draft token
  float4 *gstat;     // [kReplicas][R]: merged row max, sum-exp, argmax (bits)
  float2 *zpart;     // [kReplicas][NC][B]: slice mass of the sampled distribution (float-float)
  int4 *samp;        // [B]: sample specs written by kStatsOnly, read by kPresampled:
                     //      draft_probs row (-1: sample p), uniform bits, output index, row
  int *samp_count;   // number of specs
  const float *temperature;  // [B] softmax temperature of each sequence, or null (all 1)
  const float *top_p;        // [B] nucleus mass of each sequence, or null (no truncation)
  unsigned *nhist;           // [R][NC][kNucBins]: each CTA's bin masses of the nucleus search
                             // (fixed point, 2^31 = all of p)
  uint4 *nstate;             // [kReplicas][R]: key prefix, mass above the prefix's range, its upper mass
  __nv_bfloat16 *hidden_s;      // [B, H]: gathered hidden rows of the samples
  const __nv_bfloat16 *hidden;  // the call's hidden rows (gather source)
  // Fused KV commit (null kc: not requested): clear the rejected draft slots of
  // the caches [B, Hkv, cap, Dk] and advance ctx_lens once the decisions exist.
  uint4 *kc, *vc;
  int32_t *ctx_lens;
  int Hkv, Dk, cap;
  // Paged caches (block_table non-null): kc / vc are pools [num_pages, Hkv,
  // page_size, Dk]; slot s of sequence b is row s % page_size of page
  // block_table[b * max_pages + s / page_size]; cap = max_pages * page_size.
  const int32_t *block_table;
  int page_size, max_pages, num_pages;
  int kind;
  int pair;          // statistics pass on CTA pairs (cta_group::2), see phase A
  int nchunks;       // MMA N-chunks per tile (2 when Ncols > 256)
  int n0w;           // width of the first N-chunk
  uint32_t idesc1;   // instruction descriptor of the second N-chunk
  int h_box_rows, h_boxes;  // hidden rows per TMA box, boxes per k-chunk
  int B, R, H, V, T, NC, Ncols, Rs;
  int KC;            // k-chunks of 64 (the last may be partial)
  int KCF;           // full k-chunks (H / 64)
  int KG;            // k-chunks per pipeline stage
  int NS;            // pipeline stages per tile pass = ceil(KC / KG)
  int nrounds;
  int round_tiles[kMaxRounds];
  int HS, WS;        // hidden / W ring slots
  int BRS;           // box rows of the map used for a slice's last, partial tile
  int fastc;         // phase C through shared memory (slices <= kFastSlice, room in the rings)
  int qbulk;         // q rows may be bulk-copied (16-byte aligned rows)
  uint32_t idesc;
  uint32_t tmem_cols;
};

struct Smem {
  int w_slot, h_slot;
  int off_h, off_bar, off_misc, off_rows, off_tbuf, total;
};

__host__ __device__ inline Smem smem_layout(const Params &p) {
  Smem s;
  s.w_slot = p.KG * kWChunkBytes;
  s.h_slot = p.KG * p.h_boxes * p.h_box_rows * 128;
  s.off_h = p.WS * s.w_slot;
  s.off_bar = s.off_h + p.HS * s.h_slot;
  // 128-byte aligned: the float4 statistics in the transpose region below
  // inherit this alignment.
  s.off_misc = (s.off_bar + (2 * p.WS + 2 * p.HS + 3 + 2 * kMaxPairSlots) * 8 + 127) & ~127;
  s.off_rows = s.off_misc + 64;  // int/float [5][kMaxR] + int [3][kMaxB + 1]
  // Per epilogue warp a 32 x 33 float transpose buffer.  After the last round
  // the warps' per-row statistics (float4 [kEpiWarps][R], at most 32 KB) go to
  // the start of the W ring (at least two 16 KB slots), idle by then.
  s.off_tbuf = s.off_rows + 5 * kMaxR * 4 + 3 * (kMaxB + 1) * 4 + 4;
  s.total = s.off_tbuf + kEpiWarps * 32 * 33 * 4 + 1024;
  return s;
}

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

// barrier.red.or over `threads` threads of named barrier `id`: true on every
// thread if `pred` holds on any.
__device__ __forceinline__ bool bar_or(int id, int threads, bool pred) {
  uint32_t r;
  __syncwarp();
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "barrier.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(pred)), "r"(id), "r"(threads)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ unsigned ld_relaxed(const unsigned *p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Word offset of the grid barrier's generation counter: its own 128-byte line,
// apart from the arrival count, so the waiting CTAs' polls do not queue behind
// the arrival atomics on one L2 line.
// Data that every CTA reads right after a grid barrier (the merged row
// statistics, the slice masses) is written in kReplicas copies, and CTA c reads
// copy c % kReplicas: 152 CTAs loading the same L2 lines at once queue on them
// for several microseconds, a handful per line do not.  The barrier's
// generation word is replicated the same way, one 128-byte line per copy.
constexpr int kReplicas = 8;
constexpr int kNucBinBits = 5;                 // key bits decided per round of the nucleus search
constexpr int kNucBins = 1 << kNucBinBits;     // bins per round
constexpr int kNucRounds = 4;                  // all 20 key bits, see nuc_key
constexpr int kNucSubs = 4;                    // independent bin copies per lane (see phase B (3b))
constexpr int kGenWord = 32;      // words between the arrival count and each generation copy
constexpr int kBarBytes = 2048;  // barrier words at the workspace's start
static_assert(kGenWord * (kReplicas + 1) * 4 <= kBarBytes, "barrier words fit their region");

// Device-wide barrier among the NC co-resident CTAs (cooperative launch).  The
// last CTA to arrive resets the count and bumps the generation; the others
// poll the generation (relaxed loads with a short back-off, then an acquire
// fence) with a time limit.  Returns false if the wait expired.
// Not inlined: the kernel passes it four times after the vocabulary sweep,
// and one copy of its code stays in the instruction cache.
__device__ __noinline__ bool grid_barrier(unsigned *bar, int nctas) {
  __shared__ int s_ok;
  block_sync();
  if (threadIdx.x == 0) {
    s_ok = 1;
    unsigned *gen_p = bar + kGenWord * (1 + blockIdx.x % kReplicas);
    // Read before arriving (the arrival's release orders this load first).
    const unsigned gen = ld_relaxed(gen_p);
    unsigned arrived;
    // The arrival releases this CTA's writes (ordered before it by bar.sync).
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(arrived) : "l"(bar) : "memory");
    if (arrived == static_cast<unsigned>(nctas) - 1) {
      asm volatile("st.relaxed.gpu.global.u32 [%0], 0;" ::"l"(bar) : "memory");
      // One release fence orders everything above before all the copies.
      asm volatile("fence.acq_rel.gpu;" ::: "memory");
      for (int r = 0; r < kReplicas; ++r)
        asm volatile("red.relaxed.gpu.global.add.u32 [%0], 1;" ::"l"(bar + kGenWord * (1 + r)) : "memory");
    } else {
      const uint64_t t0 = globaltimer();
      while (ld_relaxed(gen_p) == gen) {
        if (globaltimer() - t0 > kWaitLimitNs) { s_ok = 0; break; }
        __nanosleep(20);
      }
      asm volatile("fence.acq_rel.gpu;" ::: "memory");
    }
  }
  block_sync();
  return s_ok != 0;
}

// Merge of (max, sum of exp(x - max), argmax) summaries; lowest index wins ties.
__device__ __forceinline__ void stat_merge(float &m, float &s, int &i, float om, float os, int oi) {
  const float M = fmaxf(m, om);
  if (M == -INFINITY) {
    s = 0.f;
  } else {
    s = s * ex2((m - M) * kLog2e) + os * ex2((om - M) * kLog2e);
  }
  if (om > m || (om == m && oi < i)) i = oi;
  m = M;
}

// 1 / T for sequence b: p = softmax(l / T).  A temperature that is not
// positive and finite is reported and taken as 1.
__device__ __forceinline__ float inv_temp(const Params &p, int b) {
  if (p.temperature == nullptr || b < 0) return 1.f;
  const float t = __ldg(p.temperature + b);
  if (!(t > 0.f) || !(t < INFINITY)) {
    atomicOr(p.status, SPADE_DEV_BAD_INDEX);
    return 1.f;
  }
  return 1.f / t;
}

// Top-p (nucleus) threshold search over the scaled logits l of a row.  The
// nucleus is S = {x : l_x >= tau}, tau the largest logit value whose upper
// mass F(tau) = sum_{l_x >= tau} p_x reaches top_p (tokens tied with the
// boundary are in).  The search runs on integer keys
//   L(l) = floor((l - base) * 2^15),  base = m - 31.5  (m: the row maximum),
// a monotone map of l onto [0, 2^20) for every l >= base (p below base is at
// most V e^-31.5); each of kNucRounds rounds fixes 5 more bits of the key of
// the boundary, keeping the highest bin whose upper mass still reaches top_p.
// The nucleus is then {x : L(l_x) >= L_tau}: the same key decides the bins,
// the accept test and the sampling, so all three agree bit for bit.  Logits
// within one key step (2^-15 = 3.1e-5 in l) are not told apart.
constexpr float kNucSpan = 31.5f;
constexpr int kNucKeyBits = 20;
constexpr float kNucScale = 32768.f;  // key steps per unit of l
// y = fma(l, 2^15, -base 2^15) equals (l - base) rounded, times 2^15 (scaling
// by a power of two commutes with rounding); adding 2^23 rounded toward -inf
// leaves floor(y) in the low mantissa bits for 0 <= y < 2^23 (no conversion
// instruction), and a negative key for y < 0.  Monotone in l throughout.
// nb65 = -base * 2^15 (exact).  nuc_key_bits is the float's bit pattern,
// 0x4B000000 + L for L >= 0 (the constant's low 24 bits are zero, so shifts
// of the pattern and of L differ by a constant).
constexpr int kNucKeyBias = 0x4B000000;
__device__ __forceinline__ int nuc_key_bits(float l, float nb65) {
  return __float_as_int(__fadd_rd(__fmaf_rn(l, kNucScale, nb65), 8388608.f));
}
__device__ __forceinline__ int nuc_key(float l, float base) {
  return nuc_key_bits(l, -kNucScale * base) - kNucKeyBias;
}
// top_p of sequence b when it truncates p (0 < top_p < 1), else 1.
__device__ __forceinline__ float seq_top_p(const Params &p, int b) {
  if (p.top_p == nullptr || b < 0) return 1.f;
  const float t = __ldg(p.top_p + b);
  return (t > 0.f && t < 1.f) ? t : 1.f;
}

// Float-float numbers (hi + lo, about 48 significant bits) for the sums that
// place u*Z: GB300's fp64 rate is a small fraction of fp32, so the cumulative
// masses use error-free fp32 transformations instead of doubles.
struct ff2 {
  float hi, lo;
};
// Knuth's TwoSum: s + e == a + b exactly.
__device__ __forceinline__ ff2 two_sum(float a, float b) {
  const float s = a + b;
  const float bb = s - a;
  const float e = (a - (s - bb)) + (b - bb);
  return ff2{s, e};
}
__device__ __forceinline__ ff2 ff_norm(float hi, float lo) {
  const float s = hi + lo;
  return ff2{s, lo - (s - hi)};
}
__device__ __forceinline__ ff2 ff_add(ff2 a, ff2 b) {
  const ff2 s = two_sum(a.hi, b.hi);
  return ff_norm(s.hi, s.lo + a.lo + b.lo);
}
__device__ __forceinline__ ff2 ff_add_f(ff2 a, float b) {
  const ff2 s = two_sum(a.hi, b);
  return ff_norm(s.hi, s.lo + a.lo);
}
__device__ __forceinline__ ff2 ff_sub(ff2 a, ff2 b) { return ff_add(a, ff2{-b.hi, -b.lo}); }
// a * b with the product's rounding error recovered by an fma.
__device__ __forceinline__ ff2 ff_mul_f(ff2 a, float b) {
  const float p = a.hi * b;
  float e = fmaf(a.hi, b, -p);
  e = fmaf(a.lo, b, e);
  return ff_norm(p, e);
}
__device__ __forceinline__ bool ff_gt(ff2 a, ff2 b) {
  const ff2 d = ff_sub(a, b);
  return d.hi > 0.f || (d.hi == 0.f && d.lo > 0.f);
}
__device__ __forceinline__ ff2 ff_shfl(ff2 v, int src) {
  return ff2{__shfl_sync(0xffffffffu, v.hi, src), __shfl_sync(0xffffffffu, v.lo, src)};
}
__device__ __forceinline__ ff2 warp_sum_ff(ff2 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
    v = ff_add(v, ff2{__shfl_xor_sync(0xffffffffu, v.hi, o), __shfl_xor_sync(0xffffffffu, v.lo, o)});
  return ff_shfl(v, 0);  // one value for every lane
}
// Inclusive prefix sum over the warp's lanes.
// Inclusive float-float scan over the 16 lanes of each half warp (j = lane & 15).
__device__ __forceinline__ ff2 half_scan_ff(ff2 v, int j) {
#pragma unroll
  for (int o = 1; o < 16; o <<= 1) {
    const ff2 t{__shfl_up_sync(0xffffffffu, v.hi, o, 16), __shfl_up_sync(0xffffffffu, v.lo, o, 16)};
    if (j >= o) v = ff_add(t, v);
  }
  return v;
}
__device__ __forceinline__ ff2 warp_scan_ff(ff2 v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const ff2 t{__shfl_up_sync(0xffffffffu, v.hi, o), __shfl_up_sync(0xffffffffu, v.lo, o)};
    if (lane >= o) v = ff_add(t, v);
  }
  return v;
}

// PAIR: the statistics pass on CTA pairs (tcgen05 cta_group::2); a kernel uses
// one CTA granularity throughout, so pair mode is its own instance.
template <bool PAIR>
__global__ void __launch_bounds__(kThreads, 1) verify_accept_kernel(
    const __grid_constant__ Params p, const __grid_constant__ CUtensorMap tm_w3,
    const __grid_constant__ CUtensorMap tm_w2, const __grid_constant__ CUtensorMap tm_w2s,
    const __grid_constant__ CUtensorMap tm_w3s, const __grid_constant__ CUtensorMap tm_h3,
    const __grid_constant__ CUtensorMap tm_h2) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, derived by pointer arithmetic so that the compiler
  // keeps the shared state space (plain ld/st.shared, not generic accesses).
  uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const Smem L = smem_layout(p);
  uint8_t *w_ring = smem;
  uint8_t *h_ring = smem + L.off_h;
  uint64_t *w_full = reinterpret_cast<uint64_t *>(smem + L.off_bar);
  uint64_t *w_empty = w_full + p.WS;
  uint64_t *h_full = w_empty + p.WS;
  uint64_t *h_empty = h_full + p.HS;
  uint64_t *acc_full = h_empty + p.HS;
  uint64_t *acc_empty = acc_full + 1;
  uint64_t *fin = acc_empty + 1;  // pair mode: teardown handshake
  uint64_t *pp_full = fin + 1;    // [kMaxPairSlots]: the short tile's round, see comb_ok
  uint64_t *pp_empty = pp_full + kMaxPairSlots;
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + L.off_misc);
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + L.off_misc + 8);
  int *s_any_stoch = reinterpret_cast<int *>(smem + L.off_misc + 16);
  uint64_t *q_bar = reinterpret_cast<uint64_t *>(smem + L.off_misc + 24);  // q slice bulk copies
  int32_t *s_draft = reinterpret_cast<int32_t *>(smem + L.off_rows);
  int32_t *s_seq = s_draft + kMaxR;
  int32_t *s_pos = s_seq + kMaxR;
  float *s_u = reinterpret_cast<float *>(s_pos + kMaxR);   // uniforms[n]
  float *s_qd = s_u + kMaxR;                              // q of the row's draft token
  int32_t *s_cuq = reinterpret_cast<int32_t *>(s_qd + kMaxR);
  int32_t *s_nd = s_cuq + kMaxB + 1;
  int32_t *s_md = s_nd + kMaxB;
  float *s_tbuf = reinterpret_cast<float *>(smem + L.off_tbuf);
  float4 *s_wst = reinterpret_cast<float4 *>(smem);  // after the last round (W ring)

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c = blockIdx.x;
  // This CTA's vocabulary slice [v_lo, v_hi): equal row counts (within one),
  // cut into 128-row tiles; the last tile may be partial.  Pair mode: the
  // pair's slice, cut into 256-row pair tiles whose rows 0-127 belong to the
  // even CTA and 128-255 to the odd one; tile t of this CTA starts at
  // v_lo + t * tstride + toff.
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
  const int nsl = PAIR ? p.NC / 2 : p.NC, sl = PAIR ? c >> 1 : c;
  const int v_lo = static_cast<int>(static_cast<int64_t>(sl) * p.V / nsl);
  const int v_hi = static_cast<int>(static_cast<int64_t>(sl + 1) * p.V / nsl);
  const int tstride = PAIR ? 2 * kTileV : kTileV;
  const int toff = static_cast<int>(rank) * kTileV;
  const int ntiles = (v_hi - v_lo + tstride - 1) / tstride;
  const bool short_last = !PAIR && (v_hi - v_lo) - (ntiles - 1) * kTileV <= p.BRS && p.BRS < kTileV;
  // Second pass with nothing to sample: the whole grid leaves before any set-up.
  if (p.kind == kPresampled && *p.samp_count == 0) return;

  // ---- set-up: barriers, TMEM, per-row bookkeeping -------------------------
  if (tid == 0) {
    *s_abort = 0;
    *s_any_stoch = 0;
    for (int s = 0; s < p.WS; ++s) { mbar_init(&w_full[s], 1); mbar_init(&w_empty[s], 1); }
    for (int s = 0; s < p.HS; ++s) { mbar_init(&h_full[s], 1); mbar_init(&h_empty[s], 1); }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, PAIR ? 2 * kEpiWarps : kEpiWarps);  // pair: both CTAs' epilogues
    mbar_init(fin, 1);
    for (int j = 0; j < kMaxPairSlots; ++j) { mbar_init(&pp_full[j], 1); mbar_init(&pp_empty[j], 1); }
    if (PAIR && rank == 0) {
      // Pair mode: arm every slot's first use with both CTAs' bytes.
      for (int s = 0; s < p.WS; ++s) mbar_arrive_expect_tx(&w_full[s], 2 * kWChunkBytes);
      for (int s = 0; s < p.HS; ++s) mbar_arrive_expect_tx(&h_full[s], 2 * p.h_boxes * p.h_box_rows * 128);
    }
    mbar_init(q_bar, 33);  // thread 0 (with the copies' bytes) and the 32 lanes of warp 1
    fence_mbar_init();
  }
  if (warp == 1) {
    if constexpr (PAIR) {
      tmem_alloc_pair(s_tmem, p.tmem_cols);  // collective: the same columns in both SMs
      tmem_relinquish_pair();
    } else {
      tmem_alloc(s_tmem, p.tmem_cols);
      tmem_relinquish();
    }
  }
  for (int n = tid; n < kMaxR; n += kThreads) { s_draft[n] = -1; s_seq[n] = -1; s_pos[n] = 0; }
  block_sync();
  // Row n = cu_q[b] + i is position i of sequence b; it holds draft i for i < k_b.
  if (p.kind != kPresampled) {
  for (int b = tid; b <= p.B; b += kThreads) s_cuq[b] = p.cu_q[b];
  for (int b = tid; b < p.B; b += kThreads) {
    s_nd[b] = p.n_draft[b];
    s_md[b] = p.mode[b];
  }
  for (int b = tid; b < p.B; b += kThreads) {
    const int r0 = p.cu_q[b], k = p.n_draft[b], r1 = p.cu_q[b + 1];
    if (r0 < 0 || k < 0 || r1 - r0 != k + 1 || r1 > p.R) {
      atomicOr(p.status, SPADE_DEV_BAD_INDEX);
      continue;
    }
    for (int i = 0; i <= k; ++i) {
      s_seq[r0 + i] = b;
      s_pos[r0 + i] = i;
      if (i < k) s_draft[r0 + i] = p.draft_tokens[r0 - b + i];
    }
  }
  }
  tc_fence_before();
  block_sync();
  // Pair mode: both CTAs' barriers exist before either signals the other.
  if constexpr (PAIR) cluster_sync();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  int rounds_issued = 0;  // MMA thread: accumulator rounds committed
  // Every CTA reads the same hidden rows: CTA c walks the K stages starting at
  // stage c mod NS, so at any moment about NC / NS CTAs (not all of them) load
  // the same hidden lines from L2.  Each logit's sum over K changes order only.
  const int k_rot = sl % p.NS;  // a pair walks its stages in one order
  // A round that holds only the short last tile streams one k-chunk per slot,
  // its W rows and hidden rows together, through the H ring's slots and through
  // npw slots of that size carved anew from the W ring (own barriers; each one
  // first written once round 1 has released the W slots it overlaps): at
  // Llama-3-8B sizes 6 + 3 = 9 k-chunks in flight.  That round is bound by the
  // slots' round trip (MMAs done, slot released, refilled, MMA thread woken) and
  // by the MMA thread's issue rate, not by its bytes, so it takes as many slots
  // as fit and keeps each to one chunk, released right after its own MMAs
  // (chunks spread over fewer, larger slots measured slower); a two-ring stage
  // would keep at most HS = 3 in flight.  Needs both boxes to fit an H slot.
  const bool comb_ok = p.kind != kStatsOnly && short_last && p.nchunks == 1 && p.h_boxes == 1 &&
                       (p.BRS + p.h_box_rows) * 128 <= L.h_slot;
  const int comb_pb = (p.BRS + p.h_box_rows) * 128;  // one k-chunk's W rows and hidden rows
  const int comb_npw = min(kMaxPairSlots, p.WS * L.w_slot / comb_pb);

  // ======================= phase A: logits + slice statistics =============
  if (warp == 0) {
    if constexpr (PAIR) {
     if (lane < 2 && ntiles > 0) {
      // Pair mode (statistics pass, one k-chunk per stage): this CTA's 128 W
      // rows of the pair tile (lane 1), and its half of every MMA N-chunk of
      // the hidden rows (lane 0): N-chunk 0 covers rows [0, n0w), N-chunk 1
      // rows [n0w, Ncols); the even CTA holds the first half of each, the odd
      // CTA the second.  The two rings run independently, so W (from HBM)
      // keeps its slots in flight while the hidden ring waits for the MMAs.
      // Both CTAs' copies of a stage complete on the even CTA's full barrier,
      // armed with the bytes of both before either CTA may issue them (at
      // set-up, then by the MMA thread as it takes the previous use).
      const bool is_w = lane == 1;
      tma_prefetch_desc(is_w ? &tm_w2 : &tm_h2);
      const uint64_t pol = is_w ? l2_policy_evict_first() : l2_policy_evict_last();
      const int hb = p.h_box_rows;  // n0w / 2
      const int hrow0 = static_cast<int>(rank) * hb;
      const int hrow1 = p.n0w + static_cast<int>(rank) * ((p.Ncols - p.n0w) / 2);
      uint64_t *const full = is_w ? w_full : h_full;
      uint64_t *const empty = is_w ? w_empty : h_empty;
      const uint32_t full0 = cluster_map(full, 0);
      const int slots = is_w ? p.WS : p.HS;
      uint8_t *const ring = is_w ? w_ring : h_ring;
      const int slot_bytes = is_w ? L.w_slot : L.h_slot;
      uint32_t i = 0, issued = 0, eph = 1;  // empty-barrier parity (the first pass: the preceding phase)
      int s = 0;                           // slot and parity advance by counters
      for (int t = 0; t < ntiles; ++t) {
        const int row0 = v_lo + t * tstride + toff;
        for (int it = 0; it < p.NS; ++it, ++i) {
          const int kc = it + k_rot < p.NS ? it + k_rot : it + k_rot - p.NS;
          mbar_wait(&empty[s], eph, s_abort);
          if (!*s_abort) {
            uint8_t *dst = ring + s * slot_bytes;
            if (is_w) {
              tma_load_2d_pair(dst, &tm_w2, kc * kKChunk, row0, full0 + 8u * s, pol);
            } else {
              for (int bi = 0; bi < p.h_boxes; ++bi)
                tma_load_2d_pair(dst + bi * hb * 128, &tm_h2, kc * kKChunk, bi ? hrow1 : hrow0, full0 + 8u * s, pol);
            }
            issued = i + 1;
          }
          if (++s == slots) { s = 0; eph ^= 1u; }
        }
      }
      // After an expired wait the even CTA drains the copies of both (its full
      // barriers count them); the odd CTA's shared memory stays alive until
      // the teardown handshake with the even CTA.
      if (*s_abort && rank == 0) {
        for (uint32_t j = (issued > (uint32_t)slots ? issued - slots : 0); j < issued; ++j)
          mbar_wait_unabortable(&full[j % slots], (j / slots) & 1);
      }
     }
    } else if (lane == 0 && ntiles > 0) {
      tma_prefetch_desc(&tm_w3);
      tma_prefetch_desc(&tm_w3s);
      tma_prefetch_desc(&tm_h3);
      const uint64_t pol_w = l2_policy_evict_first();
      const uint64_t pol_h = l2_policy_evict_last();
      uint32_t wi = 0, hi = 0, w_issued = 0, h_issued = 0;
      int comb_issued = 0;  // chunks of the short tile's round issued (carved slots' uses follow from it)
      // Ring slots and parities advance by counters (no per-stage divisions).
      int ws_ = 0, hs_ = 0;
      uint32_t wph_ = 0, hph_ = 0;
      int tdone = 0;
      for (int r = 0; r < p.nrounds && tdone < ntiles; ++r) {
        const int nt = min(p.round_tiles[r], ntiles - tdone);
        if (comb_ok && nt == 1 && tdone == ntiles - 1) {
          const int row0 = v_lo + tdone * kTileV;
          const int kr = c % p.KC;
          // The slots in turn: npw carved from the W ring, then the H slots;
          // slot index and pass (parity) advance by counters.
          int si = 0, use = 0;
          for (int it = 0; it < p.KC; ++it) {
            const int kc = it + kr < p.KC ? it + kr : it + kr - p.KC;
            const bool carved = si < comb_npw;
            uint8_t *dst;
            uint64_t *full;
            if (carved) {
              if (use == 0) {
                // Round 1's last use of every W slot this one overlaps is released.
                for (int s = si * comb_pb / L.w_slot; s <= ((si + 1) * comb_pb - 1) / L.w_slot; ++s)
                  mbar_wait(&w_empty[s], (s >= ws_ ? wph_ : wph_ ^ 1u) ^ 1u, s_abort);
              }
              mbar_wait(&pp_empty[si], (use & 1) ^ 1, s_abort);
              dst = w_ring + si * comb_pb;
              full = &pp_full[si];
            } else {
              mbar_wait(&h_empty[hs_], hph_ ^ 1, s_abort);
              dst = h_ring + hs_ * L.h_slot;
              full = &h_full[hs_];
            }
            if (!*s_abort) {
              mbar_arrive_expect_tx(full, comb_pb);
              tma_load_2d(dst, &tm_w2s, kc * kKChunk, row0, full, pol_w);
              tma_load_2d(dst + p.BRS * 128, &tm_h2, kc * kKChunk, 0, full, pol_h);
              if (carved) comb_issued = it + 1; else h_issued = hi + 1;
            }
            if (!carved) {
              ++hi;
              if (++hs_ == p.HS) { hs_ = 0; hph_ ^= 1u; }
            }
            if (++si == comb_npw + p.HS) { si = 0; ++use; }
          }
          tdone += nt;
          continue;
        }
        for (int it = 0; it < p.NS; ++it) {
          const int ks = it + k_rot < p.NS ? it + k_rot : it + k_rot - p.NS;
          const int c0 = ks * p.KG;
          const int nch = min(p.KG, p.KC - c0);
          const bool box3 = (nch == p.KG) && (c0 + p.KG <= p.KCF);
          {
            const int s = hs_;
            mbar_wait(&h_empty[s], hph_ ^ 1, s_abort);
            if (!*s_abort) {
              uint8_t *dst = h_ring + s * L.h_slot;
              const int hk = p.h_boxes * p.h_box_rows * 128;  // bytes per k-chunk
              mbar_arrive_expect_tx(&h_full[s], nch * hk);
              if (box3 && p.h_boxes == 1) {
                tma_load_3d(dst, &tm_h3, 0, 0, c0, &h_full[s], pol_h);
              } else {
                for (int j = 0; j < nch; ++j)
                  for (int bi = 0; bi < p.h_boxes; ++bi)
                    tma_load_2d(dst + j * hk + bi * p.h_box_rows * 128, &tm_h2, (c0 + j) * kKChunk,
                                bi * p.h_box_rows, &h_full[s], pol_h);
              }
              h_issued = hi + 1;
            }
            ++hi;
            if (++hs_ == p.HS) { hs_ = 0; hph_ ^= 1u; }
          }
          for (int j = 0; j < nt; ++j) {
            const int s = ws_;
            mbar_wait(&w_empty[s], wph_ ^ 1, s_abort);
            if (!*s_abort) {
              uint8_t *dst = w_ring + s * L.w_slot;
              const int row0 = v_lo + (tdone + j) * kTileV;
              if (short_last && tdone + j == ntiles - 1) {
                // Partial last tile: BRS-row boxes (BRS a multiple of 8), the k-chunks
                // packed at BRS * 128-byte strides: one 3-D box per stage when it
                // holds KG full chunks (small 2-D boxes stream far slower).  The
                // slot's remaining rows feed accumulator lanes that are never read.
                mbar_arrive_expect_tx(&w_full[s], nch * p.BRS * 128);
                if (box3) {
                  tma_load_3d(dst, &tm_w3s, 0, row0, c0, &w_full[s], pol_w);
                } else {
                  for (int jj = 0; jj < nch; ++jj)
                    tma_load_2d(dst + jj * p.BRS * 128, &tm_w2s, (c0 + jj) * kKChunk, row0, &w_full[s], pol_w);
                }
              } else if (box3) {
                mbar_arrive_expect_tx(&w_full[s], nch * kWChunkBytes);
                tma_load_3d(dst, &tm_w3, 0, row0, c0, &w_full[s], pol_w);
              } else {
                mbar_arrive_expect_tx(&w_full[s], nch * kWChunkBytes);
                for (int jj = 0; jj < nch; ++jj)
                  tma_load_2d(dst + jj * kWChunkBytes, &tm_w2, (c0 + jj) * kKChunk, row0, &w_full[s], pol_w);
              }
              w_issued = wi + 1;
            }
            ++wi;
            if (++ws_ == p.WS) { ws_ = 0; wph_ ^= 1u; }
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
        // Carved slot j was filled once for every issued chunk it = j (mod the cycle).
        for (int j = 0; j < comb_npw && j < comb_issued; ++j) {
          const int fills = (comb_issued - 1 - j) / (comb_npw + p.HS) + 1;
          mbar_wait_unabortable(&pp_full[j], (fills - 1) & 1);
        }
      }
    }
  } else if (warp == 1) {
    if constexpr (PAIR) {
     if (lane == 0 && ntiles > 0 && rank == 0) {
      // Pair mode, even CTA: M = 256 MMAs over both CTAs' stages (its full
      // barriers complete when both CTAs' copies have landed); the slots are
      // freed in both CTAs by one multicast commit.
      // Slot indices and phases advance by counters (no divisions per stage).
      int hs = 0, ws = 0;
      uint32_t hph = 0, wph = 0;
      const uint32_t hb_bytes = static_cast<uint32_t>(p.h_box_rows) * 128u;
      const uint32_t h_pair_bytes = 2u * p.h_boxes * hb_bytes;
      for (int t = 0; t < ntiles; ++t) {
        if (t > 0) mbar_wait_cluster(acc_empty, (t - 1) & 1, s_abort);
        tc_fence_after();
        for (int it = 0; it < p.NS; ++it) {
          // (cta-scope waits: the copies' completion on this barrier orders them
          // for the MMAs issued after it, the odd CTA's included)
          mbar_wait(&h_full[hs], hph, s_abort);
          mbar_wait(&w_full[ws], wph, s_abort);
          // Arm the slots' next use now: its copies are issued only after this
          // stage's commit frees the slots.
          mbar_arrive_expect_tx(&h_full[hs], h_pair_bytes);
          mbar_arrive_expect_tx(&w_full[ws], 2 * kWChunkBytes);
          tc_fence_after();
          const uint32_t w_addr = smem_u32(w_ring + ws * L.w_slot);
          const uint32_t h_addr = smem_u32(h_ring + hs * L.h_slot);
          for (int ci = 0; ci < p.nchunks; ++ci) {
#pragma unroll
            for (int k16 = 0; k16 < kKChunk / 16; ++k16)
              tc_mma_f16_pair(tmem + (ci ? static_cast<uint32_t>(p.n0w) : 0u),
                              smem_desc_sw128(w_addr + 32 * k16),
                              smem_desc_sw128(h_addr + ci * hb_bytes + 32 * k16), ci ? p.idesc1 : p.idesc,
                              (it | k16) != 0);
          }
          tc_commit_pair(&w_empty[ws]);
          tc_commit_pair(&h_empty[hs]);
          if (++hs == p.HS) { hs = 0; hph ^= 1u; }
          if (++ws == p.WS) { ws = 0; wph ^= 1u; }
        }
        tc_commit_pair(acc_full);
        ++rounds_issued;
      }
     } else if (lane == 0 && ntiles > 0) {
      rounds_issued = ntiles;  // odd CTA: the even CTA's commits reach its acc_full too
     }
    } else if (lane == 0 && ntiles > 0) {
      // Ring slots and parities advance by counters (no per-stage divisions).
      int ws_ = 0, hs_ = 0;
      uint32_t wph_ = 0, hph_ = 0;
      int tdone = 0, used = 0;
      for (int r = 0; r < p.nrounds && tdone < ntiles; ++r) {
        const int nt = min(p.round_tiles[r], ntiles - tdone);
        if (r > 0) mbar_wait(acc_empty, (r - 1) & 1, s_abort);
        tc_fence_after();
        if (comb_ok && nt == 1 && tdone == ntiles - 1) {
          // Slot index and pass by counters, and each chunk's two operand
          // descriptors built once (a K step of 16 adds 32 bytes, 2 in the
          // descriptor's address field): the loop issues as few instructions
          // per MMA as it can.
          const uint32_t d_tmem = tmem + static_cast<uint32_t>(used);
          const uint32_t idesc = p.idesc, boff = static_cast<uint32_t>(p.BRS) * 128u;
          const uint32_t carved0 = smem_u32(w_ring), h0 = smem_u32(h_ring);
          int si = 0;
          uint32_t cph = 0;
          for (int it = 0; it < p.KC; ++it) {
            const bool carved = si < comb_npw;
            uint32_t base;
            uint64_t *empty;
            if (carved) {
              mbar_wait(&pp_full[si], cph, s_abort);
              base = carved0 + static_cast<uint32_t>(si * comb_pb);
              empty = &pp_empty[si];
            } else {
              mbar_wait(&h_full[hs_], hph_, s_abort);
              base = h0 + static_cast<uint32_t>(hs_ * L.h_slot);
              empty = &h_empty[hs_];
              if (++hs_ == p.HS) { hs_ = 0; hph_ ^= 1u; }
            }
            if (++si == comb_npw + p.HS) { si = 0; cph ^= 1u; }
            tc_fence_after();
            const uint64_t da = smem_desc_sw128(base), db = smem_desc_sw128(base + boff);
#pragma unroll
            for (int k16 = 0; k16 < kKChunk / 16; ++k16)
              tc_mma_f16(d_tmem, da + 2u * k16, db + 2u * k16, idesc, (it | k16) != 0);
            tc_commit(empty);
          }
          tc_commit(acc_full);
          ++rounds_issued;
          used += nt * p.Rs;
          tdone += nt;
          continue;
        }
        for (int it = 0; it < p.NS; ++it) {
          const int ks = it + k_rot < p.NS ? it + k_rot : it + k_rot - p.NS;
          const int nch = min(p.KG, p.KC - ks * p.KG);
          const int hs = hs_;
          mbar_wait(&h_full[hs], hph_, s_abort);
          tc_fence_after();
          const uint32_t h_addr = smem_u32(h_ring + hs * L.h_slot);
          for (int j = 0; j < nt; ++j) {
            const int ws = ws_;
            mbar_wait(&w_full[ws], wph_, s_abort);
            tc_fence_after();
            const uint32_t w_addr = smem_u32(w_ring + ws * L.w_slot);
            // k-chunk stride in the slot: a full tile's chunks are 16 KB apart,
            // the short last tile's are packed (BRS rows each).
            const uint32_t w_chunk = (short_last && tdone + j == ntiles - 1) ? static_cast<uint32_t>(p.BRS * 128)
                                                                            : static_cast<uint32_t>(kWChunkBytes);
            const uint32_t d_tmem = tmem + static_cast<uint32_t>(used + j * p.Ncols);
            const int hk = p.h_boxes * p.h_box_rows * 128;
            for (int jj = 0; jj < nch; ++jj) {
              for (int ci = 0; ci < p.nchunks; ++ci) {
                // N-chunk ci: TMEM columns and hidden rows from noff on.  Each
                // operand's descriptor is built once per k-chunk; a K step of
                // 16 adds 32 bytes, 2 in the descriptor's address field.
                const uint32_t noff = ci ? static_cast<uint32_t>(p.n0w) : 0u;
                const uint64_t da = smem_desc_sw128(w_addr + jj * w_chunk);
                const uint64_t db = smem_desc_sw128(h_addr + jj * hk + noff * 128);
                const uint32_t idesc = ci ? p.idesc1 : p.idesc;
#pragma unroll
                for (int k16 = 0; k16 < kKChunk / 16; ++k16)
                  tc_mma_f16(d_tmem + noff, da + 2u * k16, db + 2u * k16, idesc, (it | jj | k16) != 0);
              }
            }
            tc_commit(&w_empty[ws]);
            if (++ws_ == p.WS) { ws_ = 0; wph_ ^= 1u; }
          }
          tc_commit(&h_empty[hs]);
          if (++hs_ == p.HS) { hs_ = 0; hph_ ^= 1u; }
        }
        tc_commit(acc_full);
        ++rounds_issued;
        if (p.kind != kStatsOnly) used += nt * p.Rs;  // statistics-only: one slot, reused
        tdone += nt;
      }
    }
  } else {
    // ---- epilogue warps: compaction, then slice statistics per row -------
    const int ew = warp - 2;             // 0..3
    const int q4 = warp & 3;             // TMEM lane quarter this warp may access
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    float *T = s_tbuf + ew * (32 * 33);  // this warp's transpose buffer
    // Running statistics of rows lane + 32 * j over this warp's vocab entries.
    constexpr int kRC = kMaxR / 32;  // 32-row chunks
    float rm[kRC], rs[kRC];
    int ri[kRC];
#pragma unroll
    for (int j = 0; j < kRC; ++j) { rm[j] = -INFINITY; rs[j] = 0.f; ri[j] = INT_MAX; }
    // While the first round accumulates: uniforms and q(draft) of every row.
    for (int n = tid - 64; p.kind != kPresampled && n < p.R; n += kEpiWarps * 32) {
      s_u[n] = p.uniforms[n];
      const int b = s_seq[n], d = s_draft[n];
      float qd = 0.f;
      if (b >= 0 && d >= 0 && d < p.V && s_md[b] == 1 && p.draft_probs != nullptr)
        qd = p.draft_probs[static_cast<size_t>(n - b) * p.V + d];
      s_qd[n] = qd;
    }
    __syncwarp();
    int tdone = 0, used = 0;
    for (int r = 0; r < p.nrounds && tdone < ntiles; ++r) {
      const int nt = min(p.round_tiles[r], ntiles - tdone);
      if (!mbar_wait(acc_full, r & 1, s_abort)) atomicOr(p.status, SPADE_DEV_TIMEOUT);
      tc_fence_after();
      // Compaction: this round's tiles move from stride Ncols to stride Rs, so
      // tile t of the slice ends at column t * Rs and the next round's MMAs
      // may start at once in the columns after it.
      if (p.kind != kStatsOnly && p.Ncols != p.Rs) {
        for (int j = 0; j < nt; ++j) {
          const uint32_t src = tmem + lane_base + static_cast<uint32_t>(used + j * p.Ncols);
          const uint32_t dst = tmem + lane_base + static_cast<uint32_t>(used + j * p.Rs);
          if (src == dst) continue;
          // 32-column steps, each as four 8-column accesses (TMEM addresses here
          // are only 8-column aligned) behind one wait.
          int cc = 0;
          for (; cc + 32 <= p.Rs; cc += 32) {
            uint32_t raw[32];
#pragma unroll
            for (int q = 0; q < 4; ++q) tmem_ld8(src + cc + 8 * q, raw + 8 * q);
            tmem_wait_ld();
#pragma unroll
            for (int q = 0; q < 4; ++q) tmem_st8(dst + cc + 8 * q, raw + 8 * q);
          }
          for (; cc < p.Rs; cc += 8) {
            uint32_t raw[8];
            tmem_ld8(src + cc, raw);
            tmem_wait_ld();
            tmem_st8(dst + cc, raw);
          }
        }
        tmem_wait_st();
      }
      if (p.kind != kStatsOnly) {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty);
      }
      // Statistics of this round's tiles, 32 rows at a time: one TMEM load gives
      // each lane (one vocab entry) 32 rows; a 32 x 33 shared-memory transpose
      // gives each lane one row over the warp's 32 vocab entries, reduced
      // serially -- no shuffles.
      for (int j = 0; j < nt; ++j) {
        const int t = tdone + j;
        const int vlane0 = v_lo + t * tstride + toff + q4 * 32;  // vocab id of lane 0's row
        const bool my_valid = vlane0 + lane < v_hi;       // lanes past the slice are masked
        const uint32_t col = tmem + lane_base + static_cast<uint32_t>(p.kind == kStatsOnly ? 0 : t * p.Rs);
#pragma unroll
        for (int cj = 0; cj < kRC; ++cj) {
          const int r0 = cj * 32;
          if (r0 < p.R) {
            const int nc = min(32, p.Rs - r0);  // columns of this chunk (multiple of 8)
            uint32_t raw[32];
            // Four 8-column loads (8-column aligned addresses) behind one wait.
#pragma unroll
            for (int q = 0; q < 4; ++q)
              if (8 * q < nc) tmem_ld8(col + r0 + 8 * q, raw + 8 * q);
            tmem_wait_ld();
#pragma unroll
            for (int rr = 0; rr < 32; ++rr)
              if (rr < nc) T[lane * 33 + rr] = my_valid ? __uint_as_float(raw[rr]) : -INFINITY;
            __syncwarp();
            const int n = r0 + lane;
            if (lane < nc && n < p.R) {
              // Logits at the row's temperature, l / T (T = 1 without temperatures).
              const int sq = p.kind == kPresampled ? (n < *p.samp_count ? p.samp[n].z : -1) : s_seq[n];
              const float it = inv_temp(p, sq);
              float x[32];
              float m = -INFINITY;
              int mi = 0;
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                x[i] = T[i * 33 + lane] * it;
                if (x[i] > m) { m = x[i]; mi = i; }
              }
              float sm = 0.f;
              if (m != -INFINITY) {
#pragma unroll
                for (int i = 0; i < 32; ++i) sm += ex2((x[i] - m) * kLog2e);
              }
              stat_merge(rm[cj], rs[cj], ri[cj], m, sm, m == -INFINITY ? INT_MAX : vlane0 + mi);
              const int d = s_draft[n];
              if (d >= vlane0 && d < vlane0 + 32 && d < v_hi) p.ldraft[n] = T[(d - vlane0) * 33 + lane] * it;
            }
            __syncwarp();
          }
        }
      }
      if (p.kind == kStatsOnly) {
        // The accumulator slot is read: the next tile may overwrite it (pair
        // mode: the even CTA's MMA thread counts both CTAs' epilogue warps).
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (rank == 0) mbar_arrive(acc_empty);
          else mbar_arrive_cluster(cluster_map(acc_empty, 0));
        }
      } else {
        used += nt * p.Rs;
      }
      tdone += nt;
    }
    // Merge the four warps' statistics and publish this CTA's slice partials.
    named_bar(1, kEpiWarps * 32);  // every warp is done with its transpose buffer
#pragma unroll
    for (int cj = 0; cj < kRC; ++cj) {
      const int n = cj * 32 + lane;
      if (n < p.R) s_wst[ew * p.R + n] = make_float4(rm[cj], rs[cj], __int_as_float(ri[cj]), 0.f);
    }
    named_bar(1, kEpiWarps * 32);
    for (int n = tid - 64; n < p.R; n += kEpiWarps * 32) {
      float m = -INFINITY, s = 0.f;
      int idx = INT_MAX;
      for (int w = 0; w < kEpiWarps; ++w) {
        const float4 st = s_wst[w * p.R + n];
        stat_merge(m, s, idx, st.x, st.y, __float_as_int(st.z));
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
  // (1) Rows n = c, c + NC, ... are merged by this CTA, one warp per row, from
  //     the NC slice partials (every CTA reading every partial would pile all
  //     SMs onto the same L2 lines); the merged statistics go to the workspace.
  {
    constexpr int kChunksPerPass = 5;
    for (int n = c + warp * p.NC; n < p.R; n += (kThreads / 32) * p.NC) {
      float m = -INFINITY, sm = 0.f;
      int idx = INT_MAX;
      for (int cc0 = 0; cc0 < p.NC; cc0 += 32 * kChunksPerPass) {
        float4 st[kChunksPerPass];
#pragma unroll
        for (int i = 0; i < kChunksPerPass; ++i) {
          const int cc = cc0 + i * 32 + lane;
          st[i] = cc < p.NC ? __ldcg(&p.pstat[static_cast<size_t>(cc) * p.R + n])
                            : make_float4(-INFINITY, 0.f, __int_as_float(INT_MAX), 0.f);
        }
#pragma unroll
        for (int i = 0; i < kChunksPerPass; ++i) stat_merge(m, sm, idx, st[i].x, st[i].y, __float_as_int(st[i].z));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, m, o);
        const float os = __shfl_xor_sync(0xffffffffu, sm, o);
        const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
        stat_merge(m, sm, idx, om, os, oi);
      }
      // Every copy holds lane 0's values.
      m = __shfl_sync(0xffffffffu, m, 0);
      sm = __shfl_sync(0xffffffffu, sm, 0);
      idx = __shfl_sync(0xffffffffu, idx, 0);
      // (2) The accept test of this row, from the merged statistics (every CTA
      //     then reads it with them instead of re-loading l[d] after the next
      //     barrier).  Rows past a sequence's drafts, and invalid sequences,
      //     give 0; the leading-accept count is formed after the barrier.
      int ok = 0;
      if (p.kind != kPresampled) {
        const int b = s_seq[n];
        if (b >= 0 && s_pos[n] < s_nd[b]) {
          const int d = s_draft[n];
          if (d < 0 || d >= p.V) {
            if (lane == 0) atomicOr(p.status, SPADE_DEV_BAD_INDEX);
          } else if (!(s_md[b] == 1 && p.draft_probs != nullptr)) {
            ok = (d == idx);
          } else {
            const float pd = expf(__ldcg(&p.ldraft[n]) - m) / sm;
            const float qd = s_qd[n];
            ok = (qd > 0.f) ? (s_u[n] < pd / qd) : (pd > 0.f);
          }
        }
      }
      if (lane < kReplicas)
        __stcg(&p.gstat[static_cast<size_t>(lane) * p.R + n], make_float4(m, sm, __int_as_float(idx), __int_as_float(ok)));
    }
  }
  if (!grid_barrier(p.bar, p.NC)) {
    atomicOr(p.status, SPADE_DEV_TIMEOUT);
    *s_abort = 1;
  }
  // Phase-A buffers are idle now: reuse the W ring for per-row / per-seq data.
  float *g_m = reinterpret_cast<float *>(w_ring);           // [R]
  float *g_s = g_m + kMaxR;                                 // [R]
  int *g_arg = reinterpret_cast<int *>(g_s + kMaxR);        // [R]
  int *s_ok = g_arg + kMaxR;                                // [R]
  int *s_acc = s_ok + kMaxR;                                // [B]
  int *s_rstar = s_acc + kMaxB;                             // [B]
  int *s_owner = s_rstar + kMaxB;                           // [B]
  int *s_usep = s_owner + kMaxB;                            // [B]
  int *s_stoch = s_usep + kMaxB;                            // [B]
  int *s_qidx = s_stoch + kMaxB;                            // [B] draft_probs row, -1: p
  float *s_usmp = reinterpret_cast<float *>(s_qidx + kMaxB); // [B] sampling uniform
  int *s_outb = reinterpret_cast<int *>(s_usmp + kMaxB);    // [B] next_token index
  int *s_seg = s_outb + kMaxB;  // [0..1] tile, quarter; [4], [5] row counts; [6..7] retry flags
  float2 *s_T = reinterpret_cast<float2 *>(s_seg + 16);     // [B] float-float
  float4 *s_zw = reinterpret_cast<float4 *>(s_T + kMaxB);   // [B][kEpiWarps]
  float2 *s_tw = reinterpret_cast<float2 *>(s_zw + kMaxB * kEpiWarps);  // [tiles][kEpiWarps]
  int *s_slist = reinterpret_cast<int *>(s_tw + kMaxTilesPerCta * kEpiWarps);  // [B] sampled sequences
  int *s_slpos = s_slist + kMaxB;                           // [B] position in s_slist, -1: none
  int *g_tkey = s_slpos + kMaxB;                            // [R] nucleus key threshold (INT_MIN: all of p)
  float *f_R = reinterpret_cast<float *>(g_tkey + kMaxR);   // [kFG][kFastSegs][kSegPad] residual terms
  float *f_Q = f_R + kFG * kFastSegs * kSegPad;             // [kFG][kQStride] q of staged rows
  float2 *f_seg = reinterpret_cast<float2 *>(f_Q + kFG * kQStride);  // [kFastSeqs][kFastSegs]
  uint32_t q_phase = 0;
  // (3) Every CTA reads the merged statistics and accept bits of all rows.
  for (int n = tid; n < p.R; n += kThreads) {
    const float4 g = __ldcg(&p.gstat[static_cast<size_t>(c % kReplicas) * p.R + n]);
    g_m[n] = g.x;
    g_s[n] = g.y;
    g_arg[n] = __float_as_int(g.z);
    s_ok[n] = __float_as_int(g.w);
    g_tkey[n] = INT_MIN;
  }
  for (int b = tid; p.kind != kPresampled && b < p.B; b += kThreads) {
    const int md = s_md[b];
    if (md != 0 && md != 1 && c == 0) atomicOr(p.status, SPADE_DEV_BAD_INDEX);
    // Stochastic: mode 1 with q for its drafts (a sequence without drafts
    // samples its bonus token from p and needs none).  Drafts without q are
    // reported and verified greedily.
    const bool noq = md == 1 && p.draft_probs == nullptr && s_nd[b] > 0;
    if (noq && c == 0) atomicOr(p.status, SPADE_DEV_BAD_INDEX);
    s_stoch[b] = md == 1 && !noq;
    if (p.top_p != nullptr && c == 0) {
      const float t = __ldg(p.top_p + b);
      if (!(t > 0.f && t <= 1.f)) atomicOr(p.status, SPADE_DEV_BAD_INDEX);
    }
  }
  block_sync();
  if (p.top_p != nullptr && p.kind == kResident) {
    // (3b) Top-p: the nucleus of every row of a stochastic sequence with
    //      top_p < 1 (see nuc_key).  Per round: every CTA bins its slice of
    //      each listed row and stores the bins to its own slot of the
    //      workspace (plain stores: 152 CTAs adding into the same lines
    //      serialise for hundreds of microseconds); after a grid barrier the
    //      CTA owning a row sums the slots, takes the bin and publishes the
    //      longer key prefix in kReplicas copies; after a second barrier every
    //      CTA reads it.  Bin masses are fixed point (2^31 = all of p, each
    //      term rounded to nearest): integer sums, the same in any order.
    //      Scratch:
    //      the phase-C staging area, idle until then.
    int *s_nl = reinterpret_cast<int *>(f_R);                  // [R] listed rows, ascending
    int *s_npre = s_nl + kMaxR;                                // [R] key prefix of row n (-1: not listed)
    unsigned *s_nab = reinterpret_cast<unsigned *>(s_npre + kMaxR);  // [R] mass above the prefix; at the end, F
    float *s_hp = reinterpret_cast<float *>(s_nab + kMaxR);   // [kEpiWarps][kNucSubs][kNucBins][32] lane-private bins
    if (warp == 0) {
      int base = 0;
      for (int n0 = 0; n0 < p.R; n0 += 32) {
        const int n = n0 + lane;
        const int b = n < p.R ? s_seq[n] : -1;
        const bool want = b >= 0 && s_md[b] == 1 && (p.draft_probs != nullptr || s_nd[b] == 0) &&
                          seq_top_p(p, b) < 1.f &&
                          isfinite(g_m[n]) && g_s[n] > 0.f;
        const unsigned bal = __ballot_sync(0xffffffffu, want);
        if (want) s_nl[base + __popc(bal & ((1u << lane) - 1u))] = n;
        base += __popc(bal);
      }
      if (lane == 0) s_seg[8] = base;
    }
    block_sync();
    const int nl = s_seg[8];
    for (int n = tid; n < kMaxR; n += kThreads) {
      s_npre[n] = -1;
      s_nab[n] = 0u;
    }
    block_sync();
    for (int i = tid; i < nl; i += kThreads) s_npre[s_nl[i]] = 0;
    block_sync();
#pragma unroll 1
    for (int r = 0; nl > 0 && r < kNucRounds; ++r) {
      const int sh = kNucKeyBits - kNucBinBits * (r + 1);  // this round's bin: key bits [sh, sh + 5)
      if (warp >= 2) {
        // Rows in chunks of 32.  Each warp loads its lane quarter of every
        // tile (lane = vocabulary entry, 32 columns in four 8-column loads,
        // the next tile's loads in flight while this one is binned) and
        // transposes it through its shared buffer, so that lane i owns row
        // 32 j + i.  Its bins are fp32 sums kept in kNucSubs copies: value u of
        // a batch goes to copy u % kNucSubs, so the read-add-write of four
        // values never waits on another's write (shared-memory atomics cost
        // tens of cycles per instruction here); each copy's sums follow a
        // fixed order.  Layout bin-major, lane-minor: lane i's words all sit
        // in bank i, so no access conflicts.
        const int ew = warp - 2, q4 = warp & 3;
        const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
        float *T = s_tbuf + ew * (32 * 33);
        float *hp = s_hp + ew * (kNucSubs * kNucBins * 32) + lane;
#pragma unroll 1
        for (int r0 = 0; r0 < p.R; r0 += 32) {
          const int n = r0 + lane;
          const int pre = n < p.R ? s_npre[n] : -1;
          const bool has = pre >= 0;
          if (__ballot_sync(0xffffffffu, has) == 0u) continue;  // the same on every warp
          const int nn = has ? n : r0;
          const float M = g_m[nn];
          const float nb65 = -kNucScale * __fsub_rn(M, kNucSpan);
          const float mlog = -M * kLog2e;
          const float IT = inv_temp(p, has ? s_seq[nn] : -1);
          const int pre_bits = pre + (kNucKeyBias >> (sh + kNucBinBits));  // the range's key prefix, as bits
          const int nc = min(32, p.Rs - r0);  // columns of this chunk (multiple of 8)
#pragma unroll 8
          for (int k = 0; k < kNucSubs * kNucBins; ++k) hp[k * 32] = 0.f;
          uint32_t raw[32];
#pragma unroll
          for (int q = 0; q < 4; ++q)
            if (8 * q < nc) tmem_ld8(tmem + lane_base + static_cast<uint32_t>(r0 + 8 * q), raw + 8 * q);
#pragma unroll 1
          for (int t = 0; t < ntiles; ++t) {
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (i < nc) T[lane * 33 + i] = __uint_as_float(raw[i]);
            if (t + 1 < ntiles) {
              const uint32_t col = tmem + lane_base + static_cast<uint32_t>((t + 1) * p.Rs + r0);
#pragma unroll
              for (int q = 0; q < 4; ++q)
                if (8 * q < nc) tmem_ld8(col + 8 * q, raw + 8 * q);
            }
            __syncwarp();
            const int nv = min(32, v_hi - (v_lo + t * kTileV + q4 * 32));  // valid entries, warp-uniform
            if (has) {
#pragma unroll 1
              for (int j0 = 0; j0 < nv; j0 += 8) {
                float x[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) x[u] = T[(j0 + u) * 33 + lane];
#pragma unroll
                for (int h = 0; h < 8; h += kNucSubs) {
                  float e[kNucSubs];
                  int a[kNucSubs];
#pragma unroll
                  for (int u = 0; u < kNucSubs; ++u) {
                    const float l = __fmul_rn(x[h + u], IT);
                    const int kbits = nuc_key_bits(l, nb65);
                    const bool in = j0 + h + u < nv && (kbits >> (sh + kNucBinBits)) == pre_bits;
                    e[u] = in ? ex2(__fmaf_rn(l, kLog2e, mlog)) : 0.f;
                    a[u] = (u * kNucBins + ((kbits >> sh) & (kNucBins - 1))) * 32;
                  }
                  float v[kNucSubs];
#pragma unroll
                  for (int u = 0; u < kNucSubs; ++u) v[u] = hp[a[u]];
#pragma unroll
                  for (int u = 0; u < kNucSubs; ++u) hp[a[u]] = v[u] + e[u];
                }
              }
            }
            __syncwarp();
          }
          // The four warps' bins of these rows: thread (ew, lane) adds bins
          // [8 ew, 8 ew + 8) of row r0 + lane over the warps and copies (fixed
          // order), converts them to fixed point and stores them to this CTA's slot.
          named_bar(1, kEpiWarps * 32);
          if (has) {
            constexpr int kPer = kNucBins / kEpiWarps;
            const float sc = 0x1p31f / g_s[n];  // fixed point: 2^31 = all of p
            uint4 *dst = reinterpret_cast<uint4 *>(p.nhist + (static_cast<size_t>(n) * p.NC + c) * kNucBins + ew * kPer);
#pragma unroll
            for (int k4 = 0; k4 < kPer; k4 += 4) {
              unsigned tot[4];
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                float f = 0.f;
#pragma unroll
                for (int w4 = 0; w4 < kEpiWarps; ++w4)
#pragma unroll
                  for (int u = 0; u < kNucSubs; ++u)
                    f += s_hp[((w4 * kNucSubs + u) * kNucBins + ew * kPer + k4 + k) * 32 + lane];
                tot[k] = __float2uint_rn(f * sc);
              }
              __stcg(dst + k4 / 4, make_uint4(tot[0], tot[1], tot[2], tot[3]));
            }
          }
          named_bar(1, kEpiWarps * 32);  // the next chunk clears the bins
        }
      }
      if (!grid_barrier(p.bar, p.NC)) {
        atomicOr(p.status, SPADE_DEV_TIMEOUT);
        *s_abort = 1;
      }
      // Owner of listed row i: CTA i % NC.  A slot is kNucBins / 4 16-byte
      // words (four bins each); thread t adds word t % 8 of the slots of CTAs
      // t / 8, t / 8 + 24, ..., all loads in flight.  Warp 0 then holds bins
      // 4 q .. 4 q + 3 in lane q < 8, forms the upper masses C_k (mass of keys
      // at or above bin k, plus the mass above the range) by a suffix scan
      // over the lanes and keeps the highest bin with C_k >= top_p.  Sums stay
      // below 2^32 (all of p is 2^31).
      constexpr int kWps = kNucBins / 4;        // words per slot
      constexpr int kGroups = kThreads / kWps;  // CTA groups
      uint4 *s_red = reinterpret_cast<uint4 *>(s_zw);  // [kGroups][kWps] (phase-C buffer)
#pragma unroll 1
      for (int i = c; i < nl; i += p.NC) {
        const int n = s_nl[i];
        const uint4 *src = reinterpret_cast<const uint4 *>(p.nhist + static_cast<size_t>(n) * p.NC * kNucBins) + tid % kWps;
        uint4 acc4 = make_uint4(0u, 0u, 0u, 0u);
        constexpr int kLoads = (kMaxNC + kGroups - 1) / kGroups;
        uint4 v[kLoads];
#pragma unroll
        for (int j = 0; j < kLoads; ++j) {
          const int k = tid / kWps + j * kGroups;
          v[j] = k < p.NC ? __ldcg(src + static_cast<size_t>(k) * kWps) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int j = 0; j < kLoads; ++j) {
          acc4.x += v[j].x; acc4.y += v[j].y; acc4.z += v[j].z; acc4.w += v[j].w;
        }
        s_red[tid] = acc4;  // = [tid / kWps][tid % kWps]
        block_sync();
        if (warp == 0) {
          unsigned long long bq[4] = {0, 0, 0, 0};
          if (lane < kWps) {
#pragma unroll 4
            for (int g = 0; g < kGroups; ++g) {
              const uint4 t = s_red[g * kWps + lane];
              bq[0] += t.x; bq[1] += t.y; bq[2] += t.z; bq[3] += t.w;
            }
          }

          const unsigned long long tq = bq[0] + bq[1] + bq[2] + bq[3];
          unsigned long long suf = tq;  // inclusive suffix sum over lanes >= this one
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const unsigned long long t = __shfl_down_sync(0xffffffffu, suf, o);
            if (lane + o < 32) suf += t;
          }
          // D[j] = C_{4 lane + j}; D[4] = the mass above this lane's bins.
          unsigned long long D[5];
          D[4] = s_nab[n] + (suf - tq);
#pragma unroll
          for (int j = 3; j >= 0; --j) D[j] = D[j + 1] + bq[j];
          // top_p * 2^31 is exact in fp32; the target is its ceiling.
          const unsigned long long target =
              static_cast<unsigned long long>(ceilf(seq_top_p(p, s_seq[n]) * 0x1p31f));
          const int jj = lane >= kWps ? -1 : D[3] >= target ? 3 : D[2] >= target ? 2 : D[1] >= target ? 1
                                           : D[0] >= target ? 0 : -1;
          const unsigned ge = __ballot_sync(0xffffffffu, jj >= 0);
          const int ls = ge ? 31 - __clz(ge) : 0;  // C_k falls with k: the highest lane with a hit
          unsigned long long ck = D[0], ck1 = D[1];
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (jj == j) { ck = D[j]; ck1 = D[j + 1]; }
          const int kq = __shfl_sync(0xffffffffu, jj < 0 ? 0 : jj, ls);
          ck = __shfl_sync(0xffffffffu, ck, ls);
          ck1 = __shfl_sync(0xffffffffu, ck1, ls);
          if (lane < kReplicas) {
            const int kb = ge ? 4 * ls + kq : 0;
            const uint4 ns = make_uint4(static_cast<unsigned>((s_npre[n] << kNucBinBits) | kb),
                                        static_cast<unsigned>(min(ck1, 0xffffffffull)),
                                        static_cast<unsigned>(min(ck, 0xffffffffull)), 0u);
            __stcg(&p.nstate[static_cast<size_t>(lane) * p.R + n], ns);
          }
        }
        block_sync();  // s_red is free again
      }
      if (!grid_barrier(p.bar, p.NC)) {
        atomicOr(p.status, SPADE_DEV_TIMEOUT);
        *s_abort = 1;
      }
      for (int i = tid; i < nl; i += kThreads) {
        const int n = s_nl[i];
        const uint4 ns = __ldcg(&p.nstate[static_cast<size_t>(c % kReplicas) * p.R + n]);
        s_npre[n] = static_cast<int>(ns.x);
        // The mass above the new prefix's range; after the last round F(tau).
        s_nab[n] = r + 1 < kNucRounds ? ns.y : ns.z;
      }
      block_sync();
    }
    // L_tau = the final prefix followed by zero bits; p on S renormalised by
    // S_nuc = F(tau).  The accept test of a listed draft row is taken again
    // under the nucleus (the merge step took it on all of p).
    for (int i = tid; i < nl; i += kThreads) {
      const int n = s_nl[i];
      const unsigned F = s_nab[n];
      if (F == 0u) continue;  // nothing reached top_p (not expected): all of p
      const float S = g_s[n] * (static_cast<float>(F) * 0x1p-31f);
      const int tkey = s_npre[n] << (kNucKeyBits - kNucBinBits * kNucRounds);
      const float base = __fsub_rn(g_m[n], kNucSpan);
      g_tkey[n] = tkey;
      g_s[n] = S;
      const int b = s_seq[n];
      const int d = s_draft[n];
      if (s_pos[n] < s_nd[b] && d >= 0 && d < p.V) {
        const float ld = __ldcg(&p.ldraft[n]);
        const float pd = nuc_key(ld, base) >= tkey ? expf(ld - g_m[n]) / S : 0.f;
        const float qd = s_qd[n];
        s_ok[n] = (qd > 0.f) ? (s_u[n] < pd / qd) : (pd > 0.f);
      }
    }
    block_sync();
  }
  if (p.kind != kPresampled) {
  // (4) Accepted length = leading accepts; the row that emits the next token.
  for (int b = tid; b < p.B; b += kThreads) {
    const int r0 = s_cuq[b], k = s_nd[b];
    int a = -1;
    if (r0 >= 0 && k >= 0 && s_cuq[b + 1] - r0 == k + 1 && s_cuq[b + 1] <= p.R) {
      a = 0;
      while (a < k && s_ok[r0 + a]) ++a;
    }
    s_acc[b] = a;
    s_rstar[b] = (a >= 0) ? r0 + a : -1;
    if (a < 0) s_stoch[b] = 0;
    if (s_stoch[b]) atomicOr(s_any_stoch, 1);
    // What to sample: the residual against q of draft a (a < k) or p (bonus).
    s_qidx[b] = (a >= 0 && a < k) ? r0 - b + a : -1;
    s_usmp[b] = (a >= 0) ? s_u[r0 + k] : 0.f;
    s_outb[b] = b;
    if (c == 0) {
      p.accepted_len[b] = a < 0 ? 0 : a;
      if (a < 0) p.next_token[b] = -1;
      else if (!s_stoch[b]) p.next_token[b] = g_arg[r0 + a];
    }
  }
  } else {
    // Second pass: row j holds sample j, decided by the first pass.
    const int ns = *p.samp_count;
    for (int j = tid; j < p.B; j += kThreads) {
      s_stoch[j] = j < ns;
      s_rstar[j] = j;
      if (j < ns) {
        const int4 sp = p.samp[j];
        s_qidx[j] = sp.x;
        s_usmp[j] = __int_as_float(sp.y);
        s_outb[j] = sp.z;
      }
    }
    if (tid == 0) *s_any_stoch = ns > 0;
  }
  block_sync();

  // ---- fused KV commit (Algorithm 1 context update) -----------------------
  // The decisions are known: sequence b (b = c, c + NC, ...) keeps slots
  // [0, ctx_b + a_b] and its rejected drafts' slots [ctx_b + a_b + 1, ctx_b +
  // k_b] are cleared; ctx_lens[b] advances by a_b + 1.  Warps 0-1 do it (they
  // are idle in phase C); this step's attention has finished with the cache.
  if (p.kc != nullptr && p.kind != kPresampled && warp < 2) {
    for (int b = c; b < p.B; b += p.NC) {
      const int a = s_acc[b];
      if (a < 0) continue;  // invalid sequence: reported, left untouched
      const int k = s_nd[b];
      const int ctx = p.ctx_lens[b];
      if (ctx < 0 || static_cast<int64_t>(ctx) + k + 1 > p.cap) {
        if (tid == 0) atomicOr(p.status, ctx < 0 ? SPADE_DEV_BAD_INDEX : SPADE_DEV_CAPACITY);
        continue;
      }
      const int lo = ctx + a + 1;
      const int vec = p.Dk / 8;  // 16-byte vectors per slot
      const int per_head = (k - a) * vec;
      const int total = p.Hkv * per_head;
      const uint4 z = make_uint4(0, 0, 0, 0);
      const int32_t *bt = p.block_table ? p.block_table + static_cast<int64_t>(b) * p.max_pages : nullptr;
      if (bt) {
        // Every page the rejected slots use must exist before anything is cleared.
        bool bad_page = false;
        for (int s2 = tid; s2 < k - a; s2 += 64) {
          const int pg = bt[(lo + s2) / p.page_size];
          bad_page |= pg < 0 || pg >= p.num_pages;
        }
        if (bar_or(2, 64, bad_page)) {
          if (tid == 0) atomicOr(p.status, SPADE_DEV_BAD_INDEX);
          continue;
        }
      }
      for (int e = tid; e < total; e += 64) {
        const int h = e / per_head;
        const int r = e - h * per_head;
        size_t off;
        if (bt) {
          const int slot = lo + r / vec;
          off = ((static_cast<size_t>(bt[slot / p.page_size]) * p.Hkv + h) * p.page_size + slot % p.page_size) * vec +
                r % vec;
        } else {
          off = ((static_cast<size_t>(b) * p.Hkv + h) * p.cap + lo) * vec + r;
        }
        p.kc[off] = z;
        p.vc[off] = z;
      }
      named_bar(2, 64);  // every thread has read ctx_lens[b] before it changes
      if (tid == 0) p.ctx_lens[b] = lo;
    }
  }

  if (p.kind == kStatsOnly) {
    // First pass of the two-pass path: publish one sample spec per sequence
    // that needs a draw and gather its hidden row for the second pass.
    if (tid == 0) {
      int ns = 0;
      for (int b = 0; b < p.B; ++b) s_owner[b] = s_stoch[b] ? ns++ : -1;
      s_seg[4] = ns;
    }
    block_sync();
    if (c == 0) {
      for (int b = tid; b < p.B; b += kThreads)
        if (s_owner[b] >= 0)
          p.samp[s_owner[b]] = make_int4(s_qidx[b], __float_as_int(s_usmp[b]), s_outb[b], s_rstar[b]);
      if (tid == 0) *p.samp_count = s_seg[4];
    }
    const int hv = p.H / 8;  // 16-byte vectors per hidden row
    for (int b = 0; b < p.B; ++b) {
      const int j = s_owner[b];
      if (j < 0 || j % p.NC != c) continue;
      const uint4 *src = reinterpret_cast<const uint4 *>(p.hidden + static_cast<size_t>(s_rstar[b]) * p.H);
      uint4 *dst = reinterpret_cast<uint4 *>(p.hidden_s + static_cast<size_t>(j) * p.H);
      for (int e = tid; e < hv; e += kThreads) dst[e] = src[e];
    }
  } else if (*s_any_stoch) {
    // =================== phase C: slice masses of the sampled distribution ==
    // Terms are fp32 (p = 2^((l - m) log2 e) / Z on the SFU, the same formula
    // here and in phase D, so the slice and segment masses agree); every sum is
    // float-float, so the cumulative masses that place u*Z are as exact as the
    // terms allow.  Attempt 0 sums the residual max(0, p - q) (p for a bonus
    // row).  A sequence whose residual has no mass at all falls back to p: a
    // second attempt sums p for those sequences only.  Every CTA reads the
    // same slice masses, so all take the same number of attempts.
    // The sampled sequences, in order (warp 0 compacts them).
    if (warp == 0) {
      int base = 0;
      for (int b0 = 0; b0 < p.B; b0 += 32) {
        const int b = b0 + lane;
        const bool st = b < p.B && s_stoch[b];
        const unsigned m = __ballot_sync(0xffffffffu, st);
        if (st) s_slist[base + __popc(m & ((1u << lane) - 1u))] = b;
        if (b < p.B) {
          s_slpos[b] = st ? base + __popc(m & ((1u << lane) - 1u)) : -1;
          s_usep[b] = 0;
        }
        base += __popc(m);
      }
      if (lane == 0) {
        s_seg[5] = base;
        s_seg[6] = s_seg[7] = 0;  // per attempt: some residual had no mass
      }
    }
    block_sync();
    const int ns = s_seg[5];
    const int slen = v_hi - v_lo;
    const int nseg = (slen + 31) / 32;
    const bool fastc = p.fastc && ns <= kFastSeqs;  // the same on every CTA
#pragma unroll 1  // one copy of the code: the second attempt is rare
    for (int attempt = 0; attempt < 2; ++attempt) {
      if (fastc) {
        // Per group of kFG rows:
        // (a) thread 0 starts bulk copies of the rows' q slices (their 16-byte
        //     aligned interior) and warp 1 loads the ragged ends; both arrive
        //     on q_bar.  Meanwhile the epilogue warps read the rows' logits
        //     from TMEM (lane = vocabulary entry) and form p, then, with q in
        //     shared memory, the residual r = max(0, p - q) (p for a bonus row
        //     or in the fallback attempt), stored per 32-entry segment with a
        //     one-float pad (f_R[row][segment][33]);
        // (b) every thread sums one segment of one row: four chains of
        //     compensated sums (the terms are >= 0, so ordering the two addends
        //     by size makes the error term exact);
        // (c) one warp per row adds its segment masses into the slice mass.
        //     Segment masses stay in shared memory for the in-slice search.
        // q of slice entry e sits at f_Q[row * kQStride + e + qoff], so that
        // the interior's first element lands on a 16-byte boundary.
        const int qoff = v_lo & 3;
        const int va = (v_lo + 3) & ~3, vb = v_hi & ~3;  // bulk-copied interior [va, vb)
        const bool bulk = attempt == 0 && p.qbulk && va < vb;
        const int e_tail = (va > vb ? va : vb) - v_lo;   // first entry after the interior
        for (int g0 = 0; g0 < ns; g0 += kFG) {
          const int ng = min(kFG, ns - g0);
          if (warp == 0) {
            if (lane == 0) {
              int nq = 0;
              for (int gi = 0; bulk && gi < ng; ++gi) nq += s_qidx[s_slist[g0 + gi]] >= 0;
              if (nq > 0) {
                fence_proxy_async_smem();  // earlier generic reads of f_Q come first
                mbar_arrive_expect_tx(q_bar, static_cast<uint32_t>(nq * (vb - va) * 4));
                for (int gi = 0; gi < ng; ++gi) {
                  const int qi = s_qidx[s_slist[g0 + gi]];
                  if (qi < 0) continue;
                  bulk_load(f_Q + gi * kQStride + (va - v_lo + qoff),
                            p.draft_probs + static_cast<size_t>(qi) * p.V + va,
                            static_cast<uint32_t>((vb - va) * 4), q_bar);
                }
              } else {
                mbar_arrive(q_bar);
              }
            }
          } else if (warp == 1) {
            if (attempt == 0) {
              // With bulk copies: at most three entries before va and three
              // after vb; else the whole slice.
              const int gi = lane >> 2, k = lane & 3;
              for (int row = bulk ? gi : 0; row < (bulk ? min(ng, gi + 1) : ng); ++row) {
                const int qi = s_qidx[s_slist[g0 + row]];
                if (qi < 0) continue;
                const float *q = p.draft_probs + static_cast<size_t>(qi) * p.V + v_lo;
                if (bulk) {
                  if (k < va - v_lo && k < slen) f_Q[row * kQStride + k + qoff] = __ldg(q + k);
                  if (e_tail + k < slen) f_Q[row * kQStride + e_tail + k + qoff] = __ldg(q + e_tail + k);
                } else {
                  for (int e = lane; e < slen; e += 32) f_Q[row * kQStride + e + qoff] = __ldg(q + e);
                }
              }
            }
            mbar_arrive(q_bar);  // each lane after its own stores
          } else {
            const int q4 = warp & 3;
            const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
            constexpr int kTiles = kFastSlice / kTileV;
            // Lane gi prepares row gi's parameters (kFG <= 32); each row then
            // broadcasts them.  The loop body has no divergent branch: tiles
            // past the slice re-read its last tile and store zeros.
            int n_l = -1, hq_l = 0;
            float m_l = 0.f, is_l = 0.f, it_l = 1.f;
            int tk_l = INT_MIN;
            if (lane < ng) {
              const int b = s_slist[g0 + lane];
              n_l = (attempt == 0 || s_usep[b]) ? s_rstar[b] : -1;
              hq_l = attempt == 0 && s_qidx[b] >= 0;
              if (n_l >= 0) {
                m_l = g_m[n_l];
                is_l = 1.f / g_s[n_l];
                it_l = inv_temp(p, s_outb[b]);
                tk_l = g_tkey[n_l];
              }
            }
#pragma unroll 1
            for (int gi = 0; gi < ng; ++gi) {
              const int n = __shfl_sync(0xffffffffu, n_l, gi);
              const bool hasq = __shfl_sync(0xffffffffu, hq_l, gi) != 0;
              const float M = __shfl_sync(0xffffffffu, m_l, gi), invS = __shfl_sync(0xffffffffu, is_l, gi);
              const float IT = __shfl_sync(0xffffffffu, it_l, gi);  // 1 / T of the row
              const int TK = __shfl_sync(0xffffffffu, tk_l, gi);  // nucleus key threshold
              const float BASE = __fsub_rn(M, kNucSpan);
              uint32_t raw[kTiles];
              if (n >= 0) {
#pragma unroll
                for (int t = 0; t < kTiles; ++t)
                  tmem_ld1(tmem + lane_base + static_cast<uint32_t>(min(t, ntiles - 1) * p.Rs + n), raw[t]);
                tmem_wait_ld();
              }
              if (gi == 0 && !mbar_wait_unabortable(q_bar, q_phase)) {
                // The copies read valid memory, so this wait does not give up
                // on an earlier expired wait: no copy is left in flight at exit.
                atomicOr(p.status, SPADE_DEV_TIMEOUT);
                *s_abort = 1;
              }
              if (n < 0) continue;
              const float *qs = f_Q + gi * kQStride + qoff;
              float *rrow = f_R + gi * kFastSegs * kSegPad;
              // All q loads before the first store: the compiler cannot tell
              // f_Q and f_R apart, and would otherwise wait on each load in turn.
              float qv[kTiles];
#pragma unroll
              for (int t = 0; t < kTiles; ++t) qv[t] = hasq ? qs[t * kTileV + q4 * 32 + lane] : 0.f;
#pragma unroll
              for (int t = 0; t < kTiles; ++t) {
                const int e = t * kTileV + q4 * 32 + lane;  // < kFastSlice: inside the row's buffers
                const float lv = __fmul_rn(__uint_as_float(raw[t]), IT);
                const bool in = TK == INT_MIN || nuc_key(lv, BASE) >= TK;
                const float pv = in ? ex2((lv - M) * kLog2e) * invS : 0.f;
                const float rv = hasq ? fmaxf(0.f, pv - qv[t]) : pv;
                rrow[(e >> 5) * kSegPad + (e & 31)] = e < slen ? rv : 0.f;
              }
            }
          }
          q_phase ^= 1u;
          block_sync();
          for (int task = tid; task < ng * nseg; task += kThreads) {
            const int gi = task / nseg, sg = task - gi * nseg;
            if (attempt == 1 && !s_usep[s_slist[g0 + gi]]) continue;
            const float *rr = f_R + (gi * kFastSegs + sg) * kSegPad;
            float hi[4] = {0.f, 0.f, 0.f, 0.f}, lo[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
            for (int i = 0; i < 32; ++i) {
              const float x = rr[i];
              const int k = i & 3;
              const float sm = hi[k] + x;
              lo[k] += (fmaxf(hi[k], x) - sm) + fminf(hi[k], x);
              hi[k] = sm;
            }
            const ff2 zs = ff_add(ff_add(ff_norm(hi[0], lo[0]), ff_norm(hi[1], lo[1])),
                                  ff_add(ff_norm(hi[2], lo[2]), ff_norm(hi[3], lo[3])));
            f_seg[(g0 + gi) * kFastSegs + sg] = make_float2(zs.hi, zs.lo);
          }
          block_sync();
        }
        for (int sl = warp; sl < ns; sl += kThreads / 32) {
          const int b = s_slist[sl];
          if (attempt == 1 && !s_usep[b]) continue;
          const float2 t = lane < nseg ? f_seg[sl * kFastSegs + lane] : make_float2(0.f, 0.f);
          const ff2 z = ff_shfl(warp_sum_ff(ff2{t.x, t.y}), 0);  // every copy holds lane 0's sum
          if (lane < kReplicas)
            __stcg(&p.zpart[(static_cast<size_t>(lane) * p.NC + c) * p.B + b], make_float2(z.hi, z.lo));
        }
      } else {
      if (warp >= 2) {
        const int ew = warp - 2, q4 = warp & 3;
        const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
        // Stochastic sequences in groups of kG: the TMEM reads and q loads of a
        // whole group are in flight together.
        constexpr int kG = 4;
        for (int b0 = 0; b0 < p.B;) {
          int bl[kG], nb = 0;
          while (b0 < p.B && nb < kG) {
            if (s_stoch[b0] && (attempt == 0 || s_usep[b0])) bl[nb++] = b0;
            ++b0;
          }
          if (nb == 0) break;
          const float *qrow[kG];
          int nrow[kG];
          float M[kG], invS[kG], IT[kG];
          int TK[kG];
          ff2 z[kG], zp[kG];
  #pragma unroll
          for (int g = 0; g < kG; ++g) {
            const int b = g < nb ? bl[g] : bl[0];
            nrow[g] = s_rstar[b];
            qrow[g] = (attempt == 0 && s_qidx[b] >= 0) ? p.draft_probs + static_cast<size_t>(s_qidx[b]) * p.V : nullptr;
            M[g] = g_m[nrow[g]];
            invS[g] = 1.f / g_s[nrow[g]];
            IT[g] = inv_temp(p, s_outb[b]);
            TK[g] = g_tkey[nrow[g]];
            z[g] = ff2{0.f, 0.f};
            zp[g] = ff2{0.f, 0.f};
          }
          for (int j0 = 0; j0 < ntiles; j0 += 8) {
            const int nj = min(8, ntiles - j0);
            uint32_t raw[kG][8];
            float qv[kG][8];
  #pragma unroll
            for (int g = 0; g < kG; ++g) {
  #pragma unroll
              for (int j = 0; j < 8; ++j)
                if (g < nb && j < nj)
                  tmem_ld1(tmem + lane_base + static_cast<uint32_t>((j0 + j) * p.Rs + nrow[g]), raw[g][j]);
            }
  #pragma unroll
            for (int g = 0; g < kG; ++g) {
  #pragma unroll
              for (int j = 0; j < 8; ++j) {
                const int v = v_lo + (j0 + j) * kTileV + q4 * 32 + lane;
                qv[g][j] = (g < nb && j < nj && qrow[g] && v < v_hi) ? qrow[g][v] : 0.f;
              }
            }
            tmem_wait_ld();
  #pragma unroll
            for (int g = 0; g < kG; ++g) {
  #pragma unroll
              for (int j = 0; j < 8; ++j) {
                const int v = v_lo + (j0 + j) * kTileV + q4 * 32 + lane;
                if (g < nb && j < nj && v < v_hi) {
                  const float lv = __fmul_rn(__uint_as_float(raw[g][j]), IT[g]);
                  const bool in = TK[g] == INT_MIN || nuc_key(lv, __fsub_rn(M[g], kNucSpan)) >= TK[g];
                  const float pv = in ? ex2((lv - M[g]) * kLog2e) * invS[g] : 0.f;
                  zp[g] = ff_add_f(zp[g], pv);
                  z[g] = ff_add_f(z[g], qrow[g] ? fmaxf(0.f, pv - qv[g][j]) : pv);
                }
              }
            }
          }
  #pragma unroll
          for (int g = 0; g < kG; ++g) {
            z[g] = warp_sum_ff(z[g]);
            zp[g] = warp_sum_ff(zp[g]);
            if (lane == 0 && g < nb) s_zw[bl[g] * kEpiWarps + ew] = make_float4(z[g].hi, z[g].lo, zp[g].hi, zp[g].lo);
          }
        }
      }
      block_sync();
      for (int b = tid; b < p.B; b += kThreads) {
        if (!s_stoch[b] || (attempt == 1 && !s_usep[b])) continue;
        ff2 zs{0.f, 0.f}, zps{0.f, 0.f};
        for (int w = 0; w < kEpiWarps; ++w) {
          const float4 t = s_zw[b * kEpiWarps + w];
          zs = ff_add(zs, ff2{t.x, t.y});
          zps = ff_add(zps, ff2{t.z, t.w});
        }
        const ff2 v = attempt == 0 ? zs : zps;
        for (int r = 0; r < kReplicas; ++r)
          __stcg(&p.zpart[(static_cast<size_t>(r) * p.NC + c) * p.B + b], make_float2(v.hi, v.lo));
      }
      }  // register path
      if (!grid_barrier(p.bar, p.NC)) {
        atomicOr(p.status, SPADE_DEV_TIMEOUT);
        *s_abort = 1;
      }
      // =================== phase D: owner slice of u*Z ======================
      // A half warp per sampled sequence (so one pass covers 12 sequences).
      // Lane j of the half holds the masses of the K = ceil(NC/16) slices
      // [j*K, j*K + K) (all loads in flight at once).  A scan of the lane sums
      // gives the total and the lane whose cumulative mass passes u*Z; that
      // lane's K masses are then spread over the half and scanned again, which
      // gives the owner slice (else, rounding past the total, the last slice
      // with mass).  Every CTA reaches the same owner from the same masses.
      constexpr int kZC = kMaxNC / 16;
      const int K = (p.NC + 15) / 16;
      const int half = lane >> 4, j = lane & 15;
      const unsigned hmask = 0xffffu << (16 * half);
      const float2 *zrep = p.zpart + static_cast<size_t>(c % kReplicas) * p.NC * p.B;
#pragma unroll 1
      for (int sl0 = 2 * warp; sl0 < ns; sl0 += 2 * (kThreads / 32)) {
        const int sl = sl0 + half;
        const int b = sl < ns ? s_slist[sl] : -1;
        const bool act = b >= 0 && (attempt == 0 || s_usep[b]);
        float2 zz[kZC];
#pragma unroll
        for (int k = 0; k < kZC; ++k) {
          const int cc = j * K + k;
          zz[k] = (act && k < K && cc < p.NC) ? __ldcg(&zrep[static_cast<size_t>(cc) * p.B + b])
                                              : make_float2(0.f, 0.f);
        }
        float shi = 0.f, slo = 0.f;
#pragma unroll
        for (int k = 0; k < kZC; ++k) {
          const float sm = shi + zz[k].x;
          slo += ((fmaxf(shi, zz[k].x) - sm) + fminf(shi, zz[k].x)) + zz[k].y;
          shi = sm;
        }
        const ff2 mine = ff_norm(shi, slo);
        const ff2 incl = half_scan_ff(mine, j);
        const ff2 tot{__shfl_sync(0xffffffffu, incl.hi, 15, 16), __shfl_sync(0xffffffffu, incl.lo, 15, 16)};
        const bool ok = act && tot.hi > 0.f && isfinite(tot.hi);
        if (act && !ok && j == 0) {
          s_owner[b] = -1;
          if (attempt == 0) {
            s_usep[b] = 1;  // retry on p
            s_seg[6] = 1;
          } else if (c == 0) {
            p.next_token[s_outb[b]] = -1;  // p has no mass either
          }
        }
        const ff2 Tgt = ff_mul_f(tot, ok ? s_usmp[b] : 0.f);
        ff2 before{__shfl_up_sync(0xffffffffu, incl.hi, 1, 16), __shfl_up_sync(0xffffffffu, incl.lo, 1, 16)};
        if (j == 0) before = ff2{0.f, 0.f};
        const unsigned hit = __ballot_sync(0xffffffffu, ok && mine.hi > 0.f && ff_gt(incl, Tgt)) & hmask;
        const unsigned pos = __ballot_sync(0xffffffffu, ok && mine.hi > 0.f) & hmask;
        const int l = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : -1);  // absolute lane
        // Second level: lane l's K slice masses, one per lane of the half.
        const int lsrc = l >= 0 ? (l & 15) : 0;
        float2 zk = make_float2(0.f, 0.f);
#pragma unroll
        for (int k = 0; k < kZC; ++k) {
          const float vx = __shfl_sync(0xffffffffu, zz[k].x, lsrc, 16);
          const float vy = __shfl_sync(0xffffffffu, zz[k].y, lsrc, 16);
          if (j == k) zk = make_float2(vx, vy);
        }
        const ff2 base{__shfl_sync(0xffffffffu, before.hi, lsrc, 16), __shfl_sync(0xffffffffu, before.lo, lsrc, 16)};
        const ff2 z{zk.x, zk.y};
        const ff2 inc2 = half_scan_ff(z, j);
        const ff2 reach = ff_add(base, inc2);
        const bool live = ok && l >= 0 && j < K && z.hi > 0.f;
        const unsigned hit2 = __ballot_sync(0xffffffffu, live && ff_gt(reach, Tgt)) & hmask;
        const unsigned pos2 = __ballot_sync(0xffffffffu, live) & hmask;
        const int l2 = hit2 ? __ffs(hit2) - 1 : (pos2 ? 31 - __clz(pos2) : -1);
        if (ok && l2 < 0 && j == 0) s_owner[b] = -1;  // no slice with mass (not reached: tot > 0)
        if (lane == l2) {
          if (attempt == 1 && c == 0) atomicOr(p.status, SPADE_DEV_FALLBACK);
          s_owner[b] = (l & 15) * K + j;
          const ff2 t = ff_sub(Tgt, ff_add(base, ff_sub(inc2, z)));  // target left inside the slice
          s_T[b] = make_float2(t.hi, t.lo);
        }
      }
      block_sync();
      if (s_seg[6 + attempt] == 0) break;  // a flag per attempt: no reset races the reads
    }
    block_sync();
    if (warp >= 2) {
      const int ew = warp - 2, q4 = warp & 3;
      const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
      for (int b = 0; b < p.B; ++b) {
        if (!s_stoch[b] || s_owner[b] != c) continue;
        const int n = s_rstar[b];
        const bool usep = s_usep[b] != 0;
        const float *qrow = (s_qidx[b] >= 0 && !usep) ? p.draft_probs + static_cast<size_t>(s_qidx[b]) * p.V : nullptr;
        const float M = g_m[n], invS = 1.f / g_s[n];
        const float IT = inv_temp(p, s_outb[b]);  // 1 / T of the row
        const int TK = g_tkey[n];                  // nucleus key threshold (INT_MIN: all of p)
        const float BASE = __fsub_rn(M, kNucSpan);
        // (1) mass of every 32-entry segment (tile j, lane quarter q4) of the slice:
        //     from phase C's shared-memory sums, else recomputed.
        if (fastc) {
          if (ew == 0) {
            const int sl = s_slpos[b];
            for (int sg = lane; sg < ntiles * kEpiWarps; sg += 32) {
              s_tw[sg] = sg < nseg ? f_seg[sl * kFastSegs + sg] : make_float2(0.f, 0.f);
            }
          }
        } else
        for (int j0 = 0; j0 < ntiles; j0 += 8) {
          const int nj = min(8, ntiles - j0);
          uint32_t raw[8];
          float qv[8];
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (j < nj) tmem_ld1(tmem + lane_base + static_cast<uint32_t>((j0 + j) * p.Rs + n), raw[j]);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int v = v_lo + (j0 + j) * kTileV + q4 * 32 + lane;
            qv[j] = (j < nj && qrow && v < v_hi) ? qrow[v] : 0.f;
          }
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int v = v_lo + (j0 + j) * kTileV + q4 * 32 + lane;
            float rv = 0.f;
            if (j < nj && v < v_hi) {
              const float lv = __fmul_rn(__uint_as_float(raw[j]), IT);
              const bool in = TK == INT_MIN || nuc_key(lv, BASE) >= TK;
              const float pv = in ? ex2((lv - M) * kLog2e) * invS : 0.f;
              rv = qrow ? fmaxf(0.f, pv - qv[j]) : pv;
            }
            const ff2 seg = warp_sum_ff(ff2{rv, 0.f});
            if (lane == 0 && j < nj) s_tw[(j0 + j) * kEpiWarps + q4] = make_float2(seg.hi, seg.lo);
          }
        }
        named_bar(1, kEpiWarps * 32);
        // (2) the segment holding the target, in vocabulary order.
        if (ew == 0 && lane == 0) {
          ff2 run{0.f, 0.f};
          const ff2 tgt0{s_T[b].x, s_T[b].y};
          ff2 tgt = tgt0;
          int jt = -1, qt = -1, jl = -1, ql = -1;
          for (int j = 0; j < ntiles && jt < 0; ++j) {
            for (int q = 0; q < kEpiWarps; ++q) {
              const ff2 mseg{s_tw[j * kEpiWarps + q].x, s_tw[j * kEpiWarps + q].y};
              if (mseg.hi > 0.f) { jl = j; ql = q; }
              const ff2 reach = ff_add(run, mseg);
              if (mseg.hi > 0.f && ff_gt(reach, tgt0)) { jt = j; qt = q; tgt = ff_sub(tgt0, run); break; }
              run = reach;
            }
          }
          if (jt < 0) { jt = jl; qt = ql; tgt = ff2{INFINITY, 0.f}; }  // rounding: clamp to the last mass
          s_seg[0] = jt;
          s_seg[1] = qt;
          s_T[b] = make_float2(tgt.hi, tgt.lo);
        }
        named_bar(1, kEpiWarps * 32);
        // (3) the warp owning that segment scans its 32 entries.
        const int jt = s_seg[0], qt = s_seg[1];
        if (jt >= 0 && q4 == qt) {
          uint32_t raw;
          tmem_ld1(tmem + lane_base + static_cast<uint32_t>(jt * p.Rs + n), raw);
          const int v = v_lo + jt * kTileV + q4 * 32 + lane;
          const float qv = (qrow && v < v_hi) ? qrow[v] : 0.f;
          tmem_wait_ld();
          float rv = 0.f;
          if (v < v_hi) {
            const float lv = __fmul_rn(__uint_as_float(raw), IT);
            const bool in = TK == INT_MIN || nuc_key(lv, BASE) >= TK;
            const float pv = in ? ex2((lv - M) * kLog2e) * invS : 0.f;
            rv = qrow ? fmaxf(0.f, pv - qv) : pv;
          }
          const ff2 incl = warp_scan_ff(ff2{rv, 0.f}, lane);
          const ff2 tgt{s_T[b].x, s_T[b].y};
          const unsigned hit = __ballot_sync(0xffffffffu, rv > 0.f && ff_gt(incl, tgt));
          const unsigned pos = __ballot_sync(0xffffffffu, rv > 0.f);
          if (lane == 0) {
            const int l = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
            p.next_token[s_outb[b]] = v + l;
          }
        } else if (jt < 0 && ew == 0 && lane == 0) {
          p.next_token[s_outb[b]] = -1;
        }
        named_bar(1, kEpiWarps * 32);
      }
    }
  }

  // ---- teardown: every TMEM access above has completed --------------------
  tc_fence_before();
  block_sync();
  if (warp == 1) {
    // No MMA may still write TMEM when it is released (matters only after an
    // expired wait; otherwise the epilogue already consumed the last round).
    if (lane == 0 && rounds_issued > 0) mbar_wait_unabortable(acc_full, (rounds_issued - 1) & 1);
    if constexpr (PAIR) {
      // Pair mode: the allocation is released by both CTAs together, once
      // both are done with it (bounded handshake on each other's `fin`).
      if (lane == 0) {
        mbar_arrive_cluster(cluster_map(fin, rank ^ 1u));
        const uint64_t t0 = globaltimer();
        uint32_t ok = 0;
        while (!ok) {
          asm volatile(
              "{\n\t.reg .pred p;\n\t"
              "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], 0;\n\t"
              "selp.b32 %0, 1, 0, p;\n\t}"
              : "=r"(ok)
              : "r"(smem_u32(fin))
              : "memory");
          if (!ok && globaltimer() - t0 > kWaitLimitNs) {
            atomicOr(p.status, SPADE_DEV_TIMEOUT);
            break;
          }
        }
      }
      __syncwarp();
      tc_fence_after();
      tmem_dealloc_pair(tmem, p.tmem_cols);
    } else {
      __syncwarp();
      tc_fence_after();
      tmem_dealloc(tmem, p.tmem_cols);
    }
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
  if (pl.NC > kMaxNC) pl.NC = kMaxNC;
  pl.Ncols = (R + 15) / 16 * 16;
  pl.Rs = (R + 7) / 8 * 8;
  return pl;
}

// Slices are V/NC rows (floor or ceil); returns the tiles of the longest slice
// and the box rows (multiple of 8, < 128) that cover every partial last tile,
// or 128 when no slice ends in a tile short enough to be worth a short box.
static void slice_shape(int V, int NC, int *tiles_max, int *brs) {
  const int lmin = V / NC, lmax = lmin + (V % NC ? 1 : 0);
  *tiles_max = (lmax + kTileV - 1) / kTileV;
  int last = 0;
  for (int L : {lmin, lmax}) {
    const int rows = L - ((L + kTileV - 1) / kTileV - 1) * kTileV;
    if (rows < kTileV && rows > last) last = rows;
  }
  *brs = last == 0 ? kTileV : (last + 7) / 8 * 8;
}

// Scratch of one launch: slice partials, draft logits, merged statistics, slice masses.
struct WsRegion {
  size_t pstat, ldraft, gstat, zpart, nhist, nstate, end;
};
static WsRegion ws_region(size_t off, int B, int R, int NC) {
  WsRegion w;
  w.pstat = off;
  off += round_up(static_cast<size_t>(NC) * R * 16, 256);
  w.ldraft = off;
  off += round_up(static_cast<size_t>(R) * 4, 256);
  w.gstat = off;
  off += round_up(static_cast<size_t>(kReplicas) * R * 16, 256);
  w.zpart = off;
  off += round_up(static_cast<size_t>(kReplicas) * NC * B * 8, 256);
  w.nhist = off;
  off += round_up(static_cast<size_t>(R) * NC * kNucBins * 4, 256);
  w.nstate = off;
  off += round_up(static_cast<size_t>(kReplicas) * R * 16, 256);
  w.end = off;
  return w;
}

// Whole workspace.  One launch: [barrier words][region].  Two passes:
// [barrier words][pass-1 region][sample specs][count][gathered hidden][pass-2 region].
struct WsLayout {
  bool two_pass;
  WsRegion r1, r2;
  size_t samp, count, hidden_s, end;
};

static bool resident_fits(int R, int V, int NC) {
  if (R > kMaxRes) return false;
  int tiles = 0, brs = 0, rt[kMaxRounds], nr = 0;
  slice_shape(V, NC, &tiles, &brs);
  const Plan pl = make_plan(R, V, NC);
  return tiles <= kMaxTilesPerCta && plan_rounds(tiles, pl.Ncols, pl.Rs, rt, &nr);
}

static WsLayout ws_layout(int B, int R, int H, int V, int sms) {
  WsLayout L{};
  const int NC = make_plan(R, V, sms).NC;
  L.two_pass = !resident_fits(R, V, NC);
  L.r1 = ws_region(kBarBytes, B, R, NC);
  if (!L.two_pass) {
    L.end = L.r1.end;
    return L;
  }
  size_t off = L.r1.end;
  L.samp = off;
  off += round_up(static_cast<size_t>(B) * 16, 256);
  L.count = off;
  off += 256;
  L.hidden_s = off;
  off += round_up(static_cast<size_t>(B) * H * 2, 256);
  L.r2 = ws_region(off, B, B, NC);
  L.end = L.r2.end;
  return L;
}

// 3-D view of a row-major [rows, H] bf16 matrix: dims {64, rows, H/64},
// strides {H*2, 128} bytes, box {64, box_rows, kg}; lands as [kg][box_rows][64]
// with the 128-byte swizzle, i.e. kg canonical K-major tiles back to back.
static bool encode_kslab_view(CUtensorMap *map, const void *base, int rows, int H, int box_rows,
                              int kg) {
  using EncodeFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
  static EncodeFn fn = nullptr;
  if (!fn) {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      fail(SPADE_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
      return false;
    }
    fn = reinterpret_cast<EncodeFn>(f);
  }
  cuuint64_t dims[3] = {64, static_cast<cuuint64_t>(rows), static_cast<cuuint64_t>(H / 64)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(H) * 2, 128};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), static_cast<cuuint32_t>(kg)};
  cuuint32_t es[3] = {1, 1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    fail(SPADE_ERR_CUDA, "cuTensorMapEncodeTiled (k-slab view) failed (%d)", static_cast<int>(r));
    return false;
  }
  return true;
}

struct Maps {
  CUtensorMap w3, w2, w2s, w3s, h3, h2;
};

// Fills the plan-dependent fields of `p` for a launch of kind `kind` over the
// rows of `hidden` ([R, H]) and encodes its tensor maps.
static spade_status prepare(Params &p, int kind, const void *hidden, const void *w_lm, int R,
                            int sms, Maps &m) {
  const Plan pl = make_plan(R, p.V, sms);
  p.kind = kind;
  p.R = R;
  p.T = pl.T;
  p.NC = pl.NC;
  p.Ncols = pl.Ncols;
  p.Rs = pl.Rs;
  p.KC = (p.H + kKChunk - 1) / kKChunk;
  p.KCF = p.H / kKChunk;
  int tiles_max = 0;
  slice_shape(p.V, pl.NC, &tiles_max, &p.BRS);
  if (tiles_max > kMaxTilesPerCta)
    return fail(SPADE_ERR_SHAPE, "vocabulary %d needs %d tiles per SM (max %d)", p.V, tiles_max,
                kMaxTilesPerCta);
  p.tmem_cols = kTmemCols;
  p.pair = 0;
  if (kind == kStatsOnly) {
    // One tile per round in one accumulator slot; rows beyond 256 take a
    // second MMA N-chunk.  Hidden rows arrive in <= 256-row boxes.
    if (pl.Ncols > kTmemCols) return fail(SPADE_ERR_SHAPE, "R = %d rows exceed %d", R, kTmemCols);
    p.nchunks = pl.Ncols > 256 ? 2 : 1;
    p.n0w = p.nchunks == 2 ? ((pl.Ncols / 2 + 15) / 16 * 16) : pl.Ncols;
    p.KG = 1;
    if (pl.NC % 2 == 0) {
      // CTA pairs: M = 256 MMAs (cta_group::2) over 256-row pair tiles, each
      // CTA holding half of every N-chunk's hidden rows, so an SM receives
      // 128 W rows + Ncols / 2 hidden rows per k-chunk instead of
      // 128 + Ncols: the statistics pass is bound by those bytes in flight.
      p.pair = 1;
      const int NP = pl.NC / 2;
      const int lmax = (p.V + NP - 1) / NP;
      tiles_max = (lmax + 2 * kTileV - 1) / (2 * kTileV);
      p.idesc = idesc_bf16_f32(2 * kTileV, p.n0w);
      p.idesc1 = idesc_bf16_f32(2 * kTileV, p.nchunks == 2 ? pl.Ncols - p.n0w : 16);
      p.h_boxes = p.nchunks;
      p.h_box_rows = p.n0w / 2;
      p.HS = 4;
    } else {
      p.idesc = idesc_bf16_f32(kTileV, p.n0w);
      p.idesc1 = idesc_bf16_f32(kTileV, p.nchunks == 2 ? pl.Ncols - p.n0w : 16);
      p.h_boxes = p.nchunks;
      p.h_box_rows = p.nchunks == 2 ? 256 : pl.Ncols;
      p.HS = 2;
    }
    p.nrounds = tiles_max;
    for (int r = 0; r < tiles_max; ++r) p.round_tiles[r] = 1;
  } else {
    if (!plan_rounds(tiles_max, pl.Ncols, pl.Rs, p.round_tiles, &p.nrounds))
      return fail(SPADE_ERR_SHAPE,
                  "logits of %d rows x %d vocab do not fit on chip (%d tiles per SM, %d TMEM columns each)",
                  R, p.V, tiles_max, pl.Rs);
    p.nchunks = 1;
    p.n0w = pl.Ncols;
    p.idesc = idesc_bf16_f32(kTileV, pl.Ncols);
    p.idesc1 = p.idesc;
    p.h_boxes = 1;
    p.h_box_rows = pl.Ncols;
    p.HS = 3;
    p.KG = 2;  // two k-chunks per stage (32 KB W boxes) while the rings fit
  }
  for (;;) {
    Params probe = p;
    probe.WS = 0;
    const int fixed = smem_layout(probe).total;
    p.WS = (kSmemBudget - fixed) / (p.KG * kWChunkBytes);
    if (p.WS > 8) p.WS = 8;
    if (p.WS >= 4 || p.KG == 1) break;
    p.KG = 1;
  }
  if (p.WS < 2) return fail(SPADE_ERR_SHAPE, "shared memory too small for R = %d", R);
  // Bytes of the W ring that phases B-D use (the per-row / per-sequence
  // arrays, then the staging buffers and segment masses of phase C, which
  // the nucleus search uses before phase C).
  constexpr size_t kPhaseBBytes = 4 * kMaxR * 4 + 8 * kMaxB * 4 + 16 * 4 + kMaxB * 8 +
                                  kMaxB * kEpiWarps * 16 + kMaxTilesPerCta * kEpiWarps * 8 +
                                  2 * kMaxB * 4 + kMaxR * 4;
  constexpr size_t kFastBytes = kPhaseBBytes + kFG * (kFastSegs * kSegPad + kQStride) * 4 +
                                kFastSeqs * kFastSegs * 8;
  constexpr size_t kNucBytes = kPhaseBBytes + kMaxR * 12 + kEpiWarps * kNucSubs * kNucBins * 32 * 4;  // phase B (3b)
  const size_t ring = static_cast<size_t>(p.WS) * p.KG * kWChunkBytes;
  if (ring < kPhaseBBytes) return fail(SPADE_ERR_SHAPE, "shared memory too small for R = %d", R);
  // After phase A the W and hidden rings (contiguous) are free.
  const size_t freeb = static_cast<size_t>(smem_layout(p).off_bar);
  p.fastc = freeb >= kFastBytes && (p.V + p.NC - 1) / p.NC <= kFastSlice;
  if (p.top_p != nullptr && freeb < kNucBytes)
    return fail(SPADE_ERR_SHAPE, "shared memory too small for the top-p search at R = %d", R);
  p.NS = (p.KC + p.KG - 1) / p.KG;
  if (smem_layout(p).total > kSmemMax) return fail(SPADE_ERR_SHAPE, "shared memory plan too large");

  // 2-D views (one k-chunk per box, zero fill past H) serve a ragged last
  // k-chunk and row boxes of the first pass; 3-D views fetch KG full k-chunks.
  const uint64_t pitch = static_cast<uint64_t>(p.H) * 2;
  if (!encode_tmap_bf16_sw128(&m.w2, w_lm, p.H, p.V, pitch, kKChunk, kTileV) ||
      !encode_tmap_bf16_sw128(&m.w2s, w_lm, p.H, p.V, pitch, kKChunk, p.BRS) ||
      !encode_tmap_bf16_sw128(&m.h2, hidden, p.H, R, pitch, kKChunk, p.h_box_rows))
    return SPADE_ERR_CUDA;
  if (p.KCF >= 1) {
    if (!encode_kslab_view(&m.w3, w_lm, p.V, p.H, kTileV, p.KG) ||
        !encode_kslab_view(&m.w3s, w_lm, p.V, p.H, p.BRS, p.KG) ||
        !encode_kslab_view(&m.h3, hidden, R, p.H, pl.Ncols < 256 ? pl.Ncols : 256, p.KG))
      return SPADE_ERR_CUDA;
  } else {
    m.w3 = m.w2;  // never used: every stage takes the 2-D path
    m.w3s = m.w2s;
    m.h3 = m.h2;
  }
  return SPADE_OK;
}

static spade_status launch(const Params &p, const Maps &m, cudaStream_t stream) {
  static bool configured = false;
  if (!configured) {
    for (auto kern : {verify_accept_kernel<false>, verify_accept_kernel<true>}) {
      cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMax);
      if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute(verify_accept)");
    }
    configured = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.NC);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem_layout(p).total;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;  // pair mode: CTAs 2j, 2j+1 share a cluster
  attr[1].val.clusterDim.x = 2;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.pair ? 2 : 1;
  const cudaError_t e = p.pair ? cudaLaunchKernelEx(&cfg, verify_accept_kernel<true>, p, m.w3, m.w2, m.w2s, m.w3s, m.h3, m.h2)
                               : cudaLaunchKernelEx(&cfg, verify_accept_kernel<false>, p, m.w3, m.w2, m.w2s, m.w3s, m.h3, m.h2);
  if (e != cudaSuccess) return cuda_fail(e, "verify_accept cooperative launch");
  return SPADE_OK;
}

static void set_region(Params &p, uint8_t *ws, const WsRegion &r) {
  p.pstat = reinterpret_cast<float4 *>(ws + r.pstat);
  p.ldraft = reinterpret_cast<float *>(ws + r.ldraft);
  p.gstat = reinterpret_cast<float4 *>(ws + r.gstat);
  p.zpart = reinterpret_cast<float2 *>(ws + r.zpart);
  p.nhist = reinterpret_cast<unsigned *>(ws + r.nhist);
  p.nstate = reinterpret_cast<uint4 *>(ws + r.nstate);
}

}  // namespace accept
}  // namespace spade

using namespace spade;

extern "C" int32_t spade_accept_launches(int32_t B, int32_t R, int32_t H, int32_t V) {
  if (B <= 0 || R < B || H <= 0 || V <= 0) return 0;
  int sms = 0;
  if (device_info(&sms, nullptr) != SPADE_OK) return 0;
  return accept::ws_layout(B, R, H, V, sms).two_pass ? 2 : 1;
}

extern "C" size_t spade_accept_workspace_size(int32_t B, int32_t R, int32_t H, int32_t V) {
  if (B <= 0 || R < B || H <= 0 || V <= 0) return 0;
  int sms = 0;
  if (device_info(&sms, nullptr) != SPADE_OK) return 0;
  return accept::ws_layout(B, R, H, V, sms).end;
}

extern "C" spade_status spade_accept_stats_layout(int32_t B, int32_t R, int32_t H, int32_t V,
                                                  size_t *row_stats_offset, size_t *draft_logit_offset,
                                                  int32_t *replica_stride) {
  if (!row_stats_offset || !draft_logit_offset || !replica_stride)
    return fail(SPADE_ERR_INVALID_ARG, "spade_accept_stats_layout: null output pointer");
  if (B <= 0 || R < B || H <= 0 || V <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_accept_stats_layout: bad sizes B=%d R=%d H=%d V=%d", B, R, H, V);
  int sms = 0;
  const spade_status st = device_info(&sms, nullptr);
  if (st != SPADE_OK) return st;
  // The statistics of every row are those of the first launch (the resident
  // pass, or the statistics pass of a two-pass shape).
  const accept::WsLayout L = accept::ws_layout(B, R, H, V, sms);
  *row_stats_offset = L.r1.gstat;
  *draft_logit_offset = L.r1.ldraft;
  *replica_stride = R;
  return SPADE_OK;
}

namespace spade {
namespace accept {
struct CommitArgs {
  void *k_cache, *v_cache;
  int32_t *ctx_lens;
  int Hkv, D, cap;
  const int32_t *block_table;  // paged pools when non-null
  int page_size, max_pages, num_pages;
};
static spade_status verify_accept_impl(const void *hidden, const void *w_lm,
                                       const int32_t *draft_tokens, const float *draft_probs,
                                       const float *uniforms, const int32_t *mode,
                                       const int32_t *cu_q, const int32_t *n_draft,
                                       int32_t *accepted_len, int32_t *next_token, int32_t B,
                                       int32_t R, int32_t H, int32_t V, void *workspace,
                                       size_t workspace_bytes, int32_t *status,
                                       spade_stream_t stream, const CommitArgs *cm,
                                       const float *temperature = nullptr,
                                       const float *top_p = nullptr) {
  using namespace accept;
  if (!hidden || !w_lm || !uniforms || !mode || !cu_q || !n_draft || !accepted_len ||
      !next_token || !status || (R > B && !draft_tokens))
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept: null pointer argument");
  if (B <= 0 || R < B || H <= 0 || V <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept: bad sizes B=%d R=%d H=%d V=%d", B, R, H, V);
  if (H % 8) return fail(SPADE_ERR_SHAPE, "hidden size %d must be a multiple of 8", H);
  if (R > kMaxR) return fail(SPADE_ERR_SHAPE, "R = %d verify rows exceed %d per call", R, kMaxR);
  if (B > kMaxB) return fail(SPADE_ERR_SHAPE, "B = %d sequences exceed %d per call", B, kMaxB);
  if (!aligned(hidden, 16) || !aligned(w_lm, 16))
    return fail(SPADE_ERR_INVALID_ARG, "hidden and w_lm must be 16-byte aligned");
  int sms = 0;
  spade_status st = device_info(&sms, nullptr);
  if (st != SPADE_OK) return st;

  const WsLayout L = ws_layout(B, R, H, V, sms);
  if (top_p && L.two_pass)
    return fail(SPADE_ERR_SHAPE, "top-p needs the logits resident: R = %d rows x V = %d exceed one launch", R, V);
  if (!workspace || workspace_bytes < L.end || !aligned(workspace, 256))
    return fail(SPADE_ERR_WORKSPACE, "accept workspace needs %zu bytes, 256-byte aligned (got %zu)",
                L.end, workspace_bytes);
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

  Params p{};
  p.draft_tokens = draft_tokens;
  p.draft_probs = draft_probs;
  p.temperature = temperature;
  p.top_p = top_p;
  p.qbulk = draft_probs != nullptr && aligned(draft_probs, 16) && V % 4 == 0;
  p.uniforms = uniforms;
  p.mode = mode;
  p.cu_q = cu_q;
  p.n_draft = n_draft;
  p.accepted_len = accepted_len;
  p.next_token = next_token;
  p.status = status;
  p.B = B;
  p.H = H;
  p.V = V;
  p.hidden = static_cast<const __nv_bfloat16 *>(hidden);
  p.bar = reinterpret_cast<unsigned *>(ws);
  if (cm) {
    p.kc = static_cast<uint4 *>(cm->k_cache);
    p.vc = static_cast<uint4 *>(cm->v_cache);
    p.ctx_lens = cm->ctx_lens;
    p.Hkv = cm->Hkv;
    p.Dk = cm->D;
    p.cap = cm->cap;
    p.block_table = cm->block_table;
    p.page_size = cm->page_size;
    p.max_pages = cm->max_pages;
    p.num_pages = cm->num_pages;
  }
  set_region(p, ws, L.r1);
  Maps m;
  if (!L.two_pass) {
    st = prepare(p, kResident, hidden, w_lm, R, sms, m);
    if (st != SPADE_OK) return st;
    return launch(p, m, s);
  }
  // More rows than TMEM holds: a statistics-and-decisions pass over all rows,
  // then a resident pass over the gathered rows that need a draw.
  p.samp = reinterpret_cast<int4 *>(ws + L.samp);
  p.samp_count = reinterpret_cast<int *>(ws + L.count);
  p.hidden_s = reinterpret_cast<__nv_bfloat16 *>(ws + L.hidden_s);
  st = prepare(p, kStatsOnly, hidden, w_lm, R, sms, m);
  if (st != SPADE_OK) return st;
  st = launch(p, m, s);
  if (st != SPADE_OK) return st;
  Params p2 = p;
  p2.kc = p2.vc = nullptr;  // the first pass committed
  set_region(p2, ws, L.r2);
  st = prepare(p2, kPresampled, p.hidden_s, w_lm, B, sms, m);
  if (st != SPADE_OK) return st;
  return launch(p2, m, s);
}
}  // namespace accept
}  // namespace spade

extern "C" spade_status spade_verify_accept(const void *hidden, const void *w_lm,
                                            const int32_t *draft_tokens, const float *draft_probs,
                                            const float *uniforms, const int32_t *mode,
                                            const int32_t *cu_q, const int32_t *n_draft,
                                            int32_t *accepted_len, int32_t *next_token, int32_t B,
                                            int32_t R, int32_t H, int32_t V, void *workspace,
                                            size_t workspace_bytes, int32_t *status,
                                            spade_stream_t stream) {
  return accept::verify_accept_impl(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q,
                                    n_draft, accepted_len, next_token, B, R, H, V, workspace,
                                    workspace_bytes, status, stream, nullptr);
}

extern "C" spade_status spade_verify_accept_commit(
    const void *hidden, const void *w_lm, const int32_t *draft_tokens, const float *draft_probs,
    const float *uniforms, const int32_t *mode, const int32_t *cu_q, const int32_t *n_draft,
    int32_t *accepted_len, int32_t *next_token, void *k_cache, void *v_cache, int32_t *ctx_lens,
    int32_t B, int32_t R, int32_t H, int32_t V, int32_t Hkv, int32_t D, int32_t cap,
    void *workspace, size_t workspace_bytes, int32_t *status, spade_stream_t stream) {
  if (!k_cache || !v_cache || !ctx_lens)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_commit: null cache or ctx_lens pointer");
  if (Hkv <= 0 || D <= 0 || cap <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_commit: non-positive cache size");
  if (D % 8) return fail(SPADE_ERR_SHAPE, "spade_verify_accept_commit: D = %d must be a multiple of 8", D);
  if (!aligned(k_cache, 16) || !aligned(v_cache, 16))
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_commit: caches must be 16-byte aligned");
  const accept::CommitArgs cm{k_cache, v_cache, ctx_lens, Hkv, D, cap, nullptr, 0, 0, 0};
  return accept::verify_accept_impl(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q,
                                    n_draft, accepted_len, next_token, B, R, H, V, workspace,
                                    workspace_bytes, status, stream, &cm);
}

extern "C" spade_status spade_verify_accept_commit_paged(
    const void *hidden, const void *w_lm, const int32_t *draft_tokens, const float *draft_probs,
    const float *uniforms, const int32_t *mode, const int32_t *cu_q, const int32_t *n_draft,
    int32_t *accepted_len, int32_t *next_token, void *k_pool, void *v_pool, const int32_t *block_table,
    int32_t *ctx_lens, int32_t B, int32_t R, int32_t H, int32_t V, int32_t Hkv, int32_t D, int32_t page_size,
    int32_t num_pages, int32_t max_pages, void *workspace, size_t workspace_bytes, int32_t *status,
    spade_stream_t stream) {
  if (!k_pool || !v_pool || !block_table || !ctx_lens)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_commit_paged: null pool, table or ctx_lens pointer");
  if (Hkv <= 0 || D <= 0 || page_size <= 0 || num_pages <= 0 || max_pages <= 0)
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_commit_paged: non-positive size");
  if (D % 8) return fail(SPADE_ERR_SHAPE, "spade_verify_accept_commit_paged: D = %d must be a multiple of 8", D);
  if (static_cast<int64_t>(max_pages) * page_size >= (int64_t(1) << 31))
    return fail(SPADE_ERR_CAPACITY, "max_pages * page_size exceeds 2^31");
  if (!aligned(k_pool, 16) || !aligned(v_pool, 16))
    return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_commit_paged: pools must be 16-byte aligned");
  const accept::CommitArgs cm{k_pool, v_pool, ctx_lens, Hkv, D, max_pages * page_size, block_table,
                              page_size, max_pages, num_pages};
  return accept::verify_accept_impl(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q,
                                    n_draft, accepted_len, next_token, B, R, H, V, workspace,
                                    workspace_bytes, status, stream, &cm);
}

extern "C" spade_status spade_verify_accept_temperature(
    const void *hidden, const void *w_lm, const int32_t *draft_tokens, const float *draft_probs,
    const float *uniforms, const int32_t *mode, const float *temperature, const int32_t *cu_q,
    const int32_t *n_draft, int32_t *accepted_len, int32_t *next_token, int32_t B, int32_t R, int32_t H,
    int32_t V, void *workspace, size_t workspace_bytes, int32_t *status, spade_stream_t stream) {
  if (!temperature) return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_temperature: null temperature");
  return accept::verify_accept_impl(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q, n_draft,
                                    accepted_len, next_token, B, R, H, V, workspace, workspace_bytes, status,
                                    stream, nullptr, temperature);
}

extern "C" spade_status spade_verify_accept_sampling(
    const void *hidden, const void *w_lm, const int32_t *draft_tokens, const float *draft_probs,
    const float *uniforms, const int32_t *mode, const float *temperature, const float *top_p,
    const int32_t *cu_q, const int32_t *n_draft, int32_t *accepted_len, int32_t *next_token, void *k_cache,
    void *v_cache, int32_t *ctx_lens, int32_t B, int32_t R, int32_t H, int32_t V, int32_t Hkv, int32_t D,
    int32_t cap, void *workspace, size_t workspace_bytes, int32_t *status, spade_stream_t stream) {
  const bool commit = k_cache || v_cache || ctx_lens;
  if (commit) {
    if (!k_cache || !v_cache || !ctx_lens)
      return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_sampling: give all of k_cache, v_cache, ctx_lens or none");
    if (Hkv <= 0 || D <= 0 || cap <= 0)
      return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_sampling: non-positive cache size");
    if (D % 8) return fail(SPADE_ERR_SHAPE, "spade_verify_accept_sampling: D = %d must be a multiple of 8", D);
    if (!aligned(k_cache, 16) || !aligned(v_cache, 16))
      return fail(SPADE_ERR_INVALID_ARG, "spade_verify_accept_sampling: caches must be 16-byte aligned");
  }
  const accept::CommitArgs cm{k_cache, v_cache, ctx_lens, Hkv, D, cap, nullptr, 0, 0, 0};
  return accept::verify_accept_impl(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q, n_draft,
                                    accepted_len, next_token, B, R, H, V, workspace, workspace_bytes, status,
                                    stream, commit ? &cm : nullptr, temperature, top_p);
}
