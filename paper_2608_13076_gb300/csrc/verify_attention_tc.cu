// verify_attention_tc.cu -- verify attention for head dims 64 and 128 on the
// fifth-generation tensor cores (tcgen05 MMAs with accumulators in tensor
// memory): the attention of the k_b+1 verify positions of every sequence
// against its cached keys and values, causal inside the draft block
// (Sec. III-B "Verification Stage", Algorithm 1 cloud step).
//
// Design (GB300):
//  * Keys on the MMA M side.  A unit (sequence, KV head, <= 64 query rows) has
//    few query rows (G * (k+1), e.g. 36) but thousands of keys, so the scores
//    are computed transposed: S^T[key][row] = K Q^T with M = 128 keys and
//    N = the rows rounded up to 16.  Tensor-memory lane t then holds one key's
//    scores for every row, and the softmax work spreads over all 128 lanes
//    whatever the row count.  The output is accumulated transposed too:
//    O^T[d][row] += V^T P^T with M = 128 (head dim), both operands read from
//    shared memory in MN-major form straight from the TMA tiles.  Head dim 64
//    keeps M = 128 with a V tile whose second 64-dim slab stays zero.
//  * Warp roles: warp 0 streams K and V tiles (TMA, 128 keys x all head dims
//    per box) into a two-stage ring; warp 1 issues the MMAs (one elected thread)
//    and owns the tensor-memory allocation; warps 2-9 run the softmax and the
//    epilogue, two per tensor-memory lane quadrant, each on half of the rows.
//    The next unit's Q is prefetched (cp.async) into a second buffer while
//    the current one runs.
//  * Lazy rescaling: the running row maxima only move when a score exceeds
//    them by more than 2^8 (a CTA-wide vote per chunk), so P = 2^(s - m) stays
//    <= 256 and the O^T columns in tensor memory are rescaled only then.  Row
//    maxima and per-key-lane row sums live in registers; the sums are reduced
//    across lanes once per unit.
//  * Stream-K split over 64-key slices (attn_common.cuh) with fp32 partials
//    and a log-sum-exp merge of split units.  Keys beyond the live cache (or
//    not loaded) get P = 0 and their V rows are zeroed in shared memory, so
//    whatever the unused cache slots hold cannot reach the result.
#include "attn_common.cuh"

namespace spade {
namespace attn {
namespace tc {

constexpr int kDMax = 128;                       // head dims the shared-memory tiles hold
constexpr int kKeys = 128;                       // keys per MMA chunk (two slices)
constexpr int kStages = 2;                       // K/V ring depth (chunks)
constexpr int kSoftWarps = 8;                    // softmax / epilogue warps
constexpr int kSoftThreads = 32 * kSoftWarps;
constexpr int kThreads = 64 + kSoftThreads;      // + producer warp + MMA warp
constexpr int kSlab = kKeys * 128;               // one 64-dim slab of a chunk: 16 KB
constexpr int kTile = 2 * kSlab;                 // K or V tile of a chunk: 32 KB
constexpr int kQSlab = kRowBlock * 128;          // one 64-dim slab of Q: 8 KB
constexpr int kPBytes = kKeys * 128;             // P^T: [128 keys][64 rows] bf16
constexpr uint32_t kTmemCols = 256;              // S^T x2 (64 cols each) + O^T (64 cols)
constexpr uint32_t kColS = 0, kColO = 128;
constexpr float kRescaleLog2 = 8.f;

// mbarriers.  ODone completes once per PV (chunk); OFinal once per segment,
// after its last PV, so the epilogue never waits on a parity that an older,
// still-running PV could alias.
constexpr int kBarKFull = 0, kBarVFull = 2, kBarKEmpty = 4, kBarVEmpty = 6, kBarSFull = 8,
              kBarSFree = 10, kBarPFull = 12, kBarPFree = 14, kBarODone = 16, kBarSeg = 17,
              kBarOFinal = 18, kBarQ = 19, kNumBars = 20;

struct Smem {
  static constexpr int K = 0;                               // [stage][2 slabs][128 keys][128 B]
  static constexpr int V = K + kStages * kTile;
  static constexpr int Q = V + kStages * kTile;             // [2 bufs][2 slabs][64 rows][128 B]
  static constexpr int P = Q + 4 * kQSlab;                  // [2 bufs][128 keys][128 B]
  static constexpr int PREF = P + 2 * kPBytes;              // int64 [kMaxB + 1]
  static constexpr int CTX = PREF + (kMaxB + 1) * 8;        // int32 [kMaxB]
  static constexpr int KD = CTX + kMaxB * 4;                // int32 [kMaxB]
  static constexpr int WRED = round_up_c(KD + kMaxB * 4, 128);  // float [4 quadrants][64 rows]
  static constexpr int ROWV = WRED + 4 * kRowBlock * 4;     // float [64 rows]: reduced value
  static constexpr int RMAX = ROWV + kRowBlock * 4;         // float [64 rows]: running maxima
  static constexpr int ALPHA = RMAX + kRowBlock * 4;        // float [64 rows]: rescale factors
  static constexpr int BAR = ALPHA + kRowBlock * 4;
  static constexpr int MISC = BAR + kNumBars * 8;           // abort, last, tmem base
  static constexpr int SEG0 = MISC + 64;                    // SegInfo: this CTA's first segment
  static constexpr int RANGE = SEG0 + 64;                   // CtaRange: this CTA's cost range
  static constexpr int BYTES = RANGE + 64 + 1024;           // + slack for 1024-byte alignment
};
static_assert(Smem::BAR % 8 == 0, "mbarriers need 8-byte alignment");
static_assert(Smem::RMAX % 16 == 0, "row maxima are read as float4");
static_assert(Smem::BYTES <= 225 * 1024, "shared memory budget");
static_assert(Smem::Q % 1024 == 0 && Smem::P % 1024 == 0, "swizzled tiles need 1024-byte alignment");

// Shared-memory descriptor of a 128-byte-swizzled operand.  K-major: 8-row
// groups `sbo` apart (lbo unused).  MN-major: 64-element blocks along M/N are
// `lbo` apart and 8-row groups along K are `sbo` apart.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFF) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFF) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFF) << 32;
  d |= static_cast<uint64_t>(1) << 46;  // descriptor version (sm_100 family)
  d |= static_cast<uint64_t>(2) << 61;  // 128-byte swizzle
  return d;
}

// barrier.red.or over `threads` threads of named barrier `id`.
__device__ __forceinline__ bool bar_any(int id, int threads, bool pred) {
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

// Reduce-scatter over the warp of NP values per lane (NP a power of two,
// <= 32): on return lane L holds the reduction over all 32 lanes of value
// L % NP.  Each step halves the values a lane keeps (it sends the half its
// partner keeps), so NP - 1 + log2(32 / NP) shuffles in all.  `v` is consumed.
template <int NP, bool kMax>
__device__ __forceinline__ float warp_reduce_scatter(float (&v)[NP], int lane) {
#pragma unroll
  for (int h = NP / 2; h >= 1; h /= 2) {
    const bool upper = (lane & h) != 0;
#pragma unroll
    for (int i = 0; i < h; ++i) {
      const float send = upper ? v[i] : v[i + h];
      const float keep = upper ? v[i + h] : v[i];
      const float got = __shfl_xor_sync(0xffffffffu, send, h);
      v[i] = kMax ? fmaxf(keep, got) : keep + got;
    }
  }
  float r = v[0];
#pragma unroll
  for (int o = NP; o < 32; o *= 2) {
    const float got = __shfl_xor_sync(0xffffffffu, r, o);
    r = kMax ? fmaxf(r, got) : r + got;
  }
  return r;
}

// 16-byte global -> shared copy (cp.async); src_bytes = 0 writes zeros.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// One segment of a CTA's range: the part of one unit's cost span in
// [x, seg_end); its real key slices are g.ci .. g.ci + n_here - 1.
struct SegInfo {
  Seg g;
  int64_t seg_end;
  int n_here;   // key slices in this segment (0: only the unit's virtual start)
  int nchunk;   // MMA chunks (pairs of slices, the last one possibly single)
};
__device__ __forceinline__ SegInfo seg_of(const Sched &sc, const Seg &g, int64_t x, int64_t x_end) {
  SegInfo s;
  s.g = g;
  s.seg_end = min(x_end, s.g.ust + sc.E + s.g.nch);
  const int lo = max(0, static_cast<int>(x - s.g.ust) - sc.E);
  const int hi = max(0, static_cast<int>(s.seg_end - s.g.ust) - sc.E);
  s.g.ci = lo;
  s.n_here = hi - lo;
  s.nchunk = (s.n_here + 1) / 2;
  return s;
}
__device__ __forceinline__ SegInfo seg_at(const Sched &sc, int64_t x, int64_t x_end) {
  return seg_of(sc, locate(sc, x), x, x_end);
}
// The first segment at or after cost position x that holds key slices (all
// roles skip the same empty ones); n_here == 0 when the range has none left.
__device__ __forceinline__ SegInfo next_seg(const Sched &sc, int64_t x, int64_t x_end) {
  SegInfo s = seg_at(sc, x, x_end);
  while (s.n_here == 0 && s.seg_end < x_end) s = seg_at(sc, s.seg_end, x_end);
  return s;
}
// The same, computed by a whole warp (every lane gets the result).
__device__ __forceinline__ SegInfo next_seg_warp(const Sched &sc, int64_t x, int64_t x_end, int lane) {
  SegInfo s = seg_of(sc, locate_warp(sc, x, lane), x, x_end);
  while (s.n_here == 0 && s.seg_end < x_end) s = seg_of(sc, locate_warp(sc, s.seg_end, lane), s.seg_end, x_end);
  return s;
}

// D: head dim, 64 or 128.  With D = 64 the K and V tiles hold one 64-dim slab
// and the V tiles' second slab stays zero, so O^T keeps M = 128 (its rows
// 64-127 are zero and never stored).
template <int NR, int D>
__global__ void __launch_bounds__(kThreads, 1)
    verify_attention_tc_kernel(const __grid_constant__ Params p,
                               const __grid_constant__ CUtensorMap tm_k2,
                               const __grid_constant__ CUtensorMap tm_v2,
                               const __grid_constant__ CUtensorMap tm_k1,
                               const __grid_constant__ CUtensorMap tm_v1) {
  static_assert(NR % 16 == 0 && NR >= 16 && NR <= kRowBlock, "MMA N must be 16..64, step 16");
  static_assert(D == 64 || D == kDMax, "head dim 64 or 128");
  constexpr int kD = D;
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned base, derived by pointer arithmetic so that the compiler
  // keeps the shared state space (plain ld/st.shared, not generic accesses).
  uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  int64_t *s_pref = reinterpret_cast<int64_t *>(smem + Smem::PREF);
  int32_t *s_ctx = reinterpret_cast<int32_t *>(smem + Smem::CTX);
  int32_t *s_kd = reinterpret_cast<int32_t *>(smem + Smem::KD);
  float *s_wred = reinterpret_cast<float *>(smem + Smem::WRED);
  float *s_rowv = reinterpret_cast<float *>(smem + Smem::ROWV);
  float *s_rmax = reinterpret_cast<float *>(smem + Smem::RMAX);
  float *s_alpha = reinterpret_cast<float *>(smem + Smem::ALPHA);
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + Smem::BAR);
  volatile int *s_abort = reinterpret_cast<volatile int *>(smem + Smem::MISC);
  volatile int *s_last = s_abort + 1;
  uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + Smem::MISC + 8);

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;

  if (tid == 0) { *s_abort = 0; *s_last = 0; }
  // Set-up that reads no input -- tensor-map prefetch, mbarriers, tensor
  // memory, the zero slab -- comes first: under programmatic dependent launch
  // it overlaps the end of the previous kernel in the stream.
  if (warp == 0 && lane < 2) {
    tma_prefetch_desc(lane ? &tm_v2 : &tm_k2);
    tma_prefetch_desc(lane ? &tm_v1 : &tm_k1);
  } else if (warp == 1) {
    if (lane == 0) {
      for (int s = 0; s < kStages; ++s) {
        mbar_init(&bars[kBarKFull + s], 1);
        mbar_init(&bars[kBarVFull + s], 1);
        mbar_init(&bars[kBarKEmpty + s], 1);
        mbar_init(&bars[kBarVEmpty + s], 1);
        mbar_init(&bars[kBarSFull + s], 1);
        mbar_init(&bars[kBarSFree + s], kSoftWarps);
        mbar_init(&bars[kBarPFull + s], kSoftWarps);
        mbar_init(&bars[kBarPFree + s], 1);
      }
      mbar_init(&bars[kBarODone], 1);
      mbar_init(&bars[kBarSeg], kSoftWarps);
      mbar_init(&bars[kBarQ], kSoftWarps);
      mbar_init(&bars[kBarOFinal], 1);
      fence_mbar_init();
    }
    __syncwarp();
    tmem_alloc(s_tmem, kTmemCols);
    tmem_relinquish();
  }
  if constexpr (kD == 64) {
    // The V tiles' second 64-dim slab: zeros for the whole launch (the copies
    // fill the first slab only).
    for (int e = tid; e < kStages * (kSlab / 16); e += kThreads) {
      const int st = e / (kSlab / 16), o = e % (kSlab / 16);
      *reinterpret_cast<uint4 *>(smem + Smem::V + st * kTile + kSlab + o * 16) = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
  }
  // Inputs written by earlier kernels in the stream are visible from here on.
  // The next kernel may be scheduled now: it waits for this grid to complete
  // before it reads anything this grid writes.
  griddep_wait();
  griddep_launch_dependents();
  sched_validate(p, s_ctx, s_kd, tid, kThreads);
  tc_fence_before();
  block_sync();
  tc_fence_after();
  Sched sc;
  sc.pref = s_pref; sc.ctx = s_ctx; sc.kd = s_kd;
  sc.B = p.B; sc.Hkv = p.Hkv; sc.G = p.G; sc.RB = p.RB; sc.E = p.unit_cost; sc.num_ctas = p.num_ctas;
  // Warp 0: the prefix of costs over sequences, then this CTA's range and
  // first segment (every role starts from it), all lanes together.
  SegInfo *s_seg0 = reinterpret_cast<SegInfo *>(smem + Smem::SEG0);
  CtaRange *s_range = reinterpret_cast<CtaRange *>(smem + Smem::RANGE);
  if (warp == 0) {
    sched_scan(p, sc, s_pref, lane);
    __syncwarp();
    Sched s0 = sc;
    s0.total = s_pref[p.B];
    // Never more CTAs than slices: every CTA kept has a non-empty range, so
    // the CTAs between a unit's first and last owner all contribute a partial.
    s0.num_ctas = static_cast<int>(s0.total < p.num_ctas ? s0.total : p.num_ctas);
    CtaRange r;
    r.total = s0.total;
    r.num_ctas = s0.num_ctas;
    r.active = s0.total > 0 && static_cast<int>(blockIdx.x) < s0.num_ctas;
    r.x_begin = r.x_end = 0;
    SegInfo seg0{};
    if (r.active) {
      r.x_begin = div_nn(static_cast<int64_t>(blockIdx.x) * s0.total, s0.num_ctas);
      r.x_end = div_nn(static_cast<int64_t>(blockIdx.x + 1) * s0.total, s0.num_ctas);
      seg0 = next_seg_warp(s0, r.x_begin, r.x_end, lane);
    }
    if (lane == 0) {
      *s_range = r;
      *s_seg0 = seg0;
    }
  }
  block_sync();
  const CtaRange rng = *s_range;
  sc.total = rng.total;
  sc.num_ctas = rng.num_ctas;
  if (!rng.active) {
    if (warp == 1) tmem_dealloc(*s_tmem, kTmemCols);
    return;
  }
  const int64_t x_begin = rng.x_begin;
  const int64_t x_end = rng.x_end;
  const SegInfo seg0 = *s_seg0;
  const uint32_t tmem = *s_tmem;
  const uint32_t smem_base = smem_u32(smem);

  if (warp == 0) {
    // ============================ producer: TMA ============================
    // Lane 0 loads the K tiles, lane 1 the V tiles: a K stage is refilled as
    // soon as its S product is done, without waiting behind the V stage that
    // only frees after the softmax and the PV product.
    if (lane < 2) {
      const bool is_v = lane == 1;
      const CUtensorMap *tm2 = is_v ? &tm_v2 : &tm_k2;
      const CUtensorMap *tm1 = is_v ? &tm_v1 : &tm_k1;
      const int bar_empty = is_v ? kBarVEmpty : kBarKEmpty;
      const int bar_full = is_v ? kBarVFull : kBarKFull;
      uint8_t *const ring = smem + (is_v ? Smem::V : Smem::K);
      const uint64_t pol = l2_policy_evict_first();
      uint32_t it = 0, issued = 0;
      bool expired = false;
      for (int64_t x = x_begin; x < x_end;) {
        const SegInfo si = x == x_begin ? seg0 : next_seg(sc, x, x_end);
        if (si.n_here == 0) break;
        const int row0 = (si.g.b * p.Hkv + si.g.kvh) * p.cap;
        for (int c = 0; c < si.nchunk; ++c, ++it) {
          const int st = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          const int nsl = min(2, si.n_here - 2 * c);
          const int key0 = (si.g.ci + 2 * c) * kChunk;
          // Cache rows of the chunk's slices: contiguous in a dense cache; in a
          // paged one each slice lies in one page (page sizes are multiples of
          // 64), found through the block table before the stage wait so that
          // the table load overlaps it.
          int row_a = row0 + key0, row_b = row_a + kChunk;
          if (p.block_table) {
            row_a = paged_row(p, si.g.b, si.g.kvh, key0);
            row_b = nsl == 2 ? paged_row(p, si.g.b, si.g.kvh, key0 + kChunk) : 0;
          }
          uint8_t *tile = ring + st * kTile;
          if (!mbar_wait(&bars[bar_empty + st], ph ^ 1, s_abort)) expired = true;
          if (*s_abort) continue;
          mbar_arrive_expect_tx(&bars[bar_full + st], nsl * (kSlab / kDMax) * kD);
          if (nsl == 2 && row_b == row_a + kChunk) {
            tma_load_3d(tile, tm2, 0, row_a, 0, &bars[bar_full + st], pol);
          } else {
            // One 64-key box per slice and slab; the second slice lands 64 rows in.
            for (int i = 0; i < nsl; ++i) {
              const int row = i ? row_b : row_a;
              uint8_t *dst = tile + i * kChunk * 128;
              tma_load_3d(dst, tm1, 0, row, 0, &bars[bar_full + st], pol);
              if constexpr (kD == kDMax) tma_load_3d(dst + kSlab, tm1, 0, row, 1, &bars[bar_full + st], pol);
            }
          }
          issued = it + 1;
        }
        x = si.seg_end;
      }
      if (expired || *s_abort) {
        atomicOr(p.status, SPADE_DEV_TIMEOUT);
        // Drain: every copy issued must land before the CTA's smem goes away.
        for (uint32_t j = (issued > kStages ? issued - kStages : 0); j < issued; ++j)
          mbar_wait_unabortable(&bars[bar_full + j % kStages], (j / kStages) & 1);
      }
    }
  } else if (warp == 1) {
    // ============================ MMA issuer ===============================
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(128, NR);                           // K-major A, B
      constexpr uint32_t idesc_pv = idesc_bf16_f32(128, NR) | (1u << 15) | (1u << 16);  // MN-major A, B
      bool expired = false;
      uint32_t it = 0, seg = 0;
      // O^T += V^T P^T for chunk j (first: overwrite instead of accumulate;
      // last: the segment's final product, signalled on OFinal too).
      auto issue_pv = [&](uint32_t j, bool first, bool last) {
        const int st = j % kStages;
        const uint32_t ph = (j / kStages) & 1;
        if (!mbar_wait(&bars[kBarVFull + st], ph, s_abort)) expired = true;
        if (!mbar_wait(&bars[kBarPFull + st], ph, s_abort)) expired = true;
        // The segment's first PV overwrites O^T: the previous epilogue has read it.
        if (first && !mbar_wait(&bars[kBarSeg], seg & 1, s_abort)) expired = true;
        tc_fence_after();
        if (!*s_abort) {
          const uint32_t v_addr = smem_base + Smem::V + st * kTile;
          const uint32_t p_addr = smem_base + Smem::P + st * kPBytes;
#pragma unroll
          for (int kk = 0; kk < kKeys / 16; ++kk)
            tc_mma_f16(tmem + kColO, desc_sw128(v_addr + kk * 2048, kSlab, 1024),
                       desc_sw128(p_addr + kk * 2048, kSlab, 1024), idesc_pv,
                       (first && kk == 0) ? 0u : 1u);
        }
        tc_commit(&bars[kBarVEmpty + st]);
        tc_commit(&bars[kBarPFree + st]);
        tc_commit(&bars[kBarODone]);
        if (last) tc_commit(&bars[kBarOFinal]);
      };
      for (int64_t x = x_begin; x < x_end;) {
        const SegInfo si = x == x_begin ? seg0 : next_seg(sc, x, x_end);
        if (si.n_here == 0) break;
        // Q staged: the segment's S products may start while the previous
        // segment's epilogue still reads O^T.
        if (!mbar_wait(&bars[kBarQ], seg & 1, s_abort)) expired = true;
        tc_fence_after();
        const uint32_t q_addr = smem_base + Smem::Q + (seg & 1) * 2 * kQSlab;
        for (int c = 0; c < si.nchunk; ++c, ++it) {
          const int st = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!mbar_wait(&bars[kBarKFull + st], ph, s_abort)) expired = true;
          if (!mbar_wait(&bars[kBarSFree + st], ph ^ 1, s_abort)) expired = true;
          tc_fence_after();
          if (!*s_abort) {
            const uint32_t k_addr = smem_base + Smem::K + st * kTile;
#pragma unroll
            for (int kk = 0; kk < kD / 16; ++kk) {
              const uint32_t off = (kk >> 2) * kSlab + (kk & 3) * 32;
              const uint32_t qoff = (kk >> 2) * kQSlab + (kk & 3) * 32;
              tc_mma_f16(tmem + kColS + st * 64, desc_sw128(k_addr + off, 16, 1024),
                         desc_sw128(q_addr + qoff, 16, 1024), idesc_s, kk > 0 ? 1u : 0u);
            }
          }
          tc_commit(&bars[kBarSFull + st]);
          tc_commit(&bars[kBarKEmpty + st]);
          if (c > 0) issue_pv(it - 1, c == 1, false);
        }
        issue_pv(it - 1, si.nchunk == 1, true);
        ++seg;
        x = si.seg_end;
      }
      if (expired) atomicOr(p.status, SPADE_DEV_TIMEOUT);
    }
  } else {
    // ===================== softmax and epilogue (warps 2-9) =================
    constexpr int NH = NR / 2;             // rows (S^T / O^T columns) per softmax warp
    constexpr int NP = NH <= 8 ? 8 : (NH <= 16 ? 16 : 32);  // NH padded to a power of two
    const int q4 = warp & 3;               // tensor-memory lane quadrant of this warp
    const int half = (warp - 2) >> 2;      // which half of the rows
    const int t = q4 * 32 + lane;          // key lane (softmax) / head-dim lane (epilogue)
    const int stid = tid - 64;             // 0..255
    const uint32_t tlane = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    const int c0 = half * NH;              // first row (column) of this warp
    bool expired = false;
    uint32_t it = 0, seg = 0;

    // Q of a segment into buffer qb: rows >= nrow zero-filled, 128-byte swizzle.
    auto prefetch_q = [&](const SegInfo &sq, int qb) {
      const int kdq = s_kd[sq.g.b];
      const int nrq = min(kRowBlock, p.G * (kdq + 1) - kRowBlock * sq.g.rb);
      const int qr0 = p.cu_q[sq.g.b];
      const uint32_t base = smem_base + Smem::Q + qb * 2 * kQSlab;
      for (int e = stid; e < NR * (kD / 8); e += kSoftThreads) {
        const int r = e / (kD / 8), c = e % (kD / 8);
        const bool real = r < nrq;
        const __nv_bfloat16 *src = real ? p.q + out_row(p, qr0, sq.g.kvh, sq.g.rb, r) * kD + c * 8 : p.q;
        cp_async16(base + (c >> 3) * kQSlab + r * 128 + (((c & 7) ^ (r & 7)) << 4), src, real ? 16u : 0u);
      }
    };

    SegInfo si = seg0;
    if (si.n_here > 0) prefetch_q(si, 0);
    cp_async_commit();
    for (int64_t x = x_begin; x < x_end && si.n_here > 0;) {
      const Seg g = si.g;
      SegInfo si_next = si;
      si_next.n_here = 0;
      if (si.seg_end < x_end) {
        si_next = next_seg(sc, si.seg_end, x_end);
        if (si_next.n_here > 0) prefetch_q(si_next, (seg + 1) & 1);  // that buffer's last reader (unit seg-1) is done
      }
      cp_async_commit();
      const int ctx = s_ctx[g.b];
      const int kd = s_kd[g.b];
      const int nrow = min(kRowBlock, p.G * (kd + 1) - kRowBlock * g.rb);
      const int Lkeys = ctx + kd + 1;  // live cache slots of the sequence
      const int q_row0 = p.cu_q[g.b];
      // Rows of this warp are [c0, c0 + NH); of those, r < hi are real rows.
      const int hi = nrow - c0;
      if (stid < kRowBlock) s_rmax[stid] = -INFINITY;
      cp_async_wait<1>();  // this segment's Q has landed
      fence_proxy_async_smem();
      named_bar(1, kSoftThreads);
      __syncwarp();
      // Segment 0's Q is ready now; a later segment's was signalled before the
      // previous epilogue.  O^T is free (the previous epilogue is done).
      if (lane == 0) {
        if (seg == 0) mbar_arrive(&bars[kBarQ]);
        mbar_arrive(&bars[kBarSeg]);
      }

      // Running row maxima live in s_rmax (one writer per row); the row sums of
      // this key lane in l.
      float l[NH], x_[NP];
#pragma unroll
      for (int r = 0; r < NH; ++r) l[r] = 0.f;
      const float4 *rmax4 = reinterpret_cast<const float4 *>(s_rmax + c0);

      for (int c = 0; c < si.nchunk; ++c, ++it) {
        const int st = it % kStages;
        const uint32_t ph = (it / kStages) & 1;
        const int key0 = (g.ci + 2 * c) * kChunk;  // first key of the chunk (sequence position)
        const int nk = min(2, si.n_here - 2 * c) * kChunk;
        const int kg = key0 + t;
        // Row R = 64 rb + rr (position R / G) sees key kg iff R >= (kg - ctx) G:
        // the visible rows of this key lane are rr in [lo, nrow).
        const int lo = (t < nk) ? max(0, (kg - ctx) * p.G - kRowBlock * g.rb) - c0 : NH;
        const uint32_t taddr = tlane + kColS + st * 64 + c0;

        // ---- S^T lane t, this warp's rows: scale, mask, test vs maxima ----
        if (!mbar_wait(&bars[kBarSFull + st], ph, s_abort)) expired = true;
        tc_fence_after();
#pragma unroll
        for (int j = 0; j < NH / 8; ++j) tmem_ld8(taddr + j * 8, reinterpret_cast<uint32_t *>(x_) + j * 8);
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[kBarSFree + st]);
        bool exceed = false;
#pragma unroll
        for (int r4 = 0; r4 < NH / 4; ++r4) {
          const float4 mv = rmax4[r4];
          const float mm[4] = {mv.x, mv.y, mv.z, mv.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int r = r4 * 4 + e;
            const bool vis = r >= lo && r < hi;
            // m = -inf (no visible key yet) gives +inf for a visible score: a vote.
            x_[r] = vis ? fmaf(x_[r], p.scale_log2, -mm[e]) : -INFINITY;
            exceed |= x_[r] > kRescaleLog2;
          }
        }
        // The two halves own disjoint rows: each votes and rescales on its own
        // barriers (ids 2-3 and 4-5), so neither waits for the other.
        if (bar_any(2 + half, kSoftThreads / 2, exceed)) {
          // Some score is more than 2^8 above its row's running maximum (always
          // so in a unit's first chunk): take this chunk's exact row maxima.
          // The S^T buffer is still intact (it is reused only after this
          // chunk's P is signalled).
#pragma unroll
          for (int j = 0; j < NH / 8; ++j) tmem_ld8(taddr + j * 8, reinterpret_cast<uint32_t *>(x_) + j * 8);
          tmem_wait_ld();
#pragma unroll
          for (int r = 0; r < NP; ++r)
            x_[r] = (r < NH && r >= lo && r < hi) ? x_[r] * p.scale_log2 : -INFINITY;
          {
            const float wm = warp_reduce_scatter<NP, true>(x_, lane);
            if (lane < NH) s_wred[q4 * kRowBlock + c0 + lane] = wm;
          }
          named_bar(4 + half, kSoftThreads / 2);
          const int hs = stid - half * (kSoftThreads / 2);  // thread of this half
          if (hs < NH) {
            const int row = c0 + hs;
            const float mo = s_rmax[row];
            const float mn = fmaxf(fmaxf(mo, fmaxf(s_wred[row], s_wred[kRowBlock + row])),
                                   fmaxf(s_wred[2 * kRowBlock + row], s_wred[3 * kRowBlock + row]));
            s_alpha[row] = mn > mo ? ex2(mo - mn) : 1.f;  // mo = -inf gives 0: nothing to keep
            s_rmax[row] = mn;
          }
          named_bar(4 + half, kSoftThreads / 2);
#pragma unroll
          for (int r = 0; r < NH; ++r) l[r] *= s_alpha[c0 + r];
          if (c > 0) {
            // O^T holds the chunks already multiplied in: rescale its columns
            // once the last PV has landed.  S of this chunk has completed, so
            // every PV issued before it has too: ODone is at most one phase
            // behind and its parity cannot alias.
            if (!mbar_wait(&bars[kBarODone], (it - 1) & 1, s_abort)) expired = true;
            tc_fence_after();
#pragma unroll
            for (int j = 0; j < NH / 8; ++j) {
              uint32_t o8[8];
              tmem_ld8(tlane + kColO + c0 + j * 8, o8);
              tmem_wait_ld();
#pragma unroll
              for (int e = 0; e < 8; ++e)
                o8[e] = __float_as_uint(__uint_as_float(o8[e]) * s_alpha[c0 + j * 8 + e]);
              tmem_st8(tlane + kColO + c0 + j * 8, o8);
            }
            tmem_wait_st();
          }
          // Scores relative to the new maxima (S^T reloaded: the reduction
          // consumed them).
#pragma unroll
          for (int j = 0; j < NH / 8; ++j) tmem_ld8(taddr + j * 8, reinterpret_cast<uint32_t *>(x_) + j * 8);
          tmem_wait_ld();
#pragma unroll
          for (int r = 0; r < NH; ++r)
            x_[r] = (r >= lo && r < hi) ? fmaf(x_[r], p.scale_log2, -s_rmax[c0 + r]) : -INFINITY;
        }

        // ---- P^T row of this key (this warp's rows): bf16, 128-byte swizzle ----
        if (!mbar_wait(&bars[kBarPFree + st], ph ^ 1, s_abort)) expired = true;
        {
          uint8_t *prow = smem + Smem::P + st * kPBytes + t * 128;
#pragma unroll
          for (int j = 0; j < NH / 8; ++j) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int r0 = j * 8 + 2 * e;
              const float p0 = ex2(x_[r0]), p1 = ex2(x_[r0 + 1]);
              l[r0] += p0;
              l[r0 + 1] += p1;
              w[e] = pack_bf16(p0, p1);
            }
            *reinterpret_cast<uint4 *>(prow + (((c0 / 8 + j) ^ (t & 7)) << 4)) =
                make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
        // V rows that were not loaded, or lie beyond the live cache, may hold
        // anything (NaN): zero them so that P = 0 really contributes nothing.
        // Each half of the warps clears one 64-dim slab.
        const bool zero_v = t >= nk || kg >= Lkeys;
        if (__any_sync(0xffffffffu, zero_v)) {
          if (!mbar_wait(&bars[kBarVFull + st], ph, s_abort)) expired = true;
          if (zero_v) {
            uint8_t *vrow = smem + Smem::V + st * kTile + half * kSlab + t * 128;
#pragma unroll
            for (int e = 0; e < 8; ++e) *reinterpret_cast<uint4 *>(vrow + e * 16) = make_uint4(0, 0, 0, 0);
          }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[kBarPFull + st]);
      }
      // The next segment's Q (prefetched at this segment's start) lets the MMA
      // warp start its S products during this epilogue.
      if (si_next.n_here > 0) {
        cp_async_wait<0>();
        fence_proxy_async_smem();
        named_bar(1, kSoftThreads);
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[kBarQ]);
      }

      // ---- epilogue: row sums, O^T from tensor memory, output or partial ----
      // (the maxima are read before the barriers below, after which the next
      // unit may reset them)
      const bool row_writer = q4 == 0 && lane < NH && lane < hi;
      const float m_own = row_writer ? s_rmax[c0 + lane] : 0.f;
      {
        float v[NP];
#pragma unroll
        for (int r = 0; r < NP; ++r) v[r] = r < NH ? l[r] : 0.f;
        const float ws = warp_reduce_scatter<NP, false>(v, lane);
        if (lane < NH) s_wred[q4 * kRowBlock + c0 + lane] = ws;
      }
      named_bar(1, kSoftThreads);
      if (stid < NR)
        s_rowv[stid] = (s_wred[stid] + s_wred[kRowBlock + stid]) +
                       (s_wred[2 * kRowBlock + stid] + s_wred[3 * kRowBlock + stid]);
      named_bar(1, kSoftThreads);
#pragma unroll
      for (int r = 0; r < NH; ++r) l[r] = s_rowv[c0 + r];
      // Row statistics of this warp's rows, one lane per row (quadrant-0 warps).
      const float l_own = row_writer ? s_rowv[c0 + lane] : 1.f;
      if (!mbar_wait(&bars[kBarOFinal], seg & 1, s_abort)) expired = true;
      tc_fence_after();
      const int unit = (g.b * p.Hkv + g.kvh) * p.RB + g.rb;
      const int64_t c_first = sc.owner(g.ust + sc.E);
      const int64_t c_last = sc.owner(g.ust + sc.E + g.nch - 1);
      const int nparts = static_cast<int>(c_last - c_first + 1);
      if (nparts == 1) {
        // Output row of this warp's row c0 + r, advanced row by row (one
        // division for the warp's first row instead of one per row).
        const int row0 = kRowBlock * g.rb + c0;
        int gh = row0 % p.G;
        size_t orow = static_cast<size_t>(q_row0 + row0 / p.G) * p.Hq + g.kvh * p.G + gh;
#pragma unroll
        for (int j = 0; j < NH / 8; ++j) {
          uint32_t o8[8];
          tmem_ld8(tlane + kColO + c0 + j * 8, o8);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            // l >= 1 (the row maximum's own term), so the fast divide is exact
            // to a few fp32 ulps, far below the bf16 rounding that follows.
            if (j * 8 + e < hi && t < kD)
              p.out[orow * kD + t] = __float2bfloat16_rn(__fdividef(__uint_as_float(o8[e]), l[j * 8 + e]));
            if (++gh == p.G) {
              gh = 0;
              orow += p.Hq - p.G + 1;
            } else {
              ++orow;
            }
          }
        }
        tc_fence_before();
        if (p.lse && row_writer)
          p.lse[out_row(p, q_row0, g.kvh, g.rb, c0 + lane)] = (m_own + log2f(l_own)) * 0.69314718055994531f;
      } else {
        const int64_t slot = blockIdx.x + unit;
        float *part = p.partials + slot * slot_floats(kD);
#pragma unroll
        for (int j = 0; j < NH / 8; ++j) {
          uint32_t o8[8];
          tmem_ld8(tlane + kColO + c0 + j * 8, o8);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 8; ++e)
            if (j * 8 + e < hi && t < kD) __stcg(part + (c0 + j * 8 + e) * kD + t, __uint_as_float(o8[e]));
        }
        tc_fence_before();
        if (row_writer) {
          __stcg(part + kRowBlock * kD + c0 + lane, m_own);
          __stcg(part + kRowBlock * kD + kRowBlock + c0 + lane, l_own);
        }
        named_bar(1, kSoftThreads);
        if (stid == 0) *s_last = arrive_part(&p.counters[unit], nparts);
        named_bar(1, kSoftThreads);
        if (*s_last) {
          // This CTA finished the unit last: merge every partial by log-sum-exp.
          merge_partials<kD, 5>(p, c_first + unit, nparts, nrow, g.rb, g.kvh, q_row0, warp - 2,
                                kSoftWarps, lane);
          if (stid == 0) p.counters[unit] = 0;  // every part has arrived: reset for the next call
        }
      }
      ++seg;
      x = si.seg_end;
      si = si_next;
    }
    cp_async_wait<0>();
    if (expired) atomicOr(p.status, SPADE_DEV_TIMEOUT);
  }

  tc_fence_before();
  block_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

template <int NR, int D>
static cudaError_t launch_nr(const Params &p, const CUtensorMap &k2, const CUtensorMap &v2,
                             const CUtensorMap &k1, const CUtensorMap &v1, cudaStream_t stream) {
  auto kern = verify_attention_tc_kernel<NR, D>;
  static bool configured = false;  // per template instance; the attribute is per function
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Smem::BYTES);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  // Programmatic dependent launch: the kernel's input-free set-up may overlap
  // the previous kernel in the stream (the kernel waits for it before reading
  // any input).
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.num_ctas);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Smem::BYTES;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, p, k2, v2, k1, v1);
}

}  // namespace tc

cudaError_t launch_tc(const Params &p, const CUtensorMap &k2, const CUtensorMap &v2,
                      const CUtensorMap &k1, const CUtensorMap &v1, int nr, int d, cudaStream_t stream) {
  if (d == 64) {
    switch (nr) {
      case 16: return tc::launch_nr<16, 64>(p, k2, v2, k1, v1, stream);
      case 32: return tc::launch_nr<32, 64>(p, k2, v2, k1, v1, stream);
      case 48: return tc::launch_nr<48, 64>(p, k2, v2, k1, v1, stream);
      default: return tc::launch_nr<64, 64>(p, k2, v2, k1, v1, stream);
    }
  }
  switch (nr) {
    case 16: return tc::launch_nr<16, 128>(p, k2, v2, k1, v1, stream);
    case 32: return tc::launch_nr<32, 128>(p, k2, v2, k1, v1, stream);
    case 48: return tc::launch_nr<48, 128>(p, k2, v2, k1, v1, stream);
    default: return tc::launch_nr<64, 128>(p, k2, v2, k1, v1, stream);
  }
}


}  // namespace attn
}  // namespace spade
