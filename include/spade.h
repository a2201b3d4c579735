/*
 * spade.h -- C ABI of the SPADE verify step on GB300 (sm_103a).
 *
 * SPADE (edge-cloud speculative decoding) sends a block of k draft tokens from
 * an edge draft model to a cloud verifier, which scores all k+1 positions in a
 * single forward pass and keeps the longest accepted prefix plus one corrected
 * (or bonus) token (Sec. III-B, Sec. III-C, Algorithm 1).  This library holds
 * the verifier's hot path of that step:
 *
 *   spade_verify_attention  attention of the k+1 verify positions against the
 *                           KV cache (the verifier's forward pass, Algorithm 1
 *                           "Cloud: in parallel ... in a single forward pass")
 *   spade_verify_accept     LM head o = g(x_L), softmax (Sec. III-A) fused with
 *                           the accept test alpha = min(1, p/q) and the residual
 *                           sampling from norm(max(0, p - q)) (Sec. III-C)
 *   spade_kv_commit         context update m <- m + a + 1 (Algorithm 1) on the
 *                           KV cache: keep accepted slots, clear rejected ones
 *   spade_verify_accept_commit  the two calls above fused into one launch
 *   spade_verify_qkv_rope   the verify block's QKV projection with rotary
 *                           embedding, writing its K/V into the cache slots
 *                           the attention reads
 *
 * Conventions shared by every call
 *  - Every pointer argument is a DEVICE pointer owned by the caller; the
 *    library keeps no reference after the call returns.
 *  - Calls are asynchronous on `stream` and never synchronise the host.
 *  - The return value reports host-side validation and launch errors.  Errors
 *    found on the device (bad indices, capacity overflow, an expired bounded
 *    wait) are OR-ed into the caller's device int32 `status` word (the
 *    SPADE_DEV_* bits); the caller zeroes it and reads it back when it chooses.
 *  - Every kernel targets sm_103a only; other devices get
 *    SPADE_ERR_UNSUPPORTED_DEVICE.  There is no fallback path.
 *  - spade_last_error() returns a thread-local message for the last non-OK
 *    status returned on the calling thread.
 *
 * Row layout of a verify step with B sequences: sequence b has n_draft[b] = k_b
 * drafts and k_b + 1 verify positions; position i (0 <= i <= k_b) of sequence b
 * is row cu_q[b] + i, with cu_q[0] = 0 and cu_q[b+1] = cu_q[b] + k_b + 1, so
 * R = cu_q[B] rows in total.  Position 0 is the last accepted token; position
 * i >= 1 is draft i-1.
 */
#ifndef SPADE_H_
#define SPADE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t; 0 is the legacy default stream. */
typedef struct CUstream_st *spade_stream_t;

typedef enum {
  SPADE_OK = 0,
  SPADE_ERR_INVALID_ARG = 1,       /* null pointer, negative size, bad mode   */
  SPADE_ERR_SHAPE = 2,             /* unsupported shape (e.g. D not 64/128)   */
  SPADE_ERR_CAPACITY = 3,          /* host-visible capacity bound exceeded    */
  SPADE_ERR_UNSUPPORTED_DEVICE = 4,/* current device is not sm_103            */
  SPADE_ERR_CUDA = 5,              /* a CUDA runtime / driver call failed     */
  SPADE_ERR_WORKSPACE = 6,         /* workspace missing, too small, misaligned*/
} spade_status;

/* Device status word bits (OR-ed by kernels into the caller's int32). */
#define SPADE_DEV_BAD_INDEX 0x1  /* cu_q inconsistent, n_draft > max_k, token id out of range */
#define SPADE_DEV_CAPACITY  0x2  /* ctx_lens[b] + n_draft[b] + 1 > cap                       */
#define SPADE_DEV_TIMEOUT   0x4  /* a bounded device-side wait expired; outputs are invalid  */
#define SPADE_DEV_FALLBACK  0x8  /* a residual had no positive mass; p was sampled instead   */

/* ------------------------------------------------------------------------ */
/* QKV projection + rotary embedding of the verify block (Sec. III-A/III-B)  */
/* ------------------------------------------------------------------------ */
/*
 * The verifier's projection of the verify block's hidden states into queries,
 * keys and values -- the input side of the attention in x_{l+1} = x_l +
 * f_l(x_l) (Sec. III-A) for the d+1 positions scored in the single forward
 * pass (Sec. III-B) -- with rotary position embedding, writing the block's
 * keys and values into its cache slots, ready for spade_verify_attention:
 *   y = x W^T (fp32 accumulation on the tensor cores), split into the head
 *   slices q_h (h < Hq), k_g, v_g (g < Hkv);
 *   q and k are rotated at the row's position pos = ctx_lens[b] + i (row
 *   cu_q[b] + i): the pair (dimension j, j + D/2) turns counter-clockwise by
 *   pos * rope_theta^(-2j/D); v is not rotated;
 *   q_out[cu_q[b]+i, h, :] = q_h, k_cache[b, g, ctx_b+i, :] = k_g and
 *   v_cache[b, g, ctx_b+i, :] = v_g, rounded to bf16.
 *
 *   x           bf16 [R, H] row-major (the verify rows' hidden states), H % 8 == 0
 *   w_qkv       bf16 [(Hq + 2 Hkv) D, H] row-major (nn.Linear layout): the query
 *               heads' rows, then the key heads', then the value heads';
 *               (Hq + 2 Hkv) * D a multiple of 128
 *   ctx_lens, n_draft, cu_q   int32 [B], [B], [B+1], as for the attention
 *   q_out       bf16 [R, Hq, D] written
 *   k_cache, v_cache  bf16 [B, Hkv, cap, D]: slots [ctx_b, ctx_b + n_draft[b]]
 *               written, every other slot left as it is
 *   B, R, H, Hq, Hkv, D, cap, max_k   sizes; D in {64, 128}; R <= 512
 *   rope_theta  base of the rotary frequencies (10000 for Llama-2, 500000 for
 *               Llama-3), finite and > 1
 *   status      device int32: a sequence whose block is invalid
 *               (SPADE_DEV_BAD_INDEX) or does not fit its cache
 *               (SPADE_DEV_CAPACITY) is skipped; none of its rows is written
 *   workspace   device scratch of at least spade_qkv_workspace_size(R, Hq, Hkv, D)
 *               bytes, 256-byte aligned, ZEROED ONCE by the caller after
 *               allocation; every call that completes leaves its counters
 *               zeroed again (a call that reported SPADE_DEV_TIMEOUT may not:
 *               zero the workspace again before the next one).  Calls that
 *               share a workspace must be ordered.
 * Every pointer is a 16-byte aligned device pointer.  The contraction is split
 * over every SM; the split parts' fp32 sums meet in the workspace and are
 * added in a fixed order, so results do not depend on timing.  The kernel
 * keeps every block of the grid resident at once (cooperative launch, with
 * programmatic dependent launch): the CTAs that finish a split tile wait,
 * bounded, for the other CTAs' partial sums.
 */
spade_status spade_verify_qkv_rope(const void *x, const void *w_qkv, const int32_t *ctx_lens,
                                   const int32_t *n_draft, const int32_t *cu_q, void *q_out,
                                   void *k_cache, void *v_cache, int32_t B, int32_t R, int32_t H,
                                   int32_t Hq, int32_t Hkv, int32_t D, int32_t cap, int32_t max_k,
                                   float rope_theta, void *workspace, size_t workspace_bytes,
                                   int32_t *status, spade_stream_t stream);

/* Bytes of workspace spade_verify_qkv_rope (and its paged form) needs for these
 * sizes on the current device (0 on invalid sizes). */
size_t spade_qkv_workspace_size(int32_t R, int32_t Hq, int32_t Hkv, int32_t D);

/* ------------------------------------------------------------------------ */
/* Verify attention (Sec. III-B verification stage; Algorithm 1 cloud step)  */
/* ------------------------------------------------------------------------ */
/*
 * For every sequence b, position i in [0, k_b] and query head h:
 *   out[cu_q[b]+i, h, :] = softmax(q . K^T / sqrt(D)) V
 * over the keys in slots [0, ctx_lens[b] + i] of KV head h / (Hq / Hkv).  Slots
 * [0, ctx_b) hold the committed context and slots [ctx_b, ctx_b + k_b] the
 * verify block itself (written by the caller before this call), so the mask is
 * causal inside the draft block only.  Scores are scaled by 1/sqrt(D); inputs
 * are post-RoPE; no softcap, window or ALiBi.
 *
 *   q          bf16 [R, Hq, D] row-major (row = cu_q[b] + i)
 *   k_cache    bf16 [B, Hkv, cap, D] row-major; 16-byte aligned
 *   v_cache    bf16 [B, Hkv, cap, D] row-major; 16-byte aligned
 *   ctx_lens   int32 [B] committed context length per sequence
 *   n_draft    int32 [B] draft count k_b, 0 <= k_b <= max_k
 *   cu_q       int32 [B+1] row offsets (see above)
 *   out        bf16 [R, Hq, D] written
 *   lse        float32 [R, Hq] natural-log sum-exp of the scaled scores, or NULL
 *   B, Hq, Hkv, D, cap, max_k, R   sizes; Hq % Hkv == 0; D in {64, 128};
 *              Hq / Hkv * (max_k + 1) query rows share each KV head
 *   workspace  device scratch of at least spade_attn_workspace_size(...) bytes,
 *              256-byte aligned, ZEROED ONCE by the caller after allocation;
 *              every call that completes leaves it zeroed again.  Calls that
 *              share a workspace must be ordered (same stream or events).
 *   status     device int32, SPADE_DEV_* bits OR-ed in
 * Slots beyond ctx_b + k_b are never read into the result, whatever they hold.
 */
spade_status spade_verify_attention(const void *q, const void *k_cache, const void *v_cache,
                                    const int32_t *ctx_lens, const int32_t *n_draft,
                                    const int32_t *cu_q, void *out, float *lse, int32_t B,
                                    int32_t Hq, int32_t Hkv, int32_t D, int32_t cap,
                                    int32_t max_k, int32_t R, void *workspace,
                                    size_t workspace_bytes, int32_t *status,
                                    spade_stream_t stream);

/* Bytes of workspace spade_verify_attention needs for these sizes on the
 * current device (0 on invalid sizes). */
size_t spade_attn_workspace_size(int32_t B, int32_t Hq, int32_t Hkv, int32_t D, int32_t cap,
                                 int32_t max_k);

/*
 * spade_verify_attention_noalloc -- the same attention for callers that cannot
 * allocate device memory (for example plugin hosts that pass a kernel only its
 * inputs and outputs, or serving loops whose memory pool is frozen after
 * start-up).  The paper has no counterpart: this is a deployment variant.
 *
 * Arguments are those of spade_verify_attention without the workspace.  The
 * scratch is a 32 MiB file-scope device array that every GPU loading this
 * library holds until the process exits; the call allocates nothing.
 *  - Sizes whose workspace (spade_attn_workspace_size) exceeds 32 MiB are
 *    rejected with SPADE_ERR_CAPACITY and a message giving both sizes.
 *  - The first call on each device resolves the array's device address
 *    (cudaGetSymbolAddress); make that first call before any stream capture.
 *  - Every call shares the one array and clears its merge counters first
 *    (cudaMemsetAsync on `stream`): calls that overlap on the GPU, on any
 *    streams, race and corrupt each other's results.  Order them.
 */
spade_status spade_verify_attention_noalloc(const void *q, const void *k_cache,
                                            const void *v_cache, const int32_t *ctx_lens,
                                            const int32_t *n_draft, const int32_t *cu_q, void *out,
                                            float *lse, int32_t B, int32_t Hq, int32_t Hkv,
                                            int32_t D, int32_t cap, int32_t max_k, int32_t R,
                                            int32_t *status, spade_stream_t stream);

/* ------------------------------------------------------------------------ */
/* LM head + softmax + accept/reject + residual sampling (Sec. III-A/III-C)  */
/* ------------------------------------------------------------------------ */
/*
 * logits[r, x] = sum_j hidden[r, j] * w_lm[x, j] (fp32 accumulation on the
 * tensor cores; the logits never leave the chip) and p_r = softmax(logits[r]).
 * For every sequence b (rows r_i = cu_q[b] + i, draft d_i = draft_tokens[cu_q[b]
 * - b + i] for i < k_b):
 *   greedy (mode 0):     draft i is accepted iff d_i == argmax_x logits[r_i, x]
 *                        (lowest index on ties);
 *   stochastic (mode 1): draft i is accepted iff u[r_i] < p_{r_i}(d_i) / q_i(d_i)
 *                        with q_i = draft_probs[cu_q[b] - b + i, :] (q_i(d_i) = 0
 *                        accepts iff p(d_i) > 0);
 * acceptance stops at the first rejection; a_b = number of accepted drafts is
 * written to accepted_len[b].  next_token[b] is, with r* = cu_q[b] + a_b:
 *   greedy:      argmax_x logits[r*, x];
 *   stochastic:  if a_b < k_b a draw from norm(max(0, p_{r*} - q_{a_b})), else
 *                (bonus) a draw from p_{r*}; the draw is the smallest x whose
 *                cumulative mass (ascending x, fp64) exceeds u[cu_q[b] + k_b] * Z.
 *
 *   hidden        bf16 [R, H] row-major, 16-byte aligned, H % 8 == 0
 *   w_lm          bf16 [V, H] row-major (nn.Linear layout), 16-byte aligned
 *   draft_tokens  int32 [R - B]
 *   draft_probs   float32 [R - B, V] row-major, or NULL when no stochastic
 *                 sequence has drafts (a stochastic sequence with k_b = 0
 *                 draws its token from p and reads no q); a stochastic
 *                 sequence with drafts and NULL draft_probs sets
 *                 SPADE_DEV_BAD_INDEX and is verified greedily
 *   uniforms      float32 [R] in [0, 1)
 *   mode          int32 [B], 0 greedy / 1 stochastic
 *   cu_q, n_draft int32 [B+1], [B]
 *   accepted_len  int32 [B] written;  next_token int32 [B] written
 *   workspace     scratch of spade_accept_workspace_size(...) bytes, 256-byte
 *                 aligned, ZEROED ONCE by the caller; completed calls leave the
 *                 parts that must start at zero zeroed again.
 *   status        device int32, SPADE_DEV_* bits OR-ed in
 * The kernel keeps every block of the grid resident at once (cooperative
 * launch) and meets at bounded device-wide barriers; if a barrier expires the
 * outputs are invalid and SPADE_DEV_TIMEOUT is set; zero the workspace again
 * before the next call.
 */
spade_status spade_verify_accept(const void *hidden, const void *w_lm,
                                 const int32_t *draft_tokens, const float *draft_probs,
                                 const float *uniforms, const int32_t *mode,
                                 const int32_t *cu_q, const int32_t *n_draft,
                                 int32_t *accepted_len, int32_t *next_token, int32_t B,
                                 int32_t R, int32_t H, int32_t V, void *workspace,
                                 size_t workspace_bytes, int32_t *status,
                                 spade_stream_t stream);

/*
 * spade_verify_accept with a softmax temperature per sequence: the verifier's
 * distribution is p = softmax(logits / temperature[b]) in the accept test and
 * in the residual / bonus draw (sampling "for diversity", Sec. III-A; the
 * test and p' of Sec. III-C are unchanged otherwise).  Greedy sequences take
 * the argmax, which no positive temperature changes.  draft_probs is the draft
 * model's distribution at its own temperature, as the caller produced it.
 *   temperature  float32 [B] device array, each finite and > 0 (a value that
 *                is not is taken as 1 and sets SPADE_DEV_BAD_INDEX)
 * The row statistics of spade_accept_stats_layout are then those of l / T.
 * Every other argument is that of spade_verify_accept.
 */
spade_status spade_verify_accept_temperature(const void *hidden, const void *w_lm,
                                             const int32_t *draft_tokens, const float *draft_probs,
                                             const float *uniforms, const int32_t *mode,
                                             const float *temperature, const int32_t *cu_q,
                                             const int32_t *n_draft, int32_t *accepted_len,
                                             int32_t *next_token, int32_t B, int32_t R, int32_t H,
                                             int32_t V, void *workspace, size_t workspace_bytes,
                                             int32_t *status, spade_stream_t stream);

/*
 * spade_verify_accept with the verifier's sampling options and an optional
 * fused KV commit: the general form of the calls above.
 *
 * temperature [B] (float32, device; may be null: all 1): p = softmax(l / T_b)
 *   for sequence b, as in spade_verify_accept_temperature.
 * top_p [B] (float32, device; may be null: no truncation): stochastic sequences
 *   take p truncated to its nucleus, S_b = {x : p(x) >= tau_b} with tau_b the
 *   probability of the token at which the mass of p in descending order first
 *   reaches top_p[b] (tokens tied with it included), renormalised on S_b --
 *   for the accept test, the residual max(0, p - q) and the bonus draw alike
 *   (Sec. III-A samples the verifier's distribution for diversity; the paper
 *   fixes no truncation, this is the usual nucleus rule).  top_p[b] = 1 leaves
 *   p whole; a value outside (0, 1] is reported (SPADE_DEV_BAD_INDEX) and
 *   taken as 1.  Greedy sequences are unaffected.  tau_b is located by a
 *   four-round 32-bin search over integer keys of l / T (2^15 per unit of
 *   log-probability, from 31.5 below the row maximum), so tokens whose
 *   log-probability lies within one key step (3.1e-5) below the boundary
 *   token's may also be in S_b, and tokens more than 31.5 below the
 *   maximum (at most V e^-31.5 of p) never are.  Needs the one-launch path
 *   (spade_accept_launches == 1): SPADE_ERR_SHAPE otherwise.  The row
 *   statistics of spade_accept_stats_layout stay those of the whole p (the
 *   accept bit there is the untruncated test).
 * k_cache, v_cache, ctx_lens, Hkv, D, cap: as in spade_verify_accept_commit,
 *   or all three pointers null for no commit.
 * Every other argument is that of spade_verify_accept.
 */
spade_status spade_verify_accept_sampling(const void *hidden, const void *w_lm,
                                          const int32_t *draft_tokens, const float *draft_probs,
                                          const float *uniforms, const int32_t *mode,
                                          const float *temperature, const float *top_p,
                                          const int32_t *cu_q, const int32_t *n_draft,
                                          int32_t *accepted_len, int32_t *next_token, void *k_cache,
                                          void *v_cache, int32_t *ctx_lens, int32_t B, int32_t R,
                                          int32_t H, int32_t V, int32_t Hkv, int32_t D, int32_t cap,
                                          void *workspace, size_t workspace_bytes, int32_t *status,
                                          spade_stream_t stream);

/* Bytes of workspace spade_verify_accept needs (0 on invalid sizes). */
size_t spade_accept_workspace_size(int32_t B, int32_t R, int32_t H, int32_t V);

/*
 * Kernel launches one spade_verify_accept (or spade_verify_accept_commit) call
 * makes for these sizes on the current device: 1 when the logits of all R
 * rows stay on chip, 2 when they do not (a statistics pass over all rows --
 * on pairs of SMs sharing each MMA when the grid is even -- then a pass that
 * recomputes only the rows to sample); 0 on invalid sizes.  For launch
 * accounting and graph capture; no device work.
 */
int32_t spade_accept_launches(int32_t B, int32_t R, int32_t H, int32_t V);

/*
 * Where a completed spade_verify_accept (or spade_verify_accept_commit) call
 * leaves its merged per-row softmax statistics inside the workspace, for
 * tests and diagnostics that check the on-chip logits without writing them
 * out (Sec. III-A: p = softmax(o), o = g(x_L)).  For row r (0 <= r < R):
 *   float4 at byte row_stats_offset + 16 * r: x = max_x logits[r, x],
 *     y = sum_x exp(logits[r, x] - x-component), z = argmax_x logits[r, x]
 *     (int32 bits, lowest index on ties), w = accept bit of the row (int32
 *     bits; 1 iff the row's draft passed its test);
 *   float at byte draft_logit_offset + 4 * r: logits[r, d] of the row's draft
 *     token d (rows i < k_b only; other entries are not written).
 * The statistics are stored in several copies `replica_stride` float4 apart;
 * the first copy is the one described.  Valid until the next call that uses
 * the workspace.  Returns SPADE_ERR_INVALID_ARG on null outputs or bad sizes.
 */
spade_status spade_accept_stats_layout(int32_t B, int32_t R, int32_t H, int32_t V,
                                       size_t *row_stats_offset, size_t *draft_logit_offset,
                                       int32_t *replica_stride);

/*
 * spade_verify_accept followed by spade_kv_commit, in one launch: once the
 * accept decisions are taken on the device, the same kernel clears the
 * rejected draft slots [ctx_b + a_b + 1, ctx_b + n_draft[b]] of k_cache and
 * v_cache (every KV head) and advances ctx_lens[b] by a_b + 1, exactly as
 * spade_kv_commit does (Algorithm 1's context update), so a verify step needs
 * one launch fewer.  Arguments are those of the two calls:
 *   k_cache, v_cache bf16 [B, Hkv, cap, D], 16-byte aligned, D % 8 == 0,
 *                    updated in place
 *   ctx_lens         int32 [B], read and updated in place
 * Sequences with an invalid verify block are left untouched and reported in
 * `status` (SPADE_DEV_BAD_INDEX / SPADE_DEV_CAPACITY), as by spade_kv_commit.
 * The caller must not have another kernel reading the caches or ctx_lens
 * concurrently (the step's attention is ordered before this call on `stream`).
 */
spade_status spade_verify_accept_commit(const void *hidden, const void *w_lm,
                                        const int32_t *draft_tokens, const float *draft_probs,
                                        const float *uniforms, const int32_t *mode,
                                        const int32_t *cu_q, const int32_t *n_draft,
                                        int32_t *accepted_len, int32_t *next_token,
                                        void *k_cache, void *v_cache, int32_t *ctx_lens,
                                        int32_t B, int32_t R, int32_t H, int32_t V, int32_t Hkv,
                                        int32_t D, int32_t cap, void *workspace,
                                        size_t workspace_bytes, int32_t *status,
                                        spade_stream_t stream);

/* ------------------------------------------------------------------------ */
/* KV commit (Algorithm 1 context update)                                    */
/* ------------------------------------------------------------------------ */
/*
 * For every sequence b with a_b = accepted_len[b] (0 <= a_b <= n_draft[b]):
 * slots [ctx_b + a_b + 1, ctx_b + n_draft[b]] of k_cache and v_cache (every KV
 * head) are cleared to zero and ctx_lens[b] += a_b + 1 (the last accepted
 * token plus a_b drafts are now committed; the corrected / bonus token is
 * position 0 of the next verify block).
 *   k_cache, v_cache bf16 [B, Hkv, cap, D] updated in place
 *   ctx_lens         int32 [B] updated in place
 *   accepted_len     int32 [B];  n_draft int32 [B]
 *   status           device int32 (SPADE_DEV_BAD_INDEX if a_b is out of range,
 *                    SPADE_DEV_CAPACITY if the block exceeds cap; such a
 *                    sequence is left untouched)
 */
spade_status spade_kv_commit(void *k_cache, void *v_cache, int32_t *ctx_lens,
                             const int32_t *accepted_len, const int32_t *n_draft, int32_t B,
                             int32_t Hkv, int32_t D, int32_t cap, int32_t *status,
                             spade_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Paged KV cache                                                            */
/* ------------------------------------------------------------------------ */
/*
 * The same operations on a paged KV cache, for serving batches whose context
 * lengths differ widely: keys and values live in pools of fixed-size pages,
 *   k_pool, v_pool  bf16 [num_pages, Hkv, page_size, D] row-major, 16-byte aligned
 *   block_table     int32 [B, max_pages]: block_table[b * max_pages + j] is the
 *                   page that holds slots [j * page_size, (j + 1) * page_size)
 *                   of sequence b (every KV head), 0 <= page < num_pages;
 * so slot s of sequence b, KV head g, is row s % page_size of page
 * block_table[b][s / page_size], head g.  A sequence can use up to
 * max_pages * page_size slots (its capacity, the `cap` of the dense calls);
 * page_size is a multiple of 64 for the attention.  Only the table entries of
 * the pages a call touches are read; a touched entry outside [0, num_pages)
 * sets SPADE_DEV_BAD_INDEX (the attention reads zeros for it; the commit and
 * the QKV write skip that sequence).  Every other argument, and the result,
 * is that of the dense call of the same name (spade_verify_accept_commit_paged:
 * of spade_verify_accept_commit, the commit through the table), so a paged
 * verify step is two launches like a dense one.
 */
spade_status spade_verify_attention_paged(const void *q, const void *k_pool, const void *v_pool,
                                          const int32_t *block_table, const int32_t *ctx_lens,
                                          const int32_t *n_draft, const int32_t *cu_q, void *out,
                                          float *lse, int32_t B, int32_t Hq, int32_t Hkv, int32_t D,
                                          int32_t page_size, int32_t num_pages, int32_t max_pages,
                                          int32_t max_k, int32_t R, void *workspace,
                                          size_t workspace_bytes, int32_t *status,
                                          spade_stream_t stream);

spade_status spade_kv_commit_paged(void *k_pool, void *v_pool, const int32_t *block_table,
                                   int32_t *ctx_lens, const int32_t *accepted_len,
                                   const int32_t *n_draft, int32_t B, int32_t Hkv, int32_t D,
                                   int32_t page_size, int32_t num_pages, int32_t max_pages,
                                   int32_t *status, spade_stream_t stream);

spade_status spade_verify_accept_commit_paged(
    const void *hidden, const void *w_lm, const int32_t *draft_tokens, const float *draft_probs,
    const float *uniforms, const int32_t *mode, const int32_t *cu_q, const int32_t *n_draft,
    int32_t *accepted_len, int32_t *next_token, void *k_pool, void *v_pool, const int32_t *block_table,
    int32_t *ctx_lens, int32_t B, int32_t R, int32_t H, int32_t V, int32_t Hkv, int32_t D, int32_t page_size,
    int32_t num_pages, int32_t max_pages, void *workspace, size_t workspace_bytes, int32_t *status,
    spade_stream_t stream);

spade_status spade_verify_qkv_rope_paged(const void *x, const void *w_qkv, const int32_t *block_table,
                                         const int32_t *ctx_lens, const int32_t *n_draft,
                                         const int32_t *cu_q, void *q_out, void *k_pool, void *v_pool,
                                         int32_t B, int32_t R, int32_t H, int32_t Hq, int32_t Hkv,
                                         int32_t D, int32_t page_size, int32_t num_pages,
                                         int32_t max_pages, int32_t max_k, float rope_theta,
                                         void *workspace, size_t workspace_bytes, int32_t *status,
                                         spade_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Diagnostics                                                               */
/* ------------------------------------------------------------------------ */
const char *spade_status_string(spade_status s);
const char *spade_last_error(void);
/* Library version, e.g. "spade-gb300 0.1 sm_103a". */
const char *spade_version(void);

/*
 * Self-test of the device-side timeout path that every kernel above uses for
 * its waits: launches one CTA on `stream` whose thread waits on an mbarrier
 * that nothing completes.  After limit_us microseconds of %globaltimer
 * (1 .. 1000000) the wait gives up, SPADE_DEV_TIMEOUT is OR-ed into *status
 * (device int32) and the kernel returns normally, so the context stays
 * usable.  No other effect; for health checks and tests of status reporting.
 * Returns SPADE_ERR_INVALID_ARG for a null status or a limit out of range.
 */
spade_status spade_selftest_wait_timeout(int32_t *status, int32_t limit_us, spade_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SPADE_H_ */
