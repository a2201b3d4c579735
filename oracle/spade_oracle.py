"""Float64 CPU oracle of the SPADE verify step.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports this module:
only the tests, the smoke check and the CPU-baseline leg of the benchmark do.
It shares no code with the CUDA library and is deliberately plain and slow.

What it computes (the verifier side of one speculative-decoding iteration):

* ``verify_attention`` -- causal attention of the k+1 verify positions of each
  sequence against its KV cache (the verifier's single forward pass over the
  draft block, Sec. III-B "Verification Stage" and Algorithm 1, "Cloud: in
  parallel ... in a single forward pass"; the residual block x_{l+1} = x_l +
  f_l(x_l) of Sec. III-A contains this attention).
* ``lm_logits`` -- the LM head o = g(x_L) (Sec. III-A).
* ``verify_accept`` -- softmax of the logits (Sec. III-A), the acceptance
  probability alpha(x) = min(1, p(x)/q(x)) and the residual distribution
  p'(x) = norm(max(0, p(x) - q(x))) (Sec. III-C "Verification Criterion"),
  the longest accepted prefix and the correction token (Algorithm 1).
* ``kv_commit`` -- the context update m <- m + k + 1 of Algorithm 1 applied to
  a KV cache: accepted slots stay, rejected slots are cleared.
* ``paged_gather`` / ``kv_commit_paged`` / ``kv_write_paged`` -- the same cache
  operations on a paged cache (pools of fixed-size pages and a block table).
* ``verify_qkv_rope`` / ``kv_write`` -- the projection of the verify block's
  hidden states into queries, keys and values with rotary position embedding,
  and the write of its keys and values into the block's cache slots: the
  attention input side of f_l in x_{l+1} = x_l + f_l(x_l) (Sec. III-A) for the
  d+1 positions of the single forward pass (Sec. III-B).

Readings taken where the paper is silent (each also listed in the design
notes): greedy verification accepts a draft iff it equals the verifier's
argmax (lowest index on ties); the uniform u of position i decides acceptance
iff u < p/q (q(d) = 0 accepts iff p(d) > 0); when every draft is accepted a
bonus token is drawn from p of the last row; sampling is the inverse CDF in
ascending vocabulary order, the first x whose cumulative mass exceeds u*Z; a
residual with no positive finite mass falls back to p.  Rotary embedding (the
verifier family's positional encoding; the paper names the model, Sec. IV,
not its layers) pairs dimension j with j + D/2 and rotates the pair by
pos * theta^(-2j/D), counter-clockwise; verify position i of sequence b sits
at position ctx_b + i.

Inputs are numpy arrays.  Floating inputs are the exact values of the bf16 /
fp32 tensors handed to the GPU, converted to float64 before any arithmetic.
"""
from __future__ import annotations

import math

import numpy as np

GREEDY = 0
STOCHASTIC = 1


def _f64(x):
    return np.asarray(x, dtype=np.float64)


# ----------------------------------------------------------------------------
# Attention (Sec. III-B verification stage; Algorithm 1 cloud step)
# ----------------------------------------------------------------------------
def attention_row(qv, K, V):
    """softmax(q K^T / sqrt(D)) V for one query vector over the keys given.

    Returns (o, lse) with lse the natural-log log-sum-exp of the scaled scores.
    """
    qv = _f64(qv)
    K = _f64(K)
    V = _f64(V)
    s = K @ qv / math.sqrt(qv.shape[-1])
    m = s.max()
    w = np.exp(s - m)
    den = w.sum()
    return (w @ V) / den, m + math.log(den)


def verify_attention(q, k_cache, v_cache, ctx_lens, n_draft, cu_q, rows=None):
    """Verify attention of every (row, head), or of the (row, head) pairs in ``rows``.

    q [R, Hq, D]; k_cache, v_cache [B, Hkv, cap, D]; ctx_lens, n_draft [B];
    cu_q [B+1] with row cu_q[b]+i holding position i (0 <= i <= k_b) of
    sequence b.  Position i sees keys 0 .. ctx_b + i (the committed context plus
    the draft block up to itself); query head h reads KV head h // (Hq/Hkv).
    Returns (out [R, Hq, D], lse [R, Hq]) in float64; with ``rows`` given only
    those entries are filled (the rest stay NaN).
    """
    q = np.asarray(q)
    R, Hq, D = q.shape
    B, Hkv = k_cache.shape[0], k_cache.shape[1]
    G = Hq // Hkv
    out = np.full((R, Hq, D), np.nan)
    lse = np.full((R, Hq), np.nan)
    row_seq = np.empty(R, dtype=np.int64)
    row_pos = np.empty(R, dtype=np.int64)
    for b in range(B):
        for i in range(int(n_draft[b]) + 1):
            row_seq[cu_q[b] + i] = b
            row_pos[cu_q[b] + i] = i
    pairs = rows if rows is not None else [(r, h) for r in range(R) for h in range(Hq)]
    for r, h in pairs:
        b = row_seq[r]
        last = int(ctx_lens[b]) + int(row_pos[r])
        kvh = h // G
        o, l = attention_row(q[r, h], k_cache[b, kvh, :last + 1], v_cache[b, kvh, :last + 1])
        out[r, h] = o
        lse[r, h] = l
    return out, lse


# ----------------------------------------------------------------------------
# LM head and softmax (Sec. III-A)
# ----------------------------------------------------------------------------
def lm_logits(hidden, w_lm, chunk=8192):
    """o = g(x_L): logits[r, x] = sum_j hidden[r, j] * W[x, j], float64."""
    h = _f64(hidden)
    V = w_lm.shape[0]
    out = np.empty((h.shape[0], V))
    for v0 in range(0, V, chunk):
        out[:, v0:v0 + chunk] = h @ _f64(w_lm[v0:v0 + chunk]).T
    return out


def softmax(logits):
    """P(y | prefix) = softmax(o) (Sec. III-A), temperature 1."""
    l = _f64(logits)
    e = np.exp(l - l.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def acceptance_probability(p_x, q_x):
    """alpha(x) = min(1, p(x)/q(x)) (Sec. III-C)."""
    if q_x <= 0.0:
        return 1.0 if p_x > 0.0 else 0.0
    return min(1.0, p_x / q_x)


def residual_distribution(p, q):
    """p'(x) = norm(max(0, p(x) - q(x))) (Sec. III-C), unnormalised mass and Z.

    Returns (r, Z, fell_back).  If the residual has no positive finite mass,
    it is replaced by p (reading for float or malformed q).
    """
    r = np.maximum(0.0, _f64(p) - _f64(q))
    Z = r.sum()
    if not (Z > 0.0 and np.isfinite(Z)):
        r = _f64(p).copy()
        return r, r.sum(), True
    return r, Z, False


def inverse_cdf(r, Z, u):
    """Smallest x with sum_{y<=x} r(y) > u*Z (ascending vocabulary order).

    Returns (x, margin) where margin is the distance of u*Z to the nearer edge
    of x's CDF interval divided by r(x) (0.5 = dead centre, 0 = on an edge).
    If rounding leaves u*Z beyond the total, the last x with r > 0 is taken.
    """
    c = np.cumsum(r)
    T = u * Z
    hit = np.nonzero(c > T)[0]
    pos = np.nonzero(r > 0)[0]
    x = int(hit[0]) if hit.size else int(pos[-1])
    lo = c[x] - r[x]
    margin = min(T - lo, c[x] - T) / r[x] if r[x] > 0 else 0.0
    return x, margin


def nucleus(p, top_p):
    """Top-p truncation of a distribution (sampling "for diversity", Sec. III-A, left open
    by the paper): S = {x : p(x) >= tau}, tau the probability of the token at which the
    cumulative mass in descending order first reaches top_p (tokens tied with it included);
    returns (p on S renormalised, mass margin, log gap): the distance of top_p to the nearer
    end of the boundary token's step of the cumulative mass, and ln p of the boundary token
    minus ln p of the next one (small values: a boundary that rounding could move)."""
    p = _f64(p)
    if top_p >= 1.0:
        return p, np.inf, np.inf
    order = np.argsort(-p, kind="stable")
    c = np.cumsum(p[order])
    j = int(np.nonzero(c >= top_p)[0][0]) if np.any(c >= top_p) else len(p) - 1
    tau = p[order[j]]
    keep = p >= tau
    pt = np.where(keep, p, 0.0)
    pt = pt / pt.sum()
    below = c[j - 1] if j > 0 else 0.0
    nxt = p[order[j + 1]] if j + 1 < len(p) else 0.0
    gap = np.log(tau) - np.log(nxt) if nxt > 0 else np.inf
    return pt, min(c[j] - top_p, top_p - below), gap


def _top2_margin(l):
    top = np.partition(l, -2)[-2:] if l.shape[0] > 1 else np.array([-np.inf, l[0]])
    return float(top[1] - top[0])


def verify_accept(logits, draft_tokens, draft_probs, uniforms, mode, cu_q, n_draft,
                  margin=1e-3, temperature=None, top_p=None, logit_rel_err=1.5e-5):
    """Accept/reject of every sequence, given its verifier logits.

    logits [R, V] (rows as in ``verify_attention``); draft_tokens [R-B] with
    draft i of sequence b at index cu_q[b] - b + i; draft_probs [R-B, V] (q of
    the draft model at the same positions, may be None if no sequence is
    stochastic); uniforms [R]: u[cu_q[b]+i] is the accept test of draft i,
    u[cu_q[b]+k_b] the sampling uniform; mode [B] 0 greedy / 1 stochastic.

    Returns dict with accepted_len [B], next_token [B] and diagnostics:
      flag_decision [B]  some decided position has top-2 logit margin (greedy)
                         or |u - p/q| (stochastic) below ``margin``;
      flag_sample [B]    the sampled token's u*Z lies within margin*r(x) of an
                         edge of its CDF interval, or within the spread that
                         logit errors give the cumulative mass (below; stochastic
                         only);
      fallback [B]       residual had no mass, p used instead.

    ``temperature`` [B] (optional): the verifier samples from p = softmax(l / T_b)
    (the paper mentions sampling for diversity, Sec. III-A, without fixing it);
    greedy decisions, which take the argmax, are unaffected.  ``logit_rel_err``: the
    error a computed logit l may carry, as a fraction of max(1, |l|) (fp32 sums of a bf16
    product over the hidden size); each term of p then moves by p_x times that error and
    the cumulative mass at a draw's edges by about
    sqrt(sum over the tokens with mass of (p_x * logit_rel_err * max(1, |l_x / T|))^2),
    so a draw that close to an edge is flagged too.  ``top_p`` [B] (optional): p is
    then truncated to its nucleus (``nucleus``) for stochastic sequences; a nucleus boundary
    within the margin (1e-3 of mass, 1e-4 of log probability) at a deciding row flags the
    sequence's decision.
    """
    B = len(n_draft)
    acc = np.zeros(B, dtype=np.int64)
    tok = np.zeros(B, dtype=np.int64)
    flag_dec = np.zeros(B, dtype=bool)
    flag_smp = np.zeros(B, dtype=bool)
    fallback = np.zeros(B, dtype=bool)
    for b in range(B):
        k = int(n_draft[b])
        r0 = int(cu_q[b])
        d0 = r0 - b
        stochastic = int(mode[b]) == STOCHASTIC
        t_b = 1.0 if temperature is None else float(temperature[b])
        tp_b = 1.0 if top_p is None else float(top_p[b])

        def dist(l_row):
            pn, mass_margin, log_gap = nucleus(softmax(l_row / t_b), tp_b)
            if mass_margin < margin or log_gap < 0.1 * margin:
                flag_dec[b] = True
            return pn

        a = 0
        for i in range(k):
            l = _f64(logits[r0 + i])
            d = int(draft_tokens[d0 + i])
            if not stochastic:
                ok = d == int(np.argmax(l))
                if _top2_margin(l) < margin:
                    flag_dec[b] = True
            else:
                p = dist(l)
                qd = float(draft_probs[d0 + i][d])
                u = float(uniforms[r0 + i])
                if qd > 0.0:
                    ratio = p[d] / qd
                    ok = u < ratio
                    if abs(u - ratio) < margin:
                        flag_dec[b] = True
                else:
                    ok = p[d] > 0.0
            if not ok:
                break
            a += 1
        acc[b] = a
        lr = _f64(logits[r0 + a])
        if not stochastic:
            tok[b] = int(np.argmax(lr))
            if _top2_margin(lr) < margin:
                flag_dec[b] = True
        else:
            p = dist(lr)
            if a < k:
                r, Z, fb = residual_distribution(p, draft_probs[d0 + a])
            else:
                r, Z, fb = p, p.sum(), False
            fallback[b] = fb
            x, m = inverse_cdf(r, Z, float(uniforms[r0 + k]))
            tok[b] = x
            # Two ways a draw sits on an edge: u*Z within margin * r(x) of one (a
            # relative measure), or within the spread of the cumulative mass when
            # each logit carries its own error (a peaked row moves its edges that
            # far even when the drawn token's own interval is tiny).
            lt = lr / t_b
            terms = np.where(r > 0, p * logit_rel_err * np.maximum(1.0, np.abs(lt)), 0.0)
            spread = float(np.sqrt(np.sum(terms ** 2)))
            if m < margin or m * r[x] < spread:
                flag_smp[b] = True
    return dict(accepted_len=acc, next_token=tok, flag_decision=flag_dec,
                flag_sample=flag_smp, fallback=fallback)


def verify_accept_from_hidden(hidden, w_lm, *args, **kw):
    """``verify_accept`` on logits computed by ``lm_logits`` (the full step)."""
    return verify_accept(lm_logits(hidden, w_lm), *args, **kw)


# ----------------------------------------------------------------------------
# KV commit (Algorithm 1 context update)
# ----------------------------------------------------------------------------
def kv_commit(k_cache, v_cache, ctx_lens, accepted_len, n_draft):
    """Append the accepted positions and roll back the rejected ones.

    The verify block of sequence b occupies cache slots ctx_b .. ctx_b + k_b.
    After acceptance of a_b drafts the committed context is ctx_b + a_b + 1
    (last accepted token + a_b drafts); slots ctx_b + a_b + 1 .. ctx_b + k_b
    are cleared to zero.  Returns new (k_cache, v_cache, ctx_lens) copies.
    """
    k = np.array(k_cache, copy=True)
    v = np.array(v_cache, copy=True)
    ctx = np.array(ctx_lens, dtype=np.int64, copy=True)
    for b in range(len(ctx)):
        a = int(accepted_len[b])
        lo = int(ctx[b]) + a + 1
        hi = int(ctx[b]) + int(n_draft[b]) + 1
        k[b, :, lo:hi] = 0
        v[b, :, lo:hi] = 0
        ctx[b] = lo
    return k, v, ctx


# ----------------------------------------------------------------------------
# QKV projection + rotary embedding of the verify block (Sec. III-A/III-B)
# ----------------------------------------------------------------------------
def rope_inv_freq(D, theta):
    """Rotary frequencies theta^(-2j/D), j = 0 .. D/2 - 1."""
    return float(theta) ** (-2.0 * np.arange(D // 2) / D)


def rope(x, pos, theta):
    """Rotary position embedding of vectors x [..., D] at positions pos (broadcast to
    x.shape[:-1]): the pair (x_j, x_{j+D/2}) is rotated counter-clockwise by the angle
    pos * theta^(-2j/D)."""
    x = _f64(x)
    h = x.shape[-1] // 2
    ang = np.asarray(pos, dtype=np.float64)[..., None] * rope_inv_freq(x.shape[-1], theta)
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :h], x[..., h:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def verify_positions(ctx_lens, n_draft, cu_q):
    """(sequence, position) of every verify row: row cu_q[b] + i is position ctx_b + i."""
    R = int(cu_q[len(n_draft)])
    seq = np.empty(R, dtype=np.int64)
    pos = np.empty(R, dtype=np.int64)
    for b in range(len(n_draft)):
        for i in range(int(n_draft[b]) + 1):
            seq[int(cu_q[b]) + i] = b
            pos[int(cu_q[b]) + i] = int(ctx_lens[b]) + i
    return seq, pos


def verify_qkv_rope(x, w_qkv, ctx_lens, n_draft, cu_q, Hq, Hkv, theta):
    """Queries, keys and values of the verify block.

    x [R, H] hidden states of the verify rows; w_qkv [(Hq + 2 Hkv) D, H] (nn.Linear
    layout: the query heads' rows, then the key heads', then the value heads').
    y = x W^T; q and k are rotated at each row's position (ctx_b + i), v is not.
    Returns (q [R, Hq, D], k [R, Hkv, D], v [R, Hkv, D]) in float64.
    """
    y = _f64(x) @ _f64(w_qkv).T
    R = y.shape[0]
    D = w_qkv.shape[0] // (Hq + 2 * Hkv)
    q = y[:, :Hq * D].reshape(R, Hq, D)
    k = y[:, Hq * D:(Hq + Hkv) * D].reshape(R, Hkv, D)
    v = y[:, (Hq + Hkv) * D:].reshape(R, Hkv, D)
    _, pos = verify_positions(ctx_lens, n_draft, cu_q)
    return rope(q, pos[:, None], theta), rope(k, pos[:, None], theta), v


def kv_write(k_cache, v_cache, k, v, ctx_lens, n_draft, cu_q):
    """Writes the verify block's keys and values into cache slots ctx_b .. ctx_b + k_b
    of their sequence (every KV head); returns new (k_cache, v_cache) copies."""
    kc = np.array(k_cache, dtype=np.float64, copy=True)
    vc = np.array(v_cache, dtype=np.float64, copy=True)
    seq, pos = verify_positions(ctx_lens, n_draft, cu_q)
    for r in range(len(seq)):
        kc[seq[r], :, pos[r]] = k[r]
        vc[seq[r], :, pos[r]] = v[r]
    return kc, vc


# ----------------------------------------------------------------------------
# Paged KV cache: pools [num_pages, Hkv, page, D] and a block table [B, max_pages]
# ----------------------------------------------------------------------------
def paged_slot(block_table, b, s, page):
    """(page id, row in the page) of slot s of sequence b."""
    return int(block_table[b][s // page]), s % page


def paged_gather(pool, block_table, n_slots, page):
    """Dense view [B, Hkv, n_slots, D] of a paged pool: slot s of sequence b is row
    s % page of page block_table[b][s // page]."""
    pool = np.asarray(pool)
    B = len(block_table)
    out = np.zeros((B, pool.shape[1], n_slots, pool.shape[3]), dtype=np.float64)
    for b in range(B):
        for s in range(n_slots):
            pg, r = paged_slot(block_table, b, s, page)
            out[b, :, s] = pool[pg, :, r]
    return out


def kv_commit_paged(k_pool, v_pool, block_table, ctx_lens, accepted_len, n_draft, page):
    """``kv_commit`` on a paged cache: the rejected slots ctx_b + a_b + 1 .. ctx_b + k_b of
    sequence b are cleared where the block table puts them; returns new (k_pool, v_pool,
    ctx_lens) copies."""
    k = np.array(k_pool, dtype=np.float64, copy=True)
    v = np.array(v_pool, dtype=np.float64, copy=True)
    ctx = np.array(ctx_lens, dtype=np.int64, copy=True)
    for b in range(len(ctx)):
        lo = int(ctx[b]) + int(accepted_len[b]) + 1
        for s in range(lo, int(ctx[b]) + int(n_draft[b]) + 1):
            pg, r = paged_slot(block_table, b, s, page)
            k[pg, :, r] = 0
            v[pg, :, r] = 0
        ctx[b] = lo
    return k, v, ctx


def kv_write_paged(k_pool, v_pool, block_table, k, v, ctx_lens, n_draft, cu_q, page):
    """``kv_write`` on a paged cache; returns new (k_pool, v_pool) copies."""
    kp = np.array(k_pool, dtype=np.float64, copy=True)
    vp = np.array(v_pool, dtype=np.float64, copy=True)
    seq, pos = verify_positions(ctx_lens, n_draft, cu_q)
    for r in range(len(seq)):
        pg, row = paged_slot(block_table, int(seq[r]), int(pos[r]), page)
        kp[pg, :, row] = k[r]
        vp[pg, :, row] = v[r]
    return kp, vp
