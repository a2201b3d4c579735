"""Pins of the float64 oracle against facts fixed by the paper and by mathematics.

Each ``check_*`` takes an oracle module and raises AssertionError when the
module disagrees with a fact that does not come from the oracle itself:
hand-derived worked examples, closed forms, a textbook library routine
(torch's scaled_dot_product_attention in float64), the output-equivalence
theorem of speculative decoding (Sec. III-B/III-C: greedy SD reproduces plain
argmax decoding token for token, rejection sampling reproduces p), and the
invariants of Algorithm 1.  ``test_oracle_pins.py`` runs them on the oracle;
``test_oracle_mutants.py`` runs them on copies of the oracle with planted
mistakes and requires that each mistake is caught.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np
import torch
from scipy import stats

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "worked_examples.json")


def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def _ln(s):
    return math.log(float(s.split()[1]))


# ----------------------------------------------------------------------------
# Attention
# ----------------------------------------------------------------------------
def _single_seq_cache(K, V):
    K = np.asarray(K, dtype=np.float64)[None, None]
    V = np.asarray(V, dtype=np.float64)[None, None]
    return K, V


def check_attention_worked_examples(o):
    for ex in _golden()["attention"]:
        K, V = _single_seq_cache(ex["K"], ex["V"])
        q = np.asarray(ex["q"], dtype=np.float64)[:, None, :]
        out, lse = o.verify_attention(q, K, V, [ex["ctx"]], [ex["k"]], [0, ex["k"] + 1])
        np.testing.assert_allclose(out[:, 0], np.asarray(ex["out"]), rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse[:, 0], [_ln(s) for s in ex["lse"]], rtol=0, atol=1e-12)


def _random_attention_case(rng, B, Hq, Hkv, D, ctx, kd, extra=3):
    cap = max(c + k + 1 for c, k in zip(ctx, kd)) + extra
    cu = np.concatenate([[0], np.cumsum(np.asarray(kd) + 1)])
    R = int(cu[-1])
    q = rng.standard_normal((R, Hq, D))
    kc = rng.standard_normal((B, Hkv, cap, D))
    vc = rng.standard_normal((B, Hkv, cap, D))
    return q, kc, vc, cu


def _sdpa_reference(q, kc, vc, ctx, kd, cu):
    """torch SDPA in float64 with an explicit boolean mask and GQA by repeat."""
    R, Hq, D = q.shape
    B, Hkv, cap, _ = kc.shape
    G = Hq // Hkv
    out = np.zeros((R, Hq, D))
    for b in range(B):
        rows = slice(int(cu[b]), int(cu[b + 1]))
        nq = int(kd[b]) + 1
        qb = torch.from_numpy(q[rows]).permute(1, 0, 2)              # [Hq, nq, D]
        kb = torch.from_numpy(kc[b]).repeat_interleave(G, dim=0)     # [Hq, cap, D]
        vb = torch.from_numpy(vc[b]).repeat_interleave(G, dim=0)
        mask = torch.zeros((nq, cap), dtype=torch.bool)
        for i in range(nq):
            mask[i, : int(ctx[b]) + i + 1] = True
        ob = torch.nn.functional.scaled_dot_product_attention(qb, kb, vb, attn_mask=mask)
        out[rows] = ob.permute(1, 0, 2).numpy()
    return out


def check_attention_vs_sdpa(o, seed=0):
    rng = np.random.default_rng(seed)
    for (B, Hq, Hkv, D, ctx, kd) in [(2, 4, 2, 8, [5, 3], [2, 3]),
                                    (3, 6, 3, 16, [0, 7, 1], [4, 0, 1]),
                                    (1, 2, 1, 4, [9], [5])]:
        q, kc, vc, cu = _random_attention_case(rng, B, Hq, Hkv, D, ctx, kd)
        got, _ = o.verify_attention(q, kc, vc, ctx, kd, cu)
        ref = _sdpa_reference(q, kc, vc, ctx, kd, cu)
        np.testing.assert_allclose(got, ref, rtol=1e-10, atol=1e-12)


def check_attention_special_cases(o, seed=1):
    rng = np.random.default_rng(seed)
    D = 8
    # k = 0: plain decode attention, the single query sees all ctx+1 keys.
    q, kc, vc, cu = _random_attention_case(rng, 1, 2, 2, D, [6], [0])
    got, _ = o.verify_attention(q, kc, vc, [6], [0], cu)
    for h in range(2):
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[:, h][None]), torch.from_numpy(kc[0, h, :7][None]),
            torch.from_numpy(vc[0, h, :7][None]))
        np.testing.assert_allclose(got[:, h], ref[0].numpy(), rtol=1e-10, atol=1e-12)
    # ctx = 0: causal self-attention over the verify block alone.
    q, kc, vc, cu = _random_attention_case(rng, 1, 2, 2, D, [0], [4])
    got, _ = o.verify_attention(q, kc, vc, [0], [4], cu)
    for h in range(2):
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[:, h][None]), torch.from_numpy(kc[0, h, :5][None]),
            torch.from_numpy(vc[0, h, :5][None]), is_causal=True)
        np.testing.assert_allclose(got[:, h], ref[0].numpy(), rtol=1e-10, atol=1e-12)
    # q = 0: the output is the mean of the visible values (mask width ctx+i+1).
    ctx, kd = [5], [3]
    q, kc, vc, cu = _random_attention_case(rng, 1, 2, 1, D, ctx, kd)
    q[:] = 0.0
    got, lse = o.verify_attention(q, kc, vc, ctx, kd, cu)
    for i in range(4):
        np.testing.assert_allclose(got[i, 0], vc[0, 0, : ctx[0] + i + 1].mean(0), rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse[i, 1], math.log(ctx[0] + i + 1), rtol=0, atol=1e-12)


def check_attention_gqa_mapping(o):
    # Values constant per KV head: query head h must read KV head h // G.
    B, Hq, Hkv, D, ctx, kd = 1, 6, 3, 4, [3], [2]
    rng = np.random.default_rng(2)
    q, kc, vc, cu = _random_attention_case(rng, B, Hq, Hkv, D, ctx, kd)
    for j in range(Hkv):
        vc[0, j] = float(j + 1)
    got, _ = o.verify_attention(q, kc, vc, ctx, kd, cu)
    for h in range(Hq):
        np.testing.assert_allclose(got[:, h], float(h // (Hq // Hkv) + 1), rtol=0, atol=1e-12)


# ----------------------------------------------------------------------------
# LM head
# ----------------------------------------------------------------------------
def check_logits_one_hot(o):
    rng = np.random.default_rng(3)
    V, H = 11, 5
    W = rng.standard_normal((V, H))
    hidden = np.eye(H)
    got = o.lm_logits(hidden, W, chunk=4)
    np.testing.assert_array_equal(got, W.T)
    got2 = o.lm_logits(2.0 * hidden[[1, 3]], W, chunk=3)
    np.testing.assert_array_equal(got2, 2.0 * W.T[[1, 3]])


# ----------------------------------------------------------------------------
# Acceptance / residual (Sec. III-C)
# ----------------------------------------------------------------------------
def check_acceptance_worked_examples(o):
    g = _golden()
    for ex in g["acceptance_residual"]:
        p, q = np.asarray(ex["p"]), np.asarray(ex["q"])
        for x in range(len(p)):
            assert abs(o.acceptance_probability(p[x], q[x]) - ex["alpha"][x]) < 1e-15
        r, Z, fb = o.residual_distribution(p, q)
        assert not fb
        np.testing.assert_allclose(r, ex["residual_unnormalised"], rtol=0, atol=1e-15)
        np.testing.assert_allclose(r / Z, ex["residual"], rtol=0, atol=1e-15)
    ic = g["inverse_cdf"]
    r = np.asarray(ic["r"])
    for u, x in ic["cases"]:
        assert o.inverse_cdf(r, r.sum(), u)[0] == x, (u, x)
    ga = g["greedy_argmax"]
    lg = np.asarray(ga["logits"])[None]
    res = o.verify_accept(np.repeat(lg, 2, 0), [ga["argmax"]], None, [0.5, 0.5], [0], [0, 2], [1])
    assert res["accepted_len"][0] == 1 and res["next_token"][0] == ga["argmax"]
    res = o.verify_accept(np.repeat(lg, 2, 0), [2], None, [0.5, 0.5], [0], [0, 2], [1])
    assert res["accepted_len"][0] == 0 and res["next_token"][0] == ga["argmax"]


def check_margin_worked_examples(o):
    """Flags of the parity rule on hand-derived cases: greedy top-2 gap and stochastic
    |u - p/q| below 1e-3 at a deciding position, the sampled token's edge margin, and
    no flag from rows after the first rejection."""
    g = _golden()["decision_margins"]
    thr = g["threshold"]
    for ex in g["greedy"]:
        k = ex["k"]
        res = o.verify_accept(np.asarray(ex["logits"]), ex["draft"], None, np.full(k + 1, 0.5), [0],
                              [0, k + 1], [k], margin=thr)
        assert res["accepted_len"][0] == ex["accepted"], ex["about"]
        assert res["next_token"][0] == ex["next"], ex["about"]
        assert bool(res["flag_decision"][0]) == ex["flag_decision"], ex["about"]
        assert not res["flag_sample"][0], ex["about"]
    for ex in g["stochastic"]:
        k = ex["k"]
        q = np.asarray(ex["q"]).reshape(k, -1) if k else np.zeros((0, len(ex["p"][0])))
        res = o.verify_accept(np.log(np.asarray(ex["p"])), ex["draft"], q, ex["u"], [1], [0, k + 1], [k],
                              margin=thr)
        assert res["accepted_len"][0] == ex["accepted"], ex["about"]
        assert res["next_token"][0] == ex["next"], ex["about"]
        assert bool(res["flag_decision"][0]) == ex["flag_decision"], ex["about"]
        assert bool(res["flag_sample"][0]) == ex["flag_sample"], ex["about"]
    for ex in g["sampling_margin"]["cases"]:
        r = np.asarray(ex["r"])
        x, m = o.inverse_cdf(r, r.sum(), ex["u"])
        assert x == ex["x"], ex["why"]
        assert abs(m - ex["margin"]) < 1e-9, (ex["why"], m)


def check_sample_spread_worked_examples(o):
    """The sampled-token flag from the spread logit errors give the cumulative mass: hand-derived
    bonus draws (k = 0) that the relative edge margin alone does not flag, a control, a row
    where only tokens with mass may count, and one where the logits' magnitude decides."""
    g = _golden()["sample_spread"]
    for ex in g["cases"]:
        res = o.verify_accept(np.asarray([ex["logits"]], dtype=np.float64), [], np.zeros((0, len(ex["logits"]))),
                              [ex["u"]], [1], [0, 1], [0], logit_rel_err=g["logit_rel_err"])
        assert res["next_token"][0] == ex["next"], ex["about"]
        assert bool(res["flag_sample"][0]) == ex["flag_sample"], ex["about"]
        assert not res["flag_decision"][0], ex["about"]


def check_residual_properties(o, seed=4):
    rng = np.random.default_rng(seed)
    for _ in range(50):
        V = int(rng.integers(2, 40))
        p = rng.dirichlet(np.ones(V) * 0.5)
        q = rng.dirichlet(np.ones(V) * 0.5)
        r, Z, fb = o.residual_distribution(p, q)
        assert not fb
        assert (r >= 0).all()
        assert abs((r / Z).sum() - 1.0) < 1e-12
        assert (r[q >= p] == 0).all()
        # Z equals the total variation distance = 1 - sum(min(p, q)).
        assert abs(Z - (1.0 - np.minimum(p, q).sum())) < 1e-12
    # q == p: no residual mass, p is used.
    p = rng.dirichlet(np.ones(7))
    r, Z, fb = o.residual_distribution(p, p)
    assert fb and np.allclose(r, p)


def _uniform_logits_rows(p_rows, scale=1.0):
    return np.log(np.asarray(p_rows)) * scale


def check_q_equals_p_accepts_all(o, seed=5):
    rng = np.random.default_rng(seed)
    V, k, B = 9, 4, 200
    P = rng.dirichlet(np.ones(V), size=k + 1)
    logits = np.tile(np.log(P), (B, 1))
    q = np.tile(P[:k], (B, 1))
    drafts = np.concatenate([[rng.choice(V, p=P[i]) for i in range(k)] for _ in range(B)])
    u = rng.random(B * (k + 1)) * 0.999999
    cu = np.arange(B + 1) * (k + 1)
    res = o.verify_accept(logits, drafts, q, u, np.ones(B, int), cu, np.full(B, k))
    assert (res["accepted_len"] == k).all()


def check_strict_comparison(o):
    # u exactly equal to p/q must reject (accept iff u < p/q).
    p = np.array([0.5, 0.25, 0.25])
    q = np.array([0.5, 0.5, 0.0])
    logits = np.log(np.stack([p, p]))
    res = o.verify_accept(logits, [1], q[None], [0.5, 0.3], [1], [0, 2], [1])
    assert res["accepted_len"][0] == 0
    res = o.verify_accept(logits, [1], q[None], [0.4999999, 0.3], [1], [0, 2], [1])
    assert res["accepted_len"][0] == 1
    # q(d) = 0 with p(d) > 0 accepts whatever u is.
    q2 = np.array([[0.5, 0.5, 0.0]])
    res = o.verify_accept(logits, [2], q2, [0.99, 0.3], [1], [0, 2], [1])
    assert res["accepted_len"][0] == 1


def _stochastic_trials(o, P, Q, n, seed):
    """n independent verify steps of one sequence with fixed p rows P[0..k], q rows Q[0..k-1]."""
    rng = np.random.default_rng(seed)
    k, V = Q.shape
    drafts = np.stack([rng.choice(V, size=n, p=Q[i]) for i in range(k)], axis=1).reshape(-1)
    u = rng.random(n * (k + 1))
    logits = np.tile(np.log(P), (n, 1))
    q = np.tile(Q, (n, 1))
    cu = np.arange(n + 1) * (k + 1)
    res = o.verify_accept(logits, drafts, q, u, np.ones(n, int), cu, np.full(n, k))
    return drafts.reshape(n, k), res


def check_stochastic_output_law(o, n=60000, seed=6):
    """Rejection sampling reproduces the verifier's distribution (Sec. III-B/III-C).

    The first emitted token must follow p_0; the token emitted at position 1
    (given at least one acceptance) p_1; the bonus token (all k accepted) p_k.
    """
    rng = np.random.default_rng(seed)
    V, k = 8, 2
    P = rng.dirichlet(np.ones(V) * 0.7, size=k + 1)
    Q = rng.dirichlet(np.ones(V) * 0.7, size=k)
    drafts, res = _stochastic_trials(o, P, Q, n, seed + 100)
    a, t = res["accepted_len"], res["next_token"]
    first = np.where(a >= 1, drafts[:, 0], t)
    _, pv = stats.chisquare(np.bincount(first, minlength=V), P[0] * n)
    assert pv > 1e-3, ("first token law", pv)
    sel = a >= 1
    second = np.where(a[sel] >= 2, drafts[sel, 1], t[sel])
    _, pv = stats.chisquare(np.bincount(second, minlength=V), P[1] * sel.sum())
    assert pv > 1e-3, ("second token law", pv)
    sel = a == k
    _, pv = stats.chisquare(np.bincount(t[sel], minlength=V), P[k] * sel.sum())
    assert pv > 1e-3, ("bonus token law", pv)
    # Acceptance of draft 0 has probability sum_x min(p_0(x), q_0(x)).
    pacc = np.minimum(P[0], Q[0]).sum()
    n_acc = int((a >= 1).sum())
    assert stats.binomtest(n_acc, n, pacc).pvalue > 1e-3, (n_acc / n, pacc)


def check_progress_and_bounds(o, seed=7):
    rng = np.random.default_rng(seed)
    V, k = 6, 3
    P = rng.dirichlet(np.ones(V), size=k + 1)
    Q = rng.dirichlet(np.ones(V), size=k)
    _, res = _stochastic_trials(o, P, Q, 3000, seed)
    a = res["accepted_len"]
    assert ((a >= 0) & (a <= k)).all()
    assert ((res["next_token"] >= 0) & (res["next_token"] < V)).all()


# ----------------------------------------------------------------------------
# Greedy speculative decoding == plain argmax decoding (Sec. III-B)
# ----------------------------------------------------------------------------
class _ToyLM:
    """A deterministic toy language model: hidden state of a prefix -> logits."""

    def __init__(self, V, H, seed):
        rng = np.random.default_rng(seed)
        self.E1 = rng.standard_normal((V, H))
        self.E2 = rng.standard_normal((V, H)) * 0.5
        self.P = rng.standard_normal((7, H)) * 0.3
        self.W = rng.standard_normal((V, H))

    def hidden(self, prefix):
        prev = prefix[-2] if len(prefix) > 1 else 0
        return self.E1[prefix[-1]] + self.E2[prev] + self.P[len(prefix) % 7]


def check_greedy_identity(o, seed=8):
    V, H = 16, 8
    verifier = _ToyLM(V, H, seed)
    drafter = _ToyLM(V, H, seed + 1)
    drafter.W = verifier.W + 0.8 * np.random.default_rng(seed + 2).standard_normal((V, H))
    prompt = [3, 1, 4]
    n_new = 60
    # Plain greedy decoding with the verifier alone.
    ref = list(prompt)
    while len(ref) < len(prompt) + n_new:
        ref.append(int(np.argmax(verifier.W @ verifier.hidden(ref))))
    for d in (1, 3, 5):
        y = list(prompt)
        calls = 0
        while len(y) < len(prompt) + n_new:
            drafts = []
            for _ in range(d):
                drafts.append(int(np.argmax(drafter.W @ drafter.hidden(y + drafts))))
            hid = np.stack([verifier.hidden(y + drafts[:i]) for i in range(d + 1)])
            res = o.verify_accept(o.lm_logits(hid, verifier.W), drafts, None,
                                  np.full(d + 1, 0.5), [0], [0, d + 1], [d])
            a = int(res["accepted_len"][0])
            y += drafts[:a] + [int(res["next_token"][0])]
            calls += 1
        assert y[: len(ref)] == ref, (d, y[:len(ref)], ref)
        assert calls <= n_new


# ----------------------------------------------------------------------------
# KV commit (Algorithm 1 context update)
# ----------------------------------------------------------------------------
def check_kv_commit(o, seed=9):
    rng = np.random.default_rng(seed)
    B, Hkv, D = 4, 2, 3
    ctx = np.array([5, 0, 3, 7])
    kd = np.array([3, 2, 0, 4])
    acc = np.array([1, 2, 0, 0])
    cap = 14
    kc = rng.standard_normal((B, Hkv, cap, D)) + 5.0
    vc = rng.standard_normal((B, Hkv, cap, D)) + 5.0
    k2, v2, c2 = o.kv_commit(kc, vc, ctx, acc, kd)
    np.testing.assert_array_equal(c2, ctx + acc + 1)
    for b in range(B):
        for s in range(cap):
            cleared = ctx[b] + acc[b] + 1 <= s <= ctx[b] + kd[b]
            if cleared:
                assert (k2[b, :, s] == 0).all() and (v2[b, :, s] == 0).all()
            else:
                assert (k2[b, :, s] == kc[b, :, s]).all() and (v2[b, :, s] == vc[b, :, s]).all()


# ----------------------------------------------------------------------------
# QKV projection + rotary embedding of the verify block
# ----------------------------------------------------------------------------
def check_rope_worked_examples(o):
    g = _golden()["rope"]
    theta = 4.0 / math.pi ** 2
    x = np.asarray(g["x"])
    for ex in g["cases"]:
        y = o.rope(x, ex["pos"], theta)
        np.testing.assert_allclose(y[[1, 3]], ex["pair13"], rtol=0, atol=1e-12, err_msg=ex["why"])
        # The first pair keeps its length and turns by pos radians.
        assert abs(y[0] ** 2 + y[2] ** 2 - (x[0] ** 2 + x[2] ** 2)) < 1e-12
        turn = math.atan2(y[2], y[0]) - math.atan2(x[2], x[0])
        assert abs(math.remainder(turn - ex["pair02_angle"], 2 * math.pi)) < 1e-12, ex["why"]


def check_rope_vs_complex_rotation(o, seed=10):
    """The same rotation written as a complex product in torch float64: z_j = x_j + i x_{j+D/2}
    times exp(i pos / theta^(2j/D))."""
    rng = np.random.default_rng(seed)
    for D, theta in ((8, 10000.0), (64, 500000.0), (128, 10000.0)):
        x = rng.standard_normal((5, 3, D))
        pos = rng.integers(0, 40000, size=(5, 3))
        got = o.rope(x, pos, theta)
        xt = torch.from_numpy(x)
        inv = 1.0 / (theta ** (torch.arange(0, D, 2, dtype=torch.float64) / D))
        ang = torch.from_numpy(pos).to(torch.float64)[..., None] * inv
        z = torch.complex(xt[..., :D // 2], xt[..., D // 2:]) * torch.polar(torch.ones_like(ang), ang)
        ref = torch.cat([z.real, z.imag], dim=-1).numpy()
        np.testing.assert_allclose(got, ref, rtol=1e-9, atol=1e-9)


def check_rope_relative_position(o, seed=11):
    """<rope(q, m), rope(k, n)> depends on m - n only."""
    rng = np.random.default_rng(seed)
    q, k = rng.standard_normal(64), rng.standard_normal(64)
    for m, n, t in ((5, 2, 100), (0, 9, 7), (1000, 10, 31)):
        a = o.rope(q, m, 10000.0) @ o.rope(k, n, 10000.0)
        b = o.rope(q, m + t, 10000.0) @ o.rope(k, n + t, 10000.0)
        assert abs(a - b) < 1e-9 * (1 + abs(a))
    assert abs(o.rope(q, 3, 10000.0) @ o.rope(k, 0, 10000.0) - q @ k) > 1e-6  # not trivially constant


def check_qkv_projection_layout(o, seed=12):
    """One-hot hidden rows pick columns of W^T; rows of W split q | k | v by head; only q and k
    turn (v at any position equals the projection), and row i sits at position ctx + i."""
    rng = np.random.default_rng(seed)
    Hq, Hkv, D, H = 2, 1, 4, 6
    W = rng.standard_normal(((Hq + 2 * Hkv) * D, H))
    x = np.eye(H)[[0, 3, 5]]
    ctx, kd, cu = [7], [2], [0, 3]
    q, k, v = o.verify_qkv_rope(x, W, ctx, kd, cu, Hq, Hkv, 10000.0)
    y = W.T[[0, 3, 5]]
    np.testing.assert_array_equal(v.reshape(3, -1), y[:, (Hq + Hkv) * D:])
    for i in range(3):
        for h in range(Hq):
            np.testing.assert_allclose(q[i, h], o.rope(y[i, h * D:(h + 1) * D], 7 + i, 10000.0), rtol=0, atol=1e-12)
        np.testing.assert_allclose(k[i, 0], o.rope(y[i, Hq * D:(Hq + 1) * D], 7 + i, 10000.0), rtol=0, atol=1e-12)
    # Norms of q per head are those of the projection (a rotation).
    np.testing.assert_allclose(np.linalg.norm(q, axis=-1), np.linalg.norm(y[:, :Hq * D].reshape(3, Hq, D), axis=-1),
                               rtol=1e-12)


def check_kv_write_slots(o):
    g = _golden()["qkv_write"]
    B, Hkv, cap, D = 2, 2, 6, 3
    kc = np.full((B, Hkv, cap, D), -1.0)
    vc = np.full((B, Hkv, cap, D), -2.0)
    R = g["cu_q"][-1]
    k = np.arange(R * Hkv * D, dtype=np.float64).reshape(R, Hkv, D)
    v = k + 1000.0
    k2, v2 = o.kv_write(kc, vc, k, v, g["ctx"], g["k"], g["cu_q"])
    written = set()
    for r, (b, slot) in enumerate(g["slots"]):
        np.testing.assert_array_equal(k2[b, :, slot], k[r])
        np.testing.assert_array_equal(v2[b, :, slot], v[r])
        written.add((b, slot))
    for b in range(B):
        for slot in range(cap):
            if (b, slot) not in written:
                assert (k2[b, :, slot] == -1.0).all() and (v2[b, :, slot] == -2.0).all()


# ----------------------------------------------------------------------------
# Paged KV cache
# ----------------------------------------------------------------------------
def check_paged_worked_example(o):
    g = _golden()["paged"]
    P = g["page"]
    kp = np.arange(4 * 1 * P * 2, dtype=np.float64).reshape(4, 1, P, 2) + 1.0
    vp = -kp
    k2, v2, ctx = o.kv_commit_paged(kp, vp, g["block_table"], g["ctx"], g["accepted"], g["k"], P)
    np.testing.assert_array_equal(ctx, g["new_ctx"])
    cleared = {tuple(c) for c in g["cleared"]}
    for pg in range(4):
        for r in range(P):
            if (pg, r) in cleared:
                assert (k2[pg, :, r] == 0).all() and (v2[pg, :, r] == 0).all()
            else:
                assert (k2[pg, :, r] == kp[pg, :, r]).all() and (v2[pg, :, r] == vp[pg, :, r]).all()


def check_paged_matches_dense(o, seed=13):
    """Scattering dense caches into pages by a random table and gathering them back is the
    identity; commit and write through the table equal the dense ones on the gathered view."""
    rng = np.random.default_rng(seed)
    B, Hkv, D, P, max_pages = 3, 2, 4, 4, 3
    cap = P * max_pages
    perm = rng.permutation(B * max_pages + 2)
    table = perm[:B * max_pages].reshape(B, max_pages)
    kd = np.array([2, 0, 3])
    ctx = np.array([5, 0, 8])
    cu = np.concatenate([[0], np.cumsum(kd + 1)])
    dense_k = rng.standard_normal((B, Hkv, cap, D))
    dense_v = rng.standard_normal((B, Hkv, cap, D))
    kp = np.full((B * max_pages + 2, Hkv, P, D), np.nan)
    vp = kp.copy()
    for b in range(B):
        for j in range(max_pages):
            kp[table[b, j]] = dense_k[b, :, j * P:(j + 1) * P]
            vp[table[b, j]] = dense_v[b, :, j * P:(j + 1) * P]
    np.testing.assert_array_equal(o.paged_gather(kp, table, cap, P), dense_k)
    acc = np.array([1, 0, 0])
    k2, v2, c2 = o.kv_commit_paged(kp, vp, table, ctx, acc, kd, P)
    kd2, vd2, cd2 = o.kv_commit(dense_k, dense_v, ctx, acc, kd)
    np.testing.assert_array_equal(o.paged_gather(k2, table, cap, P), kd2)
    np.testing.assert_array_equal(o.paged_gather(v2, table, cap, P), vd2)
    np.testing.assert_array_equal(c2, cd2)
    R = int(cu[-1])
    kn = rng.standard_normal((R, Hkv, D))
    vn = rng.standard_normal((R, Hkv, D))
    k3, v3 = o.kv_write_paged(kp, vp, table, kn, vn, ctx, kd, cu, P)
    kd3, vd3 = o.kv_write(dense_k, dense_v, kn, vn, ctx, kd, cu)
    np.testing.assert_array_equal(o.paged_gather(k3, table, cap, P), kd3)
    np.testing.assert_array_equal(o.paged_gather(v3, table, cap, P), vd3)
    assert np.isnan(k3[perm[B * max_pages:]]).all()  # pages outside the table untouched


# ----------------------------------------------------------------------------
# Temperature of the verifier's distribution
# ----------------------------------------------------------------------------
def check_temperature_worked_example(o):
    g = _golden()["temperature"]
    l = np.asarray(g["logits"])
    T = g["T"]
    logits = np.stack([l, l])
    a = g["accept"]
    q = np.asarray(a["q"])[None]
    res = o.verify_accept(logits, [a["draft"]], q, [a["u_accept"], 0.5], [1], [0, 2], [1], temperature=[T])
    assert res["accepted_len"][0] == 1
    res = o.verify_accept(logits, [a["draft"]], q, [a["u_reject"], 0.5], [1], [0, 2], [1], temperature=[T])
    assert res["accepted_len"][0] == 0
    for u, x in g["bonus"]:
        res = o.verify_accept(l[None], [], np.zeros((0, 3)), [u], [1], [0, 1], [0], temperature=[T])
        assert res["next_token"][0] == x, (u, x)
    # Greedy decisions ignore the temperature.
    res = o.verify_accept(logits, [1], None, [0.5, 0.5], [0], [0, 2], [1], temperature=[T])
    assert res["accepted_len"][0] == 1 and res["next_token"][0] == 1


def check_temperature_output_law(o, n=40000, seed=14):
    """Rejection sampling at temperature T reproduces softmax(l / T) (Sec. III-C with p at T)."""
    rng = np.random.default_rng(seed)
    V, k, T = 6, 1, 0.5
    L = rng.standard_normal((k + 1, V))
    P = np.exp(L / T)
    P /= P.sum(axis=1, keepdims=True)
    Q = rng.dirichlet(np.ones(V), size=k)
    drafts = rng.choice(V, size=n, p=Q[0])
    u = rng.random(n * (k + 1))
    res = o.verify_accept(np.tile(L, (n, 1)), drafts, np.tile(Q, (n, 1)), u, np.ones(n, int),
                          np.arange(n + 1) * (k + 1), np.full(n, k), temperature=np.full(n, T))
    first = np.where(res["accepted_len"] >= 1, drafts, res["next_token"])
    _, pv = stats.chisquare(np.bincount(first, minlength=V), P[0] * n)
    assert pv > 1e-3, pv


# ----------------------------------------------------------------------------
# Top-p truncation of the verifier's distribution
# ----------------------------------------------------------------------------
def check_top_p_worked_example(o):
    g = _golden()["top_p"]
    P = np.asarray(g["p"])
    l = np.log(P)
    pt, _, _ = o.nucleus(P, g["top_p"])
    np.testing.assert_allclose(pt, g["nucleus"], rtol=0, atol=1e-15)
    ex = g["exact_reach"]
    np.testing.assert_allclose(o.nucleus(P, ex["top_p"])[0], ex["nucleus"], rtol=0, atol=1e-15, err_msg=ex["why"])
    tp = [g["top_p"]]
    for ex in g["accept"]:
        res = o.verify_accept(np.stack([l, l]), [ex["draft"]], np.asarray(ex["q"])[None], [ex["u"], 0.5], [1],
                              [0, 2], [1], top_p=tp)
        assert res["accepted_len"][0] == ex["accepted"], ex["why"]
    rq = np.asarray(g["residual"]["q"])[None]
    for u, x in g["residual"]["cases"]:
        res = o.verify_accept(np.stack([l, l]), [g["residual"]["draft"]], rq, [0.0, u], [1], [0, 2], [1], top_p=tp)
        assert res["accepted_len"][0] == 0 and res["next_token"][0] == x, (u, x)
    for u, x in g["bonus"]:
        res = o.verify_accept(l[None], [], np.zeros((0, 4)), [u], [1], [0, 1], [0], top_p=tp)
        assert res["next_token"][0] == x, (u, x)
    # top_p = 1 is no truncation.
    np.testing.assert_array_equal(o.nucleus(P, 1.0)[0], P)


def check_top_p_output_law(o, n=40000, seed=15):
    """Rejection sampling with a nucleus reproduces the truncated, renormalised p."""
    rng = np.random.default_rng(seed)
    V, k, tp = 8, 1, 0.8
    L = rng.standard_normal((k + 1, V)) * 1.5
    P0 = np.exp(L[0]) / np.exp(L[0]).sum()
    Pt, _, _ = o.nucleus(P0, tp)
    Q = rng.dirichlet(np.ones(V), size=k)
    drafts = rng.choice(V, size=n, p=Q[0])
    u = rng.random(n * (k + 1))
    res = o.verify_accept(np.tile(L, (n, 1)), drafts, np.tile(Q, (n, 1)), u, np.ones(n, int),
                          np.arange(n + 1) * (k + 1), np.full(n, k), top_p=np.full(n, tp))
    first = np.where(res["accepted_len"] >= 1, drafts, res["next_token"])
    counts = np.bincount(first, minlength=V)
    assert (counts[Pt == 0] == 0).all()
    keep = Pt > 0
    _, pv = stats.chisquare(counts[keep], Pt[keep] * n)
    assert pv > 1e-3, pv


ALL_CHECKS = [
    check_attention_worked_examples, check_attention_vs_sdpa, check_attention_special_cases,
    check_attention_gqa_mapping, check_logits_one_hot, check_acceptance_worked_examples,
    check_margin_worked_examples, check_sample_spread_worked_examples, check_residual_properties, check_q_equals_p_accepts_all, check_strict_comparison,
    check_stochastic_output_law, check_progress_and_bounds, check_greedy_identity,
    check_kv_commit, check_rope_worked_examples, check_rope_vs_complex_rotation,
    check_rope_relative_position, check_qkv_projection_layout, check_kv_write_slots,
    check_paged_worked_example, check_paged_matches_dense, check_temperature_worked_example,
    check_temperature_output_law, check_top_p_worked_example, check_top_p_output_law,
]
