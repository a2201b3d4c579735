"""Shared helpers of the GPU parity tests and the smoke check.

Runs one verify step through the CUDA library (via its C-ABI binding) and the
same step through the float64 oracle, on the same seeded inputs, and compares
them under the rules of the verify step:

* attention outputs: |gpu - oracle| <= 2e-2 * max(|oracle|, rms of the oracle's
  (row, head) vector), element by element;
* accepted lengths and next tokens: bit-exact, except for sequences whose
  oracle decision margin (top-2 logit gap or |u - p/q|) or sampling margin is
  below 1e-3 -- those are counted and returned;
* KV commit: caches and context lengths bit-exact;
* on-chip logits, through the merged row statistics the LM-head kernel leaves
  in its workspace (max logit, log-sum-exp, draft-token logit):
  |gpu - oracle| <= 2e-2 * max(|oracle|, rms of the oracle's logit row).
"""
from __future__ import annotations

import numpy as np
import torch

import oracle.spade_oracle as O
import paper_2608_13076_gb300 as spade

ATTN_RTOL = 2e-2
LOGIT_RTOL = 2e-2


def to_np(t):
    if t is None:
        return None
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        t = t.float()
    return t.numpy()


def gpu_attention(wl, workspace=None, status=None):
    dev = wl["q"].device
    out = torch.empty_like(wl["q"])
    lse = torch.empty(wl["q"].shape[:2], dtype=torch.float32, device=dev)
    max_k = int(wl["n_draft"].max())
    if workspace is None:
        workspace = spade.attn_workspace(wl["B"], wl["Hq"], wl["Hkv"], wl["D"], wl["cap"], max_k, device=dev)
    if status is None:
        status = spade.status_tensor(dev)
    spade.spade_verify_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["ctx_lens"], wl["n_draft"],
                                 wl["cu_q"], out, lse, max_k=max_k, workspace=workspace, status=status)
    return out, lse, status


def gpu_accept(wl, workspace=None, status=None, temperature=None):
    dev = wl["hidden"].device
    B = wl["B"]
    acc = torch.full((B,), -7, dtype=torch.int32, device=dev)
    tok = torch.full((B,), -7, dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = spade.accept_workspace(B, wl["R"], wl["H"], wl["V"], device=dev)
    if status is None:
        status = spade.status_tensor(dev)
    spade.spade_verify_accept(wl["hidden"], wl["w_lm"], wl["draft_tokens"], wl["draft_probs"],
                              wl["uniforms"], wl["mode"], wl["cu_q"], wl["n_draft"], acc, tok,
                              workspace=workspace, status=status, temperature=temperature)
    return acc, tok, status


def gpu_accept_commit(wl, workspace=None, status=None):
    """The fused accept + KV commit call (updates wl's caches and ctx_lens in place)."""
    dev = wl["hidden"].device
    B = wl["B"]
    acc = torch.full((B,), -7, dtype=torch.int32, device=dev)
    tok = torch.full((B,), -7, dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = spade.accept_workspace(B, wl["R"], wl["H"], wl["V"], device=dev)
    if status is None:
        status = spade.status_tensor(dev)
    spade.spade_verify_accept_commit(wl["hidden"], wl["w_lm"], wl["draft_tokens"], wl["draft_probs"],
                                     wl["uniforms"], wl["mode"], wl["cu_q"], wl["n_draft"], acc, tok,
                                     wl["k_cache"], wl["v_cache"], wl["ctx_lens"], workspace=workspace,
                                     status=status)
    return acc, tok, workspace, status


def gpu_accept_sampling(wl, temperature=None, top_p=None, commit=False, workspace=None, status=None):
    """spade_verify_accept_sampling on wl (with commit: updates wl's caches and ctx_lens)."""
    dev = wl["hidden"].device
    B = wl["B"]
    acc = torch.full((B,), -7, dtype=torch.int32, device=dev)
    tok = torch.full((B,), -7, dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = spade.accept_workspace(B, wl["R"], wl["H"], wl["V"], device=dev)
    if status is None:
        status = spade.status_tensor(dev)
    cache = dict(k_cache=wl["k_cache"], v_cache=wl["v_cache"], ctx_lens=wl["ctx_lens"]) if commit else {}
    spade.spade_verify_accept_sampling(wl["hidden"], wl["w_lm"], wl["draft_tokens"], wl["draft_probs"],
                                       wl["uniforms"], wl["mode"], wl["cu_q"], wl["n_draft"], acc, tok,
                                       workspace=workspace, status=status, temperature=temperature,
                                       top_p=top_p, **cache)
    return acc, tok, status


def oracle_logits(wl):
    return O.lm_logits(to_np(wl["hidden"]), to_np(wl["w_lm"]))


def oracle_accept_from_logits(wl, logits, temperature=None, top_p=None):
    return O.verify_accept(logits, to_np(wl["draft_tokens"]), to_np(wl["draft_probs"]),
                           to_np(wl["uniforms"]), to_np(wl["mode"]), to_np(wl["cu_q"]),
                           to_np(wl["n_draft"]), temperature=temperature, top_p=top_p)


def oracle_attention(wl, rows=None):
    return O.verify_attention(to_np(wl["q"]), to_np(wl["k_cache"]), to_np(wl["v_cache"]),
                              to_np(wl["ctx_lens"]), to_np(wl["n_draft"]), to_np(wl["cu_q"]), rows=rows)


def oracle_accept(wl):
    logits = O.lm_logits(to_np(wl["hidden"]), to_np(wl["w_lm"]))
    return O.verify_accept(logits, to_np(wl["draft_tokens"]), to_np(wl["draft_probs"]),
                           to_np(wl["uniforms"]), to_np(wl["mode"]), to_np(wl["cu_q"]),
                           to_np(wl["n_draft"]))


def compare_attention(out_gpu, ref, rows=None, rtol=ATTN_RTOL):
    """Returns (n_checked, n_bad, worst ratio) of |g-o| / (rtol * max(|o|, rms))."""
    g = to_np(out_gpu).astype(np.float64)
    pairs = rows if rows is not None else [(r, h) for r in range(ref.shape[0]) for h in range(ref.shape[1])]
    bad = 0
    worst = 0.0
    for r, h in pairs:
        o = ref[r, h]
        rms = float(np.sqrt(np.mean(o * o)))
        tol = rtol * np.maximum(np.abs(o), rms)
        err = np.abs(g[r, h] - o)
        ratio = float(np.max(err / tol)) if rms > 0 else float(np.max(err))
        worst = max(worst, ratio)
        bad += int(np.sum(err > tol))
    return len(pairs), bad, worst


def compare_row_stats(stats, logits, wl, rtol=LOGIT_RTOL, margin=1e-3):
    """The LM-head kernel's merged row statistics against the oracle's float64 logits.

    stats: ``spade.read_accept_stats`` output; logits [R, V] float64.  Checks the
    max logit, the log-sum-exp (max + log sum exp(l - max)) and, for rows with a
    draft, the draft token's logit, each within rtol * max(|oracle|, rms of the
    row); the argmax bit-exactly wherever the top-2 gap is at least ``margin``.
    Returns dict with the worst error ratio per quantity and the argmax mismatches.
    """
    R = logits.shape[0]
    rms = np.sqrt(np.mean(logits * logits, axis=1))
    o_max = logits.max(axis=1)
    o_lse = o_max + np.log(np.exp(logits - o_max[:, None]).sum(axis=1))
    g_max = stats["max"].double().numpy()
    g_lse = g_max + np.log(stats["sumexp"].double().numpy())

    def ratio(g, o, rows):
        tol = rtol * np.maximum(np.abs(o[rows]), rms[rows])
        return float(np.max(np.abs(g[rows] - o[rows]) / tol)) if len(rows) else 0.0

    allr = np.arange(R)
    cu = to_np(wl["cu_q"]).astype(np.int64)
    kd = to_np(wl["n_draft"]).astype(np.int64)
    drows, dtok = [], []
    dt = to_np(wl["draft_tokens"]).astype(np.int64)
    for b in range(wl["B"]):
        for i in range(int(kd[b])):
            drows.append(int(cu[b]) + i)
            dtok.append(int(dt[int(cu[b]) - b + i]))
    drows = np.asarray(drows, dtype=np.int64)
    o_ld = np.zeros(R)
    if len(drows):
        o_ld[drows] = logits[drows, np.asarray(dtok)]
    g_ld = stats["draft_logit"].double().numpy()
    top2 = np.partition(logits, -2, axis=1)[:, -2:] if logits.shape[1] > 1 else None
    decided = (top2[:, 1] - top2[:, 0]) >= margin if top2 is not None else np.ones(R, bool)
    o_arg = logits.argmax(axis=1)
    g_arg = stats["argmax"].numpy().astype(np.int64)
    return dict(max=ratio(g_max, o_max, allr), lse=ratio(g_lse, o_lse, allr),
                draft_logit=ratio(g_ld, o_ld, drows),
                argmax_mismatch=int(np.sum((g_arg != o_arg) & decided)),
                argmax_close=int(np.sum(~decided)))


def check_commit_windows(wl_before, k_after, v_after, ctx_after, acc):
    """KV commit against ``O.kv_commit`` on every sequence's verify block.

    The commit touches only slots [ctx_b, ctx_b + k_b] of sequence b.  Those
    windows (all KV heads) are cut out of the caches as they were before the
    call, committed by the oracle with the window's own context length 0, and
    compared bit for bit with the same windows after the GPU call; everything
    outside the windows must be unchanged (compared on the device).  Returns the
    number of sequences checked.
    """
    k0, v0 = wl_before["k_cache"], wl_before["v_cache"]
    ctx0 = to_np(wl_before["ctx_lens"]).astype(np.int64)
    kd = to_np(wl_before["n_draft"]).astype(np.int64)
    a = to_np(acc).astype(np.int64)
    B, Hkv, cap, D = k0.shape
    W = int(kd.max()) + 1
    wk0 = np.zeros((B, Hkv, W, D), dtype=np.float32)
    wv0 = np.zeros_like(wk0)
    wk1 = np.zeros_like(wk0)
    wv1 = np.zeros_like(wk0)
    for b in range(B):
        lo, n = int(ctx0[b]), int(kd[b]) + 1
        wk0[b, :, :n] = to_np(k0[b, :, lo:lo + n])
        wv0[b, :, :n] = to_np(v0[b, :, lo:lo + n])
        wk1[b, :, :n] = to_np(k_after[b, :, lo:lo + n])
        wv1[b, :, :n] = to_np(v_after[b, :, lo:lo + n])
        assert torch.equal(k_after[b, :, :lo], k0[b, :, :lo]) and torch.equal(v_after[b, :, :lo], v0[b, :, :lo])
        assert torch.equal(k_after[b, :, lo + n:], k0[b, :, lo + n:])
        assert torch.equal(v_after[b, :, lo + n:], v0[b, :, lo + n:])
    rk, rv, rctx = O.kv_commit(wk0, wv0, np.zeros(B, dtype=np.int64), a, kd)
    assert np.array_equal(wk1, rk) and np.array_equal(wv1, rv)
    assert np.array_equal(to_np(ctx_after).astype(np.int64), ctx0 + rctx)
    return B


def gpu_qkv_rope(wl, x, w, q_out=None, status=None):
    """The QKV projection + rotary embedding call (writes wl's caches in place)."""
    dev = x.device
    if q_out is None:
        q_out = torch.full((wl["R"], wl["Hq"], wl["D"]), float("nan"), dtype=torch.bfloat16, device=dev)
    if status is None:
        status = spade.status_tensor(dev)
    spade.spade_verify_qkv_rope(x, w, wl["ctx_lens"], wl["n_draft"], wl["cu_q"], q_out, wl["k_cache"],
                                wl["v_cache"], Hq=wl["Hq"], Hkv=wl["Hkv"], rope_theta=wl["spec"].rope_theta,
                                max_k=int(wl["n_draft"].max()),
                                workspace=spade.qkv_workspace(wl["R"], wl["Hq"], wl["Hkv"], wl["D"], device=dev),
                                status=status)
    return q_out, status


def check_qkv_rope(wl, x, w, q_gpu, k_before, v_before, skip=()):
    """q, and the K/V written into the verify slots, against ``O.verify_qkv_rope`` (the
    attention rule per (row, head) vector); every other cache slot unchanged bit for bit.
    Sequences in ``skip`` must be left entirely untouched (q rows still NaN).
    Returns the worst tolerance ratio over q, k and v."""
    ctx, kd, cu = to_np(wl["ctx_lens"]), to_np(wl["n_draft"]), to_np(wl["cu_q"])
    q_ref, k_ref, v_ref = O.verify_qkv_rope(to_np(x), to_np(w), ctx, kd, cu, wl["Hq"], wl["Hkv"],
                                            wl["spec"].rope_theta)
    seq, pos = O.verify_positions(ctx, kd, cu)
    keep = np.array([s not in skip for s in seq])
    rows = [(r, h) for r in np.nonzero(keep)[0] for h in range(wl["Hq"])]
    worst = 0.0
    n, bad, wq = compare_attention(q_gpu, q_ref, rows=rows)
    assert bad == 0, f"q: {bad} bad elements, worst {wq:.3g}"
    worst = max(worst, wq)
    dev = q_gpu.device
    si = torch.from_numpy(seq[keep]).to(dev)
    pi = torch.from_numpy(pos[keep]).to(dev)
    for cache, before, ref, nm in ((wl["k_cache"], k_before, k_ref, "k"), (wl["v_cache"], v_before, v_ref, "v")):
        got = cache[si, :, pi]  # [rows, Hkv, D]
        kv_rows = [(r, g) for r in range(int(keep.sum())) for g in range(wl["Hkv"])]
        n, bad, wk = compare_attention(got, ref[keep], rows=kv_rows)
        assert bad == 0, f"{nm}: {bad} bad elements, worst {wk:.3g}"
        worst = max(worst, wk)
        expect = before.clone()
        expect[si, :, pi] = cache[si, :, pi]
        assert torch.equal(expect, cache), f"{nm} cache changed outside the verify slots"
    if skip:
        assert torch.isnan(q_gpu[torch.from_numpy(~keep).to(dev)].float()).all()
    return worst


def compare_accept(acc_gpu, tok_gpu, ref):
    """Bit-exact accept decisions outside flagged margins.

    Returns dict(mismatch_unflagged, flagged, mismatch_flagged)."""
    a = to_np(acc_gpu).astype(np.int64)
    t = to_np(tok_gpu).astype(np.int64)
    ra, rt = ref["accepted_len"], ref["next_token"]
    fd, fs = ref["flag_decision"], ref["flag_sample"]
    bad_a = (a != ra) & ~fd
    bad_t = (t != rt) & ~(fd | fs)
    flagged = fd | fs
    return dict(
        mismatch_unflagged=int(np.sum(bad_a | bad_t)),
        flagged=int(np.sum(flagged)),
        mismatch_flagged=int(np.sum(((a != ra) | (t != rt)) & flagged)),
        bad_seqs=[int(b) for b in np.nonzero(bad_a | bad_t)[0]],
    )
