"""Shared helpers of the GPU parity tests and the smoke check.

Runs one verify step through the CUDA library (via its C-ABI binding) and the
same step through the float64 oracle, on the same seeded inputs, and compares
them under the rules of the verify step:

* attention outputs: |gpu - oracle| <= 2e-2 * max(|oracle|, rms of the oracle's
  (row, head) vector), element by element;
* accepted lengths and next tokens: bit-exact, except for sequences whose
  oracle decision margin (top-2 logit gap or |u - p/q|) or sampling margin is
  below 1e-3 -- those are counted and returned;
* KV commit: caches and context lengths bit-exact.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle.spade_oracle as O
import paper_2608_13076_gb300 as spade

ATTN_RTOL = 2e-2


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


def gpu_accept(wl, workspace=None, status=None):
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
                              workspace=workspace, status=status)
    return acc, tok, status


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
