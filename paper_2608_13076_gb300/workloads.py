"""Seeded synthetic workloads for the SPADE verify step.

This module only draws inputs: shapes, random tensors, draft tokens, draft
distributions and uniforms.  It holds none of the verify step's arithmetic
(attention, the accept rule, residual sampling, KV commit); both the CUDA path
and the float64 oracle consume what it returns.

Workloads stand in for the paper's Spec-Bench / CNN-DailyMail runs (Sec. IV),
whose data and model weights are not available: every tensor has the shape of
a verifier step of the named model family, values drawn from seeded normal /
uniform distributions.

Draft distributions.  A real draft model's ``q`` is correlated with the
verifier's ``p``; the synthetic stand-in is ``q = softmax(l + sigma * z)`` where
``l`` are the verifier logits recomputed here in float32 (this is the *draft
model proxy*, not the verify step) and ``z ~ N(0, 1)``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

GREEDY = 0
STOCHASTIC = 1


@dataclass(frozen=True)
class WorkloadSpec:
    """Shape and draft-model recipe of one synthetic verify step."""

    name: str
    B: int
    Hq: int
    Hkv: int
    D: int
    H: int
    V: int
    ctx: tuple            # (lo, hi) inclusive range of committed context lengths
    k: tuple              # (lo, hi) inclusive range of draft lengths
    mode: str             # "greedy", "stochastic" or "mixed" (even b greedy, odd b stochastic)
    match_prob: float = 0.7     # greedy: P(draft == verifier argmax)
    noise: float = 0.5          # stochastic: std of the logit noise of q
    target_accept: float = 0.0  # stochastic: if > 0, tune noise so mean sum(min(p,q)) hits it
    greedy_draft: str = "match" # greedy drafts: "match" (match_prob) or "noisy_argmax"
    seed: int = 0
    rope_theta: float = 10000.0  # base of the rotary frequencies of the model family
    logit_scale: float = 1.0     # std of the hidden rows: logits ~ N(0, logit_scale^2)
    extra: dict = field(default_factory=dict)


# The five verifier shapes of the benchmark suite.  Seeds 1000+id; the
# stochastic variant of the Llama-2-7B step uses 2002.
SPECS = {
    "tiny": WorkloadSpec("tiny", B=1, Hq=8, Hkv=8, D=64, H=512, V=1024, ctx=(256, 256),
                         k=(4, 4), mode="greedy", match_prob=0.7, seed=1001),
    "llama2_7b_greedy": WorkloadSpec("llama2_7b_greedy", B=1, Hq=32, Hkv=32, D=128, H=4096,
                                     V=32000, ctx=(2048, 2048), k=(5, 5), mode="greedy",
                                     noise=0.5, greedy_draft="noisy_argmax", seed=1002),
    "llama2_7b_stochastic": WorkloadSpec("llama2_7b_stochastic", B=1, Hq=32, Hkv=32, D=128,
                                         H=4096, V=32000, ctx=(2048, 2048), k=(5, 5),
                                         mode="stochastic", noise=0.5, seed=2002),
    "llama3_8b": WorkloadSpec("llama3_8b", B=8, Hq=32, Hkv=8, D=128, H=4096, V=128256,
                              ctx=(4096, 4096), k=(8, 8), mode="stochastic",
                              target_accept=0.7, seed=1003, rope_theta=500000.0),
    "long_70b": WorkloadSpec("long_70b", B=4, Hq=64, Hkv=8, D=128, H=8192, V=32000,
                             ctx=(32768, 32768), k=(4, 4), mode="greedy", match_prob=0.6,
                             seed=1004, rope_theta=500000.0),
    "ragged": WorkloadSpec("ragged", B=64, Hq=40, Hkv=8, D=128, H=5120, V=152064,
                           ctx=(128, 8192), k=(1, 10), mode="mixed", match_prob=0.7,
                           noise=0.5, seed=1005, rope_theta=1000000.0),
}


def scaled(spec: WorkloadSpec, **over) -> WorkloadSpec:
    """A copy of ``spec`` with some fields replaced (smaller parity cases)."""
    d = dict(spec.__dict__)
    d.update(over)
    return WorkloadSpec(**d)


def _bf16_normal(gen, shape, std, device):
    x = torch.randn(shape, generator=gen, dtype=torch.float32, device=device)
    if std != 1.0:
        x.mul_(std)
    return x.to(torch.bfloat16)


def _verifier_logits_f32(hidden, w_lm, chunk=16384):
    """Draft-model proxy: float32 logits used only to synthesise q and drafts."""
    R = hidden.shape[0]
    out = torch.empty((R, w_lm.shape[0]), dtype=torch.float32, device=hidden.device)
    h = hidden.float()
    for v0 in range(0, w_lm.shape[0], chunk):
        out[:, v0:v0 + chunk] = h @ w_lm[v0:v0 + chunk].float().t()
    return out


def _mean_overlap(logits, noise, sigma):
    p = torch.softmax(logits, dim=-1)
    q = torch.softmax(logits + sigma * noise, dim=-1)
    return torch.minimum(p, q).sum(-1).mean().item()


def make_workload(spec: WorkloadSpec, device="cpu", cache_pad: int = 0):
    """Draw all inputs of one verify step.

    Every tensor is drawn on the CPU from one seeded generator and only then
    moved to ``device``, so a seed names the same inputs on every device (the
    GPU path, the float64 oracle and the CPU baseline all see identical data).

    Returns a dict of tensors on ``device``:
      q [R,Hq,D] bf16, k_cache/v_cache [B,Hkv,cap,D] bf16 (slots [0, ctx+k] filled,
      the rest zero), ctx_lens/n_draft [B] i32, cu_q [B+1] i32, hidden [R,H] bf16,
      w_lm [V,H] bf16, draft_tokens [R-B] i32, draft_probs [R-B,V] f32 or None,
      uniforms [R] f32 in [0,1), mode [B] i32, plus python ints B, R, cap, ...
    """
    gen = torch.Generator(device="cpu").manual_seed(spec.seed)
    dev = torch.device(device)
    cpu = torch.device("cpu")

    B = spec.B
    if spec.ctx[0] == spec.ctx[1]:
        ctx = torch.full((B,), spec.ctx[0], dtype=torch.int32)
    else:
        ctx = torch.randint(spec.ctx[0], spec.ctx[1] + 1, (B,), generator=gen, dtype=torch.int32)
    if spec.k[0] == spec.k[1]:
        kd = torch.full((B,), spec.k[0], dtype=torch.int32)
    else:
        kd = torch.randint(spec.k[0], spec.k[1] + 1, (B,), generator=gen, dtype=torch.int32)
    if spec.mode == "greedy":
        mode = torch.zeros(B, dtype=torch.int32)
    elif spec.mode == "stochastic":
        mode = torch.ones(B, dtype=torch.int32)
    else:
        mode = (torch.arange(B) % 2).to(torch.int32)

    cu_q = torch.zeros(B + 1, dtype=torch.int32)
    cu_q[1:] = torch.cumsum(kd + 1, 0)
    R = int(cu_q[-1])
    n_draft_rows = R - B
    cap = int((ctx + kd + 1).max()) + cache_pad

    q = _bf16_normal(gen, (R, spec.Hq, spec.D), 1.0, cpu)
    k_cache = torch.zeros((B, spec.Hkv, cap, spec.D), dtype=torch.bfloat16)
    v_cache = torch.zeros_like(k_cache)
    for b in range(B):
        L = int(ctx[b] + kd[b] + 1)
        k_cache[b, :, :L] = _bf16_normal(gen, (spec.Hkv, L, spec.D), 1.0, cpu)
        v_cache[b, :, :L] = _bf16_normal(gen, (spec.Hkv, L, spec.D), 1.0, cpu)
    hidden = _bf16_normal(gen, (R, spec.H), spec.logit_scale, cpu)
    w_lm = _bf16_normal(gen, (spec.V, spec.H), 1.0 / math.sqrt(spec.H), cpu)

    # Draft rows: row cu_q[b]+i (i < k_b) holds draft i of sequence b.
    draft_row_of = []
    for b in range(B):
        for i in range(int(kd[b])):
            draft_row_of.append(int(cu_q[b]) + i)
    draft_row_of = torch.tensor(draft_row_of, dtype=torch.long)
    seq_of_draft = torch.repeat_interleave(torch.arange(B), kd.long())

    logits = _verifier_logits_f32(hidden[draft_row_of], w_lm) if n_draft_rows else \
        torch.zeros((0, spec.V))
    noise = torch.randn(logits.shape, generator=gen, dtype=torch.float32)
    sigma = spec.noise
    if spec.target_accept > 0 and (mode == STOCHASTIC).any():
        lo, hi = 0.0, 20.0
        for _ in range(24):
            mid = 0.5 * (lo + hi)
            if _mean_overlap(logits, noise, mid) > spec.target_accept:
                lo = mid
            else:
                hi = mid
        sigma = 0.5 * (lo + hi)
    draft_logits = logits + sigma * noise
    q_dist = torch.softmax(draft_logits, dim=-1)

    stoch_draft = mode[seq_of_draft] == STOCHASTIC
    drafts = torch.empty(n_draft_rows, dtype=torch.int64)
    if stoch_draft.any():
        idx = stoch_draft.nonzero().flatten()
        drafts[idx] = torch.multinomial(q_dist[idx], 1, generator=gen).flatten()
    if (~stoch_draft).any():
        idx = (~stoch_draft).nonzero().flatten()
        if spec.greedy_draft == "noisy_argmax":
            drafts[idx] = draft_logits[idx].argmax(-1)
        else:
            am = logits[idx].argmax(-1)
            rnd = torch.randint(0, spec.V, (idx.numel(),), generator=gen)
            hit = torch.rand(idx.numel(), generator=gen) < spec.match_prob
            drafts[idx] = torch.where(hit, am, rnd)

    uniforms = torch.rand(R, generator=gen, dtype=torch.float32)
    draft_probs = q_dist.contiguous() if bool((mode == STOCHASTIC).any()) else None

    def mv(t):
        return None if t is None else t.to(dev)

    return dict(
        spec=spec, B=B, R=R, cap=cap, Hq=spec.Hq, Hkv=spec.Hkv, D=spec.D, H=spec.H, V=spec.V,
        q=mv(q), k_cache=mv(k_cache), v_cache=mv(v_cache),
        ctx_lens=mv(ctx), n_draft=mv(kd), cu_q=mv(cu_q),
        hidden=mv(hidden), w_lm=mv(w_lm),
        draft_tokens=mv(drafts.to(torch.int32)), draft_probs=mv(draft_probs),
        uniforms=mv(uniforms), mode=mv(mode), sigma=sigma,
    )


def make_qkv_inputs(spec: WorkloadSpec, R: int, device="cpu"):
    """Inputs of the verify block's QKV projection: hidden states x [R, H] ~ N(0, 1) and
    w_qkv [(Hq + 2 Hkv) D, H] ~ N(0, 1/H) in bf16 (so q, k, v ~ N(0, 1)), drawn on the CPU
    from their own seed (the spec's + 500) and moved to ``device``."""
    gen = torch.Generator(device="cpu").manual_seed(spec.seed + 500)
    x = _bf16_normal(gen, (R, spec.H), 1.0, "cpu")
    w = _bf16_normal(gen, ((spec.Hq + 2 * spec.Hkv) * spec.D, spec.H), 1.0 / math.sqrt(spec.H), "cpu")
    return x.to(device), w.to(device)


def to_paged(wl, page_size: int, seed: int = 0, spare_pages: int = 3, device=None):
    """The workload's dense caches scattered into paged pools.

    Each sequence's cap slots are cut into pages of ``page_size`` slots, placed in a pool
    at positions given by a seeded random permutation (so neighbouring pages of a sequence
    are far apart), with ``spare_pages`` extra pages no sequence uses, filled with NaN.
    Returns dict(k_pool, v_pool [num_pages, Hkv, page_size, D] bf16, block_table [B, max_pages]
    int32, page_size, num_pages, max_pages) on ``device`` (default: the caches' device).
    """
    dev = wl["k_cache"].device if device is None else torch.device(device)
    B, Hkv, cap, D = wl["k_cache"].shape
    max_pages = (cap + page_size - 1) // page_size
    num_pages = B * max_pages + spare_pages
    gen = torch.Generator(device="cpu").manual_seed(seed)
    perm = torch.randperm(num_pages, generator=gen)
    table = perm[:B * max_pages].reshape(B, max_pages).to(torch.int32)
    pools = []
    for cache in (wl["k_cache"], wl["v_cache"]):
        c = cache.cpu()
        padded = torch.zeros((B, Hkv, max_pages * page_size, D), dtype=c.dtype)
        padded[:, :, :cap] = c
        pool = torch.full((num_pages, Hkv, page_size, D), float("nan"), dtype=c.dtype)
        blocks = padded.reshape(B, Hkv, max_pages, page_size, D).permute(0, 2, 1, 3, 4)
        pool[table.reshape(-1).long()] = blocks.reshape(B * max_pages, Hkv, page_size, D)
        pools.append(pool.to(dev))
    return dict(k_pool=pools[0], v_pool=pools[1], block_table=table.to(dev), page_size=page_size,
                num_pages=num_pages, max_pages=max_pages)
