"""A multi-step speculative-decoding loop (Algorithm 1) on the GPU with a toy verifier.

The cloud verifier is a small random one-layer decoder whose verify step runs
through this library: the QKV projection with rotary embedding writes the
verify block's keys and values into the cache (spade_verify_qkv_rope), the
verify attention reads them (spade_verify_attention), the output projection
adds the attention to the residual stream (x_{l+1} = x_l + f_l(x_l), Sec.
III-A; a plain bf16 matmul), and the LM head with the fused accept test,
residual sampling and KV commit closes the step (spade_verify_accept_commit).
The edge drafter proposes d tokens per round from a cheap model whose logits
are the verifier's without the attention term (its residual path only), so
its q is correlated with the verifier's p, as a real draft model's is.

Each round: the drafter proposes d tokens (greedy: its argmax; stochastic: a
draw from q, which is sent along), the verifier scores the d + 1 positions in
one call, and every sequence appends its accepted drafts plus the correction
or bonus token (Algorithm 1's cloud step and context update).  The loop runs
until each sequence has produced `max_new` tokens or its end-of-sequence
token, and reports verifier calls against tokens, the quantity the paper's
cloud-call reduction is about (Sec. IV).

This is a toy model for exercising and measuring the verify path end to end;
it is not a trained model.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch

from . import (accept_workspace, attn_workspace, qkv_workspace, spade_verify_accept_commit,
               spade_verify_accept_sampling, spade_verify_attention, spade_verify_qkv_rope, status_tensor)

GREEDY = 0
STOCHASTIC = 1


@dataclass
class ToyConfig:
    V: int = 2048        # vocabulary (token V - 1 is the end-of-sequence token)
    H: int = 512         # hidden size
    Hq: int = 8          # query heads
    Hkv: int = 2         # key/value heads
    D: int = 64          # head dimension
    rope_theta: float = 10000.0
    logit_scale: float = 4.0  # sharpens the toy distributions (logits ~ N(0, scale^2))


class ToyVerifier:
    """Random one-layer decoder (embedding, attention layer, LM head) with a KV cache of
    `cap` slots for each of `B` sequences, on `device`; weights drawn on the CPU from `seed`."""

    def __init__(self, cfg: ToyConfig, B: int, cap: int, seed: int, device):
        self.cfg, self.B, self.cap = cfg, B, cap
        dev = torch.device(device)
        g = torch.Generator().manual_seed(seed)

        def normal(shape, std):
            return (torch.randn(shape, generator=g) * std).to(torch.bfloat16).to(dev)

        c = cfg
        self.emb = normal((c.V, c.H), 1.0)
        self.w_qkv = normal(((c.Hq + 2 * c.Hkv) * c.D, c.H), 1.0 / math.sqrt(c.H))
        self.w_o = normal((c.H, c.Hq * c.D), 1.0 / math.sqrt(c.Hq * c.D))
        self.w_lm = normal((c.V, c.H), c.logit_scale / math.sqrt(c.H))
        self.k_cache = torch.zeros((B, c.Hkv, cap, c.D), dtype=torch.bfloat16, device=dev)
        self.v_cache = torch.zeros_like(self.k_cache)
        self.ctx = torch.zeros(B, dtype=torch.int32, device=dev)
        self.status = status_tensor(dev)
        self.device = dev

    def draft_logits(self, tokens):
        """The drafter's logits after `tokens` [n]: the verifier's residual path without its
        attention term, fp32 [n, V]."""
        return self.emb[tokens].float() @ self.w_lm.float().t()

    def write_prefix(self, tokens, ctx, kd, cu_q, max_k):
        """K/V of prompt tokens (no output needed: one layer)."""
        x = self.emb[tokens].contiguous()
        q = torch.empty((x.shape[0], self.cfg.Hq, self.cfg.D), dtype=torch.bfloat16, device=self.device)
        spade_verify_qkv_rope(x, self.w_qkv, ctx, kd, cu_q, q, self.k_cache, self.v_cache, Hq=self.cfg.Hq,
                              Hkv=self.cfg.Hkv, rope_theta=self.cfg.rope_theta, max_k=max_k,
                              workspace=qkv_workspace(x.shape[0], self.cfg.Hq, self.cfg.Hkv, self.cfg.D,
                                                      device=self.device), status=self.status)

    def verify(self, tokens, kd, cu_q, drafts, draft_probs, uniforms, mode, max_k, temperature=None, top_p=None):
        """One verify call over the blocks (row cu_q[b] + i holds token i of sequence b's
        block, position ctx_b + i): returns (accepted_len, next_token); the cache and ctx
        are committed (accepted slots kept, rejected ones cleared, ctx += a + 1).  With
        ``temperature`` / ``top_p`` ([B] float32) the verifier's p is softmax(l / T) cut to
        its nucleus."""
        c = self.cfg
        R = tokens.numel()
        x = self.emb[tokens].contiguous()
        q = torch.empty((R, c.Hq, c.D), dtype=torch.bfloat16, device=self.device)
        spade_verify_qkv_rope(x, self.w_qkv, self.ctx, kd, cu_q, q, self.k_cache, self.v_cache, Hq=c.Hq,
                              Hkv=c.Hkv, rope_theta=c.rope_theta, max_k=max_k,
                              workspace=qkv_workspace(R, c.Hq, c.Hkv, c.D, device=self.device), status=self.status)
        out = torch.empty_like(q)
        ws = attn_workspace(self.B, c.Hq, c.Hkv, c.D, self.cap, max_k, device=self.device)
        spade_verify_attention(q, self.k_cache, self.v_cache, self.ctx, kd, cu_q, out, None, max_k=max_k,
                               workspace=ws, status=self.status)
        hidden = (x.float() + out.reshape(R, c.Hq * c.D).float() @ self.w_o.float().t()).to(torch.bfloat16)
        acc = torch.empty(self.B, dtype=torch.int32, device=self.device)
        tok = torch.empty_like(acc)
        wsa = accept_workspace(self.B, R, c.H, c.V, device=self.device)
        if temperature is None and top_p is None:
            spade_verify_accept_commit(hidden.contiguous(), self.w_lm, drafts, draft_probs, uniforms, mode, cu_q,
                                       kd, acc, tok, self.k_cache, self.v_cache, self.ctx, workspace=wsa,
                                       status=self.status)
        else:
            spade_verify_accept_sampling(hidden.contiguous(), self.w_lm, drafts, draft_probs, uniforms, mode, cu_q,
                                         kd, acc, tok, workspace=wsa, status=self.status, temperature=temperature,
                                         top_p=top_p, k_cache=self.k_cache, v_cache=self.v_cache,
                                         ctx_lens=self.ctx)
        self.last_hidden = hidden
        return acc, tok


@dataclass
class LoopResult:
    tokens: list          # per sequence: the generated tokens after the prompt (<= max_new)
    calls: int            # verifier calls of the whole batch
    calls_per_seq: list   # verifier calls until each sequence was done
    drafted: int          # drafts proposed for sequences not yet done
    accepted: int         # of those, drafts the verifier accepted
    margins: list         # with record_margins and d = 0: per sequence, the top-2 logit gap of each token


def speculative_decode(ver: ToyVerifier, prompts, d: int, max_new: int, mode: int = GREEDY, seed: int = 0,
                       eos: int | None = None, record_margins: bool = False, temperature: float | None = None,
                       top_p: float | None = None) -> LoopResult:
    """Algorithm 1 for a batch of prompts (each at least 2 tokens): rounds of d drafts and one
    verifier call, until every sequence has max_new tokens or has emitted `eos` (default
    V - 1).  d = 0 is plain decoding with the verifier alone.  Stochastic mode draws the
    drafts from q = softmax(drafter logits) and the uniforms from a CPU generator seeded
    with `seed`; `temperature` and `top_p` (one value for every sequence) shape the
    verifier's p.  The verifier's cache must hold every prompt plus max_new * (d + 1) + d + 1
    slots (sequences that are done keep stepping with the batch)."""
    B, cfg, dev = ver.B, ver.cfg, ver.device
    eos = cfg.V - 1 if eos is None else eos
    assert len(prompts) == B and all(len(p) >= 2 for p in prompts)
    need = max(len(p) for p in prompts) + max_new * (d + 1) + d + 1
    if need > ver.cap:
        raise ValueError(f"cache of {ver.cap} slots is too small; this loop needs {need}")
    gen = torch.Generator().manual_seed(seed)
    # Prefill: the prompt tokens before the last one go into the cache.
    pre = [torch.tensor(p[:-1], dtype=torch.long) for p in prompts]
    lens = torch.tensor([len(x) for x in pre], dtype=torch.int32)
    cu = torch.zeros(B + 1, dtype=torch.int32)
    cu[1:] = torch.cumsum(lens, 0)
    ver.ctx.zero_()
    ver.write_prefix(torch.cat(pre).to(dev), ver.ctx, (lens - 1).to(dev), cu.to(dev), int(lens.max()) - 1)
    ver.ctx.copy_(lens.to(dev))
    last = torch.tensor([p[-1] for p in prompts], dtype=torch.long, device=dev)
    mode_t = torch.full((B,), mode, dtype=torch.int32, device=dev)
    temp_t = None if temperature is None else torch.full((B,), temperature, dtype=torch.float32, device=dev)
    top_p_t = None if top_p is None else torch.full((B,), top_p, dtype=torch.float32, device=dev)
    kd = torch.full((B,), d, dtype=torch.int32, device=dev)
    cu_q = (torch.arange(B + 1, dtype=torch.int32) * (d + 1)).to(dev)
    out = [[] for _ in range(B)]
    margins = [[] for _ in range(B)]
    done = [False] * B
    calls, calls_per_seq, drafted, accepted = 0, [0] * B, 0, 0
    while not all(done):
        cur = last
        drafts, qrows = [], []
        for _ in range(d):
            lg = ver.draft_logits(cur)
            if mode == GREEDY:
                nxt = lg.argmax(-1)
            else:
                qd = torch.softmax(lg, dim=-1)
                nxt = torch.multinomial(qd.cpu(), 1, generator=gen).flatten().to(dev)
                qrows.append(qd)
            drafts.append(nxt)
            cur = nxt
        rows = torch.stack([last] + drafts, dim=1)  # [B, d + 1]: last accepted token, then the drafts
        dr = torch.stack(drafts, dim=1).reshape(-1).to(torch.int32) if d else \
            torch.empty(0, dtype=torch.int32, device=dev)
        qp = torch.stack(qrows, dim=1).reshape(B * d, cfg.V).contiguous() if (d and mode == STOCHASTIC) else None
        u = torch.rand(B * (d + 1), generator=gen).to(dev)
        acc, tok = ver.verify(rows.reshape(-1), kd, cu_q, dr, qp, u, mode_t, d, temperature=temp_t, top_p=top_p_t)
        calls += 1
        acc_l, tok_l = acc.tolist(), tok.tolist()
        gap_l = None
        if record_margins and d == 0:
            # Diagnostic beside the decision: the top-2 gap of the row that emitted each token.
            top = (ver.last_hidden.float() @ ver.w_lm.float().t()).topk(2, dim=-1).values
            gap_l = (top[:, 0] - top[:, 1]).tolist()
        dr_l = rows[:, 1:].tolist()
        for b in range(B):
            if not done[b]:
                calls_per_seq[b] += 1
                drafted += d
                accepted += acc_l[b]
                for t in dr_l[b][:acc_l[b]] + [tok_l[b]]:
                    if len(out[b]) < max_new and not (out[b] and out[b][-1] == eos):
                        out[b].append(t)
                        if gap_l is not None:
                            margins[b].append(gap_l[b])
                done[b] = len(out[b]) >= max_new or (bool(out[b]) and out[b][-1] == eos)
        last = tok.to(torch.long)
    if int(ver.status.item()) & ~0x8:
        raise RuntimeError(f"device status {int(ver.status.item())} in the decoding loop")
    return LoopResult(out, calls, calls_per_seq, drafted, accepted, margins)
