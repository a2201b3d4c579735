"""Seeded random shapes through the attention and the LM head / accept kernels, against the oracle.

Each case draws its shape from a fixed seed: head dims 64 and 128, GQA ratios 1-8, contexts from
empty to a few thousand slots, draft lengths 0-10, vocabularies whose slices end in ragged tiles,
hidden sizes with a partial last k-chunk, greedy / stochastic / mixed batches, the one-launch and
the two-launch LM head, and (one-launch shapes) temperature and top-p.  Sizes stay small enough for
the float64 oracle to finish in seconds.
"""
import numpy as np
import pytest
import torch

import paper_2608_13076_gb300 as spade
from paper_2608_13076_gb300 import workloads as W
from tests import parity

pytestmark = pytest.mark.gpu

N_CASES = 40


@pytest.fixture(scope="module")
def dev(gpu_lib):
    return torch.device("cuda:0")


def _spec(i):
    g = np.random.default_rng(9000 + i)
    D = int(g.choice([64, 128]))
    Hkv = int(g.choice([1, 2, 4, 8]))
    G = int(g.choice([1, 2, 4, 8]))
    B = int(g.integers(1, 40))
    k_hi = int(g.integers(0, 11))
    k_lo = int(g.integers(0, k_hi + 1))
    c_hi = int(g.choice([0, 64, 700, 3000]))
    c_lo = int(g.integers(0, c_hi + 1))
    H = int(g.choice([128, 200, 320, 512]))  # 200: a partial last k-chunk
    V = int(g.integers(300, 20000))
    mode = str(g.choice(["greedy", "stochastic", "mixed"], p=[0.2, 0.4, 0.4]))
    scale = float(g.choice([1.0, 4.0]))
    return W.WorkloadSpec(f"fuzz{i}", B=B, Hq=Hkv * G, Hkv=Hkv, D=D, H=H, V=V, ctx=(c_lo, c_hi), k=(k_lo, k_hi),
                          mode=mode, target_accept=0.7, logit_scale=scale, seed=9100 + i)


@pytest.mark.parametrize("i", range(N_CASES))
def test_attention_fuzz(dev, i):
    spec = _spec(i)
    wl = W.make_workload(spec, device=dev, cache_pad=33)
    for b in range(wl["B"]):  # unused slots poisoned: they must not reach the result
        L = int(wl["ctx_lens"][b] + wl["n_draft"][b] + 1)
        wl["k_cache"][b, :, L:] = float("nan")
        wl["v_cache"][b, :, L:] = float("nan")
    out, lse, st = parity.gpu_attention(wl)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ref, _ = parity.oracle_attention(wl)
    n, bad, worst = parity.compare_attention(out, ref)
    assert bad == 0, (spec, worst)


@pytest.mark.parametrize("i", range(N_CASES))
def test_accept_fuzz(dev, i):
    spec = _spec(i)
    wl = W.make_workload(spec, device=dev)
    B, R = wl["B"], wl["R"]
    one_launch = spade.spade_accept_launches(B, R, wl["H"], wl["V"]) == 1
    g = np.random.default_rng(9200 + i)
    temp = g.uniform(0.5, 1.6, B).astype(np.float32) if g.random() < 0.5 else None
    tp = g.uniform(0.4, 1.0, B).astype(np.float32) if (one_launch and g.random() < 0.6) else None
    acc, tok, st = parity.gpu_accept_sampling(wl, temperature=None if temp is None else torch.from_numpy(temp).to(dev),
                                              top_p=None if tp is None else torch.from_numpy(tp).to(dev))
    torch.cuda.synchronize()
    assert int(st.item()) & ~spade.DEV_FALLBACK == 0
    ref = parity.oracle_accept_from_logits(wl, parity.oracle_logits(wl), temperature=temp, top_p=tp)
    cmp = parity.compare_accept(acc, tok, ref)
    assert cmp["mismatch_unflagged"] == 0, (spec, temp is not None, tp is not None, cmp)
