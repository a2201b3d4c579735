"""GPU parity of the verifier's sampling options: top-p (nucleus) truncation of p, alone and
with temperature, through spade_verify_accept_sampling against the float64 oracle.

The workloads draw hidden rows with a larger spread (logits ~ N(0, 4^2) or wider) so that the
nucleus boundary usually sits on a token of sizeable probability: with N(0, 1) logits over
thousands of tokens every boundary step is far below the oracle's margin and each decision
would be flagged, which would leave nothing to compare.
"""
import dataclasses

import numpy as np
import pytest
import torch

import paper_2608_13076_gb300 as spade
from paper_2608_13076_gb300 import workloads as W
from tests import parity

pytestmark = pytest.mark.gpu

TOPP = {
    "topp_resident": W.WorkloadSpec("topp_resident", B=16, Hq=4, Hkv=4, D=64, H=256, V=5000, ctx=(1, 64),
                                    k=(1, 6), mode="stochastic", target_accept=0.7, logit_scale=4.0, seed=71),
    # Greedy sequences beside stochastic ones, bonus-only rows (k = 0), a ragged vocabulary tail.
    "topp_mixed_modes": W.WorkloadSpec("topp_mixed_modes", B=12, Hq=4, Hkv=4, D=64, H=256, V=3001,
                                       ctx=(1, 64), k=(0, 5), mode="mixed", target_accept=0.7,
                                       logit_scale=4.0, seed=73),
    # Slices wider than the shared-memory staging: the register path of the residual sums.
    "topp_wide_slices": W.WorkloadSpec("topp_wide_slices", B=8, Hq=4, Hkv=4, D=64, H=256, V=160000,
                                       ctx=(1, 64), k=(1, 3), mode="stochastic", target_accept=0.7,
                                       logit_scale=8.0, seed=72),
    # 256 verify rows, all listed for the nucleus search.
    "topp_many_rows": W.WorkloadSpec("topp_many_rows", B=32, Hq=4, Hkv=4, D=64, H=256, V=5000,
                                     ctx=(1, 64), k=(7, 7), mode="stochastic", target_accept=0.7,
                                     logit_scale=4.0, seed=74),
}


@pytest.fixture(scope="module")
def dev(gpu_lib):
    return torch.device("cuda:0")


def _top_p(B, seed):
    """top_p in [0.3, 0.99]; sequence 0 keeps all of p (top_p = 1)."""
    tp = np.random.default_rng(seed).uniform(0.3, 0.99, B).astype(np.float32)
    tp[0] = 1.0
    return tp


def _temperature(B, seed):
    return np.random.default_rng(seed).uniform(0.6, 1.5, B).astype(np.float32)


def _changed_unflagged(ref, ref_plain):
    """Sequences whose oracle decision changes with top-p and that neither run flags."""
    changed = (ref["accepted_len"] != ref_plain["accepted_len"]) | (ref["next_token"] != ref_plain["next_token"])
    flags = ref["flag_decision"] | ref["flag_sample"] | ref_plain["flag_decision"] | ref_plain["flag_sample"]
    return int(np.sum(changed & ~flags))


def _dev_f32(x, dev):
    return None if x is None else torch.from_numpy(x).to(dev)


@pytest.mark.parametrize("with_temp", [False, True])
@pytest.mark.parametrize("name", sorted(TOPP))
def test_accept_top_p(dev, name, with_temp):
    wl = W.make_workload(TOPP[name], device=dev)
    B = wl["B"]
    assert spade.spade_accept_launches(B, wl["R"], wl["H"], wl["V"]) == 1
    tp = _top_p(B, 5)
    T = _temperature(B, 6) if with_temp else None
    acc, tok, st = parity.gpu_accept_sampling(wl, temperature=_dev_f32(T, dev), top_p=_dev_f32(tp, dev))
    torch.cuda.synchronize()
    assert int(st.item()) & ~spade.DEV_FALLBACK == 0
    logits = parity.oracle_logits(wl)
    ref = parity.oracle_accept_from_logits(wl, logits, temperature=T, top_p=tp)
    cmp = parity.compare_accept(acc, tok, ref)
    print(f"{name} T={with_temp}: accepted {parity.to_np(acc).tolist()} flagged {cmp['flagged']}")
    assert cmp["mismatch_unflagged"] == 0, cmp
    # Not vacuous: top-p changes some unflagged decision of the oracle.
    ref_plain = parity.oracle_accept_from_logits(wl, logits, temperature=T)
    assert _changed_unflagged(ref, ref_plain) >= 1


def test_accept_top_p_full_size_commit(dev):
    """Llama-3-8B shapes (V = 128256, H = 4096, 8 sequences of 8 drafts) with temperature,
    top-p and the fused KV commit in one launch."""
    spec = dataclasses.replace(W.SPECS["llama3_8b"], name="llama3_8b_top_p", logit_scale=6.0)
    wl = W.make_workload(spec, device=dev)
    B = wl["B"]
    before = {k: wl[k].clone() for k in ("k_cache", "v_cache", "ctx_lens", "n_draft")}
    tp = _top_p(B, 7)
    T = _temperature(B, 8)
    acc, tok, st = parity.gpu_accept_sampling(wl, temperature=_dev_f32(T, dev), top_p=_dev_f32(tp, dev),
                                              commit=True)
    torch.cuda.synchronize()
    assert int(st.item()) & ~spade.DEV_FALLBACK == 0
    logits = parity.oracle_logits(wl)
    ref = parity.oracle_accept_from_logits(wl, logits, temperature=T, top_p=tp)
    cmp = parity.compare_accept(acc, tok, ref)
    print(f"llama3_8b top-p: accepted {parity.to_np(acc).tolist()} flagged {cmp['flagged']}")
    assert cmp["mismatch_unflagged"] == 0, cmp
    parity.check_commit_windows(before, wl["k_cache"], wl["v_cache"], wl["ctx_lens"], acc)


def test_top_p_one_is_the_plain_call(dev):
    """top_p = 1 everywhere leaves p whole: the same decisions, bit for bit, as the call
    without sampling options (and as the sampling entry with neither option)."""
    wl = W.make_workload(TOPP["topp_mixed_modes"], device=dev)
    B = wl["B"]
    a0, t0, s0 = parity.gpu_accept(wl)
    a1, t1, s1 = parity.gpu_accept_sampling(wl, top_p=torch.ones(B, dtype=torch.float32, device=dev))
    a2, t2, s2 = parity.gpu_accept_sampling(wl)
    torch.cuda.synchronize()
    for s in (s0, s1, s2):
        assert int(s.item()) & ~spade.DEV_FALLBACK == 0
    assert torch.equal(a0, a1) and torch.equal(t0, t1)
    assert torch.equal(a0, a2) and torch.equal(t0, t2)


def test_top_p_tiny_keeps_the_argmax(dev):
    """A nucleus of the top token alone: every stochastic sequence emits the argmax of the
    row it samples (residual or bonus), as the oracle does."""
    wl = W.make_workload(TOPP["topp_resident"], device=dev)
    B = wl["B"]
    tp = np.full(B, 1e-6, dtype=np.float32)
    acc, tok, st = parity.gpu_accept_sampling(wl, top_p=_dev_f32(tp, dev))
    torch.cuda.synchronize()
    assert int(st.item()) & ~spade.DEV_FALLBACK == 0
    logits = parity.oracle_logits(wl)
    ref = parity.oracle_accept_from_logits(wl, logits, top_p=tp)
    cmp = parity.compare_accept(acc, tok, ref)
    assert cmp["mismatch_unflagged"] == 0, cmp
    a, t = parity.to_np(acc), parity.to_np(tok)
    cu = parity.to_np(wl["cu_q"])
    for b in range(B):
        if not (ref["flag_decision"][b] or ref["flag_sample"][b]):
            assert t[b] == int(np.argmax(logits[cu[b] + a[b]])), b


def test_top_p_invalid_values_are_reported_and_taken_as_one(dev):
    wl = W.make_workload(TOPP["topp_resident"], device=dev)
    B = wl["B"]
    tp = _top_p(B, 9)
    tp[1], tp[2], tp[3], tp[4] = 0.0, -0.5, 1.5, np.nan
    acc, tok, st = parity.gpu_accept_sampling(wl, top_p=_dev_f32(tp, dev))
    torch.cuda.synchronize()
    assert int(st.item()) & spade.DEV_BAD_INDEX
    fixed = tp.copy()
    fixed[1:5] = 1.0
    ref = parity.oracle_accept_from_logits(wl, parity.oracle_logits(wl), top_p=fixed)
    cmp = parity.compare_accept(acc, tok, ref)
    assert cmp["mismatch_unflagged"] == 0, cmp


def test_top_p_needs_the_one_launch_path(dev):
    spec = W.WorkloadSpec("topp_two_pass", B=40, Hq=4, Hkv=4, D=64, H=256, V=9100, ctx=(1, 64), k=(6, 9),
                          mode="stochastic", seed=75)
    wl = W.make_workload(spec, device=dev)
    assert spade.spade_accept_launches(wl["B"], wl["R"], wl["H"], wl["V"]) == 2
    tp = torch.full((wl["B"],), 0.9, dtype=torch.float32, device=dev)
    with pytest.raises(spade.SpadeError) as e:
        parity.gpu_accept_sampling(wl, top_p=tp)
    assert e.value.status == 2


@pytest.mark.parametrize("T", [0.05, 5.0])
def test_top_p_at_extreme_temperatures(dev, T):
    """T = 0.05 scales the logits twentyfold (most tokens fall more than 31.5 below the row
    maximum, outside the search's span), T = 5 flattens p (large nuclei): both against the oracle."""
    wl = W.make_workload(TOPP["topp_resident"], device=dev)
    B = wl["B"]
    tp = _top_p(B, 11)
    temp = np.full(B, T, dtype=np.float32)
    acc, tok, st = parity.gpu_accept_sampling(wl, temperature=_dev_f32(temp, dev), top_p=_dev_f32(tp, dev))
    torch.cuda.synchronize()
    assert int(st.item()) & ~spade.DEV_FALLBACK == 0
    ref = parity.oracle_accept_from_logits(wl, parity.oracle_logits(wl), temperature=temp, top_p=tp)
    cmp = parity.compare_accept(acc, tok, ref)
    assert cmp["mismatch_unflagged"] == 0, cmp
    assert cmp["flagged"] < B, cmp  # something is left to compare


@pytest.mark.parametrize("opts", ["plain", "temperature", "top_p"])
def test_stochastic_sequences_without_drafts(dev, opts):
    """k_b = 0 everywhere: no draft rows, so draft_probs is empty (a null pointer), and every
    stochastic sequence draws its token from p (Algorithm 1's bonus draw) -- not the argmax."""
    spec = W.WorkloadSpec("stoch_k0", B=24, Hq=4, Hkv=4, D=64, H=256, V=5000, ctx=(1, 64), k=(0, 0),
                          mode="mixed", seed=77)
    wl = W.make_workload(spec, device=dev)
    B = wl["B"]
    assert wl["draft_probs"] is None or wl["draft_probs"].numel() == 0
    temp = np.full(B, 1.3, dtype=np.float32) if opts == "temperature" else None
    tp = np.full(B, 0.9, dtype=np.float32) if opts == "top_p" else None
    acc, tok, st = parity.gpu_accept_sampling(wl, temperature=_dev_f32(temp, dev), top_p=_dev_f32(tp, dev))
    torch.cuda.synchronize()
    assert int(st.item()) & ~spade.DEV_FALLBACK == 0
    logits = parity.oracle_logits(wl)
    ref = parity.oracle_accept_from_logits(wl, logits, temperature=temp, top_p=tp)
    cmp = parity.compare_accept(acc, tok, ref)
    assert cmp["mismatch_unflagged"] == 0, cmp
    # Flat logits: the draws are not the argmax for most stochastic sequences.
    am = logits.argmax(-1)
    t = parity.to_np(tok)
    stoch = parity.to_np(wl["mode"]) == 1
    assert np.sum(t[stoch] != am[stoch]) >= stoch.sum() // 2


def test_stochastic_drafts_without_q_are_reported_and_verified_greedily(dev):
    spec = W.WorkloadSpec("stoch_noq", B=8, Hq=4, Hkv=4, D=64, H=256, V=3000, ctx=(1, 64), k=(1, 5),
                          mode="stochastic", match_prob=0.7, seed=78)
    wl = W.make_workload(spec, device=dev)
    acc, tok, st = parity.gpu_accept_sampling(dict(wl, draft_probs=None))
    torch.cuda.synchronize()
    assert int(st.item()) & spade.DEV_BAD_INDEX
    greedy = dict(wl, mode=torch.zeros_like(wl["mode"]), draft_probs=None)
    acc_g, tok_g, st_g = parity.gpu_accept_sampling(greedy)
    torch.cuda.synchronize()
    assert int(st_g.item()) == 0
    assert torch.equal(acc, acc_g) and torch.equal(tok, tok_g)
