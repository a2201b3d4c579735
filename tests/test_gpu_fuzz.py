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


def _page(i):
    return int(np.random.default_rng(9300 + i).choice([16, 64, 128]))


@pytest.mark.parametrize("i", range(N_CASES))
def test_accept_commit_fuzz(dev, i):
    """The fused accept + KV commit, dense or through a shuffled block table (alternating)."""
    spec = _spec(i)
    wl = W.make_workload(spec, device=dev, cache_pad=int(np.random.default_rng(9400 + i).integers(0, 20)))
    B = wl["B"]
    acc0, tok0, st0 = parity.gpu_accept(wl)
    ws = spade.accept_workspace(B, wl["R"], wl["H"], wl["V"], device=dev)
    acc = torch.full((B,), -7, dtype=torch.int32, device=dev)
    tok = torch.full((B,), -7, dtype=torch.int32, device=dev)
    st = spade.status_tensor(dev)
    ctx = wl["ctx_lens"].clone()
    if i % 2:
        page = _page(i)
        pg = W.to_paged(wl, page, seed=i)
        k0, v0 = parity.to_np(pg["k_pool"]), parity.to_np(pg["v_pool"])
        spade.spade_verify_accept_commit_paged(wl["hidden"], wl["w_lm"], wl["draft_tokens"], wl["draft_probs"],
                                               wl["uniforms"], wl["mode"], wl["cu_q"], wl["n_draft"], acc, tok,
                                               pg["k_pool"], pg["v_pool"], pg["block_table"], ctx, workspace=ws,
                                               status=st)
        torch.cuda.synchronize()
        rk, rv, rctx = O_kv_commit_paged(k0, v0, pg, wl, acc, page)
        np.testing.assert_array_equal(parity.to_np(pg["k_pool"]), rk)
        np.testing.assert_array_equal(parity.to_np(pg["v_pool"]), rv)
    else:
        before = {k: wl[k].clone() for k in ("k_cache", "v_cache", "ctx_lens", "n_draft")}
        spade.spade_verify_accept_commit(wl["hidden"], wl["w_lm"], wl["draft_tokens"], wl["draft_probs"],
                                         wl["uniforms"], wl["mode"], wl["cu_q"], wl["n_draft"], acc, tok,
                                         wl["k_cache"], wl["v_cache"], ctx, workspace=ws, status=st)
        torch.cuda.synchronize()
        parity.check_commit_windows(before, wl["k_cache"], wl["v_cache"], ctx, acc)
        rctx = parity.to_np(before["ctx_lens"]) + parity.to_np(acc) + 1
    assert int(st0.item()) & ~spade.DEV_FALLBACK == 0 and int(st.item()) & ~spade.DEV_FALLBACK == 0
    assert torch.equal(acc, acc0) and torch.equal(tok, tok0)
    assert np.array_equal(parity.to_np(ctx), rctx)


def O_kv_commit_paged(k0, v0, pg, wl, acc, page):
    import oracle.spade_oracle as O
    return O.kv_commit_paged(k0, v0, parity.to_np(pg["block_table"]), parity.to_np(wl["ctx_lens"]),
                             parity.to_np(acc), parity.to_np(wl["n_draft"]), page)


@pytest.mark.parametrize("i", range(N_CASES))
def test_qkv_rope_fuzz(dev, i):
    """The QKV projection with rotary embedding (dense caches)."""
    spec = _spec(i)
    wl = W.make_workload(spec, device=dev, cache_pad=7)
    x, w = W.make_qkv_inputs(spec, wl["R"], device=dev)
    if (spec.Hq + 2 * spec.Hkv) * spec.D % 128:
        # The projection's rows come in 128-row tiles: such shapes are refused before any launch.
        with pytest.raises(spade.SpadeError) as e:
            parity.gpu_qkv_rope(wl, x, w)
        assert e.value.status == 2
        return
    k0, v0 = wl["k_cache"].clone(), wl["v_cache"].clone()
    q, st = parity.gpu_qkv_rope(wl, x, w)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    parity.check_qkv_rope(wl, x, w, q, k0, v0)


@pytest.mark.parametrize("i", range(0, N_CASES, 3))
def test_paged_attention_fuzz(dev, i):
    """Paged attention equals the dense attention on the gathered pages (page sizes 64, 128)."""
    spec = _spec(i)
    wl = W.make_workload(spec, device=dev, cache_pad=11)
    page = 64 if i % 2 else 128
    pg = W.to_paged(wl, page, seed=i)
    cap = pg["max_pages"] * page
    B, mp = pg["block_table"].shape

    def dense(pool):
        g = pool[pg["block_table"].reshape(-1).long()].reshape(B, mp, *pool.shape[1:]).permute(0, 2, 1, 3, 4)
        return g.reshape(B, pool.shape[1], mp * page, pool.shape[3]).contiguous()

    out, lse, st = parity.gpu_attention(dict(wl, cap=cap, k_cache=dense(pg["k_pool"]), v_cache=dense(pg["v_pool"])))
    max_k = int(wl["n_draft"].max())
    out_p = torch.empty_like(out)
    lse_p = torch.empty_like(lse)
    st_p = spade.status_tensor(dev)
    ws = spade.attn_workspace(B, wl["Hq"], wl["Hkv"], wl["D"], cap, max_k, device=dev)
    spade.spade_verify_attention_paged(wl["q"], pg["k_pool"], pg["v_pool"], pg["block_table"], wl["ctx_lens"],
                                       wl["n_draft"], wl["cu_q"], out_p, lse_p, max_k=max_k, workspace=ws, status=st_p)
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(st_p.item()) == 0
    assert torch.equal(out_p, out) and torch.equal(lse_p, lse)


TWO_PASS = [W.WorkloadSpec(f"fuzz_two_pass{j}", B=b, Hq=4, Hkv=2, D=64, H=h, V=v, ctx=(1, 64), k=(kl, 10),
                           mode=m, target_accept=0.7, logit_scale=s, seed=9500 + j)
            for j, (b, h, v, kl, m, s) in enumerate([(40, 200, 7000, 5, "mixed", 1.0), (60, 128, 3001, 3, "stochastic", 4.0),
                                                    (45, 320, 12000, 6, "greedy", 1.0), (33, 512, 9999, 7, "stochastic", 1.0)])]


@pytest.mark.parametrize("j", range(len(TWO_PASS)))
def test_two_pass_accept_fuzz(dev, j):
    """More rows than TMEM keeps resident: the statistics pass and the sampling pass."""
    wl = W.make_workload(TWO_PASS[j], device=dev)
    assert spade.spade_accept_launches(wl["B"], wl["R"], wl["H"], wl["V"]) == 2
    temp = np.random.default_rng(9600 + j).uniform(0.6, 1.5, wl["B"]).astype(np.float32) if j % 2 else None
    acc, tok, st = parity.gpu_accept_sampling(wl, temperature=None if temp is None else torch.from_numpy(temp).to(dev))
    torch.cuda.synchronize()
    assert int(st.item()) & ~spade.DEV_FALLBACK == 0
    ref = parity.oracle_accept_from_logits(wl, parity.oracle_logits(wl), temperature=temp)
    cmp = parity.compare_accept(acc, tok, ref)
    assert cmp["mismatch_unflagged"] == 0, cmp


def _wide_spec(i):
    """Wide vocabularies (slices past the shared-memory staging: the register path of the
    residual sums) and long contexts (units split across many CTAs)."""
    g = np.random.default_rng(9700 + i)
    D = int(g.choice([64, 128]))
    Hkv = int(g.choice([1, 2, 4]))
    G = int(g.choice([1, 4, 8]))
    B = int(g.integers(1, 12))
    k_hi = int(g.integers(0, 9))
    c_hi = int(g.choice([4000, 12000, 20000]))
    return W.WorkloadSpec(f"fuzz_wide{i}", B=B, Hq=Hkv * G, Hkv=Hkv, D=D, H=int(g.choice([128, 256])),
                          V=int(g.integers(100000, 160000)), ctx=(int(g.integers(0, c_hi)), c_hi),
                          k=(int(g.integers(0, k_hi + 1)), k_hi),
                          mode=str(g.choice(["stochastic", "mixed"])), target_accept=0.7,
                          logit_scale=float(g.choice([1.0, 4.0, 8.0])), seed=9800 + i)


@pytest.mark.parametrize("i", range(10))
def test_wide_fuzz(dev, i):
    spec = _wide_spec(i)
    wl = W.make_workload(spec, device=dev, cache_pad=5)
    out, lse, st = parity.gpu_attention(wl)
    B = wl["B"]
    g = np.random.default_rng(9900 + i)
    temp = g.uniform(0.5, 1.6, B).astype(np.float32) if g.random() < 0.5 else None
    one_launch = spade.spade_accept_launches(B, wl["R"], wl["H"], wl["V"]) == 1
    tp = g.uniform(0.5, 1.0, B).astype(np.float32) if (one_launch and g.random() < 0.6) else None
    acc, tok, st2 = parity.gpu_accept_sampling(wl, temperature=None if temp is None else torch.from_numpy(temp).to(dev),
                                               top_p=None if tp is None else torch.from_numpy(tp).to(dev))
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(st2.item()) & ~spade.DEV_FALLBACK == 0
    R, Hq = wl["R"], wl["Hq"]
    pairs = sorted({(int(r), int(h)) for r, h in zip(g.integers(0, R, 48), g.integers(0, Hq, 48))})
    ref, _ = parity.oracle_attention(wl, rows=pairs)
    n, bad, worst = parity.compare_attention(out, ref, rows=pairs)
    assert bad == 0, (spec, worst)
    ref_a = parity.oracle_accept_from_logits(wl, parity.oracle_logits(wl), temperature=temp, top_p=tp)
    cmp = parity.compare_accept(acc, tok, ref_a)
    assert cmp["mismatch_unflagged"] == 0, (spec, temp is not None, tp is not None, cmp)
