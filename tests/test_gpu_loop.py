"""Algorithm 1 end to end on the GPU: rounds of drafts and verifier calls through the library
with a toy one-layer verifier (paper_2608_13076_gb300.speculative)."""
import numpy as np
import pytest
import torch

from paper_2608_13076_gb300 import speculative as S

pytestmark = pytest.mark.gpu

B, MAX_NEW = 6, 40


@pytest.fixture(scope="module")
def verifier(gpu_lib):
    cfg = S.ToyConfig()
    return S.ToyVerifier(cfg, B, cap=1024, seed=3, device="cuda:0")


def _prompts(V, seed=4):
    g = np.random.default_rng(seed)
    return [list(g.integers(0, V - 1, size=int(n))) for n in g.integers(2, 40, size=B)]


def test_greedy_speculative_equals_plain_decoding(verifier):
    """Greedy verification makes the output independent of the drafts (Sec. III-B): for every
    draft length the tokens are those of plain greedy decoding with the verifier alone.  The
    two runs compute the same logits in different batch shapes, so a near tie (top-2 gap
    below 0.05, logits ~ N(0, 16)) may break the other way; a sequence may diverge only there."""
    prompts = _prompts(verifier.cfg.V)
    ref = S.speculative_decode(verifier, prompts, d=0, max_new=MAX_NEW, record_margins=True)
    assert ref.calls_per_seq == [len(t) for t in ref.tokens]  # one token per call
    for d in (1, 3, 6):
        res = S.speculative_decode(verifier, prompts, d=d, max_new=MAX_NEW)
        identical = 0
        for b in range(B):
            a, r = res.tokens[b], ref.tokens[b]
            i = next((j for j in range(min(len(a), len(r))) if a[j] != r[j]), None)
            if i is None:
                assert len(a) == len(r), (d, b)
                identical += 1
            else:
                assert ref.margins[b][i] < 0.05, (d, b, i, ref.margins[b][i])
        assert identical >= B - 1, (d, identical)
        assert sum(res.calls_per_seq) < sum(ref.calls_per_seq)  # fewer verifier calls


def test_stochastic_loop_runs_and_accepts(verifier):
    prompts = _prompts(verifier.cfg.V, seed=5)
    res = S.speculative_decode(verifier, prompts, d=4, max_new=MAX_NEW, mode=S.STOCHASTIC, seed=9)
    V = verifier.cfg.V
    for t in res.tokens:
        assert 1 <= len(t) <= MAX_NEW and all(0 <= x < V for x in t)
    assert 0 < res.accepted < res.drafted
    assert int(verifier.status.item()) & ~0x8 == 0


def test_stochastic_with_a_one_token_nucleus_equals_greedy_decoding(verifier):
    """top_p -> 0 leaves the verifier's argmax alone in its nucleus: a draft equal to it is
    accepted (p_S(d) / q(d) = 1 / q(d) >= 1 > u), any other rejected (p_S(d) = 0), and the
    residual max(0, p_S - q) has its mass on the argmax.  So stochastic speculative decoding
    through the top-p path must reproduce plain greedy decoding token for token, whatever the
    drafts and uniforms (a sequence may diverge only at a near tie, as above)."""
    prompts = _prompts(verifier.cfg.V, seed=6)
    ref = S.speculative_decode(verifier, prompts, d=0, max_new=MAX_NEW, record_margins=True)
    for d in (1, 4):
        res = S.speculative_decode(verifier, prompts, d=d, max_new=MAX_NEW, mode=S.STOCHASTIC, seed=10 + d,
                                   top_p=1e-6, temperature=0.7)
        identical = 0
        for b in range(B):
            a, r = res.tokens[b], ref.tokens[b]
            i = next((j for j in range(min(len(a), len(r))) if a[j] != r[j]), None)
            if i is None:
                assert len(a) == len(r), (d, b)
                identical += 1
            else:
                assert ref.margins[b][i] < 0.05, (d, b, i, ref.margins[b][i])
        assert identical >= B - 1, (d, identical)
        assert 0 < res.accepted < res.drafted  # drafts from q: some match the argmax, some not
    assert int(verifier.status.item()) & ~0x8 == 0
