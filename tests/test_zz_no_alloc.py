"""The allocation-free attention entry point against the workspace one.

Some callers cannot allocate device memory (plugin hosts that hand over only
inputs and outputs, serving loops with a frozen memory pool).  For them
spade_verify_attention_noalloc keeps its scratch in a static device array.
This file is collected last on purpose: it checks that entry point through the
C ABI, twice in a row on the same static scratch, against the regular entry
point with a caller workspace, and that oversized requests are refused.
"""
import ctypes

import pytest
import torch

import paper_2608_13076_gb300 as spade
from paper_2608_13076_gb300 import workloads as W
from tests import parity

pytestmark = pytest.mark.gpu

CASES = [
    # Cross-CTA split merges (long context, one KV head) and GQA with ragged rows.
    W.WorkloadSpec("noalloc_long", B=1, Hq=8, Hkv=1, D=128, H=256, V=512, ctx=(20000, 20000), k=(6, 6),
                   mode="greedy", seed=31),
    W.WorkloadSpec("noalloc_gqa", B=5, Hq=16, Hkv=4, D=128, H=256, V=512, ctx=(40, 3000), k=(0, 9),
                   mode="greedy", seed=32),
    W.WorkloadSpec("noalloc_d64", B=3, Hq=8, Hkv=8, D=64, H=256, V=512, ctx=(1, 900), k=(1, 4),
                   mode="greedy", seed=33),
]


@pytest.mark.parametrize("spec", CASES, ids=lambda s: s.name)
def test_noalloc_matches_workspace_entry_point(gpu_lib, spec):
    dev = torch.device("cuda:0")
    wl = W.make_workload(spec, device=dev)
    ref, ref_lse, st = parity.gpu_attention(wl)
    max_k = int(wl["n_draft"].max())
    outs = []
    for _ in range(2):
        out = torch.full_like(wl["q"], float("nan"))
        lse = torch.full(wl["q"].shape[:2], float("nan"), dtype=torch.float32, device=dev)
        spade.spade_verify_attention_noalloc(wl["q"], wl["k_cache"], wl["v_cache"], wl["ctx_lens"],
                                             wl["n_draft"], wl["cu_q"], out, lse, max_k=max_k, status=st)
        outs.append((out, lse))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for out, lse in outs:
        # Same kernel, same schedule, same inputs: the results are identical.
        assert torch.equal(out, ref)
        assert torch.equal(lse, ref_lse)
    # The static array starts at zero and every completed call leaves its merge
    # counters at zero again, so the clearing memset at the start of each call
    # only matters after an interrupted call; that path is checked by reading.


def test_noalloc_rejects_sizes_beyond_the_static_scratch(gpu_lib):
    lib = spade.load()
    st = spade.status_tensor("cuda:0")
    p = ctypes.c_void_p(st.data_ptr())
    # 512 sequences x 8 KV heads need far more than the 32 MiB static scratch.
    rc = lib.spade_verify_attention_noalloc(p, p, p, p, p, p, p, None, 512, 32, 8, 128, 4096, 8, 512 * 9, p,
                                            None)
    assert rc == 3  # SPADE_ERR_CAPACITY, refused before any launch
    assert b"static scratch" in lib.spade_last_error()
    # Unsupported shapes get the codes spade_verify_attention gives them.
    rc = lib.spade_verify_attention_noalloc(p, p, p, p, p, p, p, None, 1, 8, 8, 96, 64, 1, 2, p, None)
    assert rc == 2  # SPADE_ERR_SHAPE: head dim 96
    rc = lib.spade_verify_attention_noalloc(p, p, p, p, p, p, p, None, 1, 8, 3, 128, 64, 1, 2, p, None)
    assert rc == 2  # SPADE_ERR_SHAPE: Hq % Hkv != 0
