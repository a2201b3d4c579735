"""The seeded input generators (CPU): a seed names the same tensors on every call, and the
paged layout holds exactly the dense caches' data."""
import numpy as np
import torch

import oracle.spade_oracle as O
from paper_2608_13076_gb300 import workloads as W

SPEC = W.WorkloadSpec("gen_check", B=3, Hq=4, Hkv=2, D=64, H=64, V=300, ctx=(5, 90), k=(1, 4),
                      mode="mixed", seed=77)


def test_same_seed_same_tensors():
    a = W.make_workload(SPEC)
    b = W.make_workload(SPEC)
    for k, v in a.items():
        if isinstance(v, torch.Tensor):
            assert torch.equal(v, b[k]), k


def test_paged_layout_round_trip():
    wl = W.make_workload(SPEC, cache_pad=11)
    for page in (16, 64):
        pg = W.to_paged(wl, page, seed=3)
        assert pg["k_pool"].shape[0] == pg["num_pages"]
        table = pg["block_table"].numpy()
        assert len(set(table.reshape(-1).tolist())) == table.size  # every page used once
        for pool, dense in ((pg["k_pool"], wl["k_cache"]), (pg["v_pool"], wl["v_cache"])):
            got = O.paged_gather(pool.float().numpy(), table, wl["cap"], page)
            np.testing.assert_array_equal(got, dense.float().numpy())
        spare = sorted(set(range(pg["num_pages"])) - set(table.reshape(-1).tolist()))
        assert torch.isnan(pg["k_pool"][spare].float()).all()
