"""Failure detection without a GPU fault: a bounded device wait that runs out
reports CC_ERR_TIMEOUT through the status word, the kernel returns, and the
context stays usable (the same compaction then succeeds)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth.configs import ModelShape

pytestmark = pytest.mark.gpu

SHAPE = ModelShape(n_layers=1, d_model=256, n_q_heads=8, n_kv_heads=2, head_dim=64, d_ff=384,
                   vocab=1000, rope_theta=1e4, rms_eps=1e-5)


def test_withheld_flag_times_out_and_context_survives():
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    pkg.load_library()
    n = cap = 1024
    c = synth.synthetic_cache(SHAPE, [n], cap, seed=5, device="cuda")
    before = c["k"][0].float().cpu().numpy()
    # keep = every slot but the first: unit c reads slots that unit c+1 overwrites,
    # so unit 1 waits for unit 0's flag
    idx = torch.full((1, cap), -1, dtype=torch.int32, device="cuda")
    idx[0, :n - 1] = torch.arange(1, n, dtype=torch.int32, device="cuda")
    cnt = torch.tensor([n - 1], dtype=torch.int32, device="cuda")
    cache = pkg.Cache(c)
    ws = cc.alloc_workspace(cc.cc_compact_workspace_size(SHAPE, cache))
    assert cc.cc_get_status() == cc.CC_OK
    cc.cc_debug_withhold_compact_unit(0)
    cc.cc_compact_kv(SHAPE, cache, idx, cnt, ws)
    assert cc.cc_get_status() == cc.CC_ERR_TIMEOUT
    assert cc.cc_get_status() == cc.CC_OK            # read clears it
    # the context is usable: the same compaction on a fresh cache succeeds and is exact
    c2 = synth.synthetic_cache(SHAPE, [n], cap, seed=5, device="cuda")
    cache2 = pkg.Cache(c2)
    cc.cc_compact_kv(SHAPE, cache2, idx, cnt, ws)
    assert cc.cc_get_status() == cc.CC_OK
    want = oracle.compact(before, idx.cpu().numpy(), cnt.cpu().numpy())
    np.testing.assert_array_equal(c2["k"][0].float().cpu().numpy(), want)
