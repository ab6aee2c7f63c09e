"""cc_compact_kv_static: compaction for callers that cannot allocate device
memory (for example a serving loop whose whole device pool is already the KV
cache).  It must give exactly what cc_compact_kv gives with a workspace, on
two calls in a row, because its scratch is one fixed array shared by every
call on the device and keeping the previous call's contents.

This file is collected last so that a run stopping at the first failure has
already run every other test."""
import numpy as np
import pytest
import torch

import synth
from synth.configs import ModelShape

pytestmark = pytest.mark.gpu

SHAPE = ModelShape(n_layers=3, d_model=256, n_q_heads=8, n_kv_heads=2, head_dim=64,
                   d_ff=384, vocab=1000, rope_theta=1e4, rms_eps=1e-5)


def _keep(seq, cap, seed):
    r = np.random.default_rng(seed)
    idx = np.full((len(seq), cap), -1, np.int32)
    cnt = np.zeros(len(seq), np.int32)
    for b, n in enumerate(seq):
        k = np.sort(r.choice(n, size=max(1, n // 3), replace=False))
        idx[b, :len(k)] = k
        cnt[b] = len(k)
    return torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda()


def _snapshot(c):
    return [t.clone() for t in c["k"] + c["v"]] + [c["h_last"].clone(), c["tokens"].clone(),
                                                   c["pos"].clone(), c["seq_len"].clone()]


def test_static_scratch_compaction_matches_workspace_version_twice():
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    pkg.load_library()
    seq, cap = [3000, 1777], 3072
    ref = synth.synthetic_cache(SHAPE, seq, cap, seed=41, device="cuda")
    stat = {k: ([t.clone() for t in v] if isinstance(v, list) else v.clone())
            for k, v in ref.items()}
    ref_c, stat_c = pkg.Cache(ref), pkg.Cache(stat)
    ws = cc.alloc_workspace(cc.cc_compact_workspace_size(SHAPE, ref_c))
    for call, seed in enumerate((1, 2)):
        idx, cnt = _keep([int(x) for x in ref["seq_len"].tolist()], cap, seed)
        cc.cc_compact_kv(SHAPE, ref_c, idx, cnt, ws)
        cc.cc_compact_kv_static(SHAPE, stat_c, idx, cnt)
        assert cc.cc_get_status() == cc.CC_OK
        for a, b in zip(_snapshot(ref), _snapshot(stat)):
            assert torch.equal(a, b), f"call {call}"
        assert stat["seq_len"].tolist() == cnt.tolist()


def test_static_scratch_rejects_caches_beyond_its_size():
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    big = ModelShape(n_layers=64, d_model=256, n_q_heads=8, n_kv_heads=2, head_dim=64, d_ff=384,
                     vocab=1000, rope_theta=1e4, rms_eps=1e-5)
    # 128 K/V arrays of 256-byte rows move in 4 KB units of 16 slots: 2^19 / 16 = 32768
    # units per array, so about 4.2 M four-byte unit flags (16 MiB) > the 1 MiB array
    cap = 1 << 19
    tiny = torch.zeros(16, dtype=torch.bfloat16, device="cuda")   # pointers are not dereferenced
    c = {"k": [tiny] * 64, "v": [tiny] * 64, "h_last": None,
         "tokens": torch.zeros(1, 1, dtype=torch.int32, device="cuda"),
         "pos": torch.zeros(1, 1, dtype=torch.int32, device="cuda"),
         "seq_len": torch.zeros(1, dtype=torch.int32, device="cuda")}
    cache = pkg.Cache(c)
    cache.c.cap = cap      # host-side plan only: rejected before anything is enqueued
    idx = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(cc.CCError) as e:
        cc.cc_compact_kv_static(big, cache, idx, idx)
    assert e.value.code == cc.CC_ERR_WORKSPACE
