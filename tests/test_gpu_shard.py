"""cc_score_rows on the GPU: the rows of a refresh scored in the blocks a
multi-GPU plan gives each rank (here one block after another on one GPU;
no kernel waits on another), assembled by the element-wise maximum that
the MAX all-reduce computes, must equal one cc_score_layer / cc_score_full
call bit for bit; the keep-set and the compaction that follow are then
those of the single call."""
import numpy as np
import pytest
import torch

import synth
from tests._util import causal_cache, to_device, to_np
from tests.test_gpu_score import SMALL_GPU

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    import paper_2607_27600_gb300 as p
    p.load_library()
    return p


def _single_and_sharded(pkg, shape, w, c, mode, full, world, align=128):
    from paper_2607_27600_gb300 import cc, shard
    b, cap = c["tokens"].shape
    weights, cache = pkg.Weights(w), pkg.Cache(c)
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode))
    single = torch.full((b, cap), float("nan"), dtype=torch.float32, device="cuda")
    (cc.cc_score_full if full else cc.cc_score_layer)(shape, weights, cache, mode, single, ws)
    merged = torch.full((b, cap), float("-inf"), dtype=torch.float32, device="cuda")
    parts = []
    for r in range(world):
        plan = shard.RowShard(shape, full, c["seq_len"].tolist(), r, world, align, device="cuda")
        mine = torch.full((b, cap), float("nan"), dtype=torch.float32, device="cuda")
        plan.score(shape, weights, cache, mode, mine, ws)
        parts.append((plan, mine.clone()))
        merged = torch.maximum(merged, mine)
    assert cc.cc_get_status() == cc.CC_OK
    return single, merged, parts


def _check(single, merged, parts, seq_lens):
    s, m = single.cpu().numpy(), merged.cpu().numpy()
    assert np.array_equal(s.view(np.uint32), m.view(np.uint32))   # bit for bit
    for plan, mine in parts:
        x = mine.cpu().numpy()
        r = plan.rank
        for b, n in enumerate(seq_lens):
            lo, hi = plan.lo[r, b], plan.hi[r, b]
            assert np.array_equal(x[b, lo:hi].view(np.uint32), s[b, lo:hi].view(np.uint32))
            assert np.all(x[b, :lo] == -np.inf) and np.all(x[b, hi:] == -np.inf)


@pytest.mark.parametrize("world", [2, 3])
def test_llama_layer_8k_rows_in_blocks_equal_the_single_call(pkg, world):
    from paper_2607_27600_gb300 import cc
    wl = synth.WORKLOADS["llama8b-layer-8k"]
    last = wl.shape.n_layers - 1
    w = synth.model_weights(wl.shape, wl.seed, device="cuda", layers=[last], with_embed=False)
    c = synth.synthetic_cache(wl.shape, wl.seq_lens, wl.cap, wl.seed, device="cuda", layers=[last])
    single, merged, parts = _single_and_sharded(pkg, wl.shape, w, c, cc.SCORE_LOGIT, False, world)
    _check(single, merged, parts, wl.seq_lens)


@pytest.mark.parametrize("mode_name", ["logit", "logprob", "precise"])
@pytest.mark.parametrize("full", [False, True])
def test_small_ragged_batch_both_passes_and_modes(pkg, mode_name, full):
    from paper_2607_27600_gb300 import cc
    mode = {"logit": cc.SCORE_LOGIT, "logprob": cc.SCORE_LOGPROB,
            "precise": cc.SCORE_LOGIT | cc.SCORE_PRECISE}[mode_name]
    seq, cap = [300, 129, 1, 64, 0], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 21, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 22)
    w, c = to_device(w_np), to_device(c_np)
    # alignment 16: blocks that start inside the projections' 128-row tiles
    single, merged, parts = _single_and_sharded(pkg, SMALL_GPU, w, c, mode, full, 3, align=16)
    _check(single, merged, parts, seq)


@pytest.mark.parametrize("mode_name", ["logit", "logprob", "precise"])
@pytest.mark.parametrize("full", [False, True])
def test_range_only_blocks_fill_one_buffer(pkg, mode_name, full):
    """CC_SCORE_RANGE_ONLY: blocks of rows scored from the sequence ends
    backwards (the order in which a pipelined upload delivers them) into one
    buffer give the single call's scores bit for bit; entries past the
    sequence ends are never written."""
    from paper_2607_27600_gb300 import cc
    mode = {"logit": cc.SCORE_LOGIT, "logprob": cc.SCORE_LOGPROB,
            "precise": cc.SCORE_LOGIT | cc.SCORE_PRECISE}[mode_name]
    seq, cap = [300, 129, 1, 64, 0], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 23, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 24)
    w, c = to_device(w_np), to_device(c_np)
    weights, cache = pkg.Weights(w), pkg.Cache(c)
    b = len(seq)
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(SMALL_GPU, b, cap, mode))
    single = torch.empty(b, cap, dtype=torch.float32, device="cuda")
    (cc.cc_score_full if full else cc.cc_score_layer)(SMALL_GPU, weights, cache, mode, single, ws)
    filled = torch.full((b, cap), float("nan"), dtype=torch.float32, device="cuda")
    n_blocks = 4
    for k in reversed(range(n_blocks)):   # the last rows first
        lo = torch.tensor([n * k // n_blocks for n in seq], dtype=torch.int32, device="cuda")
        hi = torch.tensor([n * (k + 1) // n_blocks for n in seq], dtype=torch.int32, device="cuda")
        cc.cc_score_rows(SMALL_GPU, weights, cache, mode | cc.SCORE_RANGE_ONLY, full, lo, hi,
                         filled, ws)
    assert cc.cc_get_status() == cc.CC_OK
    s, f = single.cpu().numpy(), filled.cpu().numpy()
    for i, n in enumerate(seq):
        assert np.array_equal(f[i, :n].view(np.uint32), s[i, :n].view(np.uint32))
        assert np.all(np.isnan(f[i, n:]))


def test_sharded_refresh_keep_set_and_compaction_equal_the_single_call(pkg):
    """Two ranks' blocks, the merge, then select and compaction on a replica:
    the same keep-set and the same compacted cache as the unsharded refresh."""
    from paper_2607_27600_gb300 import cc, shard
    seq, cap, budgets = [300, 171, 64], 320, [75, 40, 16]
    w_np = to_np(synth.model_weights(SMALL_GPU, 31, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 32)
    w = pkg.Weights(to_device(w_np))
    b = len(seq)
    results = []
    for world in (1, 2):
        c = to_device(c_np)
        cache = pkg.Cache(c)
        ws = cc.alloc_workspace(cc.cc_score_workspace_size(SMALL_GPU, b, cap, cc.SCORE_LOGIT))
        cws = cc.alloc_workspace(cc.cc_compact_workspace_size(SMALL_GPU, cache))
        budget = torch.tensor(budgets, dtype=torch.int32, device="cuda")
        idx = torch.full((b, cap), -1, dtype=torch.int32, device="cuda")
        cnt = torch.zeros(b, dtype=torch.int32, device="cuda")
        merged = torch.full((b, cap), float("-inf"), dtype=torch.float32, device="cuda")
        for r in range(world):
            plan = shard.RowShard(SMALL_GPU, False, seq, r, world, 16, device="cuda")
            mine = torch.empty(b, cap, dtype=torch.float32, device="cuda")
            plan.score(SMALL_GPU, w, cache, cc.SCORE_LOGIT, mine, ws)
            merged = torch.maximum(merged, mine)   # what the MAX all-reduce computes
        cc.cc_select_keep(merged, c["seq_len"], b, cap, budget, 0, idx, cnt)
        cc.cc_compact_kv(SMALL_GPU, cache, idx, cnt, cws)
        assert cc.cc_get_status() == cc.CC_OK
        results.append((idx.cpu(), cnt.cpu(), [x.cpu() for x in c["k"] + c["v"]],
                        c["tokens"].cpu(), c["pos"].cpu(), c["h_last"].cpu()))
    (i1, n1, kv1, t1, p1, h1), (i2, n2, kv2, t2, p2, h2) = results
    assert torch.equal(n1, n2)
    for s_ in range(b):
        assert torch.equal(i1[s_, :n1[s_]], i2[s_, :n2[s_]])
    assert all(torch.equal(x, y) for x, y in zip(kv1, kv2))
    assert torch.equal(t1, t2) and torch.equal(p1, p2) and torch.equal(h1, h2)


def test_range_past_the_sequence_end_is_reported(pkg):
    """row_hi beyond seq_len (inside the buffer) is reported on the device
    and the attention skips those units (no fault)."""
    from paper_2607_27600_gb300 import cc
    seq, cap = [200], 256
    w_np = to_np(synth.model_weights(SMALL_GPU, 41, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 42)
    w, c = pkg.Weights(to_device(w_np)), to_device(c_np)
    cache = pkg.Cache(c)
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(SMALL_GPU, 1, cap, cc.SCORE_LOGIT))
    scores = torch.empty(1, cap, dtype=torch.float32, device="cuda")
    lo = torch.tensor([0], dtype=torch.int32, device="cuda")
    hi = torch.tensor([230], dtype=torch.int32, device="cuda")
    cc.cc_score_rows(SMALL_GPU, w, cache, cc.SCORE_LOGIT, False, lo, hi, scores, ws)
    assert cc.cc_get_status() == cc.CC_ERR_DEVICE_ARG
    assert cc.cc_get_status() == cc.CC_OK


@pytest.mark.parametrize("layout", ["e4m3", "paged", "head_major"])
def test_rows_in_blocks_over_cache_layout_variants(pkg, layout):
    """The same bit-for-bit equality over an e4m3 cache, a paged cache (a
    shuffled pool of 256-slot pages with a block table) and a head-major
    cache."""
    import bench
    from paper_2607_27600_gb300 import cc
    shape = synth.WORKLOADS["qwen7b-table1-fast-4096"].shape
    seq, cap = [4096, 2500], 4096
    last = shape.n_layers - 1
    w = synth.model_weights(shape, 51, device="cuda", layers=[last], with_embed=False)
    c = synth.synthetic_cache(shape, seq, cap, 52, device="cuda")
    if layout == "e4m3":
        bench.to_e4m3_cache(c)
    elif layout == "paged":
        bench.to_paged_cache(c, 256, 53)
    else:
        for key in ("k", "v"):
            c[key] = [x.permute(0, 2, 1, 3).contiguous() for x in c[key]]
        c["kv_layout"] = 1
    single, merged, parts = _single_and_sharded(pkg, shape, w, c, cc.SCORE_LOGIT, False, 3)
    _check(single, merged, parts, seq)


@pytest.mark.parametrize("layout", ["e4m3", "paged", "head_major"])
def test_range_only_blocks_over_cache_layout_variants(pkg, layout):
    """CC_SCORE_RANGE_ONLY blocks (the sequence ends first) over an e4m3, a
    paged and a head-major cache: one buffer, the single call's scores bit
    for bit (an e4m3 layer is copied to bf16 for each block's attention)."""
    import bench
    from paper_2607_27600_gb300 import cc
    shape = synth.WORKLOADS["qwen7b-table1-fast-4096"].shape
    seq, cap = [4096, 2500], 4096
    last = shape.n_layers - 1
    w = synth.model_weights(shape, 61, device="cuda", layers=[last], with_embed=False)
    c = synth.synthetic_cache(shape, seq, cap, 62, device="cuda")
    if layout == "e4m3":
        bench.to_e4m3_cache(c)
    elif layout == "paged":
        bench.to_paged_cache(c, 256, 63)
    else:
        for key in ("k", "v"):
            c[key] = [x.permute(0, 2, 1, 3).contiguous() for x in c[key]]
        c["kv_layout"] = 1
    weights, cache = pkg.Weights(w), pkg.Cache(c)
    b = len(seq)
    mode = cc.SCORE_LOGIT
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode))
    single = torch.empty(b, cap, dtype=torch.float32, device="cuda")
    cc.cc_score_layer(shape, weights, cache, mode, single, ws)
    filled = torch.full((b, cap), float("nan"), dtype=torch.float32, device="cuda")
    bounds = bench.block_bounds(seq, 3)
    for k in reversed(range(3)):
        lo = torch.tensor(bounds[k], dtype=torch.int32, device="cuda")
        hi = torch.tensor(bounds[k + 1], dtype=torch.int32, device="cuda")
        cc.cc_score_rows(shape, weights, cache, mode | cc.SCORE_RANGE_ONLY, False, lo, hi, filled, ws)
    assert cc.cc_get_status() == cc.CC_OK
    s, f = single.cpu().numpy(), filled.cpu().numpy()
    for i, n in enumerate(seq):
        assert np.array_equal(f[i, :n].view(np.uint32), s[i, :n].view(np.uint32))
        assert np.all(np.isnan(f[i, n:]))
