"""Paged K/V cache (cc_kv_cache.block_table): K and V live in page pools and
a block table maps each sequence's logical slots to pages.  Paging only
moves where rows live, so every result must equal the slot-major cache's bit
for bit; the oracle checks the same results as for the slot-major cache.
Unused pool pages hold NaN bit patterns, so a read of a wrong page shows."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth.configs import ModelShape
from tests._util import causal_cache, rel_err, to_device, to_np
from tests.test_gpu_append import SMALL_GPU, _decode_check

pytestmark = pytest.mark.gpu

TOL = 2e-2


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


def paginate(dev, page, extra=3, seed=0):
    """A paged copy of device cache dict `dev`: each K/V [B, cap, Hkv, dh]
    becomes a pool of B*cap/page + extra pages in a random order; the rest
    of the dict is copied."""
    b, cap = dev["tokens"].shape
    per = cap // page
    n_pages = b * per + extra
    perm = np.random.default_rng(seed).permutation(n_pages)[:b * per].reshape(b, per)
    table = torch.from_numpy(perm.astype(np.int32)).cuda()
    out = {k: (v.clone() if isinstance(v, torch.Tensor) else v) for k, v in dev.items()
           if k not in ("k", "v")}
    idx = torch.from_numpy(perm.reshape(-1)).cuda().long()
    for key in ("k", "v"):
        pools = []
        for x in dev[key]:
            pool = torch.empty((n_pages, page) + tuple(x.shape[2:]), dtype=x.dtype, device="cuda")
            pool.view(torch.uint8).fill_(0xFF)        # NaN bits (bf16 and e4m3)
            pool[idx] = x.reshape((b * per, page) + tuple(x.shape[2:]))
            pools.append(pool)
        out[key] = pools
    out["block_table"] = table
    out["page_size"] = page
    return out


def gather(paged, key, l):
    """Logical [B, cap, Hkv, dh] view of a paged K or V layer."""
    t = paged["block_table"].long()
    pool = paged[key][l]
    b, per = t.shape
    return pool[t.reshape(-1)].reshape((b, per * paged["page_size"]) + tuple(pool.shape[2:]))


def _bits(x):
    return x.contiguous().view(torch.uint8).cpu().numpy()


def _run_score(cc, shape, w_np, dev, full, mode=None):
    import paper_2607_27600_gb300 as pkg
    mode = cc.SCORE_LOGIT if mode is None else mode
    weights, cache = pkg.Weights(to_device(w_np)), pkg.Cache(dev)
    b, cap = dev["tokens"].shape
    scores = torch.full((b, cap), float("nan"), device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode))
    (cc.cc_score_full if full else cc.cc_score_layer)(shape, weights, cache, mode, scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
    return scores, cache


@pytest.mark.parametrize("full", [False, True])
def test_paged_scores_match_slot_major_and_oracle(cc, full):
    """Ragged batch, pages of 128 slots (3 per sequence) in a shuffled pool."""
    seq, cap = [300, 129, 1, 64], 384
    w_np = to_np(synth.model_weights(SMALL_GPU, 81, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 81)
    dev = to_device(c_np)
    flat, _ = _run_score(cc, SMALL_GPU, w_np, dev, full)
    paged, _ = _run_score(cc, SMALL_GPU, w_np, paginate(dev, 128, seed=81), full)
    np.testing.assert_array_equal(paged.cpu().numpy(), flat.cpu().numpy())
    want = (oracle.score_full if full else oracle.score_layer)(SMALL_GPU, w_np, c_np)
    assert rel_err(paged.cpu().numpy(), want) < TOL


def test_paged_importance_scores_match(cc):
    """The key-attention comparison scorer reads K tiles through the table."""
    import paper_2607_27600_gb300 as pkg
    seq, cap = [300, 129, 64], 384
    w_np = to_np(synth.model_weights(SMALL_GPU, 82, with_kv_proj=True))
    dev = to_device(causal_cache(SMALL_GPU, w_np, seq, cap, 82))
    out = []
    for d in (dev, paginate(dev, 128, seed=82)):
        scores = torch.zeros((len(seq), cap), device="cuda")
        ws = cc.alloc_workspace(cc.cc_keyattn_workspace_size(SMALL_GPU, len(seq), cap))
        cc.cc_score_importance(SMALL_GPU, pkg.Cache(d), scores, ws)
        assert cc.cc_get_status() == cc.CC_OK
        out.append(scores.cpu().numpy())
    np.testing.assert_array_equal(out[1], out[0])


def test_paged_refresh_cycle_compacts_through_the_table(cc):
    """Score, select and compact a paged cache: the gathered K/V equal the
    slot-major cache's after the same refresh, byte for byte; the table is
    unchanged; the oracle's compaction of the logical cache agrees."""
    seq, cap, budgets = [300, 129, 64], 384, [100, 129, 10]
    w_np = to_np(synth.model_weights(SMALL_GPU, 83, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 83)
    dev = to_device(c_np)
    pdev = paginate(dev, 128, seed=83)
    table_before = pdev["block_table"].clone()
    b = len(seq)
    results = []
    for d in (dev, pdev):
        scores, cache = _run_score(cc, SMALL_GPU, w_np, d, False)
        budget = torch.tensor(budgets, dtype=torch.int32, device="cuda")
        keep_idx = torch.full((b, cap), -1, dtype=torch.int32, device="cuda")
        keep_count = torch.zeros(b, dtype=torch.int32, device="cuda")
        cc.cc_select_keep(scores, d["seq_len"], b, cap, budget, 0, keep_idx, keep_count)
        ws = cc.alloc_workspace(cc.cc_compact_workspace_size(SMALL_GPU, cache))
        cc.cc_compact_kv(SMALL_GPU, cache, keep_idx, keep_count, ws)
        assert cc.cc_get_status() == cc.CC_OK
        results.append((keep_idx.cpu().numpy(), keep_count.cpu().numpy()))
    (gi, gc), (pi, pc) = results
    np.testing.assert_array_equal(pi, gi)
    np.testing.assert_array_equal(pc, gc)
    assert torch.equal(pdev["block_table"], table_before)
    for key in ("k", "v"):
        for l in range(SMALL_GPU.n_layers):
            got = gather(pdev, key, l)
            for i in range(b):
                n = int(gc[i])
                np.testing.assert_array_equal(_bits(got[i, :n]), _bits(dev[key][l][i, :n]))
                np.testing.assert_array_equal(
                    got[i, :n].float().cpu().numpy(),
                    oracle.compact(np.asarray(c_np[key][l], np.float32), gi, gc)[i, :n])
    assert pdev["seq_len"].cpu().tolist() == gc.tolist()


def _append(cc, shape, w_np, d, chunks):
    import paper_2607_27600_gb300 as pkg
    b = len(chunks)
    mx = max(len(t) for t in chunks)
    tok = np.zeros((b, mx), np.int32)
    for i, t in enumerate(chunks):
        tok[i, :len(t)] = t
    cnt = torch.tensor([len(t) for t in chunks], dtype=torch.int32, device="cuda")
    weights, cache = pkg.Weights(to_device(w_np)), pkg.Cache(d)
    ws = cc.alloc_workspace(cc.cc_append_workspace_size(shape, b, d["tokens"].shape[1]))
    cc.cc_append_chunk(shape, weights, cache, torch.from_numpy(tok).cuda(), None, cnt, mx, ws)
    assert cc.cc_get_status() == cc.CC_OK


def _same_kv(shape, flat, paged, seq_after):
    for key in ("k", "v"):
        for l in range(shape.n_layers):
            got = gather(paged, key, l)
            for i, n in enumerate(seq_after):
                np.testing.assert_array_equal(_bits(got[i, :n]), _bits(flat[key][l][i, :n]))


@pytest.mark.parametrize("case", ["small", "llama-fused", "llama-fused-e4m3"])
def test_paged_append_matches_slot_major(cc, case):
    """Chunks appended through the separate K/V projections (small shape) or
    the fused q/k/v GEMM (Llama-3-8B layer shapes, pages of 256), bf16 or
    e4m3: the pages hold exactly the slot-major cache's rows."""
    from tests.test_gpu_fp8 import fp8_views
    if case == "small":
        shape, seq, cap, page, seed = SMALL_GPU, [200, 90, 30], 384, 128, 84
        w_np = to_np(synth.model_weights(shape, seed, with_kv_proj=True))
        c_np = causal_cache(shape, w_np, seq, cap, seed)
        r = np.random.default_rng(seed)
        chunks = [r.integers(0, shape.vocab, size=m) for m in (40, 7, 0)]
    else:
        shape = ModelShape(**{**synth.configs.LLAMA3_8B.__dict__, "n_layers": 2})
        seq, cap, page, seed = [1200], 1536, 256, 85
        w = synth.model_weights(shape, seed, device="cuda", with_kv_proj=True)
        c = synth.synthetic_cache(shape, seq, cap, seed, device="cuda")
        w_np, c_np = to_np(w), to_np(c)
        chunks = [synth.tokens((300,), shape.vocab, seed, "chunk").numpy()]
    if case.endswith("e4m3"):
        _, dev = fp8_views(c_np)
    else:
        dev = to_device(c_np)
    pdev = paginate(dev, page, seed=seed)
    _append(cc, shape, w_np, dev, chunks)
    _append(cc, shape, w_np, pdev, chunks)
    after = [n + len(t) for n, t in zip(seq, chunks)]
    assert pdev["seq_len"].cpu().tolist() == after
    _same_kv(shape, dev, pdev, after)
    if case == "small":   # the slot-major result against the oracle (as in the append tests)
        on = {k: ([np.asarray(x, np.float64).copy() for x in v] if isinstance(v, list) else
                  np.asarray(v).copy()) for k, v in c_np.items()}
        for i, t in enumerate(chunks):
            if len(t):
                oracle.append_chunk(shape, w_np, on, i, t)
        for i, (n0, t) in enumerate(zip(seq, chunks)):
            if len(t):
                sl = slice(n0, n0 + len(t))
                got = gather(pdev, "k", 1)[i, sl].float().cpu().numpy()
                assert rel_err(got, on["k"][1][i, sl]) < TOL


def test_paged_decode_steps(cc):
    """Greedy decode over a paged cache (GEMV writers, key-split decode
    attention over pages of 128): next tokens and logits identical to the
    slot-major cache's, and the oracle's choice."""
    import paper_2607_27600_gb300 as pkg
    seq, cap, seed = [1500, 300, 1999], 2048, 86
    w_np = to_np(synth.model_weights(SMALL_GPU, seed, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, seed)
    dev = to_device(c_np)
    pdev = paginate(dev, 128, seed=seed)
    on = {k: ([np.asarray(x, np.float64).copy() for x in v] if isinstance(v, list) else
              np.asarray(v).copy()) for k, v in c_np.items()}
    b = len(seq)
    tok = np.random.default_rng(seed).integers(0, SMALL_GPU.vocab, size=b)
    outs = []
    for d in (dev, pdev):
        weights, cache = pkg.Weights(to_device(w_np)), pkg.Cache(d)
        ws = cc.alloc_workspace(cc.cc_decode_workspace_size(SMALL_GPU, b, cap))
        nxt = torch.empty(b, dtype=torch.int32, device="cuda")
        best = torch.empty(b, dtype=torch.float32, device="cuda")
        cc.cc_decode_step(SMALL_GPU, weights, cache, torch.from_numpy(tok.astype(np.int32)).cuda(),
                          nxt, best, ws)
        assert cc.cc_get_status() == cc.CC_OK
        outs.append((nxt.cpu().numpy(), best.cpu().numpy()))
    np.testing.assert_array_equal(outs[1][0], outs[0][0])
    np.testing.assert_array_equal(outs[1][1], outs[0][1])
    _same_kv(SMALL_GPU, dev, pdev, [n + 1 for n in seq])
    _, _, o_logits = oracle.decode_step(SMALL_GPU, w_np, on, tok)
    for i in range(b):
        _decode_check(int(outs[1][0][i]), float(outs[1][1][i]), o_logits[i])


def test_paged_bad_table_entry_is_reported(cc):
    """A block-table entry outside the pool: the kernels skip its rows (a
    tile there reads zeros) and report CC_ERR_DEVICE_ARG; the context stays
    usable; a page size that is not a whole number of key tiles is refused
    before anything runs."""
    import paper_2607_27600_gb300 as pkg
    seq, cap = [300, 64], 384
    w_np = to_np(synth.model_weights(SMALL_GPU, 87, with_kv_proj=True))
    dev = to_device(causal_cache(SMALL_GPU, w_np, seq, cap, 87))
    pdev = paginate(dev, 128, seed=87)
    pdev["block_table"][0, 1] = 10_000
    weights, cache = pkg.Weights(to_device(w_np)), pkg.Cache(pdev)
    scores = torch.zeros((2, cap), device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(SMALL_GPU, 2, cap, cc.SCORE_LOGIT))
    cc.cc_score_layer(SMALL_GPU, weights, cache, cc.SCORE_LOGIT, scores, ws)
    assert cc.cc_get_status() == cc.CC_ERR_DEVICE_ARG
    assert cc.cc_get_status() == cc.CC_OK
    bad = dict(paginate(dev, 128, seed=87))
    bad["page_size"] = 64
    with pytest.raises(cc.CCError) as e:
        cc.cc_score_layer(SMALL_GPU, weights, pkg.Cache(bad), cc.SCORE_LOGIT, scores, ws)
    assert e.value.code == cc.CC_ERR_INVALID_ARG
