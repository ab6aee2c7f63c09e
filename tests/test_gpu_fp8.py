"""GPU parity of the e4m3 K/V cache variant (cc_kv_cache.kv_format =
CC_KV_E4M3) against the oracle: the oracle sees the cache as the codes'
values (oracle.e4m3_decode(code) * scale) and quantises the rows an append
writes (oracle.kv_quantize), so both sides attend over the same cached
values."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth.configs import ModelShape
from tests._util import causal_cache, keep_set_ok, rel_err, to_device, to_np
from tests.test_gpu_append import SMALL_GPU, _decode_check

pytestmark = pytest.mark.gpu

TOL = 2e-2


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


def fp8_views(c_np, headroom=2.0):
    """(oracle view, device dict) of a float cache stored as e4m3: per layer
    scale = max |x| * headroom / 448 (room for the rows appends add)."""
    L = len(c_np["k"])
    scales, ko, vo, kd, vd = [], [], [], [], []
    for l in range(L):
        pair = []
        for src, o_list, d_list in ((c_np["k"][l], ko, kd), (c_np["v"][l], vo, vd)):
            x = np.asarray(src, np.float64)
            s = max(float(np.abs(x).max()), 1e-3) * headroom / 448.0
            codes = oracle.e4m3_encode(x / s)
            o_list.append(oracle.e4m3_decode(codes) * s)
            d_list.append(torch.from_numpy(codes).cuda())
            pair.append(s)
        scales.append(tuple(pair))
    on = {k: v for k, v in c_np.items() if k not in ("k", "v")}
    on.update(k=ko, v=vo, kv_scale=scales)
    dev = to_device({k: v for k, v in c_np.items() if k not in ("k", "v")})
    dev.update(k=kd, v=vd, kv_scale=scales)
    return on, dev


def _ordinal(codes):
    c = np.asarray(codes).astype(np.int64)
    return np.where(c & 0x80, -(c & 0x7F), c & 0x7F)


def _codes_close(got, want_values, scale, min_exact=0.75):
    """Device codes of appended rows against the oracle's (quantised) values.
    Both sides round their own projection to e4m3: the device projects
    bf16-rounded activations in fp32 (about 2^-8 relative off the oracle's
    fp64 value), one e4m3 step is 1/8 of a value, so a few to ~20 % of the
    values straddle a rounding boundary and land one code apart, and values
    far below the row's largest carry the projection's absolute error (TOL
    of the largest).  Checked: every element within one code step plus
    TOL * max; among the elements above that floor, most codes identical
    (rounding toward zero instead of to nearest would change about half) and
    the one-step flips unbiased (a scale or rounding-mode error is not)."""
    got = np.asarray(got)
    want = np.asarray(want_values, np.float64)
    amax = float(np.abs(want).max())
    err = np.abs(oracle.e4m3_decode(got) * scale - want)
    assert (err <= 0.13 * np.abs(want) + TOL * amax).all(), float((err / (amax + 1e-30)).max())
    big = np.abs(want) > TOL * amax
    ref = oracle.e4m3_encode(want / scale)
    assert (got == ref)[big].mean() >= min_exact, (got == ref)[big].mean()
    if big.sum() >= 1000:
        drift = (np.abs(_ordinal(got)) - np.abs(_ordinal(ref)))[big].mean()
        assert abs(drift) < 0.03, drift


def _score(cc, shape, w_np, dev, mode, full):
    import paper_2607_27600_gb300 as pkg
    weights, cache = pkg.Weights(to_device(w_np)), pkg.Cache(dev)
    b, cap = dev["tokens"].shape
    scores = torch.full((b, cap), float("nan"), device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode))
    (cc.cc_score_full if full else cc.cc_score_layer)(shape, weights, cache, mode, scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
    return scores.cpu().numpy(), cache


@pytest.mark.parametrize("full", [False, True])
def test_fp8_scores_small_ragged(cc, full):
    seq, cap = [300, 129, 1, 64], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 71, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 71)
    on, dev = fp8_views(c_np)
    want = (oracle.score_full if full else oracle.score_layer)(SMALL_GPU, w_np, on)
    got, _ = _score(cc, SMALL_GPU, w_np, dev, cc.SCORE_LOGIT, full)
    assert rel_err(got, want) < TOL, rel_err(got, want)
    # the quantisation is visible: the bf16 cache's scores differ
    bf = oracle.score_layer(SMALL_GPU, w_np, c_np) if not full else None
    if bf is not None:
        fin = np.isfinite(bf) & np.isfinite(want)
        assert np.abs(bf[fin] - want[fin]).max() > 0


@pytest.mark.parametrize("full", [False, True])
def test_fp8_precise_mode_small_ragged(cc, full):
    """CC_SCORE_PRECISE over an e4m3 cache: each layer's codes reach the
    attention as an exact bf16 copy, so the queries and P are split there as
    over a bf16 cache, and the scores stay within 2e-3 of the oracle's on the
    dequantised cache (an order of magnitude inside the default mode's bar)."""
    seq, cap = [300, 129, 1, 64], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 73, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 73)
    on, dev = fp8_views(c_np)
    want = (oracle.score_full if full else oracle.score_layer)(SMALL_GPU, w_np, on)
    got, _ = _score(cc, SMALL_GPU, w_np, dev, cc.SCORE_LOGIT | cc.SCORE_PRECISE, full)
    err = rel_err(got, want)
    assert err < TOL and err < 2e-3, err


@pytest.mark.parametrize("name", ["llama", "qwen"])
def test_fp8_fast_scores_model_shapes(cc, name):
    """Last-layer refresh at Llama-3-8B (G = 4) and Qwen2.5-7B (G = 7) layer
    shapes, head_dim 128, 1500 cached slots: 160 sampled rows."""
    base = synth.configs.LLAMA3_8B if name == "llama" else synth.configs.QWEN25_7B
    shape = ModelShape(**{**base.__dict__, "n_layers": 1})
    n, cap, seed = 1500, 1536, 72
    w = synth.model_weights(shape, seed, device="cuda", with_kv_proj=True)
    c = synth.synthetic_cache(shape, [n], cap, seed, device="cuda")
    w_np, c_np = to_np(w), to_np(c)
    on, dev = fp8_views(c_np)
    got, _ = _score(cc, shape, w_np, dev, cc.SCORE_LOGIT, False)
    rows = np.sort(np.random.default_rng(seed).choice(n - 1, 160, replace=False))
    want = oracle.score_layer(shape, w_np, on, rows=[rows])
    assert rel_err(got[0, rows], want[0, rows]) < TOL, rel_err(got[0, rows], want[0, rows])
    assert np.isposinf(got[0, n - 1]) and np.isneginf(got[0, n:]).all()


def test_fp8_select_and_compaction_byte_exact(cc):
    seq, cap, budgets = [300, 129, 64], 320, [100, 129, 10]
    w_np = to_np(synth.model_weights(SMALL_GPU, 73, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 73)
    on, dev = fp8_views(c_np)
    codes_before = [x.cpu().numpy().copy() for x in dev["k"] + dev["v"]]
    got, cache = _score(cc, SMALL_GPU, w_np, dev, cc.SCORE_LOGIT, False)
    b = len(seq)
    budget = torch.tensor(budgets, dtype=torch.int32, device="cuda")
    keep_idx = torch.full((b, cap), -1, dtype=torch.int32, device="cuda")
    keep_count = torch.zeros(b, dtype=torch.int32, device="cuda")
    cc.cc_select_keep(torch.from_numpy(got).cuda(), dev["seq_len"], b, cap, budget, 0, keep_idx,
                      keep_count)
    gi, gc = keep_idx.cpu().numpy(), keep_count.cpu().numpy()
    want = oracle.score_layer(SMALL_GPU, w_np, on)
    wi, wc = oracle.select_keep(want.astype(np.float32), seq, budgets)
    ok, det = keep_set_ok(gi, gc, wi, wc, want, seq, budgets)
    assert ok, det
    ws = cc.alloc_workspace(cc.cc_compact_workspace_size(SMALL_GPU, cache))
    cc.cc_compact_kv(SMALL_GPU, cache, keep_idx, keep_count, ws)
    assert cc.cc_get_status() == cc.CC_OK
    after = [x.cpu().numpy() for x in dev["k"] + dev["v"]]
    for a, bfr in zip(after, codes_before):
        np.testing.assert_array_equal(a, oracle.compact(bfr, gi, gc))
    assert dev["seq_len"].cpu().tolist() == gc.tolist()


def _append_case(cc, shape, w_np, on, dev, chunks):
    import paper_2607_27600_gb300 as pkg
    b = len(chunks)
    mx = max(len(t) for t in chunks)
    tok = np.zeros((b, mx), np.int32)
    for i, t in enumerate(chunks):
        tok[i, :len(t)] = t
    cnt = np.array([len(t) for t in chunks], np.int32)
    weights, cache = pkg.Weights(to_device(w_np)), pkg.Cache(dev)
    ws = cc.alloc_workspace(cc.cc_append_workspace_size(shape, b, dev["tokens"].shape[1]))
    n0 = dev["seq_len"].cpu().numpy().copy()
    cc.cc_append_chunk(shape, weights, cache, torch.from_numpy(tok).cuda(), None,
                       torch.from_numpy(cnt).cuda(), mx, ws)
    assert cc.cc_get_status() == cc.CC_OK
    for i, t in enumerate(chunks):
        if len(t):
            oracle.append_chunk(shape, w_np, on, i, t)
    for i, t in enumerate(chunks):
        sl = slice(int(n0[i]), int(n0[i]) + len(t))
        assert int(dev["seq_len"][i]) == n0[i] + len(t)
        if not len(t):
            continue
        for l in range(shape.n_layers):
            sk, sv = on["kv_scale"][l]
            _codes_close(dev["k"][l][i, sl].cpu().numpy(), on["k"][l][i, sl], sk)
            _codes_close(dev["v"][l][i, sl].cpu().numpy(), on["v"][l][i, sl], sv)


def test_fp8_append_small_separate_projections(cc):
    """SMALL shape (kv_dim 128: separate K and V projection GEMMs writing
    codes); ragged chunks of 40, 7 and 0 tokens after 200, 90 and 30 slots."""
    seq, cap = [200, 90, 30], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 74, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 74)
    on, dev = fp8_views(c_np)
    r = np.random.default_rng(74)
    chunks = [r.integers(0, SMALL_GPU.vocab, size=m) for m in (40, 7, 0)]
    _append_case(cc, SMALL_GPU, w_np, on, dev, chunks)


def test_fp8_append_llama_fused_projection(cc):
    """Llama-3-8B layer shapes, two layers (the fused q/k/v GEMM writes the K
    and V codes); a 300-token chunk after 1200 slots."""
    shape = ModelShape(**{**synth.configs.LLAMA3_8B.__dict__, "n_layers": 2})
    n0, cap, seed = 1200, 1536, 75
    w = synth.model_weights(shape, seed, device="cuda", with_kv_proj=True)
    c = synth.synthetic_cache(shape, [n0], cap, seed, device="cuda")
    w_np, c_np = to_np(w), to_np(c)
    on, dev = fp8_views(c_np)
    chunk = synth.tokens((300,), shape.vocab, seed, "chunk").numpy()
    _append_case(cc, shape, w_np, on, dev, [chunk])


@pytest.mark.parametrize("case", ["small", "small-long"])
def test_fp8_decode_steps(cc, case):
    """Greedy decode over an e4m3 cache (weight-streaming GEMVs write the
    codes; the CUDA-core decode attention reads them, key splits in the long
    case), teacher-forced with the oracle's tokens."""
    import paper_2607_27600_gb300 as pkg
    seq, cap = ([50, 20, 33], 64) if case == "small" else ([1500, 300, 1999], 2048)
    w_np = to_np(synth.model_weights(SMALL_GPU, 76, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 76)
    on, dev = fp8_views(c_np)
    b = len(seq)
    weights, cache = pkg.Weights(to_device(w_np)), pkg.Cache(dev)
    ws = cc.alloc_workspace(cc.cc_decode_workspace_size(SMALL_GPU, b, cap))
    tok = np.random.default_rng(76).integers(0, SMALL_GPU.vocab, size=b)
    nxt = torch.empty(b, dtype=torch.int32, device="cuda")
    best = torch.empty(b, dtype=torch.float32, device="cuda")
    for step in range(3):
        cc.cc_decode_step(SMALL_GPU, weights, cache, torch.from_numpy(tok.astype(np.int32)).cuda(),
                          nxt, best, ws)
        assert cc.cc_get_status() == cc.CC_OK
        o_next, _, o_logits = oracle.decode_step(SMALL_GPU, w_np, on, tok)
        g_next, g_best = nxt.cpu().numpy(), best.cpu().numpy()
        for i in range(b):
            _decode_check(int(g_next[i]), float(g_best[i]), o_logits[i])
            n1 = int(on["seq_len"][i])
            for l in range(SMALL_GPU.n_layers):
                sk, sv = on["kv_scale"][l]
                _codes_close(dev["k"][l][i, n1 - 1].cpu().numpy(), on["k"][l][i, n1 - 1], sk)
                _codes_close(dev["v"][l][i, n1 - 1].cpu().numpy(), on["v"][l][i, n1 - 1], sv)
        tok = o_next


def test_fp8_rejections(cc):
    """Bad format fields are refused before anything runs; the comparison
    scorers take bf16 keys only."""
    import paper_2607_27600_gb300 as pkg
    w_np = to_np(synth.model_weights(SMALL_GPU, 77, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, [40], 64, 77)
    on, dev = fp8_views(c_np)
    bad = dict(dev)
    bad["kv_scale"] = [(0.0, 1.0)] + list(dev["kv_scale"][1:])
    weights = pkg.Weights(to_device(w_np))
    scores = torch.zeros((1, 64), device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(SMALL_GPU, 1, 64, cc.SCORE_LOGIT))
    with pytest.raises(cc.CCError) as e:
        cc.cc_score_layer(SMALL_GPU, weights, pkg.Cache(bad), cc.SCORE_LOGIT, scores, ws)
    assert e.value.code == cc.CC_ERR_INVALID_ARG
    kws = cc.alloc_workspace(cc.cc_keyattn_workspace_size(SMALL_GPU, 1, 64))
    with pytest.raises(cc.CCError) as e:
        cc.cc_score_importance(SMALL_GPU, pkg.Cache(dev), scores, kws)
    assert e.value.code == cc.CC_ERR_UNSUPPORTED
