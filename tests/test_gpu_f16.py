"""The fp16 operand mode (CC_SCORE_F16) of the scoring passes, against the
CPU oracle on the same bf16 inputs: every tensor-core operand of the layers
is one fp16 value (11 significant bits to bf16's 8), so each rounding is 8x
smaller than the default mode's at the same cost.  The weight matrices are
converted once by cc_bf16_to_f16 (exact in the normal fp16 range); the
cached K/V are copied per layer inside the call.  The full-size checks of
this mode sit beside the precise mode's in test_gpu_fullsize.py."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests._util import causal_cache, keep_set_ok, rel_err, to_device, to_np
from tests.test_gpu_fp8 import fp8_views
from tests.test_gpu_score import SMALL_GPU

pytestmark = pytest.mark.gpu

TOL = 2e-2


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


@pytest.fixture(scope="module")
def tiny():
    wl = synth.WORKLOADS["tiny-512"]
    w_np = to_np(synth.model_weights(wl.shape, wl.seed, with_kv_proj=True))
    c_np = causal_cache(wl.shape, w_np, wl.seq_lens, wl.cap, wl.seed)
    return wl, w_np, c_np


def _f16(cc, w_np, c_np):
    import paper_2607_27600_gb300 as pkg
    w, c = to_device(w_np), to_device(c_np)
    return pkg.Weights(cc.f16_weights(w)), pkg.Cache(c)


def _score(cc, shape, weights, cache, mode, full):
    b, cap = cache.d["tokens"].shape
    scores = torch.full((b, cap), float("nan"), dtype=torch.float32, device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode))
    (cc.cc_score_full if full else cc.cc_score_layer)(shape, weights, cache, mode, scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
    return scores


def test_bf16_to_f16_matches_torch_conversion(cc):
    """Element by element equal to torch's own bf16 -> fp16 conversion (round
    to nearest even) over normal, subnormal-range, signed-zero, inf and NaN
    inputs, including 8-element tails; nothing reported in range."""
    g = torch.Generator().manual_seed(5)
    parts = [torch.randn(100_000, generator=g) * 0.02,                 # weights
             torch.randn(4096, generator=g) * 1e-6,                    # below 2^-14
             # 65280: the largest bf16 value inside the fp16 range (bf16(65504) is 65536)
             torch.tensor([0.0, -0.0, 65280.0, -65280.0, 2.0 ** -24, 3 * 2.0 ** -26,
                           float("inf"), -float("inf"), float("nan"), 1e-40]),
             torch.randn(6, generator=g) * 300]
    src = torch.cat(parts).to(torch.bfloat16)
    src = src[: src.numel() // 8 * 8].contiguous()
    fin = src.float()[torch.isfinite(src.float())]
    assert fin.abs().max() <= 65504
    want = src.float().half()
    got = torch.empty(src.shape, dtype=torch.float16, device="cuda")
    cc.cc_bf16_to_f16(src.cuda(), got)
    assert cc.cc_get_status() == cc.CC_OK
    got = got.cpu()
    nan = torch.isnan(want)
    assert torch.equal(torch.isnan(got), nan) and nan.sum() == 1   # NaN payloads may differ
    assert torch.equal(got[~nan].view(torch.int16), want[~nan].view(torch.int16))


def test_bf16_to_f16_range_and_argument_errors(cc):
    src = torch.full((64,), 2.0, dtype=torch.bfloat16, device="cuda")
    src[17] = 70000.0   # bf16 69632: above the fp16 range
    dst = torch.empty(64, dtype=torch.float16, device="cuda")
    cc.cc_bf16_to_f16(src, dst)
    assert cc.cc_get_status() == cc.CC_ERR_RANGE
    assert torch.isinf(dst[17]) and (dst[:17] == 2.0).all() and (dst[18:] == 2.0).all()
    lib = cc.load_library()
    stream = torch.cuda.current_stream().cuda_stream
    assert lib.cc_bf16_to_f16(src.data_ptr(), dst.data_ptr(), 60, stream) == cc.CC_ERR_INVALID_ARG
    assert lib.cc_bf16_to_f16(src.data_ptr(), src.data_ptr() + 16, 16, stream) == cc.CC_ERR_INVALID_ARG
    assert lib.cc_bf16_to_f16(src.data_ptr() + 2, dst.data_ptr(), 8, stream) == cc.CC_ERR_INVALID_ARG
    assert lib.cc_bf16_to_f16(None, None, 0, stream) == cc.CC_OK
    assert cc.cc_get_status() == cc.CC_OK


def test_tiny_f16_mode_all_rows(cc, tiny):
    """Both passes and both score definitions on every row: within the stated
    2e-2 and within 2e-3 (the default mode measures ~5e-3 here)."""
    wl, w_np, c_np = tiny
    weights, cache = _f16(cc, w_np, c_np)
    for mode, m in (("logit", cc.SCORE_LOGIT), ("logprob", cc.SCORE_LOGPROB)):
        want = oracle.score_layer(wl.shape, w_np, c_np, mode=mode)
        for full in (False, True):
            got = _score(cc, wl.shape, weights, cache, m | cc.SCORE_F16, full).cpu().numpy()
            err = rel_err(got, want)
            assert err < TOL and err < 2e-3, (mode, full, err)


@pytest.mark.parametrize("full", [False, True])
def test_small_two_layer_f16_ragged(cc, full):
    """Two layers, head_dim 64, ragged lengths (300, 129, 1, 64 in 320 slots):
    every row within 2e-3."""
    seq, cap = [300, 129, 1, 64], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 23, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 23)
    weights, cache = _f16(cc, w_np, c_np)
    want = (oracle.score_full if full else oracle.score_layer)(SMALL_GPU, w_np, c_np)
    got = _score(cc, SMALL_GPU, weights, cache, cc.SCORE_LOGIT | cc.SCORE_F16, full).cpu().numpy()
    err = rel_err(got, want)
    assert err < TOL and err < 2e-3, err


@pytest.mark.parametrize("full", [False, True])
def test_f16_mode_over_e4m3_cache(cc, full):
    """An e4m3 cache's codes are fp16 values: each layer is copied to fp16
    exactly and the scales stay folded into the softmax and the output, so
    the scores stay within 2e-3 of the oracle's on the dequantised cache."""
    import paper_2607_27600_gb300 as pkg
    seq, cap = [300, 129, 1, 64], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 75, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 75)
    on, dev = fp8_views(c_np)
    want = (oracle.score_full if full else oracle.score_layer)(SMALL_GPU, w_np, on)
    weights = pkg.Weights(cc.f16_weights(to_device(w_np)))
    got = _score(cc, SMALL_GPU, weights, pkg.Cache(dev), cc.SCORE_LOGIT | cc.SCORE_F16,
                 full).cpu().numpy()
    err = rel_err(got, want)
    assert err < TOL and err < 2e-3, err


def test_f16_keep_set_at_the_stated_bar(cc, tiny):
    """The refresh in this mode: select on the GPU's scores equals the
    oracle's select on the same fp32 scores exactly, and the keep-set meets
    the stated bar against the oracle's own scores (identical where the
    boundary gap exceeds the tolerance, else >= 99.5 % overlap)."""
    wl, w_np, c_np = tiny
    weights, cache = _f16(cc, w_np, c_np)
    got = _score(cc, wl.shape, weights, cache, cc.SCORE_LOGIT | cc.SCORE_F16, False)
    b, cap = c_np["tokens"].shape
    budget = torch.tensor(wl.budgets, dtype=torch.int32, device="cuda")
    idx = torch.full((b, cap), -1, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(b, dtype=torch.int32, device="cuda")
    cc.cc_select_keep(got, cache.d["seq_len"], b, cap, budget, 0, idx, cnt)
    assert cc.cc_get_status() == cc.CC_OK
    gi, gc = idx.cpu().numpy(), cnt.cpu().numpy()
    g_np = got.cpu().numpy()
    oi, oc = oracle.select_keep(g_np, wl.seq_lens, wl.budgets)
    assert np.array_equal(gc, oc) and np.array_equal(gi[0, :oc[0]], oi[0, :oc[0]])
    want = oracle.score_layer(wl.shape, w_np, c_np)
    wi, wc = oracle.select_keep(want.astype(np.float32), wl.seq_lens, wl.budgets)
    ok, det = keep_set_ok(gi, gc, wi, wc, want, wl.seq_lens, wl.budgets, min_overlap=0.995)
    assert ok, det


@pytest.mark.parametrize("full", [False, True])
def test_f16_row_blocks_fill_one_buffer(cc, full):
    """cc_score_rows in this mode over two row blocks (RANGE_ONLY) writes
    exactly the scores of the whole-refresh call."""
    seq, cap = [300, 129, 1, 64], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 27, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 27)
    weights, cache = _f16(cc, w_np, c_np)
    mode = cc.SCORE_LOGIT | cc.SCORE_F16
    whole = _score(cc, SMALL_GPU, weights, cache, mode, full)
    b = len(seq)
    cut = [min(n, 128) for n in seq]
    blocks = [([0] * b, cut), (cut, seq)]
    scores = torch.full((b, cap), float("nan"), dtype=torch.float32, device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(SMALL_GPU, b, cap, mode))
    for lo, hi in blocks:
        lo_t = torch.tensor(lo, dtype=torch.int32, device="cuda")
        hi_t = torch.tensor(hi, dtype=torch.int32, device="cuda")
        cc.cc_score_rows(SMALL_GPU, weights, cache, mode | cc.SCORE_RANGE_ONLY, full, lo_t, hi_t,
                         scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
    for s, n in enumerate(seq):
        assert torch.equal(scores[s, :n], whole[s, :n]), s


def test_f16_mode_reports_values_outside_the_fp16_range(cc, tiny):
    """An attention-norm gain of 1e6 puts the normalised inputs far above
    65504: the call reports CC_ERR_RANGE instead of scoring silently with
    infinities; the bf16 default mode takes the same model."""
    import paper_2607_27600_gb300 as pkg
    wl, w_np, c_np = tiny
    w_big = {**w_np, "layers": [dict(lw, attn_norm=np.full_like(lw["attn_norm"], 1e6))
                                for lw in w_np["layers"]]}
    w_dev, c_dev = to_device(w_big), to_device(c_np)
    b, cap = c_np["tokens"].shape
    for mode, weights, want in ((cc.SCORE_LOGIT | cc.SCORE_F16, cc.f16_weights(w_dev),
                                 cc.CC_ERR_RANGE),
                                (cc.SCORE_LOGIT, w_dev, cc.CC_OK)):
        scores = torch.empty(b, cap, dtype=torch.float32, device="cuda")
        ws = cc.alloc_workspace(cc.cc_score_workspace_size(wl.shape, b, cap, mode))
        cc.cc_score_layer(wl.shape, pkg.Weights(weights), pkg.Cache(c_dev), mode, scores, ws)
        assert cc.cc_get_status() == want


def test_f16_mode_rejects_the_precise_flag(cc, tiny):
    wl, w_np, c_np = tiny
    weights, cache = _f16(cc, w_np, c_np)
    b, cap = c_np["tokens"].shape
    mode = cc.SCORE_LOGIT | cc.SCORE_F16 | cc.SCORE_PRECISE
    scores = torch.empty(b, cap, dtype=torch.float32, device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(wl.shape, b, cap, cc.SCORE_PRECISE))
    with pytest.raises(cc.CCError) as e:
        cc.cc_score_layer(wl.shape, weights, cache, mode, scores, ws)
    assert e.value.code == cc.CC_ERR_INVALID_ARG


@pytest.mark.parametrize("layout", ["paged", "head_major", "e4m3_paged"])
def test_f16_cache_layouts_match_slot_major(cc, layout):
    """Qwen2.5-7B last layer (G = 7, head_dim 128), two sequences of 4096 and
    2500 slots: the fp16 mode over a paged, a head-major and a paged e4m3
    cache (each layer's K/V copied to fp16 through the block table or by
    head) writes the slot-major cache's scores bit for bit; the slot-major
    scores match the oracle on sampled rows within 2e-3."""
    import bench
    import paper_2607_27600_gb300 as pkg
    from tests.test_gpu_fullsize import host_view, sample
    shape = synth.WORKLOADS["qwen7b-table1-fast-4096"].shape
    seq, cap = [4096, 2500], 4096
    last = shape.n_layers - 1
    w = synth.model_weights(shape, 81, device="cuda", layers=[last], with_embed=False)
    c = synth.synthetic_cache(shape, seq, cap, 82, device="cuda")
    if layout == "e4m3_paged":
        bench.to_e4m3_cache(c)
    weights = pkg.Weights(cc.f16_weights(w))
    mode = cc.SCORE_LOGIT | cc.SCORE_F16
    ref = _score(cc, shape, weights, pkg.Cache(dict(c)), mode, False)
    if layout == "head_major":
        for key in ("k", "v"):
            c[key] = [None if x is None else x.permute(0, 2, 1, 3).contiguous() for x in c[key]]
        c["kv_layout"] = 1
    else:
        bench.to_paged_cache(c, 256, 83)
    got = _score(cc, shape, weights, pkg.Cache(c), mode, False)
    for i, n in enumerate(seq):
        assert torch.equal(got[i, :n].view(torch.int32), ref[i, :n].view(torch.int32)), i
    if layout == "head_major":   # the oracle once, on the slot-major draw
        c = synth.synthetic_cache(shape, seq, cap, 82, device="cuda")
        wn, cn = host_view(w, c)
        rows = sample(seq, 24, seed=84)
        want = oracle.score_layer(shape, wn, cn, rows=rows)
        r = ref.cpu().numpy()
        err = max(rel_err(r[i, rw], want[i, rw]) for i, rw in enumerate(rows))
        assert err < TOL and err < 2e-3, err


def test_binding_refuses_weights_of_the_other_operand_type(cc, tiny):
    """The C ABI reads the same weight pointers as fp16 or bf16 by the mode;
    the binding checks the tensors' dtype against it before the call."""
    import paper_2607_27600_gb300 as pkg
    wl, w_np, c_np = tiny
    w_dev, c_dev = to_device(w_np), to_device(c_np)
    b, cap = c_np["tokens"].shape
    scores = torch.empty(b, cap, dtype=torch.float32, device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(wl.shape, b, cap, cc.SCORE_LOGIT))
    cases = ((pkg.Weights(w_dev), cc.SCORE_LOGIT | cc.SCORE_F16),
             (pkg.Weights(cc.f16_weights(w_dev)), cc.SCORE_LOGIT))
    for weights, mode in cases:
        with pytest.raises(ValueError):
            cc.cc_score_layer(wl.shape, weights, pkg.Cache(c_dev), mode, scores, ws)
        with pytest.raises(ValueError):
            cc.cc_score_rows(wl.shape, weights, pkg.Cache(c_dev), mode, False, None, None, scores, ws)
    assert cc.cc_get_status() == cc.CC_OK


def test_kv_copy_that_does_not_fit_is_refused_before_any_launch(cc):
    """The per-layer K/V copy (fp16 mode, or an e4m3 cache) lives in the
    activation buffer, 2 * d_ff bytes per slot: a shape whose K and V need
    more (8 KV heads of 128 against d_ff 1024) is refused with
    CC_ERR_UNSUPPORTED before anything is enqueued; the bf16 mode over the
    bf16 cache takes it."""
    import bench
    import paper_2607_27600_gb300 as pkg
    from synth.configs import ModelShape
    shape = ModelShape(n_layers=1, d_model=256, n_q_heads=8, n_kv_heads=8, head_dim=128,
                       d_ff=1024, vocab=1000, rope_theta=1e4, rms_eps=1e-5)
    w = synth.model_weights(shape, 91, device="cuda")
    c = synth.synthetic_cache(shape, [100], 128, 92, device="cuda")
    c8 = bench.to_e4m3_cache(synth.synthetic_cache(shape, [100], 128, 92, device="cuda"))
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, 1, 128, cc.SCORE_LOGIT))
    cases = ((cc.f16_weights(w), c, cc.SCORE_LOGIT | cc.SCORE_F16),
             (w, c8, cc.SCORE_LOGIT))
    for weights, cache, mode in cases:
        scores = torch.full((1, 128), float("nan"), device="cuda")
        with pytest.raises(cc.CCError) as e:
            cc.cc_score_layer(shape, pkg.Weights(weights), pkg.Cache(cache), mode, scores, ws)
        assert e.value.code == cc.CC_ERR_UNSUPPORTED
        assert torch.isnan(scores).all()   # nothing ran
    assert cc.cc_get_status() == cc.CC_OK
    scores = torch.empty(1, 128, device="cuda")
    cc.cc_score_layer(shape, pkg.Weights(w), pkg.Cache(c), cc.SCORE_LOGIT, scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
