"""Head-major K/V buffers (cc_kv_cache.kv_layout = CC_KV_HEAD_MAJOR: k[l],
v[l] are [batch][Hkv][cap][head_dim]).  The layout only moves where each
head's vectors live, so every result must equal the slot-major cache's bit
for bit; the oracle bars of the slot-major tests hold for it as well."""
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
HEAD_MAJOR = 1


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


def head_major(dev):
    """A head-major copy of device cache dict `dev`."""
    out = {k: (v.clone() if isinstance(v, torch.Tensor) else v) for k, v in dev.items()
           if k not in ("k", "v")}
    for key in ("k", "v"):
        out[key] = [x.permute(0, 2, 1, 3).contiguous() for x in dev[key]]
    out["kv_layout"] = HEAD_MAJOR
    return out


def slot_view(hm, key, l):
    return hm[key][l].permute(0, 2, 1, 3)


def _bits(x):
    return x.contiguous().view(torch.uint8).cpu().numpy()


def _score(cc, shape, w_np, d, full):
    import paper_2607_27600_gb300 as pkg
    weights, cache = pkg.Weights(to_device(w_np)), pkg.Cache(d)
    b, cap = d["tokens"].shape
    scores = torch.full((b, cap), float("nan"), device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, cc.SCORE_LOGIT))
    (cc.cc_score_full if full else cc.cc_score_layer)(shape, weights, cache, cc.SCORE_LOGIT,
                                                       scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
    return scores, cache


@pytest.mark.parametrize("full", [False, True])
@pytest.mark.parametrize("fmt", ["bf16", "e4m3"])
def test_head_major_scores(cc, full, fmt):
    from tests.test_gpu_fp8 import fp8_views
    seq, cap = [300, 129, 1, 64], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 91, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 91)
    on, dev = fp8_views(c_np) if fmt == "e4m3" else (c_np, to_device(c_np))
    flat, _ = _score(cc, SMALL_GPU, w_np, dev, full)
    hm, _ = _score(cc, SMALL_GPU, w_np, head_major(dev), full)
    np.testing.assert_array_equal(hm.cpu().numpy(), flat.cpu().numpy())
    want = (oracle.score_full if full else oracle.score_layer)(SMALL_GPU, w_np, on)
    assert rel_err(hm.cpu().numpy(), want) < TOL


def test_head_major_importance_scores(cc):
    import paper_2607_27600_gb300 as pkg
    seq, cap = [300, 129, 64], 384
    w_np = to_np(synth.model_weights(SMALL_GPU, 92, with_kv_proj=True))
    dev = to_device(causal_cache(SMALL_GPU, w_np, seq, cap, 92))
    out = []
    for d in (dev, head_major(dev)):
        scores = torch.zeros((len(seq), cap), device="cuda")
        ws = cc.alloc_workspace(cc.cc_keyattn_workspace_size(SMALL_GPU, len(seq), cap))
        cc.cc_score_importance(SMALL_GPU, pkg.Cache(d), scores, ws)
        assert cc.cc_get_status() == cc.CC_OK
        out.append(scores.cpu().numpy())
    np.testing.assert_array_equal(out[1], out[0])


def test_head_major_refresh_cycle(cc):
    """Score, select and compact: the head-major buffers hold the slot-major
    cache's compacted rows (each row moved as Hkv segments)."""
    seq, cap, budgets = [300, 129, 64], 384, [100, 129, 10]
    w_np = to_np(synth.model_weights(SMALL_GPU, 93, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, 93)
    dev = to_device(c_np)
    hdev = head_major(dev)
    b = len(seq)
    res = []
    for d in (dev, hdev):
        scores, cache = _score(cc, SMALL_GPU, w_np, d, False)
        budget = torch.tensor(budgets, dtype=torch.int32, device="cuda")
        keep_idx = torch.full((b, cap), -1, dtype=torch.int32, device="cuda")
        keep_count = torch.zeros(b, dtype=torch.int32, device="cuda")
        cc.cc_select_keep(scores, d["seq_len"], b, cap, budget, 0, keep_idx, keep_count)
        ws = cc.alloc_workspace(cc.cc_compact_workspace_size(SMALL_GPU, cache))
        cc.cc_compact_kv(SMALL_GPU, cache, keep_idx, keep_count, ws)
        assert cc.cc_get_status() == cc.CC_OK
        res.append((keep_idx.cpu().numpy(), keep_count.cpu().numpy()))
    (gi, gc), (hi, hc) = res
    np.testing.assert_array_equal(hi, gi)
    np.testing.assert_array_equal(hc, gc)
    for key in ("k", "v"):
        for l in range(SMALL_GPU.n_layers):
            got = slot_view(hdev, key, l)
            for i in range(b):
                n = int(gc[i])
                np.testing.assert_array_equal(_bits(got[i, :n]), _bits(dev[key][l][i, :n]))
                np.testing.assert_array_equal(
                    got[i, :n].float().cpu().numpy(),
                    oracle.compact(np.asarray(c_np[key][l], np.float32), gi, gc)[i, :n])


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


@pytest.mark.parametrize("case", ["small", "llama-fused", "llama-fused-e4m3"])
def test_head_major_append(cc, case):
    """Appended K/V rows (separate projections; fused q/k/v GEMM at Llama-3-8B
    layer shapes; bf16 and e4m3) land in each head's buffer exactly as the
    slot-major cache stores them."""
    from tests.test_gpu_fp8 import fp8_views
    if case == "small":
        shape, seq, cap, seed = SMALL_GPU, [200, 90, 30], 320, 94
        w_np = to_np(synth.model_weights(shape, seed, with_kv_proj=True))
        c_np = causal_cache(shape, w_np, seq, cap, seed)
        r = np.random.default_rng(seed)
        chunks = [r.integers(0, shape.vocab, size=m) for m in (40, 7, 0)]
    else:
        shape = ModelShape(**{**synth.configs.LLAMA3_8B.__dict__, "n_layers": 2})
        seq, cap, seed = [1200], 1536, 95
        w = synth.model_weights(shape, seed, device="cuda", with_kv_proj=True)
        c = synth.synthetic_cache(shape, seq, cap, seed, device="cuda")
        w_np, c_np = to_np(w), to_np(c)
        chunks = [synth.tokens((300,), shape.vocab, seed, "chunk").numpy()]
    dev = fp8_views(c_np)[1] if case.endswith("e4m3") else to_device(c_np)
    hdev = head_major(dev)
    _append(cc, shape, w_np, dev, chunks)
    _append(cc, shape, w_np, hdev, chunks)
    after = [n + len(t) for n, t in zip(seq, chunks)]
    assert hdev["seq_len"].cpu().tolist() == after
    for key in ("k", "v"):
        for l in range(shape.n_layers):
            got = slot_view(hdev, key, l)
            for i, n in enumerate(after):
                np.testing.assert_array_equal(_bits(got[i, :n]), _bits(dev[key][l][i, :n]))


def test_head_major_decode_steps(cc):
    """Decode over head-major buffers (GEMV writers, key-split decode
    attention): next tokens and logits equal the slot-major cache's, and the
    oracle's greedy choice."""
    import paper_2607_27600_gb300 as pkg
    seq, cap, seed = [1500, 300, 1999], 2048, 96
    w_np = to_np(synth.model_weights(SMALL_GPU, seed, with_kv_proj=True))
    c_np = causal_cache(SMALL_GPU, w_np, seq, cap, seed)
    dev = to_device(c_np)
    hdev = head_major(dev)
    on = {k: ([np.asarray(x, np.float64).copy() for x in v] if isinstance(v, list) else
              np.asarray(v).copy()) for k, v in c_np.items()}
    b = len(seq)
    tok = np.random.default_rng(seed).integers(0, SMALL_GPU.vocab, size=b)
    outs = []
    for d in (dev, hdev):
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
    for key in ("k", "v"):
        for l in range(SMALL_GPU.n_layers):
            got = slot_view(hdev, key, l)
            for i, n in enumerate(seq):
                np.testing.assert_array_equal(_bits(got[i, :n + 1]), _bits(dev[key][l][i, :n + 1]))
    _, _, o_logits = oracle.decode_step(SMALL_GPU, w_np, on, tok)
    for i in range(b):
        _decode_check(int(outs[1][0][i]), float(outs[1][1][i]), o_logits[i])


def test_head_major_paged_is_refused(cc):
    import paper_2607_27600_gb300 as pkg
    from tests.test_gpu_paged import paginate
    w_np = to_np(synth.model_weights(SMALL_GPU, 97, with_kv_proj=True))
    dev = to_device(causal_cache(SMALL_GPU, w_np, [100], 256, 97))
    bad = paginate(dev, 128, seed=97)
    bad["kv_layout"] = HEAD_MAJOR
    scores = torch.zeros((1, 256), device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(SMALL_GPU, 1, 256, cc.SCORE_LOGIT))
    with pytest.raises(cc.CCError) as e:
        cc.cc_score_layer(SMALL_GPU, pkg.Weights(to_device(w_np)), pkg.Cache(bad),
                          cc.SCORE_LOGIT, scores, ws)
    assert e.value.code == cc.CC_ERR_INVALID_ARG
