"""GPU parity of the inference cycle in pre-fill (cc_append_chunk,
Algorithm CacheManagedInference / DoInference over a chunk) against the
oracle's append_chunk, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth.configs import ModelShape
from tests._util import bf16_round, causal_cache, rel_err, to_device, to_np

pytestmark = pytest.mark.gpu

TOL = 2e-2
SMALL_GPU = ModelShape(n_layers=2, d_model=256, n_q_heads=8, n_kv_heads=2, head_dim=64,
                       d_ff=384, vocab=1000, rope_theta=1e4, rms_eps=1e-5)


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


def _rel(got, want):
    """max |g - o| / max |o| (the attention tests' bar for bf16 outputs)."""
    got, want = np.asarray(got, np.float64), np.asarray(want, np.float64)
    return float(np.abs(got - want).max() / max(np.abs(want).max(), 1e-30))


def _gpu_append(cc, shape, w_np, c_np, chunks, pos=None):
    """Runs cc_append_chunk on device copies; returns the device cache (numpy)."""
    import paper_2607_27600_gb300 as pkg
    b = len(chunks)
    mx = max(1, max(len(t) for t in chunks))
    tok = np.zeros((b, mx), np.int32)
    ps = np.zeros((b, mx), np.int32)
    for i, t in enumerate(chunks):
        tok[i, :len(t)] = t
        if pos is not None:
            ps[i, :len(t)] = pos[i]
    cnt = np.array([len(t) for t in chunks], np.int32)
    w, c = to_device(w_np), to_device(c_np)
    weights, cache = pkg.Weights(w), pkg.Cache(c)
    ws = cc.alloc_workspace(cc.cc_append_workspace_size(shape, b, c["tokens"].shape[1]))
    cc.cc_append_chunk(shape, weights, cache, torch.from_numpy(tok).cuda(),
                       None if pos is None else torch.from_numpy(ps).cuda(),
                       torch.from_numpy(cnt).cuda(), mx, ws)
    status = cc.cc_get_status()
    return to_np(c), status, (weights, cache)


def _oracle_append(shape, w_np, c_np, chunks, pos=None):
    c = {k: ([np.asarray(x, np.float64).copy() for x in v] if isinstance(v, list) else
             np.asarray(v).copy()) for k, v in c_np.items()}
    for b, t in enumerate(chunks):
        if len(t):
            oracle.append_chunk(shape, w_np, c, b, t, None if pos is None else pos[b])
    return c


def _check(shape, got, want, chunks, n0, exact_memory=True):
    for b, t in enumerate(chunks):
        sl = slice(n0[b], n0[b] + len(t))
        assert got["seq_len"][b] == n0[b] + len(t)
        np.testing.assert_array_equal(got["tokens"][b, sl], want["tokens"][b, sl])
        np.testing.assert_array_equal(got["pos"][b, sl], want["pos"][b, sl])
        if not len(t):
            continue
        for l in range(shape.n_layers):
            assert _rel(got["k"][l][b, sl], want["k"][l][b, sl]) < TOL, ("k", l, b)
            assert _rel(got["v"][l][b, sl], want["v"][l][b, sl]) < TOL, ("v", l, b)
        if got.get("h_last") is not None:
            assert _rel(got["h_last"][b, sl], want["h_last"][b, sl]) < TOL, ("h_last", b)
        # memory slots untouched (exactly, unless earlier appends put values of
        # both sides' own rounding there)
        for l in range(shape.n_layers):
            if exact_memory:
                np.testing.assert_array_equal(got["k"][l][b, :n0[b]],
                                              np.asarray(want["k"][l][b, :n0[b]], np.float32))
            else:
                assert _rel(got["k"][l][b, :n0[b]], want["k"][l][b, :n0[b]]) < TOL


def _setup(shape, seq, cap, seed):
    w_np = to_np(synth.model_weights(shape, seed, with_kv_proj=True))
    c_np = causal_cache(shape, w_np, seq, cap, seed)
    return w_np, c_np


def test_append_into_empty_cache_ragged(cc):
    """Empty cache, chunks of 300 and 77 tokens: the causal forward."""
    w_np, c_np = _setup(SMALL_GPU, [0, 0], 320, seed=51)
    r = np.random.default_rng(51)
    chunks = [r.integers(0, SMALL_GPU.vocab, size=300), r.integers(0, SMALL_GPU.vocab, size=77)]
    got, status, _ = _gpu_append(cc, SMALL_GPU, w_np, c_np, chunks)
    assert status == cc.CC_OK
    want = _oracle_append(SMALL_GPU, w_np, c_np, chunks)
    _check(SMALL_GPU, got, want, chunks, [0, 0])


@pytest.mark.parametrize("variant", ["plain", "qkv_bias+rope_scaling"])
def test_append_after_compaction_then_score(cc, variant):
    """Memory built by the oracle's causal pass, compacted to a seeded keep-set
    (positions keep their original values), then a chunk appended to each
    sequence (one of them empty); the appended cache then scores like the
    oracle's appended cache."""
    import paper_2607_27600_gb300 as pkg
    shape = SMALL_GPU if variant == "plain" else ModelShape(
        **{**SMALL_GPU.__dict__, "qkv_bias": True, "rope_scaling": (8.0, 1.0, 4.0, 64)})
    w_np, c_np = _setup(shape, [200, 50, 90], 384, seed=52)
    r = np.random.default_rng(52)
    keep = np.full((3, 384), -1, np.int32)
    cnt = np.array([120, 50, 31], np.int32)
    for b, (n, j) in enumerate(zip([200, 50, 90], cnt)):
        k = np.sort(np.concatenate([r.choice(n - 1, size=j - 1, replace=False), [n - 1]]))
        keep[b, :j] = k
    for key in ("tokens", "pos", "h_last"):
        c_np[key] = oracle.compact(c_np[key], keep, cnt)
    c_np["k"] = [oracle.compact(x, keep, cnt) for x in c_np["k"]]
    c_np["v"] = [oracle.compact(x, keep, cnt) for x in c_np["v"]]
    c_np["seq_len"] = cnt.copy()
    chunks = [r.integers(0, shape.vocab, size=130), np.zeros(0, np.int64),
              r.integers(0, shape.vocab, size=255)]
    got, status, (weights, cache) = _gpu_append(cc, shape, w_np, c_np, chunks)
    assert status == cc.CC_OK
    want = _oracle_append(shape, w_np, c_np, chunks)
    _check(shape, got, want, chunks, list(cnt))
    # score the appended caches: GPU on its own, the oracle on its own
    b, cap = 3, 384
    scores = torch.full((b, cap), float("nan"), device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, cc.SCORE_LOGIT))
    cc.cc_score_layer(shape, weights, cache, cc.SCORE_LOGIT, scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
    want_s = oracle.score_layer(shape, w_np, want)
    assert rel_err(scores.cpu().numpy(), want_s) < TOL


def test_append_explicit_positions_and_bad_count(cc):
    """Given positions are stored and used for RoPE; a count past the cap is
    reported on the device and leaves that sequence as it was."""
    w_np, c_np = _setup(SMALL_GPU, [40, 60], 128, seed=53)
    r = np.random.default_rng(53)
    chunks = [r.integers(0, SMALL_GPU.vocab, size=30), r.integers(0, SMALL_GPU.vocab, size=10)]
    pos = [np.arange(1000, 1030), np.arange(500, 510) * 3]
    got, status, _ = _gpu_append(cc, SMALL_GPU, w_np, c_np, chunks, pos=pos)
    assert status == cc.CC_OK
    want = _oracle_append(SMALL_GPU, w_np, c_np, chunks, pos=pos)
    _check(SMALL_GPU, got, want, chunks, [40, 60])
    np.testing.assert_array_equal(got["pos"][0, 40:70], pos[0])
    # 100 more slots do not fit in sequence 1 (60 + 100 > 128): nothing appended there
    chunks2 = [r.integers(0, SMALL_GPU.vocab, size=5), r.integers(0, SMALL_GPU.vocab, size=100)]
    got2, status2, _ = _gpu_append(cc, SMALL_GPU, w_np, c_np, chunks2)
    assert status2 == cc.CC_ERR_DEVICE_ARG
    assert list(got2["seq_len"]) == [45, 60]
    assert cc.cc_get_status() == cc.CC_OK      # the status word was read and cleared


def test_append_short_chunks_over_long_memory_key_splits(cc):
    """Short ragged chunks (5, 20, 1 tokens) after 1500, 300 and 1999 memory
    slots: six attention units, so each unit's key tiles are split over
    several CTAs (4 on a 152-SM GPU) and merged by the combine kernel; the
    300-slot sequence has fewer tiles than splits (an empty split)."""
    seq, cap = [1500, 300, 1999], 2048
    w_np, c_np = _setup(SMALL_GPU, seq, cap, seed=57)
    r = np.random.default_rng(57)
    chunks = [r.integers(0, SMALL_GPU.vocab, size=m) for m in (5, 20, 1)]
    got, status, _ = _gpu_append(cc, SMALL_GPU, w_np, c_np, chunks)
    assert status == cc.CC_OK
    want = _oracle_append(SMALL_GPU, w_np, c_np, chunks)
    _check(SMALL_GPU, got, want, chunks, seq)


def test_append_llama_shape_chunk_over_long_memory(cc):
    """Llama-3-8B layer shapes (first two layers), a 1024-token chunk after
    8192 synthetic memory slots: every appended K/V row of both layers,
    H^(L-1) and the chunk's positions."""
    shape = ModelShape(**{**synth.configs.LLAMA3_8B.__dict__, "n_layers": 2})
    n0, h, cap = 8192, 1024, 9216
    w = synth.model_weights(shape, 7, device="cuda", with_kv_proj=True)
    c = synth.synthetic_cache(shape, [n0], cap, 7, device="cuda")
    w_np, c_np = to_np(w), to_np(c)
    chunk = synth.tokens((h,), shape.vocab, 7, "chunk").numpy()
    got, status, _ = _gpu_append(cc, shape, w_np, c_np, [chunk])
    assert status == cc.CC_OK
    want = _oracle_append(shape, w_np, c_np, [chunk])
    _check(shape, got, want, [chunk], [n0])
    np.testing.assert_array_equal(got["pos"][0, n0:n0 + h], np.arange(n0, n0 + h))


def test_cache_managed_loop_qwen_shape(cc):
    """Algorithm CacheManagedInference in chunked mode at Qwen2.5-7B layer
    shapes (two layers, q/k/v biases): 8192 memory slots, then per cycle a
    refresh (fast-pass scores on sampled rows vs the oracle; both sides compact
    to the same seeded 2048-slot keep-set, bit-exact) and an inference cycle
    appending 1024 tokens on both sides (every appended K/V row, H^(L-1))."""
    import paper_2607_27600_gb300 as pkg
    shape = ModelShape(**{**synth.configs.QWEN25_7B.__dict__, "n_layers": 2})
    n0, j, h, cap = 8192, 2048, 1024, 8192
    w = synth.model_weights(shape, 9, device="cuda", with_kv_proj=True)
    c = synth.synthetic_cache(shape, [n0], cap, 9, device="cuda")
    w_np, cn = to_np(w), to_np(c)
    cn = {k: ([np.asarray(x, np.float64) for x in v] if isinstance(v, list) else v)
          for k, v in cn.items()}
    weights, cache = pkg.Weights(w), pkg.Cache(c)
    sws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, 1, cap, cc.SCORE_LOGIT))
    cws = cc.alloc_workspace(cc.cc_compact_workspace_size(shape, cache))
    aws = cc.alloc_workspace(cc.cc_append_workspace_size(shape, 1, cap))
    r = np.random.default_rng(9)
    for cycle in range(2):
        n = int(c["seq_len"][0])
        scores = torch.full((1, cap), float("nan"), device="cuda")
        cc.cc_score_layer(shape, weights, cache, cc.SCORE_LOGIT, scores, sws)
        assert cc.cc_get_status() == cc.CC_OK
        rows = [sorted({0, n // 3, n - 2, n - 1} | set(r.choice(n, 20, replace=False).tolist()))]
        want = oracle.score_layer(shape, w_np, cn, rows=rows)
        assert rel_err(scores.cpu().numpy()[0, rows[0]], want[0, rows[0]]) < TOL, cycle
        keep = np.sort(np.concatenate([r.choice(n - 1, size=j - 1, replace=False), [n - 1]]))
        idx = np.full((1, cap), -1, np.int32)
        idx[0, :j] = keep
        cnt = np.array([j], np.int32)
        cc.cc_compact_kv(shape, cache, torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda(),
                         cws)
        for key in ("tokens", "pos", "h_last"):
            cn[key] = oracle.compact(cn[key], idx, cnt)
        cn["k"] = [oracle.compact(x, idx, cnt) for x in cn["k"]]
        cn["v"] = [oracle.compact(x, idx, cnt) for x in cn["v"]]
        cn["seq_len"] = cnt.copy()
        got_k = c["k"][1][0, :j].float().cpu().numpy()
        if cycle == 0:   # synthetic memory only: the gather is bit-exact
            np.testing.assert_array_equal(got_k, np.asarray(cn["k"][1][0, :j], np.float32))
        else:            # kept slots include both sides' own appended rows
            assert _rel(got_k, cn["k"][1][0, :j]) < TOL
        chunk = synth.tokens((1, h), shape.vocab, 9, f"loop.chunk{cycle}")
        cc.cc_append_chunk(shape, weights, cache, chunk.cuda(), None,
                           torch.tensor([h], dtype=torch.int32, device="cuda"), h, aws)
        assert cc.cc_get_status() == cc.CC_OK
        oracle.append_chunk(shape, w_np, cn, 0, chunk.numpy()[0])
        got = to_np(c)
        _check(shape, got, cn, [chunk.numpy()[0]], [j], exact_memory=(cycle == 0))
        # the cache stores bf16: the oracle keeps its own appended rows at that precision
        for x in cn["k"] + cn["v"] + [cn["h_last"]]:
            x[0, j:j + h] = bf16_round(x[0, j:j + h])


def _decode_check(next_tok, best, logits, tol=2e-2):
    """GPU greedy choice vs the oracle's logits: the argmax wherever the
    top-2 gap exceeds tol (relative to the logits' rms), else a token whose
    oracle logit is within tol of the max; the GPU's logit matches."""
    rms = np.sqrt(np.mean(logits * logits))
    srt = np.sort(logits)[::-1]
    if (srt[0] - srt[1]) / rms > tol:
        assert next_tok == int(np.argmax(logits)), (next_tok, int(np.argmax(logits)))
    else:
        assert (srt[0] - logits[next_tok]) / rms <= tol
    assert abs(best - logits[next_tok]) / max(abs(logits[next_tok]), rms) < tol


@pytest.mark.parametrize("shape_name", ["small", "small-long", "small-batch6", "llama2",
                                        "llama2-long"])
def test_decode_steps_match_oracle(cc, shape_name):
    """Greedy decode steps (teacher-forced with the oracle's tokens so both
    sides share the history): next tokens, their logits, appended K/V rows.
    The -long cases attend over enough slots that the attention splits each
    unit's key tiles across CTAs (4 and 8 splits on a 152-SM GPU); six
    sequences take the tile GEMMs instead of the weight-streaming GEMVs."""
    import paper_2607_27600_gb300 as pkg
    if shape_name.startswith("small"):
        shape, seed = SMALL_GPU, 54
        seq, cap = {"small": ([50, 20, 33], 64), "small-long": ([1500, 300, 1999], 2048),
                    # more than four sequences: the tile GEMMs with the argmax epilogue
                    "small-batch6": ([50, 20, 33, 1, 60, 41], 64)}[shape_name]
        w_np = to_np(synth.model_weights(shape, seed, with_kv_proj=True))
        c_np = causal_cache(shape, w_np, seq, cap, seed)
    else:
        shape = ModelShape(**{**synth.configs.LLAMA3_8B.__dict__, "n_layers": 2})
        seq, cap, seed = ([700], 712, 55) if shape_name == "llama2" else ([4000], 4100, 58)
        w = synth.model_weights(shape, seed, device="cuda", with_kv_proj=True)
        c = synth.synthetic_cache(shape, seq, cap, seed, device="cuda")
        w_np, c_np = to_np(w), to_np(c)
    b = len(seq)
    weights, cache = pkg.Weights(to_device(w_np)), None
    c_dev = to_device(c_np)
    cache = pkg.Cache(c_dev)
    cn = {k: ([np.asarray(x, np.float64).copy() for x in v] if isinstance(v, list) else
              np.asarray(v).copy()) for k, v in c_np.items()}
    ws = cc.alloc_workspace(cc.cc_decode_workspace_size(shape, b, cap))
    tok = np.random.default_rng(seed).integers(0, shape.vocab, size=b)
    nxt = torch.empty(b, dtype=torch.int32, device="cuda")
    best = torch.empty(b, dtype=torch.float32, device="cuda")
    for step in range(4):
        cc.cc_decode_step(shape, weights, cache, torch.from_numpy(tok.astype(np.int32)).cuda(),
                          nxt, best, ws)
        assert cc.cc_get_status() == cc.CC_OK
        o_next, o_best, o_logits = oracle.decode_step(shape, w_np, cn, tok)
        g_next, g_best = nxt.cpu().numpy(), best.cpu().numpy()
        for i in range(b):
            _decode_check(int(g_next[i]), float(g_best[i]), o_logits[i])
        got = to_np(c_dev)
        for i in range(b):
            n1 = int(cn["seq_len"][i])
            assert int(got["seq_len"][i]) == n1
            for l in range(shape.n_layers):
                assert _rel(got["k"][l][i, n1 - 1], cn["k"][l][i, n1 - 1]) < TOL
                assert _rel(got["v"][l][i, n1 - 1], cn["v"][l][i, n1 - 1]) < TOL
        # the cache stores bf16: the oracle keeps its appended rows at that precision
        for x in cn["k"] + cn["v"] + [cn["h_last"]]:
            for i in range(b):
                n1 = int(cn["seq_len"][i])
                x[i, n1 - 1] = bf16_round(x[i, n1 - 1])
        tok = o_next


def test_decode_full_cache_reports_and_skips(cc):
    import paper_2607_27600_gb300 as pkg
    w_np, c_np = _setup(SMALL_GPU, [64, 10], 64, seed=56)
    weights, c_dev = pkg.Weights(to_device(w_np)), to_device(c_np)
    cache = pkg.Cache(c_dev)
    ws = cc.alloc_workspace(cc.cc_decode_workspace_size(SMALL_GPU, 2, 64))
    nxt = torch.empty(2, dtype=torch.int32, device="cuda")
    cc.cc_decode_step(SMALL_GPU, weights, cache, torch.tensor([3, 4], dtype=torch.int32,
                                                              device="cuda"), nxt, None, ws)
    assert cc.cc_get_status() == cc.CC_ERR_DEVICE_ARG
    assert nxt.cpu().tolist()[0] == -1 and nxt.cpu().tolist()[1] >= 0
    assert c_dev["seq_len"].cpu().tolist() == [64, 11]
