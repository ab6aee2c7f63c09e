"""Captured call sequences (cc_graph_*): a decode step and a refresh cycle
recorded once and replayed over a cache whose device contents change between
replays, checked against the oracle at every replay."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests._util import bf16_round, causal_cache, keep_set_ok, rel_err, to_device, to_np
from tests.test_gpu_append import SMALL_GPU, TOL, _decode_check, _rel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


def _copy_into(dst, src):
    """Device cache tree `src` into the buffers of `dst` (same shapes)."""
    for k, v in src.items():
        if isinstance(v, list):
            for a, b in zip(dst[k], v):
                a.copy_(b)
        elif v is not None:
            dst[k].copy_(v)


def test_decode_graph_replays_match_oracle(cc):
    """One decode step captured after an eager step, then replayed four times
    with the oracle's tokens written into the same input buffer: the cache
    grows by one slot per replay (long memories: the attention takes key
    splits)."""
    import paper_2607_27600_gb300 as pkg
    shape, seq, cap, seed = SMALL_GPU, [1500, 300, 1999], 2048, 59
    w_np = to_np(synth.model_weights(shape, seed, with_kv_proj=True))
    c_np = causal_cache(shape, w_np, seq, cap, seed)
    b = len(seq)
    weights, c_dev = pkg.Weights(to_device(w_np)), to_device(c_np)
    cache = pkg.Cache(c_dev)
    cn = {k: ([np.asarray(x, np.float64).copy() for x in v] if isinstance(v, list) else
              np.asarray(v).copy()) for k, v in c_np.items()}
    ws = cc.alloc_workspace(cc.cc_decode_workspace_size(shape, b, cap))
    tok = np.random.default_rng(seed).integers(0, shape.vocab, size=b)
    tok_dev = torch.empty(b, dtype=torch.int32, device="cuda")
    nxt = torch.empty(b, dtype=torch.int32, device="cuda")
    best = torch.empty(b, dtype=torch.float32, device="cuda")
    s = torch.cuda.Stream()
    graph = None
    try:
        with torch.cuda.stream(s):
            for step in range(5):
                tok_dev.copy_(torch.from_numpy(tok.astype(np.int32)))
                if step == 0:   # eager, which also sets up the kernels
                    cc.cc_decode_step(shape, weights, cache, tok_dev, nxt, best, ws)
                else:
                    if graph is None:
                        cc.cc_graph_begin()
                        cc.cc_decode_step(shape, weights, cache, tok_dev, nxt, best, ws)
                        graph = cc.cc_graph_end()
                    cc.cc_graph_launch(graph)
                assert cc.cc_get_status() == cc.CC_OK
                o_next, _, o_logits = oracle.decode_step(shape, w_np, cn, tok)
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
                for x in cn["k"] + cn["v"] + [cn["h_last"]]:
                    for i in range(b):
                        n1 = int(cn["seq_len"][i])
                        x[i, n1 - 1] = bf16_round(x[i, n1 - 1])
                tok = o_next
    finally:
        if graph is not None:
            cc.cc_graph_destroy(graph)


def test_refresh_cycle_graph_over_two_cache_states(cc):
    """Fast scoring (the precise mode), keep-set selection and compaction
    captured once, then replayed over two different cache contents (lengths
    and budgets too) copied into the same buffers: scores within tolerance,
    the keep-set within the stated bar against the oracle's scores and exact
    against the oracle's select on the replay's own scores, compaction
    bit-exact."""
    import paper_2607_27600_gb300 as pkg
    shape, cap = SMALL_GPU, 320
    states = [([300, 129, 64], [100, 129, 10], 61), ([250, 320, 5], [60, 80, 5], 62)]
    w_np = to_np(synth.model_weights(shape, 60, with_kv_proj=True))
    weights = pkg.Weights(to_device(w_np))
    b = 3
    first = causal_cache(shape, w_np, states[0][0], cap, states[0][2])
    c_dev = to_device(first)
    cache = pkg.Cache(c_dev)
    budget = torch.zeros(b, dtype=torch.int32, device="cuda")
    scores = torch.empty((b, cap), dtype=torch.float32, device="cuda")
    keep_idx = torch.empty((b, cap), dtype=torch.int32, device="cuda")
    keep_count = torch.empty(b, dtype=torch.int32, device="cuda")
    mode = cc.SCORE_LOGIT | cc.SCORE_PRECISE
    sws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode))
    kws = cc.alloc_workspace(cc.cc_select_workspace_size(b, cap))
    cws = cc.alloc_workspace(cc.cc_compact_workspace_size(shape, cache))
    s = torch.cuda.Stream()

    def cycle():
        cc.cc_score_layer(shape, weights, cache, mode, scores, sws)
        cc.cc_select_keep(scores, c_dev["seq_len"], b, cap, budget, 0, keep_idx, keep_count, kws)
        cc.cc_compact_kv(shape, cache, keep_idx, keep_count, cws)

    graph = None
    try:
        with torch.cuda.stream(s):
            budget.copy_(torch.tensor(states[0][1], dtype=torch.int32))
            cycle()   # eager once: sets up the kernels
            assert cc.cc_get_status() == cc.CC_OK
            cc.cc_graph_begin()
            cycle()
            graph = cc.cc_graph_end()
            for seq, budgets, seed in states:
                c_np = causal_cache(shape, w_np, seq, cap, seed)
                _copy_into(c_dev, to_device(c_np))
                budget.copy_(torch.tensor(budgets, dtype=torch.int32))
                cc.cc_graph_launch(graph)
                assert cc.cc_get_status() == cc.CC_OK
                want = oracle.score_layer(shape, w_np, c_np)
                got = scores.cpu().numpy()
                assert rel_err(got, want) < TOL
                gi, gc = keep_idx.cpu().numpy(), keep_count.cpu().numpy()
                oi, oc = oracle.select_keep(got, seq, budgets)
                assert np.array_equal(gc, oc)
                for i in range(b):
                    assert np.array_equal(gi[i, :oc[i]], oi[i, :oc[i]])
                wi, wc = oracle.select_keep(want.astype(np.float32), seq, budgets)
                ok, det = keep_set_ok(gi, gc, wi, wc, want, seq, budgets)
                assert ok, det
                for name in ("tokens", "pos"):
                    np.testing.assert_array_equal(c_dev[name].cpu().numpy(),
                                                  oracle.compact(c_np[name], gi, gc))
                for name in ("k", "v"):
                    for l in range(shape.n_layers):
                        np.testing.assert_array_equal(c_dev[name][l].float().cpu().numpy(),
                                                      oracle.compact(c_np[name][l], gi, gc))
                assert c_dev["seq_len"].cpu().tolist() == gc.tolist()
    finally:
        if graph is not None:
            cc.cc_graph_destroy(graph)
