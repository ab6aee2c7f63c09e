"""cc_kv_cache.kv_ready: K/V uploads still in flight on another stream when a
call is enqueued.  The uploads are held back on their stream by a spin of
~10 ms, so a call that did not wait for the events would read the zeroed
buffers; every result must equal the resident cache's bit for bit."""
import numpy as np
import pytest
import torch

import synth
from tests._util import causal_cache, to_device, to_np
from tests.test_gpu_append import SMALL_GPU

pytestmark = pytest.mark.gpu

SPIN_CYCLES = 20_000_000   # ~10 ms at 2 GHz


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


def late_upload(dev, layers):
    """A copy of cache dict `dev` whose K/V of `layers` are zeroed now and
    uploaded from pinned host copies on a side stream after a spin; returns
    (copy, per-layer events or None)."""
    late = {k: ([x.clone() for x in v] if isinstance(v, list) else
                (v.clone() if isinstance(v, torch.Tensor) else v)) for k, v in dev.items()}
    host = {key: [x.cpu().pin_memory() for x in dev[key]] for key in ("k", "v")}
    for key in ("k", "v"):
        for l in layers:
            late[key][l].zero_()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    events = [None] * len(dev["k"])
    with torch.cuda.stream(side):
        torch.cuda._sleep(SPIN_CYCLES)
        for l in layers:
            late["k"][l].copy_(host["k"][l], non_blocking=True)
            late["v"][l].copy_(host["v"][l], non_blocking=True)
            events[l] = torch.cuda.Event()
            events[l].record(side)
    return late, events


def _bits(x):
    return x.contiguous().view(torch.uint8).cpu().numpy()


@pytest.mark.parametrize("full", [False, True])
def test_scoring_and_compaction_wait_for_the_uploads(cc, full):
    import paper_2607_27600_gb300 as pkg
    seq, cap, budgets = [300, 129, 64], 384, [100, 129, 10]
    b = len(seq)
    w_np = to_np(synth.model_weights(SMALL_GPU, 98, with_kv_proj=True))
    dev = to_device(causal_cache(SMALL_GPU, w_np, seq, cap, 98))
    weights = pkg.Weights(to_device(w_np))
    n_l = SMALL_GPU.n_layers
    layers = list(range(n_l)) if full else [n_l - 1]
    fn = cc.cc_score_full if full else cc.cc_score_layer
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(SMALL_GPU, b, cap, cc.SCORE_LOGIT))

    def score(cache):
        s = torch.full((b, cap), float("nan"), device="cuda")
        fn(SMALL_GPU, weights, cache, cc.SCORE_LOGIT, s, ws)
        return s

    ref = score(pkg.Cache(dev))
    late, events = late_upload(dev, layers)
    cache = pkg.Cache(late)
    cache.set_kv_ready(events)
    got = score(cache)
    torch.cuda.synchronize()
    assert cc.cc_get_status() == cc.CC_OK
    np.testing.assert_array_equal(got.cpu().numpy(), ref.cpu().numpy())

    # the compaction waits for every layer's event
    budget = torch.tensor(budgets, dtype=torch.int32, device="cuda")
    keep_idx = torch.full((b, cap), -1, dtype=torch.int32, device="cuda")
    keep_count = torch.zeros(b, dtype=torch.int32, device="cuda")
    cc.cc_select_keep(ref, dev["seq_len"], b, cap, budget, 0, keep_idx, keep_count)
    want = pkg.Cache({**dev, "seq_len": dev["seq_len"].clone()})
    cws = cc.alloc_workspace(cc.cc_compact_workspace_size(SMALL_GPU, want))
    cc.cc_compact_kv(SMALL_GPU, want, keep_idx, keep_count, cws)
    late2, events2 = late_upload({**late, "seq_len": dev["seq_len"]}, list(range(n_l)))
    cache2 = pkg.Cache(late2)
    cache2.set_kv_ready(events2)
    cc.cc_compact_kv(SMALL_GPU, cache2, keep_idx, keep_count, cws)
    torch.cuda.synchronize()
    assert cc.cc_get_status() == cc.CC_OK
    cnt = keep_count.cpu().numpy()
    for key in ("k", "v"):
        for l in range(n_l):
            for i in range(b):
                n = int(cnt[i])
                np.testing.assert_array_equal(_bits(late2[key][l][i, :n]),
                                              _bits(want.d[key][l][i, :n]))


def test_append_waits_for_the_uploads(cc):
    """The append writes each layer's new K/V rows and attends over the old
    ones: both after that layer's event."""
    import paper_2607_27600_gb300 as pkg
    seq, cap = [200, 90, 30], 320
    w_np = to_np(synth.model_weights(SMALL_GPU, 99, with_kv_proj=True))
    dev = to_device(causal_cache(SMALL_GPU, w_np, seq, cap, 99))
    r = np.random.default_rng(99)
    chunks = [r.integers(0, SMALL_GPU.vocab, size=m) for m in (40, 7, 1)]
    b, mx = len(chunks), 40
    tok = np.zeros((b, mx), np.int32)
    for i, t in enumerate(chunks):
        tok[i, :len(t)] = t
    tok_d = torch.from_numpy(tok).cuda()
    cnt = torch.tensor([len(t) for t in chunks], dtype=torch.int32, device="cuda")
    weights = pkg.Weights(to_device(w_np))
    ws = cc.alloc_workspace(cc.cc_append_workspace_size(SMALL_GPU, b, cap))
    late, events = late_upload(dev, list(range(SMALL_GPU.n_layers)))
    ref = pkg.Cache(dev)
    cc.cc_append_chunk(SMALL_GPU, weights, ref, tok_d, None, cnt, mx, ws)
    cache = pkg.Cache(late)
    cache.set_kv_ready(events)
    cc.cc_append_chunk(SMALL_GPU, weights, cache, tok_d, None, cnt, mx, ws)
    torch.cuda.synchronize()
    assert cc.cc_get_status() == cc.CC_OK
    after = dev["seq_len"].cpu().tolist()
    assert late["seq_len"].cpu().tolist() == after
    for key in ("k", "v"):
        for l in range(SMALL_GPU.n_layers):
            for i, n in enumerate(after):
                np.testing.assert_array_equal(_bits(late[key][l][i, :n]), _bits(dev[key][l][i, :n]))
    np.testing.assert_array_equal(_bits(late["h_last"]), _bits(dev["h_last"]))
