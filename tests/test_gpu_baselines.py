"""GPU parity of the paper's comparison scorers (Sec. 4: sliding window,
importance, H2O) through the C ABI against the oracle.

Tolerance 2e-3 (max relative error against max(|o|, rms(o))): the scores are
sums of softmax weights computed in fp32 from the same bf16 keys (exact
products), with 2-ulp exp2 and fp32 sums of at most a few thousand terms."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth.configs import ModelShape
from tests._util import rel_err, to_np

pytestmark = pytest.mark.gpu

TOL = 2e-3
SHAPE64 = ModelShape(n_layers=2, d_model=256, n_q_heads=8, n_kv_heads=2, head_dim=64,
                     d_ff=384, vocab=1000, rope_theta=1e4, rms_eps=1e-5)
SHAPE128 = ModelShape(n_layers=3, d_model=512, n_q_heads=8, n_kv_heads=4, head_dim=128,
                      d_ff=512, vocab=1000, rope_theta=1e4, rms_eps=1e-5)


@pytest.fixture(scope="module")
def pkg():
    import paper_2607_27600_gb300 as p
    p.load_library()
    return p


def _cache(shape, seq, cap, seed, stale_nan=True):
    c = synth.synthetic_cache(shape, seq, cap, seed, device="cuda", with_h_last=False)
    if stale_nan:   # slots past a sequence's end may hold any bits
        for b, n in enumerate(seq):
            for k in c["k"]:
                k[b, n:] = float("nan")
    c["h2o_acc"] = torch.zeros(len(seq), cap, dtype=torch.float32, device="cuda")
    return c


def _np_cache(c):
    return {"k": [x.float().cpu().numpy() for x in c["k"]], "pos": c["pos"].cpu().numpy(),
            "seq_len": c["seq_len"].cpu().numpy()}


def test_recency_is_the_position(pkg):
    from paper_2607_27600_gb300 import cc
    c = _cache(SHAPE64, [300, 0, 77], 320, seed=61)
    c["pos"][0, :300] = torch.arange(1000, 1300, device="cuda", dtype=torch.int32)
    scores = torch.full((3, 320), float("nan"), device="cuda")
    cc.cc_score_recency(pkg.Cache(c), scores)
    np.testing.assert_array_equal(scores.cpu().numpy(), oracle.recency_scores(_np_cache(c)))


@pytest.mark.parametrize("shape,seq,cap", [(SHAPE64, [300, 129, 1, 64], 320),
                                           (SHAPE128, [1000, 257], 1024)])
def test_importance_matches_oracle_and_is_deterministic(pkg, shape, seq, cap):
    from paper_2607_27600_gb300 import cc
    c = _cache(shape, seq, cap, seed=62)
    cache = pkg.Cache(c)
    ws = cc.alloc_workspace(cc.cc_keyattn_workspace_size(shape, len(seq), cap))
    a = torch.full((len(seq), cap), float("nan"), device="cuda")
    b = torch.full_like(a, float("nan"))
    cc.cc_score_importance(shape, cache, a, ws)
    cc.cc_score_importance(shape, cache, b, ws)
    assert cc.cc_get_status() == cc.CC_OK
    want = oracle.importance_scores(shape, _np_cache(c))
    got = a.cpu().numpy()
    for i, n in enumerate(seq):
        assert rel_err(got[i, :n], want[i, :n]) < TOL, (i, rel_err(got[i, :n], want[i, :n]))
        assert np.all(got[i, n:] == -np.inf)
    assert torch.equal(a, b)


def test_h2o_running_total_then_refresh(pkg):
    """Two accumulations (recent = 100, then a shorter sequence after a
    compaction), refresh scores with the recent slots forced, and the totals
    moved bit-exactly by the compaction."""
    from paper_2607_27600_gb300 import cc
    shape, seq, cap, recent = SHAPE128, [600, 333], 640, 100
    c = _cache(shape, seq, cap, seed=63)
    cache = pkg.Cache(c)
    ws = cc.alloc_workspace(cc.cc_keyattn_workspace_size(shape, 2, cap))
    cc.cc_h2o_accumulate(shape, cache, recent, ws)
    assert cc.cc_get_status() == cc.CC_OK
    cn = _np_cache(c)
    acc = oracle.h2o_update(shape, cn, np.zeros((2, cap)), recent)
    got = c["h2o_acc"].cpu().numpy()
    for b, n in enumerate(seq):
        assert rel_err(got[b, :n], acc[b, :n]) < TOL, b
    # refresh scores
    scores = torch.empty(2, cap, device="cuda")
    cc.cc_score_h2o(cache, recent, scores)
    np.testing.assert_array_equal(scores.cpu().numpy(),
                                  oracle.h2o_scores(got.astype(np.float64), seq, recent))
    # compaction carries the totals with the slots (bit-exact given the index list)
    keep = np.full((2, cap), -1, np.int32)
    cnt = np.array([250, 333], np.int32)
    r = np.random.default_rng(63)
    keep[0, :250] = np.sort(np.concatenate([r.choice(599, 249, replace=False), [599]]))
    keep[1, :333] = np.arange(333)
    before = got.copy()
    cws = cc.alloc_workspace(cc.cc_compact_workspace_size(shape, cache))
    cc.cc_compact_kv(shape, cache, torch.from_numpy(keep).cuda(), torch.from_numpy(cnt).cuda(), cws)
    assert cc.cc_get_status() == cc.CC_OK
    np.testing.assert_array_equal(c["h2o_acc"].cpu().numpy(), oracle.compact(before, keep, cnt))
    # a second accumulation on the compacted cache adds to the carried totals
    cc.cc_h2o_accumulate(shape, cache, recent, ws)
    cn2 = _np_cache(c)
    acc2 = oracle.h2o_update(shape, cn2, oracle.compact(before, keep, cnt).astype(np.float64), recent)
    got2 = c["h2o_acc"].cpu().numpy()
    for b, n in enumerate(cnt):
        assert rel_err(got2[b, :n], acc2[b, :n]) < TOL, b


def test_importance_paper_table1_shape(pkg):
    """Qwen2.5-7B last layer (4 KV heads x 128), a 4096-slot synthetic cache."""
    from paper_2607_27600_gb300 import cc
    wl = synth.WORKLOADS["qwen7b-table1-fast-4096"]
    shape = wl.shape
    c = synth.synthetic_cache(shape, wl.seq_lens, wl.cap, wl.seed, device="cuda",
                              layers=[shape.n_layers - 1], with_h_last=False)
    cache = pkg.Cache(c)
    ws = cc.alloc_workspace(cc.cc_keyattn_workspace_size(shape, 1, wl.cap))
    scores = torch.empty(1, wl.cap, device="cuda")
    cc.cc_score_importance(shape, cache, scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
    cn = {"k": [None] * (shape.n_layers - 1) + [c["k"][-1].float().cpu().numpy()],
          "seq_len": c["seq_len"].cpu().numpy()}
    want = oracle.importance_scores(shape, cn)
    assert rel_err(scores.cpu().numpy()[0], want[0]) < TOL
