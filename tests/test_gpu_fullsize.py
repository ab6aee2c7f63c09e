"""GPU parity at the full workload sizes, in the launch configuration bench.py
times (one cc_score_* call over the whole cache), checked on sampled rows
against the CPU oracle (rows are independent given the cache, so a sampled
row's score is exactly what the oracle computes for it alone).

Every input comes from the seeded generators (synth) and is copied to the
host for the oracle; no oracle input comes from the CUDA path.  Multi-cycle
refreshes use seeded keep-sets, compacted independently on each side.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests._util import keep_set_ok, rel_err

pytestmark = pytest.mark.gpu

TOL = 2e-2


@pytest.fixture(scope="module")
def pkg():
    import paper_2607_27600_gb300 as p
    p.load_library()
    return p


def f32(t):
    return None if t is None else t.float().cpu().numpy()


class LazyLayers(list):
    """Layer weights converted to numpy only when the oracle reaches them."""

    def __init__(self, layers):
        super().__init__(layers)

    def __getitem__(self, i):
        lw = list.__getitem__(self, i)
        return None if lw is None else {k: f32(v) for k, v in lw.items()}


class LazyTensors(list):
    def __getitem__(self, i):
        return f32(list.__getitem__(self, i))


def host_view(w, c, lazy=False):
    layers = LazyLayers(w["layers"]) if lazy else [
        None if lw is None else {k: f32(v) for k, v in lw.items()} for lw in w["layers"]]
    wn = {"embed": f32(w["embed"]), "final_norm": f32(w["final_norm"]),
          "lm_head": f32(w["lm_head"]), "layers": layers}
    if lazy:
        kk, vv = LazyTensors(c["k"]), LazyTensors(c["v"])
    else:
        kk, vv = [f32(x) for x in c["k"]], [f32(x) for x in c["v"]]
    cn = {"k": kk, "v": vv, "tokens": c["tokens"].cpu().numpy(), "pos": c["pos"].cpu().numpy(),
          "seq_len": c["seq_len"].cpu().numpy(), "h_last": f32(c["h_last"])}
    return wn, cn


def sample(seq_lens, per_seq, seed):
    r = np.random.default_rng(seed)
    out = []
    for n in seq_lens:
        pick = {0, 1, n // 2, n - 3, n - 2, n - 1} | set(r.choice(n, size=per_seq, replace=False).tolist())
        out.append(sorted(x for x in pick if 0 <= x < n))
    return out


def gpu_scores(pkg, shape, w, c, mode, full):
    from paper_2607_27600_gb300 import cc
    b, cap = c["tokens"].shape
    scores = torch.empty(b, cap, dtype=torch.float32, device="cuda")
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode))
    fn = cc.cc_score_full if full else cc.cc_score_layer
    fn(shape, pkg.Weights(w), pkg.Cache(c), mode, scores, ws)
    assert cc.cc_get_status() == cc.CC_OK
    del ws
    return scores.cpu().numpy()


def check_rows(got, want, rows):
    errs = []
    for b, r in enumerate(rows):
        errs.append(rel_err(got[b, r], want[b, r]))
    return max(errs)


def workload_inputs(wl, layers_only_last=True):
    shape = wl.shape
    fast = wl.mode == "layer"
    layers = [shape.n_layers - 1] if fast else None
    w = synth.model_weights(shape, wl.seed, device="cuda", layers=layers, with_embed=not fast)
    c = synth.synthetic_cache(shape, wl.seq_lens, wl.cap, wl.seed, device="cuda",
                              layers=layers, with_h_last=fast)
    return w, c


@pytest.mark.parametrize("name", ["llama8b-layer-8k", "llama8b-layer-32k-ragged"])
def test_fast_pass_full_size_sampled_rows(pkg, name):
    from paper_2607_27600_gb300 import cc
    wl = synth.WORKLOADS[name]
    w, c = workload_inputs(wl)
    got = gpu_scores(pkg, wl.shape, w, c, cc.SCORE_LOGIT, full=False)
    wn, cn = host_view(w, c)
    rows = sample(wl.seq_lens, 24, seed=1)
    want = oracle.score_layer(wl.shape, wn, cn, rows=rows)
    assert check_rows(got, want, rows) < TOL
    for b, n in enumerate(wl.seq_lens):    # every slot is written: -inf past the end
        assert got[b, n - 1] == np.inf and np.all(got[b, n:] == -np.inf)
        assert np.all(np.isfinite(got[b, :n - 1]))


def test_fast_pass_logprob_full_size(pkg):
    from paper_2607_27600_gb300 import cc
    wl = synth.WORKLOADS["llama8b-layer-8k"]
    w, c = workload_inputs(wl)
    got = gpu_scores(pkg, wl.shape, w, c, cc.SCORE_LOGPROB, full=False)
    wn, cn = host_view(w, c)
    rows = sample(wl.seq_lens, 6, seed=2)
    want = oracle.score_layer(wl.shape, wn, cn, mode="logprob", rows=rows)
    assert check_rows(got, want, rows) < TOL


# Two modes of the full pass (Sec. 3.1, all L layers with fresh queries).
#
# CC_SCORE_PRECISE carries every tensor-core operand that is not an exact bf16
# input as a bf16 pair hi + lo: the GEMM activations, the queries entering
# Q K^T and the probabilities entering P V (K, V and the weights are exact
# bf16 inputs).  It is held to the stated bar: max relative error 2e-2 on
# every sampled row.  tests/study_fullpass_precision.py emulates it in fp64
# ("split-all": 3e-5 after the first layer, 6e-5 after eight of 32).
#
# The default mode keeps single bf16 activations, queries and P (what a bf16
# model computes at inference, about half the precise mode's cost).  On this
# deep random model its drift is a property of the arithmetic: the study's
# "bf16-pass" rounding moves the score by up to 8.9 % (max over 96 rows and 32
# layers; per-row quantiles after layer 31: 50 % 1.7 %, 90 % 5.0 %, 99 %
# 6.9 %), so this mode's bars are derived from that spread and labelled as
# such: about 1.7x the emulated maximum at 32 layers, and at 4 layers the
# relative l2 error over the rows within 2e-2 with a worst-row cap.
#
# CC_SCORE_F16 keeps single operands at the default mode's cost but in fp16
# (11 significant bits to bf16's 8; the bf16 weights and K/V convert
# exactly): the study's "fp16-pass" emulation ends at ~1.4 % after 32 layers,
# so this mode is held to the stated bar as well.
DEFAULT_FULL4_ROW_TOL = 8e-2   # default mode, worst single row at 4 layers (measured 3.9-4.1 %)
DEFAULT_FULL32_TOL = 1.5e-1    # default mode, 32 layers
# The 28-layer Qwen2.5 pass at 512 slots: the default mode held to the 32-layer
# Llama bar (the same rounding points; fewer layers and keys).
DEFAULT_FULL28_TOL = DEFAULT_FULL32_TOL


def _full_inputs(n_layers):
    wl = synth.WORKLOADS["llama8b-full-16k"]
    shape = wl.shape.__class__(**{**wl.shape.__dict__, "n_layers": n_layers})
    w = synth.model_weights(shape, wl.seed, device="cuda")
    c = synth.synthetic_cache(shape, wl.seq_lens, wl.cap, wl.seed, device="cuda",
                              with_h_last=False)
    return wl, shape, w, c


def _full_rows(n, count, seed):
    """The edge rows (first, sequence end, the last slot's +inf) and seeded
    others: `count` distinct rows in all."""
    edge = {0, 5, n // 4 + 1, n // 2 - 1, n - 3, n - 2, n - 1}
    r = np.random.default_rng(seed)
    extra = r.choice(np.setdiff1d(np.arange(n), list(edge)), size=count - len(edge), replace=False)
    return [sorted(edge | set(extra.tolist()))]


def test_full_pass_llama_shape_first_4_layers(pkg):
    """The full-pass machinery over four layers of the Llama-3-8B shape on 64
    rows: the precise mode within the stated 2e-2 on every row; the default
    mode within 2e-2 relative l2 over the rows and its worst row within the
    derived cap."""
    from paper_2607_27600_gb300 import cc
    wl, shape, w, c = _full_inputs(4)
    precise = gpu_scores(pkg, shape, w, c, cc.SCORE_LOGIT | cc.SCORE_PRECISE, full=True)
    default = gpu_scores(pkg, shape, w, c, cc.SCORE_LOGIT, full=True)
    f16 = gpu_scores(pkg, shape, cc.f16_weights(w), c, cc.SCORE_LOGIT | cc.SCORE_F16, full=True)
    wn, cn = host_view(w, c, lazy=True)
    rows = _full_rows(wl.seq_lens[0], 64, seed=5)
    want = oracle.score_full(shape, wn, cn, rows=rows)
    print(f"4 layers, 64 rows: precise max {check_rows(precise, want, rows):.2e}, "
          f"fp16 max {check_rows(f16, want, rows):.2e}, "
          f"default max {check_rows(default, want, rows):.2e}")
    assert check_rows(precise, want, rows) < TOL
    assert check_rows(f16, want, rows) < TOL
    g, o = default[0, rows[0]].astype(np.float64), want[0, rows[0]]
    fin = np.isfinite(o)
    np.testing.assert_array_equal(g[~fin], o[~fin])
    assert np.linalg.norm(g[fin] - o[fin]) / np.linalg.norm(o[fin]) < TOL
    assert check_rows(default, want, rows) < DEFAULT_FULL4_ROW_TOL


def test_full_pass_32_layers_sampled_rows(pkg):
    """llama8b-full-16k, all 32 layers, 64 rows: the precise and fp16 modes
    within the stated 2e-2 max relative error; the default mode within its
    derived bar."""
    from paper_2607_27600_gb300 import cc
    wl, shape, w, c = _full_inputs(32)
    precise = gpu_scores(pkg, shape, w, c, cc.SCORE_LOGIT | cc.SCORE_PRECISE, full=True)
    default = gpu_scores(pkg, shape, w, c, cc.SCORE_LOGIT, full=True)
    f16 = gpu_scores(pkg, shape, cc.f16_weights(w), c, cc.SCORE_LOGIT | cc.SCORE_F16, full=True)
    torch.cuda.empty_cache()
    wn, cn = host_view(w, c, lazy=True)
    rows = _full_rows(wl.seq_lens[0], 64, seed=7)
    want = oracle.score_full(shape, wn, cn, rows=rows)
    print(f"32 layers, 64 rows: precise max {check_rows(precise, want, rows):.2e}, "
          f"fp16 max {check_rows(f16, want, rows):.2e}, "
          f"default max {check_rows(default, want, rows):.2e}")
    assert check_rows(precise, want, rows) < TOL
    assert check_rows(f16, want, rows) < TOL
    assert check_rows(default, want, rows) < DEFAULT_FULL32_TOL


def _gpu_keep(pkg, wl, w, c, mode):
    """GPU scores of the whole batch in `mode` and the GPU keep-set on them,
    which must equal the oracle's select on the same fp32 scores exactly."""
    from paper_2607_27600_gb300 import cc
    if mode & cc.SCORE_F16:
        w = cc.f16_weights(w)
    got = gpu_scores(pkg, wl.shape, w, c, mode, full=False)
    b, cap = c["tokens"].shape
    idx = torch.empty(b, cap, dtype=torch.int32, device="cuda")
    cnt = torch.empty(b, dtype=torch.int32, device="cuda")
    cc.cc_select_keep(torch.from_numpy(got).cuda(), c["seq_len"], b, cap,
                      torch.tensor(wl.budgets, dtype=torch.int32, device="cuda"), 0, idx, cnt)
    assert cc.cc_get_status() == cc.CC_OK
    gi, gc = idx.cpu().numpy(), cnt.cpu().numpy()
    oi, oc = oracle.select_keep(got, wl.seq_lens, wl.budgets)
    assert np.array_equal(gc, oc)
    for s_ in range(b):
        assert np.array_equal(gi[s_, :oc[s_]], oi[s_, :oc[s_]]), s_
    return got, gi, gc


def test_headline_keep_set_full_oracle(pkg):
    """llama8b-layer-8k end to end, with bf16 and with fp16 operands: every
    row scored by the oracle; the GPU keep-set is identical where the
    oracle's boundary gap exceeds the tolerance, else overlaps >= 99.5 %; the
    GPU select equals the oracle's select on the same fp32 scores exactly."""
    from paper_2607_27600_gb300 import cc
    wl = synth.WORKLOADS["llama8b-layer-8k"]
    w, c = workload_inputs(wl)
    runs = [_gpu_keep(pkg, wl, w, c, m) for m in (cc.SCORE_LOGIT, cc.SCORE_LOGIT | cc.SCORE_F16)]
    wn, cn = host_view(w, c)
    want = oracle.score_layer(wl.shape, wn, cn)
    wi, wc = oracle.select_keep(want.astype(np.float32), wl.seq_lens, wl.budgets)
    for got, gi, gc in runs:
        assert rel_err(got, want) < TOL
        ok, det = keep_set_ok(gi, gc, wi, wc, want, wl.seq_lens, wl.budgets)
        assert ok, det


def test_ragged_batch_keep_set_per_sequence_budget(pkg):
    """llama8b-layer-32k-ragged (Algorithm DoMemRefresh per sequence, budgets
    25 % of each length), with bf16 and with fp16 operands: the whole batch
    scored and selected on the GPU in one call each, as bench.py times it;
    the 8192-slot sequence's keep-set (budget 2048) checked against the
    oracle's scores of every one of its rows: identical where the boundary
    gap exceeds the tolerance, else >= 99.5 % overlap with near-tie swaps
    only; every sequence's keep-set equals the oracle's select on the GPU's
    own scores."""
    from paper_2607_27600_gb300 import cc
    wl = synth.WORKLOADS["llama8b-layer-32k-ragged"]
    w, c = workload_inputs(wl)
    b = c["tokens"].shape[0]
    runs = [_gpu_keep(pkg, wl, w, c, m) for m in (cc.SCORE_LOGIT, cc.SCORE_LOGIT | cc.SCORE_F16)]
    seq = int(np.argmin(wl.seq_lens))               # the 8192-slot sequence
    n = wl.seq_lens[seq]
    wn, cn = host_view(w, c)
    rows = [np.arange(n) if s_ == seq else np.array([], np.int64) for s_ in range(b)]
    want = oracle.score_layer(wl.shape, wn, cn, rows=rows)
    wi, wc = oracle.select_keep(want[seq:seq + 1].astype(np.float32), [n], [wl.budgets[seq]])
    for got, gi, gc in runs:
        assert rel_err(got[seq, :n], want[seq, :n]) < TOL
        ok, det = keep_set_ok(gi[seq:seq + 1], gc[seq:seq + 1], wi, wc, want[seq:seq + 1], [n],
                              [wl.budgets[seq]])
        assert ok, det


def seeded_keep(n, budget, seed):
    """A seeded keep-set of `budget` slots of [0, n), the last slot always in."""
    r = np.random.default_rng(seed)
    k = r.choice(n - 1, size=budget - 1, replace=False)
    return np.sort(np.concatenate([k, [n - 1]])).astype(np.int32)


def test_long_context_refresh_cycles(pkg):
    """Qwen2.5-7B-like last layer at 131072 positions, then refresh cycles of
    +4096 appended slots: cycle 1 scored in full size; between cycles both
    sides compact with the same seeded keep-set (bit-exact check) and append
    the same seeded chunk; each cycle's scores compared on sampled rows."""
    from paper_2607_27600_gb300 import cc
    wl = synth.WORKLOADS["qwen7b-layer-128k"]
    shape = wl.shape
    w, c = workload_inputs(wl)
    wn, cn = host_view(w, c)
    last = shape.n_layers - 1
    for cycle in range(wl.cycles):
        n = int(c["seq_len"][0])
        got = gpu_scores(pkg, shape, w, c, cc.SCORE_LOGIT, full=False)
        rows = sample([n], 8 if cycle == 0 else 24, seed=10 + cycle)
        want = oracle.score_layer(shape, wn, cn, rows=rows)
        assert check_rows(got, want, rows) < TOL, cycle
        if cycle + 1 == wl.cycles:
            break
        keep = seeded_keep(n, wl.budgets[0], seed=100 + cycle)
        idx = np.full((1, wl.cap), -1, np.int32)
        idx[0, :len(keep)] = keep
        cnt = np.array([len(keep)], np.int32)
        cache = pkg.Cache(c)
        cws = cc.alloc_workspace(cc.cc_compact_workspace_size(shape, cache))
        cc.cc_compact_kv(shape, cache, torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda(), cws)
        assert cc.cc_get_status() == cc.CC_OK
        for key in ("tokens", "pos"):
            cn[key] = oracle.compact(cn[key], idx, cnt)
        cn["h_last"] = oracle.compact(cn["h_last"], idx, cnt)
        cn["k"][last] = oracle.compact(cn["k"][last], idx, cnt)
        cn["v"][last] = oracle.compact(cn["v"][last], idx, cnt)
        cn["seq_len"] = cnt.copy()
        np.testing.assert_array_equal(f32(c["k"][last])[0, :len(keep)], cn["k"][last][0, :len(keep)])
        np.testing.assert_array_equal(c["pos"].cpu().numpy()[0, :len(keep)], cn["pos"][0, :len(keep)])
        # inference cycle: append the next chunk on the device, mirror it on the host
        synth.append_chunk(shape, c, wl.append, wl.seed, cycle + 1)
        s0, s1 = len(keep), len(keep) + wl.append
        for key in ("tokens", "pos"):
            cn[key][:, s0:s1] = c[key][:, s0:s1].cpu().numpy()
        cn["h_last"][:, s0:s1] = f32(c["h_last"][:, s0:s1])
        cn["k"][last][:, s0:s1] = f32(c["k"][last][:, s0:s1])
        cn["v"][last][:, s0:s1] = f32(c["v"][last][:, s0:s1])
        cn["seq_len"] = c["seq_len"].cpu().numpy()


@pytest.mark.parametrize("name", ["qwen7b-table1-fast-4096", "qwen7b-table1-full-512"])
def test_paper_table1_workloads(pkg, name):
    """The paper's efficiency benchmark shapes (Qwen2.5-7B, synthetic cache):
    the fast pass at 4096 slots on every row; the full 28-layer pass at 512
    slots on 96 rows, the precise and fp16 modes within the stated 2e-2 and
    the default mode within its derived bar; in the launch configuration
    bench.py times."""
    from paper_2607_27600_gb300 import cc
    wl = synth.WORKLOADS[name]
    fast = wl.mode == "layer"
    w, c = workload_inputs(wl)
    got = gpu_scores(pkg, wl.shape, w, c, cc.SCORE_LOGIT, full=not fast)
    wn, cn = host_view(w, c, lazy=not fast)
    if fast:
        want = oracle.score_layer(wl.shape, wn, cn)
        assert rel_err(got[0, :wl.seq_lens[0]], want[0, :wl.seq_lens[0]]) < TOL
    else:
        precise = gpu_scores(pkg, wl.shape, w, c, cc.SCORE_LOGIT | cc.SCORE_PRECISE, full=True)
        f16 = gpu_scores(pkg, wl.shape, cc.f16_weights(w), c, cc.SCORE_LOGIT | cc.SCORE_F16,
                         full=True)
        rows = _full_rows(wl.seq_lens[0], 96, seed=6)
        want = oracle.score_full(wl.shape, wn, cn, rows=rows)
        print(f"28 layers, 96 rows: precise max {check_rows(precise, want, rows):.2e}, "
              f"fp16 max {check_rows(f16, want, rows):.2e}, "
              f"default max {check_rows(got, want, rows):.2e}")
        assert check_rows(precise, want, rows) < TOL
        assert check_rows(f16, want, rows) < TOL
        assert check_rows(got, want, rows) < DEFAULT_FULL28_TOL
