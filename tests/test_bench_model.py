"""The algorithmic work behind bench.py's roofline fractions, counted by
brute force on small workloads (no GPU): attention FLOPs over the explicit
counter-causal (i, j > i) pairs, GEMM FLOPs from the operand shapes, the
compaction's bytes from the moved rows."""
import dataclasses

import pytest

import bench
import synth
from synth.configs import Workload


def _tiny(mode, seq_lens, budgets, n_layers=2):
    shape = dataclasses.replace(synth.configs.TINY, n_layers=n_layers)
    return Workload(name="t", shape=shape, mode=mode, seq_lens=seq_lens, budgets=budgets,
                    cap=max(seq_lens), seed=0, cache_from_causal_pass=False)


@pytest.mark.parametrize("mode", ["layer", "full"])
def test_flops_and_bytes_by_brute_force(mode):
    wl = _tiny(mode, [37, 5, 1], [10, 9, 1])
    s = wl.shape
    work = bench.algorithmic_work(wl)
    rows = sum(wl.seq_lens)
    # attention: per query head, QK^T and PV each cost 2 * dh per (i, j > i) pair
    pairs = sum(1 for n in wl.seq_lens for i in range(n) for j in range(i + 1, n))
    assert work["attention"] == ("tensor", 2 * 2 * s.head_dim * s.n_q_heads * pairs)
    d, qd, f = s.d_model, s.n_q_heads * s.head_dim, s.d_ff
    assert work["gemm_qrope"][1] == 2 * rows * d * qd
    assert work["gemm_oproj"][1] == 2 * rows * qd * d
    assert work["gemm_gateup"][1] == 2 * rows * d * (2 * f)   # gate and up
    assert work["gemm_down"][1] == 2 * rows * f * d
    # compaction: every kept slot's rows read once and written once (the
    # kept slot count per sequence is min(budget, n))
    kept = sum(min(b, n) for b, n in zip(wl.budgets, wl.seq_lens))
    row_bytes = 2 * s.n_layers * s.n_kv_heads * s.head_dim * 2   # K and V of every layer
    row_bytes += 2 * d if mode == "layer" else 0                 # H^(L-1)
    row_bytes += 4 + 4                                           # token, position
    assert work["compact"] == ("hbm", 2 * kept * row_bytes)
    # the pre-attention norm: the input row read (bf16 or fp32), a bf16 row written
    in_bytes = 2 if mode == "layer" else 4
    assert work["rmsnorm"] == ("hbm", rows * (in_bytes * d + 2 * d))


def test_step_flops_counts_every_layer_of_the_full_pass():
    layer, full = _tiny("layer", [64], [16], 3), _tiny("full", [64], [16], 3)
    per_layer = sum(bench.algorithmic_work(layer)[k][1] for k in
                    ("gemm_qrope", "attention", "gemm_oproj", "gemm_gateup", "gemm_down"))
    head = 2 * 64 * layer.shape.d_model
    assert bench.step_flops(layer) == per_layer + head
    assert bench.step_flops(full) == 3 * per_layer + head


def test_fp8_cache_halves_the_kv_bytes_of_the_compaction():
    wl = _tiny("full", [100], [40])
    b16, b8 = bench.algorithmic_work(wl, 2)["compact"][1], bench.algorithmic_work(wl, 1)["compact"][1]
    kv = 2 * 40 * 2 * wl.shape.n_layers * wl.shape.n_kv_heads * wl.shape.head_dim
    assert b16 - b8 == kv


def test_tensor_peak_is_sustained_for_long_timed_regions():
    peaks = {"bf16_tflops": 1916.0, "bf16_tflops_sustained": 1732.6, "hbm_gbs": 6682.5}
    assert bench.tensor_peak(peaks, 0.5) == (1916.0, "bf16 dense burst")
    assert bench.tensor_peak(peaks, 6.0) == (1732.6, "bf16 dense sustained")
    assert bench.tensor_peak({"bf16_tflops": 1900.0}, 6.0)[0] == 1900.0   # no sustained figure
    # a 1 ms launch of 1.5 TFLOP: 1500 TFLOP/s against either peak
    table = bench.kernel_table({"gemm_gateup": (2, 2.0)}, 2, {"gemm_gateup": ("tensor", 1.5e12)},
                               peaks, timed_s=6.0)
    e = table["gemm_gateup"]
    assert e["achieved"] == 1500.0
    assert e["frac"] == round(1500.0 / 1732.6, 4) and e["frac_of_burst"] == round(1500.0 / 1916.0, 4)


def test_oracle_leg_samples_and_extrapolation():
    """The oracle leg on the tiny workload (CPU tensors): the row sample is
    uniform over all positions and inside every sequence, the layer sample of a
    full pass truncates the model, and the extrapolated refresh time grows
    linearly from the sampled rows to every row (per-call fixed cost once)."""
    import numpy as np
    wl = _tiny("full", [300, 129, 64], [75, 40, 16], n_layers=4)
    w = synth.model_weights(wl.shape, 3)
    cache = synth.synthetic_cache(wl.shape, wl.seq_lens, wl.cap, 3, with_h_last=False)
    leg = bench.OracleLeg(wl, w, cache, "logit")
    assert leg.shape.n_layers == 2 and leg.layers == [0, 1]
    rows = leg.sample(leg.rows_large, seed=4)
    assert sum(len(r) for r in rows) == leg.rows_large
    for r, n in zip(rows, wl.seq_lens):
        assert all(0 <= i < n for i in r) and r == sorted(set(r))
    scores = np.random.default_rng(0).standard_normal((wl.batch, wl.cap)).astype(np.float32)
    leg.fixed = 0.5          # a known fixed cost: the extrapolation is then checkable
    measured, total, d = leg.step(scores, seed=5)
    per_row = max(0.0, d["t_rows"] - 0.5) / d["rows"]
    want = (wl.shape.n_layers / 2) * (0.5 + per_row * sum(wl.seq_lens)) + d["t_sel"] + d["t_compact"]
    assert abs(total - want) <= 1e-9 * want
    assert measured > 0
    base = leg.cpu_baseline(scores)
    assert base["kind"] == "oracle" and base["extrapolated"] and base["value"] > 0


def test_e2e_row_blocks_cover_every_slot_once_on_key_tile_boundaries():
    """The fast pass's end-to-end blocks: every slot [0, n) of a sequence in
    exactly one block, none past n, every interior start a multiple of 128
    (a block's attention then reads no key tile below its own start)."""
    seq = [32768, 8192, 300, 129, 64, 1, 0]
    for nb in (1, 2, 8, 16):
        bounds = bench.block_bounds(seq, nb)
        assert len(bounds) == nb + 1
        assert bounds[0] == [0] * len(seq) and bounds[-1] == seq
        for k in range(nb):
            for b, n in enumerate(seq):
                lo, hi = bounds[k][b], bounds[k + 1][b]
                assert 0 <= lo <= hi <= n
                assert lo % 128 == 0 or lo == n


def test_kernel_digest_ignores_comments_not_code():
    """The DRAM-traffic record stays valid through comment and layout edits
    of a kernel's sources and goes stale on any code edit."""
    import bench
    src = {"gemm.cu": "int a = 1; // one\n/* block\n comment */ int b = a  +  2;\n",
           "gemm.cuh": "", "cc_common.cuh": "", "api.cu": ""}
    base = bench.kernel_digest("gemm_gateup", read=lambda f: src[f])
    src["gemm.cu"] = "int a = 1;   // the first\nint b = a + 2; /* sum */\n"
    assert bench.kernel_digest("gemm_gateup", read=lambda f: src[f]) == base
    src["gemm.cu"] = "int a = 1;\nint b = a + 3;\n"
    assert bench.kernel_digest("gemm_gateup", read=lambda f: src[f]) != base
