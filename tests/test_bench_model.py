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
