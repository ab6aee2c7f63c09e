"""The GEMMs run as CTA pairs (clusters of two, one 256 x 256 tcgen05 product
per pair) for launches of two waves of tiles or more; smaller launches stay
on single CTAs.  This module runs the pair path everywhere a tile is 256
columns wide (CC_GEMM_PAIRS=2), so that the small seeded workloads the
oracle checks row by row reach it too: odd row-tile counts (the second CTA
of the last pair stores nothing), pairs whose two row tiles belong to
different sequences, ragged column counts and every epilogue of the refresh
(Sec. 3.1) in bf16 and fp16 operands, of the append and of the fused q/k/v
projections.  The
full-size parity tests run the default choice, which pairs the large
launches."""
import os

import numpy as np
import pytest
import torch

import synth
import tests.test_gpu_append as append_tests
import tests.test_gpu_f16 as f16_tests
import tests.test_gpu_fp8 as fp8_tests
import tests.test_gpu_kernels as kernel_tests
import tests.test_gpu_paged as paged_tests
import tests.test_gpu_score as score_tests

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def pairs_everywhere(monkeypatch):
    monkeypatch.setenv("CC_GEMM_PAIRS", "2")


# the modules' fixtures (the same library handle in each)
cc = kernel_tests.cc
pkg = score_tests.pkg
tiny = score_tests.tiny

# the oracle parity tests, rerun with every 256-wide GEMM on CTA pairs
test_linear_matches_fp64 = kernel_tests.test_linear_matches_fp64
test_tiny_single_layer_all_rows = score_tests.test_tiny_single_layer_all_rows
test_small_two_layer_full_and_fast_ragged = score_tests.test_small_two_layer_full_and_fast_ragged
test_tiny_precise_mode_all_rows = score_tests.test_tiny_precise_mode_all_rows
test_tiny_refresh_keep_set_and_compaction = score_tests.test_tiny_refresh_keep_set_and_compaction
test_model_variants_bias_and_rope_scaling = score_tests.test_model_variants_bias_and_rope_scaling
test_append_into_empty_cache_ragged = append_tests.test_append_into_empty_cache_ragged
test_append_after_compaction_then_score = append_tests.test_append_after_compaction_then_score
test_append_llama_shape_chunk_over_long_memory = (
    append_tests.test_append_llama_shape_chunk_over_long_memory)
test_fp8_append_llama_fused_projection = fp8_tests.test_fp8_append_llama_fused_projection
test_fp8_scores_small_ragged = fp8_tests.test_fp8_scores_small_ragged
test_fp8_precise_mode_small_ragged = fp8_tests.test_fp8_precise_mode_small_ragged
test_paged_append_matches_slot_major = paged_tests.test_paged_append_matches_slot_major
test_tiny_f16_mode_all_rows = f16_tests.test_tiny_f16_mode_all_rows
test_small_two_layer_f16_ragged = f16_tests.test_small_two_layer_f16_ragged


def _linear(cc, x, w):
    y = torch.empty(x.shape[0], w.shape[0], dtype=torch.float32, device="cuda")
    cc.cc_linear_f32(x, w, y)
    torch.cuda.synchronize()
    assert cc.cc_get_status() == cc.CC_OK
    return y


# row tiles: 41 (odd: the last pair's second CTA idles), 71 with a ragged
# 40-row tail; columns: 2080 = 8 tiles + 32 (the second CTA's B half of the
# last tile lies wholly past the weight rows)
@pytest.mark.parametrize("rows,n,k", [(5248, 2048, 1024), (9000, 2080, 576), (300, 96, 200)])
def test_pairs_match_single_ctas_and_fp64(cc, monkeypatch, rows, n, k):
    x = synth.normal((rows, k), 1.0, 2, f"px{rows}.{n}.{k}").cuda()
    w = synth.normal((n, k), 0.05, 2, f"pw{rows}.{n}.{k}").cuda()
    y_pair = _linear(cc, x, w)
    monkeypatch.setenv("CC_GEMM_PAIRS", "0")
    y_one = _linear(cc, x, w)
    monkeypatch.delenv("CC_GEMM_PAIRS")
    y_auto = _linear(cc, x, w)
    want = x.double().cpu() @ w.double().cpu().T
    scale = want.abs().max().item()
    for y in (y_pair, y_one, y_auto):
        err = (y.cpu().double() - want).abs().max().item()
        assert err <= 1e-4 * scale + 1e-5, (err, scale)
    # the pair's product accumulates every output in the single CTA's order
    assert torch.equal(y_pair, y_one)
    assert torch.equal(y_auto, y_one)
