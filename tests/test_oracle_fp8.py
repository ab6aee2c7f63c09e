"""Pins of the oracle's E4M3 codec (the e4m3 K/V cache variant) and of its
use in the inference cycle's append."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth.configs import ModelShape
from tests._util import to_np


def test_named_values_of_the_format():
    """Values the E4M3 definition names: 1.0 = 0 0111 000, 2.0 = 0 1000 000,
    the largest finite 448 = 0 1111 110, the smallest normal 2^-6 = 0 0001 000,
    the smallest subnormal 2^-9 = 0 0000 001, NaN = S 1111 111, -0."""
    d = oracle.e4m3_decode(np.array([0x38, 0x40, 0xB8, 0x7E, 0x08, 0x01, 0x00, 0x06], np.uint8))
    np.testing.assert_array_equal(d, [1.0, 2.0, -1.0, 448.0, 2.0 ** -6, 2.0 ** -9, 0.0, 0.75 * 2.0 ** -6])
    assert np.isnan(oracle.e4m3_decode(np.array([0x7F, 0xFF], np.uint8))).all()
    neg0 = oracle.e4m3_decode(np.array([0x80], np.uint8))[0]
    assert neg0 == 0.0 and np.signbit(neg0)


def test_round_trip_and_order():
    codes = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], np.uint8)
    np.testing.assert_array_equal(oracle.e4m3_encode(oracle.e4m3_decode(codes)), codes)
    pos = oracle.e4m3_decode(np.arange(0x7F, dtype=np.uint8))
    assert (np.diff(pos) > 0).all()          # strictly increasing magnitudes 0 .. 448
    assert len(pos) == 127


def test_ties_to_even_and_nearest():
    pos = oracle.e4m3_decode(np.arange(0x7F, dtype=np.uint8))
    mid = (pos[:-1] + pos[1:]) / 2
    got = oracle.e4m3_encode(mid).astype(int)
    lo = np.arange(126)
    want = np.where(lo % 2 == 0, lo, lo + 1)   # the even code of each pair
    np.testing.assert_array_equal(got, want)
    eps = (pos[1:] - pos[:-1]) * 1e-3
    np.testing.assert_array_equal(oracle.e4m3_encode(mid - eps), lo)
    np.testing.assert_array_equal(oracle.e4m3_encode(mid + eps), lo + 1)


def test_saturation_and_nan():
    big = np.array([448.0, 448.5, 464.0, 480.0, 1e30, np.inf])
    np.testing.assert_array_equal(oracle.e4m3_encode(big), np.full(6, 0x7E))
    np.testing.assert_array_equal(oracle.e4m3_encode(-big), np.full(6, 0xFE))
    assert oracle.e4m3_encode(np.array([np.nan]))[0] & 0x7F == 0x7F


def test_matches_torch_float8_cast_in_range():
    """torch.float8_e4m3fn (a library routine) rounds to nearest even; inside
    the finite range (|x| <= 448; beyond it the cast gives NaN rather than
    saturating) the two encoders agree on every value."""
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("torch without float8")
    r = np.random.default_rng(0)
    x = np.concatenate([r.normal(0, 1, 20000), r.normal(0, 100, 20000),
                        r.uniform(-448, 448, 20000), r.normal(0, 2.0 ** -8, 20000)])
    x = x[np.abs(x.astype(np.float32)) <= 448.0]
    want = torch.from_numpy(x.astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    got = oracle.e4m3_encode(x.astype(np.float32).astype(np.float64))
    np.testing.assert_array_equal(got, want)


def test_append_quantises_the_new_rows():
    """One-layer model: the chunk's K/V projections do not depend on the
    attention, so the e4m3 append stores exactly kv_quantize of the
    unquantised append's rows, leaves the memory rows alone, and its output
    moves by the quantisation only (nonzero, bounded)."""
    shape = ModelShape(n_layers=1, d_model=64, n_q_heads=4, n_kv_heads=2, head_dim=16,
                       d_ff=96, vocab=100, rope_theta=1e4, rms_eps=1e-5)
    w = to_np(synth.model_weights(shape, 3, with_kv_proj=True))
    cap, n0 = 40, 12
    r = np.random.default_rng(3)

    def cache():
        return {"k": [np.zeros((1, cap, 2, 16))],
                "v": [np.zeros((1, cap, 2, 16))], "tokens": np.zeros((1, cap), np.int64),
                "pos": np.tile(np.arange(cap), (1, 1)), "seq_len": np.array([0]),
                "h_last": None}

    plain, quant = cache(), cache()
    toks = r.integers(0, 100, n0 + 9)
    oracle.append_chunk(shape, w, plain, 0, toks[:n0])
    oracle.append_chunk(shape, w, quant, 0, toks[:n0])
    scales = [(0.01, 0.004)]
    quant["kv_scale"] = scales
    plain_k = plain["k"][0].copy()
    x_plain = oracle.append_chunk(shape, w, plain, 0, toks[n0:])
    x_quant = oracle.append_chunk(shape, w, quant, 0, toks[n0:])
    sl = slice(n0, n0 + 9)
    np.testing.assert_array_equal(quant["k"][0][0, sl], oracle.kv_quantize(plain["k"][0][0, sl], 0.01))
    np.testing.assert_array_equal(quant["v"][0][0, sl], oracle.kv_quantize(plain["v"][0][0, sl], 0.004))
    np.testing.assert_array_equal(quant["k"][0][0, :n0], plain_k[0, :n0])   # memory untouched
    assert 0 < np.abs(x_quant - x_plain).max() < 0.5 * np.abs(x_plain).max()
