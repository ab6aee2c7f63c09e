"""FP8 E4M3 codec of the oracle -- TEST INFRASTRUCTURE (see oracle/__init__.py).

The e4m3 K/V cache variant stores each cached key/value element as one byte:
the OCP 8-bit floating-point E4M3 format (sign bit, 4 exponent bits with
bias 7, 3 mantissa bits; no infinities; exponent 1111 with mantissa 111 is
NaN, so the largest finite magnitude is 1.75 * 2^8 = 448; exponent 0000 holds
the subnormals m/8 * 2^-6).  A cached element is code * scale, one scale per
layer for K and one for V.  The paper uses the model's own (fp16) cache; this
codec only serves the variant.

Written from that definition: the decode table is computed field by field,
the encoder rounds to the nearest table value with ties to the even code
(mantissa LSB 0) and saturates magnitudes above 448 to 448 (NaN stays NaN).
"""
import numpy as np

E4M3_MAX = 448.0


def _magnitudes():
    """Magnitude of every non-negative code 0x00..0x7F (0x7F is NaN)."""
    out = np.empty(128)
    for c in range(128):
        e, m = c >> 3, c & 7
        if e == 15 and m == 7:
            out[c] = np.nan
        elif e == 0:
            out[c] = m / 8.0 * 2.0 ** (1 - 7)
        else:
            out[c] = (1.0 + m / 8.0) * 2.0 ** (e - 7)
    return out


_MAG = _magnitudes()
_FINITE = _MAG[:127]          # codes 0x00..0x7E, ascending


def e4m3_decode(codes):
    """uint8 codes -> float64 values."""
    c = np.asarray(codes).astype(np.int64) & 0xFF
    v = _MAG[c & 0x7F]
    return np.where(c & 0x80, -v, v)


def e4m3_encode(x):
    """float values -> uint8 codes: round to nearest, ties to the even code,
    magnitudes above 448 saturate to 448, NaN -> 0x7F (sign kept)."""
    x = np.asarray(x, dtype=np.float64)
    sign = np.signbit(x).astype(np.int64) << 7
    a = np.abs(x)
    nan = np.isnan(a)
    a = np.where(nan, 0.0, np.minimum(a, E4M3_MAX))
    hi = np.searchsorted(_FINITE, a, side="left")        # first table value >= a
    hi = np.minimum(hi, 126)
    lo = np.maximum(hi - 1, 0)
    d_hi = _FINITE[hi] - a
    d_lo = a - _FINITE[lo]
    pick_hi = (d_hi < d_lo) | ((d_hi == d_lo) & (hi % 2 == 0))
    code = np.where(_FINITE[hi] == a, hi, np.where(pick_hi, hi, lo))
    code = np.where(nan, 0x7F, code)
    return (code | sign).astype(np.uint8)


def kv_quantize(x, scale):
    """A value as the e4m3 cache holds it: decode(encode(x / scale)) * scale."""
    return e4m3_decode(e4m3_encode(np.asarray(x, np.float64) / scale)) * scale
