"""Pins of the oracle's 8-bit cache format (Sec. 3.1: the storage model is per
cache format; an 8-bit format changes execution, so attention reads the
dequantised rows). The encoding is E4M3 (1 sign, 4 exponent bits with bias 7,
3 mantissa bits, no infinities, S.1111.111 = NaN, largest finite 448) with one
fp32 scale per stored row, the smallest power of two at or above amax / 448 (the
shared power-of-two scale of the OCP microscaling formats, taken per row). Every pin follows from that definition, not from the
oracle's own code: values fixed by the format, round trips, ties to even at every
midpoint, saturation, the rounding error bound, and a lossless case that must
reproduce the bf16 attention oracle exactly."""
import math

import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.filterwarnings("ignore")


def f32(x):
    return float(np.float32(x))


def bf16_bits(x):
    """Exactly representable float -> bf16 bits (truncation is exact for these)."""
    return (np.asarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


@pytest.mark.parametrize("code,value", [
    (0x00, 0.0), (0x01, 2.0 ** -9), (0x07, 7 * 2.0 ** -9), (0x08, 2.0 ** -6),
    (0x38, 1.0), (0x39, 1.125), (0x3F, 1.875), (0x40, 2.0), (0x7E, 448.0),
    (0x80, -0.0), (0xB8, -1.0), (0xC0, -2.0), (0xFE, -448.0),
])
def test_values_fixed_by_the_format(code, value):
    v = oracle.e4m3_decode(code)
    assert v == value and math.copysign(1.0, v) == math.copysign(1.0, value)


def test_nan_codes():
    assert math.isnan(oracle.e4m3_decode(0x7F)) and math.isnan(oracle.e4m3_decode(0xFF))
    assert oracle.e4m3_encode(float("nan")) == 0x7F


def test_round_trip_and_order():
    finite = [c for c in range(256) if c not in (0x7F, 0xFF)]
    for c in finite:
        assert oracle.e4m3_encode(oracle.e4m3_decode(c)) == c
    mags = [oracle.e4m3_decode(c) for c in range(0x7F)]
    assert all(a < b for a, b in zip(mags, mags[1:]))  # increasing with the code


def test_ties_to_even_and_nearest():
    for c in range(0x7E):
        lo, hi = oracle.e4m3_decode(c), oracle.e4m3_decode(c + 1)
        mid = (lo + hi) / 2  # 5 significant bits: exact in float32
        assert f32(mid) == mid
        even = c if c % 2 == 0 else c + 1
        assert oracle.e4m3_encode(mid) == even
        assert oracle.e4m3_encode(-mid) == 0x80 | even
        below = float(np.nextafter(np.float32(mid), np.float32(0)))
        above = float(np.nextafter(np.float32(mid), np.float32(1e9)))
        assert oracle.e4m3_encode(below) == c
        assert oracle.e4m3_encode(above) == c + 1


def test_saturation():
    for x in (448.0, 448.5, 464.0, 1e6, 3e38, float("inf")):
        assert oracle.e4m3_encode(x) == 0x7E
        assert oracle.e4m3_encode(-x) == 0xFE
    assert oracle.e4m3_encode(2.0 ** -11) == 0x00  # below half the smallest subnormal
    assert oracle.e4m3_encode(-(2.0 ** -11)) == 0x80


def test_row_quantization_bound_and_scale():
    rng = np.random.default_rng(5)
    for d in (64, 128, 256):
        for scale in (1e-3, 1.0, 37.0):
            x = (rng.standard_normal(d) * scale).astype(np.float32)
            bits = bf16_bits(x)
            xs = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            codes, s = oracle.quantize_row_e4m3(bits)
            amax = np.float32(np.abs(xs).max())
            r = float(np.float32(amax / np.float32(448.0)))  # amax / 448 in float arithmetic
            assert float(s) == 2.0 ** math.ceil(math.log2(r))  # smallest power of two >= r
            assert math.frexp(float(s))[0] == 0.5 and r <= float(s) < 2 * r
            deq = np.array([oracle.e4m3_decode(c) for c in codes]) * float(s)
            i = int(np.argmax(np.abs(xs)))
            assert 0x76 <= codes[i] & 0x7F <= 0x7E  # |x| / s in [224, 448]: the top binade
            if scale >= 1.0:  # a 4-bit code times a power of two: exact in fp16 here
                assert np.array_equal(deq.astype(np.float16).astype(np.float64), deq)
            # half a step: 2^-4 relative for normal codes, 2^-10 s for subnormal ones
            bound = np.maximum(np.abs(xs) * 2.0 ** -4, 2.0 ** -10 * float(s)) * (1 + 2.0 ** -18)
            assert np.all(np.abs(deq - xs) <= bound)
            neg, s2 = oracle.quantize_row_e4m3(bf16_bits(-x))
            assert s2 == s and np.array_equal(neg, codes ^ 0x80)
    codes, s = oracle.quantize_row_e4m3(np.zeros(128, dtype=np.uint16))
    assert s == 0.0 and not codes.any()


def test_lossless_rows_reproduce_bf16_attention():
    # rows whose elements lie on the E4M3 grid times 2^k, with the largest at 448 2^k:
    # the scale is exactly 2^k and quantisation loses nothing, so attention over the
    # 8-bit cache must equal the bf16 oracle's on the same values
    rng = np.random.default_rng(11)
    grid = np.array([oracle.e4m3_decode(c) for c in range(0x7F)])
    T, d, W = 97, 128, 40
    def rows(k):
        v = rng.choice(grid, size=(T, d)) * rng.choice([-1.0, 1.0], size=(T, d))
        v[:, 0] = 448.0
        return (v * 2.0 ** k).astype(np.float32)
    K, V = rows(-9), rows(-6)
    Q = (rng.standard_normal((5, d)) * 0.5).astype(np.float32)
    Qb, Kb, Vb = bf16_bits(Q), bf16_bits(K), bf16_bits(V)
    assert np.array_equal((Kb.astype(np.uint32) << 16).view(np.float32), K)
    Kc, Ks = oracle.quantize_rows_e4m3(Kb)
    Vc, Vs = oracle.quantize_rows_e4m3(Vb)
    assert np.all(Ks == np.float32(2.0 ** -9)) and np.all(Vs == np.float32(2.0 ** -6))
    assert np.array_equal(oracle.dequantize_rows_e4m3(Kc, Ks), K.astype(np.float64))
    pos = [0, 10, 39, 40, 96]
    O8, sp8 = oracle.window_attention_fp8(Qb, pos, Kc, Ks, Vc, Vs, W, 0.125)
    O16, sp16 = oracle.window_attention_bf16(Qb, pos, Kb, Vb, W, 0.125)
    np.testing.assert_allclose(O8, O16, rtol=0, atol=1e-12)
    np.testing.assert_allclose(sp8, 1.0, atol=1e-12)
