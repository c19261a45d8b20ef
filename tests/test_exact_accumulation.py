"""CPU pins of the arithmetic the tensor-core GEMM rests on (Sec. 4.2, Eq. 7, carried through the
FP8 tensor pipe).

The integer product acc[m, n] = sum_k Q_X'[m, k] Q_W'[n, k] of Eq. 7 runs on tcgen05's E4M3 kind
with FP32 accumulation.  Code q in [-8, 7] travels as the byte q + 8, which as an E4M3 number is
worth (q + 8) 2^-9 exactly; every product is then an integer multiple of 2^-18, and every partial
sum over K <= 16384 channels an integer multiple of 2^-18 below 2^24 of them, so FP32 holds it
exactly whatever the order of the additions.  The same holds for the split of K into work units:
each unit's partial and the sum of the partials are such multiples.  These tests check the E4M3
decoding from the format's definition and the exactness of FP32 sums in several orders and
splits, against int64 arithmetic."""

import numpy as np
import pytest


def e4m3_value(byte: int) -> float:
    """The OCP E4M3 number a byte encodes: sign bit, 4 exponent bits (bias 7), 3 mantissa bits;
    exponent 0 is subnormal (no implicit one).  (The one NaN pattern, S.1111.111, is not needed.)"""
    sign = -1.0 if byte & 0x80 else 1.0
    e = (byte >> 3) & 0xF
    m = byte & 0x7
    if e == 0:
        return sign * (m / 8.0) * 2.0 ** (1 - 7)
    return sign * (1.0 + m / 8.0) * 2.0 ** (e - 7)


def test_offset_code_bytes_are_exact_multiples():
    for q in range(-8, 8):
        assert e4m3_value(q + 8) == (q + 8) * 2.0 ** -9
        assert (q + 8) == (q ^ 8) & 0xF  # the byte is q XOR 8 in 4 bits
    # bytes 0..7 are subnormal, 8..15 the first normal binade: one uniform step of 2^-9
    steps = {e4m3_value(b + 1) - e4m3_value(b) for b in range(15)}
    assert steps == {2.0 ** -9}


def _products(rng, K, kind):
    if kind == "max":
        a = np.full(K, 15, np.int64)
        b = np.full(K, 15, np.int64)
    elif kind == "min":
        a = np.zeros(K, np.int64)
        b = np.zeros(K, np.int64)
    else:
        a = rng.integers(0, 16, K)
        b = rng.integers(0, 16, K)
    return a * b  # integers; the float values are these times 2^-18


def _fp32_sum(x32):
    """Sequential float32 sum, one rounding per addition."""
    return np.cumsum(x32, dtype=np.float32)[-1] if x32.size else np.float32(0)


@pytest.mark.parametrize("K", [128, 2048, 16384])
@pytest.mark.parametrize("kind", ["max", "min", "random"])
def test_fp32_sums_of_code_products_are_exact_in_any_order(K, kind):
    rng = np.random.default_rng(K)
    p = _products(rng, K, kind)
    exact = int(p.sum())
    assert exact < 2 ** 24
    scale = np.float32(2.0 ** -18)
    x = p.astype(np.float32) * scale  # exact: integers below 2^8 times a power of two
    want = np.float64(exact) * 2.0 ** -18
    orders = [np.arange(K), np.arange(K)[::-1], rng.permutation(K)]
    for order in orders:
        assert np.float64(_fp32_sum(x[order])) == want
    # blocked like the MMA: 32-channel slices summed, then accumulated
    blocks = np.array([_fp32_sum(x[i:i + 32]) for i in range(0, K, 32)], np.float32)
    assert np.float64(_fp32_sum(blocks)) == want


@pytest.mark.parametrize("parts", [2, 3, 4])
def test_split_partials_add_exactly(parts):
    """The split of K: each unit's FP32 partial over its k-range, then the tile's last unit adds
    the others to its own, in whichever order the units finish."""
    K = 16384
    rng = np.random.default_rng(parts)
    for kind in ("max", "random"):
        p = _products(rng, K, kind)
        x = p.astype(np.float32) * np.float32(2.0 ** -18)
        cuts = [K * i // parts for i in range(parts + 1)]
        partials = [_fp32_sum(x[cuts[i]:cuts[i + 1]]) for i in range(parts)]
        want = np.float64(int(p.sum())) * 2.0 ** -18
        for last in range(parts):
            acc = partials[last]
            for i in range(parts):
                if i != last:
                    acc = np.float32(acc + partials[i])
            assert np.float64(acc) == want
        # and the epilogue's scaling back to the integer sum is exact too
        assert np.float64(np.float32(acc) * np.float32(2.0 ** 18)) == int(p.sum())


def test_a_wider_sum_would_not_be_exact():
    """The bound matters: past 2^24 multiples of the step, FP32 drops a unit (the check has teeth)."""
    x = np.array([2 ** 24, 1], np.float32)
    assert np.float64(_fp32_sum(x)) != 2 ** 24 + 1
