"""GPU parity of the int4 x int4 GEMM and its dequantisation epilogue (Sec. 4.2, Eq. 7).

G2: on the oracle's codes the int32 accumulator is bit-exact for every tile shape, ragged M and
N edges and both orientations (tokens on the MMA's M side for M > 128, weights otherwise),
including the weight-major split of K over clusters of 2, 4 and 8 CTAs.
G3: the E4M3 / FP32 tensor-core path stays exact at the largest sums K = 16384 allows.
G5: outputs within 2e-3 of the tensor's maximum magnitude."""

import numpy as np
import pytest

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _codes(rng, rows, k, lo=-8, hi=7):
    return rng.integers(lo, hi + 1, (rows, k)).astype(np.int8)


def _run(M, N, K, seed, ydt="f16", with_bias=True):
    rng = np.random.default_rng(seed)
    qx = _codes(rng, M, K, -7, 7)
    qw = _codes(rng, N, K)  # the packed format also carries -8
    dx = rng.uniform(0.01, 0.3, M).astype(np.float32)
    dw = rng.uniform(0.001, 0.02, N).astype(np.float32)
    bias = rng.standard_normal(N).astype(np.float32) if with_bias else None
    layer = G.make_layer(O.pack_int4(qw), dw, 1, ydt=ydt, bias=bias)
    y, acc = G.gemm(layer, O.pack_int4(qx), dx, qx.astype(np.int64).sum(1), ydt=ydt)
    layer.close()
    ref_acc = O.int_gemm(qx, qw)
    ref_y = O.dequant_output(ref_acc, dx, dw, bias, ydt)
    return acc, ref_acc, y, ref_y


@pytest.mark.parametrize("M,N,K", [
    (1, 16, 128), (5, 48, 512), (16, 256, 2048), (17, 272, 1024), (50, 1024, 1024), (64, 4096, 1024),
    (100, 512, 4096), (128, 1024, 512), (129, 256, 512), (256, 512, 2048), (300, 272, 1024), (816, 1024, 2048),
    (816, 2048, 16384), (1000, 2048, 128),
    # weight-major split-K: a cluster of 2 with several reduction elements per thread, 5
    # k-blocks over 4 CTAs (uneven slices) with a ragged weight tile, a decode row at K = 16384
    (100, 8192, 1024), (33, 400, 640), (1, 2048, 16384),
    # token-major at larger M: 128- and 256-wide tiles with ragged last token tiles (1100, 1450)
    # beside a ragged weight tile, and several tiles per persistent CTA (640 x 16384)
    (1024, 384, 1024), (1100, 1008, 512), (1450, 2048, 1024), (2048, 4096, 256), (640, 16384, 2048),
    # CTA pairs (256-token tiles over two SMs, 128- and 256-wide): the last tile's second CTA
    # without tokens beside a ragged weight tile (600 x 8432, 260 x 13264), a ragged second CTA
    # (1450), several pair tiles per CTA (640 x 16384 above); the backbone's down projection
    (600, 8432, 1024), (1450, 4352, 1024), (260, 13264, 1024), (816, 2048, 16384),
])
def test_gemm_accumulator_bit_exact(M, N, K):
    acc, ref_acc, y, ref_y = _run(M, N, K, seed=M * 7 + N + K)
    assert np.array_equal(acc, ref_acc)
    G.assert_output_close(y, ref_y)


@pytest.mark.parametrize("ydt", ["f16", "bf16"])
def test_gemm_output_dtypes(ydt):
    acc, ref_acc, y, ref_y = _run(200, 512, 1024, seed=3, ydt=ydt)
    assert np.array_equal(acc, ref_acc)
    G.assert_output_close(y, ref_y, ydt)
    # where the float32 epilogue and the float64 oracle agree after rounding, outputs are equal
    assert np.mean(y == ref_y) > 0.99


def test_gemm_extremes_exact_at_k16384():
    """All +-7 codes at K = 16384: |acc| = 49 K = 802816, the largest sum the quantiser can
    produce, in both orientations; plus +-1 addends after a large prefix, which a truncating
    accumulator would lose."""
    K = 16384
    for M in (40, 200):
        N = 64
        qx = np.full((M, K), 7, np.int8)
        qx[1::2] = -7
        qw = np.full((N, K), 7, np.int8)
        qw[1::3] = -7
        qw[2::3, K // 2:] = np.where(np.arange(K // 2) % 2 == 0, 1, -1)
        qx[2, K // 2:] = 1
        dx = np.full(M, 0.01, np.float32)
        dw = np.full(N, 0.01, np.float32)
        layer = G.make_layer(O.pack_int4(qw), dw, 1)
        y, acc = G.gemm(layer, O.pack_int4(qx), dx, qx.astype(np.int64).sum(1))
        layer.close()
        ref = O.int_gemm(qx, qw)
        assert np.abs(ref).max() == 49 * K
        assert np.array_equal(acc, ref)


def test_gemm_zero_scale_gives_bias():
    rng = np.random.default_rng(4)
    M, N, K = 20, 64, 256
    qx = _codes(rng, M, K, -7, 7)
    qw = _codes(rng, N, K)
    bias = rng.standard_normal(N).astype(np.float32)
    layer = G.make_layer(O.pack_int4(qw), np.ones(N, np.float32), 1, bias=bias)
    y, _ = G.gemm(layer, O.pack_int4(qx), np.zeros(M, np.float32), qx.astype(np.int64).sum(1))
    layer.close()
    assert np.array_equal(y, np.broadcast_to(O.round_to_format(bias.astype(np.float64), "f16"), (M, N)))


@pytest.mark.parametrize("M,H,K", [(512, 128, 256), (600, 256, 512), (1450, 384, 1024), (520, 4096, 1024),
                                   (1450, 4224, 1024)])
def test_gated_gemm_bit_exact(M, H, K):
    """Gated layers (gate and up rows of a hidden unit in one 256-wide tile): [gate | up]
    accumulators bit-exact and h = gelu(gate) * up within the output tolerance, with ragged
    last token tiles (600, 1450) and a ragged tile of hidden units (H = 384); the two larger
    cases run on CTA pairs, the gate rows staged by one CTA and the up rows by the other, with
    the last tile's second CTA without tokens (520) or ragged (1450)."""
    rng = np.random.default_rng(M + H + K)
    qx = _codes(rng, M, K, -7, 7)
    qg, qu = _codes(rng, H, K), _codes(rng, H, K)
    dx = rng.uniform(0.01, 0.3, M).astype(np.float32)
    dg, du = (rng.uniform(0.001, 0.02, H).astype(np.float32) for _ in range(2))
    layer = Q.qvla_layer_create_gated(H, K, 1, Q.F16, Q.BF16, O.pack_int4(qg), dg, O.pack_int4(qu), du)
    y, acc = G.gemm(layer, O.pack_int4(qx), dx, qx.astype(np.int64).sum(1), ydt="bf16")
    layer.close()
    ag, au = O.int_gemm(qx, qg), O.int_gemm(qx, qu)
    assert np.array_equal(acc, np.concatenate([ag, au], axis=1))
    gate = O.dequant_output(ag, dx, dg, None, "bf16")
    up = O.dequant_output(au, dx, du, None, "bf16")
    h = O.gated_glue(gate, up)
    # The kernel rounds gate and up from float32 scale products, the oracle from float64, so
    # either may land one bf16 step away before the product; each such step, the final rounding
    # of h and the output tolerance bound the difference.
    ug, uu = G.ulp(gate, "bf16"), G.ulp(up, "bf16")
    step = np.abs(O.gated_glue(gate + ug, up) - h) + np.abs(O.gated_glue(gate, up + uu) - h)
    bound = 2e-3 * np.abs(h).max() + 2 * G.ulp(h, "bf16") + step
    assert np.all(np.isfinite(y)) and np.all(np.abs(y - O.round_to_format(h, "bf16")) <= bound)
    assert np.mean(y == O.round_to_format(h, "bf16")) > 0.95
