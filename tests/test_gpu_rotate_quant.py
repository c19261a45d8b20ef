"""GPU parity of the fused rotation + int4 activation quantisation (Sec. 4.1 Eq. 3-5 online
factor; Sec. 4.2 Eq. 5-6) against the oracle.

G1: fed the oracle's rotated float32 activations (no rotation on the GPU), codes, scales and
code sums are bit-exact.  End to end from raw fp16/bf16/fp32 activations, at most 1e-5 of the
codes differ, each by +-1 and only next to a rounding tie."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _x(m, k, seed, dtype="f16", outliers=4):
    rng = np.random.default_rng(seed)
    return W.as_dtype(W.gaussian_with_outliers(rng, m, k, outliers, 20.0), dtype)


@pytest.mark.parametrize("M,K,had", [(1, 128, 128), (37, 512, 512), (64, 2048, 2048), (9, 16384, 2048),
                                     (130, 1024, 1024), (5, 4096, 4096), (33, 384, 128)])
def test_quantize_exact_on_oracle_rotation_per_token(M, K, had):
    x = _x(M, K, seed=M + K)
    y32 = O.rotate_activations(x.double().numpy(), had)
    y32[0, :] = 0.0  # an all-zero token: Delta = 0, codes 0
    qx, dx = O.quantize_activations_per_token(y32)
    xq, xs, xsum = G.rotate_quantize_rows(torch.from_numpy(y32), 1)
    assert np.array_equal(xs, dx)
    assert np.array_equal(O.unpack_int4(xq), qx)
    assert np.array_equal(xsum, qx.astype(np.int64).sum(1))


@pytest.mark.parametrize("delta", [0.37, 0.05, 2.0])
def test_quantize_exact_on_oracle_rotation_per_step_with_clamping(delta):
    M, K = 50, 1024
    x = _x(M, K, seed=3)
    y32 = O.rotate_activations(x.double().numpy(), 1024)
    d = np.float32(delta)
    qx = O.quantize(y32, d)
    xq, xs, xsum = G.rotate_quantize_rows(torch.from_numpy(y32), 1, step_scale=float(d))
    assert np.all(xs == d)
    assert np.array_equal(O.unpack_int4(xq), qx)
    assert np.array_equal(xsum, qx.astype(np.int64).sum(1))
    if delta == 0.05:
        assert np.count_nonzero(np.abs(qx) == 7) > 0.05 * qx.size  # clamping exercised


def test_quantize_exact_ties_round_to_even():
    # values on exact half-integers of Delta = 0.5: z = 0.25 * odd
    M, K = 8, 256
    rng = np.random.default_rng(9)
    z = (rng.integers(-14, 15, (M, K)) * 0.25).astype(np.float32)
    z[:, 0] = 3.5  # row max -> Delta = 0.5 exactly
    qx, dx = O.quantize_activations_per_token(z)
    assert np.all(dx == np.float32(0.5))
    xq, xs, _ = G.rotate_quantize_rows(torch.from_numpy(z), 1)
    assert np.array_equal(O.unpack_int4(xq), qx)
    assert np.array_equal(xs, dx)


@pytest.mark.parametrize("dtype", ["f16", "bf16", "f32"])
@pytest.mark.parametrize("M,K,had", [(64, 512, 512), (200, 2048, 2048), (17, 16384, 2048), (50, 4096, 4096),
                                     (33, 1024, 64), (20, 1024, 256), (12, 2048, 16)])
def test_rotate_quantize_end_to_end(dtype, M, K, had):
    x = _x(M, K, seed=K + had, dtype=dtype)
    y32 = O.rotate_activations(x.double().numpy(), had)
    qx, dx = O.quantize_activations_per_token(y32)
    xq, xs, xsum = G.rotate_quantize_rows(x, had)
    got = O.unpack_int4(xq)
    # scales: float32 rotation on the GPU vs float64 on the oracle, a few ulp apart
    assert np.allclose(xs, dx, rtol=4e-7, atol=0)
    assert np.array_equal(xsum, got.astype(np.int64).sum(1))  # the sum is of the codes written
    frac, maxd, tie = G.code_mismatch_report(got, qx, y32.astype(np.float64) / dx.astype(np.float64)[:, None])
    assert frac <= 1e-5 and maxd <= 1, (frac, maxd)
    assert tie < 1e-4, tie


def test_rotate_quantize_per_step_end_to_end():
    case = W.single_layer_steps(seed=0)
    table = O.calibrate_step_table([x.double().numpy() for x in case.x_steps], case.had_block)
    for t in (0, 4, 9):
        x = case.x_steps[t]
        y32 = O.rotate_activations(x.double().numpy(), case.had_block)
        qx, _ = O.quantize_activations_per_step(y32, table, t)
        xq, xs, _ = G.rotate_quantize_rows(x, case.had_block, step_scale=float(table[t]))
        assert np.all(xs == table[t])
        frac, maxd, _ = G.code_mismatch_report(O.unpack_int4(xq), qx, y32 / np.float64(table[t]))
        assert frac <= 1e-5 and maxd <= 1


def test_rotated_absmax_matches_oracle():
    x = _x(300, 2048, seed=11, dtype="bf16")
    ref = O.robust_peak(O.rotate_activations(x.double().numpy(), 2048), "absmax")
    out = torch.zeros(1, dtype=torch.float32, device=G.DEV)
    Q.qvla_rotated_absmax(x.to(G.DEV), Q.BF16, 300, 2048, 2048, out, G.stream())
    got = out.item()
    assert abs(got - float(ref)) <= 4e-7 * float(ref)


def test_empty_and_single_row():
    x = _x(1, 512, seed=1)
    xq, xs, xsum = G.rotate_quantize_rows(x, 512)
    y32 = O.rotate_activations(x.double().numpy(), 512)
    qx, dx = O.quantize_activations_per_token(y32)
    assert np.allclose(xs, dx, rtol=4e-7)
    Q.qvla_rotate_quantize_rows(None, Q.F16, 0, 512, 512, None, None, None, None, G.stream())
