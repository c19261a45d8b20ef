"""GPU parity of the rotate-quantise kernel in passes (csrc/rotate_quant_pass.cu): 16-bit
activations into the GEMM's operand bytes, one CTA per pass of up to 2048 channels, the passes of
a row in a cluster that exchanges the row maximum and gathers the code sum (Sec. 4.1 Eq. 3-5,
Sec. 4.2 Eq. 5-6).

qvla_linear_quantize takes it for f16/bf16 layers at up to 64 rows; its codes, scales and code
sums must be the bits of the row-per-warp kernel, which the packed-code entry
qvla_rotate_quantize_rows still runs (and which tests/test_gpu_rotate_quant.py pins to the
oracle).  Shapes cover one to eight passes per row, passes of 128 to 2048 channels, Hadamard
blocks from 1 to 2048, per-token and per-step scales with clipping, exact ties, zero rows and
one huge value; end to end it is also checked against the oracle."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _round256(v):
    return (v + 255) // 256 * 256


def _codes_from_operand_bytes(ob):
    """Operand bytes [M][K] (q + 8, each group of 8 stored k0 k2 k4 k6 k1 k3 k5 k7) -> codes [M][K]."""
    M, K = ob.shape
    g = ob.reshape(M, K // 8, 8).astype(np.int16) - 8
    out = np.empty((M, K // 8, 8), np.int16)
    out[:, :, 0::2] = g[:, :, 0:4]
    out[:, :, 1::2] = g[:, :, 4:8]
    return out.reshape(M, K).astype(np.int8)


def _pass_kernel(x, had, step_scale=None):
    """Codes, scales and sums from qvla_linear_quantize (the pass kernel), read from its workspace."""
    M, K = x.shape
    dt = {torch.float16: "f16", torch.bfloat16: "bf16"}[x.dtype]
    layer = G.make_layer(np.zeros((16, K // 2), np.uint8), np.ones(16, np.float32), had, dt, dt)
    step = -1
    if step_scale is not None:
        Q.qvla_set_step_scales(layer, np.array([step_scale], np.float32))
        step = 0
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.full((nbytes,), 0xEE, dtype=torch.uint8, device=G.DEV)
    Q.qvla_linear_quantize(layer, x.to(G.DEV).contiguous(), M, step, work, nbytes, G.stream())
    Q.qvla_check_device(G.stream())
    w = work.cpu().numpy()
    layer.close()
    ob = w[:M * K].reshape(M, K)
    o = _round256(M * K)
    xs = w[o:o + 4 * M].view(np.float32).copy()
    o += _round256(4 * M)
    xsum = w[o:o + 4 * M].view(np.int32).astype(np.int64)
    return _codes_from_operand_bytes(ob), xs, xsum


def _row_kernel(x, had, step_scale=None):
    xq, xs, xsum = G.rotate_quantize_rows(x, had, step_scale)
    return O.unpack_int4(xq), xs, xsum.astype(np.int64)


def _input(M, K, seed, dt):
    rng = np.random.default_rng(seed)
    x = W.gaussian_with_outliers(rng, M, K, max(1, K // 500), 20.0)
    x[0] = 0.0  # an all-zero token: scale 0, codes 0
    return W.as_dtype(x, dt)


SHAPES = [(64, 2048, 2048), (4, 16384, 2048), (50, 1024, 1024), (3, 3072, 1024), (7, 384, 128), (33, 4096, 64),
          (5, 16384, 512), (5, 2048, 1), (1, 128, 128), (6, 640, 128), (50, 4096, 1024)]


@pytest.mark.parametrize("dt", ["f16", "bf16"])
@pytest.mark.parametrize("M,K,had", SHAPES)
def test_pass_kernel_equals_row_kernel_per_token(dt, M, K, had):
    x = _input(M, K, M + K + had, dt)
    q1, s1, c1 = _pass_kernel(x, had)
    q0, s0, c0 = _row_kernel(x, had)
    assert np.array_equal(s1, s0)
    assert np.array_equal(q1, q0)
    assert np.array_equal(c1, c0)
    assert np.array_equal(c1, q1.astype(np.int64).sum(1))


@pytest.mark.parametrize("dt", ["f16", "bf16"])
@pytest.mark.parametrize("M,K,had", SHAPES[:6])
@pytest.mark.parametrize("delta", [0.02, 0.3, 40.0])
def test_pass_kernel_equals_row_kernel_per_step(dt, M, K, had, delta):
    x = _input(M, K, 3 * M + K + had, dt)
    q1, s1, c1 = _pass_kernel(x, had, delta)
    q0, s0, c0 = _row_kernel(x, had, delta)
    assert np.all(s1 == np.float32(delta))
    assert np.array_equal(q1, q0)
    assert np.array_equal(c1, c0)


@pytest.mark.parametrize("K", [2048, 8192])
def test_pass_kernel_exact_ties(K):
    """No rotation (b = 1), half-integer values of the scale: every code sits on a tie and takes the
    exact rule, rounding half to even; a row of one huge value; one with the maximum in the last
    pass (the cluster exchange decides its scale)."""
    rng = np.random.default_rng(K)
    x = (rng.integers(-7, 7, (4, K)) + 0.5).astype(np.float32)  # 4 rows: the pass kernel's range
    x[1] = 0.5
    x[1, K - 3] = 7.0  # scale 1, every other value a tie at 0.5
    x[2] = 0.0
    x[2, 5] = -60000.0
    xt = torch.from_numpy(x).to(torch.float16)
    q1, s1, c1 = _pass_kernel(xt, 1)
    q0, s0, c0 = _row_kernel(xt, 1)
    assert np.array_equal(s1, s0) and np.array_equal(q1, q0) and np.array_equal(c1, c0)
    assert s1[1] == 1.0
    assert np.all(q1[1, :K - 3] == 0) and q1[1, K - 3] == 7


@pytest.mark.parametrize("M,K,had", [(64, 16384, 2048), (4, 2048, 2048)])
def test_pass_kernel_against_oracle(M, K, had):
    x = _input(M, K, 7 + M, "bf16")
    q1, s1, c1 = _pass_kernel(x, had)
    y32 = O.rotate_activations(x.double().numpy(), had)
    qx, dx = O.quantize_activations_per_token(y32)
    # float32 butterflies in a fixed order against the oracle's rotation: codes may differ by one
    # next to a rounding tie, at most 1e-5 of them (the row-per-warp kernel's bound)
    diff = q1.astype(np.int16) - qx.astype(np.int16)
    assert np.abs(diff).max() <= 1
    assert np.count_nonzero(diff) <= max(1, int(1e-5 * diff.size))
    assert np.allclose(s1, dx, rtol=2e-6, atol=0)
