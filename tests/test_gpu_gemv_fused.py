"""GPU parity of the one-launch decode linear (one token): the CUDA-core GEMV that rotates and
quantises its activations itself (Sec. 4.1 Eq. 3-5 and Sec. 4.2 Eq. 5-7 in one kernel).

qvla_w4a4_linear takes it for M = 1 where the layer allows it (rotation passes of up to 2048
channels holding whole Hadamard blocks, f16/bf16 input and output of one dtype, about one CTA
per SM).  It leaves the caller's workspace untouched, which tells the tests which path ran.  Its
outputs must be the bits of the two-launch path (the rotate-quantise kernel through
qvla_linear_quantize, then the GEMM through qvla_linear_gemm, which shares no code with its
prologue): per-token scales (the row's maximum, gathered across a split-K cluster where one
pass is not the whole row) and per-step scales, passes of 128 to 2048 channels, Hadamard blocks
from 1 to 2048, exact rounding ties, zero tokens, ragged N, gated layers and an online rotation
ahead of the quantiser.  A few cases are also checked against the oracle within the tie-aware
tolerance."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu

SENTINEL = 0xA5


def _layer(rng, N, K, had, dt, bias=True):
    wcodes = rng.integers(-8, 8, (N, K)).astype(np.int8)
    ws = rng.uniform(0.5, 2.0, N).astype(np.float32) * np.float32(2 ** -7)
    b = (rng.standard_normal(N) * 0.1).astype(np.float32) if bias else None
    return G.make_layer(O.pack_int4(wcodes), ws, had, dt, dt, b), wcodes, ws, b


def _two_launch(layer, x, step, dt):
    """The rotate-quantise kernel, then the GEMM, through their own entry points."""
    M = x.shape[0]
    xg = x.to(G.DEV).contiguous()
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=G.DEV)
    y = torch.full((M, layer.N), float("nan"), dtype=G.TORCH_DT[dt], device=G.DEV)
    Q.qvla_linear_quantize(layer, xg, M, step, work, nbytes, G.stream())
    Q.qvla_linear_gemm(layer, work, nbytes, M, y, G.stream())
    Q.qvla_check_device(G.stream())
    return y.double().cpu().numpy()


def _one_launch(layer, x, step, dt):
    """qvla_w4a4_linear with a sentinel-filled workspace: (y, whether the workspace is untouched)."""
    M = x.shape[0]
    xg = x.to(G.DEV).contiguous()
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.full((max(nbytes, 256),), SENTINEL, dtype=torch.uint8, device=G.DEV)
    y = torch.full((M, layer.N), float("nan"), dtype=G.TORCH_DT[dt], device=G.DEV)
    Q.qvla_w4a4_linear(layer, xg, M, step, y, work, nbytes, G.stream())
    Q.qvla_check_device(G.stream())
    return y.double().cpu().numpy(), bool(torch.all(work == SENTINEL).item())


def _input(rng, M, K, dt):
    x = W.gaussian_with_outliers(rng, M, K, max(1, K // 500), 20.0)
    return W.as_dtype(x, dt)


SHAPES = [(2048, 2560, 2048), (16384, 2048, 2048), (1024, 1024, 64), (384, 272, 128), (3072, 512, 1024), (2048, 128, 1),
          (16384, 16, 512), (1024, 4096, 1024)]


@pytest.mark.parametrize("dt", ["f16", "bf16"])
@pytest.mark.parametrize("K,N,had", SHAPES)
def test_one_launch_equals_two_launch_per_token(dt, K, N, had):
    rng = np.random.default_rng(K + N + had)
    layer, _, _, _ = _layer(rng, N, K, had, dt)
    for row in range(3):
        x = _input(rng, 1, K, dt)
        got, untouched = _one_launch(layer, x, -1, dt)
        assert untouched, "the one-launch linear should take this layer"
        assert np.all(np.isfinite(got))
        assert np.array_equal(got, _two_launch(layer, x, -1, dt)), f"row {row}"
    layer.close()


@pytest.mark.parametrize("dt", ["f16", "bf16"])
@pytest.mark.parametrize("K,N,had", SHAPES[:4])
def test_one_launch_equals_two_launch_per_step(dt, K, N, had):
    rng = np.random.default_rng(11 + K + N + had)
    layer, _, _, _ = _layer(rng, N, K, had, dt)
    x = _input(rng, 1, K, dt)
    # scales that clip the outlier channels (codes held at +-7) and one that clips nothing
    Q.qvla_set_step_scales(layer, np.array([0.05, 0.4, 50.0], np.float32))
    for step in range(3):
        got, untouched = _one_launch(layer, x, step, dt)
        assert untouched
        assert np.array_equal(got, _two_launch(layer, x, step, dt)), f"step {step}"
    layer.close()


@pytest.mark.parametrize("K,N,had,M,xdt", [(4096, 256, 4096, 1, "bf16"), (2048, 2560, 2048, 2, "bf16"),
                                            (2048, 512, 2048, 1, "f32")])
def test_layers_outside_the_one_launch_take_two(K, N, had, M, xdt):
    """A Hadamard block wider than one pass, more than one token, or float32 input: the two
    launches run (the workspace is written), with the same result."""
    rng = np.random.default_rng(K + N + M)
    wcodes = rng.integers(-8, 8, (N, K)).astype(np.int8)
    layer = G.make_layer(O.pack_int4(wcodes), np.full(N, 2 ** -8, np.float32), had, xdt, "bf16")
    x = _input(rng, M, K, xdt)
    got, untouched = _one_launch(layer, x, -1, "bf16")
    assert not untouched
    assert np.array_equal(got, _two_launch(layer, x, -1, "bf16"))
    layer.close()


@pytest.mark.parametrize("per_step", [False, True])
def test_one_launch_exact_ties_and_zero_tokens(per_step):
    """Half-integer values of the scale (no rotation, b = 1): every code is decided at a tie, by
    the exact rule; an all-zero token has scale 0 and codes 0; a token of one huge value."""
    K, N = 4096, 384
    rng = np.random.default_rng(5)
    layer, wcodes, ws, b = _layer(rng, N, K, 1, "f16")
    x = (rng.integers(-7, 7, (4, K)) + 0.5).astype(np.float32)
    x[1] = 0.0
    x[2, :] = 0.5
    x[2, 100] = 7.0  # per-token scale 1: every other value a tie at 0.5
    x[3, :] = 0.0
    x[3, 7] = -60000.0
    xt = torch.from_numpy(x).to(torch.float16)
    step = -1
    if per_step:
        Q.qvla_set_step_scales(layer, np.array([1.0], np.float32))
        step = 0
    rows = []
    for r in range(4):
        got, untouched = _one_launch(layer, xt[r:r + 1], step, "f16")
        assert untouched
        assert np.array_equal(got, _two_launch(layer, xt[r:r + 1], step, "f16")), f"row {r}"
        rows.append(got)
    got = np.concatenate(rows)
    if per_step:
        ref = O.w4a4_linear(xt.double().numpy(), wcodes, ws, 1, bias=b, table=np.array([1.0], np.float32), step=0,
                            out_fmt="f16")
    else:
        ref = O.w4a4_linear(xt.double().numpy(), wcodes, ws, 1, bias=b, out_fmt="f16")
    G.assert_linear_close_modulo_ties(got, ref, wcodes, ws, b, "f16")
    assert np.array_equal(got[1], O.round_to_format(b.astype(np.float64), "f16"))
    layer.close()


@pytest.mark.parametrize("dt", ["f16", "bf16"])
def test_one_launch_against_oracle(dt):
    """The backbone's down projection shape (K = 16384 in 8 Hadamard blocks of 2048, split over a
    cluster of 8 CTAs that exchange their maxima) against the oracle, three tokens one by one."""
    K, N, had = 16384, 2048, 2048
    rng = np.random.default_rng(17)
    layer, wcodes, ws, b = _layer(rng, N, K, had, dt)
    x = _input(rng, 3, K, dt)
    got = np.concatenate([_one_launch(layer, x[r:r + 1], -1, dt)[0] for r in range(3)])
    ref = O.w4a4_linear(x.double().numpy(), wcodes, ws, had, bias=b, out_fmt=dt)
    G.assert_linear_close_modulo_ties(got, ref, wcodes, ws, b, dt)
    layer.close()


@pytest.mark.parametrize("step", [-1, 0])
def test_one_launch_gated(step):
    H, K, had = 1024, 2048, 2048
    rng = np.random.default_rng(23)
    qg = rng.integers(-8, 8, (H, K)).astype(np.int8)
    qu = rng.integers(-8, 8, (H, K)).astype(np.int8)
    dg = rng.uniform(0.5, 2.0, H).astype(np.float32) * np.float32(2 ** -7)
    du = rng.uniform(0.5, 2.0, H).astype(np.float32) * np.float32(2 ** -7)
    layer = Q.qvla_layer_create_gated(H, K, had, Q.BF16, Q.BF16, O.pack_int4(qg), dg, O.pack_int4(qu), du)
    Q.qvla_set_step_scales(layer, np.array([0.3], np.float32))
    for row in range(3):
        x = _input(rng, 1, K, "bf16")
        got, untouched = _one_launch(layer, x, step, "bf16")
        assert untouched
        assert np.array_equal(got, _two_launch(layer, x, step, "bf16")), f"row {row}"
    layer.close()


def test_one_launch_with_online_rotation():
    """x . P . BlockDiag(U_b) formed ahead of the one-launch linear, as ahead of the two launches."""
    rng = np.random.default_rng(29)
    N, K, block, had = 256, 1024, 64, 512
    perm = rng.permutation(K).astype(np.int32)
    rot = np.stack([np.linalg.qr(rng.standard_normal((block, block)))[0] for _ in range(K // block)])
    layer, _, _, _ = _layer(rng, N, K, had, "f16")
    Q.qvla_layer_set_online_rotation(layer, perm, rot, block)
    for M in (1, 4):
        x = _input(rng, M, K, "f16")
        got, _ = _one_launch(layer, x, -1, "f16")
        assert np.array_equal(got, _two_launch(layer, x, -1, "f16"))
    layer.close()


def test_one_launch_stream_order():
    """Twenty linears in a row on one stream, each reading the previous one's output (the launch
    waits for its producer through programmatic dependent launch): the chain's result equals the
    two-launch chain's."""
    K = N = 2048
    rng = np.random.default_rng(31)
    layer, _, _, _ = _layer(rng, N, K, 2048, "bf16", bias=False)
    x0 = _input(rng, 1, K, "bf16").to(G.DEV)
    nbytes = Q.qvla_linear_workspace_bytes(layer, 1)
    work = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=G.DEV)
    outs = []
    for fused in (True, False):
        a = x0.clone()
        b = torch.empty_like(a)
        for _ in range(20):
            if fused:
                Q.qvla_w4a4_linear(layer, a, 1, -1, b, work, nbytes, G.stream())
            else:
                Q.qvla_linear_quantize(layer, a, 1, -1, work, nbytes, G.stream())
                Q.qvla_linear_gemm(layer, work, nbytes, 1, b, G.stream())
            a, b = b, a
        Q.qvla_check_device(G.stream())
        outs.append(a.double().cpu().numpy())
    assert np.all(np.isfinite(outs[0]))
    assert np.array_equal(outs[0], outs[1])
    layer.close()
