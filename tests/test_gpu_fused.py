"""GPU parity of the one-launch linear (qvla_w4a4_linear_fused): the DiT head's per-step-scale
linear with the rotation and the quantiser (Sec. 4.1 Eq. 3-5; Sec. 4.2 Eq. 6, second display) run
by the GEMM's own CTAs, against the oracle, on every DiT shape at M = 50 and M = 1 with clamping.

Where the Hadamard block fits one warp task (b <= 1024 at K = 1024, b <= 2048 beyond) the fused
kernel runs the butterflies in the separate rotate + quantise kernel's order, so its outputs equal
the two-launch path's bit for bit; for b = 4096 it sums the block's two halves first, a different
float32 order, so a code may move by one step at a rounding tie and the outputs are compared
within the output tolerance instead."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu

DIT_SHAPES = [(1024, 3072), (1024, 1024), (1024, 4096), (4096, 1024)]  # (K, N): qkv, o, up, down


def _layer(n, k, had, seed, xdt="f16", ydt="f16", bias=True):
    rng = np.random.default_rng(seed)
    codes = W.gaussian_codes(rng, n, k)
    ws = (rng.uniform(0.8, 1.2, n) * 0.5 / np.sqrt(k)).astype(np.float32)
    b = (rng.standard_normal(n) * 0.05).astype(np.float32) if bias else None
    return G.make_layer(W.pack_nibbles(codes), ws, had, xdt, ydt, b), codes, ws, b


def _x(m, k, seed, std=1.0, dtype="f16"):
    rng = np.random.default_rng(seed)
    return W.as_dtype(rng.standard_normal((m, k)) * std, dtype)


def _fused(layer, x, step, ydt="f16"):
    M = x.shape[0]
    y = torch.full((M, layer.N), float("nan"), dtype=G.TORCH_DT[ydt], device=G.DEV)
    Q.qvla_w4a4_linear_fused(layer, x.to(G.DEV).contiguous(), M, step, y, G.stream())
    Q.qvla_check_device(G.stream())
    return y.double().cpu().numpy()


def _two_launch(layer, x, step, ydt="f16"):
    M = x.shape[0]
    nb = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.empty(nb, dtype=torch.uint8, device=G.DEV)
    y = torch.full((M, layer.N), float("nan"), dtype=G.TORCH_DT[ydt], device=G.DEV)
    Q.qvla_linear_quantize(layer, x.to(G.DEV).contiguous(), M, step, work, nb, G.stream())
    Q.qvla_linear_gemm(layer, work, nb, M, y, G.stream())
    Q.qvla_check_device(G.stream())
    return y.double().cpu().numpy()


@pytest.mark.parametrize("M", [50, 1])
@pytest.mark.parametrize("K,N", DIT_SHAPES)
def test_fused_dit_shapes_against_oracle(K, N, M):
    layer, codes, ws, bias = _layer(N, K, K, seed=K + N)
    x = _x(M, K, seed=M + K + N, std=2.0)
    y_rot = O.rotate_activations(x.double().numpy(), K)
    peak = np.float32(np.abs(y_rot).max())
    # step 0: the batch's own peak (nothing clamps); step 1: a third of it (codes clamp at +-7)
    table = np.array([peak / np.float32(7), peak / np.float32(21)], np.float32)
    Q.qvla_set_step_scales(layer, table)
    for t in (0, 1):
        got = _fused(layer, x, t)
        ref = O.w4a4_linear(x.double().numpy(), codes, ws, K, bias=bias, table=table, step=t, out_fmt="f16")
        G.assert_linear_close_modulo_ties(got, ref, codes, ws, bias, "f16")
        if t == 1:
            assert np.count_nonzero(np.abs(ref["qx"]) == 7) > 0.05 * ref["qx"].size  # clamping exercised
        two = _two_launch(layer, x, t)
        if K <= 2048:
            assert np.array_equal(got, two)
        else:  # a different float32 order: each path within the contract on its own
            G.assert_linear_close_modulo_ties(two, ref, codes, ws, bias, "f16")
    layer.close()


@pytest.mark.parametrize("K,had", [(1024, 1), (1024, 16), (1024, 64), (1024, 256), (2048, 2048), (2048, 128),
                                   (4096, 512), (4096, 2048), (4096, 4096), (512, 512), (3072, 1024)])
@pytest.mark.parametrize("M", [3, 64, 100])
def test_fused_hadamard_blocks_and_batches(K, had, M):
    N = 256
    layer, codes, ws, bias = _layer(N, K, had, seed=K + had + M, xdt="bf16", ydt="bf16")
    x = _x(M, K, seed=7 * M + had, dtype="bf16")
    table = np.array([np.float32(np.abs(O.rotate_activations(x.double().numpy(), had)).max()) / np.float32(9)],
                     np.float32)
    Q.qvla_set_step_scales(layer, table)
    # refused: K = 3072 (not a whole number of 2048-channel warp tasks); more than 64 tokens at
    # K = 4096 (a 128-token tile leaves room for 2 k-blocks per CTA, and 16 CTAs per tile exceed
    # the cluster)
    refused = K == 3072 or (M > 64 and K >= 4096)
    try:
        got = _fused(layer, x, 0, "bf16")
    except Q.QvlaError as e:
        assert refused and e.status == 2, e
        # the linear still runs it, on two launches
        G.assert_linear_close_modulo_ties(G.linear(layer, x, step=0, ydt="bf16"),
                                          O.w4a4_linear(x.double().numpy(), codes, ws, had, bias=bias, table=table,
                                                        step=0, out_fmt="bf16"), codes, ws, bias, "bf16")
        layer.close()
        return
    assert not refused
    ref = O.w4a4_linear(x.double().numpy(), codes, ws, had, bias=bias, table=table, step=0, out_fmt="bf16")
    G.assert_linear_close_modulo_ties(got, ref, codes, ws, bias, "bf16")
    two = _two_launch(layer, x, 0, "bf16")
    if had <= (1024 if K <= 1024 else 2048):
        assert np.array_equal(got, two)
    layer.close()


def test_fused_equals_the_linear_and_repeats_exactly():
    """The one-launch path gives qvla_w4a4_linear's bits (K = 1024: the same butterfly order);
    20 launches in a row give the same bits (no race between the prologue's copies and the GEMM)."""
    K, N, M = 1024, 3072, 50
    layer, _, _, _ = _layer(N, K, K, seed=99)
    x = _x(M, K, seed=98)
    Q.qvla_set_step_scales(layer, np.array([0.4], np.float32))
    first = _fused(layer, x, 0)
    whole = G.linear(layer, x, step=0, ydt="f16")
    assert np.array_equal(first, whole)
    xg = x.to(G.DEV)
    ys = [torch.empty(M, N, dtype=torch.float16, device=G.DEV) for _ in range(20)]
    for y in ys:
        Q.qvla_w4a4_linear_fused(layer, xg, M, 0, y, G.stream())
    Q.qvla_check_device(G.stream())
    for y in ys:
        assert np.array_equal(y.double().cpu().numpy(), first)
    layer.close()


def test_fused_refusals():
    layer, _, _, _ = _layer(256, 1024, 1024, seed=5)
    x = torch.zeros(200, 1024, dtype=torch.float16, device=G.DEV)
    y = torch.zeros(200, 256, dtype=torch.float16, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:  # per-token scales: a row reduction precedes the codes
        Q.qvla_w4a4_linear_fused(layer, x, 50, -1, y, G.stream())
    assert e.value.status == 2
    with pytest.raises(Q.QvlaError) as e:  # no table yet
        Q.qvla_w4a4_linear_fused(layer, x, 50, 0, y, G.stream())
    assert e.value.status == 5
    Q.qvla_set_step_scales(layer, np.array([0.3], np.float32))
    with pytest.raises(Q.QvlaError) as e:  # more than one token tile
        Q.qvla_w4a4_linear_fused(layer, x, 129, 0, y, G.stream())
    assert e.value.status == 2
    layer.close()
    big, _, _, _ = _layer(256, 16384, 2048, seed=6)
    Q.qvla_set_step_scales(big, np.array([0.3], np.float32))
    xb = torch.zeros(4, 16384, dtype=torch.float16, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:  # K beyond 4096
        Q.qvla_w4a4_linear_fused(big, xb, 4, 0, y, G.stream())
    assert e.value.status == 2
    big.close()
