"""GPU parity of the token-major GEMM's split of K into work units (Sec. 4.2, Eq. 7).

A non-gated layer whose token-major tiles leave SMs idle splits each tile's k-blocks into 2 or 4
work units when the caller's workspace has room for their FP32 partials
(qvla_linear_workspace_bytes counts it); the tile's last unit adds the others' partials to its
own and applies the epilogue.  Every partial is a non-negative integer multiple of the same power
of two below 2^24 of them, so the sum is exact in any order: the outputs must be the bits of the
whole-tile GEMM, which runs when the workspace is one byte short of that room.  Shapes: single
CTAs with 128- and 256-wide tiles in 4 parts, CTA pairs in 2 parts (the backbone's down
projection), ragged token and weight edges; a workspace full of garbage (the rotate-quantise
kernel zeroes the unit counters) and a GEMM run twice after one quantisation (the GEMM leaves
its counters zero)."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _layer(case):
    N, K = case.w.shape
    wq = np.zeros((N, K // 2), np.uint8)
    ws = np.zeros(N, np.float32)
    Q.qvla_pack_weights_host(np.ascontiguousarray(case.w), Q.F32, N, K, had_block=case.had_block, wq=wq, wscale=ws)
    return G.make_layer(wq, ws, case.had_block, "bf16", "bf16", case.bias), wq, ws


def _linear(layer, x, nbytes, fill=None, with_work=False):
    """qvla_w4a4_linear with a workspace of nbytes (filled with `fill` first, if given)."""
    M = x.shape[0]
    y = torch.full((M, layer.N), float("nan"), dtype=torch.bfloat16, device=G.DEV)
    work = torch.empty(nbytes, dtype=torch.uint8, device=G.DEV)
    if fill is not None:
        work.fill_(fill)
    Q.qvla_w4a4_linear(layer, x.to(G.DEV).contiguous(), M, -1, y, work, nbytes, G.stream())
    Q.qvla_check_device(G.stream())
    y = y.double().cpu().numpy()
    return (y, work.cpu().numpy()) if with_work else y


def _codes_in_workspace(w, M, K):
    """The activations' codes, scales and code sums the GEMM read: operand bytes [M][K] (q + 8,
    each group of 8 stored k0 k2 k4 k6 k1 k3 k5 k7), then 256-byte aligned scales and sums."""
    g = w[:M * K].reshape(M, K // 8, 8).astype(np.int16) - 8
    q = np.empty((M, K // 8, 8), np.int16)
    q[:, :, 0::2] = g[:, :, 0:4]
    q[:, :, 1::2] = g[:, :, 4:8]
    o = (M * K + 255) // 256 * 256
    xs = w[o:o + 4 * M].view(np.float32).copy()
    o += (4 * M + 255) // 256 * 256
    xsum = w[o:o + 4 * M].view(np.int32).astype(np.int64)
    return q.reshape(M, K).astype(np.int8), xs, xsum


# (M, K, N): single 128-wide tiles in 4 parts with a ragged token tile (150); single 256-wide
# tiles in 4 parts with a ragged weight tile (300 x 2000); pairs in 2 parts with ragged tokens and
# weights (700 x 1904); the backbone's down projection (816 x 16384 -> 2048, pairs in 2 parts)
SPLIT_SHAPES = [(150, 16384, 2048), (256, 16384, 2048), (300, 16384, 2000), (700, 16384, 1904), (816, 16384, 2048)]


@pytest.mark.parametrize("M,K,N", SPLIT_SHAPES)
def test_split_equals_whole_tiles(M, K, N):
    case = W.sweep_linear(M, K, N, seed=M + N, xdtype="bf16", ydtype="bf16", with_bias=True)
    layer, wq, ws = _layer(case)
    full = Q.qvla_linear_workspace_bytes(layer, M)
    split, work = _linear(layer, case.x, full, with_work=True)
    whole = _linear(layer, case.x, full - 1)  # no room for the partials: whole tiles
    assert np.array_equal(split, whole)
    dirty = _linear(layer, case.x, full, fill=0xEE)  # counters and partials start as garbage
    assert np.array_equal(dirty, whole)
    if M <= 300:
        # the oracle's integer GEMM and dequantisation on the codes the GEMM read
        qx, xs, xsum = _codes_in_workspace(work, M, K)
        assert np.array_equal(xsum, qx.astype(np.int64).sum(1))
        ref = O.dequant_output(O.int_gemm(qx, O.unpack_int4(wq)), xs, ws, case.bias, "bf16")
        G.assert_output_close(split, ref, "bf16")
    layer.close()


def test_split_gemm_twice_after_one_quantisation():
    """qvla_linear_quantize once, then qvla_linear_gemm twice on the same workspace: the first
    GEMM's last units reset the counters, so the second is the same."""
    M, K, N = 816, 16384, 2048
    case = W.sweep_linear(M, K, N, seed=5, xdtype="bf16", ydtype="bf16")
    layer, _, _ = _layer(case)
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.full((nbytes,), 0x5A, dtype=torch.uint8, device=G.DEV)
    Q.qvla_linear_quantize(layer, case.x.to(G.DEV).contiguous(), M, -1, work, nbytes, G.stream())
    outs = []
    for _ in range(2):
        y = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device=G.DEV)
        Q.qvla_linear_gemm(layer, work, nbytes, M, y, G.stream())
        Q.qvla_check_device(G.stream())
        outs.append(y.double().cpu().numpy())
    assert np.array_equal(outs[0], outs[1])
    assert np.array_equal(outs[0], _linear(layer, case.x, nbytes - 1))
    layer.close()
