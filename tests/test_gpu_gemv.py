"""GPU parity of the decode-sized path (one to four tokens: the CUDA-core GEMV of csrc/gemv.cu).

The integer accumulators are bit-exact against the oracle's integer product (Sec. 4.2, Eq. 7),
and the outputs are the tensor-core path's bits: the same tokens inside a five-token batch (which
takes the tensor-core GEMM) give the same rows, since with per-token scales a row depends on its
own token only.  Gated layers (h = gelu(gate) * up), ragged N, bias, f16 and bf16 outputs, and
both activation forms (packed codes through qvla_gemm_w4a4, operand bytes through the linear)."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _codes_layer(rng, N, K, had, ydt, bias=True):
    wcodes = rng.integers(-7, 8, (N, K)).astype(np.int8)
    ws = rng.uniform(0.5, 2.0, N).astype(np.float32) * np.float32(2 ** -7)
    b = (rng.standard_normal(N) * 0.1).astype(np.float32) if bias else None
    return G.make_layer(O.pack_int4(wcodes), ws, had, ydt, ydt, b), wcodes, ws, b


@pytest.mark.parametrize("M", [1, 2, 3, 4])
@pytest.mark.parametrize("N,K", [(16, 128), (256, 1024), (2048, 16384), (2560, 2048), (1008, 4096)])
def test_gemv_accumulators_exact(M, N, K):
    rng = np.random.default_rng(M * 1000 + N + K)
    layer, wcodes, ws, _ = _codes_layer(rng, N, K, 1, "bf16", bias=False)
    xcodes = rng.integers(-7, 8, (M, K)).astype(np.int8)
    xcodes[0, :min(K, 64)] = 7  # an extreme run
    xs = rng.uniform(0.5, 2.0, M).astype(np.float32) * np.float32(2 ** -6)
    y, acc = G.gemm(layer, O.pack_int4(xcodes), xs, xcodes.astype(np.int64).sum(1), ydt="bf16")
    assert np.array_equal(acc, O.int_gemm(xcodes, wcodes))
    G.assert_output_close(y, O.dequant_output(acc, xs, ws, None, "bf16"), "bf16")
    layer.close()


def test_gemv_extremes_at_k16384():
    # every product +7 x +7 and -7 x +7: the largest sums the unsigned dot products carry
    N, K = 128, 16384
    wcodes = np.full((N, K), 7, np.int8)
    wcodes[1::2] = -7
    layer = G.make_layer(O.pack_int4(wcodes), np.full(N, 2 ** -12, np.float32), 1, "f16", "f16")
    xcodes = np.stack([np.full(K, 7, np.int8), np.full(K, -7, np.int8)])
    _, acc = G.gemm(layer, O.pack_int4(xcodes), np.ones(2, np.float32), xcodes.astype(np.int64).sum(1))
    assert np.array_equal(acc, O.int_gemm(xcodes, wcodes))
    layer.close()


@pytest.mark.parametrize("ydt", ["f16", "bf16"])
@pytest.mark.parametrize("M", [1, 3, 4])
@pytest.mark.parametrize("K,N,had", [(2048, 2560, 2048), (16384, 2048, 2048), (1024, 1024, 64), (4096, 1008, 4096)])
def test_gemv_linear_equals_tensor_core_rows(ydt, M, K, N, had):
    """The linear at M tokens (GEMV) against the same tokens as rows of a five-token batch
    (tensor cores), bit for bit, and against the oracle within the tie-aware tolerance."""
    case = W.sweep_linear(5, K, N, seed=M + K + N, xdtype=ydt, ydtype=ydt, had_block=had, with_bias=True)
    wq = np.zeros((N, K // 2), np.uint8)
    wsc = np.zeros(N, np.float32)
    Q.qvla_pack_weights_host(np.ascontiguousarray(case.w), Q.F32, N, K, had_block=had, wq=wq, wscale=wsc)
    layer = G.make_layer(wq, wsc, had, ydt, ydt, case.bias)
    five = G.linear(layer, case.x, ydt=ydt)
    few = G.linear(layer, case.x[:M].contiguous(), ydt=ydt)
    assert np.array_equal(few, five[:M])
    ref = O.w4a4_linear(case.x[:M].double().numpy(), O.unpack_int4(wq), wsc, had, bias=case.bias, out_fmt=ydt)
    G.assert_linear_close_modulo_ties(few, ref, O.unpack_int4(wq), wsc, case.bias, ydt)
    layer.close()


@pytest.mark.parametrize("M", [1, 2, 4])
def test_gemv_gated_layer(M):
    """The gated gate/up layer (h = bf16(gelu(gate) * up), gate and up each rounded first): the
    GEMV's accumulators are exact in the [gate | up] order and its h equals the tensor-core
    path's rows."""
    mlp = W.gated_mlp(seed=9, m=5, k=2048, hidden=1024, had_in=2048)
    H, K = mlp.w_gate.shape
    packs = []
    for w in (mlp.w_gate, mlp.w_up):
        wq = np.zeros((H, K // 2), np.uint8)
        ws = np.zeros(H, np.float32)
        Q.qvla_pack_weights_host(np.ascontiguousarray(w), Q.F32, H, K, had_block=2048, wq=wq, wscale=ws)
        packs.append((wq, ws))
    layer = Q.qvla_layer_create_gated(H, K, 2048, Q.BF16, Q.BF16, packs[0][0], packs[0][1], packs[1][0], packs[1][1])
    five = G.linear(layer, mlp.x, ydt="bf16")
    few = G.linear(layer, mlp.x[:M].contiguous(), ydt="bf16")
    assert np.array_equal(few, five[:M])
    xq, xs, xsum = G.rotate_quantize_rows(mlp.x[:M], 2048)
    _, acc = G.gemm(layer, xq, xs, xsum, ydt="bf16")
    qx = O.unpack_int4(xq)
    ref_acc = np.concatenate([O.int_gemm(qx, O.unpack_int4(p[0])) for p in packs], axis=1)
    assert np.array_equal(acc, ref_acc)
    layer.close()
