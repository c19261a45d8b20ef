"""GPU parity of the whole W4A4 linear (Sec. 4: rotate, quantise, integer GEMM, dequantise)
through qvla_w4a4_linear, on the synthetic workloads shaped like the paper's layers."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _layer_from_host_pack(w, had, xdt, ydt, bias=None, rot=None, rot_block=0):
    N, K = w.shape
    wq = np.zeros((N, K // 2), np.uint8)
    ws = np.zeros(N, np.float32)
    Q.qvla_pack_weights_host(np.ascontiguousarray(w, dtype=np.float32), Q.F32, N, K, rot=rot, rot_block=rot_block,
                             had_block=had, wq=wq, wscale=ws)
    return G.make_layer(wq, ws, had, xdt, ydt, bias), wq, ws


def test_single_layer_per_step_table_all_steps():
    """64 x 512 x 512 fp16, random orthogonal SVD stand-in folded offline, Hadamard 512,
    T = 10 per-step scales calibrated from X_t = X (1 + 0.3 t)."""
    case = W.single_layer_steps(seed=0)
    layer, wq, ws = _layer_from_host_pack(case.w, case.had_block, "f16", "f16", rot=np.ascontiguousarray(case.rot),
                                          rot_block=case.rot_block)
    table = O.calibrate_step_table([x.double().numpy() for x in case.x_steps], case.had_block)
    Q.qvla_set_step_scales(layer, table)
    assert Q.qvla_layer_info(layer) == (512, 512, 512, 10)
    wcodes = O.unpack_int4(wq)
    for t in range(10):
        x = case.x_steps[t]
        ref = O.w4a4_linear(x.double().numpy(), wcodes, ws, case.had_block, table=table, step=t, out_fmt="f16")
        got = G.linear(layer, x, step=t)
        G.assert_output_close(got, ref["y"])
        # the quantised layer approximates the unquantised product X W^T
        yref = case.x_orig_steps[t] @ case.w.astype(np.float64).T
        assert O.relative_output_error(got, yref) < 0.35
    layer.close()


@pytest.mark.parametrize("M,K,N", [(1, 1024, 1024), (16, 2048, 2048), (50, 1024, 4096), (256, 2048, 2048),
                                   (816, 2048, 1024), (300, 16384, 2048), (3200, 1024, 1024),
                                   (1, 16384, 2048), (100, 1024, 8192), (50, 4096, 1024)])
def test_linear_per_token_sweep_points(M, K, N):
    case = W.sweep_linear(M, K, N, xdtype="bf16", ydtype="bf16", with_bias=True)
    layer, wq, ws = _layer_from_host_pack(case.w, case.had_block, "bf16", "bf16", bias=case.bias)
    got = G.linear(layer, case.x, ydt="bf16")
    ref = O.w4a4_linear(case.x.double().numpy(), O.unpack_int4(wq), ws, case.had_block, bias=case.bias, out_fmt="bf16")
    G.assert_output_close(got, ref["y"], "bf16")
    layer.close()


def test_gated_mlp_gate_up_full_size_sampled():
    """The backbone MLP's gate/up projection at full size (816 x 2048 -> 32768 as one GEMM);
    the oracle checks a random sample of 512 output channels."""
    mlp = W.gated_mlp(seed=1)
    w = np.concatenate([mlp.w_gate, mlp.w_up], axis=0)
    layer, wq, ws = _layer_from_host_pack(w, mlp.had_in, "bf16", "bf16")
    got = G.linear(layer, mlp.x, ydt="bf16")
    cols = np.sort(np.random.default_rng(0).choice(w.shape[0], 512, replace=False))
    ref = O.w4a4_linear(mlp.x.double().numpy(), O.unpack_int4(wq[cols]), ws[cols], mlp.had_in, out_fmt="bf16")
    G.assert_output_close(got[:, cols], ref["y"], "bf16")
    layer.close()


def test_step_out_of_range_and_missing_table():
    rng = np.random.default_rng(1)
    w = W.gaussian_weights(rng, 32, 256, 0.02)
    layer, _, _ = _layer_from_host_pack(w, 256, "f16", "f16")
    x = torch.zeros(4, 256, dtype=torch.float16, device=G.DEV)
    y = torch.zeros(4, 32, dtype=torch.float16, device=G.DEV)
    work = torch.empty(Q.qvla_linear_workspace_bytes(layer, 4), dtype=torch.uint8, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_w4a4_linear(layer, x, 4, 0, y, work, work.numel(), G.stream())
    assert e.value.status == 5
    Q.qvla_set_step_scales(layer, np.array([0.1, 0.2], np.float32))
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_w4a4_linear(layer, x, 4, 2, y, work, work.numel(), G.stream())
    assert e.value.status == 5
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_w4a4_linear(layer, x, 4, 1, y, work, 16, G.stream())
    assert e.value.status == 1
    Q.qvla_w4a4_linear(layer, x, 4, 1, y, work, work.numel(), G.stream())
    Q.qvla_check_device(G.stream())
    assert torch.count_nonzero(y).item() == 0  # zero input, no bias
    layer.close()


def _gated_layer(mlp_w_gate, mlp_w_up, had, xdt="bf16", ydt="bf16"):
    H, K = mlp_w_gate.shape
    packs = []
    for w in (mlp_w_gate, mlp_w_up):
        wq = np.zeros((H, K // 2), np.uint8)
        ws = np.zeros(H, np.float32)
        Q.qvla_pack_weights_host(np.ascontiguousarray(w, dtype=np.float32), Q.F32, H, K, had_block=had, wq=wq, wscale=ws)
        packs.append((wq, ws))
    layer = Q.qvla_layer_create_gated(H, K, had, Q.DTYPE_CODES[xdt], Q.DTYPE_CODES[ydt], packs[0][0], packs[0][1],
                                      packs[1][0], packs[1][1])
    return layer, packs


def _oracle_h(x, packs, had, rows=None, cols=None):
    """h = bf16(gelu_tanh(gate) * up) with gate and up each a W4A4 linear rounded to bf16."""
    outs = []
    for wq, ws in packs:
        sel = slice(None) if cols is None else cols
        outs.append(O.w4a4_linear(x, O.unpack_int4(wq[sel]), ws[sel], had, out_fmt="bf16"))
    return O.round_to_format(O.gated_glue(outs[0]["y"], outs[1]["y"]), "bf16"), outs


def test_gated_mlp_layer_small():
    mlp = W.gated_mlp(seed=5, m=200, k=1024, hidden=512, had_in=1024)
    layer, packs = _gated_layer(mlp.w_gate, mlp.w_up, 1024)
    assert Q.qvla_layer_info(layer)[0] == 512
    # accumulators: [gate | up] in natural order
    x = mlp.x
    M, K = x.shape
    xq, xs, xsum = G.rotate_quantize_rows(x, 1024)
    h_ref, outs = _oracle_h(x.double().numpy(), packs, 1024)
    y, acc = G.gemm(layer, xq, xs, xsum, ydt="bf16")
    qx = O.unpack_int4(xq)
    ref_acc = np.concatenate([O.int_gemm(qx, O.unpack_int4(p[0])) for p in packs], axis=1)
    assert y.shape == (M, 512) and acc.shape == (M, 1024)
    assert np.array_equal(acc, ref_acc)
    h = G.linear(layer, x, ydt="bf16")
    G.assert_output_close(h, h_ref, "bf16")
    layer.close()


def test_gated_mlp_block_full_size_sampled():
    """The whole backbone MLP block at full size: h = gelu(gate) * up from the gated layer
    (816 x 2048 -> 16384), then the down projection 16384 -> 2048 (Hadamard 8 x 2048).
    The oracle recomputes 64 sampled hidden units of h and, from the GPU's h, 256 sampled
    output channels of the down projection."""
    mlp = W.gated_mlp(seed=1)
    layer, packs = _gated_layer(mlp.w_gate, mlp.w_up, mlp.had_in)
    h = G.linear(layer, mlp.x, ydt="bf16")
    cols = np.sort(np.random.default_rng(1).choice(mlp.w_gate.shape[0], 64, replace=False))
    h_ref, _ = _oracle_h(mlp.x.double().numpy(), packs, mlp.had_in, cols=cols)
    G.assert_output_close(h[:, cols], h_ref, "bf16")
    down, wq, ws = _layer_from_host_pack(mlp.w_down, mlp.had_hidden, "bf16", "bf16")
    h_t = torch.from_numpy(h.astype(np.float32)).to(torch.bfloat16)
    y = G.linear(down, h_t, ydt="bf16")
    ocols = np.sort(np.random.default_rng(2).choice(mlp.w_down.shape[0], 256, replace=False))
    ref = O.w4a4_linear(h_t.double().numpy(), O.unpack_int4(wq[ocols]), ws[ocols], mlp.had_hidden, out_fmt="bf16")
    G.assert_output_close(y[:, ocols], ref["y"], "bf16")
    layer.close()
    down.close()


def test_linear_halves_equal_whole_call():
    """qvla_linear_quantize + qvla_linear_gemm are the two kernels of qvla_w4a4_linear."""
    case = W.sweep_linear(300, 2048, 512, seed=31, xdtype="bf16", ydtype="bf16", with_bias=True)
    layer, _, _ = _layer_from_host_pack(case.w, case.had_block, "bf16", "bf16", bias=case.bias)
    whole = G.linear(layer, case.x, ydt="bf16")
    M = case.x.shape[0]
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.empty(nbytes, dtype=torch.uint8, device=G.DEV)
    y = torch.full((M, layer.N), float("nan"), dtype=torch.bfloat16, device=G.DEV)
    Q.qvla_linear_quantize(layer, case.x.to(G.DEV), M, -1, work, nbytes, G.stream())
    Q.qvla_linear_gemm(layer, work, nbytes, M, y, G.stream())
    Q.qvla_check_device(G.stream())
    assert np.array_equal(y.double().cpu().numpy(), whole)
    layer.close()


def test_linear_with_block_svd_and_zigzag_rotation():
    """The full composite rotation of Sec. 4.1 (Eq. 4-5): P and U_b chosen from the weights by
    the library (zigzag permutation, block SVD with block 64, the paper's setting), folded with
    Hadamard 512; the activations get x . P . BlockDiag(U_b) upstream (float64, rounded once to
    fp16) and the online path runs per token.  Both sides use the same factors."""
    rng = np.random.default_rng(41)
    M, N, K, block, had = 96, 384, 1024, 64, 512
    w = (W.gaussian_weights(rng, N, K, 0.02) * rng.uniform(0.2, 4.0, K)[None, :]).astype(np.float32)
    x = W.gaussian_with_outliers(rng, M, K, 5, 20.0)
    perm, rot = Q.qvla_block_svd_rotation(w, Q.F32, N, K, block)
    wq = np.zeros((N, K // 2), np.uint8)
    ws = np.zeros(N, np.float32)
    Q.qvla_pack_weights_host(w, Q.F32, N, K, rot=rot, rot_block=block, perm=perm, had_block=had, wq=wq, wscale=ws)
    layer = G.make_layer(wq, ws, had, "f16", "f16")
    x_up = W.as_dtype(O.upstream_activation_transform(x, perm, rot, block), "f16")
    got = G.linear(layer, x_up, ydt="f16")
    _, oscale, codes = O.pack_weights(w.astype(np.float64), had, perm=perm, rot=rot, rot_block=block)
    ref = O.w4a4_linear(x_up.double().numpy(), codes, oscale, had, out_fmt="f16")
    G.assert_output_close(got, ref["y"], "f16")
    # the quantised layer still approximates the float one (the rotation is orthogonal)
    exact = x.astype(np.float64) @ w.astype(np.float64).T
    assert O.relative_output_error(got, exact) < 0.35
    layer.close()
