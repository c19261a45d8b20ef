"""GPU parity of the single-linear throughput sweep: every point M in {1, 16, 50, 256, 816, 3200,
8192} x (K, N) in {(1024, 1024), (1024, 4096), (2048, 2048), (2048, 16384), (16384, 2048)}
through qvla_w4a4_linear with fp16 activations and fp16 outputs (Sec. 4: rotate, quantise per
token, integer GEMM, dequantise), against the oracle.

Per-token scales make every output row depend on its own input row only, so at large sizes the
oracle recomputes a sample of rows (always the first and the last, the ragged tail of the last
tile) over every output column.  On the same rows the activation codes of qvla_rotate_quantize
are held to the end-to-end bound: at most 1e-5 of them differ from the oracle's, each by +-1 and
only next to a rounding tie."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu

SWEEP_M = (1, 16, 50, 256, 816, 3200, 8192)
SWEEP_KN = ((1024, 1024), (1024, 4096), (2048, 2048), (2048, 16384), (16384, 2048))
ORACLE_ROWS = 40  # sampled rows beyond the first and the last


@pytest.fixture(scope="module")
def sweep_layers():
    """One packed layer per (K, N) with a bias: W ~ N(0, 1/K), Hadamard K (2048 blocks at K = 16384)."""
    made = {}

    def get(k, n):
        if (k, n) not in made:
            case = W.sweep_linear(1, k, n, seed=70 + k // 1024 + n // 1024, xdtype="f16", ydtype="f16",
                                  with_bias=True)
            wq = np.zeros((n, k // 2), np.uint8)
            ws = np.zeros(n, np.float32)
            Q.qvla_pack_weights_host(np.ascontiguousarray(case.w), Q.F32, n, k, had_block=case.had_block, wq=wq,
                                     wscale=ws)
            layer = G.make_layer(wq, ws, case.had_block, "f16", "f16", case.bias)
            made[(k, n)] = (layer, O.unpack_int4(wq), ws, case.had_block, case.bias)
        return made[(k, n)]

    yield get
    for layer, *_ in made.values():
        layer.close()


@pytest.mark.parametrize("K,N", SWEEP_KN)
@pytest.mark.parametrize("M", SWEEP_M)
def test_sweep_point_f16(M, K, N, sweep_layers):
    layer, wcodes, ws, had, bias = sweep_layers(K, N)
    rng = np.random.default_rng(M * 7 + K + N)
    x = W.as_dtype(W.gaussian_with_outliers(rng, M, K, max(1, round(0.005 * K)), 20.0), "f16")
    xg = x.to(G.DEV)
    y = torch.full((M, N), float("nan"), dtype=torch.float16, device=G.DEV)
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.empty(nbytes, dtype=torch.uint8, device=G.DEV)
    Q.qvla_w4a4_linear(layer, xg, M, -1, y, work, nbytes, G.stream())
    Q.qvla_check_device(G.stream())
    if M <= ORACLE_ROWS + 2:
        rows = np.arange(M)
    else:
        rows = np.unique(np.concatenate([[0, M - 1], rng.choice(np.arange(1, M - 1), ORACLE_ROWS, replace=False)]))
    rows_t = torch.from_numpy(rows).to(G.DEV)
    got = y.index_select(0, rows_t).double().cpu().numpy()
    x_rows = x[torch.from_numpy(rows)]
    ref = O.w4a4_linear(x_rows.double().numpy(), wcodes, ws, had, bias=bias, out_fmt="f16")
    G.assert_linear_close_modulo_ties(got, ref, wcodes, ws, bias, "f16")
    # the activation codes of the same rows (qvla_rotate_quantize over all M rows)
    xq = torch.zeros(M, K // 2, dtype=torch.uint8, device=G.DEV)
    xs = torch.zeros(M, dtype=torch.float32, device=G.DEV)
    Q.qvla_rotate_quantize(layer, xg, M, -1, xq, xs, None, G.stream())
    Q.qvla_check_device(G.stream())
    codes = O.unpack_int4(xq.index_select(0, rows_t).cpu().numpy())
    frac, maxd, tie = G.code_mismatch_report(codes, ref["qx"],
                                             ref["y_rot"].astype(np.float64) / ref["dx"].astype(np.float64)[:, None])
    assert frac <= 1e-5 and maxd <= 1, (frac, maxd)
    assert tie < 1e-4, tie
