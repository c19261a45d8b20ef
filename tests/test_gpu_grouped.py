"""GPU parity of per-step, per-group activation scales (Eq. 6 read per channel group; Eq. 7 per
group): qvla_w4a4_linear with a [T][G] table against the oracle's grouped linear.

Groups hold max(128, b) channels.  Each group's integer accumulator is corrected exactly and
scaled on the GPU before a float32 sum over the groups, so the outputs agree with the oracle's
float64 sum within the output tolerance (most of them bit for bit).  Covered: both GEMM
orientations (weight-major with split-K over whole groups, token-major with 128-wide tiles),
groups of 1, 2 and 8 k-blocks, a single group, ragged M and N, clamping at +-7, the library's
per-group calibration, and the refusals of the entry points that cannot take such a table."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _profiled_input(rng, m, k, t, steps):
    """Activations whose channel groups differ in spread (a log-normal profile over blocks of 64
    channels, fixed per K) and whose overall scale drifts with the step."""
    prof = np.repeat(np.exp(np.random.default_rng(k).normal(0.0, 0.8, k // 64)), 64).astype(np.float32)
    return (rng.standard_normal((m, k), dtype=np.float32) * prof[None, :] * np.float32(W.dit_input_std(t, steps)))


def _layer(rng, n, k, had, xdt="f16", ydt="f16", bias=True):
    codes = rng.integers(-7, 8, (n, k)).astype(np.int8)
    ws = (rng.uniform(0.5, 2.0, n) * 2 ** -7).astype(np.float32)
    b = (rng.standard_normal(n) * 0.05).astype(np.float32) if bias else None
    return G.make_layer(O.pack_int4(codes), ws, had, xdt, ydt, b), codes, ws, b


def _run(layer, x, step, ydt="f16"):
    return G.linear(layer, x, step=step, ydt=ydt)


@pytest.mark.parametrize("M,K,N,had", [(50, 1024, 1024, 64), (50, 4096, 1024, 128), (16, 1024, 3072, 1024),
                                       (200, 2048, 1024, 64), (1, 512, 256, 1), (130, 1024, 2048, 256),
                                       (64, 2048, 512, 2048), (33, 1024, 400, 64), (300, 1024, 272, 512)])
def test_grouped_linear_matches_oracle(M, K, N, had):
    rng = np.random.default_rng(M + K + N + had)
    layer, codes, ws, bias = _layer(rng, N, K, had)
    T = 3
    cal = [_profiled_input(np.random.default_rng(100 + t), 16, K, t, T) for t in range(T)]
    table = O.calibrate_step_table_grouped(cal, had)
    ng, size = Q.qvla_layer_scale_groups(layer)
    assert (ng, size) == (K // max(128, had), max(128, had)) and table.shape == (T, ng)
    Q.qvla_set_step_group_scales(layer, table)
    assert Q.qvla_layer_info(layer)[3] == T
    for t in range(T):
        x = W.as_dtype(_profiled_input(np.random.default_rng(200 + t), M, K, t, T), "f16")
        got = _run(layer, x, t)
        ref = O.grouped_linear(x.double().numpy(), codes, ws, had, table, t, bias=bias, out_fmt="f16")
        G.assert_output_close(got, ref["y"], "f16")
        assert np.mean(got == ref["y"]) > 0.9
    layer.close()


def test_grouped_clamping_and_library_calibration():
    """A table calibrated by the library (qvla_rotated_absmax_groups) on a 16-row draw, then an
    evaluation draw that exceeds it: codes clamp at +-7 in some groups."""
    M, K, N, had, T = 50, 1024, 1024, 64, 4
    rng = np.random.default_rng(5)
    layer, codes, ws, bias = _layer(rng, N, K, had)
    table = np.zeros((T, K // 128), np.float32)
    for t in range(T):
        xc = W.as_dtype(_profiled_input(np.random.default_rng(300 + t), 16, K, t, T), "f16")
        peak = torch.zeros(K // 128, dtype=torch.float32, device=G.DEV)
        Q.qvla_rotated_absmax_groups(xc.to(G.DEV), Q.F16, 16, K, had, peak, G.stream())
        lib = peak.cpu().numpy()
        ref = O.calibrate_step_table_grouped([xc.double().numpy()], had)[0] * np.float32(7)
        assert np.allclose(lib, ref, rtol=4e-7, atol=0)
        table[t] = lib / np.float32(7)
    Q.qvla_set_step_group_scales(layer, table)
    clamped = 0
    for t in range(T):
        x = W.as_dtype(_profiled_input(np.random.default_rng(400 + t), M, K, t, T), "f16")
        ref = O.grouped_linear(x.double().numpy(), codes, ws, had, table, t, bias=bias, out_fmt="f16")
        clamped += int(np.count_nonzero(np.abs(ref["qx"]) == 7))
        G.assert_output_close(_run(layer, x, t), ref["y"], "f16")
    assert clamped > 0
    layer.close()


def test_grouped_bf16_output_and_step_range():
    M, K, N, had = 40, 2048, 768, 128
    rng = np.random.default_rng(6)
    layer, codes, ws, bias = _layer(rng, N, K, had, "bf16", "bf16", bias=False)
    table = (rng.uniform(0.05, 0.5, (2, K // 128))).astype(np.float32)
    Q.qvla_set_step_group_scales(layer, table)
    x = W.as_dtype(_profiled_input(rng, M, K, 1, 2), "bf16")
    ref = O.grouped_linear(x.double().numpy(), codes, ws, had, table, 1, out_fmt="bf16")
    G.assert_output_close(_run(layer, x, 1, "bf16"), ref["y"], "bf16")
    with pytest.raises(Q.QvlaError) as e:
        _run(layer, x, 2, "bf16")
    assert e.value.status == 5
    layer.close()


def test_grouped_table_rules():
    """Per-token calls are unaffected by a grouped table; the table's width must be the layer's
    group count; a per-step table replaces a grouped one; the entry points without a step path
    for groups refuse it; gated layers take no grouped table."""
    M, K, N, had = 20, 1024, 256, 64
    rng = np.random.default_rng(7)
    layer, codes, ws, bias = _layer(rng, N, K, had)
    table = rng.uniform(0.05, 0.5, (2, 8)).astype(np.float32)
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_set_step_group_scales(layer, table[:, :4])
    assert e.value.status == 1
    Q.qvla_set_step_group_scales(layer, table)
    x = W.as_dtype(_profiled_input(rng, M, K, 0, 2), "f16")
    ref = O.w4a4_linear(x.double().numpy(), codes, ws, had, bias=bias, out_fmt="f16")
    G.assert_output_close(_run(layer, x, -1), ref["y"], "f16")  # per token
    nb = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.empty(nb, dtype=torch.uint8, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_linear_quantize(layer, x.to(G.DEV), M, 0, work, nb, G.stream())
    assert e.value.status == 2
    xq = torch.zeros(M, K // 2, dtype=torch.uint8, device=G.DEV)
    xs = torch.zeros(M, dtype=torch.float32, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_rotate_quantize(layer, x.to(G.DEV), M, 0, xq, xs, None, G.stream())
    assert e.value.status == 2
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_w4a8_linear(layer, x.to(G.DEV), M, 0, torch.zeros(M, N, dtype=torch.float16, device=G.DEV), work,
                           nb, G.stream())
    assert e.value.status in (1, 2)
    tab1 = np.array([0.2, 0.3], np.float32)
    Q.qvla_set_step_scales(layer, tab1)  # back to one scale per step
    ref = O.w4a4_linear(x.double().numpy(), codes, ws, had, bias=bias, table=tab1, step=1, out_fmt="f16")
    G.assert_output_close(_run(layer, x, 1), ref["y"], "f16")
    layer.close()
    gq = O.pack_int4(rng.integers(-7, 8, (128, K)).astype(np.int8))
    gl = Q.qvla_layer_create_gated(128, K, had, Q.F16, Q.F16, gq, np.ones(128, np.float32), gq,
                                   np.ones(128, np.float32))
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_set_step_group_scales(gl, table)
    assert e.value.status == 2
    gl.close()
