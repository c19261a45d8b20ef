"""The allocation-free linear against the ordinary one.

qvla_w4a4_linear_noalloc serves callers that cannot allocate device memory while running (a
robot controller's real-time loop that reserves everything at start-up, or a plug-in whose
host runtime owns all device memory): it takes no workspace and uses the library's fixed
8 MiB scratch instead.  These tests call it through the C ABI twice in a row, with different
inputs, and compare each result with qvla_w4a4_linear on the same input, within the output
tolerance the other parity tests use.  The file sorts last so that a run stopping at the first
failure has already run every other test; it also passes on its own in a fresh process.
"""

import numpy as np
import pytest
import torch

from paper_2605_28803_gb300 import qvla as Q
from paper_2605_28803_gb300 import workloads as W
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def _layer(case, xdt, ydt):
    N, K = case.w.shape
    wq = np.zeros((N, K // 2), np.uint8)
    ws = np.zeros(N, np.float32)
    Q.qvla_pack_weights_host(np.ascontiguousarray(case.w), Q.F32, N, K, had_block=case.had_block, wq=wq, wscale=ws)
    return G.make_layer(wq, ws, case.had_block, xdt, ydt, case.bias)


def _noalloc(layer, x, step, ydt):
    M = x.shape[0]
    y = torch.full((M, layer.N), float("nan"), dtype=G.TORCH_DT[ydt], device=G.DEV)
    Q.qvla_w4a4_linear_noalloc(layer, x.to(G.DEV).contiguous(), M, step, y, G.stream())
    Q.qvla_check_device(G.stream())
    return y.double().cpu().numpy()


def test_noalloc_matches_linear_per_token_two_calls():
    a = W.sweep_linear(816, 2048, 1024, seed=21, xdtype="bf16", ydtype="bf16", with_bias=True)
    b = W.sweep_linear(300, 2048, 1024, seed=22, xdtype="bf16", ydtype="bf16", with_bias=True)
    layer = _layer(a, "bf16", "bf16")
    for x in (a.x, b.x):  # two calls in a row; the second must not see the first's scratch
        got = _noalloc(layer, x, -1, "bf16")
        ref = G.linear(layer, x, ydt="bf16")
        G.assert_output_close(got, ref, "bf16")
    layer.close()


def test_noalloc_matches_linear_per_step_two_calls():
    case = W.single_layer_steps(seed=3, m=64, k=1024, n=512, had_block=1024)
    N, K = case.w.shape
    wq = np.zeros((N, K // 2), np.uint8)
    ws = np.zeros(N, np.float32)
    Q.qvla_pack_weights_host(np.ascontiguousarray(case.w), Q.F32, N, K, rot=np.ascontiguousarray(case.rot),
                             rot_block=case.rot_block, had_block=case.had_block, wq=wq, wscale=ws)
    layer = G.make_layer(wq, ws, case.had_block, "f16", "f16")
    Q.qvla_set_step_scales(layer, np.linspace(0.3, 0.05, 10).astype(np.float32))
    for t in (2, 7):
        got = _noalloc(layer, case.x_steps[t], t, "f16")
        ref = G.linear(layer, case.x_steps[t], step=t, ydt="f16")
        G.assert_output_close(got, ref, "f16")
    layer.close()


def test_noalloc_rejects_more_rows_than_its_scratch_holds():
    case = W.sweep_linear(16, 16384, 256, seed=23, xdtype="bf16", ydtype="bf16")
    layer = _layer(case, "bf16", "bf16")
    too_many = (Q.NOALLOC_SCRATCH_BYTES // (16384 // 2)) + 1  # codes alone exceed the scratch
    x = torch.zeros(too_many, 16384, dtype=torch.bfloat16, device=G.DEV)
    y = torch.zeros(too_many, 256, dtype=torch.bfloat16, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_w4a4_linear_noalloc(layer, x, too_many, -1, y, G.stream())
    assert e.value.status == 2 and "scratch" in str(e.value)
    layer.close()


def test_noalloc_counts_the_online_rotation_in_its_scratch():
    # A layer with an online x.P.BlockDiag(U_b) keeps x' in the scratch as well: 2000 rows of
    # K = 2048 fit without it (operand bytes and sums) but not with 2000 x 2048 bf16 values more.
    # (N = 2560: 16 x 10 tiles of 128 x 256, enough for every SM, so the workspace has no
    # split-of-K part.)
    K, N, M = 2048, 2560, 2000
    case = W.sweep_linear(16, K, N, seed=24, xdtype="bf16", ydtype="bf16")
    layer = _layer(case, "bf16", "bf16")
    assert Q.qvla_linear_workspace_bytes(layer, M) <= Q.NOALLOC_SCRATCH_BYTES
    Q.qvla_layer_set_online_rotation(layer, perm=np.arange(K - 1, -1, -1, dtype=np.int32), rot=None, rot_block=16)
    assert Q.qvla_linear_workspace_bytes(layer, M) > Q.NOALLOC_SCRATCH_BYTES
    x = torch.zeros(M, K, dtype=torch.bfloat16, device=G.DEV)
    y = torch.zeros(M, N, dtype=torch.bfloat16, device=G.DEV)
    with pytest.raises(Q.QvlaError) as e:
        Q.qvla_w4a4_linear_noalloc(layer, x, M, -1, y, G.stream())
    assert e.value.status == 2 and "scratch" in str(e.value)
    layer.close()
