"""The device-side failure path: a bounded wait that runs out.

A test hook (include/qvla_debug.h) makes the GEMM's load warp issue no copy and shortens the wait
limit to 20 ms, so the converters' waits for the staged tiles, the MMA thread's wait for the
expanded tiles and the epilogue's wait for the accumulator all run out.  The kernel must record
QVLA_ERR_TIMEOUT, issue no MMA, leave the output untouched and return; qvla_check_device reports
it once and clears it, and the next launch is bit-exact.  The held kernel has no copy, MMA or
asynchronous store outstanding when it returns (it is the token-major single-CTA form: no cluster
exchange), so nothing faults or hangs."""

import numpy as np
import pytest
import torch

from oracle import qvla_oracle as O
from paper_2605_28803_gb300 import qvla as Q
from tests import gpu_helpers as G

pytestmark = pytest.mark.gpu


def test_a_wait_that_runs_out_reports_timeout_and_the_next_launch_is_clean():
    rng = np.random.default_rng(61)
    M, K, N = 256, 512, 256
    wcodes = rng.integers(-7, 8, (N, K)).astype(np.int8)
    layer = G.make_layer(O.pack_int4(wcodes), np.full(N, 0.01, np.float32), 512, "f16", "f16")
    xcodes = rng.integers(-7, 8, (M, K)).astype(np.int8)
    xq, xs = O.pack_int4(xcodes), np.full(M, 0.02, np.float32)
    xsum = xcodes.astype(np.int64).sum(1)
    y0, acc0 = G.gemm(layer, xq, xs, xsum)
    assert np.array_equal(acc0, O.int_gemm(xcodes, wcodes))

    xqg = torch.from_numpy(xq).to(G.DEV)
    xsg = torch.from_numpy(xs).to(G.DEV)
    xsumg = torch.from_numpy(xsum.astype(np.int32)).to(G.DEV)
    y = torch.full((M, N), float("nan"), dtype=torch.float16, device=G.DEV)
    Q.qvla_check_device(G.stream())
    Q.qvla_debug_set_hooks(20_000_000, True)
    try:
        Q.qvla_gemm_w4a4(layer, xqg, xsg, xsumg, M, y, None, G.stream())
        with pytest.raises(Q.QvlaError) as e:
            Q.qvla_check_device(G.stream())
        assert e.value.status == 6
        assert torch.isnan(y).all().item()  # nothing was written
    finally:
        Q.qvla_debug_set_hooks(0, False)
    Q.qvla_check_device(G.stream())  # the error word was cleared by the first check
    y1, acc1 = G.gemm(layer, xq, xs, xsum)
    assert np.array_equal(acc1, acc0) and np.array_equal(y1, y0)
    layer.close()


@pytest.mark.parametrize("M", [1, 2])
def test_a_decode_gemv_wait_that_runs_out(M):
    """The decode GEMV split over a cluster of CTAs: with the hook, no CTA sends its row maximum
    (one launch, M = 1, K = 16384) or its partial sums (M = 1 and 2), so every receiving wait runs
    out.  No asynchronous store is issued, so none is outstanding when the CTAs return.  The
    kernel reports QVLA_ERR_TIMEOUT, writes nothing, and the next call is bit-exact."""
    rng = np.random.default_rng(67 + M)
    N, K = 2048, 16384
    wcodes = rng.integers(-8, 8, (N, K)).astype(np.int8)
    layer = G.make_layer(O.pack_int4(wcodes), np.full(N, 2 ** -9, np.float32), 2048, "bf16", "bf16")
    x = torch.from_numpy(rng.standard_normal((M, K), dtype=np.float32)).to(torch.bfloat16)
    y0 = G.linear(layer, x, ydt="bf16")
    xg = x.to(G.DEV)
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.empty(nbytes, dtype=torch.uint8, device=G.DEV)
    y = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device=G.DEV)
    Q.qvla_check_device(G.stream())
    Q.qvla_debug_set_hooks(20_000_000, True)
    try:
        Q.qvla_w4a4_linear(layer, xg, M, -1, y, work, nbytes, G.stream())
        with pytest.raises(Q.QvlaError) as e:
            Q.qvla_check_device(G.stream())
        assert e.value.status == 6
        assert torch.isnan(y).all().item()
    finally:
        Q.qvla_debug_set_hooks(0, False)
    Q.qvla_check_device(G.stream())
    assert np.array_equal(G.linear(layer, x, ydt="bf16"), y0)
    layer.close()


def test_a_rotate_quantize_pass_wait_that_runs_out():
    """The few-row rotate-quantise kernel with a row of 8 passes in a cluster: with the hook, no pass
    sends its maximum or its code sum, so the waits run out; the launch reports QVLA_ERR_TIMEOUT
    and returns with no asynchronous store outstanding, and the next call is bit-exact."""
    rng = np.random.default_rng(71)
    M, K = 2, 16384
    layer = G.make_layer(np.zeros((16, K // 2), np.uint8), np.ones(16, np.float32), 2048, "bf16", "bf16")
    x = torch.from_numpy(rng.standard_normal((M, K), dtype=np.float32)).to(torch.bfloat16).to(G.DEV)
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    ref = torch.zeros(nbytes, dtype=torch.uint8, device=G.DEV)
    Q.qvla_linear_quantize(layer, x, M, -1, ref, nbytes, G.stream())
    Q.qvla_check_device(G.stream())
    work = torch.zeros(nbytes, dtype=torch.uint8, device=G.DEV)
    Q.qvla_debug_set_hooks(20_000_000, True)
    try:
        Q.qvla_linear_quantize(layer, x, M, -1, work, nbytes, G.stream())
        with pytest.raises(Q.QvlaError) as e:
            Q.qvla_check_device(G.stream())
        assert e.value.status == 6
    finally:
        Q.qvla_debug_set_hooks(0, False)
    Q.qvla_check_device(G.stream())
    work.zero_()
    Q.qvla_linear_quantize(layer, x, M, -1, work, nbytes, G.stream())
    Q.qvla_check_device(G.stream())
    assert torch.equal(work, ref)  # codes, scales and sums (the padding is zero in both)
    layer.close()
