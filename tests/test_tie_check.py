"""The tie-aware output check of the GPU parity tests, exercised on the CPU with the oracle alone:
outputs that differ from the oracle's only through activation codes moved by one step at a
rounding tie pass; a code moved away from a tie, or moved by two steps, fails."""

import numpy as np
import pytest

from oracle import qvla_oracle as O
from tests import gpu_helpers as G


def _case(seed=3, m=6, k=256, n=96):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((m, k))
    wcodes = rng.integers(-7, 8, (n, k)).astype(np.int8)
    ws = (rng.uniform(0.5, 1.5, n) * 0.01).astype(np.float32)
    bias = (rng.standard_normal(n) * 0.05).astype(np.float32)
    delta = np.float32(np.abs(O.rotate_activations(x, k)).max() / 7)  # a per-step scale
    return x, wcodes, ws, bias, delta, (2, 17)  # the tie goes on rotated value (2, 17)


def _ref_with_tie():
    x, wcodes, ws, bias, delta, (r, kk) = _case()
    ref = O.w4a4_linear(x, wcodes, ws, 256, bias=bias, table=np.array([delta]), step=0, out_fmt="f16")
    # move the chosen rotated value onto a tie (k + 0.5) Delta exactly, and requantise that row
    t = ref["y_rot"][r, kk] / np.float32(delta)
    half = np.float32((np.floor(t) + 0.5) * np.float64(delta))
    ref["y_rot"][r, kk] = half
    ref["qx"][r] = O.quantize(ref["y_rot"][r:r + 1], np.full((1, 1), delta, np.float32))[0]
    acc = O.int_gemm(ref["qx"], wcodes)
    ref["y"] = O.dequant_output(acc, ref["dx"], ws, bias, "f16")
    return ref, wcodes, ws, bias, r, kk


def _moved(ref, wcodes, ws, bias, r, kk, step):
    q = ref["qx"].astype(np.int64).copy()
    q[r, kk] += step
    return O.dequant_output(O.int_gemm(q, wcodes), ref["dx"], ws, bias, "f16")


def test_a_code_moved_across_its_tie_passes():
    ref, wcodes, ws, bias, r, kk = _ref_with_tie()
    t = np.float64(ref["y_rot"][r, kk]) / np.float64(ref["dx"][r])
    step = 1 if ref["qx"][r, kk] == np.floor(t) else -1
    got = _moved(ref, wcodes, ws, bias, r, kk, step)
    assert np.any(np.abs(got - ref["y"]) > 2e-3 * np.abs(ref["y"]).max())  # the plain check would fail
    adj = G.assert_linear_close_modulo_ties(got, ref, wcodes, ws, bias, "f16", max_flip_frac=1.0)
    assert np.array_equal(adj[r], got[r])


@pytest.mark.parametrize("which", ["away_from_tie", "two_steps"])
def test_other_code_changes_fail(which):
    ref, wcodes, ws, bias, r, kk = _ref_with_tie()
    if which == "away_from_tie":
        t = ref["y_rot"][r].astype(np.float64) / np.float64(ref["dx"][r])
        far = int(np.argmax(np.abs(t - np.floor(t) - 0.5) * (np.abs(t) < 6)))  # nearest to an integer: no tie
        got = _moved(ref, wcodes, ws, bias, r, far, 1)
    else:
        got = _moved(ref, wcodes, ws, bias, r, kk, 2)
    with pytest.raises(AssertionError):
        G.assert_linear_close_modulo_ties(got, ref, wcodes, ws, bias, "f16", max_flip_frac=1.0)
