"""Pins of the CPU oracle to things other than itself (CPU only).

The paper prints no worked numeric example, so every oracle function is pinned by one
or more of: a hand-worked fixture under tests/golden/, a library routine it reduces to
in a special case, a closed form or invariant the paper states, or brute force on tiny
inputs.  Each pin is a ``check_*`` function of the oracle module; ``test_mutants``
plants plausible mistakes in the oracle (on the CPU) and shows that some pin fails.
"""

import math

import numpy as np
import pytest
import scipy.linalg
import scipy.special
import torch

from oracle import qvla_oracle as O
from tests.conftest import read_golden


# --------------------------------------------------------------------------------------
# Pins
# --------------------------------------------------------------------------------------

def check_hadamard_matches_scipy(o):
    """Sylvester order (reading R1) is what scipy.linalg.hadamard builds."""
    for n in [1, 2, 4, 8, 64, 512, 2048]:
        assert np.array_equal(o.sylvester_hadamard(n), scipy.linalg.hadamard(n)), n


def check_hadamard_orthogonal(o):
    """H H^T = n I exactly (Sec. 4.1: normalised H is orthogonal)."""
    for n in [2, 16, 256, 1024]:
        h = o.sylvester_hadamard(n).astype(np.float64)
        assert np.array_equal(h @ h.T, n * np.eye(n)), n


def check_hadamard_golden(o):
    g = read_golden("hadamard4.txt")
    h4 = np.array([[int(v) for v in r] for r in g["_rows"]])
    assert np.array_equal(o.sylvester_hadamard(4), h4)
    assert np.allclose(o.normalized_hadamard(4), h4 / 2.0, rtol=0, atol=0)


def check_rotate_matches_library_blockdiag(o):
    """Block rotation = x . scipy block_diag(H_b/sqrt(b), ...) (Eq. 4 with U = I)."""
    rng = np.random.default_rng(11)
    for k, b in [(64, 16), (512, 512), (1024, 256), (96, 32)]:
        x = rng.standard_normal((5, k))
        r = scipy.linalg.block_diag(*([scipy.linalg.hadamard(b) / math.sqrt(b)] * (k // b)))
        assert np.allclose(o.block_hadamard_rotate(x, b), x @ r, rtol=1e-12, atol=1e-12), (k, b)


def check_rotate_linf_bound(o):
    """The Fig. 2 caption bounds ||z H||_inf by ||z||_2 / sqrt(n).  As printed that fails
    (z = ones gives sqrt(n) against 1); what holds is ||z H||_inf <= ||z||_1 / sqrt(n),
    which equals ||z||_2 / sqrt(n) for a single dominant channel (one-hot z), the case
    Sec. 4.1 describes.  Also: H preserves the 2-norm and is an involution."""
    rng = np.random.default_rng(12)
    for n in [8, 128, 2048]:
        z = rng.standard_normal((20, n))
        z[:, 3] *= 50.0
        y = o.block_hadamard_rotate(z, n)
        assert np.all(np.max(np.abs(y), axis=1) <= np.sum(np.abs(z), axis=1) / math.sqrt(n) * (1 + 1e-12))
        ones = o.block_hadamard_rotate(np.ones((1, n)), n)
        assert np.isclose(np.max(np.abs(ones)), math.sqrt(n))  # the printed 2-norm form fails here
        assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(z, axis=1), rtol=1e-12)
        assert np.allclose(o.block_hadamard_rotate(y, n), z, rtol=1e-11, atol=1e-11)
        e = np.zeros((1, n))
        e[0, 5] = 3.0
        ye = o.block_hadamard_rotate(e, n)
        assert np.allclose(np.abs(ye), 3.0 / math.sqrt(n), rtol=1e-14)
        assert np.allclose(ye[0], 3.0 * scipy.linalg.hadamard(n)[5] / math.sqrt(n), rtol=1e-14)


def check_rotation_invariance(o):
    """Y = XW = (XR)(R^T W) for orthogonal R (Sec. 4.1), with R = P . BlockDiag(U_b) .
    BlockDiag(H).  The activation side is built here from explicit matrices (a
    permutation matrix and scipy's block_diag), independently of the oracle, so a weight
    fold that disagrees with the upstream transform (e.g. U^T for U) fails."""
    rng = np.random.default_rng(13)
    k, n, m = 256, 48, 9
    x = rng.standard_normal((m, k))
    w = rng.standard_normal((n, k))
    perm = rng.permutation(k)
    rot = np.stack([np.linalg.qr(rng.standard_normal((64, 64)))[0] for _ in range(k // 64)])
    pmat = np.eye(k)[:, perm]                      # (x P)[j] = x[perm[j]]
    umat = scipy.linalg.block_diag(*rot)
    x_up = x @ pmat @ umat
    assert np.allclose(o.upstream_activation_transform(x, perm, rot, 64), x_up, rtol=1e-12, atol=1e-12)
    for had in [64, 256]:
        hmat = scipy.linalg.block_diag(*([scipy.linalg.hadamard(had) / math.sqrt(had)] * (k // had)))
        xr = x_up @ hmat
        wr = o.fold_weights(w, had, perm, rot, 64)
        ref = x @ w.T
        assert np.allclose(xr @ wr.T, ref, rtol=1e-11, atol=1e-11 * np.abs(ref).max())
        assert np.allclose(wr, w @ pmat @ umat @ hmat, rtol=1e-11, atol=1e-11)
        assert not np.allclose(xr, x)


def check_zigzag_golden(o):
    g = read_golden("zigzag_worked.txt")
    w = np.array([[float(v) for v in g["w"]]])
    perm = o.zigzag_permutation(w, int(g["block"][0]))
    assert perm.tolist() == [int(v) for v in g["perm"]]
    energy = (w * w).sum(axis=0)
    assert [energy[perm[:4]].sum(), energy[perm[4:]].sum()] == [float(v) for v in g["block_energy"]]


def check_zigzag_rule(o):
    """The i-th channel of the energy order lands in block i mod 2nb, or 2nb - 1 - (i mod 2nb)
    past the turn (the zigzag written as one index formula), in dealing order; the result is a
    permutation and spreads energy more evenly than contiguous blocks of the sorted list."""
    rng = np.random.default_rng(21)
    for k, block in [(256, 64), (64, 8), (96, 32)]:
        w = rng.standard_normal((40, k)) * rng.uniform(0.1, 5.0, k)[None, :]
        perm = o.zigzag_permutation(w, block)
        assert sorted(perm.tolist()) == list(range(k))
        nb = k // block
        energy = (w * w).sum(axis=0)
        order = sorted(range(k), key=lambda j: (-energy[j], j))
        expect = [[] for _ in range(nb)]
        for i, j in enumerate(order):
            t = i % (2 * nb)
            expect[t if t < nb else 2 * nb - 1 - t].append(j)
        assert perm.tolist() == [j for blk in expect for j in blk]
        be = energy[perm].reshape(nb, block).sum(axis=1)
        bc = np.sort(energy)[::-1].reshape(nb, block).sum(axis=1)
        assert be.max() - be.min() < bc.max() - bc.min()


def check_block_svd_golden(o):
    g = read_golden("svd_worked.txt")
    w = np.array([[float(v) for v in g["w_row0"]], [float(v) for v in g["w_row1"]]])
    u = np.array([[float(v) for v in g["u_times_sqrt10_row0"]], [float(v) for v in g["u_times_sqrt10_row1"]]])
    rot = o.block_svd_rotation(w, 2)
    assert np.allclose(rot[0], u / math.sqrt(10.0), rtol=0, atol=1e-14)
    rows = rot[0].T @ w.T
    assert np.allclose((rows * rows).sum(axis=1), [float(v) for v in g["sigma_squared"]], rtol=1e-13)


def check_block_svd_properties(o):
    """Each U_b is orthogonal; the rows of U_b^T W_b carry energies sigma_i^2 in descending
    order (Sec. 4.1: the rotated block's row energy is its singular spectrum), with sigma from
    scipy's svdvals; the largest entry of every column is positive; and the composite fold
    with P and these U_b still preserves X W^T."""
    rng = np.random.default_rng(22)
    k, n, block = 128, 48, 32
    w = rng.standard_normal((n, k)) * rng.uniform(0.2, 3.0, k)[None, :]
    perm = o.zigzag_permutation(w, block)
    rot = o.block_svd_rotation(w, block, perm)
    wp = w[:, perm]
    for b in range(k // block):
        u = rot[b]
        assert np.allclose(u.T @ u, np.eye(block), atol=1e-13)
        wb = wp[:, b * block:(b + 1) * block].T
        rows = u.T @ wb
        sig = scipy.linalg.svdvals(wb)
        assert np.allclose((rows * rows).sum(axis=1), sig ** 2, rtol=1e-10)
        idx = np.argmax(np.abs(u), axis=0)
        assert np.all(u[idx, np.arange(block)] > 0)
    x = rng.standard_normal((5, k))
    xr = o.block_hadamard_rotate(o.upstream_activation_transform(x, perm, rot, block), 64)
    wr = o.fold_weights(w, 64, perm, rot, block)
    ref = x @ w.T
    assert np.allclose(xr @ wr.T, ref, rtol=1e-11, atol=1e-11 * np.abs(ref).max())


def check_quantizer_8bit_bruteforce(o):
    """k = 8 (q_max = 127, Eq. 5): Delta = max / 127 and each code is the nearest candidate in
    [-127, 127], ties to even, by exhaustive search in exact float64 arithmetic."""
    rng = np.random.default_rng(23)
    z = (rng.standard_normal(3000) * 5).astype(np.float32)
    z[:4] = [0.5, -1.5, 2.5, 3.5]
    d = o.absmax_scale(z, qmax=127)
    assert d == np.float32(np.float32(np.max(np.abs(z))) / np.float32(127))
    codes = o.quantize(z, np.float32(1.0), 127)
    assert codes[:4].tolist() == [0, -2, 2, 4]
    q = o.quantize(z, d, 127)
    cand = np.arange(-127, 128, dtype=np.float64)
    t = z.astype(np.float64) / np.float64(d)
    dist = np.abs(t[:, None] - cand[None, :])
    best = dist.min(axis=1)
    for i in range(len(z)):
        c = cand[dist[i] == best[i]]
        expect = c[0] if len(c) == 1 else c[np.argmin(np.abs(c) % 2)]
        assert q[i] == expect
    assert q.min() >= -127 and q.max() <= 127 and np.count_nonzero(np.abs(q) == 127) >= 1


def check_w4a8_linear(o):
    """The W4A8 linear is the same recipe with 8-bit activation codes: its integer product is
    the exhaustive sum of int8 x int4 codes, and on outlier-heavy data it approximates the
    float product better than W4A4."""
    rng = np.random.default_rng(24)
    m, n, k, had = 6, 10, 64, 64
    x = rng.standard_normal((m, k))
    x[:, 3] *= 20
    w = rng.standard_normal((n, k)) * 0.05
    _, ws, wc = o.pack_weights(w, had)
    r8 = o.w4a4_linear(x, wc, ws, had, out_fmt="f32", act_bits=8)
    r4 = o.w4a4_linear(x, wc, ws, had, out_fmt="f32", act_bits=4)
    assert np.abs(r8["qx"]).max() == 127 and np.abs(r4["qx"]).max() == 7
    acc = np.zeros((m, n), dtype=np.int64)
    for i in range(m):
        for j in range(n):
            acc[i, j] = sum(int(r8["qx"][i, t]) * int(wc[j, t]) for t in range(k))
    assert np.array_equal(r8["acc"], acc)
    ref = x @ w.T
    assert o.relative_output_error(r8["y"], ref) < o.relative_output_error(r4["y"], ref)


def check_quantizer_golden(o):
    g = read_golden("quantizer_worked.txt")
    z = np.array([float(v) for v in g["z"]], dtype=np.float32)
    d = o.absmax_scale(z)
    assert d == np.float32(g["delta"][0])
    assert np.array_equal(o.quantize(z, d), np.array([int(v) for v in g["codes"]]))
    ds = np.float32(g["step_delta"][0])
    assert np.array_equal(o.quantize(z, ds), np.array([int(v) for v in g["step_codes"]]))


def check_quantizer_bruteforce(o):
    """Each code is the candidate in [-7, 7] nearest to z / Delta, ties to the even one
    (Eq. 6 with reading R4), found by exhaustive search with exact float64 arithmetic."""
    rng = np.random.default_rng(14)
    z = (rng.standard_normal(4000) * 3).astype(np.float32)
    # exact ties and clamped values
    z[:40] = (np.arange(-20, 20) + 0.5).astype(np.float32) * np.float32(0.5)
    for d in [np.float32(0.5), np.float32(0.37), np.float32(1.3)]:
        q = o.quantize(z, d)
        cand = np.arange(-7, 8, dtype=np.float64)
        dist = np.abs(z.astype(np.float64)[:, None] - np.float64(d) * cand[None, :])  # exact
        best = dist.min(axis=1, keepdims=True)
        ok = dist == best
        # among equally near candidates take the even one
        choice = np.where(ok.sum(1) > 1, np.where(ok & (cand[None, :] % 2 == 0), cand[None, :], 99).min(1),
                          cand[np.argmax(ok, axis=1)])
        assert np.array_equal(q, choice.astype(np.int8)), d


def check_quantizer_bounds(o):
    """Codes lie in [-7, 7]; |z - Delta q| <= Delta/2 where no clamp applies; the
    per-token maximum maps to +-7; an all-zero row has Delta = 0 and codes 0."""
    rng = np.random.default_rng(15)
    y = (rng.standard_normal((30, 256)) * rng.uniform(0.1, 10, (30, 1))).astype(np.float32)
    y[7] = 0.0
    q, d = o.quantize_activations_per_token(y)
    assert q.min() >= -7 and q.max() <= 7
    err = np.abs(y.astype(np.float64) - d.astype(np.float64)[:, None] * q)
    assert np.all(err <= d.astype(np.float64)[:, None] / 2 * (1 + 1e-6))
    am = np.argmax(np.abs(y), axis=1)
    for r in range(30):
        if r == 7:
            assert d[r] == 0 and np.all(q[r] == 0)
        else:
            assert abs(int(q[r, am[r]])) == 7


def check_pack_golden_and_roundtrip(o):
    g = read_golden("pack_worked.txt")
    codes = np.array([int(v) for v in g["codes"]], dtype=np.int8)
    want = np.array([int(v, 16) for v in g["bytes"]], dtype=np.uint8)
    assert np.array_equal(o.pack_int4(codes), want)
    allc = np.array([[a, b] for a in range(-8, 8) for b in range(-8, 8)], dtype=np.int8).reshape(1, -1)
    assert np.array_equal(o.unpack_int4(o.pack_int4(allc)), allc)


def check_int_gemm_bruteforce(o):
    """Exhaustive nested loops on tiny non-square shapes, and the +-7 extremes at K = 16384."""
    rng = np.random.default_rng(16)
    for m, n, k in [(3, 5, 7), (1, 8, 64), (6, 2, 33)]:
        a = rng.integers(-8, 8, (m, k)).astype(np.int8)
        b = rng.integers(-8, 8, (n, k)).astype(np.int8)
        ref = np.zeros((m, n), dtype=np.int64)
        for i in range(m):
            for j in range(n):
                s = 0
                for t in range(k):
                    s += int(a[i, t]) * int(b[j, t])
                ref[i, j] = s
        got = o.int_gemm(a, b)
        assert got.shape == (m, n) and np.array_equal(got, ref), (m, n, k)
    k = 16384
    a = np.full((2, k), 7, np.int8)
    a[1] = -7
    b = np.full((3, k), 7, np.int8)
    b[2, ::2] = -7
    got = o.int_gemm(a, b)
    assert np.array_equal(got, np.array([[49 * k, 49 * k, 0], [-49 * k, -49 * k, 0]]))


def check_round_to_format(o):
    """Single round-to-nearest-even into f16 / f32 agrees with numpy's direct float64
    conversions; into bf16 it agrees with torch's float32 -> bfloat16 conversion."""
    rng = np.random.default_rng(17)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.uniform(-9, 5, 20000),
                        [65504.0, 65519.99, 65520.0, -70000.0, 6e-8, 3e-8, 2.9e-8, 0.0, 1.0 + 2 ** -11, 1.0 + 3 * 2 ** -11]])
    assert np.array_equal(o.round_to_format(x, "f16"), x.astype(np.float16).astype(np.float64))
    assert np.array_equal(o.round_to_format(x, "f32"), x.astype(np.float32).astype(np.float64))
    x32 = x.astype(np.float32)
    tb = torch.from_numpy(x32).to(torch.bfloat16).double().numpy()
    assert np.array_equal(o.round_to_format(x32.astype(np.float64), "bf16"), tb)


def check_linear_golden(o):
    """The hand-worked W4A4 linear (K = 4, H_4, two output channels)."""
    g = read_golden("linear_worked.txt")
    x = np.array([[float(v) for v in g["x"]]])
    w = np.array([[float(v) for v in g["w0"]], [float(v) for v in g["w1"]]])
    packed, wscale, wcodes = o.pack_weights(w, 4)
    assert np.array_equal(wcodes[0], [int(v) for v in g["qw0"]])
    assert np.array_equal(wcodes[1], [int(v) for v in g["qw1"]])
    r = o.w4a4_linear(x, wcodes, wscale, 4, out_fmt="f16")
    assert np.array_equal(r["qx"][0], [int(v) for v in g["qx"]])
    assert np.array_equal(r["acc"][0], [int(v) for v in g["acc"]])
    assert np.array_equal(r["y"][0], [float(v) for v in g["y_f16"]])


def check_dequant_special_cases(o):
    """Delta_x = Delta_w = 1 and no bias gives fp16(acc) exactly for |acc| <= 2048; a zero
    activation scale gives the bias alone."""
    acc = np.arange(-2048, 2049, dtype=np.int64).reshape(1, -1)
    y = o.dequant_output(acc, np.ones(1, np.float32), np.ones(acc.shape[1], np.float32), None, "f16")
    assert np.array_equal(y, acc.astype(np.float64))
    bias = np.linspace(-3, 3, 7).astype(np.float32)
    y = o.dequant_output(np.full((2, 7), 1234, np.int64), np.zeros(2, np.float32), np.ones(7, np.float32), bias, "f32")
    assert np.array_equal(y, np.broadcast_to(bias.astype(np.float64), (2, 7)))
    y = o.dequant_output(np.full((1, 7), 3, np.int64), np.full(1, 0.5, np.float32), np.full(7, 0.25, np.float32), bias, "f32")
    assert np.allclose(y, 0.375 + bias.astype(np.float64), rtol=1e-7)


def check_step_lookup(o):
    """The scale of step t is table[t], exactly; t outside [0, T) is an error; per-step
    codes are Eq. 6 with that scale."""
    table = np.array([0.1, 0.2, 0.3, 0.4], dtype=np.float32)
    for t in range(4):
        assert o.step_scale_lookup(table, t) == table[t]
    for t in (-1, 4):
        with pytest.raises(IndexError):
            o.step_scale_lookup(table, t)
    y = np.linspace(-2, 2, 64, dtype=np.float32).reshape(2, 32)
    q, d = o.quantize_activations_per_step(y, table, 2)
    assert np.all(d == table[2])
    assert np.array_equal(q, o.quantize(y, np.float32(table[2])))


def check_calibration(o):
    """A table calibrated by absmax on X_t (Eq. 6, per-tensor reading) maps the largest
    rotated entry of X_t to +-7 and clamps nothing; q999 <= absmax; a different draw can clamp."""
    rng = np.random.default_rng(18)
    xs = [rng.standard_normal((16, 128)) * (1 + 0.3 * t) for t in range(4)]
    table = o.calibrate_step_table(xs, 128)
    assert table.dtype == np.float32 and table.shape == (4,)
    for t, x in enumerate(xs):
        y = o.rotate_activations(x, 128)
        assert table[t] == np.float32(np.max(np.abs(y))) / np.float32(7)
        q, _ = o.quantize_activations_per_step(y, table, t)
        assert np.abs(q).max() == 7
        assert np.count_nonzero(np.abs(y.astype(np.float64) / np.float64(table[t])) > 7.5) == 0
    t999 = o.calibrate_step_table(xs, 128, "q999")
    assert np.all(t999 <= table) and np.all(t999 > 0.5 * table)
    other = [rng.standard_normal((16, 128)) * 3.0]
    y = o.rotate_activations(other[0], 128)
    q, _ = o.quantize_activations_per_step(y, t999, 0)
    assert np.count_nonzero(np.abs(y / t999[0]) > 7.5) > 0 and np.abs(q).max() == 7


def check_weight_roundtrip(o):
    """Per-channel RTN: |W' - Delta_w q| <= Delta_w / 2 for every folded weight."""
    rng = np.random.default_rng(19)
    w = rng.standard_normal((40, 256)) * 0.02
    wf = o.fold_weights(w, 64)
    packed, scale, codes = o.pack_weights(w, 64)
    wf32 = wf.astype(np.float32).astype(np.float64)
    assert np.all(np.abs(wf32 - scale.astype(np.float64)[:, None] * codes) <= scale.astype(np.float64)[:, None] / 2 * (1 + 1e-6))
    assert np.array_equal(o.unpack_int4(packed), codes)


def check_end_to_end_band(o):
    """Relative output error ||Y_q - XW^T||_F / ||XW^T||_F of the whole W4A4 linear lies in a
    sane band for Gaussian data with outlier channels, and the Hadamard rotation lowers it
    (Sec. 4.1: H spreads activation outliers; the Table 4 ablation direction)."""
    rng = np.random.default_rng(20)
    m, k, n = 64, 512, 256
    x = rng.standard_normal((m, k))
    x[:, rng.choice(k, 4, replace=False)] *= 20
    w = rng.standard_normal((n, k)) / math.sqrt(k)
    ref = x @ w.T
    errs = {}
    for had in (1, 512):
        _, ws, wc = o.pack_weights(w, had)
        r = o.w4a4_linear(x, wc, ws, had, out_fmt="f32")
        errs[had] = o.relative_output_error(r["y"], ref)
    assert 0.02 < errs[512] < 0.25, errs
    assert errs[512] < 0.7 * errs[1], errs


def _correlated_calibration(rng, n, k, mix=0.6):
    """Calibration rows with correlated channels: Z (I + mix A), Z and A Gaussian."""
    a = rng.standard_normal((k, k)) / np.sqrt(k)
    return rng.standard_normal((n, k)) @ (np.eye(k) + mix * a)


def check_gptq_two_columns_closed_form(o):
    """K = 2: after column 0 is rounded, column 1 absorbs its error d0 = w0 - Delta q0 as
    w1 + d0 H01 / H11 (minimising the quadratic error over the free column), on the damped H."""
    rng = np.random.default_rng(31)
    for _ in range(20):
        w = rng.standard_normal((5, 2))
        x = _correlated_calibration(rng, 40, 2, mix=1.5)
        h = o.gptq_hessian(x)
        codes, scale = o.gptq_quantize(w, h, block=2, damp=0.01)
        hd = h + 0.01 * np.mean(np.diag(h)) * np.eye(2)
        w32 = w.astype(np.float32).astype(np.float64)
        d = scale.astype(np.float64)
        q0 = np.clip(np.rint(w32[:, 0] / d), -7, 7)
        w1 = w32[:, 1] + (w32[:, 0] - d * q0) * hd[0, 1] / hd[1, 1]
        q1 = np.clip(np.rint(w1 / d), -7, 7)
        assert np.array_equal(codes[:, 0], q0) and np.array_equal(codes[:, 1], q1)


def check_gptq_identity_hessian_is_rtn(o):
    """With a diagonal Hessian no error crosses columns: GPTQ returns the RTN codes and scales."""
    rng = np.random.default_rng(32)
    w = rng.standard_normal((16, 64))
    h = np.diag(rng.uniform(0.5, 2.0, 64))
    codes, scale = o.gptq_quantize(w, h, block=16)
    rc, rs = o.quantize_weights(w)
    assert np.array_equal(scale, rs) and np.array_equal(codes, rc)


def _obq_sequential(w, h, damp):
    """The GPTQ result restated in the optimal-brain-quantiser form: one row at a time, column i
    rounded, the remaining weights moved by -(w_i - Delta q_i) Hinv[i, :] / Hinv[i, i], and the
    inverse Hessian updated by eliminating i (no Cholesky factor, no blocks)."""
    w = np.asarray(w, dtype=np.float64).astype(np.float32).astype(np.float64)
    k = w.shape[1]
    hd = h + damp * np.mean(np.diag(h)) * np.eye(k)
    out = np.zeros(w.shape, dtype=np.int8)
    for n in range(w.shape[0]):
        d = float(np.float32(np.abs(w[n].astype(np.float32)).max()) / np.float32(7))
        row = w[n].copy()
        hinv = np.linalg.inv(hd)
        for i in range(k):
            q = np.clip(np.rint(row[i] / d), -7, 7) if d > 0 else 0.0
            out[n, i] = int(q)
            row -= (row[i] - d * q) * hinv[i, :] / hinv[i, i]
            hinv = hinv - np.outer(hinv[:, i], hinv[i, :]) / hinv[i, i]
    return out


def check_gptq_matches_obq_sequential(o):
    """The Cholesky-and-blocks GPTQ equals the sequential OBQ elimination on small correlated
    problems, for block sizes 1, 5 and K."""
    rng = np.random.default_rng(33)
    w = rng.standard_normal((6, 12)) * 0.1
    h = o.gptq_hessian(_correlated_calibration(rng, 64, 12, mix=1.0))
    ref = _obq_sequential(w, h, 0.01)
    for block in (1, 5, 12):
        codes, _ = o.gptq_quantize(w, h, block=block, damp=0.01)
        assert np.array_equal(codes, ref), block


def check_gptq_block_invariance_and_loss(o):
    """Batching the updates in blocks does not change the result (block 1, 128, K), and on
    correlated calibration data GPTQ's error tr(dW H dW^T) is below RTN's on every draw."""
    rng = np.random.default_rng(34)
    for seed in range(3):
        r = np.random.default_rng(seed + 100)
        x = o.block_hadamard_rotate(_correlated_calibration(r, 512, 256), 64)
        w = o.block_hadamard_rotate(r.standard_normal((32, 256)) / 16.0, 64)
        h = o.gptq_hessian(x)
        c1, s1 = o.gptq_quantize(w, h, block=1)
        c2, _ = o.gptq_quantize(w, h, block=128)
        c3, _ = o.gptq_quantize(w, h, block=256)
        assert np.array_equal(c1, c2) and np.array_equal(c1, c3)
        rc, rs = o.quantize_weights(w)
        assert np.array_equal(s1, rs)
        lg = o.weight_proxy_loss(w, c1, s1, h)
        lr = o.weight_proxy_loss(w, rc, rs, h)
        assert lg < 0.9 * lr, (lg, lr)
    del rng


def check_gptq_dead_column(o):
    """A calibration channel that is always zero leaves H_kk = 0: that column is dead, its codes
    are 0, and the rest stays finite and within +-7."""
    rng = np.random.default_rng(35)
    x = _correlated_calibration(rng, 64, 32)
    x[:, 5] = 0.0
    w = rng.standard_normal((8, 32))
    h = o.gptq_hessian(x)
    h[5, :] = 0.0
    h[:, 5] = 0.0
    codes, scale = o.gptq_quantize(w, h)
    assert np.all(codes[:, 5] == 0) and np.all(np.abs(codes) <= 7) and np.all(np.isfinite(scale))


def check_grouped_equal_scales_reduce_to_per_tensor(o):
    """With every group of step t at the same scale the grouped linear is the per-tensor one."""
    rng = np.random.default_rng(41)
    x = rng.standard_normal((6, 512)) * 2.0
    wc = rng.integers(-7, 8, (32, 512)).astype(np.int8)
    ws = rng.uniform(0.01, 0.02, 32).astype(np.float32)
    tab = np.array([0.3, 0.7], np.float32)
    grouped = np.repeat(tab[:, None], 4, axis=1)
    for t in range(2):
        a = o.grouped_linear(x, wc, ws, 1, grouped, t, out_fmt="f32")["y"]
        b = o.w4a4_linear(x, wc, ws, 1, table=tab, step=t, out_fmt="f32")["y"]
        assert np.array_equal(a, b)


def check_grouped_linear_bruteforce(o):
    """Nested loops over m, n, k: y = sum_k Delta_{g(k)} q_x[m,k] q_w[n,k] Delta_W[n] + b, with
    channel k in group k // max(128, b); codes by the nearest candidate per channel."""
    rng = np.random.default_rng(42)
    K, had = 256, 64
    x = rng.standard_normal((3, K)) * 3.0
    wc = rng.integers(-7, 8, (4, K)).astype(np.int8)
    ws = rng.uniform(0.01, 0.02, 4).astype(np.float32)
    bias = rng.standard_normal(4)
    table = np.array([[0.2, 0.9], [1.3, 0.05]], np.float32)
    out = o.grouped_linear(x, wc, ws, had, table, 1, bias=bias, out_fmt="f32")
    y32 = o.rotate_activations(x, had)
    for m in range(3):
        for k in range(K):
            d = float(table[1, k // 128])
            t = float(y32[m, k]) / d
            best = min(range(-7, 8), key=lambda q: (abs(t - q), q % 2))
            assert out["qx"][m, k] == best
    for m in range(3):
        for n in range(4):
            acc = sum(float(table[1, k // 128]) * int(out["qx"][m, k]) * int(wc[n, k]) for k in range(K))
            ref = acc * float(ws[n]) + bias[n]
            assert abs(out["y"][m, n] - ref) <= 2 ** -23 * max(1.0, abs(ref)), (m, n)


def check_grouped_calibration(o):
    """Each group's calibration peak maps to code +-7 exactly at its own scale; the group size is
    max(128, b)."""
    rng = np.random.default_rng(43)
    xs = [rng.standard_normal((8, 512)) * (1.0 + t) * np.repeat(rng.uniform(0.5, 4.0, 4), 128)[None, :]
          for t in range(3)]
    tab = o.calibrate_step_table_grouped(xs, 64)
    assert tab.shape == (3, 4)
    assert o.step_group_size(512, 64) == 128 and o.step_group_size(4096, 1024) == 1024
    for t in range(3):
        y = o.rotate_activations(xs[t], 64)
        q, _ = o.quantize_activations_per_step_grouped(y, tab, t, 128)
        for g in range(4):
            assert np.abs(q[:, g * 128:(g + 1) * 128]).max() == 7


def check_gelu_golden(o):
    """The tanh-form GELU of the gated MLP glue (reading R7) at hand-worked points
    (tests/golden/gelu_worked.txt), and the glue h = gelu(gate) * up."""
    g = read_golden("gelu_worked.txt")
    x = np.array([float(v) for v in g["x"]])
    want = np.array([float(v) for v in g["gelu"]])
    assert np.allclose(o.gelu_tanh(x), want, rtol=0, atol=5e-15)
    gate = np.array([float(v) for v in g["gate"]])
    up = np.array([float(v) for v in g["up"]])
    assert np.allclose(o.gated_glue(gate, up), np.array([float(v) for v in g["h"]]), rtol=0, atol=5e-15)


def check_gelu_library_and_identities(o):
    """gelu_tanh equals torch's GELU with approximate='tanh' (float64) on a grid over +-10;
    its odd part is x/2 (gelu(x) - gelu(-x) = x for the tanh form); it tends to x above and to
    0 below; it differs from the exact erf form (the other GELU) by more than rounding."""
    x = np.linspace(-10.0, 10.0, 4001)
    lib = torch.nn.functional.gelu(torch.from_numpy(x), approximate="tanh").numpy()
    assert np.allclose(o.gelu_tanh(x), lib, rtol=1e-14, atol=1e-15)
    assert np.allclose(o.gelu_tanh(x) - o.gelu_tanh(-x), x, rtol=0, atol=1e-13)
    assert abs(o.gelu_tanh(np.array([30.0]))[0] - 30.0) < 1e-12 and abs(o.gelu_tanh(np.array([-30.0]))[0]) < 1e-12
    erf_form = torch.nn.functional.gelu(torch.from_numpy(x), approximate="none").numpy()
    assert np.abs(o.gelu_tanh(x) - erf_form).max() > 1e-4
    rng = np.random.default_rng(44)
    gate, up = rng.standard_normal(64) * 3, rng.standard_normal(64)
    lib_h = torch.nn.functional.gelu(torch.from_numpy(gate), approximate="tanh").numpy() * up
    assert np.allclose(o.gated_glue(gate, up), lib_h, rtol=1e-14, atol=1e-15)


def check_q999_golden(o):
    """The q999 peak statistic (Eq. 6's sigma_hat as the appendix measures it) on a hand-worked
    case (tests/golden/q999_worked.txt): the 0.999 quantile of |y| with linear interpolation."""
    g = read_golden("q999_worked.txt")
    n = int(g["n"][0])
    y = np.array([(-1) ** i * i for i in range(n)], dtype=np.float64)
    assert o.robust_peak(y, "q999") == np.float32(float(g["q999"][0]))
    assert o.robust_peak(y, "absmax") == np.float32(float(g["absmax"][0]))
    # the same statistic through the calibration of a per-step table: sigma_hat / 7 of the rotated
    # activations; with b = 1 (no rotation) the activations are y itself
    tab = o.calibrate_step_table([y.reshape(8, n // 8)], 1, "q999")
    assert tab[0] == np.float32(998.001) / np.float32(7)


PINS = {f.__name__: f for f in [
    check_hadamard_matches_scipy, check_hadamard_orthogonal, check_hadamard_golden,
    check_rotate_matches_library_blockdiag, check_rotate_linf_bound, check_rotation_invariance,
    check_quantizer_golden, check_quantizer_bruteforce, check_quantizer_bounds,
    check_pack_golden_and_roundtrip, check_int_gemm_bruteforce, check_round_to_format,
    check_linear_golden, check_dequant_special_cases, check_step_lookup, check_calibration,
    check_weight_roundtrip, check_end_to_end_band,
    check_zigzag_golden, check_zigzag_rule, check_block_svd_golden, check_block_svd_properties,
    check_quantizer_8bit_bruteforce, check_w4a8_linear,
    check_gptq_two_columns_closed_form, check_gptq_identity_hessian_is_rtn, check_gptq_matches_obq_sequential,
    check_gptq_block_invariance_and_loss, check_gptq_dead_column,
    check_grouped_equal_scales_reduce_to_per_tensor, check_grouped_linear_bruteforce, check_grouped_calibration,
    check_gelu_golden, check_gelu_library_and_identities, check_q999_golden,
]}


@pytest.mark.parametrize("name", sorted(PINS))
def test_pin(name):
    PINS[name](O)


# --------------------------------------------------------------------------------------
# Planted mistakes: each must make at least one pin fail
# --------------------------------------------------------------------------------------

def _mut_hadamard_order(n):
    h = np.ones((1, 1), dtype=np.int64)
    while h.shape[0] < n:
        h = np.block([[h, -h], [h, h]])  # still orthogonal, wrong order
    return h


_real_rotate = O.block_hadamard_rotate
_real_quantize = O.quantize
_real_int_gemm = O.int_gemm
_real_dequant = O.dequant_output
_real_apply_block_rotation = O.apply_block_rotation
_real_block_svd = O.block_svd_rotation
_real_round = O.round_to_format


def _mut_rotate_unnormalised(x, b):
    return _real_rotate(x, b) * math.sqrt(b)


def _mut_rot_transposed(x, rot, rot_block):
    if rot is None:
        return np.asarray(x, np.float64)
    return _real_apply_block_rotation(x, np.transpose(np.asarray(rot), (0, 2, 1)), rot_block)


def _mut_quantize_floor(z, d):
    z64 = z.astype(np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.floor(z64 / np.float64(d) if np.ndim(d) == 0 else z64 / d.astype(np.float64))
    return np.clip(np.nan_to_num(r), -7, 7).astype(np.int8)


def _mut_quantize_half_away(z, d):
    z64 = z.astype(np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        t = z64 / np.broadcast_to(np.asarray(d, np.float64), z.shape)
    r = np.sign(t) * np.floor(np.abs(t) + 0.5)
    return np.clip(np.nan_to_num(r), -7, 7).astype(np.int8)


def _mut_quantize_clamp8(z, d):
    z64 = z.astype(np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.rint(z64 / np.broadcast_to(np.asarray(d, np.float64), z.shape))
    return np.clip(np.nan_to_num(r), -8, 8).astype(np.int8)


def _mut_scale_by_8(z, axis=None):
    return (np.asarray(np.max(np.abs(z), axis=axis), np.float32) / np.float32(8)).astype(np.float32)


def _mut_pack_swapped(q):
    u = (np.asarray(q).astype(np.int16) & 0xF).astype(np.uint8)
    return (u[..., 1::2] | (u[..., 0::2] << 4)).astype(np.uint8)


def _mut_unpack_no_sign(b):
    b = np.asarray(b, np.uint8)
    out = np.empty(b.shape[:-1] + (b.shape[-1] * 2,), dtype=np.int16)
    out[..., 0::2] = b & 0xF
    out[..., 1::2] = b >> 4
    return out.astype(np.int8)


def _mut_gemm_transposed(qx, qw):
    return (qx.astype(np.float64) @ qw.astype(np.float64).T).T.astype(np.int64)


def _mut_gemm_dropped_term(qx, qw):
    return (qx[..., 1:].astype(np.float64) @ qw[..., 1:].astype(np.float64).T).astype(np.int64)


def _mut_dequant_no_dw(acc, dx, dw, bias=None, out_fmt="f16"):
    return _real_dequant(acc, dx, np.ones_like(np.asarray(dw)), bias, out_fmt)


def _mut_dequant_bias_twice(acc, dx, dw, bias=None, out_fmt="f16"):
    b2 = None if bias is None else 2 * np.asarray(bias)
    return _real_dequant(acc, dx, dw, b2, out_fmt)


def _mut_lookup_off_by_one(table, t):
    table = np.asarray(table, np.float32)
    if not (0 <= t < table.shape[0]):
        raise IndexError(t)
    return table[max(t - 1, 0)]


def _mut_round_truncate(x, fmt):
    mant, emin, emax = O._FORMATS[fmt]
    x = np.asarray(x, np.float64)
    out = x.copy()
    fin = np.isfinite(x) & (x != 0)
    _, e = np.frexp(x[fin])
    qexp = np.maximum(e, emin + 1) - (mant + 1)
    out[fin] = np.ldexp(np.trunc(np.ldexp(x[fin], -qexp)), qexp)
    return out


def _mut_quantize_ignores_qmax(z, d, qmax=7):
    return _real_quantize(z, d, 7)


def _mut_zigzag_round_robin(w, block):
    w = np.asarray(w, np.float64)
    k = w.shape[1]
    nb = k // block
    order = np.argsort(-(w * w).sum(axis=0), kind="stable")
    perm = np.empty(k, dtype=np.int64)
    for i, j in enumerate(order):
        perm[(i % nb) * block + i // nb] = j
    return perm


def _mut_svd_ascending(w, block, perm=None):
    return _real_block_svd(w, block, perm)[:, :, ::-1].copy()


def _mut_svd_transposed(w, block, perm=None):
    return np.transpose(_real_block_svd(w, block, perm), (0, 2, 1)).copy()


def _gptq_variant(sign=1.0, use_h=False, scale_err=True, tail=True):
    """A GPTQ with one planted mistake (the oracle's steps otherwise)."""
    def gptq(w_folded, h, block=128, damp=0.01):
        w = np.asarray(w_folded, dtype=np.float64).astype(np.float32).astype(np.float64)
        n_rows, k = w.shape
        scale = O.absmax_scale(w.astype(np.float32), axis=1)
        d = scale.astype(np.float64)
        h = np.array(h, dtype=np.float64, copy=True)
        dead = np.diag(h) == 0
        h[dead, dead] = 1.0
        w[:, dead] = 0.0
        h[np.diag_indices(k)] += damp * np.mean(np.diag(h))
        u = np.linalg.cholesky(h if use_h else np.linalg.inv(h)).T
        codes = np.zeros((n_rows, k), dtype=np.int8)
        for i1 in range(0, k, block):
            i2 = min(i1 + block, k)
            err = np.zeros((n_rows, i2 - i1))
            for i in range(i1, i2):
                col = w[:, i]
                q = np.clip(np.rint(np.where(d > 0, col / np.where(d > 0, d, 1), 0.0)), -7, 7)
                codes[:, i] = q.astype(np.int8)
                e = (col - d * q) / (u[i, i] if scale_err else 1.0)
                w[:, i:i2] -= sign * np.outer(e, u[i, i:i2])
                err[:, i - i1] = e
            if tail:
                w[:, i2:] -= sign * (err @ u[i1:i2, i2:])
        return codes, scale
    return gptq


def _mut_group_of_next_channel(y, table, t, group, qmax=7):
    table = np.asarray(table, dtype=np.float32)
    d = table[t]
    per_channel = np.roll(np.repeat(d, group), 1)
    return O.quantize(y, per_channel[None, :], qmax), d


def _mut_group_first_only(y, table, t, group, qmax=7):
    table = np.asarray(table, dtype=np.float32)
    d = table[t]
    return O.quantize(y, np.full((1, y.shape[1]), d[0], np.float32), qmax), d


def _mut_group_size_fixed_128(k, had_block):
    return 128


def _mut_gelu_coefficient(x):
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.04715 * x ** 3)))


def _mut_gelu_no_sqrt_2_over_pi(x):
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + np.tanh(x + 0.044715 * x ** 3))


def _mut_gelu_erf_form(x):
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + scipy.special.erf(x / math.sqrt(2.0)))


def _mut_glue_swapped(gate, up):
    return O.gelu_tanh(up) * np.asarray(gate, dtype=np.float64)


def _mut_q999_at_099(y, estimator="absmax"):
    a = np.abs(np.asarray(y, dtype=np.float64)).ravel()
    if estimator == "q999":
        return np.float32(np.quantile(a, 0.99))
    return np.float32(a.max(initial=0.0))


def _mut_q999_nearest(y, estimator="absmax"):
    a = np.abs(np.asarray(y, dtype=np.float64)).ravel()
    if estimator == "q999":
        return np.float32(np.quantile(a, 0.999, method="nearest"))
    return np.float32(a.max(initial=0.0))


def _mut_q999_signed(y, estimator="absmax"):
    a = np.asarray(y, dtype=np.float64).ravel()
    if estimator == "q999":
        return np.float32(np.quantile(a, 0.999))
    return np.float32(np.abs(a).max(initial=0.0))


MUTANTS = {
    "hadamard_wrong_order": ("sylvester_hadamard", _mut_hadamard_order),
    "rotate_unnormalised": ("block_hadamard_rotate", _mut_rotate_unnormalised),
    "svd_factor_transposed": ("apply_block_rotation", _mut_rot_transposed),
    "quantize_floor": ("quantize", _mut_quantize_floor),
    "quantize_half_away": ("quantize", _mut_quantize_half_away),
    "quantize_clamp_8": ("quantize", _mut_quantize_clamp8),
    "scale_divides_by_8": ("absmax_scale", _mut_scale_by_8),
    "pack_nibbles_swapped": ("pack_int4", _mut_pack_swapped),
    "unpack_no_sign_extension": ("unpack_int4", _mut_unpack_no_sign),
    "gemm_transposed_output": ("int_gemm", _mut_gemm_transposed),
    "gemm_dropped_term": ("int_gemm", _mut_gemm_dropped_term),
    "dequant_drops_weight_scale": ("dequant_output", _mut_dequant_no_dw),
    "dequant_bias_twice": ("dequant_output", _mut_dequant_bias_twice),
    "step_lookup_off_by_one": ("step_scale_lookup", _mut_lookup_off_by_one),
    "round_truncates": ("round_to_format", _mut_round_truncate),
    "zigzag_without_turns": ("zigzag_permutation", _mut_zigzag_round_robin),
    "quantize_8bit_clamps_at_7": ("quantize", _mut_quantize_ignores_qmax),
    "svd_columns_ascending": ("block_svd_rotation", _mut_svd_ascending),
    "svd_factor_transposed_in_pack": ("block_svd_rotation", _mut_svd_transposed),
    "gptq_update_sign_flipped": ("gptq_quantize", _gptq_variant(sign=-1.0)),
    "gptq_cholesky_of_hessian": ("gptq_quantize", _gptq_variant(use_h=True)),
    "gptq_error_not_scaled": ("gptq_quantize", _gptq_variant(scale_err=False)),
    "gptq_no_update_past_block": ("gptq_quantize", _gptq_variant(tail=False)),
    "grouped_scale_shifted_one_channel": ("quantize_activations_per_step_grouped", _mut_group_of_next_channel),
    "grouped_scale_first_group_only": ("quantize_activations_per_step_grouped", _mut_group_first_only),
    "group_size_ignores_hadamard_block": ("step_group_size", _mut_group_size_fixed_128),
    "gelu_cubic_coefficient": ("gelu_tanh", _mut_gelu_coefficient),
    "gelu_without_sqrt_2_over_pi": ("gelu_tanh", _mut_gelu_no_sqrt_2_over_pi),
    "gelu_erf_form": ("gelu_tanh", _mut_gelu_erf_form),
    "glue_gate_and_up_swapped": ("gated_glue", _mut_glue_swapped),
    "q999_at_0_99": ("robust_peak", _mut_q999_at_099),
    "q999_nearest_rank": ("robust_peak", _mut_q999_nearest),
    "q999_without_abs": ("robust_peak", _mut_q999_signed),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutants(name, monkeypatch, request):
    attr, fn = MUTANTS[name]
    # the normalised Hadamard is cached: rebuild it from the mutant, and again after it is undone
    O._normalized_hadamard_cached.cache_clear()
    request.addfinalizer(O._normalized_hadamard_cached.cache_clear)
    monkeypatch.setattr(O, attr, fn)
    failed = []
    for pin_name, pin in PINS.items():
        try:
            pin(O)
        except Exception:  # an assertion, or the mutant breaking a shape contract
            failed.append(pin_name)
    assert failed, f"no pin caught the planted mistake {name}"
