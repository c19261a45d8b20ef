"""CPU oracle for the Omega-QVLA W4A4 quantized linear -- TEST INFRASTRUCTURE ONLY.

This module restates the method of arxiv 2605.28803 ("Omega-QVLA") as plain, slow,
obviously-correct numpy.  It exists to check the CUDA path, never to serve it:
only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
reference leg may import it.  The product package never imports it, and the two
share no code (no kernels, headers, tables, helpers, pre- or post-processing).

What is computed, in the paper's order (Sec. 4):
  * Sec. 4.1, Eq. 3-5: the composite rotation X' = X P R_hat, W' = P^T R_hat^T W with
    R_hat = BlockDiag(U_b H_c).  Written out as dense float64 products.
  * Sec. 4.1 (Eq. 4 and the permutation after it): the offline choice of P (channels sorted
    by weight energy, dealt across blocks in zigzag order) and of U_b (the left singular
    vectors of each block's row partition, from numpy's SVD).
  * Sec. 4.2, Eq. 5: Delta_Z = max|Z| / q_max, q_max = 2^(k-1) - 1 = 7 at k = 4.
  * Sec. 4.2, Eq. 6 (first display): Q_Z = clamp(round(Z / Delta_Z), -q_max, q_max).
  * Sec. 4.2: weight scales per output channel, backbone activation scales per token,
    DiT activation scales from a per-step table (Eq. 6, second display) looked up by t.
  * Sec. 4.2, Eq. 7: X'W' ~= Delta_X' Delta_W' Q_X' Q_W' (the integer GEMM and the
    dequantisation), plus the bias of the linear Y = XW + b (Sec. 3.2).
  * Sec. 5.1 implementation details and the appendix on weight-quantisation solvers: the
    LLM side's GPTQ-style weight codes (block size 128, damping ratio 0.01), written from
    the published GPTQ algorithm the paper names.

Precision.  Rotations, folds and the dequantised output are float64, rounded once
to the output format.  Where floating point decides an integer (an int4 code) the
decision is taken on the exact quotient of the float32 operands Z / Delta, rounded
half to even: ``quantize`` explains why float64 division makes that decision
exactly.  Delta itself is a float32 value: float32(max|Z|) / 7 in float32.

Readings of the paper that this file fixes (each is also listed in the design notes):
  R1  H is the Sylvester (natural-order) Hadamard matrix, normalised by 1/sqrt(b).
  R2  The online rotation is the block Hadamard only; P and the SVD factors U_b are
      applied upstream to activations and folded into the weights offline.
  R3  Codes are clamped to [-7, 7] (Eq. 6); -8 is never produced.
  R4  round() is round-half-to-even on the exact quotient; Delta = 0 gives code 0.
  R5  The per-step table holds one float32 scale per (layer, step): the per-tensor
      reading of Eq. 6 (the paper's table is per channel).
  R6  Packed int4: byte j of a row holds code 2j in its low nibble and code 2j+1 in
      its high nibble, each as a 4-bit two's-complement integer.
  R7  The down-projection glue of the gated MLP is gelu_tanh(gate) * up.
  R20 The q999 peak statistic is the 0.999 quantile of |y| with linear interpolation between
      order statistics.
  R14 The zigzag deals the energy-sorted channels (ties: lower index first) forwards in even
      rounds and backwards in odd ones; Eq. 5's W' = P^T R_hat^T W is read as the fold that
      keeps X W unchanged, R_hat^T P^T W.
  R15 U_b's columns are ordered by descending singular value, each signed so that its
      largest-magnitude entry is positive (the SVD fixes them only up to sign).
  R18 The per-step table of Eq. 6 is also provided per channel group: one float32 per
      (layer, step, group of max(128, b) channels) -- a k-block of the integer GEMM or a
      Hadamard block; each group's integer partial is scaled by its Delta before the sum.
  R17 GPTQ keeps the RTN per-channel scale (max |W'_n| / 7 of the folded weights) and
      quantises the columns in natural order; its Hessian is H = 2/n X'^T X' of calibration
      activations in the folded basis, damped by 0.01 mean(diag H); a column with
      H_kk = 0 is dead (its weights become 0 and H_kk 1).

Functions with no pin in the paper (the paper prints no worked numeric example) are
pinned by closed forms, invariants, library special cases and brute force in
``tests/test_oracle_pins.py``; none is "parity unpinned".
"""

from __future__ import annotations

import functools
import math

import numpy as np

# Sec. 4.2, Eq. 5-6: q_max = 2^(k-1) - 1 with k = 4 bits for both weights and activations.
BITS = 4
QMAX = 2 ** (BITS - 1) - 1


# --------------------------------------------------------------------------------------
# Sec. 4.1 -- rotations
# --------------------------------------------------------------------------------------

def sylvester_hadamard(n: int) -> np.ndarray:
    """Unnormalised Hadamard matrix of order n (a power of two), entries +-1, int64.

    Sec. 4.1, "Hadamard rotation" / Eq. 3: the paper composes the SVD factor with a
    normalised Hadamard matrix H in {+-1/sqrt(C_in)}^(C_in x C_in).  Reading R1: the
    Sylvester construction H_1 = [1], H_2m = [[H_m, H_m], [H_m, -H_m]].
    """
    if n < 1 or n & (n - 1):
        raise ValueError(f"Hadamard order must be a power of two, got {n}")
    h = np.ones((1, 1), dtype=np.int64)
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


def normalized_hadamard(n: int) -> np.ndarray:
    """H / sqrt(n) in float64: the orthogonal matrix of Sec. 4.1 / Eq. 3.  Built once per
    order and returned read-only (the stacks rotate thousands of rows with the same H)."""
    return _normalized_hadamard_cached(n)


@functools.lru_cache(maxsize=8)
def _normalized_hadamard_cached(n: int) -> np.ndarray:
    h = sylvester_hadamard(n).astype(np.float64) / math.sqrt(n)
    h.setflags(write=False)
    return h


def block_hadamard_rotate(x: np.ndarray, had_block: int) -> np.ndarray:
    """x . BlockDiag(H_b, ..., H_b) with H_b the normalised Hadamard of order b, float64.

    Sec. 4.1, "Block-wise Implementation" / Eq. 4: R_hat is block diagonal; its online
    factor is the Hadamard H_c of each block (reading R2).  Written as one dense
    product per block of b consecutive channels.  x: [..., K] with K % b == 0.
    """
    x = np.asarray(x, dtype=np.float64)
    k = x.shape[-1]
    if k % had_block:
        raise ValueError(f"K={k} is not a multiple of the Hadamard block {had_block}")
    hb = normalized_hadamard(had_block)
    blocks = x.reshape(*x.shape[:-1], k // had_block, had_block)
    return (blocks @ hb).reshape(x.shape)


def apply_permutation(x: np.ndarray, perm) -> np.ndarray:
    """x . P for the channel permutation P of Sec. 4.1 (Eq. 5): column j of the
    result is column perm[j] of x.  perm=None is the identity."""
    x = np.asarray(x, dtype=np.float64)
    if perm is None:
        return x
    perm = np.asarray(perm)
    if sorted(perm.tolist()) != list(range(x.shape[-1])):
        raise ValueError("perm is not a permutation of the channel axis")
    return x[..., perm]


def apply_block_rotation(x: np.ndarray, rot, rot_block: int | None) -> np.ndarray:
    """x . BlockDiag(U_1, ..., U_nb) for the SVD factors U_b of Eq. 4 (float64).

    rot: None (U = I) or an array [K / rot_block, rot_block, rot_block] of orthogonal
    blocks; a dense K x K factor is rot_block = K.
    """
    x = np.asarray(x, dtype=np.float64)
    if rot is None:
        return x
    rot = np.asarray(rot, dtype=np.float64)
    k = x.shape[-1]
    nb = k // rot_block
    if rot.shape != (nb, rot_block, rot_block):
        raise ValueError(f"rot must have shape {(nb, rot_block, rot_block)}, got {rot.shape}")
    out = np.empty_like(x)
    for b in range(nb):
        sl = slice(b * rot_block, (b + 1) * rot_block)
        out[..., sl] = x[..., sl] @ rot[b]
    return out


def fold_weights(w: np.ndarray, had_block: int, perm=None, rot=None, rot_block=None) -> np.ndarray:
    """Offline fold of the composite rotation into the weights, float64.

    Eq. 5 writes W' = P^T R_hat^T W for W in C_in x C_out.  The weights here are stored
    [C_out, C_in] (row n = output channel n, y = x W^T), so the same fold reads
    W'_rows = W_rows . P . R_hat with R_hat = BlockDiag(U_b) . BlockDiag(H_c) (Eq. 3-4).
    """
    wr = apply_permutation(w, perm)
    wr = apply_block_rotation(wr, rot, rot_block)
    return block_hadamard_rotate(wr, had_block)


def zigzag_permutation(w: np.ndarray, block: int) -> np.ndarray:
    """The channel permutation P of Sec. 4.1 (after Eq. 4): input channels sorted by descending
    weight energy sum_n W[n, j]^2 (ties by channel index), dealt across the K/block blocks in
    zigzag order -- round r visits the blocks forwards for even r, backwards for odd r -- each
    block taking its channels in the order dealt.  Returns perm (int64 [K]): column j of X P is
    column perm[j] of X, i.e. block b holds channels perm[b block : (b + 1) block]."""
    w = np.asarray(w, dtype=np.float64)
    k = w.shape[1]
    if k % block:
        raise ValueError(f"K={k} is not a multiple of the block {block}")
    nb = k // block
    energy = (w * w).sum(axis=0)
    order = np.argsort(-energy, kind="stable")
    perm = np.empty(k, dtype=np.int64)
    for i, j in enumerate(order):
        r, pos = divmod(i, nb)
        b = pos if r % 2 == 0 else nb - 1 - pos
        perm[b * block + r] = j
    return perm


def block_svd_rotation(w: np.ndarray, block: int, perm=None) -> np.ndarray:
    """The SVD factors U_b of Eq. 4 for the weights stored [C_out, C_in]: after the permutation,
    block b of the input channels is W_b = (W P)[:, b]^T (block x C_out, the paper's row
    partition) and U_b its block x block left singular vectors, columns ordered by descending
    singular value (reading R2 of U_SVD(W_b^T)).  Each column's sign makes its largest-magnitude
    entry positive (the first, on a tie).  Returns rot [K/block, block, block] float64, to be
    used as x . BlockDiag(U_b)."""
    wp = apply_permutation(np.asarray(w, dtype=np.float64), perm)
    k = wp.shape[1]
    nb = k // block
    rot = np.empty((nb, block, block), dtype=np.float64)
    for b in range(nb):
        wb = wp[:, b * block:(b + 1) * block].T
        u, _, _ = np.linalg.svd(wb, full_matrices=True)
        idx = np.argmax(np.abs(u), axis=0)
        u = u * np.where(u[idx, np.arange(block)] < 0, -1.0, 1.0)[None, :]
        rot[b] = u
    return rot


def upstream_activation_transform(x: np.ndarray, perm=None, rot=None, rot_block=None) -> np.ndarray:
    """X . P . BlockDiag(U_b): the part of X' = X P R_hat (Eq. 5) applied upstream of the
    online kernel (reading R2).  Float64; the caller rounds to the activation dtype."""
    return apply_block_rotation(apply_permutation(x, perm), rot, rot_block)


# --------------------------------------------------------------------------------------
# Sec. 4.2 -- symmetric uniform quantiser
# --------------------------------------------------------------------------------------

def qmax_of(bits: int) -> int:
    """q_max = 2^(k-1) - 1 for k-bit symmetric codes (Sec. 4.2, Eq. 5): 7 at k = 4, 127 at k = 8."""
    return 2 ** (bits - 1) - 1


def absmax_scale(z: np.ndarray, axis=None, qmax: int = QMAX) -> np.ndarray:
    """Delta_Z = max|Z| / q_max (Sec. 4.2, Eq. 5), in float32 as the stored scale.

    z must already be float32 (the values the quantiser sees).  The maximum of float32
    magnitudes is exact; the division by q_max is one IEEE float32 division.
    """
    z = np.asarray(z)
    if z.dtype != np.float32:
        raise TypeError("absmax_scale expects float32 input")
    m = np.max(np.abs(z), axis=axis)
    return (np.asarray(m, dtype=np.float32) / np.float32(qmax)).astype(np.float32)


def quantize(z: np.ndarray, delta: np.ndarray, qmax: int = QMAX) -> np.ndarray:
    """Q_Z = clamp(round(Z / Delta), -q_max, q_max) (Sec. 4.2, Eq. 6), int8 codes.

    z and delta are float32 (delta broadcasts against z).  Reading R4: round() is
    half-to-even on the exact real quotient of the two float32 operands.  That quotient
    is evaluated in float64: for float32 z = a 2^i and delta = d 2^j (|a|, |d| < 2^24)
    a quotient that is not itself a half-integer lies at least 2^-25 (relative) from
    every half-integer, far more than float64's 2^-53 rounding error, so np.rint of the
    float64 quotient takes the exact decision.  Delta = 0 (an all-zero row) gives 0.
    """
    z = np.asarray(z)
    delta = np.asarray(delta)
    if z.dtype != np.float32 or delta.dtype != np.float32:
        raise TypeError("quantize expects float32 operands")
    z64 = z.astype(np.float64)
    d64 = np.broadcast_to(delta.astype(np.float64), z.shape)
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.rint(z64 / d64)
    r = np.where(d64 == 0.0, 0.0, r)
    r = np.where(np.isnan(r), 0.0, r)
    return np.clip(r, -qmax, qmax).astype(np.int8)


def dequantize(q: np.ndarray, delta: np.ndarray) -> np.ndarray:
    """Q(Z) = Delta_Z Q_Z (Sec. 4.2, after Eq. 6), float64."""
    return np.asarray(delta, dtype=np.float64) * np.asarray(q, dtype=np.float64)


# --------------------------------------------------------------------------------------
# Packed int4 layout (reading R6; the paper only says "packed layout")
# --------------------------------------------------------------------------------------

def pack_int4(q: np.ndarray) -> np.ndarray:
    """int8 codes [..., K] (K even, each in [-8, 7]) -> uint8 [..., K/2]."""
    q = np.asarray(q)
    if q.shape[-1] % 2:
        raise ValueError("K must be even to pack int4 pairs")
    if q.min(initial=0) < -8 or q.max(initial=0) > 7:
        raise ValueError("codes out of int4 range")
    u = (q.astype(np.int16) & 0xF).astype(np.uint8)
    return (u[..., 0::2] | (u[..., 1::2] << 4)).astype(np.uint8)


def unpack_int4(b: np.ndarray) -> np.ndarray:
    """uint8 [..., K/2] -> int8 codes [..., K] (inverse of pack_int4)."""
    b = np.asarray(b, dtype=np.uint8)
    lo = (b & 0xF).astype(np.int16)
    hi = (b >> 4).astype(np.int16)
    lo = np.where(lo >= 8, lo - 16, lo)
    hi = np.where(hi >= 8, hi - 16, hi)
    out = np.empty(b.shape[:-1] + (b.shape[-1] * 2,), dtype=np.int8)
    out[..., 0::2] = lo
    out[..., 1::2] = hi
    return out


# --------------------------------------------------------------------------------------
# Weights (offline) and activations (online)
# --------------------------------------------------------------------------------------

def quantize_weights(w_folded: np.ndarray):
    """Per-output-channel symmetric int4 RTN of the folded weights (Sec. 4.2: Delta_W'
    per output channel at bit-width k_w; RTN on the DiT side, Sec. 5.1).

    w_folded: float64 [N, K]; it is rounded once to float32, the precision of the
    stored scale and of the code decision.  Returns (codes int8 [N, K], scales f32 [N]).
    """
    wf = np.asarray(w_folded, dtype=np.float64).astype(np.float32)
    scale = absmax_scale(wf, axis=1)
    codes = quantize(wf, scale[:, None])
    return codes, scale


def gptq_hessian(x_folded: np.ndarray) -> np.ndarray:
    """H = 2/n X'^T X' (float64 [K, K]) of n calibration rows already in the folded basis
    X' = X P R_hat: the Hessian of the layer-wise squared error ||X'W'^T - X'Q^T||^2 that GPTQ
    minimises."""
    x = np.asarray(x_folded, dtype=np.float64)
    return (2.0 / x.shape[0]) * (x.T @ x)


def gptq_quantize(w_folded: np.ndarray, h: np.ndarray, block: int = 128, damp: float = 0.01):
    """GPTQ-style int4 weight codes (Sec. 5.1: the LLM side's solver, block size 128, damping
    ratio 0.01), from the published GPTQ algorithm (reading R17):

      1. scales as RTN: Delta_W[n] = float32(max |W'_n|) / 7 of the float32-rounded weights;
      2. dead columns (H_kk = 0) are zeroed; H += damp * mean(diag H) * I;
      3. U = the upper Cholesky factor of H^-1 (H^-1 = U^T U);
      4. for each column i in order: q = clamp(round(w_i / Delta), +-7); the scaled error
         e = (w_i - Delta q) / U_ii is subtracted, times U_ij, from every later column j;
         within a block of `block` columns the later columns of the block are updated at
         once, the columns after the block by one product at the end of the block.

    w_folded: float64 [N, K]; h: float64 [K, K].  Returns (codes int8 [N, K], scales f32 [N]).
    """
    w = np.asarray(w_folded, dtype=np.float64).astype(np.float32).astype(np.float64)
    n_rows, k = w.shape
    scale = absmax_scale(w.astype(np.float32), axis=1)
    d = scale.astype(np.float64)[:, None]
    h = np.array(h, dtype=np.float64, copy=True)
    dead = np.diag(h) == 0
    h[dead, dead] = 1.0
    w[:, dead] = 0.0
    h[np.diag_indices(k)] += damp * np.mean(np.diag(h))
    hinv = np.linalg.inv(h)
    u = np.linalg.cholesky(hinv).T  # upper: hinv = u^T u
    codes = np.zeros((n_rows, k), dtype=np.int8)
    for i1 in range(0, k, block):
        i2 = min(i1 + block, k)
        err = np.zeros((n_rows, i2 - i1))
        for i in range(i1, i2):
            col = w[:, i]
            with np.errstate(divide="ignore", invalid="ignore"):
                t = np.where(d[:, 0] > 0, col / d[:, 0], 0.0)
            q = np.clip(np.rint(t), -QMAX, QMAX)
            codes[:, i] = q.astype(np.int8)
            e = (col - d[:, 0] * q) / u[i, i]
            w[:, i:i2] -= np.outer(e, u[i, i:i2])
            err[:, i - i1] = e
        w[:, i2:] -= err @ u[i1:i2, i2:]
    return codes, scale


def weight_proxy_loss(w_folded: np.ndarray, codes: np.ndarray, scale: np.ndarray, h: np.ndarray) -> float:
    """tr((W' - Delta Q) H (W' - Delta Q)^T): the calibration error GPTQ reduces."""
    dw = np.asarray(w_folded, dtype=np.float64) - np.asarray(scale, np.float64)[:, None] * codes
    return float(np.einsum("nk,kl,nl->", dw, np.asarray(h, np.float64), dw))


def pack_weights(w: np.ndarray, had_block: int, perm=None, rot=None, rot_block=None):
    """The offline weight path: fold (Eq. 5), per-channel quantise (Eq. 5-6), pack.

    Returns (packed uint8 [N, K/2], scales f32 [N], codes int8 [N, K]).
    """
    codes, scale = quantize_weights(fold_weights(w, had_block, perm, rot, rot_block))
    return pack_int4(codes), scale, codes


def rotate_activations(x: np.ndarray, had_block: int) -> np.ndarray:
    """The online rotation of Eq. 5 (block Hadamard, reading R2) rounded once to float32:
    the rotated activations the quantiser sees.  x holds the (fp16/bf16/fp32) input values."""
    return block_hadamard_rotate(np.asarray(x, dtype=np.float64), had_block).astype(np.float32)


def quantize_activations_per_token(y: np.ndarray, qmax: int = QMAX):
    """Backbone activations: one scale per token (Sec. 4.2), Eq. 5-6 along each row.
    y: float32 [M, K] rotated activations.  Returns (codes int8 [M, K], scales f32 [M])."""
    scale = absmax_scale(y, axis=1, qmax=qmax)
    return quantize(y, scale[:, None], qmax), scale


def step_scale_lookup(table, t: int) -> np.float32:
    """Sec. 4.2: at inference the scale of the current step t is retrieved from the
    per-step table (reading R5: one float32 per step).  t outside [0, T) is an error."""
    table = np.asarray(table, dtype=np.float32)
    if not (0 <= t < table.shape[0]):
        raise IndexError(f"step {t} outside the table of {table.shape[0]} steps")
    return table[t]


def quantize_activations_per_step(y: np.ndarray, table, t: int, qmax: int = QMAX):
    """DiT activations: the step-t scale replaces Delta_Z in Eq. 6 (Sec. 4.2)."""
    d = step_scale_lookup(table, t)
    scale = np.full(y.shape[0], d, dtype=np.float32)
    return quantize(y, scale[:, None], qmax), scale


def step_group_size(k: int, had_block: int) -> int:
    """Channels per scale of the per-step, per-group table (reading R18): max(128, b) -- one
    128-channel k-block of the integer GEMM, or one Hadamard block when that is larger (after a
    Hadamard block every channel of the block has the same spread, so a finer scale is moot)."""
    g = max(128, had_block)
    if k % g:
        raise ValueError(f"K={k} is not a multiple of the group size {g}")
    return g


def quantize_activations_per_step_grouped(y: np.ndarray, table, t: int, group: int, qmax: int = QMAX):
    """DiT activations with the per-step, per-group table of Eq. 6 (reading R18): channel k of
    step t is quantised with table[t, k // group].  Returns (codes int8 [M, K], scales f32 [G])."""
    table = np.asarray(table, dtype=np.float32)
    if not (0 <= t < table.shape[0]):
        raise IndexError(f"step {t} outside the table of {table.shape[0]} steps")
    d = table[t]
    if d.shape[0] * group != y.shape[1]:
        raise ValueError("table width times group size must equal K")
    per_channel = np.repeat(d, group)
    return quantize(y, per_channel[None, :], qmax), d


def grouped_linear(x: np.ndarray, w_codes: np.ndarray, w_scale: np.ndarray, had_block: int, table, step: int,
                   bias=None, out_fmt: str = "f16", act_bits: int = 4):
    """The online linear with per-step, per-group activation scales (Eq. 6 per channel group,
    Eq. 7 per group): y = sum_g Delta_g Delta_W acc_g + b, where acc_g is the integer product
    over group g's channels.  Float64 sum over the groups, rounded once to the output format."""
    qmax = qmax_of(act_bits)
    y32 = rotate_activations(x, had_block)
    group = step_group_size(y32.shape[1], had_block)
    qx, d = quantize_activations_per_step_grouped(y32, table, step, group, qmax)
    n_groups = d.shape[0]
    acc = [int_gemm(qx[:, g * group:(g + 1) * group], w_codes[:, g * group:(g + 1) * group]) for g in range(n_groups)]
    y = np.zeros(acc[0].shape)
    for g in range(n_groups):
        y += np.float64(d[g]) * acc[g].astype(np.float64)
    y = y * np.asarray(w_scale, dtype=np.float64)[None, :]
    if bias is not None:
        y = y + np.asarray(bias, dtype=np.float64)[None, :]
    return {"y_rot": y32, "qx": qx, "dx": d, "acc_groups": acc, "y": round_to_format(y, out_fmt)}


def calibrate_step_table_grouped(x_steps, had_block: int, estimator: str = "absmax", qmax: int = QMAX) -> np.ndarray:
    """Per-step, per-group table [T, G] (reading R18): Delta_{t,g} = sigma_hat of group g's
    channels of the rotated X_t, over q_max, float32."""
    rows = []
    for x in x_steps:
        y = rotate_activations(x, had_block)
        group = step_group_size(y.shape[1], had_block)
        rows.append([np.float32(robust_peak(y[:, g * group:(g + 1) * group], estimator)) / np.float32(qmax)
                     for g in range(y.shape[1] // group)])
    return np.asarray(rows, dtype=np.float32)


def robust_peak(y: np.ndarray, estimator: str = "absmax") -> np.float32:
    """sigma_hat of Eq. 6: a robust peak estimate of a calibration tensor.

    "absmax" is max|y|; "q999" is the 99.9th percentile of |y| (the appendix on per-step
    scaling measures q999), read as the 0.999 quantile with linear interpolation between order
    statistics (reading R20).  Returned as float32.
    """
    a = np.abs(np.asarray(y, dtype=np.float64)).ravel()
    if estimator == "absmax":
        return np.float32(a.max(initial=0.0))
    if estimator == "q999":
        return np.float32(np.quantile(a, 0.999))
    raise ValueError(f"unknown estimator {estimator}")


def calibrate_step_table(x_steps, had_block: int, estimator: str = "absmax") -> np.ndarray:
    """Per-step scale table of Eq. 6 (per-tensor reading R5): for each step t,
    Delta_t = sigma_hat(rotated X_t) / q_max, float32, from calibration activations."""
    out = []
    for x in x_steps:
        y = rotate_activations(x, had_block)
        out.append(np.float32(robust_peak(y, estimator)) / np.float32(QMAX))
    return np.asarray(out, dtype=np.float32)


# --------------------------------------------------------------------------------------
# Eq. 7 -- integer GEMM and dequantisation
# --------------------------------------------------------------------------------------

def int_gemm(qx: np.ndarray, qw: np.ndarray) -> np.ndarray:
    """acc[m, n] = sum_k Q_X'[m, k] Q_W'[n, k]: the integer product of Eq. 7, int64.

    Evaluated with a float64 matrix product: every product is an integer of magnitude
    <= 128 x 8 = 1024 (8-bit activation codes against int4 weights; <= 64 for int4 x int4) and
    every partial sum an integer of magnitude <= 1024 K < 2^53, all exactly representable, so
    the result is the exact integer whatever the summation order.
    """
    qx = np.asarray(qx)
    qw = np.asarray(qw)
    if qx.shape[-1] != qw.shape[-1]:
        raise ValueError("reduction lengths differ")
    if qx.shape[-1] * 1024 >= 2 ** 53:
        raise ValueError("K too large for an exact float64 product")
    return (qx.astype(np.float64) @ qw.astype(np.float64).T).astype(np.int64)


_FORMATS = {
    # name: (explicit mantissa bits, min normal exponent, max exponent)
    "f16": (10, -14, 15),
    "bf16": (7, -126, 127),
    "f32": (23, -126, 127),
}


def round_to_format(x: np.ndarray, fmt: str) -> np.ndarray:
    """Round float64 values once, to nearest-even, to an IEEE-style binary format
    ("f16", "bf16", "f32"), with gradual underflow and overflow to +-inf.  Returned
    as float64 values of that format."""
    mant, emin, emax = _FORMATS[fmt]
    x = np.asarray(x, dtype=np.float64)
    out = x.copy()
    fin = np.isfinite(x) & (x != 0)
    xf = x[fin]
    _, e = np.frexp(xf)  # xf = f * 2^e with 0.5 <= |f| < 1
    qexp = np.maximum(e, emin + 1) - (mant + 1)  # exponent of one unit in the last place
    r = np.ldexp(np.rint(np.ldexp(xf, -qexp)), qexp)
    maxfin = (2.0 - 2.0 ** -mant) * 2.0 ** emax
    r = np.where(np.abs(r) > maxfin, np.copysign(np.inf, r), r)
    out[fin] = r
    return out


def dequant_output(acc: np.ndarray, dx: np.ndarray, dw: np.ndarray, bias=None, out_fmt: str = "f16") -> np.ndarray:
    """y[m, n] = Delta_X'[m] Delta_W'[n] acc[m, n] + b[n] (Eq. 7 plus the bias of
    Y = XW + b, Sec. 3.2), float64, rounded once to the output format."""
    y = np.asarray(acc, dtype=np.float64) * np.asarray(dx, dtype=np.float64)[:, None]
    y = y * np.asarray(dw, dtype=np.float64)[None, :]
    if bias is not None:
        y = y + np.asarray(bias, dtype=np.float64)[None, :]
    return round_to_format(y, out_fmt)


def w4a4_linear(x: np.ndarray, w_codes: np.ndarray, w_scale: np.ndarray, had_block: int,
                bias=None, table=None, step: int | None = None, out_fmt: str = "f16", act_bits: int = 4):
    """The online quantized linear of Sec. 4: rotate (Eq. 5), quantise per token or with
    the step-t table scale (Eq. 5-6), integer GEMM and dequantisation (Eq. 7).

    x: activations [M, K] already in the P.U basis (reading R2), as fp16/bf16/fp32 values.
    act_bits: 4 (W4A4) or 8 (W4A8, the paper's deployed precision: the same recipe with
    k = 8, q_max = 127, for the activations only).
    Returns a dict with the rotated activations, codes, scales, int accumulator and y.
    """
    qmax = qmax_of(act_bits)
    y32 = rotate_activations(x, had_block)
    if step is None:
        qx, dx = quantize_activations_per_token(y32, qmax)
    else:
        qx, dx = quantize_activations_per_step(y32, table, step, qmax)
    acc = int_gemm(qx, w_codes)
    out = dequant_output(acc, dx, w_scale, bias, out_fmt)
    return {"y_rot": y32, "qx": qx, "dx": dx, "acc": acc, "y": out}


# --------------------------------------------------------------------------------------
# Glue of the gated MLP (reading R7) and the unquantised reference
# --------------------------------------------------------------------------------------

def gelu_tanh(x: np.ndarray) -> np.ndarray:
    """GELU, tanh form, float64: x/2 (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3))), the activation
    of the gated MLP of the Pi-0.5 / PaliGemma backbone (Sec. 5.1; reading R7)."""
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def gated_glue(gate: np.ndarray, up: np.ndarray) -> np.ndarray:
    """h = gelu_tanh(gate) * up, float64 (reading R7)."""
    return gelu_tanh(gate) * np.asarray(up, dtype=np.float64)


def relative_output_error(y_q: np.ndarray, y_ref: np.ndarray) -> float:
    """||Y_q - Y||_F / ||Y||_F, the relative output error of the appendix on weight
    solvers; a sanity band for a whole W4A4 linear, not a parity criterion."""
    y_q = np.asarray(y_q, dtype=np.float64)
    y_ref = np.asarray(y_ref, dtype=np.float64)
    return float(np.linalg.norm(y_q - y_ref) / np.linalg.norm(y_ref))
