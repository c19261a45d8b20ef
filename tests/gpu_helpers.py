"""Shared helpers of the GPU parity tests: run libqvla through its C ABI on torch tensors."""

import numpy as np
import torch

from paper_2605_28803_gb300 import qvla as Q

DEV = torch.device("cuda:0")
TORCH_DT = {"f16": torch.float16, "bf16": torch.bfloat16, "f32": torch.float32}
OUT_FMT = {"f16": "f16", "bf16": "bf16"}


def stream():
    return torch.cuda.current_stream()


def rotate_quantize_rows(x: torch.Tensor, had: int, step_scale=None):
    """GPU rotate + quantise of an [M, K] tensor; returns (packed codes uint8 [M, K/2], scale f32 [M], sum int [M])."""
    M, K = x.shape
    xdt = {torch.float16: Q.F16, torch.bfloat16: Q.BF16, torch.float32: Q.F32}[x.dtype]
    xg = x.to(DEV).contiguous()
    xq = torch.zeros(M, K // 2, dtype=torch.uint8, device=DEV)
    xs = torch.full((M,), -1.0, dtype=torch.float32, device=DEV)
    xsum = torch.full((M,), -999999, dtype=torch.int32, device=DEV)
    ss = None
    if step_scale is not None:
        ss = torch.tensor([step_scale], dtype=torch.float32, device=DEV)
    Q.qvla_rotate_quantize_rows(xg, xdt, M, K, had, ss, xq, xs, xsum, stream())
    Q.qvla_check_device(stream())
    return xq.cpu().numpy(), xs.cpu().numpy(), xsum.cpu().numpy()


def make_layer(wq: np.ndarray, ws: np.ndarray, had: int, xdt="f16", ydt="f16", bias=None):
    N, K2 = wq.shape
    return Q.qvla_layer_create(N, K2 * 2, had, Q.DTYPE_CODES[xdt], Q.DTYPE_CODES[ydt], np.ascontiguousarray(wq),
                               np.ascontiguousarray(ws, dtype=np.float32),
                               None if bias is None else np.ascontiguousarray(bias, dtype=np.float32))


def gemm(layer, xq: np.ndarray, xs: np.ndarray, xsum: np.ndarray, ydt="f16"):
    """GPU integer GEMM + epilogue; returns (y float64 [M,N], acc int64 [M,N])."""
    M = xq.shape[0]
    N = layer.N
    xqg = torch.from_numpy(np.ascontiguousarray(xq)).to(DEV)
    xsg = torch.from_numpy(np.ascontiguousarray(xs, dtype=np.float32)).to(DEV)
    xsumg = torch.from_numpy(np.ascontiguousarray(xsum, dtype=np.int32)).to(DEV)
    y = torch.full((M, N), float("nan"), dtype=TORCH_DT[ydt], device=DEV)
    acc = torch.full((M, 2 * N if layer.gated else N), -2 ** 31, dtype=torch.int32, device=DEV)
    Q.qvla_gemm_w4a4(layer, xqg, xsg, xsumg, M, y, acc, stream())
    Q.qvla_check_device(stream())
    return y.double().cpu().numpy(), acc.cpu().numpy().astype(np.int64)


def linear(layer, x: torch.Tensor, step: int = -1, ydt="f16"):
    M = x.shape[0]
    xg = x.to(DEV).contiguous()
    y = torch.full((M, layer.N), float("nan"), dtype=TORCH_DT[ydt], device=DEV)
    nbytes = Q.qvla_linear_workspace_bytes(layer, M)
    work = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=DEV)
    Q.qvla_w4a4_linear(layer, xg, M, step, y, work, nbytes, stream())
    Q.qvla_check_device(stream())
    return y.double().cpu().numpy()


def ulp(v: np.ndarray, fmt: str) -> np.ndarray:
    """One unit in the last place of the output format at |v| (normal range)."""
    mant = {"f16": 10, "bf16": 7, "f32": 23}[fmt]
    e = np.floor(np.log2(np.maximum(np.abs(v), 1e-30)))
    return np.exp2(e - mant)


def assert_output_close(got: np.ndarray, ref: np.ndarray, fmt: str = "f16", rel: float = 2e-3):
    """max |y - y_ref| <= rel * max |y_ref| over the tensor: the per-tensor reading of the 2e-3
    maximum relative error stated for fp16 outputs.  bf16 keeps 8 significant bits, so one
    rounding flip alone moves an output by up to 2^-7 of its magnitude; for bf16 each element
    may also differ by one bf16 ulp at its value."""
    assert np.all(np.isfinite(got)), "non-finite output"
    scale = np.abs(ref).max()
    bound = rel * scale + (ulp(ref, "bf16") if fmt == "bf16" else 0.0)
    err = np.abs(got - ref)
    worst = np.argmax(err - bound)
    assert np.all(err <= bound), (f"|y - ref| = {err.flat[worst]:.4g} > bound {np.broadcast_to(bound, err.shape).flat[worst]:.4g}"
                                  f" (max |ref| {scale:.4g})")


def code_mismatch_report(got: np.ndarray, ref: np.ndarray, y_over_delta: np.ndarray):
    """Fraction of differing codes, largest difference, and how near to a rounding tie the
    differing positions lie (|frac(y/Delta)| distance from .5)."""
    d = got.astype(np.int16) - ref.astype(np.int16)
    nz = np.nonzero(d)
    frac = len(nz[0]) / d.size
    maxd = int(np.abs(d).max()) if d.size else 0
    tie_dist = np.abs(np.abs(y_over_delta[nz] - np.floor(y_over_delta[nz])) - 0.5) if len(nz[0]) else np.zeros(0)
    return frac, maxd, (float(tie_dist.max()) if tie_dist.size else 0.0)


def assert_linear_close_modulo_ties(got: np.ndarray, ref: dict, wcodes: np.ndarray, wscale: np.ndarray, bias=None,
                                    fmt: str = "f16", tie: float = 1e-4, max_flip_frac: float = 1e-5,
                                    max_candidates: int = 8) -> np.ndarray:
    """The end-to-end contract of the linear: at most max_flip_frac of the activation codes differ
    from the oracle's, each by one step and only at a rounding tie, and the outputs are within the
    output tolerance of the oracle's arithmetic on the codes used.

    ref is O.w4a4_linear's result.  A row of `got` outside assert_output_close's tolerance must be
    matched by the oracle's own output for that row with some of its near-tie codes (the exact
    quotient within `tie` of a half-integer, not clamped) moved to the other side of the tie.
    Returns the reference with those rows replaced (for exact-match statistics)."""
    from oracle import qvla_oracle as O

    y = ref["y"]
    scale = np.abs(y).max()
    bound = 2e-3 * scale + (ulp(y, "bf16") if fmt == "bf16" else 0.0)
    bound = np.broadcast_to(bound, y.shape)
    assert np.all(np.isfinite(got)), "non-finite output"
    bad_rows = np.nonzero(np.any(np.abs(got - y) > bound, axis=1))[0]
    adjusted = y.copy()
    if bad_rows.size == 0:
        return adjusted
    t = ref["y_rot"].astype(np.float64) / np.asarray(ref["dx"], np.float64)[:, None]
    frac = t - np.floor(t)
    near = (np.abs(frac - 0.5) < tie) & (np.abs(t) < 7.0)
    flips = 0
    for r in bad_rows:
        cand = np.nonzero(near[r])[0]
        assert 0 < cand.size <= max_candidates, f"row {r} differs with {cand.size} codes near a tie"
        matched = None
        for size in range(1, cand.size + 1):
            for subset in __import__("itertools").combinations(cand.tolist(), size):
                q = ref["qx"][r].astype(np.int64).copy()
                for k in subset:  # the other integer next to the tie
                    lo = int(np.floor(t[r, k]))
                    q[k] = lo + 1 if q[k] == lo else lo
                acc = O.int_gemm(q[None, :], wcodes)
                yr = O.dequant_output(acc, np.asarray(ref["dx"])[r:r + 1], wscale, bias, fmt)[0]
                if np.all(np.abs(got[r] - yr) <= bound[r]):
                    matched = (size, yr)
                    break
            if matched:
                break
        assert matched, f"row {r} differs from the oracle by more than moving its near-tie codes explains"
        flips += matched[0]
        adjusted[r] = matched[1]
    assert flips <= max(1.0, max_flip_frac * ref["qx"].size), f"{flips} codes moved at ties"
    return adjusted
