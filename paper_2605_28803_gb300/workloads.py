"""Seeded synthetic inputs shaped like the backbone and DiT layers of the paper's VLA models.

This module only draws random numbers: it holds none of the quantized linear's
arithmetic.  The paper evaluates on LIBERO rollouts of Pi-0.5 / GR00T N1.5, which need
a simulator and model weights; these generators stand in for them with the layer shapes,
dtypes and outlier structure of those models:

* Gaussian activations with a few outlier channels scaled by a fixed factor;
* heavy-tailed (Student-t) channels for the backbone MLP input;
* weights ~ N(0, sigma^2) with sigma = 0.02 or 1/sqrt(K);
* a random orthogonal matrix standing in for the SVD factor (QR of a Gaussian,
  with the sign fix diag(R) > 0);
* per-step activation magnitudes for the DiT head, drifting geometrically across steps.

Every draw uses numpy's PCG64 ``default_rng(seed)`` in a fixed order, so the same seed
gives the same tensors on every machine.
"""

from __future__ import annotations

from dataclasses import dataclass, replace, field

import numpy as np
import torch

_TORCH_DTYPES = {"f16": torch.float16, "bf16": torch.bfloat16, "f32": torch.float32}


def as_dtype(x: np.ndarray, dtype: str) -> torch.Tensor:
    """A float array as a CPU torch tensor of the activation/weight dtype."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(_TORCH_DTYPES[dtype])


def random_orthogonal(rng: np.random.Generator, n: int) -> np.ndarray:
    """A random orthogonal n x n matrix (float64): Q of a Gaussian's QR, sign-fixed."""
    a = rng.standard_normal((n, n))
    q, r = np.linalg.qr(a)
    return q * np.sign(np.diag(r))[None, :]


def gaussian_with_outliers(rng, m: int, k: int, n_outliers: int, factor: float) -> np.ndarray:
    """X ~ N(0, 1) [m, k] (float32) with n_outliers fixed channels multiplied by factor."""
    x = rng.standard_normal((m, k), dtype=np.float32)
    if n_outliers:
        idx = rng.choice(k, n_outliers, replace=False)
        x[:, idx] *= np.float32(factor)
    return x


def gaussian_with_heavy_channels(rng, m: int, k: int, frac: float, nu: float) -> np.ndarray:
    """X ~ N(0, 1) [m, k] (float32) whose channels in a random fraction frac are Student-t(nu)."""
    x = rng.standard_normal((m, k), dtype=np.float32)
    n_heavy = max(1, int(round(frac * k)))
    idx = rng.choice(k, n_heavy, replace=False)
    x[:, idx] = rng.standard_t(nu, size=(m, n_heavy)).astype(np.float32)
    return x


def gaussian_weights(rng, n: int, k: int, sigma: float) -> np.ndarray:
    """W ~ N(0, sigma^2) [n, k], float32, stored [out_features, in_features]."""
    return rng.standard_normal((n, k), dtype=np.float32) * np.float32(sigma)


# --------------------------------------------------------------------------------------
# The workloads (sizes are those of the paper's Pi-0.5-shaped layers)
# --------------------------------------------------------------------------------------

@dataclass
class SingleLayerWithSteps:
    """One linear whose input is scaled per denoising step (DiT-style per-step scales)."""
    x_steps: list            # T activation tensors [M, K] (torch, dtype), in the rotated basis
    x_orig_steps: list       # the same before the upstream SVD-factor rotation (float64)
    w: np.ndarray            # [N, K] float32 values of the given wdtype
    rot: np.ndarray | None   # [K/rot_block, rot_block, rot_block] float64, or None
    rot_block: int | None
    had_block: int
    xdtype: str
    ydtype: str


def single_layer_steps(seed: int = 0, m: int = 64, k: int = 512, n: int = 512, steps: int = 10,
                       n_outliers: int = 4, outlier_factor: float = 20.0, w_sigma: float = 0.02,
                       step_growth: float = 0.3, had_block: int = 512) -> SingleLayerWithSteps:
    """Single W4A4 layer (64 x 512 x 512 by default): X fp16 ~ N(0,1) with 4 channels x20,
    W fp16 ~ N(0, 0.02^2), a random orthogonal stand-in for the SVD factor (folded into W
    and applied upstream to X), Hadamard block 512, T = 10 steps with X_t = X (1 + 0.3 t).
    Draw order: X, outlier channels, W, U."""
    rng = np.random.default_rng(seed)
    x = gaussian_with_outliers(rng, m, k, n_outliers, outlier_factor).astype(np.float64)
    w = as_dtype(gaussian_weights(rng, n, k, w_sigma), "f16").float().numpy()
    u = random_orthogonal(rng, k)
    xs, xo = [], []
    for t in range(steps):
        xt = x * (1.0 + step_growth * t)
        xo.append(xt)
        xs.append(as_dtype(xt @ u, "f16"))
    return SingleLayerWithSteps(xs, xo, w, u[None], k, had_block, "f16", "f16")


@dataclass
class GatedMLP:
    """Backbone-shaped gated MLP: gate/up K -> H each, GELU-gated product, down H -> K."""
    x: torch.Tensor          # [M, K] bf16
    w_gate: np.ndarray       # [H, K] float32
    w_up: np.ndarray         # [H, K]
    w_down: np.ndarray       # [K, H]
    had_in: int
    had_hidden: int
    xdtype: str = "bf16"


def gated_mlp(seed: int = 1, m: int = 816, k: int = 2048, hidden: int = 16384,
              heavy_frac: float = 0.01, nu: float = 2.0, had_in: int = 2048, had_hidden: int = 2048) -> GatedMLP:
    """Prefix of M = 816 tokens (3 x 256 image + 48 text), hidden 2048, MLP 2048 -> 2 x 16384
    -> 2048.  X ~ N(0,1) bf16 with 1% Student-t(2) channels, W ~ N(0, 1/fan_in).
    Draw order: X, heavy channels, W_gate, W_up, W_down."""
    rng = np.random.default_rng(seed)
    x = gaussian_with_heavy_channels(rng, m, k, heavy_frac, nu)
    wg = gaussian_weights(rng, hidden, k, 1.0 / np.sqrt(k))
    wu = gaussian_weights(rng, hidden, k, 1.0 / np.sqrt(k))
    wd = gaussian_weights(rng, k, hidden, 1.0 / np.sqrt(hidden))
    return GatedMLP(as_dtype(x, "bf16"), wg, wu, wd, had_in, had_hidden)


@dataclass
class LinearCase:
    """One linear of a sweep: activations, weights and the rotation block."""
    x: torch.Tensor
    w: np.ndarray
    bias: np.ndarray | None
    had_block: int
    xdtype: str
    ydtype: str
    extra: dict = field(default_factory=dict)


def sweep_linear(m: int, k: int, n: int, seed: int = 4, outlier_frac: float = 0.005,
                 outlier_factor: float = 20.0, xdtype: str = "bf16", ydtype: str = "bf16",
                 had_block: int | None = None, with_bias: bool = False) -> LinearCase:
    """One point of the single-linear sweep: X ~ N(0,1) with 0.5% channels x20,
    W ~ N(0, 1/K).  Hadamard block = K up to 4096, else 2048.  Draw order: X, outlier
    channels, W, bias."""
    rng = np.random.default_rng(seed)
    x = gaussian_with_outliers(rng, m, k, max(1, int(round(outlier_frac * k))), outlier_factor)
    w = gaussian_weights(rng, n, k, 1.0 / np.sqrt(k))
    bias = rng.standard_normal(n).astype(np.float32) * np.float32(0.1) if with_bias else None
    if had_block is None:
        had_block = k if k <= 4096 else 2048
    return LinearCase(as_dtype(x, xdtype), w, bias, had_block, xdtype, ydtype)


def sweep_input_device(m: int, k: int, seed: int, device, dtype: str = "f16", outlier_frac: float = 0.005,
                       outlier_factor: float = 20.0) -> torch.Tensor:
    """Sweep activations drawn on the device with torch's seeded generator (the largest sweep
    points hold 134 M values, seconds of host drawing): N(0,1) [m, k] with round(0.5% K)
    channels x20.  Draw order: X, then the outlier channels."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    x = torch.randn(m, k, generator=g, device=device, dtype=torch.float32)
    idx = torch.randperm(k, generator=g, device=device)[:max(1, int(round(outlier_frac * k)))]
    x[:, idx] *= outlier_factor
    return x.to(_TORCH_DTYPES[dtype])


def dit_input_std(t: int, steps: int = 10, start: float = 4.0, end: float = 0.5) -> float:
    """Per-step input magnitude of the DiT head: geometric drift from 4.0 at t = 0 to 0.5
    at t = T-1, i.e. sigma_t = 4 (1/8)^(t / 9) for T = 10."""
    return start * (end / start) ** (t / (steps - 1))


def dit_step_inputs(rng, m: int, k: int, steps: int = 10) -> list:
    """Activations of one DiT linear for every step: N(0, sigma_t^2) [m, k] float32."""
    base = rng.standard_normal((m, k), dtype=np.float32)
    return [base * np.float32(dit_input_std(t, steps)) for t in range(steps)]


DIT_LAYER_SHAPES = (("q", 1024, 1024), ("k", 1024, 1024), ("v", 1024, 1024), ("o", 1024, 1024),
                    ("up", 1024, 4096), ("down", 4096, 1024))
"""(name, in_features K, out_features N) of one DiT block of the action head."""

BACKBONE_LAYER_SHAPES = (("q", 2048, 2048), ("k", 2048, 256), ("v", 2048, 256), ("o", 2048, 2048),
                         ("gate", 2048, 16384), ("up", 2048, 16384), ("down", 16384, 2048))
"""(name, K, N) of one backbone decoder layer (Gemma-2B-like, 18 layers)."""


# --------------------------------------------------------------------------------------
# Layer stacks: pre-rotated, pre-quantised weights drawn directly as int4 codes
# --------------------------------------------------------------------------------------

def pack_nibbles(codes: np.ndarray) -> np.ndarray:
    """int8 codes [..., K] in [-8, 7] -> the packed storage layout (byte j: code 2j in the low
    nibble, code 2j+1 in the high nibble, 4-bit two's complement), uint8 [..., K/2]."""
    u = (np.asarray(codes).astype(np.int16) & 0xF).astype(np.uint8)
    return np.ascontiguousarray(u[..., 0::2] | (u[..., 1::2] << 4))


@dataclass
class StackWeights:
    """One linear of a stack: its weights as int4 codes (what the offline fold and quantiser
    would produce) with per-output-channel scales.  For a gated layer the rows are the H gate
    rows, then the H up rows."""
    name: str
    k: int
    n: int                    # output features (H for a gated layer)
    had_block: int
    packed: np.ndarray        # uint8 [rows, k/2]
    wscale: np.ndarray        # float32 [rows]
    bias: np.ndarray | None   # float32 [rows] or None
    gated: bool = False
    codes: np.ndarray | None = None  # int8 [rows, k] when drawn as codes

    def weight_codes(self) -> np.ndarray:
        """int8 codes [rows, k], unpacked from the storage layout when not kept."""
        if self.codes is not None:
            return self.codes
        b = self.packed
        out = np.empty(b.shape[:-1] + (b.shape[-1] * 2,), dtype=np.int8)
        lo = (b & 0xF).astype(np.int16)
        hi = (b >> 4).astype(np.int16)
        out[..., 0::2] = np.where(lo > 7, lo - 16, lo)
        out[..., 1::2] = np.where(hi > 7, hi - 16, hi)
        return out


def gaussian_codes(rng, rows: int, k: int, sigma: float = 2.0) -> np.ndarray:
    """Weight codes shaped like per-channel int4 codes of Gaussian weights: N(0, sigma^2)
    rounded to integers and clipped to [-7, 7], int8 [rows, k]."""
    return np.clip(np.rint(rng.standard_normal((rows, k), dtype=np.float32) * np.float32(sigma)), -7, 7).astype(np.int8)


def _weight_scales(rng, rows: int, k: int) -> np.ndarray:
    """Per-channel scales of weights ~ N(0, 1/K): about max|w| / 7 ~ 0.5 / sqrt(K), +-20%."""
    return (rng.uniform(0.8, 1.2, rows) * 0.5 / np.sqrt(k)).astype(np.float32)


DIT_STACK_LAYERS = (("qkv", 1024, 3072), ("o", 1024, 1024), ("up", 1024, 4096), ("down", 4096, 1024))
"""(name, K, N) of one DiT block as run: Q, K and V read the same input with the same per-step
table, so they form one 1024 -> 3072 linear whose output columns are [Q | K | V]."""


def dit_stack(seed: int = 2, layers: int = 18) -> list:
    """Weights of the DiT action head's 18 blocks: per block qkv 1024 -> 3072, o 1024 -> 1024,
    up 1024 -> 4096, down 4096 -> 1024, Hadamard block = K, with biases.  Codes ~ rounded
    N(0, 2^2) in [-7, 7].  Draw order per layer and linear: codes, scales, bias."""
    rng = np.random.default_rng(seed)
    out = []
    for layer in range(layers):
        for name, k, n in DIT_STACK_LAYERS:
            codes = gaussian_codes(rng, n, k)
            ws = _weight_scales(rng, n, k)
            bias = (rng.standard_normal(n, dtype=np.float32) * np.float32(0.05)).astype(np.float32)
            out.append(StackWeights(f"{layer}.{name}", k, n, k, pack_nibbles(codes), ws, bias, codes=codes))
    return out


def dit_layer_input(seed: int, index: int, t: int, m: int, k: int, steps: int = 10,
                    channel_profile: bool = False) -> np.ndarray:
    """Input of linear `index` of the DiT stack at denoising step t: N(0, sigma_t^2) [m, k]
    float32 with sigma_t drifting from 4.0 (t = 0) to 0.5 (t = T-1).  Each (index, t) has its
    own stream, so any subset can be drawn.  channel_profile: every block of 64 channels is
    also multiplied by its own log-normal factor (spread 0.8, fixed per linear), the uneven
    channel magnitudes that per-group scales are for."""
    rng = np.random.default_rng([seed, index, t])
    x = rng.standard_normal((m, k), dtype=np.float32) * np.float32(dit_input_std(t, steps))
    if channel_profile:
        prof = np.exp(np.random.default_rng([seed, index, 7919]).normal(0.0, 0.8, k // 64)).astype(np.float32)
        x *= np.repeat(prof, 64)[None, :]
    return x


def dit_stack_blocks(weights, had_block: int = 64) -> list:
    """The same DiT weights with the paper's rotation block (Sec. 5.1: block size 64) as the
    layers' Hadamard block, for per-group step scales over 128-channel groups."""
    return [replace(w, had_block=had_block) for w in weights]


BACKBONE_STACK_LAYERS = (("qkv", 2048, 2560, False), ("o", 2048, 2048, False), ("gate_up", 2048, 16384, True),
                         ("down", 16384, 2048, False))
"""(name, K, N, gated) of one backbone layer as run: Q (2048) and K/V (256 each) share their
input and form one 2048 -> 2560 linear; gate and up (2048 -> 16384 each) form one gated layer
whose output is gelu(gate) * up."""


def backbone_stack(seed: int = 3, layers: int = 18, had_wide: int = 2048) -> list:
    """Weights of the 18-layer backbone (hidden 2048, MLP 16384): 1.98 G int4 codes drawn as
    uniform random bytes (codes uniform in [-8, 7]; the packed format carries -8), with
    per-channel scales and no bias.  Hadamard block = K for K = 2048, 8 x 2048 blocks for
    K = 16384.  Draw order per layer and linear: bytes, scales."""
    rng = np.random.default_rng(seed)
    out = []
    for layer in range(layers):
        for name, k, n, gated in BACKBONE_STACK_LAYERS:
            rows = 2 * n if gated else n
            packed = rng.integers(0, 256, (rows, k // 2), dtype=np.uint8)
            ws = _weight_scales(rng, rows, k)
            out.append(StackWeights(f"{layer}.{name}", k, n, min(k, had_wide), packed, ws, None, gated=gated))
    return out


def backbone_layer_input(seed: int, index: int, m: int, k: int, frac: float = 0.002, factor: float = 20.0) -> np.ndarray:
    """Input of linear `index` of the backbone stack: N(0, 1) [m, k] float32 with a fixed 0.2%
    of channels (per linear) scaled x20."""
    rng = np.random.default_rng([seed, index])
    n_out = max(1, int(round(frac * k)))
    idx = rng.choice(k, n_out, replace=False)
    x = rng.standard_normal((m, k), dtype=np.float32)
    x[:, idx] *= np.float32(factor)
    return x
