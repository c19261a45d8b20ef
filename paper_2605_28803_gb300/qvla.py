"""ctypes binding of libqvla (include/qvla.h): the same entry points, argument marshalling only.

Tensors are passed as raw pointers (``tensor.data_ptr()``) and streams as
``torch.cuda.Stream.cuda_stream``; every step of the computation runs in libqvla's kernels.
A non-zero status raises QvlaError with the library's message.  Importing this module loads
the in-tree libqvla.so and fails loudly if it has not been built.
"""

from __future__ import annotations

import ctypes
import os

import numpy as np

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libqvla.so")

F16, BF16, F32 = 0, 1, 2
DTYPE_CODES = {"f16": F16, "bf16": BF16, "f32": F32}

STATUS = {0: "QVLA_OK", 1: "QVLA_ERR_INVALID_ARG", 2: "QVLA_ERR_UNSUPPORTED", 3: "QVLA_ERR_CUDA",
          4: "QVLA_ERR_OOM", 5: "QVLA_ERR_STEP_RANGE", 6: "QVLA_ERR_TIMEOUT"}

# every symbol include/*.h declares, with (restype, argtypes)
_P, _I, _S, _D = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_double
SIGNATURES = {
    "qvla_last_error": (ctypes.c_char_p, []),
    "qvla_abi_version": (_I, []),
    "qvla_pack_weights_host": (_I, [_P, _I, _I, _I, _P, _I, _P, _I, _P, _P, _P]),
    "qvla_block_svd_rotation": (_I, [_P, _I, _I, _I, _I, _P, _P]),
    "qvla_gptq_pack_host": (_I, [_P, _I, _I, _I, _P, _I, _I, _P, _I, _P, _I, _I, _D, _P, _P, _P]),
    "qvla_layer_create": (_I, [_I, _I, _I, _I, _I, _P, _P, _P, ctypes.POINTER(_P)]),
    "qvla_layer_create_gated": (_I, [_I, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, ctypes.POINTER(_P)]),
    "qvla_pack_weights": (_I, [_P, _I, _I, _I, _P, _I, _P, _I, _P, _I, _I, ctypes.POINTER(_P)]),
    "qvla_layer_destroy": (_I, [_P]),
    "qvla_set_step_scales": (_I, [_P, _P, _I]),
    "qvla_set_step_group_scales": (_I, [_P, _P, _I, _I]),
    "qvla_layer_scale_groups": (_I, [_P, _P, _P]),
    "qvla_layer_set_online_rotation": (_I, [_P, _P, _P, _I]),
    "qvla_online_rotate": (_I, [_P, _P, _I, _P, _P]),
    "qvla_rotated_absmax_groups": (_I, [_P, _I, _I, _I, _I, _P, _P]),
    "qvla_layer_info": (_I, [_P, _P, _P, _P, _P]),
    "qvla_rotate_quantize": (_I, [_P, _P, _I, _I, _P, _P, _P, _P]),
    "qvla_rotate_quantize_rows": (_I, [_P, _I, _I, _I, _I, _P, _P, _P, _P, _P]),
    "qvla_rotated_absmax": (_I, [_P, _I, _I, _I, _I, _P, _P]),
    "qvla_gemm_w4a4": (_I, [_P, _P, _P, _P, _I, _P, _P, _P]),
    "qvla_linear_workspace_bytes": (_S, [_P, _I]),
    "qvla_w4a4_linear": (_I, [_P, _P, _I, _I, _P, _P, _S, _P]),
    "qvla_linear_quantize": (_I, [_P, _P, _I, _I, _P, _S, _P]),
    "qvla_linear_gemm": (_I, [_P, _P, _S, _I, _P, _P]),
    "qvla_w4a4_linear_noalloc": (_I, [_P, _P, _I, _I, _P, _P]),
    "qvla_w4a4_linear_fused": (_I, [_P, _P, _I, _I, _P, _P]),
    "qvla_rotate_quantize_rows_a8": (_I, [_P, _I, _I, _I, _I, _P, _P, _P, _P, _P]),
    "qvla_w4a8_workspace_bytes": (_S, [_P, _I]),
    "qvla_w4a8_linear": (_I, [_P, _P, _I, _I, _P, _P, _S, _P]),
    "qvla_gemm_w4a8": (_I, [_P, _P, _P, _I, _P, _P, _P, _S, _P]),
    "qvla_check_device": (_I, [_P]),
    "qvla_debug_set_hooks": (_I, [ctypes.c_ulonglong, _I]),
    "qvla_debug_gemm_plan": (_I, [_I, _I, _I, _I, _I, _I, _P, _P]),
}


class QvlaError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status


def load_library(path: str = _LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(f"libqvla.so is not built ({path}); run __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = load_library()


def lib() -> ctypes.CDLL:
    return _lib


def _check(status: int) -> None:
    if status != 0:
        raise QvlaError(status, _lib.qvla_last_error().decode())


def _ptr(t) -> int | None:
    """Raw address of a torch tensor / numpy array (None passes NULL)."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        return None
    return stream if isinstance(stream, int) else stream.cuda_stream


def qvla_abi_version() -> int:
    return _lib.qvla_abi_version()


def qvla_pack_weights_host(W: np.ndarray, wdt: int, N: int, K: int, rot=None, rot_block: int = 0, perm=None,
                           had_block: int = 1, wq=None, wscale=None, wsum=None) -> None:
    """Host-only fold + quantise + pack into caller-provided numpy buffers."""
    _check(_lib.qvla_pack_weights_host(_ptr(W), wdt, N, K, _ptr(rot), rot_block, _ptr(perm), had_block,
                                       _ptr(wq), _ptr(wscale), _ptr(wsum)))


def qvla_gptq_pack_host(W: np.ndarray, wdt: int, N: int, K: int, X: np.ndarray, xdt: int, n_cal: int, rot=None,
                        rot_block: int = 0, perm=None, had_block: int = 1, block: int = 128, damp: float = 0.01,
                        wq=None, wscale=None, wsum=None) -> None:
    """Host-only fold + GPTQ codes against calibration rows X + pack into caller-provided buffers."""
    _check(_lib.qvla_gptq_pack_host(_ptr(W), wdt, N, K, _ptr(X), xdt, n_cal, _ptr(rot), rot_block, _ptr(perm),
                                    had_block, block, float(damp), _ptr(wq), _ptr(wscale), _ptr(wsum)))


def qvla_block_svd_rotation(W: np.ndarray, wdt: int, N: int, K: int, block: int):
    """The zigzag permutation and block SVD factors chosen from the weights; returns
    (perm int32 [K], rot float64 [K/block, block, block])."""
    perm = np.empty(max(K, 1), dtype=np.int32)
    ok = block > 0 and K > 0 and K % block == 0
    rot = np.empty((K // block, block, block) if ok else (1,), dtype=np.float64)  # the library rejects bad shapes
    _check(_lib.qvla_block_svd_rotation(_ptr(np.ascontiguousarray(W)), wdt, N, K, block, _ptr(perm), _ptr(rot)))
    return perm, rot


class Layer:
    """Owner of a qvla_layer handle; ``close()`` (or garbage collection) destroys it."""

    def __init__(self, handle: int, N: int, K: int, had_block: int, xdt: int, ydt: int, gated: bool = False):
        self.handle, self.N, self.K, self.had_block, self.xdt, self.ydt = handle, N, K, had_block, xdt, ydt
        self.gated = gated  # N is the output width (H); the weight rows are 2H

    def close(self) -> None:
        if self.handle:
            _check(_lib.qvla_layer_destroy(self.handle))
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def qvla_layer_create(N: int, K: int, had_block: int, xdt: int, ydt: int, wq: np.ndarray, wscale: np.ndarray,
                      bias=None) -> Layer:
    h = ctypes.c_void_p()
    _check(_lib.qvla_layer_create(N, K, had_block, xdt, ydt, _ptr(wq), _ptr(wscale), _ptr(bias), ctypes.byref(h)))
    return Layer(h.value, N, K, had_block, xdt, ydt)


def qvla_layer_create_gated(H: int, K: int, had_block: int, xdt: int, ydt: int, wq_gate: np.ndarray,
                            wscale_gate: np.ndarray, wq_up: np.ndarray, wscale_up: np.ndarray, bias_gate=None,
                            bias_up=None) -> Layer:
    """Gate + up projections of a gated MLP as one layer whose output is h = gelu(gate) * up."""
    h = ctypes.c_void_p()
    _check(_lib.qvla_layer_create_gated(H, K, had_block, xdt, ydt, _ptr(wq_gate), _ptr(wscale_gate), _ptr(wq_up),
                                        _ptr(wscale_up), _ptr(bias_gate), _ptr(bias_up), ctypes.byref(h)))
    return Layer(h.value, H, K, had_block, xdt, ydt, gated=True)


def qvla_pack_weights(W: np.ndarray, wdt: int, N: int, K: int, rot=None, rot_block: int = 0, perm=None,
                      had_block: int = 1, bias=None, xdt: int = F16, ydt: int = F16) -> Layer:
    h = ctypes.c_void_p()
    _check(_lib.qvla_pack_weights(_ptr(W), wdt, N, K, _ptr(rot), rot_block, _ptr(perm), had_block, _ptr(bias),
                                  xdt, ydt, ctypes.byref(h)))
    return Layer(h.value, N, K, had_block, xdt, ydt)


def qvla_layer_destroy(layer: Layer) -> None:
    layer.close()


def qvla_set_step_scales(layer: Layer, scales: np.ndarray) -> None:
    scales = np.ascontiguousarray(scales, dtype=np.float32)
    _check(_lib.qvla_set_step_scales(layer.handle, _ptr(scales), int(scales.shape[0])))


def qvla_set_step_group_scales(layer: Layer, scales: np.ndarray) -> None:
    """Per-step, per-group table [T, G] (float32)."""
    arr = np.ascontiguousarray(scales, dtype=np.float32)
    if arr.ndim != 2:
        raise ValueError("scales must be [T, G]")
    _check(_lib.qvla_set_step_group_scales(layer.handle, _ptr(arr), arr.shape[0], arr.shape[1]))


def qvla_layer_set_online_rotation(layer: Layer, perm=None, rot=None, rot_block: int = 0) -> None:
    """Online x . P . BlockDiag(U_b) ahead of the layer's quantiser (perm int32 [K], rot float64
    [K/rot_block, rot_block, rot_block]); both None removes it."""
    p = None if perm is None else np.ascontiguousarray(perm, dtype=np.int32)
    r = None if rot is None else np.ascontiguousarray(rot, dtype=np.float64)
    _check(_lib.qvla_layer_set_online_rotation(layer.handle, _ptr(p), _ptr(r), int(rot_block)))


def qvla_online_rotate(layer: Layer, x, M: int, out, stream=None) -> None:
    _check(_lib.qvla_online_rotate(layer.handle, _ptr(x), M, _ptr(out), _stream(stream)))


def qvla_layer_scale_groups(layer: Layer):
    g, size = ctypes.c_int(), ctypes.c_int()
    _check(_lib.qvla_layer_scale_groups(layer.handle, ctypes.byref(g), ctypes.byref(size)))
    return g.value, size.value


def qvla_rotated_absmax_groups(x, xdt: int, M: int, K: int, had_block: int, absmax, stream=None) -> None:
    _check(_lib.qvla_rotated_absmax_groups(_ptr(x), xdt, M, K, had_block, _ptr(absmax), _stream(stream)))


def qvla_layer_info(layer: Layer):
    n, k, b, t = ctypes.c_int(), ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check(_lib.qvla_layer_info(layer.handle, ctypes.byref(n), ctypes.byref(k), ctypes.byref(b), ctypes.byref(t)))
    return n.value, k.value, b.value, t.value


def qvla_rotate_quantize(layer: Layer, x, M: int, step: int, xq, xscale, xsum=None, stream=None) -> None:
    _check(_lib.qvla_rotate_quantize(layer.handle, _ptr(x), M, step, _ptr(xq), _ptr(xscale), _ptr(xsum),
                                     _stream(stream)))


def qvla_rotate_quantize_rows(x, xdt: int, M: int, K: int, had_block: int, step_scale, xq, xscale, xsum=None,
                              stream=None) -> None:
    _check(_lib.qvla_rotate_quantize_rows(_ptr(x), xdt, M, K, had_block, _ptr(step_scale), _ptr(xq), _ptr(xscale),
                                          _ptr(xsum), _stream(stream)))


def qvla_rotated_absmax(x, xdt: int, M: int, K: int, had_block: int, absmax, stream=None) -> None:
    _check(_lib.qvla_rotated_absmax(_ptr(x), xdt, M, K, had_block, _ptr(absmax), _stream(stream)))


def qvla_gemm_w4a4(layer: Layer, xq, xscale, xsum, M: int, y, acc=None, stream=None) -> None:
    _check(_lib.qvla_gemm_w4a4(layer.handle, _ptr(xq), _ptr(xscale), _ptr(xsum), M, _ptr(y), _ptr(acc),
                               _stream(stream)))


def qvla_linear_workspace_bytes(layer: Layer, M: int) -> int:
    return int(_lib.qvla_linear_workspace_bytes(layer.handle, M))


def qvla_w4a4_linear(layer: Layer, x, M: int, step: int, y, workspace, workspace_bytes: int, stream=None) -> None:
    _check(_lib.qvla_w4a4_linear(layer.handle, _ptr(x), M, step, _ptr(y), _ptr(workspace), workspace_bytes,
                                 _stream(stream)))


def qvla_linear_quantize(layer: Layer, x, M: int, step: int, workspace, workspace_bytes: int, stream=None) -> None:
    _check(_lib.qvla_linear_quantize(layer.handle, _ptr(x), M, step, _ptr(workspace), workspace_bytes,
                                     _stream(stream)))


def qvla_linear_gemm(layer: Layer, workspace, workspace_bytes: int, M: int, y, stream=None) -> None:
    _check(_lib.qvla_linear_gemm(layer.handle, _ptr(workspace), workspace_bytes, M, _ptr(y), _stream(stream)))


NOALLOC_SCRATCH_BYTES = 8 << 20


def qvla_w4a4_linear_fused(layer: Layer, x, M: int, step: int, y, stream=None) -> None:
    """The one-launch linear (small batch, per-step scale); QvlaError status 2 where it does not apply."""
    _check(_lib.qvla_w4a4_linear_fused(layer.handle, _ptr(x), M, step, _ptr(y), _stream(stream)))


def qvla_w4a4_linear_noalloc(layer: Layer, x, M: int, step: int, y, stream=None) -> None:
    """qvla_w4a4_linear without a caller workspace: for callers that cannot allocate device
    memory while running; the library's fixed 8 MiB scratch takes the workspace's place."""
    _check(_lib.qvla_w4a4_linear_noalloc(layer.handle, _ptr(x), M, step, _ptr(y), _stream(stream)))


def qvla_rotate_quantize_rows_a8(x, xdt: int, M: int, K: int, had_block: int, step_scale, xq, xscale, xsum=None,
                                 stream=None) -> None:
    _check(_lib.qvla_rotate_quantize_rows_a8(_ptr(x), xdt, M, K, had_block, _ptr(step_scale), _ptr(xq),
                                             _ptr(xscale), _ptr(xsum), _stream(stream)))


def qvla_w4a8_workspace_bytes(layer: Layer, M: int) -> int:
    return int(_lib.qvla_w4a8_workspace_bytes(layer.handle, M))


def qvla_w4a8_linear(layer: Layer, x, M: int, step: int, y, workspace, workspace_bytes: int, stream=None) -> None:
    _check(_lib.qvla_w4a8_linear(layer.handle, _ptr(x), M, step, _ptr(y), _ptr(workspace), workspace_bytes,
                                 _stream(stream)))


def qvla_gemm_w4a8(layer: Layer, xq, xscale, M: int, y, acc, workspace, workspace_bytes: int, stream=None) -> None:
    _check(_lib.qvla_gemm_w4a8(layer.handle, _ptr(xq), _ptr(xscale), M, _ptr(y), _ptr(acc), _ptr(workspace),
                               workspace_bytes, _stream(stream)))


def qvla_check_device(stream=None) -> None:
    _check(_lib.qvla_check_device(_stream(stream)))


def qvla_debug_set_hooks(wait_limit_ns: int = 0, hold_gemm_loads: bool = False) -> None:
    """Test hooks (include/qvla_debug.h): the device wait limit (0 = default) and whether GEMM
    load warps hold back every copy."""
    _check(_lib.qvla_debug_set_hooks(int(wait_limit_ns), 1 if hold_gemm_loads else 0))


GEMM_SHAPES = ("single 128x128", "single 128x256", "pair 256x128", "pair 256x256")


def qvla_debug_gemm_plan(M: int, K: int, N: int, gated: bool = False, num_sms: int = 152,
                         split_room: bool = True) -> tuple[str, int]:
    """The token-major GEMM's launch plan (include/qvla_debug.h): (tile shape, work units per
    tile) for M > 128 tokens of an M x K -> N layer (N weight rows, 2H when gated).  Host only."""
    shape, parts = ctypes.c_int(-1), ctypes.c_int(0)
    _check(_lib.qvla_debug_gemm_plan(M, K, N, 1 if gated else 0, num_sms, 1 if split_room else 0,
                                     ctypes.addressof(shape), ctypes.addressof(parts)))
    return GEMM_SHAPES[shape.value], parts.value
