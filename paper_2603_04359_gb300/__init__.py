"""Block Concentration-Alignment Transform (CAT) W4A4 linear layer on GB300 (sm_103a).

A thin ctypes binding of the C ABI in ``include/cat_w4a4.h``: every function below has the name
of the C entry point it calls, takes torch tensors, allocates outputs with torch on the tensors'
device when none are given, passes raw pointers and the current CUDA stream, and raises
``CatError`` on a non-zero status.  All arithmetic runs in the library's CUDA kernels (or, for
``cat_build_transform_host``, in its host code); there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional, Tuple

import numpy as np
import torch

__all__ = [
    "CatError", "library_path", "load_library", "exported_symbols",
    "cat_calib_cov", "cat_quantize_weights", "cat_build_transform_host", "cat_transform_quantize_act",
    "cat_w4a4_linear", "cat_sqnr", "cat_device_status", "cat_version", "KIND",
    "cat_dp_planes", "cat_transform_quantize_act_dp", "cat_quantize_weights_dp", "cat_linear_dp",
    "cat_block_transform", "cat_dequantize_codes", "cat_gemm_f32", "one_sided_sqnr", "cat_set_wait_limit_ns",
    "cat_transform_quantize_act_hd", "cat_fwht_rows", "cat_gram_f32", "cat_alignment_ceiling_host",
    "cat_split_transform", "cat_split_transform_bytes", "cat_transform_quantize_act_split",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libcatw4a4.so")
_HEADER = os.path.join(os.path.dirname(_HERE), "include", "cat_w4a4.h")
_lib: Optional[ctypes.CDLL] = None

KIND = {"identity": 0, "rht": 1, "cat": 2, "cat_diag": 3, "cat_hd": 4}
_DTYPE = {torch.float32: 0, torch.bfloat16: 1}
_STATUS = {0: "CAT_OK", 1: "CAT_ERR_INVALID_ARG", 2: "CAT_ERR_SHAPE", 3: "CAT_ERR_ALIGNMENT", 4: "CAT_ERR_NUMERIC",
           5: "CAT_ERR_UNSUPPORTED", 6: "CAT_ERR_CUDA", 7: "CAT_ERR_TIMEOUT"}


class CatError(RuntimeError):
    def __init__(self, func: str, status: int, message: str):
        super().__init__(f"{func}: {_STATUS.get(status, status)}: {message}")
        self.status = status


def library_path() -> str:
    return _LIB_PATH


def load_library() -> ctypes.CDLL:
    """Load ``libcatw4a4.so`` (built in-tree by ``paper_2603_04359_gb300.build``); fail loudly if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise ImportError(f"{_LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(_LIB_PATH)
    P, I64, I32, I = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int
    sigs = {
        "cat_status_string": ([I], ctypes.c_char_p),
        "cat_last_error": ([], ctypes.c_char_p),
        "cat_version": ([], I),
        "cat_kernel_launches": ([], ctypes.c_ulonglong),
        "cat_calib_cov": ([P, I, I64, I64, I32, P, I, P], I),
        "cat_quantize_weights": ([P, I, I64, I64, I32, I, P, I64, P, P, P, P, P], I),
        "cat_quantize_weights_noalloc": ([P, I, I64, I64, I32, I, P, I64, P, P, P, P, P], I),
        "cat_build_transform_host": ([I, I64, I32, P, I64, P, P, P, P], I),
        "cat_transform_quantize_act": ([P, I, I64, I64, I32, P, P, P, P], I),
        "cat_w4a4_linear": ([P, P, P, P, I64, I64, I64, P, P, P], I),
        "cat_sqnr": ([P, P, I64, P, P], I),
        "cat_w4a4_linear_sqnr": ([P, P, P, P, I64, I64, I64, P, P, P, P], I),
        "cat_device_status": ([P, P], I),
        "cat_block_row_stats": ([P, I, I64, I64, I32, P, I, P, P, P, P], I),
        "cat_dp_planes": ([I32], I32),
        "cat_set_wait_limit_ns": ([ctypes.c_uint64], I),
        "cat_block_transform": ([P, I, I64, I64, I32, P, I, P, P], I),
        "cat_dequantize_codes": ([P, P, I64, I64, P, P], I),
        "cat_gemm_f32": ([P, P, I64, I64, I64, P, P], I),
        "cat_transform_quantize_act_hd": ([P, I, I64, I64, I32, P, P, P, P], I),
        "cat_split_transform": ([P, I64, I32, P, P], I),
        "cat_split_transform_bytes": ([I64, I32], I64),
        "cat_transform_quantize_act_split": ([P, I, I64, I64, I32, P, P, P, P, P], I),
        "cat_fwht_rows": ([P, I64, I64, P], I),
        "cat_gram_f32": ([P, I, I64, I64, P, P], I),
        "cat_alignment_ceiling_host": ([P, P, I64, P], I),
        "cat_transform_quantize_act_dp": ([P, I, I64, I64, I32, P, I32, I32, P, P, P, P], I),
        "cat_quantize_weights_dp": ([P, I, I64, I64, I32, I, P, I64, P, I32, I32, P, P, P, P, P], I),
        "cat_linear_dp": ([P, I32, I32, P, P, P, I32, P, P, I64, I64, I64, P, P, P], I),
        "cat_codes_to_e4m3": ([P, I64, I64, P, P], I),
        "cat_transform_quantize_act_e8": ([P, I, I64, I64, I32, P, P, P, P, P], I),
        "cat_w4a4_linear_e8": ([P, P, P, P, I64, I64, I64, P, P, P], I),
        "cat_w4a4_linear_sqnr_e8": ([P, P, P, P, I64, I64, I64, P, P, P, P], I),
    }
    for name, (args, res) in sigs.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    _lib = lib
    return lib


def exported_symbols() -> list:
    """Names of the entry points declared in ``include/cat_w4a4.h``."""
    with open(_HEADER) as f:
        text = f.read()
    return sorted(set(re.findall(r"^\s*(?:cat_status|const char\*|int|int32_t|int64_t|unsigned long long)\s+(cat_\w+)\s*\(", text,
                                 re.M)))


def _check(func: str, status: int) -> None:
    if status != 0:
        msg = load_library().cat_last_error().decode()
        raise CatError(func, status, msg)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(device: torch.device):
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _dtype(t: torch.Tensor) -> int:
    if t.dtype not in _DTYPE:
        raise TypeError(f"unsupported dtype {t.dtype}; expected float32 or bfloat16")
    return _DTYPE[t.dtype]


def _need(t: torch.Tensor, name: str) -> None:
    if not (t.is_cuda and t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous CUDA tensor")


def _expect(t: torch.Tensor, name: str, dtype: torch.dtype, shape: tuple, device: torch.device) -> None:
    """Check a tensor handed to the library (an input it reads or an output it writes): contiguous,
    on ``device``, of the given dtype and shape.  The library trusts sizes, so a wrong buffer would
    be read or written past its end; this raises ValueError before any call."""
    if not isinstance(t, torch.Tensor):
        raise ValueError(f"{name} must be a torch tensor")
    _need(t, name)
    if t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")
    if t.dtype != dtype:
        raise ValueError(f"{name} has dtype {t.dtype}, expected {dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")


def cat_version() -> int:
    return int(load_library().cat_version())


def cat_kernel_launches() -> int:
    """Kernels the library has launched in this process (diagnostic host counter)."""
    return int(load_library().cat_kernel_launches())


def cat_calib_cov(x: torch.Tensor, k: int, out: Optional[torch.Tensor] = None, accumulate: bool = False) -> torch.Tensor:
    """Sums of x_b x_b^T over tokens for every k x k diagonal block: float64 [d/k, k, k]."""
    _need(x, "x")
    n, d = x.shape
    if out is None:
        out = torch.empty((d // k, k, k), dtype=torch.float64, device=x.device)
    _expect(out, "out", torch.float64, (d // k, k, k), x.device)
    _check("cat_calib_cov", load_library().cat_calib_cov(_ptr(x), _dtype(x), n, d, k, _ptr(out), int(accumulate),
                                                         _stream(x.device)))
    return out


def cat_quantize_weights(W: torch.Tensor, k: int, kind: str, sigma_x: Optional[torch.Tensor] = None, n_calib: int = 0,
                         rht_signs=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """Offline weight preparation.  Returns (T_blocks float32 [d_in/k,k,k], Wq uint8 [d_out, d_in/2],
    w_scale float32 [d_out])."""
    _need(W, "W")
    d_out, d_in = W.shape
    dev = W.device
    T = torch.empty((d_in // k, k, k), dtype=torch.float32, device=dev)
    Wq = torch.empty((d_out, d_in // 2), dtype=torch.uint8, device=dev)
    sw = torch.empty((d_out,), dtype=torch.float32, device=dev)
    signs = None
    if rht_signs is not None:
        signs = np.ascontiguousarray(np.asarray(rht_signs, dtype=np.float32))
    if sigma_x is not None:
        _expect(sigma_x, "sigma_x", torch.float64, (d_in // k, k, k), dev)
    if signs is not None and signs.shape != (d_in,):
        raise ValueError(f"rht_signs has shape {signs.shape}, expected ({d_in},)")
    st = load_library().cat_quantize_weights(
        _ptr(W), _dtype(W), d_out, d_in, k, KIND[kind], _ptr(sigma_x), int(n_calib),
        None if signs is None else signs.ctypes.data_as(ctypes.c_void_p), _ptr(T), _ptr(Wq), _ptr(sw), _stream(dev))
    _check("cat_quantize_weights", st)
    return T, Wq, sw


def cat_quantize_weights_noalloc(W: torch.Tensor, k: int, kind: str, sigma_x: Optional[torch.Tensor] = None,
                                 n_calib: int = 0, rht_signs=None, out=None) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """cat_quantize_weights with the library's static scratch instead of device allocations
    (d_in * k <= 1048576).  ``out`` = (T_blocks, Wq, w_scale) preallocated by the caller, or None."""
    _need(W, "W")
    d_out, d_in = W.shape
    dev = W.device
    if out is None:
        out = (torch.empty((d_in // k, k, k), dtype=torch.float32, device=dev),
               torch.empty((d_out, d_in // 2), dtype=torch.uint8, device=dev),
               torch.empty((d_out,), dtype=torch.float32, device=dev))
    T, Wq, sw = out
    _expect(T, "out[0] (T_blocks)", torch.float32, (d_in // k, k, k), dev)
    _expect(Wq, "out[1] (Wq)", torch.uint8, (d_out, d_in // 2), dev)
    _expect(sw, "out[2] (w_scale)", torch.float32, (d_out,), dev)
    signs = None
    if rht_signs is not None:
        signs = np.ascontiguousarray(np.asarray(rht_signs, dtype=np.float32))
        if signs.shape != (d_in,):
            raise ValueError(f"rht_signs has shape {signs.shape}, expected ({d_in},)")
    if sigma_x is not None:
        _expect(sigma_x, "sigma_x", torch.float64, (d_in // k, k, k), dev)
    st = load_library().cat_quantize_weights_noalloc(
        _ptr(W), _dtype(W), d_out, d_in, k, KIND[kind], _ptr(sigma_x), int(n_calib),
        None if signs is None else signs.ctypes.data_as(ctypes.c_void_p), _ptr(T), _ptr(Wq), _ptr(sw), _stream(dev))
    _check("cat_quantize_weights_noalloc", st)
    return T, Wq, sw


def cat_build_transform_host(kind: str, d_in: int, k: int, sigma_x: Optional[np.ndarray] = None, n_calib: int = 0,
                             sigma_w: Optional[np.ndarray] = None, rht_signs=None) -> Tuple[np.ndarray, np.ndarray]:
    """Host float64 block transform (T, T^{-1}), each [d_in/k, k, k]."""
    nb = d_in // k
    T = np.zeros((nb, k, k), dtype=np.float64)
    Ti = np.zeros((nb, k, k), dtype=np.float64)
    sx = None if sigma_x is None else np.ascontiguousarray(sigma_x, dtype=np.float64)
    sw = None if sigma_w is None else np.ascontiguousarray(sigma_w, dtype=np.float64)
    sg = None if rht_signs is None else np.ascontiguousarray(rht_signs, dtype=np.float32)
    vp = lambda a: None if a is None else a.ctypes.data_as(ctypes.c_void_p)  # noqa: E731
    st = load_library().cat_build_transform_host(KIND[kind], d_in, k, vp(sx), int(n_calib), vp(sw), vp(sg), vp(T),
                                                 vp(Ti))
    _check("cat_build_transform_host", st)
    return T, Ti


def cat_transform_quantize_act(x: torch.Tensor, T_blocks: torch.Tensor, k: int, xq: Optional[torch.Tensor] = None,
                               x_scale: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """x' = T x, per-token INT4 codes (SM4x8 uint8 [n, d_in/2]) and steps (float32 [n])."""
    _need(x, "x")
    _need(T_blocks, "T_blocks")
    n, d_in = x.shape
    if xq is None:
        xq = torch.empty((n, d_in // 2), dtype=torch.uint8, device=x.device)
    if x_scale is None:
        x_scale = torch.empty((n,), dtype=torch.float32, device=x.device)
    _expect(T_blocks, "T_blocks", torch.float32, (d_in // k, k, k), x.device)
    _expect(xq, "xq", torch.uint8, (n, d_in // 2), x.device)
    _expect(x_scale, "x_scale", torch.float32, (n,), x.device)
    _check("cat_transform_quantize_act", load_library().cat_transform_quantize_act(
        _ptr(x), _dtype(x), n, d_in, k, _ptr(T_blocks), _ptr(xq), _ptr(x_scale), _stream(x.device)))
    return xq, x_scale


def _linear_args(xq, x_scale, Wq, w_scale, y) -> None:
    n, half = xq.shape
    d_out = Wq.shape[0]
    dev = xq.device
    _expect(xq, "xq", torch.uint8, (n, half), dev)
    _expect(x_scale, "x_scale", torch.float32, (n,), dev)
    _expect(Wq, "Wq", torch.uint8, (d_out, half), dev)
    _expect(w_scale, "w_scale", torch.float32, (d_out,), dev)
    _expect(y, "y", torch.float32, (n, d_out), dev)


def cat_split_transform_bytes(d_in: int, k: int) -> int:
    """Bytes of cat_split_transform's planes (0: no tensor-core transform for this d_in and k)."""
    return int(load_library().cat_split_transform_bytes(d_in, k))


def cat_split_transform(T_blocks: torch.Tensor, k: int) -> torch.Tensor:
    """T's three bf16 planes per channel group in the tensor-core transform's layout: uint8
    [cat_split_transform_bytes(d_in, k)]."""
    nb = T_blocks.shape[0]
    d_in = nb * k
    _expect(T_blocks, "T_blocks", torch.float32, (nb, k, k), T_blocks.device)
    nbytes = cat_split_transform_bytes(d_in, k)
    if nbytes <= 0:
        raise CatError("cat_split_transform", 5, f"no tensor-core transform for d_in = {d_in}, k = {k}")
    planes = torch.empty((nbytes,), dtype=torch.uint8, device=T_blocks.device)
    _check("cat_split_transform", load_library().cat_split_transform(_ptr(T_blocks), d_in, k, _ptr(planes),
                                                                     _stream(T_blocks.device)))
    return planes


def cat_transform_quantize_act_split(x: torch.Tensor, T_blocks: torch.Tensor, T_planes: Optional[torch.Tensor], k: int,
                                     xq: Optional[torch.Tensor] = None,
                                     x_scale: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """cat_transform_quantize_act with T's pre-split planes (cat_split_transform)."""
    _need(x, "x")
    n, d_in = x.shape
    if xq is None:
        xq = torch.empty((n, d_in // 2), dtype=torch.uint8, device=x.device)
    if x_scale is None:
        x_scale = torch.empty((n,), dtype=torch.float32, device=x.device)
    _expect(T_blocks, "T_blocks", torch.float32, (d_in // k, k, k), x.device)
    if T_planes is not None:
        _expect(T_planes, "T_planes", torch.uint8, (cat_split_transform_bytes(d_in, k),), x.device)
    _expect(xq, "xq", torch.uint8, (n, d_in // 2), x.device)
    _expect(x_scale, "x_scale", torch.float32, (n,), x.device)
    _check("cat_transform_quantize_act_split", load_library().cat_transform_quantize_act_split(
        _ptr(x), _dtype(x), n, d_in, k, _ptr(T_blocks), _ptr(T_planes), _ptr(xq), _ptr(x_scale), _stream(x.device)))
    return xq, x_scale


def cat_transform_quantize_act_e8(x: torch.Tensor, T_blocks: torch.Tensor, T_planes: Optional[torch.Tensor], k: int,
                                  xq8: Optional[torch.Tensor] = None,
                                  x_scale: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """cat_transform_quantize_act_split with the codes as byte codes: (xq8 uint8 [n, d_in], x_scale [n])."""
    _need(x, "x")
    n, d_in = x.shape
    if xq8 is None:
        xq8 = torch.empty((n, d_in), dtype=torch.uint8, device=x.device)
    if x_scale is None:
        x_scale = torch.empty((n,), dtype=torch.float32, device=x.device)
    _expect(T_blocks, "T_blocks", torch.float32, (d_in // k, k, k), x.device)
    if T_planes is not None:
        _expect(T_planes, "T_planes", torch.uint8, (cat_split_transform_bytes(d_in, k),), x.device)
    _expect(xq8, "xq8", torch.uint8, (n, d_in), x.device)
    _expect(x_scale, "x_scale", torch.float32, (n,), x.device)
    _check("cat_transform_quantize_act_e8", load_library().cat_transform_quantize_act_e8(
        _ptr(x), _dtype(x), n, d_in, k, _ptr(T_blocks), _ptr(T_planes), _ptr(xq8), _ptr(x_scale), _stream(x.device)))
    return xq8, x_scale


def cat_w4a4_linear(xq: torch.Tensor, x_scale: torch.Tensor, Wq: torch.Tensor, w_scale: torch.Tensor,
                    y: Optional[torch.Tensor] = None, acc_out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """y[t, o] = (sum_i q_x q_w) * s_x[t] * s_w[o] (float32 [n, d_out]); optionally the int32 accumulators."""
    for t, name in ((xq, "xq"), (x_scale, "x_scale"), (Wq, "Wq"), (w_scale, "w_scale")):
        _need(t, name)
    n, half = xq.shape
    d_out = Wq.shape[0]
    if y is None:
        y = torch.empty((n, d_out), dtype=torch.float32, device=xq.device)
    _linear_args(xq, x_scale, Wq, w_scale, y)
    if acc_out is not None:
        _expect(acc_out, "acc_out", torch.int32, (n, d_out), xq.device)
    _check("cat_w4a4_linear", load_library().cat_w4a4_linear(
        _ptr(xq), _ptr(x_scale), _ptr(Wq), _ptr(w_scale), n, 2 * half, d_out, _ptr(y), _ptr(acc_out),
        _stream(xq.device)))
    return y


def cat_w4a4_linear_sqnr(xq: torch.Tensor, x_scale: torch.Tensor, Wq: torch.Tensor, w_scale: torch.Tensor,
                         y_ref: torch.Tensor, y: Optional[torch.Tensor] = None,
                         out: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """cat_w4a4_linear and cat_sqnr against y_ref in one call: (y float32 [n, d_out], float64 [3])."""
    for t, name in ((xq, "xq"), (x_scale, "x_scale"), (Wq, "Wq"), (w_scale, "w_scale"), (y_ref, "y_ref")):
        _need(t, name)
    n, half = xq.shape
    d_out = Wq.shape[0]
    if y is None:
        y = torch.empty((n, d_out), dtype=torch.float32, device=xq.device)
    if out is None:
        out = torch.empty((3,), dtype=torch.float64, device=xq.device)
    _linear_args(xq, x_scale, Wq, w_scale, y)
    _expect(y_ref, "y_ref", torch.float32, (n, d_out), xq.device)
    _expect(out, "out", torch.float64, (3,), xq.device)
    _check("cat_w4a4_linear_sqnr", load_library().cat_w4a4_linear_sqnr(
        _ptr(xq), _ptr(x_scale), _ptr(Wq), _ptr(w_scale), n, 2 * half, d_out, _ptr(y), _ptr(y_ref), _ptr(out),
        _stream(xq.device)))
    return y, out


def cat_codes_to_e4m3(codes: torch.Tensor, out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """SM4x8 codes uint8 [rows, d/2] -> byte codes uint8 [rows, d] (one E4M3 byte per code)."""
    _need(codes, "codes")
    if codes.dtype != torch.uint8 or codes.dim() != 2:
        raise ValueError("codes must be a 2-D uint8 tensor")
    rows, half = codes.shape
    if out is None:
        out = torch.empty((rows, 2 * half), dtype=torch.uint8, device=codes.device)
    _expect(out, "out", torch.uint8, (rows, 2 * half), codes.device)
    _check("cat_codes_to_e4m3", load_library().cat_codes_to_e4m3(_ptr(codes), rows, 2 * half, _ptr(out),
                                                                 _stream(codes.device)))
    return out


def _linear_args_e8(xq8, x_scale, Wq8, w_scale, y) -> None:
    n, d_in = xq8.shape
    d_out = Wq8.shape[0]
    dev = xq8.device
    _expect(xq8, "xq8", torch.uint8, (n, d_in), dev)
    _expect(x_scale, "x_scale", torch.float32, (n,), dev)
    _expect(Wq8, "Wq8", torch.uint8, (d_out, d_in), dev)
    _expect(w_scale, "w_scale", torch.float32, (d_out,), dev)
    _expect(y, "y", torch.float32, (n, d_out), dev)


def cat_w4a4_linear_e8(xq8: torch.Tensor, x_scale: torch.Tensor, Wq8: torch.Tensor, w_scale: torch.Tensor,
                       y: Optional[torch.Tensor] = None, acc_out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """cat_w4a4_linear on byte codes xq8 [n, d_in], Wq8 [d_out, d_in]: the same y (and accumulators)."""
    for t, name in ((xq8, "xq8"), (x_scale, "x_scale"), (Wq8, "Wq8"), (w_scale, "w_scale")):
        _need(t, name)
    n, d_in = xq8.shape
    d_out = Wq8.shape[0]
    if y is None:
        y = torch.empty((n, d_out), dtype=torch.float32, device=xq8.device)
    _linear_args_e8(xq8, x_scale, Wq8, w_scale, y)
    if acc_out is not None:
        _expect(acc_out, "acc_out", torch.int32, (n, d_out), xq8.device)
    _check("cat_w4a4_linear_e8", load_library().cat_w4a4_linear_e8(
        _ptr(xq8), _ptr(x_scale), _ptr(Wq8), _ptr(w_scale), n, d_in, d_out, _ptr(y), _ptr(acc_out),
        _stream(xq8.device)))
    return y


def cat_w4a4_linear_sqnr_e8(xq8: torch.Tensor, x_scale: torch.Tensor, Wq8: torch.Tensor, w_scale: torch.Tensor,
                            y_ref: torch.Tensor, y: Optional[torch.Tensor] = None,
                            out: Optional[torch.Tensor] = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """cat_w4a4_linear_sqnr on byte codes: (y float32 [n, d_out], float64 [3])."""
    for t, name in ((xq8, "xq8"), (x_scale, "x_scale"), (Wq8, "Wq8"), (w_scale, "w_scale"), (y_ref, "y_ref")):
        _need(t, name)
    n, d_in = xq8.shape
    d_out = Wq8.shape[0]
    if y is None:
        y = torch.empty((n, d_out), dtype=torch.float32, device=xq8.device)
    if out is None:
        out = torch.empty((3,), dtype=torch.float64, device=xq8.device)
    _linear_args_e8(xq8, x_scale, Wq8, w_scale, y)
    _expect(y_ref, "y_ref", torch.float32, (n, d_out), xq8.device)
    _expect(out, "out", torch.float64, (3,), xq8.device)
    _check("cat_w4a4_linear_sqnr_e8", load_library().cat_w4a4_linear_sqnr_e8(
        _ptr(xq8), _ptr(x_scale), _ptr(Wq8), _ptr(w_scale), n, d_in, d_out, _ptr(y), _ptr(y_ref), _ptr(out),
        _stream(xq8.device)))
    return y, out


def cat_sqnr(y_ref: torch.Tensor, y_hat: torch.Tensor, out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """float64 [3] on the device: (sum y^2, sum (y - y_hat)^2, SQNR dB)."""
    _need(y_ref, "y_ref")
    _need(y_hat, "y_hat")
    if out is None:
        out = torch.empty((3,), dtype=torch.float64, device=y_ref.device)
    _expect(y_hat, "y_hat", torch.float32, tuple(y_ref.shape), y_ref.device)
    _expect(out, "out", torch.float64, (3,), y_ref.device)
    if y_ref.dtype != torch.float32:
        raise ValueError("y_ref must be float32")
    _check("cat_sqnr", load_library().cat_sqnr(_ptr(y_ref), _ptr(y_hat), y_ref.numel(), _ptr(out),
                                               _stream(y_ref.device)))
    return out


def cat_block_row_stats(V: torch.Tensor, k: int, M: torch.Tensor, transpose: bool = False):
    """Row statistics of V transformed block by block (v'_b = M_b v_b, or M_b^T v_b when
    ``transpose``): (row ||v'||^2 float32 [rows], row max |v'| float32 [rows], float64 [3]
    {sum ||v'||^2, sum (2 max |v'|)^2, 10 log10 of their ratio}) on V's device."""
    _need(V, "V")
    _need(M, "M")
    rows, d = V.shape
    _expect(M, "M", torch.float32, (d // k, k, k), V.device)
    row_sumsq = torch.empty((rows,), dtype=torch.float32, device=V.device)
    row_amax = torch.empty((rows,), dtype=torch.float32, device=V.device)
    out3 = torch.empty((3,), dtype=torch.float64, device=V.device)
    _check("cat_block_row_stats", load_library().cat_block_row_stats(
        _ptr(V), _dtype(V), rows, d, k, _ptr(M), 1 if transpose else 0, _ptr(row_sumsq), _ptr(row_amax), _ptr(out3),
        _stream(V.device)))
    return row_sumsq, row_amax, out3


def cat_dp_planes(bits: int) -> int:
    """Digit planes of b-bit codes (1 for b <= 4, else 2)."""
    return int(load_library().cat_dp_planes(int(bits)))


def cat_transform_quantize_act_dp(x: torch.Tensor, T_blocks: torch.Tensor, k: int, bits: int, asymmetric: bool = False,
                                  out=None):
    """x' = T x and its per-token b-bit codes as digit planes: (planes uint8 [D, n, d_in], x_scale float32 [n],
    x_zero int32 [n] or None)."""
    _need(x, "x")
    n, d_in = x.shape
    D = cat_dp_planes(bits)
    if D == 0:
        raise ValueError("bits must be in 2..8")
    if out is None:
        out = (torch.empty((D, n, d_in), dtype=torch.uint8, device=x.device),
               torch.empty((n,), dtype=torch.float32, device=x.device),
               torch.empty((n,), dtype=torch.int32, device=x.device) if asymmetric else None)
    planes, sx, zx = out
    _expect(T_blocks, "T_blocks", torch.float32, (d_in // k, k, k), x.device)
    _expect(planes, "planes", torch.uint8, (D, n, d_in), x.device)
    _expect(sx, "x_scale", torch.float32, (n,), x.device)
    if asymmetric:
        _expect(zx, "x_zero", torch.int32, (n,), x.device)
    _check("cat_transform_quantize_act_dp", load_library().cat_transform_quantize_act_dp(
        _ptr(x), _dtype(x), n, d_in, k, _ptr(T_blocks), int(bits), int(bool(asymmetric)), _ptr(planes), _ptr(sx),
        _ptr(zx) if asymmetric else None, _stream(x.device)))
    return planes, sx, (zx if asymmetric else None)


def cat_quantize_weights_dp(W: torch.Tensor, k: int, kind: str, bits: int, sigma_x: Optional[torch.Tensor] = None,
                            n_calib: int = 0, rht_signs=None, l24_range: bool = False, rowsum: bool = False):
    """Offline weight preparation at b bits: (T_blocks float32 [d_in/k, k, k], planes uint8 [D, d_out, d_in],
    w_scale float32 [d_out], w_rowsum int32 [d_out] or None)."""
    _need(W, "W")
    d_out, d_in = W.shape
    dev = W.device
    D = cat_dp_planes(bits)
    if D == 0:
        raise ValueError("bits must be in 2..8")
    T = torch.empty((d_in // k, k, k), dtype=torch.float32, device=dev)
    planes = torch.empty((D, d_out, d_in), dtype=torch.uint8, device=dev)
    sw = torch.empty((d_out,), dtype=torch.float32, device=dev)
    rs = torch.empty((d_out,), dtype=torch.int32, device=dev) if rowsum else None
    signs = None
    if rht_signs is not None:
        signs = np.ascontiguousarray(np.asarray(rht_signs, dtype=np.float32))
        if signs.shape != (d_in,):
            raise ValueError(f"rht_signs has shape {signs.shape}, expected ({d_in},)")
    if sigma_x is not None:
        _expect(sigma_x, "sigma_x", torch.float64, (d_in // k, k, k), dev)
    st = load_library().cat_quantize_weights_dp(
        _ptr(W), _dtype(W), d_out, d_in, k, KIND[kind], _ptr(sigma_x), int(n_calib),
        None if signs is None else signs.ctypes.data_as(ctypes.c_void_p), int(bits), int(bool(l24_range)), _ptr(T),
        _ptr(planes), _ptr(sw), _ptr(rs), _stream(dev))
    _check("cat_quantize_weights_dp", st)
    return T, planes, sw, rs


def cat_linear_dp(x_planes: torch.Tensor, bits_x: int, x_scale: torch.Tensor, w_planes: torch.Tensor, bits_w: int,
                  w_scale: torch.Tensor, x_zero: Optional[torch.Tensor] = None, w_rowsum: Optional[torch.Tensor] = None,
                  y: Optional[torch.Tensor] = None, acc_out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """y[t, o] = (sum_i (q_x - z_t) q_w) * s_x[t] * s_w[o] from digit-plane codes (float32 [n, d_out])."""
    Dx, n, d_in = x_planes.shape
    Dw, d_out, d_in_w = w_planes.shape
    dev = x_planes.device
    if Dx != cat_dp_planes(bits_x) or Dw != cat_dp_planes(bits_w) or d_in_w != d_in:
        raise ValueError("digit planes do not match the bit widths or each other")
    asym = x_zero is not None
    if asym and w_rowsum is None:
        raise ValueError("asymmetric activations need w_rowsum")
    if y is None:
        y = torch.empty((n, d_out), dtype=torch.float32, device=dev)
    _expect(x_planes, "x_planes", torch.uint8, (Dx, n, d_in), dev)
    _expect(w_planes, "w_planes", torch.uint8, (Dw, d_out, d_in), dev)
    _expect(x_scale, "x_scale", torch.float32, (n,), dev)
    _expect(w_scale, "w_scale", torch.float32, (d_out,), dev)
    _expect(y, "y", torch.float32, (n, d_out), dev)
    if asym:
        _expect(x_zero, "x_zero", torch.int32, (n,), dev)
        _expect(w_rowsum, "w_rowsum", torch.int32, (d_out,), dev)
    if acc_out is not None:
        _expect(acc_out, "acc_out", torch.int32, (n, d_out), dev)
    _check("cat_linear_dp", load_library().cat_linear_dp(
        _ptr(x_planes), int(bits_x), int(asym), _ptr(x_scale), _ptr(x_zero), _ptr(w_planes), int(bits_w), _ptr(w_scale),
        _ptr(w_rowsum) if asym else None, n, d_in, d_out, _ptr(y), _ptr(acc_out), _stream(dev)))
    return y


def cat_block_transform(V: torch.Tensor, k: int, M: torch.Tensor, transpose: bool = False) -> torch.Tensor:
    """v'_b = M_b v_b (or M_b^T v_b) for every row: float32 [rows, d]."""
    _need(V, "V")
    rows, d = V.shape
    _expect(M, "M", torch.float32, (d // k, k, k), V.device)
    out = torch.empty((rows, d), dtype=torch.float32, device=V.device)
    _check("cat_block_transform", load_library().cat_block_transform(
        _ptr(V), _dtype(V), rows, d, k, _ptr(M), 1 if transpose else 0, _ptr(out), _stream(V.device)))
    return out


def cat_dequantize_codes(codes: torch.Tensor, scale: torch.Tensor) -> torch.Tensor:
    """s_r * q from SM4x8 codes [rows, d/2] and steps [rows]: float32 [rows, d]."""
    rows, half = codes.shape
    _expect(codes, "codes", torch.uint8, (rows, half), codes.device)
    _expect(scale, "scale", torch.float32, (rows,), codes.device)
    out = torch.empty((rows, 2 * half), dtype=torch.float32, device=codes.device)
    _check("cat_dequantize_codes", load_library().cat_dequantize_codes(
        _ptr(codes), _ptr(scale), rows, 2 * half, _ptr(out), _stream(codes.device)))
    return out


def cat_gemm_f32(A: torch.Tensor, B: torch.Tensor) -> torch.Tensor:
    """C = A B^T in float32 (A [m, k], B [n, k])."""
    m, kd = A.shape
    n = B.shape[0]
    _expect(A, "A", torch.float32, (m, kd), A.device)
    _expect(B, "B", torch.float32, (n, kd), A.device)
    C = torch.empty((m, n), dtype=torch.float32, device=A.device)
    _check("cat_gemm_f32", load_library().cat_gemm_f32(_ptr(A), _ptr(B), m, n, kd, _ptr(C), _stream(A.device)))
    return C


def one_sided_sqnr(x: torch.Tensor, W: torch.Tensor, k: int, T: torch.Tensor, Tinv: torch.Tensor, xq: torch.Tensor,
                   x_scale: torch.Tensor, Wq: torch.Tensor, w_scale: torch.Tensor, y_ref: torch.Tensor):
    """The measured one-sided SQNRs of Lemmas 2 and 3 in dB, (activations only, weights only), composed
    of the library calls above and cat_sqnr against y_ref = W x."""
    xt = cat_block_transform(x, k, T)
    wt = cat_block_transform(W, k, Tinv, transpose=True)
    y_x = cat_gemm_f32(cat_dequantize_codes(xq, x_scale), wt)
    y_w = cat_gemm_f32(xt, cat_dequantize_codes(Wq, w_scale))
    return float(cat_sqnr(y_ref, y_x)[2].item()), float(cat_sqnr(y_ref, y_w)[2].item())


def cat_transform_quantize_act_hd(x: torch.Tensor, M_blocks: torch.Tensor, k: int) -> Tuple[torch.Tensor, torch.Tensor]:
    """x' = H_d (M_block x) and its per-token INT4 codes (kind "cat_hd"): (SM4x8 uint8 [n, d_in/2], float32 [n])."""
    _need(x, "x")
    n, d_in = x.shape
    _expect(M_blocks, "M_blocks", torch.float32, (d_in // k, k, k), x.device)
    xq = torch.empty((n, d_in // 2), dtype=torch.uint8, device=x.device)
    sx = torch.empty((n,), dtype=torch.float32, device=x.device)
    _check("cat_transform_quantize_act_hd", load_library().cat_transform_quantize_act_hd(
        _ptr(x), _dtype(x), n, d_in, k, _ptr(M_blocks), _ptr(xq), _ptr(sx), _stream(x.device)))
    return xq, sx


def cat_fwht_rows(V: torch.Tensor) -> torch.Tensor:
    """In place: every row of the float32 V [rows, d] becomes H_d v / sqrt(d)."""
    rows, d = V.shape
    _expect(V, "V", torch.float32, (rows, d), V.device)
    _check("cat_fwht_rows", load_library().cat_fwht_rows(_ptr(V), rows, d, _stream(V.device)))
    return V


def cat_gram_f32(X: torch.Tensor) -> torch.Tensor:
    """X^T X in float32 [d, d] for X [n, d] (float32 or bf16)."""
    _need(X, "X")
    n, d = X.shape
    C = torch.empty((d, d), dtype=torch.float32, device=X.device)
    _check("cat_gram_f32", load_library().cat_gram_f32(_ptr(X), _dtype(X), n, d, _ptr(C), _stream(X.device)))
    return C


def cat_alignment_ceiling_host(sigma_x: np.ndarray, sigma_w: np.ndarray) -> Tuple[float, float, float]:
    """Eq. 9 on the host from full Sigma_x, Sigma_w [d, d]: (A_max, sum mu, sum sqrt mu)."""
    sx = np.ascontiguousarray(sigma_x, dtype=np.float64)
    sw = np.ascontiguousarray(sigma_w, dtype=np.float64)
    d = sx.shape[0]
    if sx.shape != (d, d) or sw.shape != (d, d):
        raise ValueError("sigma_x and sigma_w must be square and of the same size")
    out = np.zeros(3)
    vp = lambda a: a.ctypes.data_as(ctypes.c_void_p)  # noqa: E731
    _check("cat_alignment_ceiling_host", load_library().cat_alignment_ceiling_host(vp(sx), vp(sw), d, vp(out)))
    return float(out[0]), float(out[1]), float(out[2])


def cat_set_wait_limit_ns(ns: int) -> None:
    """Testing aid: bound (ns) of the pipeline waits of the weight-streaming and digit-plane GEMMs on the
    current device; 0 restores the default (1 s)."""
    _check("cat_set_wait_limit_ns", load_library().cat_set_wait_limit_ns(int(ns)))


def cat_device_status(device: Optional[torch.device] = None) -> Tuple[int, int]:
    """Synchronize the current stream and return (status, raw status word); clears the word."""
    dev = device or torch.device("cuda", torch.cuda.current_device())
    detail = ctypes.c_uint32(0)
    st = load_library().cat_device_status(_stream(dev), ctypes.byref(detail))
    return int(st), int(detail.value)
