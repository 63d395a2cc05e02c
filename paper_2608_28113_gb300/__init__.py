"""GB300-native (sm_103a) H-Scale hot path: Python binding of ``libhscale.so``.

The functions here have the names of the C entry points in ``include/hscale.h`` and
only marshal arguments: they take torch CUDA tensors, check dtype/shape/device, pass
raw device pointers and the current CUDA stream through ctypes, and raise
``HScaleError`` on a non-zero status.  Every step of the path runs in the CUDA
kernels; there is no CPU fallback: if the compiled library is missing, loading it
raises.

Paper map: ``hscale_hessian_diag_accumulate`` is h = diag(X^T X) (Sec. 3.2, Eq. 4);
``hscale_rtn_scales`` the global scale and RTN codes (Sec. 3.3, Eq. 7);
``hscale_refine_scales`` Algorithm 1 (Eqs. 6-13); ``hscale_pack_nvfp4`` the final
re-quantization (Sec. 3.3); ``hscale_fourover6_codes`` the 4over6 start of Algorithm 2.
"""
from __future__ import annotations

import ctypes
import pathlib
import threading

import torch

__all__ = [
    "HScaleError", "load", "library_path", "hscale_status_string", "hscale_abi_version",
    "hscale_device_error_flags",
    "hscale_hessian_diag_accumulate", "hscale_hessian_diag_accumulate_ex", "HSCALE_HESSIAN_X_READY",
    "hscale_hessian_sum_partials", "hscale_amax_bits", "hscale_global_scale_from_amax",
    "hscale_rtn_workspace_bytes", "hscale_rtn_scales",
    "hscale_rtn_scales_noalloc",
    "hscale_refine_scales", "hscale_refine_scales_ex", "hscale_refine_scales_4over6",
    "hscale_refine_scales_strided", "hscale_refine_workspace_bytes", "hscale_refine_scales_ws",
    "hscale_pack_nvfp4", "hscale_fourover6_codes",
    "hscale_dequant_residual", "hscale_output_error_workspace_bytes", "hscale_output_error",
    "residual_ld", "hscale_selftest_bounded_wait", "hscale_hessian_full_workspace_bytes",
    "hscale_hessian_full_accumulate", "hscale_gptq_factor_workspace_bytes", "hscale_gptq_factor",
    "hscale_gptq_workspace_bytes", "hscale_gptq_hscale", "EXPORTED_SYMBOLS",
]

_PKG = pathlib.Path(__file__).resolve().parent
_LIB_PATH = _PKG / "_build" / "libhscale.so"
_lock = threading.Lock()
_lib = None

# every entry point of include/hscale.h, with its ctypes signature
_P, _I64, _I32, _SZ = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_size_t
_SIGNATURES = {
    "hscale_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "hscale_abi_version": (ctypes.c_int, []),
    "hscale_device_error_flags": (ctypes.c_int, [_P]),
    "hscale_selftest_bounded_wait": (ctypes.c_int, [ctypes.c_uint32, _P]),
    "hscale_hessian_diag_accumulate": (ctypes.c_int, [_P, _I64, _I64, _I64, _P, _P]),
    "hscale_hessian_diag_accumulate_ex": (ctypes.c_int, [_P, _I64, _I64, _I64, _P, ctypes.c_uint32, _P]),
    "hscale_hessian_sum_partials": (ctypes.c_int, [_P, _I64, _I64, _I64, _P, _P]),
    "hscale_amax_bits": (ctypes.c_int, [_P, _I64, _I64, _P, _P]),
    "hscale_global_scale_from_amax": (ctypes.c_int, [_P, _P, _P]),
    "hscale_rtn_workspace_bytes": (_SZ, []),
    "hscale_rtn_scales": (ctypes.c_int, [_P, _I64, _I64, _P, _P, _P, _SZ, _P]),
    "hscale_rtn_scales_noalloc": (ctypes.c_int, [_P, _I64, _I64, _P, _P, _P]),
    "hscale_refine_scales": (ctypes.c_int, [_P, _P, _I64, _I64, _P, _P, _I32, _I32, _P, _P, _P]),
    "hscale_refine_scales_ex": (ctypes.c_int, [_P, _P, _I64, _I64, _P, _P, _I32, _I32, _P, _P, _I32, _P]),
    "hscale_refine_scales_4over6": (ctypes.c_int, [_P, _P, _I64, _I64, _P, _I32, _I32, _P, _P, _I32, _P]),
    "hscale_refine_scales_strided": (ctypes.c_int, [_P, _I64, _P, _I64, _I64, _P, _P, _I64, _I32, _I32, _I32,
                                                    _P, _I64, _P, _I64, _I32, _P]),
    "hscale_refine_workspace_bytes": (_SZ, []),
    "hscale_refine_scales_ws": (ctypes.c_int, [_P, _P, _I64, _I64, _P, _P, _I32, _I32, _I32, _P, _P, _I32, _P, _SZ,
                                               _P]),
    "hscale_pack_nvfp4": (ctypes.c_int, [_P, _I64, _I64, _P, _P, _P, _P]),
    "hscale_fourover6_codes": (ctypes.c_int, [_P, _I64, _I64, _P, _P, _P]),
    "hscale_dequant_residual": (ctypes.c_int, [_P, _I64, _I64, _P, _P, _P, _P, _I64, _P]),
    "hscale_output_error_workspace_bytes": (ctypes.c_size_t, [_I64, _I64]),
    "hscale_output_error": (ctypes.c_int, [_P, _I64, _I64, _I64, _P, _I64, _I64, _P, _P, ctypes.c_size_t, _P]),
    "hscale_hessian_full_workspace_bytes": (ctypes.c_size_t, [_I64, _I64]),
    "hscale_hessian_full_accumulate": (ctypes.c_int, [_P, _I64, _I64, _I64, _P, _I64, _P, ctypes.c_size_t, _P]),
    "hscale_gptq_factor_workspace_bytes": (ctypes.c_size_t, [_I64]),
    "hscale_gptq_factor": (ctypes.c_int, [_P, _I64, _I64, ctypes.c_float, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "hscale_gptq_workspace_bytes": (ctypes.c_size_t, [_I64, _I64, _I32]),
    "hscale_gptq_hscale": (ctypes.c_int, [_P, _I64, _I64, _P, _P, _P, _P, _I32, _I32, _I32, _P, _P, _P,
                                          ctypes.c_size_t, _P]),
}
EXPORTED_SYMBOLS = tuple(_SIGNATURES)


class HScaleError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} failed with status {status}: {hscale_status_string(status)}")
        self.status = status


def library_path() -> pathlib.Path:
    return _LIB_PATH


def load(build_if_missing: bool = False) -> ctypes.CDLL:
    """The loaded CUDA library.  Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not _LIB_PATH.exists():
            if not build_if_missing:
                raise ImportError(f"{_LIB_PATH} is missing: build it with "
                                  "`python -c 'import __graft_entry__ as g; g.build()'`")
            from . import build as _build
            _build.build()
        lib = ctypes.CDLL(str(_LIB_PATH))
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def hscale_status_string(status: int) -> str:
    return load().hscale_status_string(int(status)).decode()


def hscale_abi_version() -> int:
    return int(load().hscale_abi_version())


def hscale_selftest_bounded_wait(polls: int, stream=None) -> None:
    """Launch the bounded-wait self-test (the wait runs out and sets device flag bit 0)."""
    _check("hscale_selftest_bounded_wait", load().hscale_selftest_bounded_wait(int(polls), _stream_ptr(stream)))


def hscale_device_error_flags() -> int:
    """Synchronise and return (then clear) the device failure flags; 0 = none."""
    v = ctypes.c_uint32(0)
    _check("hscale_device_error_flags", load().hscale_device_error_flags(ctypes.byref(v)))
    return int(v.value)


def _stream_ptr(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


def _check(fn: str, status: int) -> None:
    if status != 0:
        raise HScaleError(fn, status)


def _ptr(t: torch.Tensor | None):
    return None if t is None else t.data_ptr()


def _need(t: torch.Tensor, dtype, name: str):
    if not isinstance(t, torch.Tensor) or t.dtype != dtype or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor of dtype {dtype}")


HSCALE_HESSIAN_X_READY = 1


def hscale_hessian_diag_accumulate(x: torch.Tensor, h: torch.Tensor, stream=None) -> torch.Tensor:
    """h[j] += sum_t x[t, j]^2 for a bf16 chunk x [tokens, n] (row stride >= n)."""
    return hscale_hessian_diag_accumulate_ex(x, h, 0, stream)


def hscale_hessian_diag_accumulate_ex(x: torch.Tensor, h: torch.Tensor, flags: int = 0,
                                      stream=None) -> torch.Tensor:
    """hscale_hessian_diag_accumulate with flags; HSCALE_HESSIAN_X_READY declares that nothing
    still running writes x, so the kernel may overlap the previous kernel on the stream."""
    _need(x, torch.bfloat16, "x")
    _need(h, torch.float32, "h")
    if x.dim() != 2 or x.stride(1) != 1:
        raise ValueError("x must be 2-D with unit column stride")
    tokens, n = x.shape
    if h.numel() != n or not h.is_contiguous():
        raise ValueError("h must be a contiguous float32 vector of length n")
    ld = x.stride(0) if tokens > 1 else n
    _check("hscale_hessian_diag_accumulate_ex",
           load().hscale_hessian_diag_accumulate_ex(_ptr(x), tokens, n, ld, _ptr(h), int(flags),
                                                    _stream_ptr(stream)))
    return h


def hscale_hessian_sum_partials(partials: torch.Tensor, h: torch.Tensor, stream=None) -> torch.Tensor:
    """h = rank-order fp32 sum of the rows of partials [parts, n] (each a rank's partial h)."""
    _need(partials, torch.float32, "partials")
    _need(h, torch.float32, "h")
    if partials.dim() != 2 or partials.stride(1) != 1:
        raise ValueError("partials must be 2-D [parts, n] with unit column stride")
    parts, n = partials.shape
    if h.numel() != n or not h.is_contiguous():
        raise ValueError("h must be a contiguous float32 vector of length n")
    ld = partials.stride(0) if parts > 1 else n
    _check("hscale_hessian_sum_partials",
           load().hscale_hessian_sum_partials(_ptr(partials), parts, n, ld, _ptr(h), _stream_ptr(stream)))
    return h


def hscale_amax_bits(w: torch.Tensor, amax_bits: torch.Tensor, stream=None) -> torch.Tensor:
    """amax_bits (int32 [1], device) = bf16 bit pattern of max|W| (for an all-reduce MAX)."""
    _need(w, torch.bfloat16, "w")
    _need(amax_bits, torch.int32, "amax_bits")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    _check("hscale_amax_bits", load().hscale_amax_bits(_ptr(w), m, n, _ptr(amax_bits), _stream_ptr(stream)))
    return amax_bits


def hscale_global_scale_from_amax(amax_bits: torch.Tensor, global_scale: torch.Tensor, stream=None) -> None:
    """global_scale[0] = s_g of a matrix whose amax word is amax_bits[0]."""
    _need(amax_bits, torch.int32, "amax_bits")
    _need(global_scale, torch.float32, "global_scale")
    _check("hscale_global_scale_from_amax",
           load().hscale_global_scale_from_amax(_ptr(amax_bits), _ptr(global_scale), _stream_ptr(stream)))


def hscale_rtn_workspace_bytes() -> int:
    return int(load().hscale_rtn_workspace_bytes())


def hscale_rtn_scales(w: torch.Tensor, global_scale: torch.Tensor, codes: torch.Tensor | None,
                      workspace: torch.Tensor, stream=None) -> None:
    """s_g = amax|W| / 2688 into global_scale[0]; RTN codes [m, n/16] into codes."""
    _need(w, torch.bfloat16, "w")
    _need(global_scale, torch.float32, "global_scale")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if codes is not None:
        _need(codes, torch.uint8, "codes")
        if codes.numel() != m * (n // 16) or not codes.is_contiguous():
            raise ValueError("codes must be contiguous [m, n/16]")
    if not workspace.is_cuda:
        raise TypeError("workspace must live on the GPU")
    nbytes = workspace.numel() * workspace.element_size()
    _check("hscale_rtn_scales",
           load().hscale_rtn_scales(_ptr(w), m, n, _ptr(global_scale), _ptr(codes),
                                    _ptr(workspace), nbytes, _stream_ptr(stream)))


def hscale_rtn_scales_noalloc(w: torch.Tensor, global_scale: torch.Tensor,
                              codes: torch.Tensor | None, stream=None) -> None:
    """hscale_rtn_scales for callers that cannot allocate: no workspace argument; the
    library's fixed per-GPU scratch array is used instead (calls must not overlap)."""
    _need(w, torch.bfloat16, "w")
    _need(global_scale, torch.float32, "global_scale")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if codes is not None:
        _need(codes, torch.uint8, "codes")
        if codes.numel() != m * (n // 16) or not codes.is_contiguous():
            raise ValueError("codes must be contiguous [m, n/16]")
    _check("hscale_rtn_scales_noalloc",
           load().hscale_rtn_scales_noalloc(_ptr(w), m, n, _ptr(global_scale), _ptr(codes),
                                            _stream_ptr(stream)))


def hscale_refine_scales(w: torch.Tensor, h: torch.Tensor | None, global_scale: torch.Tensor,
                         init_codes: torch.Tensor | None, down: int, up: int,
                         codes_out: torch.Tensor, packed_out: torch.Tensor | None,
                         stream=None) -> None:
    """Algorithm 1 over every group of W, with the final re-quantization and packing."""
    hscale_refine_scales_ex(w, h, global_scale, init_codes, down, up, codes_out, packed_out, 0, stream)


def hscale_refine_scales_ex(w: torch.Tensor, h: torch.Tensor | None, global_scale: torch.Tensor,
                            init_codes: torch.Tensor | None, down: int, up: int,
                            codes_out: torch.Tensor, packed_out: torch.Tensor | None,
                            ctas_per_sm: int, stream=None) -> None:
    """hscale_refine_scales with at most ``ctas_per_sm`` resident CTAs per SM (0: all)."""
    _need(w, torch.bfloat16, "w")
    _need(global_scale, torch.float32, "global_scale")
    _need(codes_out, torch.uint8, "codes_out")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if h is not None:
        _need(h, torch.float32, "h")
        if h.numel() != n or not h.is_contiguous():
            raise ValueError("h must be a contiguous float32 vector of length n")
    for name, t, size in (("init_codes", init_codes, m * (n // 16)),
                          ("codes_out", codes_out, m * (n // 16)),
                          ("packed_out", packed_out, m * (n // 2))):
        if t is not None:
            _need(t, torch.uint8, name)
            if t.numel() != size or not t.is_contiguous():
                raise ValueError(f"{name} must be contiguous with {size} bytes")
    _check("hscale_refine_scales_ex",
           load().hscale_refine_scales_ex(_ptr(w), _ptr(h), m, n, _ptr(global_scale), _ptr(init_codes),
                                          int(down), int(up), _ptr(codes_out), _ptr(packed_out),
                                          int(ctas_per_sm), _stream_ptr(stream)))


def hscale_refine_workspace_bytes() -> int:
    return int(load().hscale_refine_workspace_bytes())


def hscale_refine_scales_ws(w: torch.Tensor, h: torch.Tensor | None, global_scale: torch.Tensor,
                            init_codes: torch.Tensor | None, fourover6: int, down: int, up: int,
                            codes_out: torch.Tensor, packed_out: torch.Tensor | None, ctas_per_sm: int,
                            workspace: torch.Tensor | None, stream=None) -> None:
    """hscale_refine_scales_ex (fourover6 = 0) or _4over6 (fourover6 = 1) with long searches'
    units shared out at run time through ``workspace`` (a device uint8 tensor of at least
    hscale_refine_workspace_bytes() bytes, or None for the static deal)."""
    _need(w, torch.bfloat16, "w")
    _need(global_scale, torch.float32, "global_scale")
    _need(codes_out, torch.uint8, "codes_out")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if h is not None:
        _need(h, torch.float32, "h")
        if h.numel() != n or not h.is_contiguous():
            raise ValueError("h must be a contiguous float32 vector of length n")
    for name, t, size in (("init_codes", init_codes, m * (n // 16)),
                          ("codes_out", codes_out, m * (n // 16)),
                          ("packed_out", packed_out, m * (n // 2))):
        if t is not None:
            _need(t, torch.uint8, name)
            if t.numel() != size or not t.is_contiguous():
                raise ValueError(f"{name} must be contiguous with {size} bytes")
    nbytes = 0
    if workspace is not None:
        _need(workspace, torch.uint8, "workspace")
        nbytes = workspace.numel()
    _check("hscale_refine_scales_ws",
           load().hscale_refine_scales_ws(_ptr(w), _ptr(h), m, n, _ptr(global_scale), _ptr(init_codes),
                                          int(fourover6), int(down), int(up), _ptr(codes_out), _ptr(packed_out),
                                          int(ctas_per_sm), _ptr(workspace), nbytes, _stream_ptr(stream)))


def hscale_refine_scales_4over6(w: torch.Tensor, h: torch.Tensor | None, global_scale: torch.Tensor,
                                down: int, up: int, codes_out: torch.Tensor, packed_out: torch.Tensor | None,
                                ctas_per_sm: int = 0, stream=None) -> None:
    """Algorithm 2 in one pass: 4over6 initial codes decided in the search, then the search."""
    _need(w, torch.bfloat16, "w")
    _need(global_scale, torch.float32, "global_scale")
    _need(codes_out, torch.uint8, "codes_out")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if h is not None:
        _need(h, torch.float32, "h")
        if h.numel() != n or not h.is_contiguous():
            raise ValueError("h must be a contiguous float32 vector of length n")
    for name, t, size in (("codes_out", codes_out, m * (n // 16)),
                          ("packed_out", packed_out, m * (n // 2))):
        if t is not None:
            _need(t, torch.uint8, name)
            if t.numel() != size or not t.is_contiguous():
                raise ValueError(f"{name} must be contiguous with {size} bytes")
    _check("hscale_refine_scales_4over6",
           load().hscale_refine_scales_4over6(_ptr(w), _ptr(h), m, n, _ptr(global_scale), int(down), int(up),
                                              _ptr(codes_out), _ptr(packed_out), int(ctas_per_sm),
                                              _stream_ptr(stream)))


def _row_view(t: torch.Tensor, name: str, dtype, rows: int, cols: int) -> int:
    """Row stride (elements) of a 2-D view with unit column stride; checks its shape."""
    _need(t, dtype, name)
    if t.dim() != 2 or tuple(t.shape) != (rows, cols) or (cols > 1 and t.stride(1) != 1):
        raise ValueError(f"{name} must be a [{rows}, {cols}] view with contiguous rows")
    return t.stride(0) if rows > 1 else max(cols, t.stride(0))


def hscale_refine_scales_strided(w: torch.Tensor, h: torch.Tensor | None, global_scale: torch.Tensor,
                                 init_codes: torch.Tensor | None, fourover6: bool, down: int, up: int,
                                 codes_out: torch.Tensor, packed_out: torch.Tensor | None,
                                 ctas_per_sm: int = 0, stream=None) -> None:
    """The search on 2-D views (e.g. ``W[:, c0:c1]``, ``codes[:, c0/16:c1/16]``,
    ``packed[:, c0/2:c1/2]``)."""
    if w.dim() != 2:
        raise ValueError("w must be a 2-D view")
    m, n = w.shape
    ld_w = _row_view(w, "w", torch.bfloat16, m, n)
    _need(global_scale, torch.float32, "global_scale")
    if h is not None:
        _need(h, torch.float32, "h")
        if h.numel() != n or not h.is_contiguous():
            raise ValueError("h must be a contiguous float32 vector of length n")
    ld_c = _row_view(codes_out, "codes_out", torch.uint8, m, n // 16)
    ld_i = 0 if init_codes is None else _row_view(init_codes, "init_codes", torch.uint8, m, n // 16)
    ld_p = 0 if packed_out is None else _row_view(packed_out, "packed_out", torch.uint8, m, n // 2)
    _check("hscale_refine_scales_strided",
           load().hscale_refine_scales_strided(_ptr(w), ld_w, _ptr(h), m, n, _ptr(global_scale), _ptr(init_codes),
                                               ld_i, int(bool(fourover6)), int(down), int(up), _ptr(codes_out), ld_c,
                                               _ptr(packed_out), ld_p, int(ctas_per_sm), _stream_ptr(stream)))


def hscale_pack_nvfp4(w: torch.Tensor, global_scale: torch.Tensor, codes: torch.Tensor,
                      packed_out: torch.Tensor, stream=None) -> None:
    """FP4 nibbles of W under the given codes."""
    _need(w, torch.bfloat16, "w")
    _need(global_scale, torch.float32, "global_scale")
    _need(codes, torch.uint8, "codes")
    _need(packed_out, torch.uint8, "packed_out")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if codes.numel() != m * (n // 16) or packed_out.numel() != m * (n // 2):
        raise ValueError("codes must be [m, n/16] and packed_out [m, n/2]")
    _check("hscale_pack_nvfp4",
           load().hscale_pack_nvfp4(_ptr(w), m, n, _ptr(global_scale), _ptr(codes),
                                    _ptr(packed_out), _stream_ptr(stream)))


def hscale_fourover6_codes(w: torch.Tensor, global_scale: torch.Tensor, codes: torch.Tensor,
                           stream=None) -> None:
    """Algorithm 2's 4over6 initial codes [m, n/16] (input to hscale_refine_scales)."""
    _need(w, torch.bfloat16, "w")
    _need(global_scale, torch.float32, "global_scale")
    _need(codes, torch.uint8, "codes")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if codes.numel() != m * (n // 16) or not codes.is_contiguous():
        raise ValueError("codes must be contiguous [m, n/16]")
    _check("hscale_fourover6_codes",
           load().hscale_fourover6_codes(_ptr(w), m, n, _ptr(global_scale), _ptr(codes),
                                         _stream_ptr(stream)))


def residual_ld(n: int) -> int:
    """Row length (elements) of the [hi | lo] residual matrix for n input features."""
    return 2 * 64 * ((int(n) + 63) // 64)


def hscale_dequant_residual(w: torch.Tensor, global_scale: torch.Tensor, codes: torch.Tensor,
                            packed: torch.Tensor, dw2: torch.Tensor, stream=None) -> None:
    """dW = W - W_hat of packed NVFP4 weights into dw2 [m, ld] bf16 as [hi | lo] halves."""
    _need(w, torch.bfloat16, "w")
    _need(global_scale, torch.float32, "global_scale")
    _need(codes, torch.uint8, "codes")
    _need(packed, torch.uint8, "packed")
    _need(dw2, torch.bfloat16, "dw2")
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if codes.numel() != m * (n // 16) or packed.numel() != m * (n // 2):
        raise ValueError("codes must be [m, n/16] and packed [m, n/2]")
    if dw2.dim() != 2 or dw2.shape[0] != m or dw2.stride(1) != 1 or dw2.shape[1] < residual_ld(n):
        raise ValueError("dw2 must be [m, >= residual_ld(n)] with unit column stride")
    _check("hscale_dequant_residual",
           load().hscale_dequant_residual(_ptr(w), m, n, _ptr(global_scale), _ptr(codes), _ptr(packed),
                                          _ptr(dw2), dw2.stride(0), _stream_ptr(stream)))


def hscale_output_error_workspace_bytes(tokens: int, m: int) -> int:
    return int(load().hscale_output_error_workspace_bytes(int(tokens), int(m)))


def hscale_output_error(x: torch.Tensor, dw2: torch.Tensor, m: int, out_sum: torch.Tensor,
                        workspace: torch.Tensor, stream=None) -> None:
    """out_sum (fp64, device) += ||X dW^T||_F^2 for x [tokens, n] (row stride ld_x)."""
    _need(x, torch.bfloat16, "x")
    _need(dw2, torch.bfloat16, "dw2")
    _need(out_sum, torch.float64, "out_sum")
    if x.dim() != 2 or x.stride(1) != 1 or dw2.dim() != 2 or dw2.stride(1) != 1:
        raise ValueError("x and dw2 must be 2-D with unit column stride")
    tokens, n = x.shape
    _check("hscale_output_error",
           load().hscale_output_error(_ptr(x), tokens, n, x.stride(0), _ptr(dw2), dw2.stride(0), int(m),
                                      _ptr(out_sum), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                      _stream_ptr(stream)))


def _workspace(nbytes: int, device) -> torch.Tensor:
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def hscale_hessian_full_accumulate(x: torch.Tensor, H: torch.Tensor, workspace: torch.Tensor | None = None,
                                   stream=None) -> None:
    """Upper triangle of H (fp32 [n, n]) += X^T X for x [tokens, n] bf16 on the tensor cores.
    A workspace is needed (and allocated here if not given) only for x whose rows are not
    16-byte aligned."""
    _need(x, torch.bfloat16, "x")
    _need(H, torch.float32, "H")
    if x.dim() != 2 or x.stride(1) != 1 or H.dim() != 2 or H.stride(1) != 1:
        raise ValueError("x and H must be 2-D with unit column stride")
    tokens, n = x.shape
    direct = x.data_ptr() % 16 == 0 and x.stride(0) % 8 == 0
    if workspace is None and not direct:
        workspace = _workspace(load().hscale_hessian_full_workspace_bytes(tokens, n), x.device)
    _check("hscale_hessian_full_accumulate",
           load().hscale_hessian_full_accumulate(_ptr(x), tokens, n, x.stride(0), _ptr(H), H.stride(0),
                                                 _ptr(workspace) if workspace is not None else None,
                                                 workspace.numel() if workspace is not None else 0,
                                                 _stream_ptr(stream)))


def hscale_gptq_factor(H: torch.Tensor, damp: float, U: torch.Tensor, dead: torch.Tensor | None,
                       info: torch.Tensor, workspace: torch.Tensor | None = None, stream=None) -> None:
    """U (fp32 [n, n], upper) with U^T U = (H + damp * mean(diag H) I)^-1, as GPTQ forms it."""
    _need(H, torch.float32, "H")
    _need(U, torch.float32, "U")
    _need(info, torch.int32, "info")
    n = H.shape[0]
    if U.shape != (n, n) or not U.is_contiguous() or info.numel() < 3:
        raise ValueError("U must be contiguous [n, n] and info hold 3 int32")
    if dead is not None:
        _need(dead, torch.uint8, "dead")
    if workspace is None:
        nbytes = load().hscale_gptq_factor_workspace_bytes(n)
        if nbytes == 0:
            raise HScaleError("hscale_gptq_factor_workspace_bytes", 5)
        workspace = _workspace(nbytes, H.device)
    _check("hscale_gptq_factor",
           load().hscale_gptq_factor(_ptr(H), n, H.stride(0), float(damp), _ptr(U), _ptr(dead), _ptr(info),
                                     _ptr(workspace), workspace.numel(), _stream_ptr(stream)))


def hscale_gptq_hscale(w: torch.Tensor, U: torch.Tensor, h: torch.Tensor, global_scale: torch.Tensor,
                       dead: torch.Tensor | None, block: int, down: int, up: int, codes_out: torch.Tensor,
                       packed_out: torch.Tensor, workspace: torch.Tensor | None = None, stream=None) -> None:
    """Algorithm 3: GPTQ over blocks of `block` columns with H-Scale as the local quantizer."""
    _need(w, torch.bfloat16, "w")
    for name, t, dt in (("U", U, torch.float32), ("h", h, torch.float32), ("global_scale", global_scale, torch.float32),
                        ("codes_out", codes_out, torch.uint8), ("packed_out", packed_out, torch.uint8)):
        _need(t, dt, name)
    if not w.is_contiguous() or w.dim() != 2:
        raise ValueError("w must be a contiguous 2-D tensor")
    m, n = w.shape
    if workspace is None:
        workspace = _workspace(load().hscale_gptq_workspace_bytes(m, n, block), w.device)
    _check("hscale_gptq_hscale",
           load().hscale_gptq_hscale(_ptr(w), m, n, _ptr(U), _ptr(h), _ptr(global_scale), _ptr(dead), int(block),
                                     int(down), int(up), _ptr(codes_out), _ptr(packed_out), _ptr(workspace),
                                     workspace.numel(), _stream_ptr(stream)))


def hscale_hessian_full_workspace_bytes(tokens: int, n: int) -> int:
    return int(load().hscale_hessian_full_workspace_bytes(int(tokens), int(n)))


def hscale_gptq_factor_workspace_bytes(n: int) -> int:
    return int(load().hscale_gptq_factor_workspace_bytes(int(n)))


def hscale_gptq_workspace_bytes(m: int, n: int, block: int) -> int:
    return int(load().hscale_gptq_workspace_bytes(int(m), int(n), int(block)))
