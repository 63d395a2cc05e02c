"""CPU oracle for the H-Scale hot path -- TEST INFRASTRUCTURE ONLY.

A plain fp64 restatement of the paper's method (``hscale_oracle.c``), loaded with
ctypes.  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg may import this package; the CUDA product path never does, and this package
never imports the product package.  Inputs are raw bfloat16 bit patterns as
``numpy.uint16`` arrays, so both sides see exactly the same bytes.

Function map (paper equations in their order of appearance):
  hessian_accumulate   h += diag(X^T X)                      Sec. 3.2, Eq. 4
  global_scale         s_g = amax|W| / (6*448)               Sec. 3.1 (formula is a reading)
  rtn_codes            iota(Q_fp8(amax_group / (6 s_g)))     Sec. 3.3, Eq. 7
  refine               Algorithm 1 with diagnostics          Eqs. 8-13
  fourover6_codes      Algorithm 2's 4over6 initialization   Sec. 3.5, Algorithm 2
  refine_f64           Algorithm 1 on fp64 weights           (local quantizer of Algorithm 3)
  hessian_full         H += X^T X                            GPTQ Hessian of Algorithm 3
  gptq_factor          damped inverse-Cholesky factor        Algorithm 3 (as in GPTQ)
  gptq_hscale          GPTQ with H-Scale as local quantizer  Algorithm 3
  pack                 final FP4 quantization                Sec. 3.3, Eq. 2
  quantize_at_scale    Eq. 2 at a real scale (App. A.1 microcase)
  dequant_residual     dW = W - W_hat of packed NVFP4         Eqs. 1-3
  output_error         ||X dW^T||_F^2                        Eq. 3
"""
from __future__ import annotations

import ctypes
import os
import pathlib
import subprocess
import threading

import numpy as np

_HERE = pathlib.Path(__file__).resolve().parent
_SRC = _HERE / "hscale_oracle.c"
_BUILD = _HERE / "_build"
_LIB_PATH = _BUILD / "liboracle.so"
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> pathlib.Path:
    """Compile the C oracle with gcc (OpenMP if the compiler has it)."""
    _BUILD.mkdir(exist_ok=True)
    if not force and _LIB_PATH.exists() and _LIB_PATH.stat().st_mtime >= _SRC.stat().st_mtime:
        return _LIB_PATH
    base = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", "-Wall"]
    tmp = _BUILD / f"liboracle.{os.getpid()}.so"
    for extra in (["-fopenmp"], []):
        cmd = base + extra + ["-o", str(tmp), str(_SRC), "-lm"]
        if subprocess.run(cmd, capture_output=True).returncode == 0:
            os.replace(tmp, _LIB_PATH)
            return _LIB_PATH
    raise RuntimeError("could not compile the CPU oracle: " + " ".join(base))


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(str(build()))
        P = ctypes.c_void_p
        i64, i32, f32, f64 = ctypes.c_int64, ctypes.c_int, ctypes.c_float, ctypes.c_double
        sig = {
            "oracle_set_threads": (None, [i32]),
            "oracle_max_threads": (i32, []),
            "oracle_e4m3_decode": (f64, [ctypes.c_uint8]),
            "oracle_e2m1_decode": (f64, [ctypes.c_uint8]),
            "oracle_hessian_accumulate": (None, [P, i64, i64, i64, P]),
            "oracle_global_scale": (f32, [P, i64, P]),
            "oracle_rtn_codes": (None, [P, i64, i64, f32, P]),
            "oracle_refine": (None, [P, P, i64, i64, f32, P, i32, i32, P, P, P, P, P, P, P]),
            "oracle_group_errors": (None, [P, P, f32, P, i32, P]),
            "oracle_pack": (None, [P, i64, i64, f32, P, P]),
            "oracle_fourover6_codes": (None, [P, i64, i64, f32, P, P]),
            "oracle_quantize_at_scale": (None, [P, i64, f64, P, P]),
            "oracle_output_error": (f64, [P, i64, i64, P, i64]),
            "oracle_dequant_residual": (None, [P, i64, i64, f32, P, P, P]),
            "oracle_refine_f64": (None, [P, P, i64, i64, f32, i32, i32, P, P, P, P]),
            "oracle_hessian_full": (None, [P, i64, i64, i64, P]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _u16(a) -> np.ndarray:
    a = np.asarray(a)
    if a.dtype != np.uint16:
        raise TypeError("bf16 inputs are passed as uint16 bit patterns")
    return np.ascontiguousarray(a)


def set_threads(n: int) -> None:
    _load().oracle_set_threads(int(n))


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def e4m3_decode_table() -> np.ndarray:
    """Value of every E4M3 byte 0..255 (NaN at 0x7F / 0xFF)."""
    lib = _load()
    return np.array([lib.oracle_e4m3_decode(b) for b in range(256)], dtype=np.float64)


def e2m1_decode_table() -> np.ndarray:
    """Value of every E2M1 nibble 0..15."""
    lib = _load()
    return np.array([lib.oracle_e2m1_decode(b) for b in range(16)], dtype=np.float64)


def hessian_accumulate(x_u16: np.ndarray, h: np.ndarray, ld: int | None = None,
                       tokens: int | None = None, n: int | None = None) -> np.ndarray:
    """h (float64 [n], in place) += sum over tokens of x^2.  x is [tokens, ld] uint16."""
    x = _u16(x_u16)
    if x.ndim != 2:
        raise ValueError("x must be 2-D")
    T = x.shape[0] if tokens is None else tokens
    nn = x.shape[1] if n is None else n
    L = x.shape[1] if ld is None else ld
    if h.dtype != np.float64 or not h.flags.c_contiguous or h.shape[0] < nn:
        raise ValueError("h must be a contiguous float64 array of length n")
    _load().oracle_hessian_accumulate(_ptr(x), T, nn, L, _ptr(h))
    return h


def global_scale(w_u16: np.ndarray) -> tuple[np.float32, float]:
    """(s_g as float32, amax as float)."""
    w = _u16(w_u16)
    amax = ctypes.c_double(0.0)
    s = _load().oracle_global_scale(_ptr(w), w.size, ctypes.byref(amax))
    return np.float32(s), float(amax.value)


def rtn_codes(w_u16: np.ndarray, s_g) -> np.ndarray:
    w = _u16(w_u16)
    m, n = w.shape
    codes = np.empty((m, n // 16), dtype=np.uint8)
    _load().oracle_rtn_codes(_ptr(w), m, n, float(np.float32(s_g)), _ptr(codes))
    return codes


def refine(w_u16: np.ndarray, h_f32: np.ndarray | None, s_g, init_codes: np.ndarray | None,
           down: int, up: int) -> dict:
    """Algorithm 1 with diagnostics.  Returns a dict of numpy arrays:
    codes [m, n/16] u8, packed [m, n/2] u8, near_tie, delta, e_best, e_init, e_second."""
    w = _u16(w_u16)
    m, n = w.shape
    ng = n // 16
    h = None
    if h_f32 is not None:
        h = np.ascontiguousarray(h_f32, dtype=np.float32)
        if h.shape[0] != n:
            raise ValueError("h must have n entries")
    ic = None
    if init_codes is not None:
        ic = np.ascontiguousarray(init_codes, dtype=np.uint8).reshape(m, ng)
    out = {
        "codes": np.empty((m, ng), np.uint8),
        "packed": np.empty((m, n // 2), np.uint8),
        "near_tie": np.empty((m, ng), np.uint8),
        "delta": np.empty((m, ng), np.int16),
        "e_best": np.empty((m, ng), np.float64),
        "e_init": np.empty((m, ng), np.float64),
        "e_second": np.empty((m, ng), np.float64),
    }
    _load().oracle_refine(_ptr(w), _ptr(h), m, n, float(np.float32(s_g)), _ptr(ic), int(down),
                          int(up), _ptr(out["codes"]), _ptr(out["packed"]), _ptr(out["near_tie"]),
                          _ptr(out["delta"]), _ptr(out["e_best"]), _ptr(out["e_init"]),
                          _ptr(out["e_second"]))
    return out


def group_errors(g16_u16: np.ndarray, h16: np.ndarray | None, s_g, codes) -> np.ndarray:
    """E(code) of one 16-element group for every code in ``codes``."""
    g = _u16(g16_u16).reshape(16)
    h = None if h16 is None else np.ascontiguousarray(h16, dtype=np.float32).reshape(16)
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    err = np.empty(c.size, np.float64)
    _load().oracle_group_errors(_ptr(g), _ptr(h), float(np.float32(s_g)), _ptr(c), c.size,
                                _ptr(err))
    return err


def fourover6_codes(w_u16: np.ndarray, s_g) -> tuple[np.ndarray, np.ndarray]:
    """Algorithm 2's initial codes [m, n/16] and the anchor near-tie flags."""
    w = _u16(w_u16)
    m, n = w.shape
    codes = np.empty((m, n // 16), np.uint8)
    nt = np.empty((m, n // 16), np.uint8)
    _load().oracle_fourover6_codes(_ptr(w), m, n, float(np.float32(s_g)), _ptr(codes), _ptr(nt))
    return codes, nt


def pack(w_u16: np.ndarray, s_g, codes: np.ndarray) -> np.ndarray:
    w = _u16(w_u16)
    m, n = w.shape
    c = np.ascontiguousarray(codes, dtype=np.uint8).reshape(m, n // 16)
    out = np.empty((m, n // 2), np.uint8)
    _load().oracle_pack(_ptr(w), m, n, float(np.float32(s_g)), _ptr(c), _ptr(out))
    return out


def quantize_at_scale(w: np.ndarray, s: float) -> tuple[np.ndarray, np.ndarray]:
    """Eq. 2 at a real scale: (w_hat, signed magnitude codes)."""
    ww = np.ascontiguousarray(w, dtype=np.float64)
    wh = np.empty_like(ww)
    codes = np.empty(ww.shape, np.int8)
    _load().oracle_quantize_at_scale(_ptr(ww), ww.size, float(s), _ptr(wh), _ptr(codes))
    return wh, codes


def dequant_residual(w_u16: np.ndarray, s_g, codes: np.ndarray, packed: np.ndarray) -> np.ndarray:
    """dW = W - W_hat (fp64 [m, n]) for packed NVFP4 weights with per-group codes."""
    w = _u16(w_u16)
    m, n = w.shape
    c = np.ascontiguousarray(codes, dtype=np.uint8).reshape(m, n // 16)
    p = np.ascontiguousarray(packed, dtype=np.uint8).reshape(m, n // 2)
    out = np.empty((m, n), np.float64)
    _load().oracle_dequant_residual(_ptr(w), m, n, float(np.float32(s_g)), _ptr(c), _ptr(p), _ptr(out))
    return out


def output_error(X: np.ndarray, dW: np.ndarray) -> float:
    """||X dW^T||_F^2 (Eq. 3)."""
    Xd = np.ascontiguousarray(X, dtype=np.float64)
    D = np.ascontiguousarray(np.atleast_2d(dW), dtype=np.float64)
    return float(_load().oracle_output_error(_ptr(Xd), Xd.shape[0], Xd.shape[1], _ptr(D),
                                             D.shape[0]))


def refine_f64(w: np.ndarray, h_f32: np.ndarray | None, s_g, down: int, up: int) -> dict:
    """Algorithm 1 with RTN initial codes on fp64 weights [m, n]: codes, w_hat (signed
    dequantized values), packed nibbles, near_tie flags."""
    wv = np.ascontiguousarray(w, dtype=np.float64)
    m, n = wv.shape
    h = None if h_f32 is None else np.ascontiguousarray(h_f32, dtype=np.float32).reshape(n)
    out = {"codes": np.empty((m, n // 16), np.uint8), "w_hat": np.empty((m, n), np.float64),
           "packed": np.empty((m, n // 2), np.uint8), "near_tie": np.empty((m, n // 16), np.uint8)}
    _load().oracle_refine_f64(_ptr(wv), _ptr(h), m, n, float(np.float32(s_g)), int(down), int(up),
                              _ptr(out["codes"]), _ptr(out["w_hat"]), _ptr(out["packed"]), _ptr(out["near_tie"]))
    return out


def hessian_full(x_u16: np.ndarray, H: np.ndarray, ld: int | None = None, n: int | None = None) -> np.ndarray:
    """H (fp64 [n, n], in place) += X^T X for x [tokens, ld] uint16 (first n columns)."""
    x = _u16(x_u16)
    nn = x.shape[1] if n is None else n
    L = x.shape[1] if ld is None else ld
    if H.dtype != np.float64 or not H.flags.c_contiguous or H.shape != (nn, nn):
        raise ValueError("H must be a contiguous float64 [n, n] array")
    _load().oracle_hessian_full(_ptr(x), x.shape[0], nn, L, _ptr(H))
    return H


def gptq_factor(H: np.ndarray, damp: float = 0.01) -> tuple[np.ndarray, np.ndarray]:
    """The damped inverse-Cholesky factor of Algorithm 3, formed as GPTQ forms it: dead
    columns (H_jj = 0) get H_jj = 1, the diagonal gets damp * mean(diag H), and U is the
    upper Cholesky factor of (H + damp I)^-1, so U^T U = (H + damp I)^-1.  Returns
    (U, dead-column mask).  numpy's Cholesky and inverse serve as library steps."""
    Hd = np.array(H, dtype=np.float64, copy=True)
    dead = np.diag(Hd) == 0
    Hd[dead, dead] = 1.0
    Hd[np.diag_indices_from(Hd)] += damp * float(np.mean(np.diag(Hd)))
    Hinv = np.linalg.inv(Hd)
    Hinv = 0.5 * (Hinv + Hinv.T)
    U = np.linalg.cholesky(Hinv).T
    return U, dead


def gptq_hscale(w_u16: np.ndarray, U: np.ndarray, h_f32: np.ndarray, s_g, block: int, down: int, up: int,
                dead: np.ndarray | None = None) -> dict:
    """Algorithm 3 (GPTQ + H-Scale) on bf16 weights: for each block of B columns, quantize
    the current weights with H-Scale (RTN start, window (down, up), h of the block), form
    E = (W_b - W_hat_b) / diag(U_b), and update the later columns by
    W[:, i+B:] -= E U[i:i+B, i+B:].  Returns codes, packed nibbles, w_hat (fp64) and the
    near-tie flags of every block quantization."""
    W = (_u16(w_u16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    m, n = W.shape
    if dead is not None:
        W[:, dead] = 0.0
    if block % 16 or n % block:
        raise ValueError("block must be a multiple of 16 dividing n")
    h = np.ascontiguousarray(h_f32, dtype=np.float32).reshape(n)
    out = {"codes": np.empty((m, n // 16), np.uint8), "packed": np.empty((m, n // 2), np.uint8),
           "w_hat": np.empty((m, n), np.float64), "near_tie": np.empty((m, n // 16), np.uint8)}
    for i in range(0, n, block):
        q = refine_f64(W[:, i:i + block], h[i:i + block], s_g, down, up)
        out["codes"][:, i // 16:(i + block) // 16] = q["codes"]
        out["packed"][:, i // 2:(i + block) // 2] = q["packed"]
        out["near_tie"][:, i // 16:(i + block) // 16] = q["near_tie"]
        out["w_hat"][:, i:i + block] = q["w_hat"]
        E = (W[:, i:i + block] - q["w_hat"]) / np.diag(U)[i:i + block]
        if i + block < n:
            W[:, i + block:] -= E @ U[i:i + block, i + block:]
    return out
