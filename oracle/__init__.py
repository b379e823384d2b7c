"""CPU oracle for the compression operators of arXiv 2401.07788 (test infrastructure).

This package is TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import it.  It wraps ``oracle.c`` (plain,
single-threaded C, built with ``-O2 -ffp-contract=off``) through ctypes and exchanges
numpy arrays.  It imports nothing from the CUDA library and the library imports
nothing from here.

Operators (paper sections): TopK §2.3, error feedback and EF21 §2.4, AQ-SGD §2.5,
min-max quantisation §2.2.  Stochastic rounding and its splitmix64 generator are not in
the paper; they follow the counter definition in ``oracle.c``.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]

_lock = threading.Lock()
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB_PATH) -> str:
    """Compile ``oracle.c`` into a shared library with gcc and return its path."""
    if not force and out == _LIB_PATH and os.path.exists(out) and (
        os.path.getmtime(out) >= os.path.getmtime(src)
    ):
        return out
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + ".tmp%d" % os.getpid()
    cmd = ["gcc", *_CFLAGS, "-I", _HERE, src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


_F32P = np.ctypeslib.ndpointer(dtype=np.float32, flags="C_CONTIGUOUS")
_I32P = np.ctypeslib.ndpointer(dtype=np.int32, flags="C_CONTIGUOUS")
_I64P = np.ctypeslib.ndpointer(dtype=np.int64, flags="C_CONTIGUOUS")
_U32P = np.ctypeslib.ndpointer(dtype=np.uint32, flags="C_CONTIGUOUS")
_i64 = ctypes.c_int64


def load(path: str | None = None) -> ctypes.CDLL:
    """Load (building if needed) the oracle library and declare its signatures."""
    global _lib
    with _lock:
        if path is None and _lib is not None:
            return _lib
        lib = ctypes.CDLL(path or build())
        lib.orc_splitmix64.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        lib.orc_splitmix64.restype = ctypes.c_uint64
        lib.orc_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        lib.orc_uniform.restype = ctypes.c_float
        lib.orc_topk_compress.argtypes = [_F32P, _i64, _i64, _i64, _F32P, _I32P]
        lib.orc_topk_decompress.argtypes = [_F32P, _I32P, _i64, _i64, _i64, _F32P]
        lib.orc_topk_gather.argtypes = [_F32P, _i64, _i64, _I32P, _i64, _F32P]
        lib.orc_ef_topk_compress.argtypes = [_F32P, _F32P, _i64, _i64, _i64, _F32P, _I32P]
        lib.orc_ef21_topk_compress.argtypes = [_F32P, _F32P, _i64, _i64, _i64, _F32P, _I32P]
        lib.orc_efmix_topk_compress.argtypes = [_F32P, _F32P, _i64, _i64, _i64, _F32P, _I32P]
        lib.orc_aqsgd_compress.argtypes = [_F32P, _F32P, _i64, _I64P, _i64, _i64, _i64, _i64,
                                           _F32P, _I32P]
        lib.orc_aqsgd_decompress.argtypes = [_F32P, _I32P, _F32P, _i64, _I64P, _i64, _i64,
                                             _i64, _i64]
        lib.orc_quant_row_words.argtypes = [_i64, ctypes.c_int]
        lib.orc_quant_row_words.restype = _i64
        lib.orc_quant_compress.argtypes = [_F32P, _i64, _i64, ctypes.c_int, ctypes.c_int,
                                           ctypes.c_uint64, _U32P, _F32P, _F32P]
        lib.orc_quant_decompress.argtypes = [_U32P, _F32P, _F32P, _i64, _i64, ctypes.c_int,
                                             _F32P]
        lib.orc_aqsgd_quant_compress.argtypes = [_F32P, _F32P, _i64, _I64P, _i64, _i64, _i64,
                                                 ctypes.c_int, ctypes.c_int, ctypes.c_uint64,
                                                 _U32P, _F32P, _F32P]
        lib.orc_aqsgd_quant_decompress.argtypes = [_U32P, _F32P, _F32P, _F32P, _i64, _I64P, _i64,
                                                   _i64, _i64, ctypes.c_int]
        for name in ("orc_aqsgd_quant_compress", "orc_aqsgd_quant_decompress"):
            getattr(lib, name).restype = None
        for name in ("orc_topk_compress", "orc_topk_decompress", "orc_topk_gather",
                     "orc_ef_topk_compress", "orc_efmix_topk_compress",
                     "orc_ef21_topk_compress", "orc_aqsgd_compress", "orc_aqsgd_decompress",
                     "orc_quant_compress", "orc_quant_decompress"):
            getattr(lib, name).restype = None
        if path is None:
            _lib = lib
        return lib


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


def _rows_cols(x: np.ndarray) -> tuple[int, int]:
    if x.ndim == 1:
        return 1, x.shape[0]
    return int(np.prod(x.shape[:-1])), x.shape[-1]


# --------------------------------------------------------------------------------------
# numpy-level API (shapes: x [..., L] is treated as rows x L)
# --------------------------------------------------------------------------------------

def splitmix64(seed: int, counter: int, lib=None) -> int:
    return int((lib or load()).orc_splitmix64(seed, counter))


def uniform(seed: int, i: int, lib=None) -> float:
    return float((lib or load()).orc_uniform(seed, i))


def topk_compress(x, k: int, lib=None):
    """TopK (§2.3) per row; returns (vals [R,k] f32, idx [R,k] i32)."""
    x = _f32(x)
    R, L = _rows_cols(x)
    vals = np.empty((R, k), np.float32)
    idx = np.empty((R, k), np.int32)
    (lib or load()).orc_topk_compress(x, R, L, k, vals, idx)
    return vals, idx


def topk_decompress(vals, idx, row_len: int, lib=None):
    vals = _f32(vals)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    R, k = _rows_cols(vals)
    y = np.empty((R, row_len), np.float32)
    (lib or load()).orc_topk_decompress(vals, idx, R, row_len, k, y)
    return y


def topk_gather(g, idx, lib=None):
    """TopK index reuse (§3.2, Table 5): the values of g at the kept indices idx [R, k]."""
    g = _f32(g)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    R, L = _rows_cols(g)
    k = idx.shape[-1]
    assert idx.size == R * k and (idx.size == 0 or (idx.min() >= 0 and idx.max() < L))
    vals = np.empty((R, k), np.float32)
    (lib or load()).orc_topk_gather(g, R, L, idx, k, vals)
    return vals


def ef_topk_compress(x, e, k: int, lib=None):
    """Error feedback (§2.4). ``e`` (float32, C-contiguous) is updated in place."""
    x = _f32(x)
    assert e.dtype == np.float32 and e.flags.c_contiguous and e.shape == x.shape
    R, L = _rows_cols(x)
    vals = np.empty((R, k), np.float32)
    idx = np.empty((R, k), np.int32)
    (lib or load()).orc_ef_topk_compress(x, e, R, L, k, vals, idx)
    return vals, idx


def efmix_topk_compress(x, e, k: int, lib=None):
    """EF-mixed (§2.4). ``e`` (float32, C-contiguous) is updated in place."""
    x = _f32(x)
    assert e.dtype == np.float32 and e.flags.c_contiguous and e.shape == x.shape
    R, L = _rows_cols(x)
    vals = np.empty((R, k), np.float32)
    idx = np.empty((R, k), np.int32)
    (lib or load()).orc_efmix_topk_compress(x, e, R, L, k, vals, idx)
    return vals, idx


def ef21_topk_compress(x, g, k: int, lib=None):
    """EF21 (§2.4). ``g`` is updated in place."""
    x = _f32(x)
    assert g.dtype == np.float32 and g.flags.c_contiguous and g.shape == x.shape
    R, L = _rows_cols(x)
    vals = np.empty((R, k), np.float32)
    idx = np.empty((R, k), np.int32)
    (lib or load()).orc_ef21_topk_compress(x, g, R, L, k, vals, idx)
    return vals, idx


def aqsgd_compress(x, buf, sample_ids, k: int, lib=None):
    """AQ-SGD with TopK (§2.5). x [n_ids, rows_per_sample, L]; buf [S, rows_per_sample, L]
    updated in place. Returns payload rows in the order of ``sample_ids``."""
    x = _f32(x)
    assert buf.dtype == np.float32 and buf.flags.c_contiguous
    ids = np.ascontiguousarray(sample_ids, dtype=np.int64)
    n_ids = ids.shape[0]
    S, rps, L = buf.shape
    assert x.shape == (n_ids, rps, L)
    vals = np.empty((n_ids * rps, k), np.float32)
    idx = np.empty((n_ids * rps, k), np.int32)
    (lib or load()).orc_aqsgd_compress(x, buf, S, ids, n_ids, rps, L, k, vals, idx)
    return vals, idx


def aqsgd_decompress(vals, idx, buf_recv, sample_ids, lib=None):
    vals = _f32(vals)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    ids = np.ascontiguousarray(sample_ids, dtype=np.int64)
    S, rps, L = buf_recv.shape
    k = vals.shape[-1]
    (lib or load()).orc_aqsgd_decompress(vals, idx, buf_recv, S, ids, ids.shape[0], rps, L, k)


def quant_row_words(row_len: int, bits: int, lib=None) -> int:
    return int((lib or load()).orc_quant_row_words(row_len, bits))


def quant_compress(x, bits: int, stochastic: bool = False, seed: int = 0, lib=None):
    """Min-max quantisation (§2.2). Returns (codes [R,W] u32, scale [R], minv [R])."""
    lib = lib or load()
    x = _f32(x)
    R, L = _rows_cols(x)
    W = quant_row_words(L, bits, lib)
    codes = np.empty((R, W), np.uint32)
    scale = np.empty(R, np.float32)
    minv = np.empty(R, np.float32)
    lib.orc_quant_compress(x, R, L, bits, 1 if stochastic else 0, seed, codes, scale, minv)
    return codes, scale, minv


def quant_decompress(codes, scale, minv, row_len: int, bits: int, lib=None):
    codes = np.ascontiguousarray(codes, dtype=np.uint32)
    scale = _f32(scale)
    minv = _f32(minv)
    R = scale.shape[0]
    y = np.empty((R, row_len), np.float32)
    (lib or load()).orc_quant_decompress(codes, scale, minv, R, row_len, bits, y)
    return y


def aqsgd_quant_compress(x, buf, sample_ids, bits: int, stochastic: bool = False, seed: int = 0,
                         lib=None):
    """AQ-SGD with quantisation (§2.5). x [n_ids, rps, L]; buf [S, rps, L] updated in place.
    Returns (codes, scale, minv) of the gathered rows."""
    x = _f32(x)
    assert buf.dtype == np.float32 and buf.flags.c_contiguous
    ids = np.ascontiguousarray(sample_ids, dtype=np.int64)
    n_ids = ids.shape[0]
    S, rps, L = buf.shape
    assert x.shape == (n_ids, rps, L)
    lib = lib or load()
    R = n_ids * rps
    W = quant_row_words(L, bits, lib)
    codes = np.zeros((R, W), np.uint32)
    scale = np.empty(R, np.float32)
    minv = np.empty(R, np.float32)
    lib.orc_aqsgd_quant_compress(x, buf, S, ids, n_ids, rps, L, bits, 1 if stochastic else 0,
                                 seed, codes, scale, minv)
    return codes, scale, minv


def aqsgd_quant_decompress(codes, scale, minv, buf_recv, sample_ids, bits: int, lib=None):
    ids = np.ascontiguousarray(sample_ids, dtype=np.int64)
    S, rps, L = buf_recv.shape
    assert buf_recv.dtype == np.float32 and buf_recv.flags.c_contiguous
    (lib or load()).orc_aqsgd_quant_decompress(
        np.ascontiguousarray(codes, dtype=np.uint32), _f32(scale), _f32(minv), buf_recv, S, ids,
        ids.shape[0], rps, L, bits)
    return buf_recv
