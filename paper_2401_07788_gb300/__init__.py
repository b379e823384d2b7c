"""Python binding of libmpcomp: GB300 (sm_103a) kernels for the activation and gradient
compression operators of arXiv 2401.07788 ("Activations and Gradients Compression for
Model-Parallel Training").

Each ``mpc_*`` function here has the name of the C entry point it calls (declared in
``include/mpcomp.h``) and only marshals arguments: it checks that tensors are contiguous
CUDA tensors of the right dtype, allocates outputs and workspaces with PyTorch when the
caller does not pass them, and passes raw device pointers and the current CUDA stream to
the library.  Every operator runs in the library's kernels; there is no fallback.  If
``libmpcomp.so`` has not been built, the first call raises ``MpcError``.
"""

from __future__ import annotations

import ctypes
import os

import torch

from ._build import LIB_PATH

__all__ = [
    "MpcError", "lib", "mpc_topk_workspace_bytes", "mpc_topk_compress", "mpc_topk_decompress",
    "mpc_topk_gather", "mpc_efmix_workspace_bytes", "mpc_efmix_topk_compress",
    "mpc_ef_topk_compress", "mpc_ef21_topk_compress", "mpc_aqsgd_compress",
    "mpc_aqsgd_decompress", "mpc_quant_codes_words", "mpc_quant_workspace_bytes",
    "mpc_quant_compress", "mpc_quant_decompress", "mpc_aqsgd_quant_workspace_bytes",
    "mpc_aqsgd_quant_compress", "mpc_aqsgd_quant_decompress", "mpc_get_status", "mpc_last_error",
    "mpc_set_knob", "MPC_KNOB_SPIN_LIMIT", "MPC_KNOB_TOPK_PATH", "MPC_KNOB_PDL", "STATUS_NAMES",
]

STATUS_NAMES = {0: "MPC_OK", 1: "MPC_ERR_INVALID_ARG", 2: "MPC_ERR_UNSUPPORTED",
                3: "MPC_ERR_WORKSPACE", 4: "MPC_ERR_CUDA", 5: "MPC_ERR_TIMEOUT",
                6: "MPC_ERR_DEVICE"}
MPC_KNOB_SPIN_LIMIT = 1
MPC_KNOB_TOPK_PATH = 2
MPC_KNOB_PDL = 3

_VP = ctypes.c_void_p
_I64 = ctypes.c_int64
_SZ = ctypes.c_size_t
_INT = ctypes.c_int
_U64 = ctypes.c_uint64

_SIGNATURES = {
    "mpc_version": ([], _INT),
    "mpc_topk_workspace_bytes": ([_I64, _I64, _I64], _SZ),
    "mpc_topk_compress": ([_VP, _I64, _I64, _I64, _VP, _VP, _VP, _SZ, _VP], _INT),
    "mpc_topk_decompress": ([_VP, _VP, _I64, _I64, _I64, _VP, _VP], _INT),
    "mpc_topk_gather": ([_VP, _I64, _I64, _VP, _I64, _VP, _VP], _INT),
    "mpc_efmix_workspace_bytes": ([_I64, _I64, _I64], _SZ),
    "mpc_efmix_topk_compress": ([_VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _SZ, _VP], _INT),
    "mpc_ef_topk_compress": ([_VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _SZ, _VP], _INT),
    "mpc_ef21_topk_compress": ([_VP, _VP, _I64, _I64, _I64, _VP, _VP, _VP, _SZ, _VP], _INT),
    "mpc_aqsgd_compress": ([_VP, _VP, _I64, _VP, _I64, _I64, _I64, _I64, _VP, _VP, _VP, _SZ,
                            _VP], _INT),
    "mpc_aqsgd_decompress": ([_VP, _VP, _VP, _I64, _VP, _I64, _I64, _I64, _I64, _VP], _INT),
    "mpc_quant_codes_words": ([_I64, _I64, _INT], _SZ),
    "mpc_quant_workspace_bytes": ([_I64, _I64, _INT], _SZ),
    "mpc_quant_compress": ([_VP, _I64, _I64, _INT, _INT, _U64, _VP, _VP, _VP, _VP, _SZ, _VP],
                           _INT),
    "mpc_quant_decompress": ([_VP, _VP, _VP, _I64, _I64, _INT, _VP, _VP], _INT),
    "mpc_aqsgd_quant_workspace_bytes": ([_I64, _I64, _I64, _INT], _SZ),
    "mpc_aqsgd_quant_compress": ([_VP, _VP, _I64, _VP, _I64, _I64, _I64, _INT, _INT, _U64, _VP,
                                  _VP, _VP, _VP, _SZ, _VP], _INT),
    "mpc_aqsgd_quant_decompress": ([_VP, _VP, _VP, _VP, _I64, _VP, _I64, _I64, _I64, _INT, _VP],
                                   _INT),
    "mpc_quant_compress_noalloc": ([_VP, _I64, _I64, _INT, _INT, _U64, _VP, _VP, _VP, _VP],
                                   _INT),
    "mpc_get_status": ([_VP], _INT),
    "mpc_last_error": ([], ctypes.c_char_p),
    "mpc_set_knob": ([_INT, _I64], _INT),
}

_lib = None


class MpcError(RuntimeError):
    """A libmpcomp call returned an error status."""

    def __init__(self, status: int, message: str):
        super().__init__("%s: %s" % (STATUS_NAMES.get(status, status), message))
        self.status = status


def lib(path: str | None = None) -> ctypes.CDLL:
    """The loaded libmpcomp.so with its C signatures declared."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise MpcError(2, "libmpcomp.so is not built at %s; run "
                          "`python -c 'import __graft_entry__ as g; g.build()'`" % p)
    handle = ctypes.CDLL(p)
    for name, (args, res) in _SIGNATURES.items():
        fn = getattr(handle, name)
        fn.argtypes = args
        fn.restype = res
    if path is None:
        _lib = handle
    return handle


def _check(status: int) -> None:
    if status != 0:
        raise MpcError(status, lib().mpc_last_error().decode(errors="replace"))


def _ptr(t: torch.Tensor | None):
    return None if t is None else _VP(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return _VP(s.cuda_stream)


def _cuda(t: torch.Tensor, dtype: torch.dtype, name: str) -> torch.Tensor:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise MpcError(1, "%s must be a CUDA tensor" % name)
    if t.dtype != dtype:
        raise MpcError(1, "%s must be %s, got %s" % (name, dtype, t.dtype))
    if not t.is_contiguous():
        raise MpcError(1, "%s must be contiguous" % name)
    return t


def _rows_cols(x: torch.Tensor) -> tuple[int, int]:
    if x.dim() == 0:
        raise MpcError(1, "x must have at least one dimension")
    L = x.shape[-1]
    return (x.numel() // L if L else 0), L


def _workspace(nbytes: int, ws, device) -> tuple:
    if nbytes == 0:
        return ws, (0 if ws is None else ws.numel() * ws.element_size())
    if ws is None:
        ws = torch.empty(nbytes, dtype=torch.uint8, device=device)
    return ws, ws.numel() * ws.element_size()


# ---------------------------------------------------------------------------------------
# TopK (§2.3), error feedback and EF21 (§2.4)
# ---------------------------------------------------------------------------------------

def mpc_topk_workspace_bytes(rows: int, row_len: int, k: int) -> int:
    return int(lib().mpc_topk_workspace_bytes(rows, row_len, k))


def _topk_outputs(x, k, vals, idx):
    R, L = _rows_cols(x)
    if vals is None:
        vals = torch.empty((R, k), dtype=torch.float32, device=x.device)
    if idx is None:
        idx = torch.empty((R, k), dtype=torch.int32, device=x.device)
    _cuda(vals, torch.float32, "vals")
    _cuda(idx, torch.int32, "idx")
    if vals.numel() != R * k or idx.numel() != R * k:
        raise MpcError(1, "vals/idx must hold rows*k = %d entries" % (R * k))
    return R, L, vals, idx


def mpc_topk_compress(x, k: int, vals=None, idx=None, ws=None, stream=None):
    """TopK per row of x (last dimension = row).  Returns (vals [R,k], idx [R,k])."""
    _cuda(x, torch.float32, "x")
    R, L, vals, idx = _topk_outputs(x, k, vals, idx)
    ws, wsb = _workspace(mpc_topk_workspace_bytes(R, L, k) if R else 0, ws, x.device)
    _check(lib().mpc_topk_compress(_ptr(x), R, L, k, _ptr(vals), _ptr(idx), _ptr(ws), wsb,
                                   _stream(stream)))
    return vals, idx


def mpc_ef_topk_compress(x, err, k: int, vals=None, idx=None, ws=None, stream=None):
    """Error feedback: TopK of x + err; err is rewritten in place."""
    _cuda(x, torch.float32, "x")
    _cuda(err, torch.float32, "err")
    if err.shape != x.shape:
        raise MpcError(1, "err must have the shape of x")
    R, L, vals, idx = _topk_outputs(x, k, vals, idx)
    ws, wsb = _workspace(mpc_topk_workspace_bytes(R, L, k) if R else 0, ws, x.device)
    _check(lib().mpc_ef_topk_compress(_ptr(x), _ptr(err), R, L, k, _ptr(vals), _ptr(idx),
                                      _ptr(ws), wsb, _stream(stream)))
    return vals, idx


def mpc_efmix_workspace_bytes(rows: int, row_len: int, k: int) -> int:
    return int(lib().mpc_efmix_workspace_bytes(rows, row_len, k))


def mpc_efmix_topk_compress(x, err, k: int, vals=None, idx=None, ws=None, stream=None):
    """EF-mixed (§2.4); ``err`` is updated in place."""
    _cuda(x, torch.float32, "x")
    _cuda(err, torch.float32, "err")
    if err.shape != x.shape:
        raise MpcError(1, "err must have the shape of x")
    R, L, vals, idx = _topk_outputs(x, k, vals, idx)
    ws, wsb = _workspace(mpc_efmix_workspace_bytes(R, L, k) if R else 0, ws, x.device)
    _check(lib().mpc_efmix_topk_compress(_ptr(x), _ptr(err), R, L, k, _ptr(vals), _ptr(idx),
                                         _ptr(ws), wsb, _stream(stream)))
    return vals, idx


def mpc_ef21_topk_compress(x, g, k: int, vals=None, idx=None, ws=None, stream=None):
    """EF21: TopK of x - g; g takes the sent values in place."""
    _cuda(x, torch.float32, "x")
    _cuda(g, torch.float32, "g")
    if g.shape != x.shape:
        raise MpcError(1, "g must have the shape of x")
    R, L, vals, idx = _topk_outputs(x, k, vals, idx)
    ws, wsb = _workspace(mpc_topk_workspace_bytes(R, L, k) if R else 0, ws, x.device)
    _check(lib().mpc_ef21_topk_compress(_ptr(x), _ptr(g), R, L, k, _ptr(vals), _ptr(idx),
                                        _ptr(ws), wsb, _stream(stream)))
    return vals, idx


def mpc_topk_decompress(vals, idx, row_len: int, y=None, stream=None):
    """Dense [R, row_len] from a TopK payload."""
    _cuda(vals, torch.float32, "vals")
    _cuda(idx, torch.int32, "idx")
    R, k = _rows_cols(vals)
    if y is None:
        y = torch.empty((R, row_len), dtype=torch.float32, device=vals.device)
    _cuda(y, torch.float32, "y")
    _check(lib().mpc_topk_decompress(_ptr(vals), _ptr(idx), R, row_len, k, _ptr(y),
                                     _stream(stream)))
    return y


def mpc_topk_gather(g, idx, vals=None, stream=None):
    """TopK index reuse (§3.2): the values of g [R, L] at the payload indices idx [R, k]."""
    _cuda(g, torch.float32, "g")
    _cuda(idx, torch.int32, "idx")
    R, L = _rows_cols(g)
    Ri, k = _rows_cols(idx)
    if Ri != R:
        raise MpcError(1, "idx must have one row per row of g")
    if vals is None:
        vals = torch.empty((R, k), dtype=torch.float32, device=g.device)
    _cuda(vals, torch.float32, "vals")
    _check(lib().mpc_topk_gather(_ptr(g), R, L, _ptr(idx), k, _ptr(vals), _stream(stream)))
    return vals


# ---------------------------------------------------------------------------------------
# AQ-SGD (§2.5)
# ---------------------------------------------------------------------------------------

def mpc_aqsgd_compress(x, buf, sample_ids, k: int, vals=None, idx=None, ws=None, stream=None):
    """x [n_ids, rps, L]; buf [num_samples, rps, L] updated in place; sample_ids int64."""
    _cuda(x, torch.float32, "x")
    _cuda(buf, torch.float32, "buf")
    _cuda(sample_ids, torch.int64, "sample_ids")
    if buf.dim() != 3 or x.dim() != 3 or x.shape[1:] != buf.shape[1:]:
        raise MpcError(1, "x must be [n_ids, rps, L] and buf [num_samples, rps, L]")
    S, rps, L = buf.shape
    n_ids = sample_ids.numel()
    if x.shape[0] != n_ids:
        raise MpcError(1, "x.shape[0] must equal the number of sample ids")
    R = n_ids * rps
    if vals is None:
        vals = torch.empty((R, k), dtype=torch.float32, device=x.device)
    if idx is None:
        idx = torch.empty((R, k), dtype=torch.int32, device=x.device)
    _cuda(vals, torch.float32, "vals")
    _cuda(idx, torch.int32, "idx")
    _check(lib().mpc_aqsgd_compress(_ptr(x), _ptr(buf), S, _ptr(sample_ids), n_ids, rps, L, k,
                                    _ptr(vals), _ptr(idx), _ptr(ws), 0 if ws is None else
                                    ws.numel() * ws.element_size(), _stream(stream)))
    return vals, idx


def mpc_aqsgd_decompress(vals, idx, buf_recv, sample_ids, stream=None):
    """Receiver: buf_recv[ids] += decompressed payload (in place)."""
    _cuda(vals, torch.float32, "vals")
    _cuda(idx, torch.int32, "idx")
    _cuda(buf_recv, torch.float32, "buf_recv")
    _cuda(sample_ids, torch.int64, "sample_ids")
    S, rps, L = buf_recv.shape
    k = vals.shape[-1]
    _check(lib().mpc_aqsgd_decompress(_ptr(vals), _ptr(idx), _ptr(buf_recv), S,
                                      _ptr(sample_ids), sample_ids.numel(), rps, L, k,
                                      _stream(stream)))
    return buf_recv


# ---------------------------------------------------------------------------------------
# Min-max quantisation (§2.2)
# ---------------------------------------------------------------------------------------

def mpc_quant_codes_words(rows: int, row_len: int, bits: int) -> int:
    return int(lib().mpc_quant_codes_words(rows, row_len, bits))


def mpc_quant_workspace_bytes(rows: int, row_len: int, bits: int) -> int:
    return int(lib().mpc_quant_workspace_bytes(rows, row_len, bits))


def mpc_quant_compress(x, bits: int, stochastic: bool = False, seed: int = 0, codes=None,
                       scale=None, minv=None, ws=None, stream=None):
    """Returns (codes [R, W] int32 holding uint32 words, scale [R], minv [R])."""
    _cuda(x, torch.float32, "x")
    R, L = _rows_cols(x)
    words = mpc_quant_codes_words(R, L, bits)
    if words == 0 and R > 0:
        raise MpcError(1, "bits=%d is not supported" % bits)
    W = words // R if R else 0
    if codes is None:
        codes = torch.empty((R, W), dtype=torch.int32, device=x.device)
    if scale is None:
        scale = torch.empty(R, dtype=torch.float32, device=x.device)
    if minv is None:
        minv = torch.empty(R, dtype=torch.float32, device=x.device)
    _cuda(codes, torch.int32, "codes")
    _cuda(scale, torch.float32, "scale")
    _cuda(minv, torch.float32, "minv")
    ws, wsb = _workspace(mpc_quant_workspace_bytes(R, L, bits) if R else 0, ws, x.device)
    _check(lib().mpc_quant_compress(_ptr(x), R, L, bits, 1 if stochastic else 0,
                                    seed & 0xFFFFFFFFFFFFFFFF, _ptr(codes), _ptr(scale),
                                    _ptr(minv), _ptr(ws), wsb, _stream(stream)))
    return codes, scale, minv


def mpc_quant_decompress(codes, scale, minv, row_len: int, bits: int, y=None, stream=None):
    _cuda(codes, torch.int32, "codes")
    _cuda(scale, torch.float32, "scale")
    _cuda(minv, torch.float32, "minv")
    R = scale.numel()
    if y is None:
        y = torch.empty((R, row_len), dtype=torch.float32, device=scale.device)
    _cuda(y, torch.float32, "y")
    _check(lib().mpc_quant_decompress(_ptr(codes), _ptr(scale), _ptr(minv), R, row_len, bits,
                                      _ptr(y), _stream(stream)))
    return y


def mpc_aqsgd_quant_workspace_bytes(n_ids: int, rows_per_sample: int, row_len: int,
                                    bits: int) -> int:
    return int(lib().mpc_aqsgd_quant_workspace_bytes(n_ids, rows_per_sample, row_len, bits))


def _aqsgd_shapes(x_shape, buf, sample_ids):
    if buf.dim() != 3:
        raise MpcError(1, "buf must be [num_samples, rps, L]")
    S, rps, L = buf.shape
    n_ids = sample_ids.numel()
    if x_shape is not None and tuple(x_shape) != (n_ids, rps, L):
        raise MpcError(1, "x must be [n_ids, rps, L] with buf [num_samples, rps, L]")
    return S, rps, L, n_ids


def mpc_aqsgd_quant_compress(x, buf, sample_ids, bits: int, stochastic: bool = False,
                             seed: int = 0, codes=None, scale=None, minv=None, ws=None,
                             stream=None):
    """AQ-SGD with quantisation (§2.5). x [n_ids, rps, L]; buf [num_samples, rps, L]
    updated in place; returns (codes [R, W] int32 of uint32 words, scale [R], minv [R])
    with R = n_ids * rps."""
    _cuda(x, torch.float32, "x")
    _cuda(buf, torch.float32, "buf")
    _cuda(sample_ids, torch.int64, "sample_ids")
    S, rps, L, n_ids = _aqsgd_shapes(x.shape, buf, sample_ids)
    R = n_ids * rps
    words = mpc_quant_codes_words(R, L, bits)
    if words == 0 and R > 0:
        raise MpcError(1, "bits=%d is not supported" % bits)
    W = words // R if R else 0
    if codes is None:
        codes = torch.empty((R, W), dtype=torch.int32, device=x.device)
    if scale is None:
        scale = torch.empty(R, dtype=torch.float32, device=x.device)
    if minv is None:
        minv = torch.empty(R, dtype=torch.float32, device=x.device)
    _cuda(codes, torch.int32, "codes")
    _cuda(scale, torch.float32, "scale")
    _cuda(minv, torch.float32, "minv")
    need = mpc_aqsgd_quant_workspace_bytes(n_ids, rps, L, bits) if R else 0
    ws, wsb = _workspace(need, ws, x.device)
    _check(lib().mpc_aqsgd_quant_compress(_ptr(x), _ptr(buf), S, _ptr(sample_ids), n_ids, rps,
                                          L, bits, 1 if stochastic else 0,
                                          seed & 0xFFFFFFFFFFFFFFFF, _ptr(codes), _ptr(scale),
                                          _ptr(minv), _ptr(ws), wsb, _stream(stream)))
    return codes, scale, minv


def mpc_aqsgd_quant_decompress(codes, scale, minv, buf_recv, sample_ids, bits: int,
                               stream=None):
    """Receiver: buf_recv[ids] += Dequant(codes) (in place)."""
    _cuda(codes, torch.int32, "codes")
    _cuda(scale, torch.float32, "scale")
    _cuda(minv, torch.float32, "minv")
    _cuda(buf_recv, torch.float32, "buf_recv")
    _cuda(sample_ids, torch.int64, "sample_ids")
    S, rps, L, n_ids = _aqsgd_shapes(None, buf_recv, sample_ids)
    _check(lib().mpc_aqsgd_quant_decompress(_ptr(codes), _ptr(scale), _ptr(minv),
                                            _ptr(buf_recv), S, _ptr(sample_ids), n_ids, rps,
                                            L, bits, _stream(stream)))
    return buf_recv


# ---------------------------------------------------------------------------------------
# Status and knobs
# ---------------------------------------------------------------------------------------

def mpc_get_status(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device status as a code."""
    return int(lib().mpc_get_status(_stream(stream)))


def mpc_last_error() -> str:
    return lib().mpc_last_error().decode(errors="replace")


def mpc_set_knob(knob: int, value: int) -> None:
    _check(lib().mpc_set_knob(knob, value))


# The compression block between pipeline stages (§2.1) built on the calls above.
from .boundary import CompressionBoundary, Quant, Reuse, TopK, with_boundaries  # noqa: E402

__all__ += ["CompressionBoundary", "Quant", "TopK", "Reuse", "with_boundaries"]
