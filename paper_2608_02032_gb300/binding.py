"""ctypes binding of ``libdart.so`` with the C entry points' names.

Argument marshalling only: every function checks that the tensors it is
given live on the GPU and are contiguous, passes their device pointers and
the current CUDA stream to the C ABI (``include/dart.h``) and turns a
non-zero ``dart_status`` into :class:`DartError`. All computation happens in
the library's CUDA kernels; there is no CPU path. If ``libdart.so`` has not
been built, :func:`lib` raises instead of falling back to anything.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdart.so")

DART_OK = 0
DART_F32, DART_BF16 = 0, 1
DART_OP_CHUNK_SCAN, DART_OP_SMA_FORWARD, DART_OP_DECODE_STEP = 0, 1, 2
DART_OP_SMA_BACKWARD, DART_OP_SCAN_BACKWARD, DART_OP_PREFILL_HOST = 3, 4, 5
STATUS_NAMES = {0: "DART_OK", 1: "DART_ERR_INVALID_ARG", 2: "DART_ERR_UNSUPPORTED",
                3: "DART_ERR_WORKSPACE", 4: "DART_ERR_CUDA", 5: "DART_ERR_TIMEOUT",
                6: "DART_ERR_TOO_LARGE"}

TORCH_DTYPE = {DART_F32: torch.float32, DART_BF16: torch.bfloat16}
DART_DTYPE = {torch.float32: DART_F32, torch.bfloat16: DART_BF16}

EXPORTED = ("dart_status_string", "dart_last_cuda_error", "dart_workspace_size",
            "dart_chunk_scan", "dart_sma_forward", "dart_decode_step", "dart_sma_forward_noalloc",
            "dart_launch_count", "dart_set_wait_limit_ns", "dart_get_device_status",
            "dart_sma_backward", "dart_chunk_scan_backward", "dart_test_withhold_copies",
            "dart_prefill_host", "dart_sma_forward_with_logits", "dart_sma_backward_with_logits",
            "dart_block_workspace_size", "dart_block_forward", "dart_sma_tiles_size",
            "dart_chunk_scan_with_tiles", "dart_sma_forward_with_tiles")


class DartError(RuntimeError):
    """A DART C-ABI call returned an error status."""

    def __init__(self, fn: str, status: int, detail: str = ""):
        self.status = status
        super().__init__(f"{fn}: {detail or STATUS_NAMES.get(status, status)}")


class dart_dims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int64), ("seqlen", ctypes.c_int64),
                ("nheads", ctypes.c_int64), ("ngroups", ctypes.c_int64),
                ("headdim", ctypes.c_int64), ("dstate", ctypes.c_int64),
                ("chunk", ctypes.c_int64), ("in_dtype", ctypes.c_int32),
                ("mem_dtype", ctypes.c_int32), ("out_dtype", ctypes.c_int32),
                ("eps", ctypes.c_float)]


class dart_block_dims(ctypes.Structure):
    _fields_ = [("core", dart_dims), ("d_model", ctypes.c_int64), ("conv_width", ctypes.c_int64),
                ("norm_eps", ctypes.c_float)]


def make_block_dims(batch, seqlen, d_model, nheads, ngroups=1, headdim=64, dstate=128, chunk=256,
                    conv_width=4, out_dtype=DART_F32, eps=1e-6, norm_eps=1e-5) -> dart_block_dims:
    """Sizes of one whole block (bf16 input and weights; ``out_dtype`` of its output)."""
    core = make_dims(batch, seqlen, nheads, ngroups, headdim, dstate, chunk, DART_BF16, DART_F32, out_dtype, eps)
    return dart_block_dims(core, d_model, conv_width, norm_eps)


def _code(dt):
    return DART_DTYPE[dt] if isinstance(dt, torch.dtype) else int(dt)


def make_dims(batch, seqlen, nheads, ngroups, headdim, dstate, chunk, dtype=DART_BF16,
              mem_dtype=DART_F32, out_dtype=DART_F32, eps=1e-6) -> dart_dims:
    """Sizes and dtypes of one call. ``dtype`` is the token-input type; memories
    and outputs default to fp32 (see include/dart.h for the supported triples)."""
    return dart_dims(batch, seqlen, nheads, ngroups, headdim, dstate, chunk, _code(dtype),
                     _code(mem_dtype), _code(out_dtype), eps)


_lib = None
_vp = ctypes.c_void_p


def lib() -> ctypes.CDLL:
    """Load libdart.so (raises if it is missing: build it with ``build.build()``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run python -m paper_2608_02032_gb300.build")
        L = ctypes.CDLL(LIB_PATH)
        dp = ctypes.POINTER(dart_dims)
        L.dart_status_string.restype = ctypes.c_char_p
        L.dart_status_string.argtypes = [ctypes.c_int]
        L.dart_last_cuda_error.restype = ctypes.c_int
        L.dart_workspace_size.restype = ctypes.c_size_t
        L.dart_workspace_size.argtypes = [dp, ctypes.c_int]
        L.dart_chunk_scan.restype = ctypes.c_int
        L.dart_chunk_scan.argtypes = [dp] + [_vp] * 10 + [ctypes.c_size_t, _vp]
        L.dart_sma_forward.restype = ctypes.c_int
        L.dart_sma_forward.argtypes = [dp] + [_vp] * 11 + [ctypes.c_size_t, _vp]
        L.dart_prefill_host.restype = ctypes.c_int
        L.dart_prefill_host.argtypes = [dp] + [_vp] * 10 + [ctypes.c_size_t, _vp]
        L.dart_decode_step.restype = ctypes.c_int
        L.dart_decode_step.argtypes = ([dp, ctypes.c_int64, ctypes.c_int64] + [_vp] * 14
                                       + [ctypes.c_size_t, _vp])
        L.dart_sma_forward_noalloc.restype = ctypes.c_int
        L.dart_sma_forward_noalloc.argtypes = [dp] + [_vp] * 10
        L.dart_launch_count.restype = ctypes.c_uint64
        L.dart_launch_count.argtypes = []
        L.dart_set_wait_limit_ns.restype = None
        L.dart_set_wait_limit_ns.argtypes = [ctypes.c_uint64]
        L.dart_get_device_status.restype = ctypes.c_int
        L.dart_get_device_status.argtypes = [_vp]
        L.dart_get_device_status.restype = ctypes.c_int
        L.dart_test_withhold_copies.argtypes = [ctypes.c_int]
        L.dart_test_withhold_copies.restype = None
        L.dart_sma_backward.argtypes = [dp] + [_vp] * 14 + [ctypes.c_size_t, _vp]
        L.dart_sma_backward.restype = ctypes.c_int
        L.dart_sma_forward_with_logits.restype = ctypes.c_int
        L.dart_sma_forward_with_logits.argtypes = [dp] + [_vp] * 12 + [ctypes.c_size_t, _vp]
        L.dart_sma_backward_with_logits.restype = ctypes.c_int
        L.dart_sma_backward_with_logits.argtypes = [dp] + [_vp] * 15 + [ctypes.c_size_t, _vp]
        L.dart_chunk_scan_backward.argtypes = [dp] + [_vp] * 13 + [ctypes.c_size_t, _vp]
        L.dart_chunk_scan_backward.restype = ctypes.c_int
        bp = ctypes.POINTER(dart_block_dims)
        L.dart_block_workspace_size.argtypes = [bp]
        L.dart_block_workspace_size.restype = ctypes.c_size_t
        L.dart_block_forward.argtypes = [bp] + [_vp] * 11 + [ctypes.c_size_t, _vp]
        L.dart_sma_tiles_size.restype = ctypes.c_size_t
        L.dart_sma_tiles_size.argtypes = [dp]
        L.dart_chunk_scan_with_tiles.restype = ctypes.c_int
        L.dart_chunk_scan_with_tiles.argtypes = [dp] + [_vp] * 11 + [ctypes.c_size_t, _vp]
        L.dart_sma_forward_with_tiles.restype = ctypes.c_int
        L.dart_sma_forward_with_tiles.argtypes = [dp] + [_vp] * 10
        L.dart_block_forward.restype = ctypes.c_int
        _lib = L
    return _lib


def _ptr(t: torch.Tensor | None, name: str):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor (the DART library has no CPU path)")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return _vp(t.data_ptr())


def _host_ptr(t: torch.Tensor, name: str):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.is_cuda:
        raise ValueError(f"{name} must be a host tensor (page-locked for the copies to overlap)")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return _vp(t.data_ptr())


def _stream(stream) -> _vp:
    if stream is None:
        stream = torch.cuda.current_stream()
    if isinstance(stream, torch.cuda.Stream):
        return _vp(stream.cuda_stream)
    return _vp(int(stream))


def _check(fn: str, status: int):
    if status != DART_OK:
        detail = lib().dart_status_string(status).decode()
        if status == 4:
            detail += f" (cudaError {lib().dart_last_cuda_error()})"
        raise DartError(fn, status, detail)


def dart_workspace_size(dims: dart_dims, op: int) -> int:
    return int(lib().dart_workspace_size(ctypes.byref(dims), op))


def _ws(workspace):
    if workspace is None:
        return None, 0
    return _ptr(workspace, "workspace"), workspace.numel() * workspace.element_size()


def dart_chunk_scan(dims, X, dt, A, Bm, Cm, Y_ssd, M, rM=None, final_state=None, workspace=None,
                    stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_chunk_scan", lib().dart_chunk_scan(
        ctypes.byref(dims), _ptr(X, "X"), _ptr(dt, "dt"), _ptr(A, "A"), _ptr(Bm, "Bm"),
        _ptr(Cm, "Cm"), _ptr(Y_ssd, "Y_ssd"), _ptr(M, "M"), _ptr(rM, "rM"),
        _ptr(final_state, "final_state"), w, nb, _stream(stream)))


def dart_sma_tiles_size(dims) -> int:
    return int(lib().dart_sma_tiles_size(ctypes.byref(dims)))


def dart_chunk_scan_with_tiles(dims, X, dt, A, Bm, Cm, Y_ssd, M, rM, final_state, tiles, workspace=None,
                               stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_chunk_scan_with_tiles", lib().dart_chunk_scan_with_tiles(
        ctypes.byref(dims), _ptr(X, "X"), _ptr(dt, "dt"), _ptr(A, "A"), _ptr(Bm, "Bm"),
        _ptr(Cm, "Cm"), _ptr(Y_ssd, "Y_ssd"), _ptr(M, "M"), _ptr(rM, "rM"),
        _ptr(final_state, "final_state"), _ptr(tiles, "tiles"), w, nb, _stream(stream)))


def dart_sma_forward_with_tiles(dims, tiles, Q, Cm, E, z, Y_ssd, Y, R=None, lse=None, stream=None) -> None:
    _check("dart_sma_forward_with_tiles", lib().dart_sma_forward_with_tiles(
        ctypes.byref(dims), _ptr(tiles, "tiles"), _ptr(Q, "Q"), _ptr(Cm, "Cm"), _ptr(E, "E"),
        _ptr(z, "z"), _ptr(Y_ssd, "Y_ssd"), _ptr(Y, "Y"), _ptr(R, "R"), _ptr(lse, "lse"),
        _stream(stream)))


def dart_sma_forward(dims, M, rM, Q, Cm, E, z, Y_ssd, Y, R=None, lse=None, workspace=None,
                     stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_sma_forward", lib().dart_sma_forward(
        ctypes.byref(dims), _ptr(M, "M"), _ptr(rM, "rM"), _ptr(Q, "Q"), _ptr(Cm, "Cm"),
        _ptr(E, "E"), _ptr(z, "z"), _ptr(Y_ssd, "Y_ssd"), _ptr(Y, "Y"), _ptr(R, "R"),
        _ptr(lse, "lse"), w, nb, _stream(stream)))


def dart_sma_forward_noalloc(dims, M, Q, Cm, E, z, Y_ssd, Y, R=None, lse=None, stream=None) -> None:
    """dart_sma_forward with rM = NULL for callers that cannot allocate: its
    scratch is a fixed 4 MiB array inside the library (see include/dart.h)."""
    _check("dart_sma_forward_noalloc", lib().dart_sma_forward_noalloc(
        ctypes.byref(dims), _ptr(M, "M"), _ptr(Q, "Q"), _ptr(Cm, "Cm"), _ptr(E, "E"),
        _ptr(z, "z"), _ptr(Y_ssd, "Y_ssd"), _ptr(Y, "Y"), _ptr(R, "R"), _ptr(lse, "lse"),
        _stream(stream)))


def dart_decode_step(dims, pos, m_cap, cache, state, partial, x, dt, A, b, c, q, e, z, y,
                     lse=None, workspace=None, stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_decode_step", lib().dart_decode_step(
        ctypes.byref(dims), int(pos), int(m_cap), _ptr(cache, "cache"), _ptr(state, "state"),
        _ptr(partial, "partial"), _ptr(x, "x"), _ptr(dt, "dt"), _ptr(A, "A"), _ptr(b, "b"),
        _ptr(c, "c"), _ptr(q, "q"), _ptr(e, "e"), _ptr(z, "z"), _ptr(y, "y"), _ptr(lse, "lse"),
        w, nb, _stream(stream)))


def dart_prefill_host(dims, X, dt, A, Bm, Cm, Q, E, z, Y, workspace=None, stream=None) -> None:
    """Host tensors in (X, dt, A, Bm, Cm, Q, E, z) and out (Y); a device workspace."""
    w, nb = _ws(workspace)
    _check("dart_prefill_host", lib().dart_prefill_host(
        ctypes.byref(dims), _host_ptr(X, "X"), _host_ptr(dt, "dt"), _host_ptr(A, "A"),
        _host_ptr(Bm, "Bm"), _host_ptr(Cm, "Cm"), _host_ptr(Q, "Q"), _host_ptr(E, "E"),
        _host_ptr(z, "z"), _host_ptr(Y, "Y"), w, nb, _stream(stream)))


def dart_sma_forward_with_logits(dims, M, rM, Q, Cm, E, z, Y_ssd, Y, R, lse, logits, workspace=None,
                                 stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_sma_forward_with_logits", lib().dart_sma_forward_with_logits(
        ctypes.byref(dims), _ptr(M, "M"), _ptr(rM, "rM"), _ptr(Q, "Q"), _ptr(Cm, "Cm"), _ptr(E, "E"),
        _ptr(z, "z"), _ptr(Y_ssd, "Y_ssd"), _ptr(Y, "Y"), _ptr(R, "R"), _ptr(lse, "lse"),
        _ptr(logits, "logits"), w, nb, _stream(stream)))


def dart_sma_backward_with_logits(dims, M, rM, Q, Cm, E, z, lse, logits, dY, dM, dQ, dC, dE, dz,
                                  workspace=None, stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_sma_backward_with_logits", lib().dart_sma_backward_with_logits(
        ctypes.byref(dims), _ptr(M, "M"), _ptr(rM, "rM"), _ptr(Q, "Q"), _ptr(Cm, "Cm"), _ptr(E, "E"),
        _ptr(z, "z"), _ptr(lse, "lse"), _ptr(logits, "logits"), _ptr(dY, "dY"), _ptr(dM, "dM"),
        _ptr(dQ, "dQ"), _ptr(dC, "dC"), _ptr(dE, "dE"), _ptr(dz, "dz"), w, nb, _stream(stream)))


def dart_sma_backward(dims, M, rM, Q, Cm, E, z, lse, dY, dM, dQ, dC, dE, dz, workspace=None,
                      stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_sma_backward", lib().dart_sma_backward(
        ctypes.byref(dims), _ptr(M, "M"), _ptr(rM, "rM"), _ptr(Q, "Q"), _ptr(Cm, "Cm"),
        _ptr(E, "E"), _ptr(z, "z"), _ptr(lse, "lse"), _ptr(dY, "dY"), _ptr(dM, "dM"),
        _ptr(dQ, "dQ"), _ptr(dC, "dC"), _ptr(dE, "dE"), _ptr(dz, "dz"), w, nb, _stream(stream)))


def dart_chunk_scan_backward(dims, X, dt, A, Bm, Cm, dY, dM, dX, ddt, dA, dB, dC, workspace=None,
                             stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_chunk_scan_backward", lib().dart_chunk_scan_backward(
        ctypes.byref(dims), _ptr(X, "X"), _ptr(dt, "dt"), _ptr(A, "A"), _ptr(Bm, "Bm"),
        _ptr(Cm, "Cm"), _ptr(dY, "dY"), _ptr(dM, "dM"), _ptr(dX, "dX"), _ptr(ddt, "ddt"),
        _ptr(dA, "dA"), _ptr(dB, "dB"), _ptr(dC, "dC"), w, nb, _stream(stream)))


def dart_block_workspace_size(dims: dart_block_dims) -> int:
    return int(lib().dart_block_workspace_size(ctypes.byref(dims)))


def dart_block_forward(dims, U, W_in, conv_w, conv_b, dt_bias, A_log, D, norm_w, W_out, out, workspace=None,
                       stream=None) -> None:
    w, nb = _ws(workspace)
    _check("dart_block_forward", lib().dart_block_forward(
        ctypes.byref(dims), _ptr(U, "U"), _ptr(W_in, "W_in"), _ptr(conv_w, "conv_w"), _ptr(conv_b, "conv_b"),
        _ptr(dt_bias, "dt_bias"), _ptr(A_log, "A_log"), _ptr(D, "D"), _ptr(norm_w, "norm_w"),
        _ptr(W_out, "W_out"), _ptr(out, "out"), w, nb, _stream(stream)))


def dart_get_device_status(stream=None) -> None:
    _check("dart_get_device_status", lib().dart_get_device_status(_stream(stream)))


def dart_launch_count() -> int:
    """Kernels the library has launched in this process."""
    return int(lib().dart_launch_count())


def dart_test_withhold_copies(on: bool) -> None:
    """Failure-path test hook: tensor-core SMA launches issue no operand copies while on."""
    lib().dart_test_withhold_copies(1 if on else 0)


def dart_set_wait_limit_ns(limit_ns: int) -> None:
    """Bound on each device-side wait of the tensor-core kernels (0 = default 2 s)."""
    lib().dart_set_wait_limit_ns(int(limit_ns))
