"""Allocating wrappers over the C ABI: the calls a PyTorch user makes.

Each wrapper allocates its outputs and workspace with PyTorch on the inputs'
device and calls one entry point of ``libdart.so`` on the current stream.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import binding as B


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype not in B.DART_DTYPE:
        raise TypeError(f"unsupported dtype {t.dtype}; use float32 or bfloat16")
    return B.DART_DTYPE[t.dtype]


def _workspace(dims, op, device) -> torch.Tensor | None:
    n = B.dart_workspace_size(dims, op)
    if n == 0:
        return None
    return torch.empty(n, dtype=torch.uint8, device=device)


@dataclass
class ScanOut:
    Y_ssd: torch.Tensor  # (Bsz, L, H, P)
    M: torch.Tensor      # (Bsz, M, H, N, P) chunk state memories
    rM: torch.Tensor     # (Bsz, M, H, N) inverse RMS of each memory row
    final_state: torch.Tensor | None  # (Bsz, H, N, P) fp32


def chunk_scan(X, dt, A, Bm, Cm, chunk: int, eps: float = 1e-6, final_state: bool = False,
               workspace: torch.Tensor | None = None, mem_dtype=torch.float32,
               out_dtype=torch.float32) -> ScanOut:
    """Chunked SSD scan with chunk state memories (``dart_chunk_scan``)."""
    Bsz, L, H, P = X.shape
    G, N = Bm.shape[2], Bm.shape[3]
    code = _dtype_code(X)
    dims = B.make_dims(Bsz, L, H, G, P, N, chunk, code, mem_dtype, out_dtype, eps=eps)
    M = -(-L // chunk)  # ceil: a ragged last chunk keeps its (partial) memory
    dev = X.device
    Y = torch.empty(X.shape, dtype=out_dtype, device=dev)
    Mem = torch.empty(Bsz, M, H, N, P, dtype=mem_dtype, device=dev)
    rM = torch.empty(Bsz, M, H, N, dtype=torch.float32, device=dev)
    fs = torch.empty(Bsz, H, N, P, dtype=torch.float32, device=dev) if final_state else None
    ws = workspace if workspace is not None else _workspace(dims, B.DART_OP_CHUNK_SCAN, dev)
    B.dart_chunk_scan(dims, X, dt, A, Bm, Cm, Y, Mem, rM, fs, ws)
    return ScanOut(Y, Mem, rM, fs)


@dataclass
class SmaOut:
    Y: torch.Tensor             # (Bsz, L, H, P) gated merge
    R: torch.Tensor | None      # (Bsz, L, H, P) SMA readout
    lse: torch.Tensor           # (Bsz, L, H) fp32 logsumexp over earlier chunks
    logits: torch.Tensor | None = None  # (Bsz, H, M, L) fp32, saved for the backward


def sma_forward(Mem, rM, Q, Cm, E, z, Y_ssd, chunk: int, eps: float = 1e-6, want_R: bool = True,
                workspace: torch.Tensor | None = None, save_logits: bool = False) -> SmaOut:
    """State-memory attention and gated merge (``dart_sma_forward``). ``save_logits``
    (tensor-core shapes) also keeps the logits for ``sma_backward``
    (``dart_sma_forward_with_logits``)."""
    Bsz, L, H, P = Y_ssd.shape
    G, N = Q.shape[2], Q.shape[3]
    dims = B.make_dims(Bsz, L, H, G, P, N, chunk, _dtype_code(Q), _dtype_code(Mem),
                       _dtype_code(Y_ssd), eps=eps)
    dev = Y_ssd.device
    Y = torch.empty_like(Y_ssd)
    R = torch.empty_like(Y_ssd) if want_R else None
    lse = torch.empty(Bsz, L, H, dtype=torch.float32, device=dev)
    ws = workspace if workspace is not None else _workspace(dims, B.DART_OP_SMA_FORWARD, dev)
    if save_logits:
        logits = torch.empty(Bsz, H, L // chunk, L, dtype=torch.float32, device=dev)
        B.dart_sma_forward_with_logits(dims, Mem, rM, Q, Cm, E, z, Y_ssd, Y, R, lse, logits, ws)
        return SmaOut(Y, R, lse, logits)
    B.dart_sma_forward(dims, Mem, rM, Q, Cm, E, z, Y_ssd, Y, R, lse, ws)
    return SmaOut(Y, R, lse)


def prefill_forward(X, dt, A, Bm, Cm, Q, E, z, chunk: int, eps: float = 1e-6, want_R=False,
                    mem_dtype=torch.float32, out_dtype=torch.float32, save_logits: bool = False):
    """Whole DART hot path of one block for a prefill: scan, SMA and merge
    (``save_logits``: keep the SMA logits for ``layer_backward``)."""
    s = chunk_scan(X, dt, A, Bm, Cm, chunk, eps, mem_dtype=mem_dtype, out_dtype=out_dtype)
    o = sma_forward(s.M, s.rM, Q, Cm, E, z, s.Y_ssd, chunk, eps, want_R=want_R, save_logits=save_logits)
    return s, o


def prefill_from_host(X, dt, A, Bm, Cm, Q, E, z, chunk: int, eps: float = 1e-6,
                      out_dtype=torch.float32, Y=None, workspace=None, stream=None):
    """The prefill (scan, SMA, merge) from host tensors to a host tensor
    (``dart_prefill_host``): copies overlapped with the kernels, head group by head
    group. Inputs should be page-locked (``pin_memory()``); ``Y`` (allocated
    page-locked when not given) is complete once ``stream`` (default: the current
    stream) is synchronised. ``workspace`` is device memory reused across calls.
    Returns (Y, workspace)."""
    Bsz, L, H, P = X.shape
    G, N = Bm.shape[2], Bm.shape[3]
    dims = B.make_dims(Bsz, L, H, G, P, N, chunk, _dtype_code(X), B.DART_F32, out_dtype, eps=eps)
    if Y is None:
        Y = torch.empty(Bsz, L, H, P, dtype=out_dtype).pin_memory()
    if workspace is None:
        workspace = torch.empty(B.dart_workspace_size(dims, B.DART_OP_PREFILL_HOST), dtype=torch.uint8,
                                device="cuda")
    if stream is None:
        stream = torch.cuda.current_stream()
    B.dart_prefill_host(dims, X, dt, A, Bm, Cm, Q, E, z, Y, workspace, stream)
    return Y, workspace


def decode_step(cache, state, partial, x, dt, A, b, c, q, e, z, pos: int, chunk: int,
                eps: float = 1e-6, out_dtype=torch.float32):
    """One decode step (``dart_decode_step``); cache, state and partial are updated in place.

    Returns (y ``Bsz x H x P``, lse ``Bsz x H``).
    """
    Bsz, m_cap, H, N, P = cache.shape
    G = b.shape[1]
    dims = B.make_dims(Bsz, 1, H, G, P, N, chunk, _dtype_code(x), _dtype_code(cache),
                       out_dtype, eps=eps)
    y = torch.empty(x.shape, dtype=out_dtype, device=x.device)
    lse = torch.empty(Bsz, H, dtype=torch.float32, device=x.device)
    B.dart_decode_step(dims, pos, m_cap, cache, state, partial, x, dt, A, b, c, q, e, z, y, lse)
    return y, lse


@dataclass
class LayerGrads:
    dX: torch.Tensor    # (Bsz, L, H, P) fp32
    ddt: torch.Tensor   # (Bsz, L, H) fp32
    dA: torch.Tensor    # (H,) fp32
    dB: torch.Tensor    # (Bsz, L, G, N) fp32
    dC: torch.Tensor    # (Bsz, L, G, N) fp32, SSD + SMA parts
    dQ: torch.Tensor    # (Bsz, L, G, N) fp32
    dE: torch.Tensor    # (Bsz, L, G, P) fp32
    dz: torch.Tensor    # (Bsz, L, H) fp32
    dM: torch.Tensor    # (Bsz, M, H, N, P) fp32 gradient of the chunk memories


def sma_backward(Mem, rM, Q, Cm, E, z, lse, dY, chunk: int, eps: float = 1e-6,
                 workspace: torch.Tensor | None = None, logits: torch.Tensor | None = None):
    """Backward of ``sma_forward`` (``dart_sma_backward``, or
    ``dart_sma_backward_with_logits`` given the forward's saved logits):
    (dM, dQ, dC, dE, dz), all fp32."""
    Bsz, L, H, P = dY.shape
    G, N = Q.shape[2], Q.shape[3]
    dims = B.make_dims(Bsz, L, H, G, P, N, chunk, _dtype_code(Q), _dtype_code(Mem),
                       B.DART_F32, eps=eps)
    dev = dY.device
    f32 = dict(dtype=torch.float32, device=dev)
    dM = torch.empty(Mem.shape, **f32)
    dQ, dC, dE = torch.empty(Q.shape, **f32), torch.empty(Cm.shape, **f32), torch.empty(E.shape, **f32)
    dz = torch.empty(Bsz, L, H, **f32)
    ws = workspace if workspace is not None else _workspace(dims, B.DART_OP_SMA_BACKWARD, dev)
    if logits is not None:
        B.dart_sma_backward_with_logits(dims, Mem, rM, Q, Cm, E, z, lse, logits, dY, dM, dQ, dC, dE, dz, ws)
    else:
        B.dart_sma_backward(dims, Mem, rM, Q, Cm, E, z, lse, dY, dM, dQ, dC, dE, dz, ws)
    return dM, dQ, dC, dE, dz


def chunk_scan_backward(X, dt, A, Bm, Cm, dY, dM, chunk: int, dC=None, eps: float = 1e-6,
                        workspace: torch.Tensor | None = None):
    """Backward of ``chunk_scan`` (``dart_chunk_scan_backward``): (dX, ddt, dA, dB, dC), fp32.

    ``dC``, when given (fp32), is accumulated into (e.g. the SMA part); else it starts at zero.
    """
    Bsz, L, H, P = X.shape
    G, N = Bm.shape[2], Bm.shape[3]
    dims = B.make_dims(Bsz, L, H, G, P, N, chunk, _dtype_code(X), B.DART_F32, B.DART_F32, eps=eps)
    dev = X.device
    f32 = dict(dtype=torch.float32, device=dev)
    dX, ddt, dA = torch.empty(X.shape, **f32), torch.empty(dt.shape, **f32), torch.empty(A.shape, **f32)
    dB = torch.empty(Bm.shape, **f32)
    dC = torch.zeros(Cm.shape, **f32) if dC is None else dC
    ws = workspace if workspace is not None else _workspace(dims, B.DART_OP_SCAN_BACKWARD, dev)
    B.dart_chunk_scan_backward(dims, X, dt, A, Bm, Cm, dY, dM, dX, ddt, dA, dB, dC, ws)
    return dX, ddt, dA, dB, dC


def layer_backward(X, dt, A, Bm, Cm, Q, E, z, dY, scan: ScanOut, sma: SmaOut, chunk: int,
                   eps: float = 1e-6) -> LayerGrads:
    """Backward of ``prefill_forward`` for a loss gradient dY on Y: SMA backward, whose
    memory gradient and dC feed the scan backward."""
    dM, dQ, dC, dE, dz = sma_backward(scan.M, scan.rM, Q, Cm, E, z, sma.lse, dY, chunk, eps,
                                      logits=sma.logits)
    dX, ddt, dA, dB, dC = chunk_scan_backward(X, dt, A, Bm, Cm, dY, dM, chunk, dC=dC, eps=eps)
    return LayerGrads(dX, ddt, dA, dB, dC, dQ, dE, dz, dM)


def block_forward(U, W_in, conv_w, conv_b, dt_bias, A_log, D, norm_w, W_out, heads: int, chunk: int = 256,
                  groups: int = 1, headdim: int = 64, dstate: int = 128, eps: float = 1e-6,
                  norm_eps: float = 1e-5, out_dtype=torch.float32, workspace=None) -> torch.Tensor:
    """One whole DART block for a prefill (``dart_block_forward``): in-projection,
    convolution, the hot path, D skip, gated RMSNorm and out-projection. U and the
    projection weights are bf16, the small parameters fp32; returns out
    (Bsz, L, d_model) in ``out_dtype``."""
    Bsz, L, d_model = U.shape
    dims = B.make_block_dims(Bsz, L, d_model, heads, groups, headdim, dstate, chunk, conv_w.shape[1],
                             B.DART_DTYPE[out_dtype], eps, norm_eps)
    out = torch.empty(Bsz, L, d_model, dtype=out_dtype, device=U.device)
    ws = workspace
    if ws is None:
        ws = torch.empty(max(B.dart_block_workspace_size(dims), 256), dtype=torch.uint8, device=U.device)
    B.dart_block_forward(dims, U, W_in, conv_w, conv_b, dt_bias, A_log, D, norm_w, W_out, out, ws)
    return out
