"""CPU oracle for the DART hot path (arXiv 2608.02032) -- TEST INFRASTRUCTURE.

A plain, slow, fp64 implementation of what the hot path computes, written
straight from the paper's definitions in ``dart_oracle.c`` and wrapped here
with numpy. It exists to check the CUDA path and for nothing else: only the
test suite, ``__graft_entry__.smoke()`` and the CPU-baseline / reference legs
of ``bench.py`` may import it. The product package never imports it, and it
imports nothing from the product package.

Every function takes and returns numpy arrays; inputs of any float dtype are
converted to float64. Layouts are the paper's (App. B.2 table of tensor
shapes): X ``Bsz x L x H x P``, dt ``Bsz x L x H``, A ``H``, B/C/Q
``Bsz x L x G x N``, E ``Bsz x L x G x P``, memories ``Bsz x M x H x N x P``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dart_oracle.c")
_SO = os.path.join(_HERE, "liboracle.so")
_lib = None

_i64 = ctypes.c_int64
_dp = ctypes.POINTER(ctypes.c_double)
_ip = ctypes.POINTER(ctypes.c_int64)


def build(force: bool = False) -> str:
    """Compile ``dart_oracle.c`` into ``liboracle.so`` (gcc, -O2, OpenMP, no fast-math)."""
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
        )
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_SO)
        lib.oracle_num_threads.restype = ctypes.c_int
        lib.oracle_ssd_recurrence.argtypes = [_i64] * 6 + [_dp] * 7
        lib.oracle_chunk_memories.argtypes = [_i64] * 7 + [_dp] * 5
        lib.oracle_sma.argtypes = [_i64] * 7 + [ctypes.c_double] + [_dp] * 4 + [_i64, _ip] + [_dp] * 3
        lib.oracle_merge.argtypes = [_i64, _i64] + [_dp] * 4
        lib.oracle_memory_inverse_rms.argtypes = [_i64, _i64, ctypes.c_double, _dp, _dp]
        lib.oracle_decode_step.argtypes = (
            [_i64] * 6 + [ctypes.c_double, _i64, _i64] + [_dp] * 13
        )
        lib.oracle_ssd_backward.argtypes = [_i64] * 7 + [_dp] * 12
        lib.oracle_sma_backward.argtypes = [_i64] * 7 + [ctypes.c_double] + [_dp] * 11
        for f in ("oracle_ssd_recurrence", "oracle_chunk_memories", "oracle_sma",
                  "oracle_merge", "oracle_decode_step", "oracle_memory_inverse_rms",
                  "oracle_ssd_backward", "oracle_sma_backward"):
            getattr(lib, f).restype = None
        _lib = lib
    return _lib


def num_threads() -> int:
    """OpenMP threads the oracle uses (OMP_NUM_THREADS, else all cores)."""
    return int(_load().oracle_num_threads())


def _f64(a) -> np.ndarray:
    if hasattr(a, "detach"):  # torch tensor
        a = a.detach().cpu().double().numpy()
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a: np.ndarray | None):
    if a is None:
        return None
    return a.ctypes.data_as(_dp)


def ssd_recurrence(X, dt, A, Bm, Cm):
    """Token recurrence of Sec. 2 / App. A. Returns (Y ``Bsz x L x H x P``, H_last ``Bsz x H x N x P``)."""
    X, dt, A, Bm, Cm = map(_f64, (X, dt, A, Bm, Cm))
    Bsz, L, H, P = X.shape
    G, N = Bm.shape[2], Bm.shape[3]
    Y = np.empty_like(X)
    Hl = np.empty((Bsz, H, N, P))
    _load().oracle_ssd_recurrence(Bsz, L, H, G, P, N, _ptr(X), _ptr(dt), _ptr(A), _ptr(Bm),
                                  _ptr(Cm), _ptr(Y), _ptr(Hl))
    return Y, Hl


def chunk_memories(X, dt, A, Bm, S: int):
    """Chunk state memories of Sec. 3 / App. A. Returns dH ``Bsz x M x H x N x P``."""
    X, dt, A, Bm = map(_f64, (X, dt, A, Bm))
    Bsz, L, H, P = X.shape
    G, N = Bm.shape[2], Bm.shape[3]
    M = -(-L // S)
    dH = np.empty((Bsz, M, H, N, P))
    _load().oracle_chunk_memories(Bsz, L, H, G, P, N, S, _ptr(X), _ptr(dt), _ptr(A), _ptr(Bm),
                                  _ptr(dH))
    return dH


def sma(dH, Q, Cm, E, S: int, eps: float, H: int | None = None, tokens=None, want_g=False):
    """State-memory attention of Sec. 3 / App. B.1 with the exact two-pass softmax.

    ``tokens``: None for every (b, t, h), else an ``n x 3`` int array of
    (b, t, h). Returns (R, lse[, g]); for ``tokens=None`` R is
    ``Bsz x L x H x P`` and lse ``Bsz x L x H``, else ``n x P`` and ``n``.
    """
    dH, Q, Cm, E = map(_f64, (dH, Q, Cm, E))
    Bsz, M, Hm, N, P = dH.shape
    H = Hm if H is None else H
    L, G = Q.shape[1], Q.shape[2]
    assert M == -(-L // S), "memory count must be ceil(L / S)"
    if tokens is None:
        ntok = Bsz * L * H
        tok = None
        R = np.empty((Bsz, L, H, P))
        lse = np.empty((Bsz, L, H))
    else:
        tok = np.ascontiguousarray(np.asarray(tokens, dtype=np.int64).reshape(-1, 3))
        ntok = tok.shape[0]
        R = np.empty((ntok, P))
        lse = np.empty((ntok,))
    g = np.empty((ntok, M)) if want_g else None
    _load().oracle_sma(Bsz, L, H, G, P, N, S, float(eps), _ptr(dH), _ptr(Q), _ptr(Cm), _ptr(E),
                       ntok, None if tok is None else tok.ctypes.data_as(_ip),
                       _ptr(R), _ptr(lse), _ptr(g))
    if want_g:
        return R, lse, g.reshape(R.shape[:-1] + (M,))
    return R, lse


def memory_inverse_rms(dH, eps: float):
    """Inverse RMS of each memory row along P (App. B.1): shape ``dH.shape[:-1]``."""
    dH = _f64(dH)
    P = dH.shape[-1]
    r = np.empty(dH.shape[:-1])
    _load().oracle_memory_inverse_rms(r.size, P, float(eps), _ptr(dH), _ptr(r))
    return r


def merge(Yssd, z, R):
    """Gated residual merge of Sec. 3: Y = Y_ssd + SiLU(z) R (z has one entry per row of P)."""
    Yssd, z, R = map(_f64, (Yssd, z, R))
    P = Yssd.shape[-1]
    rows = Yssd.size // P
    assert z.size == rows and R.shape == Yssd.shape
    Y = np.empty_like(Yssd)
    _load().oracle_merge(rows, P, _ptr(Yssd), _ptr(z), _ptr(R), _ptr(Y))
    return Y


def decode_step(cache, state, partial, x, dt, A, b, c, q, e, z, pos: int, S: int, eps: float):
    """One decode step (the oracle's reading of the paper's inference cache).

    Returns (y ``Bsz x H x P``, lse ``Bsz x H``, cache', state', partial'); the
    inputs are not modified.
    """
    cache, state, partial = (np.array(_f64(a), copy=True) for a in (cache, state, partial))
    x, dt, A, b, c, q, e, z = map(_f64, (x, dt, A, b, c, q, e, z))
    Bsz, m_cap, H, N, P = cache.shape
    G = b.shape[1]
    y = np.empty((Bsz, H, P))
    lse = np.empty((Bsz, H))
    _load().oracle_decode_step(Bsz, H, G, P, N, S, float(eps), int(pos), m_cap, _ptr(cache),
                               _ptr(state), _ptr(partial), _ptr(x), _ptr(dt), _ptr(A), _ptr(b),
                               _ptr(c), _ptr(q), _ptr(e), _ptr(z), _ptr(y), _ptr(lse))
    return y, lse, cache, state, partial


def forward(X, dt, A, Bm, Cm, Q, E, z, S: int, eps: float):
    """Whole prefill path: (Y_ssd, dH, R, lse, Y) from the definitions above."""
    Yssd, _ = ssd_recurrence(X, dt, A, Bm, Cm)
    dH = chunk_memories(X, dt, A, Bm, S)
    R, lse = sma(dH, Q, Cm, E, S, eps)
    Y = merge(Yssd, z, R)
    return Yssd, dH, R, lse, Y


def ssd_backward(X, dt, A, Bm, Cm, dY, dMem, S: int):
    """Gradients of the SSD scan (chain rule on the token recurrence of Sec. 2 / App. A).

    dY: gradient w.r.t. Y_ssd (``Bsz x L x H x P``); dMem: gradient w.r.t. the
    chunk memories (``Bsz x M x H x N x P``) or None. Returns (dX, d_dt, dA, dB,
    dC); dB and dC are summed over the heads of a group.
    """
    X, dt, A, Bm, Cm, dY = map(_f64, (X, dt, A, Bm, Cm, dY))
    dMem = None if dMem is None else _f64(dMem)
    Bsz, L, H, P = X.shape
    G, N = Bm.shape[2], Bm.shape[3]
    dX, ddt, dA = np.empty_like(X), np.empty_like(dt), np.empty_like(A)
    dB, dC = np.empty_like(Bm), np.empty_like(Cm)
    _load().oracle_ssd_backward(Bsz, L, H, G, P, N, S, _ptr(X), _ptr(dt), _ptr(A), _ptr(Bm),
                                _ptr(Cm), _ptr(dY), _ptr(dMem), _ptr(dX), _ptr(ddt), _ptr(dA),
                                _ptr(dB), _ptr(dC))
    return dX, ddt, dA, dB, dC


def sma_backward(dH, Q, Cm, E, z, dY, S: int, eps: float):
    """Gradients of state-memory attention + gated merge (Sec. 3 / App. B.1) w.r.t.
    the memories, Q, C, E and the gate logit z, for a loss gradient dY on
    Y = Y_ssd + SiLU(z) R. Returns (dMem, dQ, dC, dE, dz); the gradient w.r.t.
    Y_ssd is dY itself.
    """
    dH, Q, Cm, E, z, dY = map(_f64, (dH, Q, Cm, E, z, dY))
    Bsz, M, H, N, P = dH.shape
    L, G = Q.shape[1], Q.shape[2]
    dMem, dQ, dC, dE = np.empty_like(dH), np.empty_like(Q), np.empty_like(Cm), np.empty_like(E)
    dz = np.empty((Bsz, L, H))
    _load().oracle_sma_backward(Bsz, L, H, G, P, N, S, float(eps), _ptr(dH), _ptr(Q), _ptr(Cm),
                                _ptr(E), _ptr(z), _ptr(dY), _ptr(dMem), _ptr(dQ), _ptr(dC),
                                _ptr(dE), _ptr(dz))
    return dMem, dQ, dC, dE, dz


def backward(X, dt, A, Bm, Cm, Q, E, z, dY, S: int, eps: float):
    """Whole-layer backward for a loss gradient dY on Y: (dX, d_dt, dA, dB, dC, dQ, dE, dz).

    The SMA backward's memory gradient feeds the scan backward, and dC sums
    the SSD and SMA contributions.
    """
    dH = chunk_memories(X, dt, A, Bm, S)
    dMem, dQ, dC_sma, dE, dz = sma_backward(dH, Q, Cm, E, z, dY, S, eps)
    dX, ddt, dA, dB, dC_ssd = ssd_backward(X, dt, A, Bm, Cm, dY, dMem, S)
    return dX, ddt, dA, dB, dC_ssd + dC_sma, dQ, dE, dz
