"""Shared test plumbing: tolerance metric, device transfer, oracle/GPU runners.

Inputs always come from ``paper_2608_02032_gb300.workloads`` (seeded, CPU);
expected values always come from ``oracle`` on those same inputs. The GPU
side is called only through the C ABI (``binding``/``api``).
"""
from __future__ import annotations

import numpy as np
import torch

# max |gpu - oracle| / RMS(oracle) per output tensor
TOL = {"f32": 1e-4, "bf16": 2e-2}
TORCH = {"f32": torch.float32, "bf16": torch.bfloat16}


def rel_err(got, ref) -> float:
    """max|got - ref| / RMS(ref) over entries where ref is finite; non-finite
    entries of ref (lse = -inf) must be matched exactly."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    fin = np.isfinite(ref)
    if not np.all(fin):
        assert np.array_equal(got[~fin], ref[~fin]), "non-finite entries differ"
    if not np.any(fin):
        return 0.0
    rms = np.sqrt(np.mean(ref[fin] ** 2))
    if rms == 0.0:
        return float(np.max(np.abs(got[fin])))
    return float(np.max(np.abs(got[fin] - ref[fin])) / rms)


def dev(t: torch.Tensor, dtype: str | torch.dtype, device="cuda") -> torch.Tensor:
    if isinstance(dtype, str):
        dtype = TORCH[dtype]
    return t.to(device=device, dtype=dtype).contiguous()


def host(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().double().numpy()


def gpu_prefill(inp: dict, w, want_R=True) -> dict:
    """Run dart_chunk_scan + dart_sma_forward on the GPU; returns CPU float64 arrays."""
    from paper_2608_02032_gb300 import api

    dt_ = w.dtype
    X, Bm, Cm, Q, E, z = (dev(inp[k], dt_) for k in ("X", "Bm", "Cm", "Q", "E", "z"))
    dtv, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s = api.chunk_scan(X, dtv, A, Bm, Cm, w.chunk, w.eps, final_state=True)
    o = api.sma_forward(s.M, s.rM, Q, Cm, E, z, s.Y_ssd, w.chunk, w.eps, want_R=want_R)
    torch.cuda.synchronize()
    out = dict(Y_ssd=host(s.Y_ssd), M=host(s.M), rM=host(s.rM), final_state=host(s.final_state),
               Y=host(o.Y), lse=host(o.lse))
    if want_R:
        out["R"] = host(o.R)
    return out


def oracle_prefill(inp: dict, w) -> dict:
    import oracle

    Yssd, Hl = oracle.ssd_recurrence(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"])
    dH = oracle.chunk_memories(inp["X"], inp["dt"], inp["A"], inp["Bm"], w.chunk)
    R, lse = oracle.sma(dH, inp["Q"], inp["Cm"], inp["E"], w.chunk, w.eps)
    Y = oracle.merge(Yssd, inp["z"], R)
    rM = oracle.memory_inverse_rms(dH, w.eps)
    return dict(Y_ssd=Yssd, M=dH, rM=rM, final_state=Hl, R=R, lse=lse, Y=Y)
