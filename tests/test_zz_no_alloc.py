"""dart_sma_forward_noalloc against dart_sma_forward and against the oracle.

The no-allocation entry point serves callers that can neither allocate device
memory nor pass a workspace: a host framework that hands a plugin only its
input and output buffers, a service that forbids allocation after start-up,
a process under a fixed device-memory budget. Its scratch (the inverse RMS of
every memory row) is a fixed array inside the library, shared by every call.

Here it is called through the C ABI on two problems in a row. Before the
second call the shared scratch is poisoned with NaN by a call on all-NaN
memories of the larger problem, so that an entry the second call read without
writing it first would surface as NaN. Each result is compared with the regular
entry point's (rM = NULL, caller workspace) and with the oracle, at the
tolerance the other GPU tests use. The entry point always runs the CUDA-core
SMA kernel, so on tensor-core shapes it agrees with dart_sma_forward within the
bf16-input tolerance, not bit for bit. Collected last on purpose.
"""
import numpy as np
import pytest
import torch

from helpers import TOL, dev, host, oracle_prefill, rel_err
from paper_2608_02032_gb300 import api, binding
from paper_2608_02032_gb300.workloads import Workload, prefill_inputs

pytestmark = pytest.mark.gpu


def _case(w):
    inp = prefill_inputs(w)
    X, Bm, Cm, Q, E, z = (dev(inp[k], w.dtype) for k in ("X", "Bm", "Cm", "Q", "E", "z"))
    dtv, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s = api.chunk_scan(X, dtv, A, Bm, Cm, w.chunk, w.eps)
    return inp, (s, Q, Cm, E, z)


def _regular(w, s, Q, Cm, E, z):
    o = api.sma_forward(s.M, None, Q, Cm, E, z, s.Y_ssd, w.chunk, w.eps, want_R=True)
    return o.Y, o.R, o.lse


def _noalloc(w, s, Q, Cm, E, z, M=None):
    Bsz, L, H, P = s.Y_ssd.shape
    dims = binding.make_dims(Bsz, L, H, w.groups, P, w.dstate, w.chunk, Q.dtype, s.M.dtype,
                             s.Y_ssd.dtype, eps=w.eps)
    Y = torch.full_like(s.Y_ssd, float("nan"))
    R = torch.full_like(s.Y_ssd, float("nan"))
    lse = torch.full((Bsz, L, H), float("nan"), dtype=torch.float32, device=s.Y_ssd.device)
    binding.dart_sma_forward_noalloc(dims, s.M if M is None else M, Q, Cm, E, z, s.Y_ssd, Y, R, lse)
    return Y, R, lse


def test_noalloc_matches_sma_forward_and_oracle_on_two_calls_in_a_row(oracle_mod):
    assert torch.cuda.is_available(), "GPU test needs a CUDA device"
    binding.lib()
    # the first takes the tensor-core SMA in dart_sma_forward, the second the CUDA-core one
    cases = [Workload("noalloc_a", 2, 4, 1024, 64, 128, 128, seed=501),
             Workload("noalloc_b", 1, 2, 512, 32, 64, 64, dtype="f32", seed=502)]
    prepared = [(w, *_case(w)) for w in cases]
    for i, (w, inp, args) in enumerate(prepared):  # two calls in a row, different sizes and dtypes
        if i == 1:
            # poison the shared scratch: r of all-NaN memories of the larger problem
            w0, _, a0 = prepared[0]
            nan_M = torch.full_like(a0[0].M, float("nan"))
            poison = _noalloc(w0, *a0, M=nan_M)
            torch.cuda.synchronize()
            assert torch.isnan(poison[0][:, w0.chunk:]).any()  # the poison reached the outputs
        got = _noalloc(w, *args)
        torch.cuda.synchronize()
        want = _regular(w, *args)
        torch.cuda.synchronize()
        tol = TOL[w.dtype]
        ref = oracle_prefill(inp, w)
        for name, g, r in zip(("Y", "R", "lse"), got, want):
            gh = host(g)
            assert not np.isnan(gh).any(), (w.name, name, "stale scratch read")
            assert rel_err(gh, host(r)) <= tol, (w.name, name, "vs dart_sma_forward")
            assert rel_err(gh, ref[name]) <= tol, (w.name, name, "vs oracle")
    binding.dart_get_device_status()
