"""dart_sma_forward_noalloc against dart_sma_forward.

The no-allocation entry point serves callers that can neither allocate device
memory nor pass a workspace: a host framework that hands a plugin only its
input and output buffers, a service that forbids allocation after start-up,
a process under a fixed device-memory budget. Its scratch (the inverse RMS of
every memory row) is a fixed array inside the library. Here it is called
through the C ABI twice in a row, on two different problems, and each result
is compared with the regular entry point's (rM = NULL, caller workspace) at
the tolerance the other GPU tests use. Collected last on purpose.
"""
import pytest
import torch

from helpers import TOL, dev, host, rel_err
from paper_2608_02032_gb300 import api, binding
from paper_2608_02032_gb300.workloads import Workload, prefill_inputs

pytestmark = pytest.mark.gpu


def _case(w):
    inp = prefill_inputs(w)
    X, Bm, Cm, Q, E, z = (dev(inp[k], w.dtype) for k in ("X", "Bm", "Cm", "Q", "E", "z"))
    dtv, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s = api.chunk_scan(X, dtv, A, Bm, Cm, w.chunk, w.eps)
    return s, Q, Cm, E, z


def _regular(w, s, Q, Cm, E, z):
    o = api.sma_forward(s.M, None, Q, Cm, E, z, s.Y_ssd, w.chunk, w.eps, want_R=True)
    return o.Y, o.R, o.lse


def _noalloc(w, s, Q, Cm, E, z):
    Bsz, L, H, P = s.Y_ssd.shape
    dims = binding.make_dims(Bsz, L, H, w.groups, P, w.dstate, w.chunk, Q.dtype, s.M.dtype,
                             s.Y_ssd.dtype, eps=w.eps)
    Y = torch.full_like(s.Y_ssd, float("nan"))
    R = torch.full_like(s.Y_ssd, float("nan"))
    lse = torch.full((Bsz, L, H), float("nan"), dtype=torch.float32, device=s.Y_ssd.device)
    binding.dart_sma_forward_noalloc(dims, s.M, Q, Cm, E, z, s.Y_ssd, Y, R, lse)
    return Y, R, lse


def test_noalloc_matches_sma_forward_on_two_calls_in_a_row():
    assert torch.cuda.is_available(), "GPU test needs a CUDA device"
    binding.lib()
    cases = [Workload("noalloc_a", 2, 4, 1024, 64, 128, 128, seed=501),
             Workload("noalloc_b", 1, 2, 512, 32, 64, 64, dtype="f32", seed=502)]
    prepared = [(w, _case(w)) for w in cases]
    for w, args in prepared:  # two calls in a row, different sizes and dtypes
        got = _noalloc(w, *args)
        torch.cuda.synchronize()
        want = _regular(w, *args)
        torch.cuda.synchronize()
        tol = TOL[w.dtype]
        for name, g, r in zip(("Y", "R", "lse"), got, want):
            assert rel_err(host(g), host(r)) <= tol, (w.name, name)
    binding.dart_get_device_status()
