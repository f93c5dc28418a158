"""Failure detection without a GPU fault, one case per tensor-core entry point.

With the test hook on, one ring-fed kernel of the call issues none of its
copies (dart_sma_forward: the SMA kernel's operands; dart_chunk_scan: the
state passing's chunk slabs; dart_sma_backward: the row kernels' operands;
dart_chunk_scan_backward: the reverse passing's slabs), so the waits on them
can only run out: each is bounded (here 2 ms), after which the kernel drains
what it started, frees its tensor memory and records DART_ERR_TIMEOUT, which
dart_get_device_status reports. The context stays usable: the next call, with
the hook off and the default bound, matches the oracle."""
import contextlib

import pytest
import torch

import oracle
from helpers import TOL, dev, gpu_prefill, host, oracle_prefill, rel_err
from paper_2608_02032_gb300 import api, binding
from paper_2608_02032_gb300.workloads import Workload, memory_grad_input, prefill_inputs

pytestmark = pytest.mark.gpu

W = Workload("timeout_case", 1, 4, 1024, 64, 128, 128, seed=2201)
# eight heads and G = 1: the tensor-core scan (forward and backward) and SMA backward
W8 = Workload("timeout_case_h8", 1, 8, 512, 64, 128, 128, seed=2202)


@contextlib.contextmanager
def _withheld():
    """Copies withheld and waits bounded at 2 ms inside; the call must report a timeout."""
    binding.dart_get_device_status()  # clean status before the hook
    binding.dart_set_wait_limit_ns(2_000_000)
    binding.dart_test_withhold_copies(True)
    try:
        yield
        with pytest.raises(binding.DartError) as exc:
            binding.dart_get_device_status()
        assert exc.value.status == 5  # DART_ERR_TIMEOUT
    finally:
        binding.dart_test_withhold_copies(False)
        binding.dart_set_wait_limit_ns(0)
    binding.dart_get_device_status()  # the status word was cleared by the read above


def _bf16(inp, *names):
    return [dev(inp[k], "bf16") for k in names]


def test_sma_forward_withheld_operands_time_out_and_the_context_recovers():
    inp = prefill_inputs(W)
    X, Bm, Cm, Q, E, z = _bf16(inp, "X", "Bm", "Cm", "Q", "E", "z")
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    scan = api.chunk_scan(X, dt, A, Bm, Cm, W.chunk, W.eps)
    with _withheld():
        api.sma_forward(scan.M, scan.rM, Q, Cm, E, z, scan.Y_ssd, W.chunk, W.eps)
    got = gpu_prefill(inp, W)
    ref = oracle_prefill(inp, W)
    for k in ("Y_ssd", "Y", "lse"):
        assert rel_err(got[k], ref[k]) <= TOL["bf16"], k


def test_chunk_scan_withheld_slabs_time_out_and_the_context_recovers():
    inp = prefill_inputs(W8)
    X, Bm, Cm = _bf16(inp, "X", "Bm", "Cm")
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    with _withheld():
        api.chunk_scan(X, dt, A, Bm, Cm, W8.chunk, W8.eps, final_state=True)
    got = gpu_prefill(inp, W8)
    ref = oracle_prefill(inp, W8)
    for k in ("Y_ssd", "M", "final_state", "Y"):
        assert rel_err(got[k], ref[k]) <= TOL["bf16"], k


def _layer_case(w):
    inp = prefill_inputs(w, with_grad=True)
    X, Bm, Cm, Q, E, z, dY = _bf16(inp, "X", "Bm", "Cm", "Q", "E", "z", "dY")
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s, o = api.prefill_forward(X, dt, A, Bm, Cm, Q, E, z, w.chunk, w.eps)
    return inp, (X, dt, A, Bm, Cm, Q, E, z, dY), s, o


def test_sma_backward_withheld_operands_time_out_and_the_context_recovers():
    inp, (X, dt, A, Bm, Cm, Q, E, z, dY), s, o = _layer_case(W8)
    with _withheld():
        api.sma_backward(s.M, s.rM, Q, Cm, E, z, o.lse, dY, W8.chunk, W8.eps)
    gr = api.layer_backward(X, dt, A, Bm, Cm, Q, E, z, dY, s, o, W8.chunk, W8.eps)
    torch.cuda.synchronize()
    ref = oracle.backward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"], inp["Q"], inp["E"],
                          inp["z"], inp["dY"], W8.chunk, W8.eps)
    for n, g, r in zip(["dX", "ddt", "dA", "dB", "dC", "dQ", "dE", "dz"],
                       [gr.dX, gr.ddt, gr.dA, gr.dB, gr.dC, gr.dQ, gr.dE, gr.dz], ref):
        assert rel_err(host(g), r) <= TOL["bf16"], n


def test_chunk_scan_backward_withheld_slabs_time_out_and_the_context_recovers():
    inp = prefill_inputs(W8, with_grad=True)
    dMem = memory_grad_input(W8)
    X, Bm, Cm, dY = _bf16(inp, "X", "Bm", "Cm", "dY")
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    dM = dev(dMem, torch.float32)
    with _withheld():
        api.chunk_scan_backward(X, dt, A, Bm, Cm, dY, dM, W8.chunk, eps=W8.eps)
    got = api.chunk_scan_backward(X, dt, A, Bm, Cm, dY, dM, W8.chunk, eps=W8.eps)
    torch.cuda.synchronize()
    ref = oracle.ssd_backward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"], inp["dY"], dMem, W8.chunk)
    for n, g, r in zip(["dX", "ddt", "dA", "dB", "dC"], got, ref):
        assert rel_err(host(g), r) <= TOL["bf16"], n
