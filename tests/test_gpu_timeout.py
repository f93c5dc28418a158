"""Failure detection without a GPU fault. With the test hook on, the
tensor-core SMA kernel issues no operand copies, so its waits can only run
out: each is bounded (here 2 ms), after which the kernel drains what it
started, frees its tensor memory and reports DART_ERR_TIMEOUT through
dart_get_device_status. The context stays usable and the next call is correct."""
import pytest
import torch

from helpers import TOL, dev, gpu_prefill, oracle_prefill, rel_err
from paper_2608_02032_gb300 import api, binding
from paper_2608_02032_gb300.workloads import Workload, prefill_inputs

pytestmark = pytest.mark.gpu

W = Workload("timeout_case", 1, 4, 1024, 64, 128, 128, seed=2201)


def test_withheld_operands_time_out_and_the_context_recovers():
    inp = prefill_inputs(W)
    X, Bm, Cm, Q, E, z = (dev(inp[k], "bf16") for k in ("X", "Bm", "Cm", "Q", "E", "z"))
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    scan = api.chunk_scan(X, dt, A, Bm, Cm, W.chunk, W.eps)
    binding.dart_get_device_status()  # clean status before the hook
    binding.dart_set_wait_limit_ns(2_000_000)
    binding.dart_test_withhold_copies(True)
    try:
        api.sma_forward(scan.M, scan.rM, Q, Cm, E, z, scan.Y_ssd, W.chunk, W.eps)
        with pytest.raises(binding.DartError) as exc:
            binding.dart_get_device_status()
        assert exc.value.status == 5  # DART_ERR_TIMEOUT
    finally:
        binding.dart_test_withhold_copies(False)
        binding.dart_set_wait_limit_ns(0)
    binding.dart_get_device_status()  # the status word was cleared by the read above
    got = gpu_prefill(inp, W)
    ref = oracle_prefill(inp, W)
    for k in ("Y_ssd", "Y", "lse"):
        assert rel_err(got[k], ref[k]) <= TOL["bf16"], k
