"""The product path has no CPU fallback: without the compiled library, or given
host tensors where the library wants device ones, the binding raises before
anything is computed."""
import pytest
import torch

from paper_2608_02032_gb300 import api, binding
from paper_2608_02032_gb300.workloads import WORKLOADS, prefill_inputs


def test_missing_library_raises(monkeypatch):
    monkeypatch.setattr(binding, "LIB_PATH", "/nonexistent/libdart.so")
    monkeypatch.setattr(binding, "_lib", None)
    with pytest.raises(RuntimeError, match="not built"):
        binding.lib()


@pytest.fixture(scope="module")
def built():
    from paper_2608_02032_gb300 import build

    build.build()  # the library exists: the refusal below is the binding's, not a missing file


def test_host_tensors_are_refused_by_the_device_entry_points(built):
    inp = prefill_inputs(WORKLOADS["tiny_fp32"])
    w = WORKLOADS["tiny_fp32"]
    with pytest.raises(ValueError, match="CUDA tensor"):
        api.chunk_scan(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"], w.chunk, w.eps)
    with pytest.raises(ValueError, match="CUDA tensor"):
        binding._ptr(torch.zeros(4), "X")


def test_host_buffer_entry_wants_contiguous_host_tensors():
    with pytest.raises(ValueError, match="contiguous"):
        binding._host_ptr(torch.zeros(4, 4).t(), "X")
    with pytest.raises(TypeError):
        binding._host_ptr([0.0], "X")
