"""dart_prefill_host: the prefill from host buffers to a host buffer, with the
copies overlapped with the kernels head group by head group, against the
device entry points on the same inputs (which the other tests check against
the oracle). Per head the same kernels run, so the results agree to fp32
rounding (in practice bit for bit)."""
import pytest
import torch

from helpers import host, rel_err
from paper_2608_02032_gb300 import api
from paper_2608_02032_gb300.workloads import Workload, prefill_inputs

pytestmark = pytest.mark.gpu


def _inputs(w):
    inp = prefill_inputs(w)
    dt_ = {"X": torch.bfloat16, "Bm": torch.bfloat16, "Cm": torch.bfloat16, "Q": torch.bfloat16,
           "E": torch.bfloat16, "z": torch.bfloat16, "dt": torch.float32, "A": torch.float32}
    return {k: inp[k].to(t).contiguous() for k, t in dt_.items()}


@pytest.mark.parametrize("w", [
    Workload("host_h32", 1, 32, 2048, 64, 128, 256, seed=51),              # eight groups of 4 heads
    Workload("host_b2_h16", 2, 16, 1024, 64, 128, 128, seed=52),           # four groups, S = 128
    Workload("host_h24", 1, 24, 1024, 64, 128, 64, seed=57),               # six groups, S = 64
    Workload("host_h8", 1, 8, 512, 64, 128, 256, seed=58),                 # two groups: fewer than the streams
    Workload("host_h6", 1, 6, 512, 64, 128, 128, seed=53),                 # one group (H % 4 != 0)
    Workload("host_g2", 1, 16, 512, 64, 128, 128, groups=2, seed=54),      # one group (G = 2)
    Workload("host_small", 1, 16, 512, 32, 64, 64, seed=55),               # the CUDA-core kernels
], ids=lambda w: w.name)
def test_prefill_from_host_matches_the_device_path(w):
    inp = _inputs(w)
    d = {k: t.cuda() for k, t in inp.items()}
    _, o = api.prefill_forward(d["X"], d["dt"], d["A"], d["Bm"], d["Cm"], d["Q"], d["E"], d["z"], w.chunk,
                               w.eps)
    torch.cuda.synchronize()
    ref = host(o.Y)
    h = {k: t.pin_memory() for k, t in inp.items()}
    ws = None
    for _ in range(2):  # the workspace is reused by the second call
        Y, ws = api.prefill_from_host(h["X"], h["dt"], h["A"], h["Bm"], h["Cm"], h["Q"], h["E"], h["z"],
                                      w.chunk, w.eps, workspace=ws)
        torch.cuda.current_stream().synchronize()
        assert not Y.is_cuda and Y.is_pinned()
        err = rel_err(Y.numpy(), ref)
        assert err <= 1e-6, f"{w.name}: {err:.2e}"


def test_prefill_from_host_orders_after_earlier_work_on_the_stream():
    """Inputs written on the device by earlier work on the same stream and copied back
    to the host buffers just before the call are the ones the call reads."""
    w = Workload("host_order", 1, 16, 1024, 64, 128, 256, seed=56)
    inp = _inputs(w)
    h = {k: t.pin_memory() for k, t in inp.items()}
    Y1, ws = api.prefill_from_host(h["X"], h["dt"], h["A"], h["Bm"], h["Cm"], h["Q"], h["E"], h["z"],
                                   w.chunk, w.eps)
    torch.cuda.current_stream().synchronize()
    first = Y1.clone()
    # scale X on the device and bring it back into the same pinned buffer, on the stream
    Xd = inp["X"].cuda() * 2
    h["X"].copy_(Xd, non_blocking=True)
    Y2, _ = api.prefill_from_host(h["X"], h["dt"], h["A"], h["Bm"], h["Cm"], h["Q"], h["E"], h["z"],
                                  w.chunk, w.eps, workspace=ws)
    torch.cuda.current_stream().synchronize()
    d = {k: t.cuda() for k, t in inp.items()}
    _, o = api.prefill_forward(Xd, d["dt"], d["A"], d["Bm"], d["Cm"], d["Q"], d["E"], d["z"], w.chunk, w.eps)
    torch.cuda.synchronize()
    assert rel_err(Y2.numpy(), host(o.Y)) <= 1e-6
    assert not torch.equal(first, Y2)
