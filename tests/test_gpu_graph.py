"""The hot path inside a CUDA graph.

The library launches on the caller's stream, takes its scratch from the
caller's workspace and never synchronises or allocates, so a whole prefill
step (dart_chunk_scan + dart_sma_forward) and a whole training step (the
forward and both backwards) can be captured once and replayed. Each replay
is compared with the eager calls on the same buffers: the forward bit for
bit (its kernels are deterministic), the backward within fp32 rounding (its
row and column sums add partial results with atomics, in varying order).
A second set of inputs copied into the captured buffers checks that the
replay reads the buffers rather than values frozen at capture.
"""
import pytest
import torch

from helpers import host, rel_err
from paper_2608_02032_gb300 import binding as Bd
from paper_2608_02032_gb300.workloads import Workload, prefill_inputs

pytestmark = pytest.mark.gpu


class _Step:
    """Buffers of one DART layer step on the device and its launches through the C ABI."""

    def __init__(self, w, train: bool):
        self.w, self.train = w, train
        Bsz, L, H, G, P, N = w.batch, w.seqlen, w.heads, w.groups, w.headdim, w.dstate
        M = w.nchunks
        f32 = dict(dtype=torch.float32, device="cuda")
        bf = dict(dtype=torch.bfloat16, device="cuda")
        self.inp = {"X": torch.empty(Bsz, L, H, P, **bf), "Bm": torch.empty(Bsz, L, G, N, **bf),
                    "Cm": torch.empty(Bsz, L, G, N, **bf), "Q": torch.empty(Bsz, L, G, N, **bf),
                    "E": torch.empty(Bsz, L, G, P, **bf), "z": torch.empty(Bsz, L, H, **bf),
                    "dY": torch.empty(Bsz, L, H, P, **bf), "dt": torch.empty(Bsz, L, H, **f32),
                    "A": torch.empty(H, **f32)}
        self.out = {"Yssd": torch.empty(Bsz, L, H, P, **f32), "Y": torch.empty(Bsz, L, H, P, **f32),
                    "M": torch.empty(Bsz, M, H, N, P, **f32), "rM": torch.empty(Bsz, M, H, N, **f32),
                    "lse": torch.empty(Bsz, L, H, **f32)}
        if train:
            self.out.update({"dM": torch.empty(Bsz, M, H, N, P, **f32),
                             "dQ": torch.empty(Bsz, L, G, N, **f32), "dC": torch.empty(Bsz, L, G, N, **f32),
                             "dE": torch.empty(Bsz, L, G, P, **f32), "dz": torch.empty(Bsz, L, H, **f32),
                             "dX": torch.empty(Bsz, L, H, P, **f32), "ddt": torch.empty(Bsz, L, H, **f32),
                             "dA": torch.empty(H, **f32), "dB": torch.empty(Bsz, L, G, N, **f32)})
        self.dims = Bd.make_dims(Bsz, L, H, G, P, N, w.chunk, Bd.DART_BF16, mem_dtype=Bd.DART_F32,
                                 out_dtype=Bd.DART_F32, eps=w.eps)

        def ws(op):
            return torch.empty(max(Bd.dart_workspace_size(self.dims, op), 256), dtype=torch.uint8,
                               device="cuda")
        self.ws = {"scan": ws(Bd.DART_OP_CHUNK_SCAN), "sma": ws(Bd.DART_OP_SMA_FORWARD)}
        if train:
            self.ws.update({"sbwd": ws(Bd.DART_OP_SMA_BACKWARD), "cbwd": ws(Bd.DART_OP_SCAN_BACKWARD)})

    def load(self, seed: int):
        src = prefill_inputs(self.w.with_(seed=seed), with_grad=True)
        for k, t in self.inp.items():
            t.copy_(src[k].to(t.dtype))

    def run(self, stream):
        i, o, d, ws = self.inp, self.out, self.dims, self.ws
        Bd.dart_chunk_scan(d, i["X"], i["dt"], i["A"], i["Bm"], i["Cm"], o["Yssd"], o["M"], o["rM"], None,
                           ws["scan"], stream)
        Bd.dart_sma_forward(d, o["M"], o["rM"], i["Q"], i["Cm"], i["E"], i["z"], o["Yssd"], o["Y"], None,
                            o["lse"], ws["sma"], stream)
        if self.train:
            Bd.dart_sma_backward(d, o["M"], o["rM"], i["Q"], i["Cm"], i["E"], i["z"], o["lse"], i["dY"],
                                 o["dM"], o["dQ"], o["dC"], o["dE"], o["dz"], ws["sbwd"], stream)
            Bd.dart_chunk_scan_backward(d, i["X"], i["dt"], i["A"], i["Bm"], i["Cm"], i["dY"], o["dM"],
                                        o["dX"], o["ddt"], o["dA"], o["dB"], o["dC"], ws["cbwd"], stream)

    def snapshot(self):
        return {k: t.clone() for k, t in self.out.items()}

    def clear(self):
        for t in self.out.values():
            t.fill_(float("nan"))


def _eager(step, seed):
    step.load(seed)
    step.run(torch.cuda.current_stream())
    torch.cuda.synchronize()
    return step.snapshot()


def _capture(step):
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):  # first launches (function attributes) outside the capture
        step.run(side)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step.run(torch.cuda.current_stream())
    torch.cuda.synchronize()
    return g


def _replay(step, g, seed):
    step.load(seed)
    step.clear()
    g.replay()
    torch.cuda.synchronize()
    return step.snapshot()


def test_prefill_step_replays_bitwise_from_a_cuda_graph():
    w = Workload("graph_fwd", 2, 16, 1024, 64, 128, 256, seed=41)  # tensor-core path, 4 chunks
    step = _Step(w, train=False)
    ref = {s: _eager(step, s) for s in (41, 42)}
    g = _capture(step)
    for s in (42, 41):  # the second set first: the replay must not reuse captured values
        got = _replay(step, g, s)
        for k in got:
            assert torch.equal(got[k], ref[s][k]), f"{k} differs after replay (seed {s})"


def test_training_step_replays_from_a_cuda_graph():
    w = Workload("graph_train", 2, 8, 1024, 64, 128, 256, seed=43)
    step = _Step(w, train=True)
    ref = {s: _eager(step, s) for s in (43, 44)}
    g = _capture(step)
    # dA is one sum per head over every token, added by atomics in an order that
    # varies from run to run (eager or replayed); its spread reaches ~2e-5 of its RMS
    tol = {"dA": 2e-4}
    for s in (44, 43):
        got = _replay(step, g, s)
        for k in got:
            assert not torch.isnan(got[k]).any(), f"{k}: not written by the replay (seed {s})"
            err = rel_err(host(got[k]), host(ref[s][k]))
            assert err <= tol.get(k, 1e-5), f"{k}: {err:.2e} after replay (seed {s})"
