"""Parity of the backward entry points (dart_chunk_scan_backward,
dart_sma_backward) against the fp64 oracle's hand-derived backward, which the
CPU tests pin by finite differences. Inputs come from the seeded generators;
expected values from the oracle on the same (bf16-rounded) inputs."""
import pytest
import torch

import oracle
from helpers import TOL, dev, host, rel_err
from paper_2608_02032_gb300 import api, binding
from paper_2608_02032_gb300.workloads import WORKLOADS, Workload, memory_grad_input, prefill_inputs

pytestmark = pytest.mark.gpu

CASES = [
    WORKLOADS["tiny_fp32"],
    Workload("bwd_f32_s32_g2", 1, 4, 256, 32, 32, 32, groups=2, dtype="f32", seed=2101),
    Workload("bwd_f32_s16", 2, 2, 128, 16, 16, 16, dtype="f32", seed=2102),
    Workload("bwd_bf16_s128", 1, 4, 512, 64, 128, 128, seed=2103),
    Workload("bwd_bf16_s256", 2, 4, 1024, 64, 128, 256, seed=2104),
    # three head pairs and seven memories: many jobs per tile through the two-stage rings
    Workload("bwd_bf16_h6_s128", 1, 6, 1024, 64, 128, 128, seed=2106),
    # eight heads: the tensor-core scan backward (head groups of 8)
    Workload("bwd_bf16_h8_s256", 1, 8, 1024, 64, 128, 256, seed=2107),
    Workload("bwd_bf16_h8_s128", 2, 8, 512, 64, 128, 128, seed=2108),
    # G = 2: the tensor-core backward once per group of 8 heads (scan and SMA)
    Workload("bwd_bf16_h16_g2_s128", 1, 16, 512, 64, 128, 128, groups=2, seed=2109),
    # G = 2 with 4 heads per group: the SMA backward per group on the tensor cores, the scan on FFMA
    Workload("bwd_bf16_h8_g2_s256", 2, 8, 1024, 64, 128, 256, groups=2, seed=2110),
]


def _tol(w):
    return TOL[w.dtype]


@pytest.mark.parametrize("w", CASES, ids=lambda w: w.name)
def test_scan_backward_matches_oracle(w):
    inp = prefill_inputs(w, with_grad=True)
    dMem = memory_grad_input(w)
    ref = oracle.ssd_backward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"], inp["dY"],
                              dMem, w.chunk)
    X, Bm, Cm, dY = (dev(inp[k], w.dtype) for k in ("X", "Bm", "Cm", "dY"))
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    got = api.chunk_scan_backward(X, dt, A, Bm, Cm, dY, dev(dMem, torch.float32), w.chunk, eps=w.eps)
    torch.cuda.synchronize()
    errs = {name: rel_err(host(g), r) for name, g, r in zip(["dX", "ddt", "dA", "dB", "dC"], got, ref)}
    print(w.name, {k: f"{v:.2e}" for k, v in errs.items()})
    for name, err in errs.items():
        assert err <= _tol(w), f"{name}: {err:.3e}"


def test_scan_backward_accumulates_into_dC_and_takes_no_memory_gradient():
    w = WORKLOADS["tiny_fp32"]
    inp = prefill_inputs(w, with_grad=True)
    ref = oracle.ssd_backward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"], inp["dY"],
                              None, w.chunk)
    X, Bm, Cm, dY = (dev(inp[k], "f32") for k in ("X", "Bm", "Cm", "dY"))
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    base = torch.full(Cm.shape, 0.25, dtype=torch.float32, device="cuda")
    got = api.chunk_scan_backward(X, dt, A, Bm, Cm, dY, None, w.chunk, dC=base.clone())
    torch.cuda.synchronize()
    assert rel_err(host(got[4]) - 0.25, ref[4]) <= TOL["f32"]
    assert rel_err(host(got[0]), ref[0]) <= TOL["f32"]


@pytest.mark.parametrize("w", CASES, ids=lambda w: w.name)
def test_sma_backward_matches_oracle(w):
    """Memories and lse from the oracle, so the check covers the backward alone."""
    inp = prefill_inputs(w, with_grad=True)
    D = oracle.chunk_memories(inp["X"], inp["dt"], inp["A"], inp["Bm"], w.chunk)
    _, lse = oracle.sma(D, inp["Q"], inp["Cm"], inp["E"], w.chunk, w.eps)
    ref = oracle.sma_backward(D, inp["Q"], inp["Cm"], inp["E"], inp["z"], inp["dY"], w.chunk, w.eps)
    Q, Cm, E, z, dY = (dev(inp[k], w.dtype) for k in ("Q", "Cm", "E", "z", "dY"))
    Mem = dev(torch.from_numpy(D).float(), torch.float32)
    got = api.sma_backward(Mem, None, Q, Cm, E, z, dev(torch.from_numpy(lse).float(), torch.float32),
                           dY, w.chunk, w.eps)
    torch.cuda.synchronize()
    errs = {name: rel_err(host(g), r) for name, g, r in zip(["dM", "dQ", "dC", "dE", "dz"], got, ref)}
    print(w.name, {k: f"{v:.2e}" for k, v in errs.items()})
    for name, err in errs.items():
        assert err <= _tol(w), f"{name}: {err:.3e}"


@pytest.mark.parametrize("w", [CASES[0], CASES[3], CASES[6], CASES[8]], ids=lambda w: w.name)
def test_layer_backward_matches_oracle(w):
    """Forward through the library, then the layer backward: SMA backward's dM and
    dC feed the scan backward."""
    inp = prefill_inputs(w, with_grad=True)
    ref = oracle.backward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"], inp["Q"], inp["E"],
                          inp["z"], inp["dY"], w.chunk, w.eps)
    X, Bm, Cm, Q, E, z, dY = (dev(inp[k], w.dtype) for k in ("X", "Bm", "Cm", "Q", "E", "z", "dY"))
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s, o = api.prefill_forward(X, dt, A, Bm, Cm, Q, E, z, w.chunk, w.eps)
    gr = api.layer_backward(X, dt, A, Bm, Cm, Q, E, z, dY, s, o, w.chunk, w.eps)
    torch.cuda.synchronize()
    got = [gr.dX, gr.ddt, gr.dA, gr.dB, gr.dC, gr.dQ, gr.dE, gr.dz]
    errs = {n: rel_err(host(g), r) for n, g, r in zip(["dX", "ddt", "dA", "dB", "dC", "dQ", "dE", "dz"], got, ref)}
    print(w.name, {k: f"{v:.2e}" for k, v in errs.items()})
    for name, err in errs.items():
        assert err <= _tol(w), f"{name}: {err:.3e}"


@pytest.mark.parametrize("w", [CASES[3], CASES[6], CASES[7], CASES[8]], ids=lambda w: w.name)
def test_layer_backward_with_saved_logits(w):
    """The training pair that keeps the forward's logits: the backward takes its
    softmax weights from them instead of recomputing the logit chains. Against the
    oracle, and against the recomputing backward (the same weights; the gradients
    differ only by the order of their fp32 atomic additions)."""
    inp = prefill_inputs(w, with_grad=True)
    ref = oracle.backward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"], inp["Q"], inp["E"],
                          inp["z"], inp["dY"], w.chunk, w.eps)
    X, Bm, Cm, Q, E, z, dY = (dev(inp[k], w.dtype) for k in ("X", "Bm", "Cm", "Q", "E", "z", "dY"))
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s, o = api.prefill_forward(X, dt, A, Bm, Cm, Q, E, z, w.chunk, w.eps, save_logits=True)
    assert o.logits is not None
    gr = api.layer_backward(X, dt, A, Bm, Cm, Q, E, z, dY, s, o, w.chunk, w.eps)
    s2, o2 = api.prefill_forward(X, dt, A, Bm, Cm, Q, E, z, w.chunk, w.eps)
    gr2 = api.layer_backward(X, dt, A, Bm, Cm, Q, E, z, dY, s2, o2, w.chunk, w.eps)
    torch.cuda.synchronize()
    assert torch.equal(o.Y, o2.Y) and torch.equal(o.lse, o2.lse)  # the forward itself is unchanged
    names = ["dX", "ddt", "dA", "dB", "dC", "dQ", "dE", "dz"]
    got = [gr.dX, gr.ddt, gr.dA, gr.dB, gr.dC, gr.dQ, gr.dE, gr.dz]
    rec = [gr2.dX, gr2.ddt, gr2.dA, gr2.dB, gr2.dC, gr2.dQ, gr2.dE, gr2.dz]
    # dA: one sum per head over every token, atomics in run-dependent order
    tol_same = {"dA": 2e-4}
    for n, g, r, g2 in zip(names, got, ref, rec):
        assert rel_err(host(g), r) <= _tol(w), n
        assert rel_err(host(g), host(g2)) <= tol_same.get(n, 1e-5), n
    assert rel_err(host(gr.dM), host(gr2.dM)) <= 1e-5


def test_grouped_backward_runs_per_group_on_the_tensor_cores():
    """At G = 2 with 8 heads per group, each backward runs the G = 1 tensor-core
    kernels once per group on copied slices: per group at least 7 (scan) and 7
    (SMA) copies in and 4 and 5 copies out besides the backward's own kernels, far
    more launches than the CUDA-core backward makes. Parity is checked above."""
    w = CASES[8]
    inp = prefill_inputs(w, with_grad=True)
    X, Bm, Cm, Q, E, z, dY = (dev(inp[k], w.dtype) for k in ("X", "Bm", "Cm", "Q", "E", "z", "dY"))
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s, o = api.prefill_forward(X, dt, A, Bm, Cm, Q, E, z, w.chunk, w.eps)
    torch.cuda.synchronize()
    n0 = binding.dart_launch_count()
    gM, gQ, gC, gE, gz = api.sma_backward(s.M, s.rM, Q, Cm, E, z, o.lse, dY, w.chunk, w.eps)
    n1 = binding.dart_launch_count()
    api.chunk_scan_backward(X, dt, A, Bm, Cm, dY, gM, w.chunk, dC=gC, eps=w.eps)
    n2 = binding.dart_launch_count()
    torch.cuda.synchronize()
    assert n1 - n0 >= 2 * (7 + 5) and n2 - n1 >= 2 * (7 + 4), (n1 - n0, n2 - n1)


def test_backward_single_chunk_has_no_sma_gradient():
    """S = L: no token has history, so the SMA gradients are exactly zero."""
    w = Workload("bwd_one_chunk", 1, 2, 128, 32, 16, 128, dtype="f32", seed=2105)
    inp = prefill_inputs(w, with_grad=True)
    X, Bm, Cm, Q, E, z, dY = (dev(inp[k], "f32") for k in ("X", "Bm", "Cm", "Q", "E", "z", "dY"))
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s, o = api.prefill_forward(X, dt, A, Bm, Cm, Q, E, z, w.chunk, w.eps)
    dM, dQ, dC, dE, dz = api.sma_backward(s.M, s.rM, Q, Cm, E, z, o.lse, dY, w.chunk, w.eps)
    torch.cuda.synchronize()
    for t in (dM, dQ, dC, dE, dz):
        assert torch.count_nonzero(t).item() == 0


@pytest.mark.parametrize("name", ["train_b8_l4k_s256", "train_b8_l4k_s128"])
def test_training_step_full_size_on_one_batch(name):
    """The training workload at full size (B8 H24 L4096), forward (keeping the SMA
    logits) and layer backward through the library exactly as the bench's training
    step runs them; the oracle
    computes batch 0 (batches are independent) and every per-batch gradient is
    compared there. dA sums over the batch, so it is checked on the small cases."""
    w = WORKLOADS[name]
    inp = prefill_inputs(w, with_grad=True)
    X, Bm, Cm, Q, E, z, dY = (dev(inp[k], w.dtype) for k in ("X", "Bm", "Cm", "Q", "E", "z", "dY"))
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s, o = api.prefill_forward(X, dt, A, Bm, Cm, Q, E, z, w.chunk, w.eps, save_logits=True)
    gr = api.layer_backward(X, dt, A, Bm, Cm, Q, E, z, dY, s, o, w.chunk, w.eps)
    torch.cuda.synchronize()
    one = {k: inp[k][:1] for k in ("X", "dt", "Bm", "Cm", "Q", "E", "z", "dY")}
    ref = oracle.backward(one["X"], one["dt"], inp["A"], one["Bm"], one["Cm"], one["Q"], one["E"],
                          one["z"], one["dY"], w.chunk, w.eps)
    got = [gr.dX, gr.ddt, None, gr.dB, gr.dC, gr.dQ, gr.dE, gr.dz]
    names = ["dX", "ddt", "dA", "dB", "dC", "dQ", "dE", "dz"]
    errs = {n: rel_err(host(g[:1]), r) for n, g, r in zip(names, got, ref) if g is not None}
    print(name, {k: f"{v:.2e}" for k, v in errs.items()})
    for n, err in errs.items():
        assert err <= _tol(w), f"{n}: {err:.3e}"


@pytest.mark.parametrize("w", [CASES[0], CASES[6]], ids=lambda w: w.name)
def test_independent_sma_read_vector(w):
    """The variant with an independent SMA read vector (the ablation of Sec. 5 that
    replaces the shared C_t of V_{t,c} = C_t Delta H_[c] by its own projection): the
    scan reads C, state-memory attention reads C_sma. Forward outputs, and the two
    read-vector gradients kept apart (dC from the scan backward with no SMA part
    passed in, dC_sma from the SMA backward), against the oracle run on the same split."""
    inp = prefill_inputs(w, with_grad=True)
    g = torch.Generator().manual_seed(w.seed + 77)
    C_sma = (torch.randn(inp["Cm"].shape, generator=g, dtype=torch.float64) / w.dstate ** 0.5)
    if w.dtype == "bf16":
        C_sma = C_sma.to(torch.bfloat16).double()
    # oracle: the scan with C, SMA and its backward with C_sma
    Yssd, _ = oracle.ssd_recurrence(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"])
    dH = oracle.chunk_memories(inp["X"], inp["dt"], inp["A"], inp["Bm"], w.chunk)
    R, lse = oracle.sma(dH, inp["Q"], C_sma, inp["E"], w.chunk, w.eps)
    Y = oracle.merge(Yssd, inp["z"], R)
    dMem, dQ, dCs, dE, dz = oracle.sma_backward(dH, inp["Q"], C_sma, inp["E"], inp["z"], inp["dY"], w.chunk, w.eps)
    dX, ddt, dA, dB, dC = oracle.ssd_backward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"], inp["dY"],
                                              dMem, w.chunk)
    # GPU
    X, Bm, Cm, Q, E, z, dY = (dev(inp[k], w.dtype) for k in ("X", "Bm", "Cm", "Q", "E", "z", "dY"))
    Cs = dev(C_sma, w.dtype)
    dt, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s = api.chunk_scan(X, dt, A, Bm, Cm, w.chunk, w.eps)
    o = api.sma_forward(s.M, s.rM, Q, Cs, E, z, s.Y_ssd, w.chunk, w.eps)
    gM, gQ, gCs, gE, gz = api.sma_backward(s.M, s.rM, Q, Cs, E, z, o.lse, dY, w.chunk, w.eps)
    gX, gdt, gA, gB, gC = api.chunk_scan_backward(X, dt, A, Bm, Cm, dY, gM, w.chunk, eps=w.eps)
    torch.cuda.synchronize()
    tol = _tol(w)
    for n, got, ref in (("Y", o.Y, Y), ("lse", o.lse, lse), ("dX", gX, dX), ("ddt", gdt, ddt), ("dA", gA, dA),
                        ("dB", gB, dB), ("dC", gC, dC), ("dC_sma", gCs, dCs), ("dQ", gQ, dQ), ("dE", gE, dE),
                        ("dz", gz, dz)):
        assert rel_err(host(got), ref) <= tol, n
