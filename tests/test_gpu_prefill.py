"""Parity of the CUDA prefill path (dart_chunk_scan + dart_sma_forward) with the oracle.

Element-by-element at sizes the oracle finishes in seconds; on sampled heads
and tokens at the full L = 16K workload. Tolerance: max|gpu - oracle| /
RMS(oracle) <= 1e-4 (fp32) or 2e-2 (bf16 inputs, fp32 accumulation), per
output tensor; lse = -inf rows (chunk 0) must match exactly.
"""
import numpy as np
import pytest
import torch

from helpers import TOL, dev, gpu_prefill, host, oracle_prefill, rel_err
from paper_2608_02032_gb300 import api, binding
from paper_2608_02032_gb300.workloads import WORKLOADS, Workload, prefill_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    binding.lib()  # fails loudly if libdart.so is missing


def _compare(got, ref, tol, keys=("Y_ssd", "M", "rM", "final_state", "R", "lse", "Y")):
    errs = {k: rel_err(got[k], ref[k]) for k in keys if k in got}
    bad = {k: v for k, v in errs.items() if not v <= tol}
    assert not bad, f"tolerance {tol} exceeded: {bad} (all: {errs})"
    return errs


def test_tiny_fp32_workload_matches_oracle(oracle_mod):
    w = WORKLOADS["tiny_fp32"]
    inp = prefill_inputs(w)
    _compare(gpu_prefill(inp, w), oracle_prefill(inp, w), TOL["f32"])


def test_prefill_b4_l2k_bf16_matches_oracle(oracle_mod):
    w = WORKLOADS["prefill_b4_l2k"]
    inp = prefill_inputs(w)
    _compare(gpu_prefill(inp, w), oracle_prefill(inp, w), TOL["bf16"])


SWEEP = [
    # (L, S, P, N, H, G, dtype)
    (64, 16, 32, 16, 2, 1, "f32"),
    (96, 32, 16, 64, 2, 1, "f32"),
    (192, 64, 64, 128, 2, 1, "f32"),
    (384, 128, 32, 64, 3, 1, "f32"),
    (512, 256, 64, 128, 2, 1, "f32"),
    (256, 256, 64, 128, 2, 1, "bf16"),   # M = 1: no token has history
    (512, 256, 64, 128, 2, 1, "bf16"),   # M = 2
    (768, 256, 64, 128, 4, 2, "bf16"),   # M = 3, two groups
    (320, 64, 32, 32, 2, 1, "bf16"),     # ragged last token tile inside chunks
    (1024, 128, 64, 128, 2, 1, "bf16"),
    # tensor-core SMA shapes (bf16, P 64, N 128, two heads per job, one CTA per 128-token tile);
    # at H = 4 the scan runs on the tensor cores too
    (512, 128, 64, 128, 4, 1, "bf16"),     # first tile of each chunk ... M = 4
    (256, 128, 64, 128, 4, 1, "bf16"),     # M = 2
    (128, 128, 64, 128, 4, 1, "bf16"),     # M = 1: only chunk-0 tiles
    (384, 128, 64, 128, 4, 1, "bf16"),     # L not a multiple of 256, M = 3
    (768, 128, 64, 128, 2, 1, "bf16"),     # M = 6
    (1024, 256, 64, 128, 8, 1, "bf16"),    # two head groups
    (768, 256, 64, 128, 8, 2, "bf16"),     # G = 2, four heads per group
    # tensor-core scan shapes (bf16, P 64, N 128, S in {64, 128, 256}, H / G a multiple of 4)
    (512, 128, 64, 128, 8, 1, "bf16"),
    (1024, 256, 64, 128, 4, 1, "bf16"),    # four heads: one chunk-state CTA per chunk
    (512, 256, 64, 128, 12, 1, "bf16"),    # twelve heads: three chunk-state CTAs, output heads per CTA divide 12
    (1024, 256, 64, 128, 16, 2, "bf16"),   # G = 2, eight heads per group
    (1024, 64, 64, 128, 8, 1, "bf16"),     # S = 64: one chunk per 128-row tile, rows 64 .. 127 idle
    (512, 64, 64, 128, 16, 2, "bf16"),     # S = 64, G = 2
    (1000, 64, 64, 128, 8, 1, "bf16"),     # S = 64 and ragged: 1024 padded tokens
    (100, 256, 64, 128, 8, 1, "bf16"),     # L < S: one partial chunk, no token has history
    (129, 128, 64, 128, 8, 1, "bf16"),     # one full chunk and a one-token chunk: only the last token reads a memory
    # ragged L (L % S != 0): the last memory holds the partial chunk
    (1000, 256, 64, 128, 8, 1, "bf16"),    # tensor-core scan and SMA on 1024 padded tokens
    (1000, 256, 64, 128, 4, 1, "bf16"),    # the same with four heads (one chunk-state CTA per chunk)
    (1000, 256, 64, 128, 2, 1, "bf16"),    # CUDA-core scan, tensor-core SMA
    (300, 64, 32, 32, 2, 1, "f32"),        # CUDA-core path, 5 memories, 44-token last chunk
    (97, 32, 16, 16, 3, 1, "f32"),         # a last chunk of one token (97 = 3 x 32 + 1)
    # tensor-core SMA with S < 128: a tile spans chunks, each token keeps its own history
    (1024, 64, 64, 128, 4, 1, "bf16"),     # S = 64: 16 memories
    (512, 32, 64, 128, 2, 1, "bf16"),      # S = 32: four chunks per tile
    (1000, 64, 64, 128, 2, 1, "bf16"),     # S = 64 and ragged (1024 padded tokens)
]


@pytest.mark.parametrize("L,S,P,N,H,G,dtype", SWEEP)
def test_size_sweep_matches_oracle(oracle_mod, L, S, P, N, H, G, dtype):
    w = Workload("sweep", 2, H, L, P, N, S, groups=G, dtype=dtype, seed=77 + L + S + P + N)
    inp = prefill_inputs(w)
    _compare(gpu_prefill(inp, w), oracle_prefill(inp, w), TOL[dtype])


@pytest.mark.parametrize("mem,out", [("bf16", "f32"), ("bf16", "bf16")])
def test_bf16_storage_of_memories_and_outputs(oracle_mod, mem, out):
    """bf16 memories (and outputs). Each stored memory is the oracle's memory
    rounded to bf16 (within an ulp, 2^-8 relative: the GPU rounds its fp32 sum).
    SMA then reads the stored memories, so R, lse and Y are checked against the
    oracle's SMA over its own memories rounded to bf16 (round to nearest even,
    on the CPU), at the bf16-input tolerance; bf16 outputs add their own
    rounding (2^-8 relative)."""
    w = Workload("bf16_store", 2, 2, 512, 64, 128, 128, seed=10)
    inp = prefill_inputs(w)
    X, Bm, Cm, Q, E, z = (dev(inp[k], "bf16") for k in ("X", "Bm", "Cm", "Q", "E", "z"))
    dtv, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    to = {"bf16": torch.bfloat16, "f32": torch.float32}[out]
    s, o = api.prefill_forward(X, dtv, A, Bm, Cm, Q, E, z, w.chunk, w.eps, want_R=True,
                               mem_dtype=torch.bfloat16, out_dtype=to)
    torch.cuda.synchronize()
    ref = oracle_prefill(inp, w)
    g, r = host(s.M), ref["M"]
    assert np.all(np.abs(g - r) <= 2.0 ** -8 * np.abs(r) + 1e-6 * np.abs(r).max())
    dH16 = torch.from_numpy(ref["M"]).to(torch.bfloat16).double().numpy()
    R16, lse16 = oracle_mod.sma(dH16, inp["Q"], inp["Cm"], inp["E"], w.chunk, w.eps)
    Y16 = oracle_mod.merge(ref["Y_ssd"], inp["z"], R16)
    assert rel_err(host(o.lse), lse16) <= TOL["bf16"]
    for k, got, want in (("Y_ssd", s.Y_ssd, ref["Y_ssd"]), ("R", o.R, R16), ("Y", o.Y, Y16)):
        g = host(got)
        if out == "f32":
            assert rel_err(g, want) <= TOL["bf16"], k
        else:
            rms = np.sqrt(np.mean(want ** 2))
            assert np.all(np.abs(g - want) <= 2.0 ** -8 * np.abs(want) + TOL["bf16"] * rms), k


def test_single_chunk_has_no_readout(oracle_mod):
    """S = L: every token is in chunk 0, so R = 0, lse = -inf and Y = Y_ssd exactly."""
    w = Workload("one_chunk", 1, 2, 256, 64, 128, 256, seed=5)
    got = gpu_prefill(prefill_inputs(w), w)
    assert np.all(got["R"] == 0) and np.all(np.isneginf(got["lse"]))
    assert np.array_equal(got["Y"], got["Y_ssd"])


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_zero_gate_reproduces_mamba2_bitwise(oracle_mod, dtype):
    """z = 0 (W_G = 0, Sec. 3): Y is bit-identical to the SSD output."""
    w = Workload("zero_gate", 1, 2, 512, 64, 128, 128, dtype=dtype, seed=6)
    inp = prefill_inputs(w)
    inp["z"] = torch.zeros_like(inp["z"])
    got = gpu_prefill(inp, w)
    assert np.array_equal(got["Y"], got["Y_ssd"])
    assert np.any(got["R"] != 0)


def test_rms_computed_inside_when_not_given(oracle_mod):
    w = Workload("rm_null", 1, 2, 512, 64, 128, 128, seed=8)
    inp = prefill_inputs(w)
    X, Bm, Cm, Q, E, z = (dev(inp[k], "bf16") for k in ("X", "Bm", "Cm", "Q", "E", "z"))
    dtv, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    s = api.chunk_scan(X, dtv, A, Bm, Cm, w.chunk, w.eps)
    o1 = api.sma_forward(s.M, s.rM, Q, Cm, E, z, s.Y_ssd, w.chunk, w.eps)
    o2 = api.sma_forward(s.M, None, Q, Cm, E, z, s.Y_ssd, w.chunk, w.eps)
    torch.cuda.synchronize()
    # the two r computations sum the squares in different orders; a 1-ulp change
    # of r moves the bf16 hi/lo split of r*M on the tensor-core path (~2e-5)
    assert rel_err(host(o1.Y), host(o2.Y)) <= 2e-4
    assert rel_err(host(o1.lse), host(o2.lse)) <= 1e-5  # -inf rows must match exactly


def test_outputs_stay_inside_their_buffers(oracle_mod):
    """Canary bands around every output of both calls stay untouched."""
    w = Workload("canary", 1, 2, 512, 64, 128, 128, seed=9)
    inp = prefill_inputs(w)
    Bsz, L, H, P, N, S = 1, 512, 2, 64, 128, 128
    M = L // S
    X, Bm, Cm, Q, E, z = (dev(inp[k], "bf16") for k in ("X", "Bm", "Cm", "Q", "E", "z"))
    dtv, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    pad = 4096

    def guarded(n, dtype):
        buf = torch.full((n + 2 * pad,), 7.0, dtype=dtype, device="cuda")
        return buf, buf[pad:pad + n]

    bufs = {}
    f32 = torch.float32
    for name, n, dtp in [("Y", Bsz * L * H * P, f32), ("M", Bsz * M * H * N * P, f32),
                         ("rM", Bsz * M * H * N, f32), ("fs", Bsz * H * N * P, f32),
                         ("Yo", Bsz * L * H * P, f32), ("R", Bsz * L * H * P, f32),
                         ("lse", Bsz * L * H, f32)]:
        bufs[name] = guarded(n, dtp)
    dims = binding.make_dims(Bsz, L, H, 1, P, N, S, binding.DART_BF16, eps=w.eps)
    ws = torch.empty(binding.dart_workspace_size(dims, binding.DART_OP_CHUNK_SCAN), dtype=torch.uint8,
                     device="cuda")
    binding.dart_chunk_scan(dims, X, dtv, A, Bm, Cm, bufs["Y"][1], bufs["M"][1], bufs["rM"][1],
                            bufs["fs"][1], ws)
    ws2 = torch.empty(binding.dart_workspace_size(dims, binding.DART_OP_SMA_FORWARD), dtype=torch.uint8,
                      device="cuda")
    binding.dart_sma_forward(dims, bufs["M"][1], bufs["rM"][1], Q, Cm, E, z, bufs["Y"][1],
                             bufs["Yo"][1], bufs["R"][1], bufs["lse"][1], ws2)
    torch.cuda.synchronize()
    for name, (buf, _) in bufs.items():
        assert torch.all(buf[:pad] == 7.0) and torch.all(buf[-pad:] == 7.0), name


def test_l16k_workload_sampled_heads_and_tokens(oracle_mod):
    """The full L = 16K, H = 32 workload in the benchmark's launch configuration,
    checked on three heads: Y_ssd and the memories of every token/chunk of those
    heads, R, lse and Y on 768 sampled tokens."""
    import oracle

    w = WORKLOADS["prefill_l16k"]
    inp = prefill_inputs(w)
    got = gpu_prefill(inp, w)
    heads = [0, 17, 31]
    rng = np.random.default_rng(0)
    toks = np.concatenate([rng.choice(np.arange(w.chunk, w.seqlen), 250, replace=False),
                           [0, w.chunk - 1, w.chunk, w.seqlen - 1, 3 * w.chunk + 5, w.seqlen - w.chunk]])
    for h in heads:
        sl = {k: inp[k][:, :, h:h + 1] for k in ("X", "dt", "z")}
        Yssd, Hl = oracle.ssd_recurrence(sl["X"], sl["dt"], inp["A"][h:h + 1], inp["Bm"], inp["Cm"])
        dH = oracle.chunk_memories(sl["X"], sl["dt"], inp["A"][h:h + 1], inp["Bm"], w.chunk)
        assert rel_err(got["Y_ssd"][:, :, h:h + 1], Yssd) <= TOL["bf16"]
        assert rel_err(got["M"][:, :, h:h + 1], dH) <= TOL["bf16"]
        assert rel_err(got["final_state"][:, h:h + 1], Hl) <= TOL["bf16"]
        tl = np.stack([np.zeros_like(toks), toks, np.zeros_like(toks)], 1)
        R, lse = oracle.sma(dH, inp["Q"], inp["Cm"], inp["E"], w.chunk, w.eps, tokens=tl)
        Y = oracle.merge(Yssd[0, toks, 0], sl["z"][0, toks, 0], R)
        assert rel_err(got["R"][0, toks, h], R) <= TOL["bf16"]
        assert rel_err(got["lse"][0, toks, h], lse) <= TOL["bf16"]
        assert rel_err(got["Y"][0, toks, h], Y) <= TOL["bf16"]


TILE_CASES = [
    # (B, H, G, L, S, mem, out): the tensor-core shapes of both calls
    (1, 8, 1, 1024, 256, "f32", "f32"),
    (2, 16, 2, 512, 128, "f32", "f32"),   # G = 2
    (1, 8, 1, 512, 64, "f32", "f32"),     # S = 64: a tile spans two chunks in the SMA
    (1, 8, 1, 512, 128, "bf16", "bf16"),  # bf16 memories: the tiles hold the stored (rounded) values
    (2, 4, 1, 512, 256, "f32", "f32"),    # four heads: one chunk-state CTA per chunk
    (1, 12, 1, 768, 128, "f32", "f32"),   # twelve heads
]


@pytest.mark.parametrize("Bsz,H,G,L,S,mem,out", TILE_CASES)
def test_sma_tiles_from_the_scan_match_the_regular_calls_bit_for_bit(oracle_mod, Bsz, H, G, L, S, mem, out):
    """dart_chunk_scan_with_tiles + dart_sma_forward_with_tiles: the chunk-state kernel
    writes the SMA's operand tiles; every output equals the regular pair's, bit for
    bit, and the oracle's within the bf16 tolerance."""
    w = Workload("tiles", Bsz, H, L, 64, 128, S, groups=G, seed=3300 + L + S + H)
    inp = prefill_inputs(w)
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16}
    X, Bm, Cm, Q, E, z = (dev(inp[k], "bf16") for k in ("X", "Bm", "Cm", "Q", "E", "z"))
    dtv, A = dev(inp["dt"], torch.float32), dev(inp["A"], torch.float32)
    dims = binding.make_dims(Bsz, L, H, G, 64, 128, S, binding.DART_BF16, binding.DART_DTYPE[tdt[mem]],
                             binding.DART_DTYPE[tdt[out]], eps=w.eps)
    nb = binding.dart_sma_tiles_size(dims)
    assert nb > 0
    Mc = L // S
    outs = []
    for fused in (False, True):
        Yssd = torch.empty(Bsz, L, H, 64, dtype=tdt[out], device="cuda")
        M = torch.empty(Bsz, Mc, H, 128, 64, dtype=tdt[mem], device="cuda")
        rM = torch.empty(Bsz, Mc, H, 128, dtype=torch.float32, device="cuda")
        Y, R = torch.empty_like(Yssd), torch.empty_like(Yssd)
        lse = torch.empty(Bsz, L, H, dtype=torch.float32, device="cuda")
        ws = torch.empty(binding.dart_workspace_size(dims, binding.DART_OP_CHUNK_SCAN), dtype=torch.uint8,
                         device="cuda")
        if fused:
            tiles = torch.full((nb,), 0xFF, dtype=torch.uint8, device="cuda")  # NaN-poisoned
            binding.dart_chunk_scan_with_tiles(dims, X, dtv, A, Bm, Cm, Yssd, M, rM, None, tiles, ws)
            binding.dart_sma_forward_with_tiles(dims, tiles, Q, Cm, E, z, Yssd, Y, R, lse)
        else:
            binding.dart_chunk_scan(dims, X, dtv, A, Bm, Cm, Yssd, M, rM, None, ws)
            wss = torch.empty(binding.dart_workspace_size(dims, binding.DART_OP_SMA_FORWARD), dtype=torch.uint8,
                              device="cuda")
            binding.dart_sma_forward(dims, M, rM, Q, Cm, E, z, Yssd, Y, R, lse, wss)
        torch.cuda.synchronize()
        outs.append((Yssd, M, rM, Y, R, lse))
    for name, a, b in zip(("Y_ssd", "M", "rM", "Y", "R", "lse"), outs[0], outs[1]):
        assert torch.equal(a, b), name
    if mem == "f32" and out == "f32":
        ref = oracle_prefill(inp, w)
        for name, got in (("Y", outs[1][3]), ("R", outs[1][4]), ("lse", outs[1][5])):
            assert rel_err(host(got), ref[name]) <= TOL["bf16"], name


def test_sma_tiles_refuse_other_shapes():
    dims = lambda **kw: binding.make_dims(kw.get("B", 1), kw.get("L", 512), kw.get("H", 8), kw.get("G", 1),
                                         kw.get("P", 64), kw.get("N", 128), kw.get("S", 128),
                                         kw.get("dt", binding.DART_BF16), eps=1e-6)
    assert binding.dart_sma_tiles_size(dims()) > 0
    assert binding.dart_sma_tiles_size(dims(H=4)) > 0
    for bad in (dict(L=500), dict(H=2), dict(H=6), dict(P=32), dict(dt=binding.DART_F32), dict(S=32)):
        assert binding.dart_sma_tiles_size(dims(**bad)) == 0, bad
    with pytest.raises(binding.DartError):
        t = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
        binding.dart_sma_forward_with_tiles(dims(H=6), t, t, t, t, t, t, t)
