"""Parity of the CUDA decode step (dart_decode_step) with the oracle."""
import numpy as np
import pytest
import torch

from helpers import TOL, dev, host, rel_err
from paper_2608_02032_gb300 import api, binding
from paper_2608_02032_gb300.workloads import (WORKLOADS, Workload, decode_cache_slab, decode_state,
                                              decode_state_slab, decode_token_inputs, prefill_inputs)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    binding.lib()


def _token_dev(tok, dtype):
    out = {k: dev(tok[k], dtype) for k in ("x", "b", "c", "q", "e", "z")}
    out["dt"] = dev(tok["dt"], torch.float32)
    out["A"] = dev(tok["A"], torch.float32)
    return out


def test_decode_b64_workload_sampled_rows(oracle_mod):
    """The full decode workload (64 x 32 heads, 64 cached memories = 2 GiB bf16,
    pos = 16384, a chunk start) in the benchmark's launch configuration; y, lse
    and the updated state/partial are checked on three batch rows (all heads)."""
    w = WORKLOADS["decode_b64"]
    tok = decode_token_inputs(w)
    m_cap = w.mem + 1
    cache = torch.empty(w.batch, m_cap, w.heads, w.dstate, w.headdim, dtype=torch.bfloat16, device="cuda")
    state = torch.empty(w.batch, w.heads, w.dstate, w.headdim, dtype=torch.float32, device="cuda")
    for b in range(w.batch):
        cache[b] = decode_cache_slab(w, b, m_cap).to("cuda", torch.bfloat16)
        state[b] = decode_state_slab(w, b).cuda()
    partial = torch.zeros_like(state)
    t = _token_dev(tok, "bf16")
    y, lse = api.decode_step(cache, state, partial, t["x"], t["dt"], t["A"], t["b"], t["c"], t["q"],
                             t["e"], t["z"], w.pos, w.chunk, w.eps)
    torch.cuda.synchronize()
    for b in (0, 37, 63):
        sl = lambda k: tok[k][b:b + 1]
        yo, lo, _, so, po = oracle_mod.decode_step(
            decode_cache_slab(w, b, m_cap)[None], decode_state_slab(w, b)[None],
            np.zeros((1, w.heads, w.dstate, w.headdim)), sl("x"), sl("dt"), tok["A"], sl("b"),
            sl("c"), sl("q"), sl("e"), sl("z"), w.pos, w.chunk, w.eps)
        assert rel_err(host(y[b:b + 1]), yo) <= TOL["bf16"]
        assert rel_err(host(lse[b:b + 1]), lo) <= TOL["bf16"]
        assert rel_err(host(state[b:b + 1]), so) <= 1e-5
        assert rel_err(host(partial[b:b + 1]), po) <= 1e-5


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_prefill_then_decode_equals_longer_prefill(oracle_mod, dtype):
    """GPU prefill of L0 tokens, then GPU decode of k tokens across two chunk
    boundaries, against the oracle prefill of L0 + k tokens: y at every decode
    position, and the memories the decode appends."""
    S, L0, k = 16, 32, 40
    w = Workload("dec_consistency", 2, 3, L0 + k, 32, 64, S, dtype=dtype, seed=21)
    inp = prefill_inputs(w)
    Yssd, dH, R, lse, Y = oracle_mod.forward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"],
                                             inp["Q"], inp["E"], inp["z"], S, w.eps)
    pre = {key: dev(inp[key][:, :L0], dtype) for key in ("X", "Bm", "Cm")}
    dt_pre = dev(inp["dt"][:, :L0], torch.float32)
    A = dev(inp["A"], torch.float32)
    # fp32 cache: the property is the decode semantics (bf16 storage of the cache
    # perturbs the logits by ~1e-2 and is covered by the storage tests)
    s = api.chunk_scan(pre["X"], dt_pre, A, pre["Bm"], pre["Cm"], S, w.eps, final_state=True)
    m_cap = -(-(L0 + k) // S)
    cache = torch.zeros(w.batch, m_cap, w.heads, w.dstate, w.headdim, dtype=s.M.dtype, device="cuda")
    cache[:, : L0 // S] = s.M
    state = s.final_state.clone()
    partial = torch.zeros_like(state)
    tol = TOL[dtype]
    for pos in range(L0, L0 + k):
        t = {key: dev(inp[src][:, pos], dtype) for key, src in
             (("x", "X"), ("b", "Bm"), ("c", "Cm"), ("q", "Q"), ("e", "E"), ("z", "z"))}
        y, l = api.decode_step(cache, state, partial, t["x"], dev(inp["dt"][:, pos], torch.float32), A,
                               t["b"], t["c"], t["q"], t["e"], t["z"], pos, S, w.eps)
        assert rel_err(host(y), Y[:, pos]) <= tol, pos
        assert rel_err(host(l), lse[:, pos]) <= tol, pos
    torch.cuda.synchronize()
    assert rel_err(host(cache[:, : (L0 + k) // S]), dH[:, : (L0 + k) // S]) <= tol


def test_ragged_prefill_hands_off_mid_chunk_to_decode(oracle_mod):
    """A prefill of L0 = 300 tokens (S = 128: two full chunks and 44 tokens of a
    third) on the tensor-core shapes, then decode from pos = 300 across the end of
    that chunk (pos 383 appends it) into the next: the prefill's last memory is the
    running partial memory and its final state the running state. Against the
    oracle prefill of L0 + k tokens: y at every decode position, the completed
    memories in the cache."""
    S, L0, k = 128, 300, 100
    w = Workload("dec_ragged", 2, 2, L0 + k, 64, 128, S, seed=23)
    inp = prefill_inputs(w)
    Yssd, dH, R, lse, Y = oracle_mod.forward(inp["X"], inp["dt"], inp["A"], inp["Bm"], inp["Cm"],
                                             inp["Q"], inp["E"], inp["z"], S, w.eps)
    pre = {key: dev(inp[key][:, :L0], "bf16") for key in ("X", "Bm", "Cm", "Q", "E", "z")}
    dt_pre = dev(inp["dt"][:, :L0], torch.float32)
    A = dev(inp["A"], torch.float32)
    s, o = api.prefill_forward(pre["X"], dt_pre, A, pre["Bm"], pre["Cm"], pre["Q"], pre["E"], pre["z"], S,
                               w.eps)
    s_fs = api.chunk_scan(pre["X"], dt_pre, A, pre["Bm"], pre["Cm"], S, w.eps, final_state=True)
    torch.cuda.synchronize()
    assert s.M.shape[1] == 3  # ceil(300 / 128): the third memory is the partial chunk
    assert rel_err(host(o.Y), Y[:, :L0]) <= TOL["bf16"]
    m_cap = -(-(L0 + k) // S)
    cache = torch.zeros(w.batch, m_cap, w.heads, w.dstate, w.headdim, dtype=torch.float32, device="cuda")
    cache[:, : L0 // S] = s.M[:, : L0 // S]
    partial = s.M[:, L0 // S].contiguous()  # the running partial memory of chunk 2
    state = s_fs.final_state.clone()
    for pos in range(L0, L0 + k):
        t = {key: dev(inp[src][:, pos], "bf16") for key, src in
             (("x", "X"), ("b", "Bm"), ("c", "Cm"), ("q", "Q"), ("e", "E"), ("z", "z"))}
        y, l = api.decode_step(cache, state, partial, t["x"], dev(inp["dt"][:, pos], torch.float32), A,
                               t["b"], t["c"], t["q"], t["e"], t["z"], pos, S, w.eps)
        assert rel_err(host(y), Y[:, pos]) <= TOL["bf16"], pos
        assert rel_err(host(l), lse[:, pos]) <= TOL["bf16"], pos
    torch.cuda.synchronize()
    assert rel_err(host(cache[:, :3]), dH[:, :3]) <= TOL["bf16"]


def test_decode_mid_chunk_updates_state_and_partial(oracle_mod):
    """pos inside a chunk: the partial memory decays and accumulates (no reset)."""
    w = Workload("dec_mid", 3, 4, 1, 64, 128, 64, seed=31, mem=5, pos=5 * 64 + 17)
    tok = decode_token_inputs(w)
    hs = decode_state(w, m_cap=6)
    cache, state, partial = (dev(hs[k], d) for k, d in
                             (("cache", "bf16"), ("state", torch.float32), ("partial", torch.float32)))
    t = _token_dev(tok, "bf16")
    y, lse = api.decode_step(cache, state, partial, t["x"], t["dt"], t["A"], t["b"], t["c"], t["q"],
                             t["e"], t["z"], w.pos, w.chunk, w.eps)
    torch.cuda.synchronize()
    yo, lo, co, so, po = oracle_mod.decode_step(hs["cache"], hs["state"], hs["partial"], tok["x"],
                                                tok["dt"], tok["A"], tok["b"], tok["c"], tok["q"],
                                                tok["e"], tok["z"], w.pos, w.chunk, w.eps)
    assert rel_err(host(y), yo) <= TOL["bf16"]
    assert rel_err(host(lse), lo) <= TOL["bf16"]
    assert rel_err(host(state), so) <= 1e-5
    assert rel_err(host(partial), po) <= 1e-5
    assert torch.equal(cache.float().cpu(), hs["cache"])  # no chunk completed: cache untouched


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_decode_chunk_end_appends_the_partial_memory(oracle_mod, dtype):
    """(pos + 1) % S == 0: the completed partial memory becomes cache slot pos / S
    (stored in the cache's dtype: bf16 rounding to nearest for a bf16 cache)."""
    w = Workload("dec_end", 2, 2, 1, 32, 64, 32, dtype=dtype, seed=33, mem=3, pos=3 * 32 + 31)
    tok = decode_token_inputs(w)
    hs = decode_state(w, m_cap=4)
    cache = dev(hs["cache"], dtype)
    state, partial = (dev(hs[k], torch.float32) for k in ("state", "partial"))
    t = _token_dev(tok, dtype)
    y, lse = api.decode_step(cache, state, partial, t["x"], t["dt"], t["A"], t["b"], t["c"], t["q"],
                             t["e"], t["z"], w.pos, w.chunk, w.eps)
    torch.cuda.synchronize()
    yo, lo, co, so, po = oracle_mod.decode_step(hs["cache"], hs["state"], hs["partial"], tok["x"],
                                                tok["dt"], tok["A"], tok["b"], tok["c"], tok["q"],
                                                tok["e"], tok["z"], w.pos, w.chunk, w.eps)
    assert rel_err(host(y), yo) <= TOL[dtype]
    assert torch.equal(cache[:, :3].float().cpu(), hs["cache"][:, :3])  # earlier slots untouched
    got = host(cache[:, 3])
    if dtype == "f32":
        assert rel_err(got, po) <= 1e-5
    else:
        assert np.all(np.abs(got - po) <= 2.0 ** -8 * np.abs(po) + 1e-7 * np.abs(po).max())


def test_decode_first_chunk_has_no_readout(oracle_mod):
    """pos < S: no completed memory, so y = c state and lse = -inf."""
    w = Workload("dec_first", 2, 2, 1, 32, 16, 16, dtype="f32", seed=41, mem=0, pos=3)
    tok = decode_token_inputs(w)
    hs = decode_state(w, m_cap=1)
    cache, state, partial = (dev(hs[k], torch.float32) for k in ("cache", "state", "partial"))
    t = _token_dev(tok, "f32")
    y, lse = api.decode_step(cache, state, partial, t["x"], t["dt"], t["A"], t["b"], t["c"], t["q"],
                             t["e"], t["z"], w.pos, w.chunk, w.eps)
    torch.cuda.synchronize()
    yo, lo, _, so, po = oracle_mod.decode_step(hs["cache"], hs["state"], hs["partial"], tok["x"],
                                               tok["dt"], tok["A"], tok["b"], tok["c"], tok["q"],
                                               tok["e"], tok["z"], w.pos, w.chunk, w.eps)
    assert np.all(np.isneginf(host(lse)))
    assert rel_err(host(y), yo) <= TOL["f32"]
    assert rel_err(host(partial), po) <= 1e-5
