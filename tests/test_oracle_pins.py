"""Pins of the CPU oracle against facts the paper and the mathematics fix.

Each test ties one oracle function to something other than itself: another
formulation the paper proves equal (the SSD attention form, the App. A
chunked scan), a closed form, an invariant, or a special case that reduces to
a textbook routine. Chosen so that a dropped term, a wrong decay index, a
wrong normalisation axis or a transposed operand fails at least one of them.
"""
import math
import os

import numpy as np
import pytest

TOL = 1e-11


def _rng_inputs(seed, Bsz, L, H, G, P, N, Amin=-3.0):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((Bsz, L, H, P))
    Bm = rng.standard_normal((Bsz, L, G, N)) / math.sqrt(N)
    Cm = rng.standard_normal((Bsz, L, G, N)) / math.sqrt(N)
    Q = rng.standard_normal((Bsz, L, G, N))
    E = rng.standard_normal((Bsz, L, G, P))
    dt = np.log1p(np.exp(rng.normal(-1.0, 0.5, (Bsz, L, H))))
    A = -np.exp(rng.uniform(0.0, -Amin, H)) + 0.5
    z = rng.standard_normal((Bsz, L, H))
    return dict(X=X, Bm=Bm, Cm=Cm, Q=Q, E=E, dt=dt, A=A, z=z)


def _rel(a, b):
    return np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300)


# ---------------------------------------------------------------- recurrence

def test_recurrence_is_causal_linear_attention_without_decay(oracle_mod):
    """a_t = 1 and dt = 1 turn the SSD layer into causal linear attention
    Y = tril(C B^T) X (Sec. 2: CB^T X has the form QK^T V)."""
    d = _rng_inputs(1, 2, 17, 4, 2, 3, 5)
    dt = np.ones_like(d["dt"])
    A = np.zeros(4)
    Y, _ = oracle_mod.ssd_recurrence(d["X"], dt, A, d["Bm"], d["Cm"])
    for b in range(2):
        for h in range(4):
            g = h // 2  # H / G = 2 heads per group
            CBt = d["Cm"][b, :, g] @ d["Bm"][b, :, g].T
            ref = np.tril(CBt) @ d["X"][b, :, h]
            assert _rel(Y[b, :, h], ref) < TOL


def test_recurrence_matches_ssd_masked_attention_form(oracle_mod):
    """Sec. 2: Y = (L_SSD o C B^T) X with (L_SSD)_{ij} = prod_{k=j+1}^{i} a_k for
    i >= j, here with the write scaled by dt (so X -> dt X)."""
    d = _rng_inputs(2, 1, 23, 3, 1, 4, 6)
    Y, _ = oracle_mod.ssd_recurrence(d["X"], d["dt"], d["A"], d["Bm"], d["Cm"])
    L = 23
    for h in range(3):
        a = np.exp(d["dt"][0, :, h] * d["A"][h])
        Lssd = np.zeros((L, L))
        for i in range(L):
            for j in range(i + 1):
                Lssd[i, j] = np.prod(a[j + 1:i + 1])
        CBt = d["Cm"][0, :, 0] @ d["Bm"][0, :, 0].T
        ref = (Lssd * CBt) @ (d["dt"][0, :, h, None] * d["X"][0, :, h])
        assert _rel(Y[0, :, h], ref) < TOL


# -------------------------------------------------------------- chunk memories

@pytest.mark.parametrize("L,S", [(48, 16), (50, 16), (7, 8)])
def test_chunked_scan_of_appendix_a_reproduces_recurrence(oracle_mod, L, S):
    """App. A: H_[c] = A_{a_c:b_c} H_[c-1] + dH_[c] and Y_t = Y^intra + C_t A_{a_c:t} H_[c-1]
    rebuild the token recurrence from the oracle's chunk memories (ragged last
    chunk included)."""
    Bsz, H, G, P, N = 2, 2, 1, 3, 4
    d = _rng_inputs(3, Bsz, L, H, G, P, N)
    Y, Hlast = oracle_mod.ssd_recurrence(d["X"], d["dt"], d["A"], d["Bm"], d["Cm"])
    dH = oracle_mod.chunk_memories(d["X"], d["dt"], d["A"], d["Bm"], S)
    M = -(-L // S)
    assert dH.shape == (Bsz, M, H, N, P)
    for b in range(Bsz):
        for h in range(H):
            a = np.exp(d["dt"][b, :, h] * d["A"][h])
            Hprev = np.zeros((N, P))
            for c in range(M):
                lo, hi = c * S, min((c + 1) * S, L)
                for t in range(lo, hi):
                    intra = np.zeros(P)
                    for s in range(lo, t + 1):
                        w = np.prod(a[s + 1:t + 1]) * d["dt"][b, s, h]
                        intra += w * (d["Cm"][b, t, 0] @ d["Bm"][b, s, 0]) * d["X"][b, s, h]
                    inter = np.prod(a[lo:t + 1]) * (d["Cm"][b, t, 0] @ Hprev)
                    assert _rel(Y[b, t, h], intra + inter) < 1e-10
                Hprev = np.prod(a[lo:hi]) * Hprev + dH[b, c, h]
            assert _rel(Hlast[b, h], Hprev) < 1e-10


def test_scan_outputs_are_linear_in_x(oracle_mod):
    """For fixed dt, A, B, C the recurrence and the chunk memories are linear in X
    (App. A): Y_ssd and M_j of a X1 + b X2 are a Y(X1) + b Y(X2) and the same for
    the memories."""
    d1 = _rng_inputs(15, 2, 24, 2, 1, 3, 5)
    X2 = np.random.default_rng(115).standard_normal(d1["X"].shape)
    a, b = 0.75, -1.5
    args = (d1["dt"], d1["A"], d1["Bm"], d1["Cm"])
    Y1, _ = oracle_mod.ssd_recurrence(d1["X"], *args)
    Y2, _ = oracle_mod.ssd_recurrence(X2, *args)
    Y3, _ = oracle_mod.ssd_recurrence(a * d1["X"] + b * X2, *args)
    assert _rel(Y3, a * Y1 + b * Y2) < 1e-12
    margs = (d1["dt"], d1["A"], d1["Bm"], 8)
    M1 = oracle_mod.chunk_memories(d1["X"], *margs)
    M2 = oracle_mod.chunk_memories(X2, *margs)
    M3 = oracle_mod.chunk_memories(a * d1["X"] + b * X2, *margs)
    assert _rel(M3, a * M1 + b * M2) < 1e-12


def test_decayed_sum_of_memories_is_final_state(oracle_mod):
    """Unrolling App. A eq. (mamba2_chunk_state): H_{L-1} = sum_c A_{e(c)+1:L-1} dH_[c]."""
    L, S, H = 40, 8, 3
    d = _rng_inputs(4, 1, L, H, 1, 5, 7)
    _, Hlast = oracle_mod.ssd_recurrence(d["X"], d["dt"], d["A"], d["Bm"], d["Cm"])
    dH = oracle_mod.chunk_memories(d["X"], d["dt"], d["A"], d["Bm"], S)
    for h in range(H):
        cum = d["dt"][0, :, h] * d["A"][h]
        tot = np.zeros_like(Hlast[0, h])
        for c in range(L // S):
            e = (c + 1) * S - 1
            tot += np.exp(cum[e + 1:].sum()) * dH[0, c, h]
        assert _rel(tot, Hlast[0, h]) < 1e-12


def test_single_chunk_memory_is_the_state(oracle_mod):
    """S = L: the one chunk memory is the whole recurrent state (empty decay at the end)."""
    d = _rng_inputs(5, 2, 19, 2, 1, 3, 4)
    _, Hlast = oracle_mod.ssd_recurrence(d["X"], d["dt"], d["A"], d["Bm"], d["Cm"])
    dH = oracle_mod.chunk_memories(d["X"], d["dt"], d["A"], d["Bm"], 19)
    assert _rel(dH[:, 0], Hlast) < 1e-12


# ------------------------------------------------------------------------ SMA

def _small_sma_case(seed=6, Bsz=2, L=40, H=3, G=1, P=4, N=6, S=8):
    d = _rng_inputs(seed, Bsz, L, H, G, P, N)
    dH = np.random.default_rng(seed + 100).standard_normal((Bsz, -(-L // S), H, N, P))
    return d, dH, S


def test_sma_weights_form_a_distribution_over_earlier_chunks(oracle_mod):
    d, dH, S = _small_sma_case()
    R, lse, g = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], S, 1e-6, want_g=True)
    L = d["Q"].shape[1]
    for t in range(L):
        nh = t // S
        gt = g[:, t]
        assert np.all(gt >= 0)
        assert np.all(gt[..., nh:] == 0)
        if nh:
            assert np.allclose(gt.sum(-1), 1.0, atol=1e-14, rtol=0)
        else:
            assert np.all(R[:, t] == 0) and np.all(np.isneginf(lse[:, t]))


def test_sma_online_softmax_of_algorithm_1_matches_two_pass(oracle_mod):
    """Alg. 1 / App. C online recurrences (m, d, O) over the oracle's logits
    (recovered as l = lse + log g) reproduce R = sum_j g_j C_t dH_j."""
    d, dH, S = _small_sma_case(seed=7)
    R, lse, g = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], S, 1e-6, want_g=True)
    for b, t, h in [(0, 39, 1), (1, 17, 2), (0, 8, 0)]:
        nh = t // S
        ell = lse[b, t, h] + np.log(g[b, t, h, :nh])
        m, den, O = -np.inf, 0.0, np.zeros(dH.shape[-1])
        for j in range(nh):
            V = d["Cm"][b, t, 0] @ dH[b, j, h]
            mn = max(m, ell[j])
            den = np.exp(m - mn) * den + np.exp(ell[j] - mn)
            O = np.exp(m - mn) * O + np.exp(ell[j] - mn) * V
            m = mn
        assert _rel(O / den, R[b, t, h]) < 1e-12
        assert abs(m + np.log(den) - lse[b, t, h]) < 1e-12


def test_sma_single_memory_gives_value_readout(oracle_mod):
    """Tokens of chunk 1 see one memory: R_t = C_t dH_[0] whatever Q and E are."""
    d, dH, S = _small_sma_case(seed=8)
    R, lse = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], S, 1e-6)
    for t in range(S, 2 * S):
        for h in range(3):
            ref = np.einsum("bn,bnp->bp", d["Cm"][:, t, 0], dH[:, 0, h])
            assert _rel(R[:, t, h], ref) < 1e-13


def test_sma_zero_query_gives_uniform_average(oracle_mod):
    """Q = 0 makes every logit 0: g uniform, R = mean_j C_t dH_j, lse = log(#memories)."""
    d, dH, S = _small_sma_case(seed=9)
    Q = np.zeros_like(d["Q"])
    R, lse = oracle_mod.sma(dH, Q, d["Cm"], d["E"], S, 1e-6)
    for t in [20, 33, 39]:
        nh = t // S
        for h in range(3):
            V = np.einsum("bn,bjnp->bjp", d["Cm"][:, t, 0], dH[:, :nh, h])
            assert _rel(R[:, t, h], V.mean(1)) < 1e-13
            assert np.allclose(lse[:, t, h], math.log(nh), rtol=0, atol=1e-14)


def test_sma_rank_one_memories_closed_form(oracle_mod):
    """dH_j[n,p] = alpha_j beta_n gamma_p and e = gamma give, as eps -> 0,
    r_{j,n} = 1/(|alpha_j| beta_n rms(gamma)) (inverse RMS along P, App. B.1),
    K_{j,n} = sign(alpha_j) P, so l_j = sign(alpha_j) P sum_n Qbar_n / sqrt(N);
    V_j = alpha_j (C_t . beta) gamma."""
    P, N, S = 5, 4, 2  # N != P so a normalisation over the wrong axis shows
    alpha = np.array([0.7, -2.5, 1.3])
    beta = np.array([0.5, 1.0, 2.0, 3.0])
    gamma = np.array([1.0, -2.0, 0.5, 3.0, -1.5])
    L = S * (len(alpha) + 1)
    M = L // S
    dH = np.zeros((1, M, 1, N, P))
    for j, a in enumerate(alpha):
        dH[0, j, 0] = a * np.outer(beta, gamma)
    q = np.array([2.0, -2.0, 2.0, 2.0])  # rms 2, so Qbar = (1, -1, 1, 1), sum 2
    c = np.array([0.3, -0.1, 0.2, 0.4])
    Q = np.tile(q, (1, L, 1, 1))
    E = np.tile(gamma, (1, L, 1, 1))
    Cm = np.tile(c, (1, L, 1, 1))
    t = L - 1
    R, lse, g = oracle_mod.sma(dH, Q, Cm, E, S, 1e-14, tokens=[[0, t, 0]], want_g=True)
    ell = np.sign(alpha) * P * 2.0 / math.sqrt(N)
    gref = np.exp(ell - ell.max()) / np.exp(ell - ell.max()).sum()
    Rref = sum(gj * aj * (c @ beta) * gamma for gj, aj in zip(gref, alpha))
    assert np.allclose(g[0, :3], gref, rtol=1e-9, atol=0)
    assert _rel(R[0], Rref) < 1e-9
    assert abs(lse[0] - math.log(np.exp(ell).sum())) < 1e-9


def test_sma_logits_are_scale_invariant_in_q_and_e(oracle_mod):
    """RMSNorm makes the routing independent of the scale of Q and E (up to eps)."""
    d, dH, S = _small_sma_case(seed=10)
    R1, l1, g1 = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], S, 1e-12, want_g=True)
    R2, l2, g2 = oracle_mod.sma(dH, 7.0 * d["Q"], d["Cm"], 0.25 * d["E"], S, 1e-12, want_g=True)
    assert np.max(np.abs(g1 - g2)) < 1e-9 and _rel(R2, R1) < 1e-9


def test_sma_memory_scale_moves_values_not_routing(oracle_mod):
    """The key path reads r (.) M_j, whose row scale r cancels a uniform scale of M_j
    (App. B.1), while the value path reads M_j itself: scaling every memory by alpha
    leaves the weights and lse unchanged (up to eps) and scales R by alpha."""
    d, dH, S = _small_sma_case(seed=14)
    alpha = 3.5
    R1, l1, g1 = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], S, 1e-30, want_g=True)
    R2, l2, g2 = oracle_mod.sma(alpha * dH, d["Q"], d["Cm"], d["E"], S, 1e-30, want_g=True)
    fin = np.isfinite(l1)
    assert np.max(np.abs(g1 - g2)) < 1e-12 and np.max(np.abs(l1[fin] - l2[fin])) < 1e-12
    assert _rel(R2, alpha * R1) < 1e-12


def test_sma_is_causal_over_chunks(oracle_mod):
    """Token t reads memories j < chunk(t) only: changing later memories changes nothing."""
    d, dH, S = _small_sma_case(seed=11)
    R1, l1 = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], S, 1e-6)
    dH2 = dH.copy()
    dH2[:, 3:] += 5.0
    R2, l2 = oracle_mod.sma(dH2, d["Q"], d["Cm"], d["E"], S, 1e-6)
    assert np.array_equal(R1[:, : 4 * S], R2[:, : 4 * S])
    assert not np.allclose(R1[:, 4 * S:], R2[:, 4 * S:])


def test_sma_single_chunk_sequence_has_no_readout(oracle_mod):
    """S = L (M = 1): no token has history, so R = 0 and lse = -inf everywhere."""
    d = _rng_inputs(12, 1, 16, 2, 1, 3, 4)
    dH = np.random.default_rng(0).standard_normal((1, 1, 2, 4, 3))
    R, lse = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], 16, 1e-6)
    assert np.all(R == 0) and np.all(np.isneginf(lse))


def test_token_list_matches_full_evaluation(oracle_mod):
    d, dH, S = _small_sma_case(seed=13)
    R, lse = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], S, 1e-6)
    toks = np.array([[1, 39, 2], [0, 9, 0], [1, 3, 1]])
    Rs, ls = oracle_mod.sma(dH, d["Q"], d["Cm"], d["E"], S, 1e-6, tokens=toks)
    for i, (b, t, h) in enumerate(toks):
        assert np.array_equal(Rs[i], R[b, t, h])
        assert ls[i] == lse[b, t, h] or (np.isneginf(ls[i]) and np.isneginf(lse[b, t, h]))


def test_memory_inverse_rms_closed_forms(oracle_mod):
    """App. B.1: r = (mean_p dH^2 + eps)^-1/2 along the value axis P: a row of
    constant a gives (a^2 + eps)^-1/2; the row (3, 4) gives (12.5 + eps)^-1/2."""
    eps = 1e-6
    dH = np.zeros((1, 2, 1, 3, 2))
    dH[0, 0, 0, 0] = [2.0, 2.0]
    dH[0, 0, 0, 1] = [3.0, 4.0]
    dH[0, 1, 0, 2] = [-5.0, -5.0]
    r = oracle_mod.memory_inverse_rms(dH, eps)
    assert r.shape == (1, 2, 1, 3)
    assert abs(r[0, 0, 0, 0] - 1 / math.sqrt(4.0 + eps)) < 1e-15
    assert abs(r[0, 0, 0, 1] - 1 / math.sqrt(12.5 + eps)) < 1e-15
    assert abs(r[0, 1, 0, 2] - 1 / math.sqrt(25.0 + eps)) < 1e-15
    assert abs(r[0, 0, 0, 2] - 1 / math.sqrt(eps)) < 1e-9


# ---------------------------------------------------------------------- merge

def test_zero_gate_reproduces_mamba2_exactly(oracle_mod):
    """Sec. 3: with W_G = 0 the gate logit is 0, SiLU(0) = 0, and Y = C_t H_t exactly
    (the SMA-removal ablation of Sec. 5 is the same operation)."""
    rng = np.random.default_rng(14)
    Yssd = rng.standard_normal((3, 5, 2, 4))
    R = rng.standard_normal((3, 5, 2, 4))
    Y = oracle_mod.merge(Yssd, np.zeros((3, 5, 2)), R)
    assert np.array_equal(Y, Yssd)


def test_gate_is_silu(oracle_mod):
    """SiLU(ln 3) = ln 3 * sigmoid(ln 3) = 0.75 ln 3; SiLU(z) -> z for large z."""
    z = np.array([[math.log(3.0), 40.0, -40.0]])
    Y = oracle_mod.merge(np.zeros((1, 3, 1)), z, np.ones((1, 3, 1)))
    assert abs(Y[0, 0, 0] - 0.75 * math.log(3.0)) < 1e-15
    assert abs(Y[0, 1, 0] - 40.0) < 1e-12
    assert abs(Y[0, 2, 0]) < 1e-15


# --------------------------------------------------------------------- decode

def test_prefill_then_decode_equals_longer_prefill(oracle_mod):
    """Prefill L tokens, then decode k more: y, the running state and the
    appended memories equal the prefill of L + k tokens."""
    Bsz, H, G, P, N, S, eps = 2, 2, 1, 3, 4, 8, 1e-6
    L0, k = 13, 12  # decode crosses the chunk boundaries at tokens 15 and 23
    Lt = L0 + k
    d = _rng_inputs(15, Bsz, Lt, H, G, P, N)
    Yssd, dH, R, lse, Y = oracle_mod.forward(d["X"], d["dt"], d["A"], d["Bm"], d["Cm"], d["Q"],
                                             d["E"], d["z"], S, eps)
    pre = {k_: v[:, :L0] for k_, v in d.items() if k_ not in ("A",)}
    _, state = oracle_mod.ssd_recurrence(pre["X"], pre["dt"], d["A"], pre["Bm"], pre["Cm"])
    mem0 = oracle_mod.chunk_memories(pre["X"], pre["dt"], d["A"], pre["Bm"], S)
    m_cap = -(-Lt // S)
    cache = np.zeros((Bsz, m_cap, H, N, P))
    cache[:, : L0 // S] = mem0[:, : L0 // S]
    partial = mem0[:, L0 // S] if L0 % S else np.zeros((Bsz, H, N, P))
    for pos in range(L0, Lt):
        y, l, cache, state, partial = oracle_mod.decode_step(
            cache, state, partial, d["X"][:, pos], d["dt"][:, pos], d["A"], d["Bm"][:, pos],
            d["Cm"][:, pos], d["Q"][:, pos], d["E"][:, pos], d["z"][:, pos], pos, S, eps)
        assert _rel(y, Y[:, pos]) < 1e-11
        if pos // S > 0:
            assert np.max(np.abs(l - lse[:, pos])) < 1e-11
    for j in range(Lt // S):
        assert _rel(cache[:, j], dH[:, j]) < 1e-11


# ---------------------------------------------------------------- cache ratio

def _golden_cache_ratio():
    path = os.path.join(os.path.dirname(__file__), "golden", "cache_ratio.txt")
    rows = [ln.split() for ln in open(path) if ln.strip() and not ln.startswith("#")]
    S, N, ratio, saving, retr = rows[0]
    return int(S), int(N), float(ratio), float(saving), float(retr)


def test_cache_ratio_is_the_papers_25_percent(oracle_mod):
    """Sec. 4: M N P / (2 L P) = N / (2 S) = 0.25 at S = 256, N = 128 (75 % saving),
    counted from the element counts of the memories the oracle actually keeps."""
    S, N, ratio, saving, retr = _golden_cache_ratio()
    P, L = 2, 4 * S
    X = np.zeros((1, L, 1, P))
    dt = np.zeros((1, L, 1))
    Bm = np.zeros((1, L, 1, N))
    dH = oracle_mod.chunk_memories(X, dt, np.zeros(1), Bm, S)
    kv_elems = 2 * L * P  # keys and values of every token
    assert dH.size / kv_elems == pytest.approx(ratio, abs=0)
    assert 1 - dH.size / kv_elems == pytest.approx(saving, abs=0)
    # leading-order SMA retrieval cost: L * M pairs of 2 N P contractions against
    # L^2 * P for token attention (Sec. 4 "Training Complexity")
    assert (L * (L // S) * N * P) / (L * L * P) == pytest.approx(retr, abs=0)
