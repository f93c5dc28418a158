"""Pins of the oracle's backward functions (CPU, no GPU).

The paper prints no backward equations, so the oracle's gradients are the
chain rule written out by hand. They are pinned to things other than
themselves: central finite differences of the (separately pinned) forward
oracle in fp64, and closed forms of special cases.
"""
import numpy as np
import pytest

import oracle

EPS = 1e-6
FD_H = 1e-6


def _inputs(rng, Bsz=1, L=64, H=2, G=1, P=8, N=8):
    X = rng.standard_normal((Bsz, L, H, P)) / np.sqrt(P)
    dt = np.log1p(np.exp(rng.normal(-2.0, 0.5, (Bsz, L, H))))  # softplus, as the workloads draw it
    A = -np.exp(rng.uniform(0.0, np.log(16.0), H))
    Bm = rng.standard_normal((Bsz, L, G, N)) / np.sqrt(N)
    Cm = rng.standard_normal((Bsz, L, G, N)) / np.sqrt(N)
    Q = rng.standard_normal((Bsz, L, G, N)) / np.sqrt(N)
    E = rng.standard_normal((Bsz, L, G, P)) / np.sqrt(P)
    z = rng.standard_normal((Bsz, L, H))
    return X, dt, A, Bm, Cm, Q, E, z


def _fd(loss, arrays, idx_lists):
    """Central differences of loss() w.r.t. the listed flat entries of each array."""
    out = []
    for a, idx in zip(arrays, idx_lists):
        g = np.zeros(len(idx))
        flat = a.reshape(-1)
        for k, i in enumerate(idx):
            v = flat[i]
            flat[i] = v + FD_H
            lp = loss()
            flat[i] = v - FD_H
            lm = loss()
            flat[i] = v
            g[k] = (lp - lm) / (2 * FD_H)
        out.append(g)
    return out


def _rel(a, b):
    scale = max(np.abs(b).max(), 1e-300)
    return np.abs(a - b).max() / scale


@pytest.mark.parametrize("L,S,G", [(64, 16, 1), (56, 16, 1), (48, 16, 2)])
def test_ssd_backward_matches_finite_differences(L, S, G):
    rng = np.random.default_rng(11 + L + G)
    H, P, N = 2, 8, 6
    X, dt, A, Bm, Cm, *_ = _inputs(rng, L=L, H=H, G=G, P=P, N=N)
    M = -(-L // S)
    Wy = rng.standard_normal((1, L, H, P))
    Wm = rng.standard_normal((1, M, H, N, P))

    def loss():
        Y, _ = oracle.ssd_recurrence(X, dt, A, Bm, Cm)
        D = oracle.chunk_memories(X, dt, A, Bm, S)
        return float((Wy * Y).sum() + (Wm * D).sum())

    dX, ddt, dA, dB, dC = oracle.ssd_backward(X, dt, A, Bm, Cm, Wy, Wm, S)
    arrays = [X, dt, A, Bm, Cm]
    grads = [dX, ddt, dA, dB, dC]
    idx = [np.arange(a.size) for a in arrays]
    fds = _fd(loss, arrays, idx)
    for name, g, f in zip(["X", "dt", "A", "B", "C"], grads, fds):
        assert _rel(g.reshape(-1), f) < 1e-6, name


def test_ssd_backward_without_memory_gradient_is_the_recurrence_adjoint():
    """dMem = None must equal dMem = 0, and only dY then drives the result."""
    rng = np.random.default_rng(5)
    X, dt, A, Bm, Cm, *_ = _inputs(rng, L=32)
    dY = rng.standard_normal(X.shape)
    a = oracle.ssd_backward(X, dt, A, Bm, Cm, dY, None, 16)
    b = oracle.ssd_backward(X, dt, A, Bm, Cm, dY, np.zeros((1, 2, 2, 8, 8)), 16)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_ssd_backward_linear_attention_closed_form():
    """a_t = 1, dt = 1 (Sec. 2, SSD with an all-ones mask): Y = tril(C B^T) X, so
    dX = tril(C B^T)^T dY, dC = tril(dY X^T) B and dB = tril(dY X^T)^T C."""
    rng = np.random.default_rng(7)
    L, P, N, S = 40, 6, 5, 8
    X = rng.standard_normal((1, L, 1, P))
    dt = np.ones((1, L, 1))
    A = np.zeros(1)
    Bm = rng.standard_normal((1, L, 1, N))
    Cm = rng.standard_normal((1, L, 1, N))
    dY = rng.standard_normal((1, L, 1, P))
    dX, ddt, dA, dB, dC = oracle.ssd_backward(X, dt, A, Bm, Cm, dY, None, S)
    x, b, c, dy = X[0, :, 0], Bm[0, :, 0], Cm[0, :, 0], dY[0, :, 0]
    att = np.tril(c @ b.T)
    datt = np.tril(dy @ x.T)
    np.testing.assert_allclose(dX[0, :, 0], att.T @ dy, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dC[0, :, 0], datt @ b, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dB[0, :, 0], datt.T @ c, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("G", [1, 2])
def test_sma_backward_matches_finite_differences(G):
    rng = np.random.default_rng(21 + G)
    L, S, H, P, N = 64, 16, 2, 8, 12  # N != P, so a normalisation over the wrong axis shows
    X, dt, A, Bm, Cm, Q, E, z = _inputs(rng, L=L, H=H, G=G, P=P, N=N)
    D = oracle.chunk_memories(X, dt, A, Bm, S)
    Yssd = rng.standard_normal((1, L, H, P))
    W = rng.standard_normal((1, L, H, P))

    def loss():
        R, _ = oracle.sma(D, Q, Cm, E, S, EPS)
        return float((W * oracle.merge(Yssd, z, R)).sum())

    dMem, dQ, dC, dE, dz = oracle.sma_backward(D, Q, Cm, E, z, W, S, EPS)
    arrays = [D, Q, Cm, E, z]
    grads = [dMem, dQ, dC, dE, dz]
    fds = _fd(loss, arrays, [np.arange(a.size) for a in arrays])
    for name, g, f in zip(["Mem", "Q", "C", "E", "z"], grads, fds):
        assert _rel(g.reshape(-1), f) < 1e-6, name


def test_sma_backward_gate_closed_form_at_zero_logit():
    """SiLU'(0) = 1/2, so dz = (dY . R) / 2 where z = 0; tokens without history get 0."""
    rng = np.random.default_rng(3)
    L, S = 48, 16
    X, dt, A, Bm, Cm, Q, E, z = _inputs(rng, L=L)
    z[:] = 0.0
    D = oracle.chunk_memories(X, dt, A, Bm, S)
    dY = rng.standard_normal((1, L, 2, 8))
    R, _ = oracle.sma(D, Q, Cm, E, S, EPS)
    *_, dz = oracle.sma_backward(D, Q, Cm, E, z, dY, S, EPS)
    np.testing.assert_allclose(dz, 0.5 * (dY * R).sum(-1), rtol=1e-12, atol=1e-14)
    assert np.all(dz[:, :S] == 0.0)


def test_layer_backward_matches_finite_differences_on_a_sample():
    """The whole layer: the SMA memory gradient feeds the scan backward, and dC
    sums both paths. Checked on a random sample of entries of every input."""
    rng = np.random.default_rng(31)
    L, S = 48, 16
    inputs = list(_inputs(rng, L=L, P=6, N=10))
    W = rng.standard_normal((1, L, 2, 6))

    def loss():
        *_, Y = oracle.forward(*inputs, S, EPS)
        return float((W * Y).sum())

    grads = oracle.backward(*inputs, W, S, EPS)
    # backward order: dX, d_dt, dA, dB, dC, dQ, dE, dz ; inputs: X, dt, A, Bm, Cm, Q, E, z
    idx = [rng.choice(a.size, size=min(a.size, 40), replace=False) for a in inputs]
    fds = _fd(loss, inputs, idx)
    for name, g, f, i in zip(["X", "dt", "A", "B", "C", "Q", "E", "z"], grads, fds, idx):
        assert _rel(g.reshape(-1)[i], f) < 1e-6, name
