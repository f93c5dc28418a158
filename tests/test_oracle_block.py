"""Pins of the whole-block oracle (oracle/block.py) against facts its definitions
fix: convolution taps, causality, the zero gate reducing DART to Mamba-2 (Sec. 3,
W_G initialised to zero), the scale invariance and the axis of the output
RMSNorm. CPU only."""
import numpy as np
import pytest

import oracle
import oracle.block as ob
from paper_2608_02032_gb300.workloads import BlockWorkload, block_inputs

W = BlockWorkload("block_pin", 2, 96, 64, 2, headdim=16, dstate=8, chunk=32, seed=7)


@pytest.fixture(scope="module")
def inp():
    oracle.build()
    return {k: v.double().numpy() for k, v in block_inputs(W).items()}


def _run(inp, norm_eps=W.norm_eps, **kw):
    a = dict(inp)
    a.update(kw)
    return ob.block_forward(a["U"], a["W_in"], a["conv_w"], a["conv_b"], a["dt_bias"], a["A_log"], a["D"],
                            a["norm_w"], a["W_out"], W.heads, W.groups, W.dstate, W.headdim, W.chunk, W.eps,
                            norm_eps)


def _rows(name):
    """Row slice of W_in for one column block of the in-projection."""
    di, GN, H, GP = W.d_inner, W.groups * W.dstate, W.heads, W.groups * W.headdim
    o = 0
    for n, size in (("z", di), ("x", di), ("B", GN), ("C", GN), ("dt", H), ("Q", GN), ("E", GP), ("gate", 1)):
        if n == name:
            return slice(o, o + size)
        o += size
    raise KeyError(name)


def test_in_projection_width():
    assert W.d_in_proj == 2 * 32 + 3 * 8 + 2 + 16 + 1
    assert ob.in_proj_width(W.d_inner, W.heads, W.groups, W.dstate, W.headdim) == W.d_in_proj


def test_conv_delta_taps_are_identity_and_causal_shift():
    rng = np.random.default_rng(0)
    xs = rng.standard_normal((2, 10, 3))
    w = np.zeros((3, 4))
    w[:, 3] = 1.0  # the last tap reads the current token
    assert np.array_equal(ob.causal_conv(xs, w, np.zeros(3)), xs)
    w = np.zeros((3, 4))
    w[:, 0] = 1.0  # the first tap reads three tokens back, zeros before the sequence
    out = ob.causal_conv(xs, w, np.zeros(3))
    assert np.array_equal(out[:, 3:], xs[:, :-3]) and np.all(out[:, :3] == 0)
    # a bias alone, and per-channel taps
    assert np.allclose(ob.causal_conv(np.zeros((1, 4, 3)), np.ones((3, 4)), np.arange(3.0)), np.arange(3.0))


def test_block_is_causal(inp):
    out, _ = _run(inp)
    U2 = inp["U"].copy()
    U2[:, 50] += 1.0
    out2, _ = _run(inp, U=U2)
    assert np.array_equal(out[:, :50], out2[:, :50])
    assert np.abs(out2[:, 50] - out[:, 50]).max() > 1e-3


def test_zero_gate_is_mamba2(inp):
    """W_G = 0 (the paper's initialisation): G_t = SiLU(0) = 0, so the path output is
    the SSM readout alone and the block no longer depends on the Q and E projections."""
    W_in = inp["W_in"].copy()
    W_in[_rows("gate")] = 0.0
    out, im = _run(inp, W_in=W_in)
    p = im["path"]
    Yssd, _ = oracle.ssd_recurrence(p["X"], p["dt"], p["A"], p["Bm"], p["Cm"])
    assert np.array_equal(im["Y"], Yssd)
    W_in2 = W_in.copy()
    rng = np.random.default_rng(1)
    for name in ("Q", "E"):
        W_in2[_rows(name)] = rng.standard_normal(W_in2[_rows(name)].shape)
    out2, _ = _run(inp, W_in=W_in2)
    assert np.array_equal(out, out2)
    # and with the gate on, Q and E do matter
    out3, _ = _run(inp, W_in=np.where(np.arange(W.d_in_proj)[:, None] == _rows("gate").start, 1.0, W_in2))
    assert np.abs(out3 - out2).max() > 1e-6


def _no_ssm(inp):
    """B = 0 (its in-projection rows and conv bias zeroed): no state is written, so
    Y_ssd, the memories and R vanish and the block output comes from the D skip."""
    W_in = inp["W_in"].copy()
    W_in[_rows("B")] = 0.0
    cb = inp["conv_b"].copy()
    cb[W.d_inner:W.d_inner + W.groups * W.dstate] = 0.0
    return dict(W_in=W_in, conv_b=cb)


def test_output_norm_is_scale_invariant(inp):
    kw = _no_ssm(inp)
    out, im = _run(inp, norm_eps=1e-14, **kw)  # the invariance holds up to eps / mean square
    assert np.all(im["Y"] == 0)
    out2, _ = _run(inp, D=3.0 * inp["D"], norm_eps=1e-14, **kw)
    assert np.abs(out2 - out).max() <= 1e-9 * np.abs(out).max()


def test_output_norm_runs_over_d_inner(inp):
    """Only head 0 carries signal: normalised over all of d_inner (unit weight), its
    entries have mean square H; a per-head norm would give 1."""
    kw = _no_ssm(inp)
    D = np.zeros(W.heads)
    D[0] = 1.0
    _, im = _run(inp, D=D, norm_w=np.ones(W.d_inner), norm_eps=1e-14, **kw)
    yn = im["yn"]
    assert np.all(yn[..., W.headdim:] == 0)
    ms = np.mean(yn[..., :W.headdim] ** 2, axis=-1)
    assert np.allclose(ms, W.heads, rtol=1e-9)


def test_gate_passes_through_silu(inp):
    """Every token's input the same vector and W_G set so that the gate logit is -20:
    G = SiLU(-20) ~ -4e-8, so the readout barely moves the path output, while a
    linear gate would subtract 20 R."""
    U = np.broadcast_to(inp["U"][:1, :1], inp["U"].shape).copy()
    W_in = inp["W_in"].copy()
    W_in[_rows("gate")] = -20.0 * U[0, 0] / np.dot(U[0, 0], U[0, 0])
    _, im = _run(inp, U=U, W_in=W_in)
    p = im["path"]
    assert np.allclose(p["z"], -20.0)
    Yssd, _ = oracle.ssd_recurrence(p["X"], p["dt"], p["A"], p["Bm"], p["Cm"])
    dH = oracle.chunk_memories(p["X"], p["dt"], p["A"], p["Bm"], W.chunk)
    R, _ = oracle.sma(dH, p["Q"], p["Cm"], p["E"], W.chunk, W.eps)
    assert np.abs(R).max() > 1e-3
    assert np.abs(im["Y"] - Yssd).max() <= 1e-7 * np.abs(R).max()


def test_q_and_e_come_from_the_input_row_and_x_from_the_convolution(inp):
    """Q_t = U_t W_Q and E_t = U_t W_E (Sec. 3) read only token t; x (convolved, width 4)
    reads tokens t - 3 .. t. A change of U at one token moves Q and E at that token and
    x at it and the three after."""
    _, im = _run(inp)
    U2 = inp["U"].copy()
    U2[:, 40] += 0.5
    _, im2 = _run(inp, U=U2)
    p, p2 = im["path"], im2["path"]
    for k in ("Q", "E"):
        diff = np.abs(p2[k] - p[k]).reshape(W.batch, W.seqlen, -1).max(axis=(0, 2))
        assert np.all(diff[np.arange(W.seqlen) != 40] == 0) and diff[40] > 0, k
    dx = np.abs(p2["X"] - p["X"]).reshape(W.batch, W.seqlen, -1).max(axis=(0, 2))
    assert np.all(dx[:40] == 0) and np.all(dx[40:44] > 0) and np.all(dx[44:] == 0)


def test_in_projection_column_blocks(inp):
    """Each named row block of W_in feeds its own input of the path: changing the Q rows
    changes Q alone, changing the x rows leaves Q, E, dt and the gate alone."""
    _, im = _run(inp)
    rng = np.random.default_rng(3)
    W_q = inp["W_in"].copy()
    W_q[_rows("Q")] += rng.standard_normal(W_q[_rows("Q")].shape)
    _, iq = _run(inp, W_in=W_q)
    assert np.abs(iq["path"]["Q"] - im["path"]["Q"]).max() > 0
    for k in ("X", "Bm", "Cm", "E", "dt", "z", "zn"):
        assert np.array_equal(iq["path"][k], im["path"][k]), k
    W_x = inp["W_in"].copy()
    W_x[_rows("x")] += rng.standard_normal(W_x[_rows("x")].shape)
    _, ix = _run(inp, W_in=W_x)
    assert np.abs(ix["path"]["X"] - im["path"]["X"]).max() > 0
    for k in ("Q", "E", "dt", "z", "zn", "Bm", "Cm"):
        assert np.array_equal(ix["path"][k], im["path"][k]), k
