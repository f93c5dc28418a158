"""CPU oracle of one whole DART block -- TEST INFRASTRUCTURE.

The hot path (scan, chunk memories, state-memory attention, merge) comes from
``oracle`` (plain fp64 C); this module adds the steps of the block around it,
in fp64 numpy, each from its plain definition. The paper (Sec. 3) forms Q, E
and the gate from the block input U_t, shares C with the SSM branch and adds
the gated SMA readout to the SSM readout, Y_t = C_t H_t + G_t R_t; for the rest
it follows the Mamba-2 block (App. D.2: head dimension 64, one shared B, C
group, convolution width 4, RMSNorm). Readings where the paper says no more:

  * in-projection columns, in this order: z (d_inner), x (d_inner), B (G N),
    C (G N), dt (H), Q (G N), E (G P), gate (1);
  * the causal depthwise convolution and SiLU act on x, B and C (Mamba-2's
    xBC), not on Q, E or the gate (the paper writes Q_t = U_t W_Q, E_t = U_t W_E);
  * dt = softplus(dt_raw + dt_bias), A = -exp(A_log);
  * one gate logit per token, shared by the heads (App. D.2, "a scalar SMA
    residual gate per token"): G_t = SiLU(U_t W_G);
  * D skip after the merge: y = C_t H_t + G_t R_t + D_h x_t;
  * gated RMSNorm over d_inner: RMSNorm(y * SiLU(z)) * w, then the
    out-projection;
  * precision of the hot path's token inputs: with ``path_dtype="bf16"`` the
    x, B, C (after the convolution), Q, E and gate logits are rounded to bf16
    (round to nearest even) before the scan and SMA, the storage type of the
    bf16 configuration's token inputs; everything else stays fp64.

Weights use ``nn.Linear`` layouts: W_in (D_in x d_model), W_out (d_model x
d_inner), conv_w (conv channels x width), the tap k multiplying x[t - width + 1 + k].
Only tests/, the smoke check and bench.py's CPU legs import this module.
"""
from __future__ import annotations

import numpy as np

import oracle


def _f64(a):
    if hasattr(a, "detach"):
        a = a.detach().cpu().double().numpy()
    return np.ascontiguousarray(a, dtype=np.float64)


def in_proj_width(d_inner: int, H: int, G: int, N: int, P: int) -> int:
    """Columns of the in-projection: z, x, B, C, dt, Q, E, gate."""
    return 2 * d_inner + 2 * G * N + H + G * N + G * P + 1


def split_in_proj(zx, d_inner: int, H: int, G: int, N: int, P: int) -> dict:
    """The in-projection output (``... x D_in``) cut into its named column blocks."""
    sizes = [("z", d_inner), ("x", d_inner), ("B", G * N), ("C", G * N), ("dt", H), ("Q", G * N),
             ("E", G * P), ("gate", 1)]
    out, o = {}, 0
    for name, n in sizes:
        out[name] = zx[..., o:o + n]
        o += n
    assert o == zx.shape[-1]
    return out


def silu(v):
    return v / (1.0 + np.exp(-v))


def softplus(v):
    return np.logaddexp(0.0, v)


def causal_conv(xs, w, b):
    """Depthwise causal convolution along tokens: out[t, ch] = b[ch] + sum_k w[ch, k]
    xs[t - W + 1 + k, ch], with zeros before the first token. xs: Bsz x L x C."""
    xs, w, b = _f64(xs), _f64(w), _f64(b)
    Bsz, L, Cc = xs.shape
    W = w.shape[1]
    out = np.broadcast_to(b, xs.shape).copy()
    for k in range(W):
        shift = W - 1 - k  # tap k reads the token `shift` steps back
        if shift >= L:
            continue
        out[:, shift:, :] += w[:, k] * xs[:, : L - shift, :]
    return out


def rms_norm_gated(y, z, w, eps: float):
    """RMSNorm(y * SiLU(z)) * w over the last axis."""
    g = _f64(y) * silu(_f64(z))
    return g / np.sqrt(np.mean(g * g, axis=-1, keepdims=True) + eps) * _f64(w)


def _bf16(a):
    """Round to bf16 (nearest even), back in fp64."""
    import torch

    return torch.from_numpy(np.ascontiguousarray(a)).to(torch.bfloat16).double().numpy()


def block_inputs_to_path(U, W_in, conv_w, conv_b, dt_bias, A_log, H: int, G: int, N: int, P: int,
                         path_dtype: str = "f64"):
    """The in-projection, the convolution and the step-size / decay parameters: the
    inputs of the hot path (X, dt, A, B, C, Q, E, gate logits per head) and z.
    ``path_dtype="bf16"`` rounds X, B, C, Q, E and the gate logits to bf16."""
    U, W_in = _f64(U), _f64(W_in)
    Bsz, L, _ = U.shape
    d_inner = H * P
    zx = U @ W_in.T
    parts = split_in_proj(zx, d_inner, H, G, N, P)
    xBC = np.concatenate([parts["x"], parts["B"], parts["C"]], axis=-1)
    xBC = silu(causal_conv(xBC, conv_w, conv_b))
    X = xBC[..., :d_inner].reshape(Bsz, L, H, P)
    Bm = xBC[..., d_inner:d_inner + G * N].reshape(Bsz, L, G, N)
    Cm = xBC[..., d_inner + G * N:].reshape(Bsz, L, G, N)
    dt = softplus(parts["dt"] + _f64(dt_bias))
    A = -np.exp(_f64(A_log))
    Q = parts["Q"].reshape(Bsz, L, G, N)
    E = parts["E"].reshape(Bsz, L, G, P)
    gate = np.broadcast_to(parts["gate"], (Bsz, L, H)).copy()  # one logit per token, every head
    if path_dtype == "bf16":
        X, Bm, Cm, Q, E, gate = (_bf16(a) for a in (X, Bm, Cm, Q, E, gate))
    else:
        assert path_dtype == "f64", path_dtype
    return dict(X=X, dt=dt, A=A, Bm=Bm, Cm=Cm, Q=Q, E=E, z=gate, zn=parts["z"])


def block_forward(U, W_in, conv_w, conv_b, dt_bias, A_log, D, norm_w, W_out, H: int, G: int, N: int,
                  P: int, S: int, eps: float, norm_eps: float, path=None, path_dtype: str = "f64"):
    """Whole DART block for a prefill: returns (out ``Bsz x L x d_model``, intermediates).

    ``path``: optional replacement of the hot-path result Y (``Bsz x L x H x P``),
    for tests that pin the surrounding steps alone.
    """
    p = block_inputs_to_path(U, W_in, conv_w, conv_b, dt_bias, A_log, H, G, N, P, path_dtype)
    if path is None:
        Yssd, _ = oracle.ssd_recurrence(p["X"], p["dt"], p["A"], p["Bm"], p["Cm"])
        dH = oracle.chunk_memories(p["X"], p["dt"], p["A"], p["Bm"], S)
        R, lse = oracle.sma(dH, p["Q"], p["Cm"], p["E"], S, eps)
        Y = oracle.merge(Yssd, p["z"], R)
    else:
        Y = _f64(path)
    Bsz, L = Y.shape[0], Y.shape[1]
    y = Y + _f64(D)[None, None, :, None] * p["X"]  # D skip
    yn = rms_norm_gated(y.reshape(Bsz, L, H * P), p["zn"], norm_w, norm_eps)
    out = yn @ _f64(W_out).T
    return out, dict(path=p, Y=Y, y=y, yn=yn)
