"""Seeded synthetic inputs for the DART hot path.

This module only draws random numbers. It holds none of the method's
arithmetic, so both the CUDA path and the CPU oracle can take their inputs
from it. Every draw uses a CPU ``torch.Generator`` so the same seed gives the
same values on any machine.

Distributions (the paper trains on text; its kernel benchmark feeds
precomputed synthetic tensors, Sec. 5.3 "Kernel Forward Time and Inference
Cache", so these stand in for that):
  X ~ N(0,1)/sqrt(P);  B, C ~ N(0,1)/sqrt(N);  Q ~ N(0,1)/sqrt(N);
  E ~ N(0,1)/sqrt(P);  dt = softplus(N(-2, 0.5)) per (b, t, h), fp32;
  A = -exp(U(0, ln 16)) per head, fp32 (so A lies in [-16, -1]);
  z (gate logit) ~ N(0,1);  upstream gradient dY ~ N(0,1).
Draw order: X, B, C, Q, E, dt, A, z, dY. bf16 workloads round X, B, C, Q, E,
z and dY to bf16 once here, so every consumer sees identical values.

Decode workloads add a cache of ``m`` chunk memories drawn N(0, 0.02^2)
(bf16) and a running state drawn N(0, 0.02^2) (fp32); each batch row's cache
slab is drawn from its own generator, so a sample of rows can be re-drawn on
its own without materialising the whole 2 GiB cache on the host.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import torch


@dataclass(frozen=True)
class Workload:
    """Sizes of one DART hot-path workload (notation of the paper)."""

    name: str
    batch: int
    heads: int
    seqlen: int
    headdim: int  # P
    dstate: int  # N
    chunk: int  # S
    groups: int = 1  # G (the paper uses G = 1 for B, C, Q, E)
    dtype: str = "bf16"  # storage type of X, B, C, Q, E, z, Y and the memories
    seed: int = 0
    eps: float = 1e-6
    # decode only
    mem: int = 0  # cached chunk memories per (b, h)
    pos: int = 0  # tokens already absorbed
    notes: str = field(default="", compare=False)

    @property
    def nchunks(self) -> int:
        return -(-self.seqlen // self.chunk)

    @property
    def tokens(self) -> int:
        return self.batch * self.seqlen

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    "tiny_fp32": Workload("tiny_fp32", 1, 2, 512, 32, 16, 64, dtype="f32", seed=1000,
                          notes="B1 H2 L512 P32 N16 S64, fp32"),
    "prefill_b4_l2k": Workload("prefill_b4_l2k", 4, 16, 2048, 64, 128, 256, seed=1001,
                               notes="B4 H16 L2048 P64 N128 S256, bf16"),
    "prefill_l16k": Workload("prefill_l16k", 1, 32, 16384, 64, 128, 256, seed=1002,
                             notes="B1 H32 L16384 P64 N128 S256, bf16, 64 chunk memories"),
    "prefill_l8k": Workload("prefill_l8k", 1, 32, 8192, 64, 128, 256, seed=1006,
                            notes="B1 H32 L8192 P64 N128 S256, bf16 (profiling size)"),
    "decode_b64": Workload("decode_b64", 64, 32, 1, 64, 128, 256, seed=1003, mem=64, pos=16384,
                           notes="B64 H32 P64 N128 S256, 64 cached memories, pos 16384"),
    "decode_b16": Workload("decode_b16", 16, 32, 1, 64, 128, 256, seed=1007, mem=64, pos=16384,
                           notes="B16 H32 P64 N128 S256, 64 cached memories (profiling size)"),
    "train_b8_l4k_s128": Workload("train_b8_l4k_s128", 8, 24, 4096, 64, 128, 128, seed=1004,
                                  notes="B8 H24 L4096 P64 N128 S128, bf16"),
    "train_b8_l4k_s256": Workload("train_b8_l4k_s256", 8, 24, 4096, 64, 128, 256, seed=1005,
                                  notes="B8 H24 L4096 P64 N128 S256, bf16"),
}


def _round(t: torch.Tensor, dtype: str) -> torch.Tensor:
    if dtype == "bf16":
        return t.to(torch.bfloat16).to(torch.float32)
    return t


def prefill_inputs(w: Workload, with_grad: bool = False) -> dict:
    """Seeded prefill inputs as CPU fp32 tensors (bf16-exact values for bf16 workloads)."""
    g = torch.Generator().manual_seed(w.seed)
    B, L, H, G, P, N = w.batch, w.seqlen, w.heads, w.groups, w.headdim, w.dstate
    X = torch.randn(B, L, H, P, generator=g) / math.sqrt(P)
    Bm = torch.randn(B, L, G, N, generator=g) / math.sqrt(N)
    Cm = torch.randn(B, L, G, N, generator=g) / math.sqrt(N)
    Q = torch.randn(B, L, G, N, generator=g) / math.sqrt(N)
    E = torch.randn(B, L, G, P, generator=g) / math.sqrt(P)
    dt = torch.nn.functional.softplus(-2.0 + 0.5 * torch.randn(B, L, H, generator=g))
    A = -torch.exp(torch.rand(H, generator=g) * math.log(16.0))
    z = torch.randn(B, L, H, generator=g)
    out = dict(X=X, Bm=Bm, Cm=Cm, Q=Q, E=E, z=z)
    out = {k: _round(v, w.dtype) for k, v in out.items()}
    out["dt"] = dt.float()
    out["A"] = A.float()
    if with_grad:
        out["dY"] = _round(torch.randn(B, L, H, P, generator=g), w.dtype)
    return out


def memory_grad_input(w: Workload, scale: float = 0.1) -> torch.Tensor:
    """Seeded gradient w.r.t. the chunk memories, ``B x M x H x N x P`` fp32 ~ N(0, scale^2)
    (drawn from its own generator, seed + 7919, after nothing else)."""
    g = torch.Generator().manual_seed(w.seed + 7919)
    return scale * torch.randn(w.batch, w.nchunks, w.heads, w.dstate, w.headdim, generator=g)


def decode_token_inputs(w: Workload) -> dict:
    """Seeded per-token decode inputs: x, dt, A, b, c, q, e, z (CPU fp32)."""
    g = torch.Generator().manual_seed(w.seed)
    B, H, G, P, N = w.batch, w.heads, w.groups, w.headdim, w.dstate
    x = torch.randn(B, H, P, generator=g) / math.sqrt(P)
    b = torch.randn(B, G, N, generator=g) / math.sqrt(N)
    c = torch.randn(B, G, N, generator=g) / math.sqrt(N)
    q = torch.randn(B, G, N, generator=g) / math.sqrt(N)
    e = torch.randn(B, G, P, generator=g) / math.sqrt(P)
    dt = torch.nn.functional.softplus(-2.0 + 0.5 * torch.randn(B, H, generator=g))
    A = -torch.exp(torch.rand(H, generator=g) * math.log(16.0))
    z = torch.randn(B, H, generator=g)
    out = {k: _round(v, w.dtype) for k, v in dict(x=x, b=b, c=c, q=q, e=e, z=z).items()}
    out["dt"] = dt.float()
    out["A"] = A.float()
    return out


def decode_cache_slab(w: Workload, b: int, m_cap: int | None = None) -> torch.Tensor:
    """Cache slab of batch row ``b``: ``m_cap x H x N x P`` memories ~ N(0, 0.02^2).

    Only the first ``w.mem`` memories are drawn; slots beyond them are zero.
    """
    m_cap = w.mem if m_cap is None else m_cap
    g = torch.Generator().manual_seed(w.seed * 1_000_003 + 7919 * (b + 1))
    slab = torch.zeros(m_cap, w.heads, w.dstate, w.headdim)
    slab[: w.mem] = 0.02 * torch.randn(w.mem, w.heads, w.dstate, w.headdim, generator=g)
    return _round(slab, w.dtype)


def decode_state_slab(w: Workload, b: int) -> torch.Tensor:
    """Running state of batch row ``b``: ``H x N x P`` fp32 ~ N(0, 0.02^2)."""
    g = torch.Generator().manual_seed(w.seed * 1_000_003 + 104_729 * (b + 1) + 1)
    return 0.02 * torch.randn(w.heads, w.dstate, w.headdim, generator=g)


def decode_partial_slab(w: Workload, b: int) -> torch.Tensor:
    """Partial-chunk memory of batch row ``b``: ``H x N x P`` fp32 ~ N(0, 0.01^2)
    (only read when ``w.pos`` is not a chunk start)."""
    g = torch.Generator().manual_seed(w.seed * 1_000_003 + 15_485_863 * (b + 1) + 2)
    return 0.01 * torch.randn(w.heads, w.dstate, w.headdim, generator=g)


def decode_state(w: Workload, m_cap: int | None = None) -> dict:
    """Whole decode state on the host: cache (Bsz x m_cap x H x N x P), state and
    partial (Bsz x H x N x P). For small workloads; large ones go slab by slab."""
    m_cap = w.mem if m_cap is None else m_cap
    return dict(
        cache=torch.stack([decode_cache_slab(w, b, m_cap) for b in range(w.batch)]),
        state=torch.stack([decode_state_slab(w, b) for b in range(w.batch)]),
        partial=torch.stack([decode_partial_slab(w, b) for b in range(w.batch)]),
    )


# ---------------------------------------------------------------- whole block
@dataclass(frozen=True)
class BlockWorkload:
    """Sizes of one DART block (the hot path inside a Mamba-2 style block): d_inner =
    H P, in-projection of width 2 d_inner + 3 G N + H + G P + 1."""

    name: str
    batch: int
    seqlen: int
    d_model: int
    heads: int
    headdim: int = 64  # P
    dstate: int = 128  # N
    chunk: int = 256  # S
    groups: int = 1
    conv: int = 4  # convolution width
    seed: int = 0
    eps: float = 1e-6  # RMSNorm of Q, E and the memory rows
    norm_eps: float = 1e-5  # the gated output RMSNorm
    notes: str = field(default="", compare=False)

    @property
    def d_inner(self) -> int:
        return self.heads * self.headdim

    @property
    def d_in_proj(self) -> int:
        G, N, P = self.groups, self.dstate, self.headdim
        return 2 * self.d_inner + 3 * G * N + self.heads + G * P + 1

    @property
    def tokens(self) -> int:
        return self.batch * self.seqlen


BLOCK_WORKLOADS = {
    # the DART 380M block shape (d_model 1024, expand 2: 32 heads of 64) at L = 16K
    "block_l16k": BlockWorkload("block_l16k", 1, 16384, 1024, 32, seed=1010,
                                notes="B1 L16384 d_model 1024 H32 P64 N128 S256, bf16"),
    "block_small": BlockWorkload("block_small", 2, 512, 256, 8, chunk=128, seed=1011,
                                 notes="B2 L512 d_model 256 H8 P64 N128 S128, bf16"),
}


def block_inputs(w: BlockWorkload) -> dict:
    """Seeded block input and weights as CPU fp32 tensors (U, W_in and W_out bf16-exact).

    U ~ N(0, 1); the in-projection rows ~ N(0, 1/d_model), except the dt rows ~
    N(0, 0.25/d_model) (with dt_bias ~ N(-2, 0.1^2) the step size is softplus of
    about N(-2, 0.5^2), as in the hot-path workloads); conv_w, conv_b ~
    U(-1/sqrt(width), 1/sqrt(width)); A_log ~ U(0, ln 16); D ~ N(1, 0.1^2);
    norm_w ~ N(1, 0.1^2); W_out ~ N(0, 1/d_inner). Draw order: U, W_in, conv_w,
    conv_b, dt_bias, A_log, D, norm_w, W_out.
    """
    g = torch.Generator().manual_seed(w.seed)
    d, di, H = w.d_model, w.d_inner, w.heads
    conv_ch = di + 2 * w.groups * w.dstate
    U = torch.randn(w.batch, w.seqlen, d, generator=g)
    W_in = torch.randn(w.d_in_proj, d, generator=g) / math.sqrt(d)
    dt0 = 2 * di + 2 * w.groups * w.dstate  # first dt row
    W_in[dt0:dt0 + H] *= 0.5
    bound = 1.0 / math.sqrt(w.conv)
    conv_w = (torch.rand(conv_ch, w.conv, generator=g) * 2 - 1) * bound
    conv_b = (torch.rand(conv_ch, generator=g) * 2 - 1) * bound
    dt_bias = -2.0 + 0.1 * torch.randn(H, generator=g)
    A_log = torch.rand(H, generator=g) * math.log(16.0)
    D = 1.0 + 0.1 * torch.randn(H, generator=g)
    norm_w = 1.0 + 0.1 * torch.randn(di, generator=g)
    W_out = torch.randn(d, di, generator=g) / math.sqrt(di)
    return dict(U=_round(U, "bf16"), W_in=_round(W_in, "bf16"), conv_w=conv_w, conv_b=conv_b,
                dt_bias=dt_bias, A_log=A_log, D=D, norm_w=norm_w, W_out=_round(W_out, "bf16"))
