"""Seeded synthetic inputs for the Free Energy Mixer read.

This module only draws random numbers: it holds none of the read's
arithmetic, and both the CUDA path and the float64 oracle consume what it
returns.  All draws come from one CPU ``torch.Generator`` per call, in the
order Q, K, V, beta, so a (workload, seed) pair fixes every input.

Shapes follow the paper's uses of the read: Q, K, V are [B, H, T, d] (one d for
queries, keys and values, the score scale of Sec. 1), beta is the per-head,
per-channel inverse temperature [H, d] (the per-channel beta_max of Sec.
2.3.2).  beta is drawn log-uniformly so every workload spans the averaging
regime (small beta) and the selecting regime (large beta).
"""
from __future__ import annotations

import dataclasses
import math

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    T: int
    d: int
    causal: bool
    dtype: str               # "bf16" or "f32": the element type of Q, K, V
    beta_lo: float
    beta_hi: float
    v_dist: str = "normal"   # "normal" or "student_t3"
    const_channels: int = 0  # channels 0..n-1 of every (b, h) held constant over t

    @property
    def flops(self) -> float:
        """Flash-attention FLOP count of the read: 4*B*H*T*T*d, halved when causal."""
        f = 4.0 * self.B * self.H * self.T * self.T * self.d
        return f / 2 if self.causal else f

    def describe(self) -> dict:
        return {"workload": self.name, "B": self.B, "H": self.H, "T": self.T, "d": self.d,
                "causal": self.causal, "in_dtype": self.dtype,
                "beta": f"log-uniform[{self.beta_lo:g},{self.beta_hi:g}]", "v": self.v_dist,
                "const_channels": self.const_channels}


# The five synthetic workloads.  The ViT-S one borrows only the shape of a
# ViT-S/16 image transformer (197 tokens, 6 heads of 64); nothing of a dataset.
WORKLOADS = {
    w.name: w
    for w in [
        Workload("tiny_f32_causal", 1, 1, 64, 16, True, "f32", 0.1, 10.0),
        Workload("vit_s_full_prior", 64, 6, 197, 64, False, "bf16", 0.05, 20.0),
        Workload("lm_causal_d64", 8, 12, 2048, 64, True, "bf16", 0.05, 20.0),
        Workload("lm_causal_d128", 4, 16, 8192, 128, True, "bf16", 0.05, 20.0),
        Workload("long_causal_student_t", 1, 32, 32768, 128, True, "bf16", 1e-3, 100.0,
                 v_dist="student_t3", const_channels=4),
    ]
}

HEADLINE = "lm_causal_d128"


def _normal(gen: torch.Generator, shape) -> torch.Tensor:
    return torch.randn(shape, generator=gen, dtype=torch.float32)


def _student_t3_unit_var(gen: torch.Generator, shape) -> torch.Tensor:
    """Student-t with 3 degrees of freedom scaled to unit variance.

    t = Z / sqrt(X / 3) with Z ~ N(0,1) and X ~ chi^2_3 = sum of three squared
    standard normals; Var(t) = 3, so the draw is divided by sqrt(3)."""
    z = _normal(gen, shape)
    x = _normal(gen, shape).square_()
    x += _normal(gen, shape).square_()
    x += _normal(gen, shape).square_()
    return z.div_(x.div_(3.0).sqrt_()).div_(math.sqrt(3.0))


def make_inputs(w: Workload, seed: int = 0, T: int | None = None, B: int | None = None,
                H: int | None = None):
    """Draw (q, k, v, beta) for workload ``w`` on the CPU.

    q, k, v are [B, H, T, d] in the workload's element type (bf16 or fp32),
    contiguous; beta is [H, d] float32.  ``T``/``B``/``H`` override the sizes
    (for reduced parity cases with the same distributions)."""
    B = w.B if B is None else B
    H = w.H if H is None else H
    T = w.T if T is None else T
    gen = torch.Generator(device="cpu").manual_seed(seed)
    q, k, v = _draw_qkv(gen, w, (B, H, T, w.d))
    beta = _draw_beta(gen, w, H)
    dt = _dtype(w)
    return q.to(dt).contiguous(), k.to(dt).contiguous(), v.to(dt).contiguous(), beta.contiguous()


def _draw_qkv(gen: torch.Generator, w: Workload, shape):
    q = _normal(gen, shape)
    k = _normal(gen, shape)
    if w.v_dist == "normal":
        v = _normal(gen, shape)
    elif w.v_dist == "student_t3":
        v = _student_t3_unit_var(gen, shape)
    else:
        raise ValueError(w.v_dist)
    if w.const_channels:
        c = w.const_channels
        v[..., :c] = v[..., :1, :c]
    return q, k, v


def _draw_beta(gen: torch.Generator, w: Workload, H: int) -> torch.Tensor:
    u = torch.rand((H, w.d), generator=gen, dtype=torch.float64)
    return torch.exp(math.log(w.beta_lo) + u * (math.log(w.beta_hi) - math.log(w.beta_lo))).float()


def _dtype(w: Workload):
    return torch.bfloat16 if w.dtype == "bf16" else torch.float32


def make_batch_shard(w: Workload, rank: int, world: int, seed: int = 0):
    """Rank ``rank``'s share of one global batch of ``world * w.B`` sequences.

    The read is independent per (b, h), so the global batch shards over the batch
    dimension with no exchange: rank r holds sequences r*B .. r*B + B - 1, each drawn
    from its own generator (seeded by ``seed`` and the sequence's global index), and
    every rank draws the same beta [H, d] (from the generator seeded by ``seed``).  The
    shards of all ranks, concatenated over the batch, are exactly
    ``make_batch_shard(w with B = world * w.B, 0, 1, seed)``."""
    if not 0 <= rank < world:
        raise ValueError("rank out of range")
    shape = (1, w.H, w.T, w.d)
    parts = []
    for b in range(rank * w.B, (rank + 1) * w.B):
        gen = torch.Generator(device="cpu").manual_seed((seed * 1_000_003 + 1 + b) % (1 << 63))
        parts.append(_draw_qkv(gen, w, shape))
    beta = _draw_beta(torch.Generator(device="cpu").manual_seed(seed), w, w.H)
    dt = _dtype(w)
    q, k, v = (torch.cat([p[i] for p in parts]).to(dt).contiguous() for i in range(3))
    return q, k, v, beta.contiguous()


def make_custom(B: int, H: int, T: int, d: int, *, dtype: str = "bf16", beta_lo: float = 0.05,
                beta_hi: float = 20.0, seed: int = 0, v_dist: str = "normal", const_channels: int = 0):
    """Inputs of an arbitrary shape drawn with the same recipe."""
    w = Workload("custom", B, H, T, d, True, dtype, beta_lo, beta_hi, v_dist, const_channels)
    return make_inputs(w, seed=seed)


def beta_grid(H: int, d: int, values) -> torch.Tensor:
    """beta [H, d] cycling through ``values`` along the channels (for beta sweeps)."""
    vals = torch.tensor(list(values), dtype=torch.float32)
    idx = torch.arange(H * d) % vals.numel()
    return vals[idx].reshape(H, d).contiguous()
