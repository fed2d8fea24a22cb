"""Checks that pin the oracle's two-level gated read (Sec. 3, "Two-Level
Gated FEM") to what the paper and the mathematics fix:

  G1  lambda = 0, g = 1: the read is the prior mean mu_t = sum_i p_t(i) v_i,
      i.e. softmax attention, formed here with numpy (Eq. "inner-gate-main")
  G2  lambda = 1, g = 1: the read is Fmax, checked against the one-pass form
      of App. "One-pass implementation": (1/beta) log sum_i p_t(i)
      exp(beta v_i) from the numpy prior, a different evaluation path from the
      oracle's difference of log-sum-exps
  G3  general gates: out = g ((1 - lambda) mu + lambda Fmax) with mu and Fmax
      from G1/G2 (Eqs. "inner-gate-main", "fem-two-gates-main")
  G4  hidden temperature (Prop. "ltl-hidden", App. "fem-ltl"): for lambda in
      (0, 1) the inner read equals F(beta*) at a unique beta* in [0, beta_max],
      increasing in lambda, and KL(p || q^(beta*))/beta* = lambda
      KL(p || q^(beta_max))/beta_max (the fraction of the achievable KL
      improvement, with F(beta) - mu = KL(p || q^(beta))/beta)

mu, Fmax, priors and KL terms are formed with numpy from the inputs, never
from the oracle (except F(beta) inside the G4 bisection, which is the read
the proposition is about).
"""
from __future__ import annotations

import numpy as np
from scipy.special import logsumexp

import oracle
from tests.oracle_pins import _inputs, _prior


def _gates(seed, shape):
    r = np.random.default_rng(seed)
    lam = r.uniform(0.0, 1.0, size=shape)
    g = np.log1p(np.exp(r.standard_normal(shape)))  # softplus, > 0
    g = g / np.sqrt((g * g).mean(axis=-1, keepdims=True))  # RMS-normalised over channels
    return lam, g


def _mu_np(p, v):
    return np.einsum("bhti,bhij->bhtj", p, v)


def _fmax_np(p, v, beta):
    # (1/beta_j) log sum_i p_i exp(beta_j v_ij), per (b, h, t, j), via log p + beta v
    with np.errstate(divide="ignore"):
        logp = np.log(p)  # -inf off the support
    B, H, T, d = v.shape
    out = np.empty((B, H, T, d))
    for h in range(H):
        for j in range(d):
            a = logp[:, h] + beta[h, j] * v[:, h, None, :, j]  # [B, T, T]
            out[:, h, :, j] = logsumexp(a, axis=-1) / beta[h, j]
    return out


def check_g1_mean_branch(lib):
    for causal in (True, False):
        q, k, v, bmax = _inputs(21, 2, 2, 9, 5, beta_lo=0.05, beta_hi=20)
        shape = q.shape
        out, _ = oracle.gated_read(q, k, v, bmax, np.zeros(shape), np.ones(shape), causal, nthreads=1, lib=lib)
        p, _ = _prior(q, k, causal)
        assert np.allclose(out, _mu_np(p, v), rtol=0, atol=1e-12), np.abs(out - _mu_np(p, v)).max()


def check_g2_max_branch(lib):
    for causal in (True, False):
        q, k, v, bmax = _inputs(22, 1, 3, 8, 4, beta_lo=0.05, beta_hi=20)
        shape = q.shape
        out, _ = oracle.gated_read(q, k, v, bmax, np.ones(shape), np.ones(shape), causal, nthreads=1, lib=lib)
        p, _ = _prior(q, k, causal)
        ref = _fmax_np(p, v, bmax)
        assert np.allclose(out, ref, rtol=0, atol=1e-10), np.abs(out - ref).max()


def check_g3_gates(lib):
    for causal in (True, False):
        q, k, v, bmax = _inputs(23, 2, 2, 7, 6, beta_lo=0.05, beta_hi=20)
        lam, g = _gates(5, q.shape)
        out, lse = oracle.gated_read(q, k, v, bmax, lam, g, causal, nthreads=1, lib=lib)
        p, s = _prior(q, k, causal)
        ref = g * ((1 - lam) * _mu_np(p, v) + lam * _fmax_np(p, v, bmax))
        assert np.allclose(out, ref, rtol=0, atol=1e-10), np.abs(out - ref).max()
        assert np.allclose(lse, logsumexp(s, axis=-1), rtol=0, atol=1e-12)


def check_g4_hidden_temperature(lib):
    q, k, v, bmax = _inputs(24, 1, 1, 6, 3, beta_lo=0.5, beta_hi=8)
    causal = True
    p, _ = _prior(q, k, causal)
    t = 5  # a row with six visible keys
    pt = p[0, 0, t, : t + 1]
    ones = np.ones(q.shape)

    def F(beta_scalar, j):
        beta = np.full(bmax.shape, beta_scalar)
        out, _ = oracle.fem_read(q, k, v, beta, causal, nthreads=1, lib=lib)
        return out[0, 0, t, j]

    def kl_over_beta(beta, j):
        # KL(p || q^(beta)) / beta with q^(beta) proportional to p exp(beta v), in numpy
        vj = v[0, 0, : t + 1, j]
        logq = np.log(pt) + beta * vj - logsumexp(np.log(pt) + beta * vj)
        return float(np.sum(pt * (np.log(pt) - logq)) / beta)

    for j in range(3):
        mu = float(pt @ v[0, 0, : t + 1, j])
        fm = F(bmax[0, j], j)
        assert fm > mu  # Jensen, non-constant channel
        prev = 0.0
        for lam_s in (0.1, 0.35, 0.6, 0.9):
            lam = np.full(q.shape, lam_s)
            target = oracle.gated_read(q, k, v, bmax, lam, ones, causal, nthreads=1, lib=lib)[0][0, 0, t, j]
            lo, hi = 0.0, float(bmax[0, j])
            for _ in range(80):  # F is strictly increasing in beta (Thm. "fem-main")
                mid = 0.5 * (lo + hi)
                lo, hi = (mid, hi) if F(mid, j) < target else (lo, mid)
            bstar = 0.5 * (lo + hi)
            assert abs(F(bstar, j) - target) < 1e-9
            assert prev < bstar < bmax[0, j]
            prev = bstar
            assert abs(kl_over_beta(bstar, j) - lam_s * kl_over_beta(float(bmax[0, j]), j)) < 1e-8


ALL_CHECKS = [check_g1_mean_branch, check_g2_max_branch, check_g3_gates, check_g4_hidden_temperature]
