"""Checks that pin the oracle's FEM read over a GLA prior (App. "Gated Linear
Attention (GLA) Prior") to what the paper and the mathematics fix:

  L1  no decay and constant features: the prior is uniform over i <= t, so
      F = (logsumexp_{i<=t}(beta v_i) - log(t + 1))/beta (scipy)
  L2  beta = 0: the prior mean equals the streaming ratio of Eq. "gla-assoc",
      <D_t qf_t, A_t> / <D_t qf_t, B_t> with A_t = sum_r D_r^-1 kf_r v_r and
      B_t = sum_r D_r^-1 kf_r accumulated step by step in numpy
  L3  the first step sees one key: F = v_0 for every beta
  L4  strong decay (g = -60): the prior sits on i = t, so F = v_t
  L5  keys and values after t do not change row t (the mask, Eq. "gla-score-appendix")
  L6  log Z_t from the streaming normaliser <D_t qf_t, B_t>
"""
from __future__ import annotations

import numpy as np
from scipy.special import logsumexp

import oracle


def _inputs(seed, B, H, T, m, d, g_scale=0.3, beta_lo=0.05, beta_hi=20.0):
    r = np.random.default_rng(seed)
    qf = np.maximum(r.standard_normal((B, H, T, m)), 0.0) + 0.05
    kf = np.maximum(r.standard_normal((B, H, T, m)), 0.0) + 0.05
    v = r.standard_normal((B, H, T, d))
    g = -g_scale * r.uniform(0.0, 1.0, size=(B, H, T))
    beta = np.exp(r.uniform(np.log(beta_lo), np.log(beta_hi), size=(H, d)))
    return qf, kf, v, g, beta


def check_l1_uniform(lib=None):
    qf, kf, v, g, beta = _inputs(41, 1, 2, 9, 4, 5)
    qf[:] = 1.0
    kf[:] = 1.0
    g[:] = 0.0
    out, _ = oracle.gla_read(qf, kf, v, g, beta)
    for t in range(9):
        for h in range(2):
            ref = (logsumexp(beta[h][None, :] * v[0, h, : t + 1], axis=0) - np.log(t + 1)) / beta[h]
            assert np.allclose(out[0, h, t], ref, rtol=0, atol=1e-12)


def check_l2_mean_is_streaming_ratio(lib=None):
    qf, kf, v, g, beta = _inputs(42, 2, 2, 12, 6, 4)
    beta[:] = 0.0
    out, _ = oracle.gla_read(qf, kf, v, g, beta)
    B, H, T, m = qf.shape
    for b in range(B):
        for h in range(H):
            A = np.zeros((m, v.shape[-1]))
            Bs = np.zeros(m)
            G = 0.0
            for t in range(T):
                G += g[b, h, t]
                A += np.exp(-G) * np.outer(kf[b, h, t], v[b, h, t])
                Bs += np.exp(-G) * kf[b, h, t]
                num = np.exp(G) * qf[b, h, t] @ A
                den = np.exp(G) * qf[b, h, t] @ Bs
                assert np.allclose(out[b, h, t], num / den, rtol=0, atol=1e-10)


def check_l3_first_step(lib=None):
    qf, kf, v, g, beta = _inputs(43, 1, 3, 5, 4, 6)
    out, _ = oracle.gla_read(qf, kf, v, g, beta)
    assert np.allclose(out[:, :, 0], v[:, :, 0], rtol=0, atol=1e-12)


def check_l4_strong_decay(lib=None):
    qf, kf, v, g, beta = _inputs(44, 1, 2, 7, 4, 5, beta_lo=0.5, beta_hi=5.0)
    g[:] = -60.0
    out, _ = oracle.gla_read(qf, kf, v, g, beta)
    assert np.allclose(out, v, rtol=0, atol=1e-9)


def check_l5_mask(lib=None):
    qf, kf, v, g, beta = _inputs(45, 1, 2, 10, 4, 3)
    out, lz = oracle.gla_read(qf, kf, v, g, beta)
    kf2, v2 = kf.copy(), v.copy()
    kf2[:, :, 6:] *= 3.0
    v2[:, :, 6:] += 5.0
    out2, lz2 = oracle.gla_read(qf, kf2, v2, g, beta)
    assert np.array_equal(out[:, :, :6], out2[:, :, :6]) and np.array_equal(lz[:, :, :6], lz2[:, :, :6])


def check_l6_log_normaliser(lib=None):
    qf, kf, v, g, beta = _inputs(46, 1, 2, 8, 5, 3)
    _, lz = oracle.gla_read(qf, kf, v, g, beta)
    for h in range(2):
        Bs = np.zeros(5)
        G = 0.0
        for t in range(8):
            G += g[0, h, t]
            Bs += np.exp(-G) * kf[0, h, t]
            assert abs(lz[0, h, t] - np.log(np.exp(G) * qf[0, h, t] @ Bs)) < 1e-12


ALL_CHECKS = [check_l1_uniform, check_l2_mean_is_streaming_ratio, check_l3_first_step, check_l4_strong_decay,
              check_l5_mask, check_l6_log_normaliser]
