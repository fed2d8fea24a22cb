"""Checks that pin the float64 oracle to what the paper and the mathematics fix.

Every check takes an oracle library handle (``oracle.load()`` or a deliberately
mutated build of it) and raises AssertionError when the oracle disagrees with
the fact it encodes.  The facts come from the paper's statements about the
read F_{t,j}(beta) = (1/beta) log sum_i p_t(i) exp(beta v_{i,j}):

  P1  one-key support (causal row 0): F = v_0 exactly (Sec. 2.3 definition)
  P2  constant channel: F = const for every beta (Thm. "fem-main": F is
      strictly increasing unless v is p-a.s. constant; Prop. "app-bounds" range)
  P3  mu <= F <= v*, v* + log p(i*)/beta <= F, and F = mu at beta = 0
      (Prop. "app-bounds"; the beta -> 0 limit of Prop. "app-baseline")
  P4  small beta: F = mu + beta/2 Var_p(v) + O(beta^2), and F - mu =
      KL(p || q)/beta (Prop. "app-baseline", Eq. "fem-fixed")
  P5  monotone in beta with dF/dbeta = KL(q || p)/beta^2 (Eq. "app-beta-deriv")
  P6  shift and scale laws (Prop. "app-prior" (ii))
  P7  uniform prior: F = (logsumexp(beta v) - log n)/beta, against scipy
  P8  50-digit brute force on tiny shapes (stored golden values written by
      oracle/make_golden.py, and live mpmath where it is installed)
  P9  channel-wise argmax toy data (App. "toy-argmax"): with a uniform prior
      over T = 128 keys and beta = 100, F = v* - ln(128)/100 to 1e-12
  P10 mask preservation (Prop. "app-prior" (i)) and key-permutation invariance
  P11 invariance of the softmax prior under a common rotation of q and k
  P12 concentration at large beta (Prop. "app-bounds"): |F - v*| <= -log p(i*)/beta
  P13 lse_t = LSE_i s_{t,i} (checked with the scores formed by numpy)

Everything that the checks compute themselves (mu, variances, KL terms,
maxima, scores) is formed with numpy from the inputs, never from the oracle.
"""
from __future__ import annotations

import json
import os

import numpy as np
from scipy.special import logsumexp

import oracle

GOLDEN_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rng(seed):
    return np.random.default_rng(seed)


def _inputs(seed, B, H, T, d, beta=None, beta_lo=1e-3, beta_hi=1e3, v_scale=1.0):
    r = _rng(seed)
    q = r.standard_normal((B, H, T, d))
    k = r.standard_normal((B, H, T, d))
    v = r.standard_normal((B, H, T, d)) * v_scale
    if beta is None:
        beta = np.exp(r.uniform(np.log(beta_lo), np.log(beta_hi), size=(H, d)))
    return q, k, v, np.broadcast_to(np.asarray(beta, dtype=np.float64), (H, d)).copy()


def _prior(q, k, causal):
    """numpy softmax prior p[b,h,t,i] (zero outside the support) and scores."""
    d = q.shape[-1]
    s = np.einsum("bhtc,bhic->bhti", q, k) / np.sqrt(d)
    T = q.shape[2]
    if causal:
        mask = np.tril(np.ones((T, T), dtype=bool))
        s = np.where(mask, s, -np.inf)
    p = np.exp(s - s.max(-1, keepdims=True))
    p /= p.sum(-1, keepdims=True)
    return p, s


def _visible_max(v, causal):
    """v*[b,h,t,j] = max over the support of v[b,h,i,j], and its index."""
    if causal:
        vm = np.maximum.accumulate(v, axis=2)
        T = v.shape[2]
        arg = np.zeros(v.shape, dtype=np.int64)
        for t in range(T):
            arg[:, :, t, :] = np.argmax(v[:, :, : t + 1, :], axis=2)
        return vm, arg
    vm = np.broadcast_to(v.max(axis=2, keepdims=True), v.shape)
    arg = np.broadcast_to(np.argmax(v, axis=2)[:, :, None, :], v.shape)
    return vm, arg


def _run(lib, q, k, v, beta, causal):
    return oracle.fem_read(q, k, v, beta, causal, nthreads=1, lib=lib)


def check_p1_single_key(lib):
    q, k, v, beta = _inputs(1, 2, 3, 7, 5)
    beta[:, 0] = 0.0
    out, _ = _run(lib, q, k, v, beta, True)
    np.testing.assert_allclose(out[:, :, 0, :], v[:, :, 0, :], rtol=0, atol=1e-12)


def check_p2_constant_channel(lib):
    q, k, v, beta = _inputs(2, 1, 2, 9, 6)
    const = np.array([0.37, -1.5, 2.25])
    v[..., :3] = const
    beta[:, 0] = 0.0
    beta[:, 1] = 100.0
    beta[:, 2] = 1e-3
    for causal in (True, False):
        out, _ = _run(lib, q, k, v, beta, causal)
        np.testing.assert_allclose(out[..., :3], np.broadcast_to(const, out[..., :3].shape), rtol=0, atol=1e-12)


def check_p3_bounds(lib):
    q, k, v, beta = _inputs(3, 2, 2, 11, 8)
    beta[:, 0] = 0.0
    for causal in (True, False):
        out, _ = _run(lib, q, k, v, beta, causal)
        p, _ = _prior(q, k, causal)
        mu = np.einsum("bhti,bhij->bhtj", p, v)
        vstar, istar = _visible_max(v, causal)
        pstar = np.take_along_axis(p, np.ascontiguousarray(istar), axis=3)
        b = np.broadcast_to(beta[None, :, None, :], out.shape)
        tol = 1e-11
        assert np.all(out >= mu - tol), "F below the prior mean (Jensen bound)"
        assert np.all(out <= vstar + tol), "F above the visible maximum"
        pos = b > 0
        lower = vstar + np.log(pstar) / np.where(pos, b, 1.0)
        assert np.all(out[pos] >= lower[pos] - tol), "F below v* + log p(i*)/beta"
        np.testing.assert_allclose(out[..., 0], mu[..., 0], rtol=0, atol=1e-12)


def check_p4_small_beta(lib):
    q, k, v, _ = _inputs(4, 1, 2, 10, 5)
    H, d = 2, 5
    for causal in (True, False):
        p, _ = _prior(q, k, causal)
        mu = np.einsum("bhti,bhij->bhtj", p, v)
        var = np.einsum("bhti,bhij->bhtj", p, v * v) - mu * mu
        dev = np.abs(v[:, :, None, :, :] - mu[:, :, :, None, :]).max(axis=3)
        for bval in (1e-4, 1e-3):
            out, _ = _run(lib, q, k, v, np.full((H, d), bval), causal)
            resid = np.abs(out - mu - 0.5 * bval * var)
            bound = bval * bval * dev ** 3 / 6.0 * 1.5 + 1e-11
            assert np.all(resid <= bound), "small-beta expansion mu + beta/2 Var violated"
        for bval in (0.3, 2.0, 9.0):
            out, _ = _run(lib, q, k, v, np.full((H, d), bval), causal)
            w = p[..., None] * np.exp(bval * (v[:, :, None, :, :] - v.max(axis=2)[:, :, None, None, :]))
            qpost = w / w.sum(axis=3, keepdims=True)
            with np.errstate(divide="ignore", invalid="ignore"):
                term = np.where(p[..., None] > 0, p[..., None] * (np.log(p[..., None]) - np.log(qpost)), 0.0)
            kl = term.sum(axis=3)
            np.testing.assert_allclose(out - mu, kl / bval, rtol=1e-9, atol=1e-11)


def check_p5_monotone_and_derivative(lib):
    q, k, v, _ = _inputs(5, 1, 1, 8, 4)
    grid = np.geomspace(1e-2, 1e2, 25)
    causal = True
    outs = np.stack([_run(lib, q, k, v, np.full((1, 4), g), causal)[0] for g in grid])
    assert np.all(np.diff(outs, axis=0) >= -1e-12), "F not non-decreasing in beta"
    p, _ = _prior(q, k, causal)
    for bval in (0.2, 1.5, 6.0):
        h = 1e-5
        fp = _run(lib, q, k, v, np.full((1, 4), bval * (1 + h)), causal)[0]
        fm = _run(lib, q, k, v, np.full((1, 4), bval * (1 - h)), causal)[0]
        fd = (fp - fm) / (2 * bval * h)
        w = p[..., None] * np.exp(bval * (v[:, :, None, :, :] - v.max(axis=2)[:, :, None, None, :]))
        qpost = w / w.sum(axis=3, keepdims=True)
        with np.errstate(divide="ignore", invalid="ignore"):
            term = np.where(qpost > 0, qpost * (np.log(qpost) - np.log(np.where(p[..., None] > 0, p[..., None], 1.0))), 0.0)
        kl_qp = term.sum(axis=3)
        np.testing.assert_allclose(fd, kl_qp / bval ** 2, rtol=1e-5, atol=1e-8)


def check_p6_shift_scale(lib):
    q, k, v, beta = _inputs(6, 1, 2, 9, 5, beta_lo=1e-2, beta_hi=30.0)
    c = np.array([3.7, -2.0, 0.5, 11.0, -0.25])
    a = 2.5
    for causal in (True, False):
        base, _ = _run(lib, q, k, v, beta, causal)
        shifted, _ = _run(lib, q, k, v + c, beta, causal)
        np.testing.assert_allclose(shifted, base + c, rtol=0, atol=1e-11)
        scaled, _ = _run(lib, q, k, a * v, beta, causal)
        base_ab, _ = _run(lib, q, k, v, a * beta, causal)
        np.testing.assert_allclose(scaled, a * base_ab, rtol=0, atol=1e-11)


def check_p7_uniform_prior(lib):
    q, k, v, beta = _inputs(7, 1, 2, 12, 6, beta_lo=1e-2, beta_hi=50.0)
    q[:] = 0.0
    for causal in (True, False):
        out, lse = _run(lib, q, k, v, beta, causal)
        T = q.shape[2]
        for t in range(T):
            n = t + 1 if causal else T
            for h in range(2):
                for j in range(6):
                    b = beta[h, j]
                    want = (logsumexp(b * v[0, h, :n, j]) - np.log(n)) / b
                    assert abs(out[0, h, t, j] - want) <= 1e-12 * max(1.0, abs(want)), (causal, t, h, j)
                assert abs(lse[0, h, t] - np.log(n)) <= 1e-13


def _golden_cases():
    with open(os.path.join(GOLDEN_DIR, "bruteforce_tiny.json")) as f:
        return json.load(f)["cases"]


def check_p8_bruteforce_golden(lib):
    for case in _golden_cases():
        q = np.array(case["q"], dtype=np.float64)
        k = np.array(case["k"], dtype=np.float64)
        v = np.array(case["v"], dtype=np.float64)
        beta = np.array(case["beta"], dtype=np.float64)
        out, lse = _run(lib, q, k, v, beta, case["causal"])
        want = np.array([[float(x) for x in row] for row in case["out"]]).reshape(out.shape)
        want_lse = np.array([float(x) for x in case["lse"]]).reshape(lse.shape)
        np.testing.assert_allclose(out, want, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(lse, want_lse, rtol=1e-13, atol=1e-13)


def check_p9_toy_argmax(lib):
    """App. "toy-argmax" data: winner a_j per channel at 1 + eps_j, others N(0, 0.05^2)."""
    r = _rng(9)
    T, D, delta, sigma = 128, 512, 1.0, 0.05
    v = r.normal(0.0, sigma, size=(1, 1, T, D))
    a = r.integers(0, T, size=D)
    v[0, 0, a, np.arange(D)] = delta + r.normal(0.0, sigma, size=D)
    q = np.zeros((1, 1, T, D))
    k = r.standard_normal((1, 1, T, D))
    beta = np.full((1, D), 100.0)
    out, _ = _run(lib, q, k, v, beta, False)
    vstar = v[0, 0].max(axis=0)
    want = vstar - np.log(T) / 100.0
    np.testing.assert_allclose(out[0, 0, -1], want, rtol=0, atol=1e-12)


def check_p10_mask_and_permutation(lib):
    q, k, v, beta = _inputs(10, 1, 2, 10, 4, beta_lo=1e-2, beta_hi=40.0)
    out_c, lse_c = _run(lib, q, k, v, beta, True)
    for t in (0, 3, 9):
        sub_o, sub_l = _run(lib, q[:, :, : t + 1], k[:, :, : t + 1], v[:, :, : t + 1], beta, False)
        np.testing.assert_allclose(out_c[:, :, t], sub_o[:, :, t], rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse_c[:, :, t], sub_l[:, :, t], rtol=0, atol=1e-12)
    perm = _rng(100).permutation(10)
    out_f, _ = _run(lib, q, k, v, beta, False)
    out_p, _ = _run(lib, q, k[:, :, perm], v[:, :, perm], beta, False)
    np.testing.assert_allclose(out_f, out_p, rtol=0, atol=1e-12)


def check_p11_rotation(lib):
    q, k, v, beta = _inputs(11, 1, 1, 9, 6, beta_lo=1e-2, beta_hi=20.0)
    R, _ = np.linalg.qr(_rng(111).standard_normal((6, 6)))
    for causal in (True, False):
        base, _ = _run(lib, q, k, v, beta, causal)
        rot, _ = _run(lib, q @ R, k @ R, v, beta, causal)
        np.testing.assert_allclose(rot, base, rtol=0, atol=1e-11)


def check_p12_large_beta(lib):
    q, k, v, _ = _inputs(12, 1, 2, 10, 5)
    beta = np.full((2, 5), 1e4)
    for causal in (True, False):
        out, _ = _run(lib, q, k, v, beta, causal)
        p, _ = _prior(q, k, causal)
        vstar, istar = _visible_max(v, causal)
        pstar = np.take_along_axis(p, np.ascontiguousarray(istar), axis=3)
        gap = vstar - out
        assert np.all(gap >= -1e-12)
        assert np.all(gap <= -np.log(pstar) / 1e4 + 1e-12)


def check_p13_lse(lib):
    q, k, v, beta = _inputs(13, 2, 2, 9, 7)
    for causal in (True, False):
        _, lse = _run(lib, q, k, v, beta, causal)
        _, s = _prior(q, k, causal)
        np.testing.assert_allclose(lse, logsumexp(s, axis=-1), rtol=0, atol=1e-12)


ALL_CHECKS = [
    check_p1_single_key,
    check_p2_constant_channel,
    check_p3_bounds,
    check_p4_small_beta,
    check_p5_monotone_and_derivative,
    check_p6_shift_scale,
    check_p7_uniform_prior,
    check_p8_bruteforce_golden,
    check_p9_toy_argmax,
    check_p10_mask_and_permutation,
    check_p11_rotation,
    check_p12_large_beta,
    check_p13_lse,
]
