"""The oracle's TDC convolution against the paper's statements (CPU only):

  T1  the rank-one streaming form of Prop. "tdc-lowrank": C_t = C_{t-1} + u_t / f_t,
      h_t = f_t C_t with f_t = exp(-(s_1 + ... + s_t)) (numpy, moderate T)
  T2  s = 0: no decay, h_t is the running sum of u
  T3  large s: the kernel keeps only i = t, h_t = u_t
  T4  linearity in u and causality (inputs after t do not change h_t)
"""
import numpy as np

import oracle


def _inputs(seed, B=2, T=40, Hc=6, s_scale=0.2):
    r = np.random.default_rng(seed)
    s = s_scale * np.log1p(np.exp(r.standard_normal((B, T, Hc))))  # softplus rates >= 0
    u = r.standard_normal((B, T, Hc))
    return s, u


def test_t1_streaming_form():
    s, u = _inputs(51)
    h = oracle.tdc_conv(s, u)
    f = np.exp(-np.cumsum(s, axis=1))
    C = np.cumsum(u / f, axis=1)
    assert np.allclose(h, f * C, rtol=1e-10, atol=1e-12)


def test_t2_no_decay():
    s, u = _inputs(52)
    assert np.allclose(oracle.tdc_conv(np.zeros_like(s), u), np.cumsum(u, axis=1), rtol=0, atol=1e-12)


def test_t3_fast_decay():
    s, u = _inputs(53)
    assert np.allclose(oracle.tdc_conv(np.full_like(s, 80.0), u), u, rtol=0, atol=1e-12)


def test_t4_linear_and_causal():
    s, u = _inputs(54)
    u2 = np.random.default_rng(55).standard_normal(u.shape)
    assert np.allclose(oracle.tdc_conv(s, 2 * u - 3 * u2), 2 * oracle.tdc_conv(s, u) - 3 * oracle.tdc_conv(s, u2),
                       rtol=0, atol=1e-10)
    s3, u3 = s.copy(), u.copy()
    s3[:, 25:] += 1.0
    u3[:, 25:] -= 4.0
    assert np.array_equal(oracle.tdc_conv(s, u)[:, :25], oracle.tdc_conv(s3, u3)[:, :25])
