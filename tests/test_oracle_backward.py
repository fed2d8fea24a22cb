"""The oracle's gradients of the read against independent facts (CPU only):

  B1  central finite differences of the forward oracle (Sec. 2.3 read) in
      float64, for q, k, v and beta, on a small causal and a full-prior case
  B2  for a unit output cotangent e_{t,j}: dv_{.,j} is the posterior q_{t,.,j},
      a probability vector (Prop. "app-geom": ||grad_v F||_1 = 1)
  B3  the score gradients of every row sum to zero (sum_i (q_i - p_i) = 0)
  B4  beta = 0: dbeta = Var_p(v)/2 per row (the second cumulant, Prop. "app-baseline")
"""
import numpy as np
import pytest

import oracle
from tests.oracle_pins import _inputs, _prior


def _loss(q, k, v, beta, dout, causal):
    out, _ = oracle.fem_read(q, k, v, beta, causal, nthreads=1)
    return float((out * dout).sum())


@pytest.mark.parametrize("causal", [True, False])
def test_b1_finite_differences(causal):
    q, k, v, beta = _inputs(61, 1, 2, 5, 3, beta_lo=0.2, beta_hi=5.0)
    beta[0, 1] = 0.0
    dout = np.random.default_rng(62).standard_normal(q.shape)
    dq, dk, dv, db = oracle.fem_backward(q, k, v, beta, dout, causal)
    eps = 1e-6
    for name, x, g in (("q", q, dq), ("k", k, dk), ("v", v, dv), ("beta", beta, db)):
        it = np.nditer(x, flags=["multi_index"])
        for _ in it:
            idx = it.multi_index
            if name == "beta" and x[idx] == 0.0:
                continue  # one-sided at the boundary beta = 0
            xp, xm = x.copy(), x.copy()
            xp[idx] += eps
            xm[idx] -= eps
            args = {"q": q, "k": k, "v": v, "beta": beta}
            args[name] = xp
            fp = _loss(args["q"], args["k"], args["v"], args["beta"], dout, causal)
            args[name] = xm
            fm = _loss(args["q"], args["k"], args["v"], args["beta"], dout, causal)
            num = (fp - fm) / (2 * eps)
            assert abs(num - g[idx]) <= 1e-6 * max(1.0, abs(num)), (name, idx, num, g[idx])


def test_b2_posterior_is_a_distribution():
    q, k, v, beta = _inputs(63, 1, 1, 7, 4, beta_lo=0.1, beta_hi=10.0)
    for t, j in ((6, 0), (3, 2)):
        dout = np.zeros(q.shape)
        dout[0, 0, t, j] = 1.0
        _, _, dv, _ = oracle.fem_backward(q, k, v, beta, dout, True)
        col = dv[0, 0, :, j]
        assert np.all(col >= 0) and abs(col.sum() - 1.0) < 1e-12 and np.all(col[t + 1 :] == 0)


def test_b3_score_gradients_sum_to_zero():
    q, k, v, beta = _inputs(64, 1, 2, 6, 4, beta_lo=0.1, beta_hi=10.0)
    dout = np.random.default_rng(65).standard_normal(q.shape)
    dq, _, _, _ = oracle.fem_backward(q, k, v, beta, dout, True)
    # dq = dS K / sqrt(d); with K replaced by ones the rows give sum_i dS_{t,i}
    dq1, _, _, _ = oracle.fem_backward(q, np.ones_like(k), v, beta, dout, True)
    assert np.abs(dq1).max() < 1e-12


def test_b4_zero_beta_is_half_the_variance():
    q, k, v, beta = _inputs(66, 1, 1, 6, 3)
    beta[:] = 0.0
    dout = np.zeros(q.shape)
    dout[0, 0, 4, 1] = 1.0
    _, _, _, db = oracle.fem_backward(q, k, v, beta, dout, True)
    p, _ = _prior(q, k, True)
    pt, vj = p[0, 0, 4], v[0, 0, :, 1]
    mu = pt @ vj
    assert abs(db[0, 1] - 0.5 * (pt @ (vj - mu) ** 2)) < 1e-12
