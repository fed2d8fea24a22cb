"""Gradients of the fp32 read on the GPU against the float64 oracle (needs a GB300).

fp32 arithmetic over O(T) terms per gradient: bound 1e-4 of each gradient's
largest magnitude (at least 1), element by element.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_07160_gb300 import build, fem
from paper_2602_07160_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return fem.load()


@pytest.mark.parametrize("B,H,T,d,causal", [(1, 2, 1, 16, True), (2, 2, 33, 32, True), (1, 2, 100, 64, False),
                                            (2, 1, 257, 128, True), (1, 3, 150, 64, True),
                                            # channels not a multiple of 32 per lane, and d > 128
                                            (1, 2, 65, 96, False), (1, 1, 70, 200, True)])
def test_backward_matches_oracle(B, H, T, d, causal):
    q, k, v, beta = W.make_custom(B, H, T, d, dtype="f32", seed=T + d)
    beta[0, :2] = 0.0
    dout = torch.randn(q.shape, generator=torch.Generator().manual_seed(T), dtype=torch.float32)
    dev = torch.device("cuda", 0)
    qd, kd, vd, bd, dod = (x.to(dev).contiguous() for x in (q, k, v, beta, dout))
    out, lse = fem.fem_fwd_f32(qd, kd, vd, bd, causal=causal)
    dq, dk, dv, db = fem.fem_bwd_f32(qd, kd, vd, bd, out, lse, dod, causal=causal)
    fem.check_device_error()
    ref = oracle.fem_backward(q, k, v, beta, dout, causal)
    for name, got, want in zip(("dq", "dk", "dv", "dbeta"), (dq, dk, dv, db), ref):
        g = got.cpu().double().numpy()
        assert np.isfinite(g).all(), name
        err = np.abs(g - want).max()
        assert err <= 1e-4 * max(1.0, float(np.abs(want).max())), (name, err, float(np.abs(want).max()))
