"""The attention-mode comparator on the GPU (needs a GB300).

fem_attn_fwd runs the read's tensor-core kernel with V itself in place of the
value bank: plain softmax attention, the read's beta -> 0 limit (Prop.
"app-baseline").  It is checked against the oracle at beta = 0 (the prior mean)
at the bf16 read's tolerance, on shapes with ragged tails, both masks and
both head dimensions.
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


@pytest.mark.parametrize("B,H,T,d,causal", [(1, 2, 300, 128, True), (2, 2, 129, 64, True), (1, 3, 197, 64, False),
                                            (1, 2, 256, 128, False), (1, 1, 1, 128, True)])
def test_attention_mode_matches_the_prior_mean(B, H, T, d, causal):
    q, k, v, _ = W.make_custom(B, H, T, d, seed=3 * T + d)
    dev = torch.device("cuda", 0)
    out = torch.full(q.shape, float("nan"), device=dev)
    out, lse = fem.fem_attn_fwd(*(x.to(dev) for x in (q, k, v)), causal=causal, out=out)
    fem.check_device_error()
    ref, ref_lse = oracle.fem_read(q, k, v, torch.zeros(H, d), causal)
    o = out.cpu().double().numpy()
    assert np.isfinite(o).all()
    err = np.abs(o - ref)
    assert err.max() <= 2e-2 and err.mean() <= 2e-3, (err.max(), err.mean())
    assert np.abs(lse.cpu().double().numpy() - ref_lse).max() <= 2e-3


def test_attention_mode_headline_shape_sampled():
    w = W.WORKLOADS["lm_causal_d128"]
    q, k, v, _ = W.make_inputs(w)
    dev = torch.device("cuda", 0)
    out, lse = fem.fem_attn_fwd(*(x.to(dev) for x in (q, k, v)), causal=True)
    fem.check_device_error()
    rows = np.unique(np.concatenate([np.arange(256), np.random.default_rng(2).choice(w.B * w.H * w.T, 600,
                                                                                       replace=False)]))
    ref, _ = oracle.fem_read_rows(q, k, v, torch.zeros(w.H, w.d), True, rows)
    got = out.reshape(-1, w.d)[torch.from_numpy(rows).to(dev)].cpu().double().numpy()
    err = np.abs(got - ref)
    assert err.max() <= 2e-2 and err.mean() <= 2e-3, (err.max(), err.mean())
