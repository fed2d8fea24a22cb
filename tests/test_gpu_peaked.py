"""GPU read against the float64 oracle on peaked priors (needs a GB300).

With Q and K drawn at a scale sigma the scores q.k/sqrt(d) spread over
tens of nats, so the prior weights of most keys are far below the largest
one.  At large beta the free energy (1/beta) log sum_i p(i) e^{beta v_i}
(Sec. 2.3, Eq. "fem-free-energy-main") is then often governed by a key of
tiny prior weight and large value, or by a heavy key whose value lies far
below the channel's maximum: the products p(i) e^{beta v_i} span a range
that neither a 16-bit prior weight nor a 16-bit value-bank entry holds.  The
read must still agree with the definition; entries whose rounding error
cannot be bounded are recomputed exactly, so these tests check the whole
path.  Tolerances are the bf16 ones of the other parity tests.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_07160_gb300 import build, fem
from paper_2602_07160_gb300 import workloads as W

pytestmark = pytest.mark.gpu

BF16_MAX, BF16_MEAN = 2e-2, 2e-3
LSE_MAX = 2e-3
BETA_SWEEP = [0.0, 1e-4, 1e-3, 1e-2, 0.1, 0.5, 1.0, 5.0, 20.0, 100.0, 1e3]


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return fem.load()


def _scaled(q, k, sigma):
    return ((q.float() * sigma).to(torch.bfloat16).contiguous(),
            (k.float() * sigma).to(torch.bfloat16).contiguous())


def _gpu(q, k, v, beta, causal):
    dev = torch.device("cuda", 0)
    out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=dev)
    out, lse = fem.fem_fwd(*(x.to(dev) for x in (q, k, v, beta)), causal=causal, out=out)
    fem.check_device_error()
    return out.cpu().double().numpy(), lse.cpu().double().numpy()


def _assert_close(out, ref, what):
    assert np.isfinite(out).all(), f"{what}: {int((~np.isfinite(out)).sum())} non-finite outputs"
    err = np.abs(out - ref)
    mx, mn = float(err.max()), float(err.mean())
    where = np.unravel_index(int(err.argmax()), err.shape)
    assert mx <= BF16_MAX and mn <= BF16_MEAN, f"{what}: max {mx:.3e} at {where}, mean {mn:.3e}"


@pytest.mark.parametrize("sigma", [1.5, 2.0, 3.0])
@pytest.mark.parametrize("d,causal", [(64, True), (128, True), (64, False), (128, False)])
def test_peaked_prior_beta_sweep(sigma, d, causal):
    """Score spreads of about 15 to 60 nats over 520 keys (four tiles and a ragged tail),
    beta from 0 to 1e3 along the channels."""
    q, k, v, _ = W.make_custom(1, 2, 520, d, seed=7)
    q, k = _scaled(q, k, sigma)
    beta = W.beta_grid(2, d, BETA_SWEEP)
    out, lse = _gpu(q, k, v, beta, causal)
    ref, ref_lse = oracle.fem_read(q, k, v, beta, causal)
    _assert_close(out, ref, f"sigma={sigma} d={d} causal={causal}")
    assert np.abs(lse - ref_lse).max() <= LSE_MAX * max(1.0, np.abs(ref_lse).max() / 10)


@pytest.mark.parametrize("d,causal", [(64, True), (128, True), (128, False)])
def test_planted_heavy_key_with_low_value(d, causal):
    """Every row puts about 25 nats more score on one planted key, whose values in half the
    channels sit below every other value of the channel: at large beta the read is carried
    by keys of prior weight near e^-25 and the heavy key's bank entry underflows."""
    B, H, T = 1, 2, 400
    q, k, v, _ = W.make_custom(B, H, T, d, seed=21)
    gen = torch.Generator().manual_seed(5)
    kf, vf = k.float(), v.float()
    t = torch.arange(T)
    pick = (torch.rand(B, H, T, generator=gen) * ((t + 1) if causal else T)).long()
    pick = torch.minimum(pick, (t if causal else torch.full_like(t, T - 1)))
    qf = 25.0 / d ** 0.5 * torch.gather(kf, 2, pick[..., None].expand(B, H, T, d))
    low = vf.amin(dim=2, keepdim=True) - 0.5
    half = torch.arange(d) % 2 == 0
    for b in range(B):
        for h in range(H):
            keys = pick[b, h].unique()
            vf[b, h, keys[:, None], half] = low[b, h, 0, half]
    q, v = qf.to(torch.bfloat16).contiguous(), vf.to(torch.bfloat16).contiguous()
    beta = W.beta_grid(H, d, [0.0, 0.05, 1.0, 5.0, 20.0, 100.0])
    out, _ = _gpu(q, k, v, beta, causal)
    ref, _ = oracle.fem_read(q, k, v, beta, causal)
    _assert_close(out, ref, f"planted d={d} causal={causal}")


def test_peaked_prior_headline_shape_sampled():
    """B4 H16 T8192 d128 causal with sigma = 2 (score spread about 30 nats) and the
    workload's beta, checked on sampled rows including the first and last tiles."""
    w = W.WORKLOADS["lm_causal_d128"]
    q, k, v, beta = W.make_inputs(w)
    q, k = _scaled(q, k, 2.0)
    out, lse = _gpu(q, k, v, beta, True)
    r = np.random.default_rng(1)
    rows = np.unique(np.concatenate([np.arange(256), (w.B * w.H - 1) * w.T + np.arange(w.T - 128, w.T),
                                     r.choice(w.B * w.H * w.T, 800, replace=False)]))
    ref, ref_lse = oracle.fem_read_rows(q, k, v, beta, True, rows)
    _assert_close(out.reshape(-1, w.d)[rows], ref, "headline sigma=2")
    assert np.abs(lse.reshape(-1)[rows] - ref_lse).max() <= LSE_MAX * 10
