"""The two-level gated read on the GPU against the float64 oracle (needs a GB300).

out = g ((1 - lambda) mu + lambda Fmax) (Sec. 3, "Two-Level Gated FEM"), with
gates drawn as the paper parameterises them (lambda a sigmoid output in
[0, 1], g a softplus output normalised to RMS 1 over the channels).  The
tolerance is the bf16 read's (max abs 2e-2, mean abs 2e-3) scaled by the
largest |g|, since the outer gate multiplies the read's error.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_07160_gb300 import build, fem
from paper_2602_07160_gb300 import workloads as W

pytestmark = pytest.mark.gpu

BF16_MAX, BF16_MEAN = 2e-2, 2e-3


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return fem.load()


def _gates(seed, shape):
    g = torch.Generator().manual_seed(seed)
    lam = torch.sigmoid(torch.randn(shape, generator=g, dtype=torch.float32) * 2)
    gate = torch.nn.functional.softplus(torch.randn(shape, generator=g, dtype=torch.float32))
    gate = gate / gate.pow(2).mean(-1, keepdim=True).sqrt()
    return lam, gate


CASES = [
    # B, H, T, d, causal
    (1, 2, 300, 64, True),
    (2, 2, 129, 128, True),
    (1, 3, 256, 128, False),
    (2, 2, 197, 64, False),
]


@pytest.mark.parametrize("B,H,T,d,causal", CASES)
def test_gated_read_matches_oracle(B, H, T, d, causal):
    q, k, v, bmax = W.make_custom(B, H, T, d, seed=11 * T + d)
    lam, gate = _gates(T + d, q.shape)
    dev = torch.device("cuda", 0)
    args = [x.to(dev) for x in (q, k, v, bmax, lam, gate)]
    out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=dev)
    out, lse = fem.fem_fwd_gated(*args, causal=causal, out=out)
    fem.check_device_error()
    ref, ref_lse = oracle.gated_read(q, k, v, bmax, lam, gate, causal)
    o = out.cpu().double().numpy()
    assert np.isfinite(o).all()
    err = np.abs(o - ref)
    scale = max(1.0, float(gate.abs().max()))
    assert err.max() <= BF16_MAX * scale and err.mean() <= BF16_MEAN, (err.max(), err.mean())
    assert np.abs(lse.cpu().double().numpy() - ref_lse).max() <= 2e-3


def test_gated_read_limits_match_the_plain_reads():
    """lambda = 0 gives g times the beta = 0 read, lambda = 1 and g = 1 the read at beta_max."""
    B, H, T, d, causal = 1, 2, 200, 128, True
    q, k, v, bmax = W.make_custom(B, H, T, d, seed=5)
    dev = torch.device("cuda", 0)
    qd, kd, vd, bd = (x.to(dev) for x in (q, k, v, bmax))
    _, gate = _gates(3, q.shape)
    gate = gate.to(dev)
    zeros, ones = torch.zeros(q.shape, device=dev), torch.ones(q.shape, device=dev)
    mu, _ = fem.fem_fwd(qd, kd, vd, torch.zeros_like(bd), causal=causal)
    fmax, lse_f = fem.fem_fwd(qd, kd, vd, bd, causal=causal)
    o0, lse0 = fem.fem_fwd_gated(qd, kd, vd, bd, zeros, gate, causal=causal)
    o1, _ = fem.fem_fwd_gated(qd, kd, vd, bd, ones, ones, causal=causal)
    fem.check_device_error()
    # (1 - 0) mu + 0 (F - mu) = mu, then times g; the plain read adds its diagonal
    # tile's P E to the accumulator in the epilogue (fp32, another summation order)
    assert torch.allclose(o0, mu * gate, rtol=1e-6, atol=1e-6)
    assert torch.allclose(o1, fmax, rtol=0, atol=1e-5)
    assert torch.equal(lse0, lse_f)


@pytest.mark.parametrize("d", [64, 128])
def test_gated_read_fixup_rows(d):
    """Spikes in small-valued beta_max = 20 channels move the bank shift in the
    middle of diagonal tiles, so rows before each spike are completed by the
    fix-up: there the gated output combines the fix-up's exact F with the mean
    the tensor-core kernel set aside for the entry."""
    B, H, T = 1, 2, 3000
    q, k, v, bmax = W.make_custom(B, H, T, d, seed=7)
    bmax[:, :8] = 20.0
    vf = v.float()
    vf[..., :8] *= 0.1
    for p in (5, 20 * 128 + 64, 23 * 128 + 40):
        vf[:, :, p, :8] = 3.0
    v = vf.to(torch.bfloat16).contiguous()
    lam, gate = _gates(d, q.shape)
    dev = torch.device("cuda", 0)
    out, lse = fem.fem_fwd_gated(*(x.to(dev) for x in (q, k, v, bmax, lam, gate)), causal=True)
    fem.check_device_error()
    assert fem.last_fixup_rows() >= 2 * (5 + 64 + 40)
    ref, ref_lse = oracle.gated_read(q, k, v, bmax, lam, gate, True)
    err = np.abs(out.cpu().double().numpy() - ref)
    scale = max(1.0, float(gate.abs().max()))
    assert err.max() <= BF16_MAX * scale and err.mean() <= BF16_MEAN, (err.max(), err.mean())
    assert np.abs(lse.cpu().double().numpy() - ref_lse).max() <= 2e-3


def test_gated_read_headline_shape_sampled():
    """The one-pass gated kernel (its own TMEM and shared-memory layout at d = 128: two score
    buffers, two K stages, two accumulators) at B4 H16 T8192 causal with the paper's gate
    parameterisation, checked on sampled rows that include the first and last key tiles."""
    w = W.WORKLOADS["lm_causal_d128"]
    q, k, v, bmax = W.make_inputs(w)
    lam, gate = _gates(17, q.shape)
    dev = torch.device("cuda", 0)
    out, lse = fem.fem_fwd_gated(*(x.to(dev) for x in (q, k, v, bmax, lam, gate)), causal=True)
    fem.check_device_error()
    r = np.random.default_rng(4)
    rows = np.unique(np.concatenate([np.arange(384), (w.B * w.H - 1) * w.T + np.arange(w.T - 128, w.T),
                                     r.choice(w.B * w.H * w.T, 1200, replace=False)]))
    ref, ref_lse = oracle.gated_read_rows(q, k, v, bmax, lam, gate, True, rows)
    got = out.reshape(-1, w.d)[torch.from_numpy(rows).to(dev)].cpu().double().numpy()
    assert np.isfinite(got).all()
    err = np.abs(got - ref)
    scale = max(1.0, float(gate.abs().max()))
    assert err.max() <= BF16_MAX * scale and err.mean() <= BF16_MEAN, (err.max(), err.mean())
    assert np.abs(lse.reshape(-1)[torch.from_numpy(rows).to(dev)].cpu().double().numpy() - ref_lse).max() <= 2e-3


@pytest.mark.parametrize("d", [64, 128])
def test_gated_read_peaked_prior(d):
    """Q and K scaled by 2 (score spread of about 30 nats) with beta_max up to 1e3: the gated
    kernel's guard routes the entries its 16-bit operands cannot hold to the exact fix-up."""
    q, k, v, _ = W.make_custom(1, 2, 400, d, seed=31)
    q = (q.float() * 2).to(torch.bfloat16)
    k = (k.float() * 2).to(torch.bfloat16)
    bmax = W.beta_grid(2, d, [0.05, 1.0, 5.0, 20.0, 100.0, 1e3])
    lam, gate = _gates(5, q.shape)
    dev = torch.device("cuda", 0)
    for causal in (True, False):
        out, _ = fem.fem_fwd_gated(*(x.to(dev) for x in (q, k, v, bmax, lam, gate)), causal=causal)
        fem.check_device_error()
        ref, _ = oracle.gated_read(q, k, v, bmax, lam, gate, causal)
        o = out.cpu().double().numpy()
        assert np.isfinite(o).all()
        err = np.abs(o - ref)
        scale = max(1.0, float(gate.abs().max()))
        assert err.max() <= BF16_MAX * scale and err.mean() <= BF16_MEAN, (causal, err.max(), err.mean())
