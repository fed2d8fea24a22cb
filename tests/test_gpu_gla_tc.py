"""The GLA-prior read chunked on the tensor cores (fem_gla_fwd_tc) on the GPU (needs a GB300).

bf16 operands with fp32 accumulation and an fp32 state: the bound is the bf16
read's, max abs 2e-2 and mean abs 2e-3 against the float64 oracle (the O(T^2)
definition), on shapes that span one step, several 128-step chunks and ragged
tails, beta from 0 to 20 across both forms of the bank (the linear form below
1/4, the shifted one above), strong and weak decay.  At the bench's shape the
reference is the fp32 scan (fem_gla_fwd, itself held to 1e-4 of the oracle).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_07160_gb300 import build, fem

pytestmark = pytest.mark.gpu

MAX_TOL, MEAN_TOL = 2e-2, 2e-3


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return fem.load()


def _inputs(seed, B, H, T, g_scale=0.3, v_scale=1.0):
    g = torch.Generator().manual_seed(seed)
    qf = torch.relu(torch.randn((B, H, T, 64), generator=g)) + 0.05
    kf = torch.relu(torch.randn((B, H, T, 64), generator=g)) + 0.05
    v = torch.randn((B, H, T, 64), generator=g) * v_scale
    logdecay = -g_scale * torch.rand((B, H, T), generator=g)
    beta = torch.exp(torch.empty((H, 64)).uniform_(np.log(0.05), np.log(20.0), generator=g))
    beta[0, :3] = 0.0
    return qf, kf, v, logdecay, beta


def _run(qf, kf, v, logdecay, beta):
    dev = torch.device("cuda", 0)
    args = [x.to(dev) for x in (qf, kf, v, logdecay, beta)]
    out = torch.full(v.shape, float("nan"), dtype=torch.float32, device=dev)
    out, logz = fem.fem_gla_fwd_tc(*args, out=out)
    fem.check_device_error()
    return out.cpu().double().numpy(), logz.cpu().double().numpy()


@pytest.mark.parametrize("B,H,T,g_scale", [(1, 2, 1, 0.3), (1, 2, 100, 0.3), (2, 2, 257, 0.3), (1, 3, 300, 0.02),
                                            (1, 2, 384, 2.0)])
def test_gla_tc_matches_oracle(B, H, T, g_scale):
    qf, kf, v, logdecay, beta = _inputs(T + B, B, H, T, g_scale)
    out, logz = _run(qf, kf, v, logdecay, beta)
    ref, ref_logz = oracle.gla_read(qf, kf, v, logdecay, beta)
    assert np.isfinite(out).all()
    err = np.abs(out - ref)
    assert err.max() <= MAX_TOL and err.mean() <= MEAN_TOL, (err.max(), err.mean())
    assert np.abs(logz - ref_logz).max() <= 1e-2


def test_gla_tc_beta_sweep_and_wide_values():
    """beta straddling the two forms' boundary and values spread three times wider than N(0, 1).

    A bf16 operand is rounded to within 2^-8 of itself, so a row that sees few keys carries up to
    2^-8 |E| of error in its read: 2^-8 |v - c| for a linear channel (E = expm1(beta (v - c)) / beta
    ~ v - c at small beta), 2^-8 / beta for a shifted one.  The bound scales with the values'
    spread; with values 3 x N(0, 1) it is taken as 3 x the N(0, 1) bound."""
    v_scale = 3.0
    qf, kf, v, logdecay, _ = _inputs(5, 1, 2, 260, 0.1, v_scale=v_scale)
    vals = [0.0, 1e-3, 0.1, 0.24, 0.26, 1.0, 5.0, 20.0]
    beta = torch.tensor([vals[i % len(vals)] for i in range(2 * 64)], dtype=torch.float32).reshape(2, 64)
    out, _ = _run(qf, kf, v, logdecay, beta)
    ref, _ = oracle.gla_read(qf, kf, v, logdecay, beta)
    err = np.abs(out - ref)
    assert np.isfinite(out).all()
    w = np.unravel_index(int(err.argmax()), err.shape)
    assert err.max() <= MAX_TOL * v_scale and err.mean() <= MEAN_TOL * v_scale, (err.max(), err.mean(), w,
                                                                                  float(beta[w[1], w[3]]))


def test_gla_tc_bench_shape_against_the_scan():
    B, H, T = 4, 16, 8192
    qf, kf, v, logdecay, beta = _inputs(1, B, H, T)
    dev = torch.device("cuda", 0)
    args = [x.to(dev) for x in (qf, kf, v, logdecay, beta)]
    ref, ref_logz = fem.fem_gla_fwd(*args)
    out, logz = fem.fem_gla_fwd_tc(*args)
    fem.check_device_error()
    err = (out - ref).abs()
    assert torch.isfinite(out).all()
    assert err.max().item() <= MAX_TOL and err.mean().item() <= MEAN_TOL, (err.max().item(), err.mean().item())
    assert (logz - ref_logz).abs().max().item() <= 1e-2


def test_gla_tc_refuses_other_widths():
    dev = torch.device("cuda", 0)
    qf = torch.ones((1, 1, 8, 32), device=dev)
    v = torch.ones((1, 1, 8, 64), device=dev)
    with pytest.raises(fem.FemError) as e:
        fem.fem_gla_fwd_tc(qf, qf, v, torch.zeros((1, 1, 8), device=dev), torch.ones((1, 64), device=dev))
    assert e.value.status == 2
