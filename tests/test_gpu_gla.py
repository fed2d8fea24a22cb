"""FEM over a GLA prior on the GPU against the float64 oracle (needs a GB300).

fp32 inputs and fp32 arithmetic: the bound is the fp32 read's 1e-4 (max abs)
with beta in [0.05, 20] and exact zeros; log Z to 1e-4 as well.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_07160_gb300 import build, fem

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return fem.load()


def _inputs(seed, B, H, T, m, d, g_scale=0.3):
    g = torch.Generator().manual_seed(seed)
    qf = torch.relu(torch.randn((B, H, T, m), generator=g)) + 0.05
    kf = torch.relu(torch.randn((B, H, T, m), generator=g)) + 0.05
    v = torch.randn((B, H, T, d), generator=g)
    logdecay = -g_scale * torch.rand((B, H, T), generator=g)
    beta = torch.exp(torch.empty((H, d)).uniform_(np.log(0.05), np.log(20.0), generator=g))
    beta[0, : min(3, d)] = 0.0
    return qf, kf, v, logdecay, beta


@pytest.mark.parametrize("B,H,T,m,d", [(1, 2, 1, 16, 8), (2, 2, 100, 32, 31), (1, 3, 257, 64, 64),
                                       (2, 1, 600, 64, 100), (1, 2, 2000, 64, 155)])
def test_gla_read_matches_oracle(B, H, T, m, d):
    qf, kf, v, logdecay, beta = _inputs(T + m + d, B, H, T, m, d)
    dev = torch.device("cuda", 0)
    args = [x.to(dev).contiguous() for x in (qf, kf, v, logdecay, beta)]
    out = torch.full(v.shape, float("nan"), dtype=torch.float32, device=dev)
    out, logz = fem.fem_gla_fwd(*args, out=out)
    fem.check_device_error()
    ref, ref_lz = oracle.gla_read(qf, kf, v, logdecay, beta)
    o = out.cpu().double().numpy()
    assert np.isfinite(o).all()
    err = np.abs(o - ref)
    assert err.max() <= 1e-4, (err.max(), np.unravel_index(err.argmax(), err.shape))
    assert np.abs(logz.cpu().double().numpy() - ref_lz).max() <= 1e-4


def test_gla_strong_decay_reads_the_current_value():
    """g = -60: the prior sits on the current step, so o_t = v_t for every beta."""
    qf, kf, v, logdecay, beta = _inputs(7, 1, 2, 300, 32, 20)
    logdecay[:] = -60.0
    dev = torch.device("cuda", 0)
    out, _ = fem.fem_gla_fwd(*[x.to(dev).contiguous() for x in (qf, kf, v, logdecay, beta)])
    fem.check_device_error()
    assert (out.cpu() - v).abs().max().item() <= 1e-5
