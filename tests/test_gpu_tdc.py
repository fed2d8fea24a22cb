"""The TDC convolution on the GPU against the float64 oracle (needs a GB300).

fp32 arithmetic: bound 1e-4 relative to the scale of h (its running sums grow
with the decay horizon), element by element.
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


@pytest.mark.parametrize("B,T,Hc,s_scale", [(1, 1, 8, 0.2), (2, 127, 32, 0.2), (2, 129, 64, 0.05),
                                            (1, 1000, 48, 0.2), (4, 2000, 64, 0.01),
                                            # 157 segments (several per combine lane) and more
                                            # channels than a block's threads
                                            (1, 5000, 40, 0.01), (1, 1200, 300, 0.05),
                                            # the longest sequence of the one-launch form, and the
                                            # first of the three launches
                                            (1, 16384, 4, 0.01), (1, 16385, 4, 0.01)])
def test_tdc_matches_oracle(B, T, Hc, s_scale):
    g = torch.Generator().manual_seed(T + Hc)
    s = s_scale * torch.nn.functional.softplus(torch.randn((B, T, Hc), generator=g))
    u = torch.randn((B, T, Hc), generator=g)
    h = torch.full((B, T, Hc), float("nan"), device="cuda")  # poisoned: every element must be written
    fem.fem_tdc_conv(s.cuda(), u.cuda(), out=h)
    fem.check_device_error()
    ref = oracle.tdc_conv(s, u)
    err = np.abs(h.cpu().double().numpy() - ref)
    scale = max(1.0, float(np.abs(ref).max()))
    assert err.max() <= 1e-4 * scale, (err.max(), scale)
