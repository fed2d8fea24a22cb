"""The bounded-wait failure path on the device (needs a GB300).

Every wait of the library's kernels gives up after a limit, records the fact
in a per-device error word and lets the kernel return, so a stuck copy or
contraction ends in FEM_ERR_TIMEOUT instead of a hung GPU.  Here the wait
runs out on purpose, on an mbarrier that nothing completes (the library's
wait probe, 1 ms), and the tests check that the host sees the timeout once,
that the word is cleared, and that the next read still matches the oracle.
No copy or tensor-core operation is left in flight by the probe.
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


def test_wait_probe_reports_timeout_then_clears():
    fem.check_device_error()  # start from a clean word
    fem.probe_wait_timeout(1000)
    with pytest.raises(fem.FemError) as e:
        fem.check_device_error()
    assert e.value.status == 4  # FEM_ERR_TIMEOUT
    fem.check_device_error()  # cleared: no error now


def test_read_after_timeout_still_matches_oracle():
    fem.probe_wait_timeout(500)
    with pytest.raises(fem.FemError):
        fem.check_device_error()
    q, k, v, beta = W.make_custom(1, 2, 300, 128, seed=12)
    dev = torch.device("cuda", 0)
    out, lse = fem.fem_fwd(*(x.to(dev) for x in (q, k, v, beta)), causal=True)
    fem.check_device_error()
    ref, _ = oracle.fem_read(q, k, v, beta, True)
    err = np.abs(out.cpu().double().numpy() - ref)
    assert err.max() <= 2e-2 and err.mean() <= 2e-3


def test_probe_rejects_bad_limits():
    with pytest.raises(fem.FemError) as e:
        fem.probe_wait_timeout(0)
    assert e.value.status == 1
    with pytest.raises(fem.FemError) as e:
        fem.probe_wait_timeout(2_000_000)
    assert e.value.status == 1
