"""bf16 read at head dimensions 16 and 32 on the GPU against the float64 oracle (needs a GB300).

These head dimensions run on the library's CUDA-core kernel (fp32 products and
sums of the bf16 inputs, no 16-bit operand anywhere), so the output is held to
the fp32 path's bound, 1e-4, against the oracle evaluated on the same
bf16-rounded inputs upcast to double.  The cases cover one key, ragged tails,
both priors, a beta sweep from 0 to 1e3, the workspace, no-allocation and
host-buffer entry points.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2602_07160_gb300 import build, fem
from paper_2602_07160_gb300 import workloads as W

pytestmark = pytest.mark.gpu

F32_MAX = 1e-4
LSE_MAX = 1e-4


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return fem.load()


CASES = [
    # B, H, T, d, causal
    (1, 2, 1, 16, True),
    (2, 2, 127, 16, True),
    (1, 3, 300, 32, True),
    (2, 2, 129, 32, False),
    (1, 2, 197, 16, False),
]


@pytest.mark.parametrize("B,H,T,d,causal", CASES)
def test_small_head_dim_matches_oracle(B, H, T, d, causal):
    q, k, v, beta = W.make_custom(B, H, T, d, seed=3 * T + d)
    dev = torch.device("cuda", 0)
    out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=dev)
    out, lse = fem.fem_fwd(*(x.to(dev) for x in (q, k, v, beta)), causal=causal, out=out)
    fem.check_device_error()
    ref, ref_lse = oracle.fem_read(q, k, v, beta, causal)
    o = out.cpu().double().numpy()
    assert np.isfinite(o).all()
    assert np.abs(o - ref).max() <= F32_MAX
    assert np.abs(lse.cpu().double().numpy() - ref_lse).max() <= LSE_MAX
    assert fem.last_fixup_rows() == 0


@pytest.mark.parametrize("d", [16, 32])
def test_small_head_dim_beta_sweep(d):
    q, k, v, _ = W.make_custom(1, 2, 200, d, seed=d)
    beta = W.beta_grid(2, d, [0.0, 1e-3, 0.05, 1.0, 5.0, 20.0, 100.0, 1e3])
    dev = torch.device("cuda", 0)
    out, _ = fem.fem_fwd(*(x.to(dev) for x in (q, k, v, beta)), causal=True)
    fem.check_device_error()
    ref, _ = oracle.fem_read(q, k, v, beta, True)
    assert np.abs(out.cpu().double().numpy() - ref).max() <= F32_MAX


def test_small_head_dim_other_entry_points():
    B, H, T, d = 2, 2, 150, 32
    q, k, v, beta = W.make_custom(B, H, T, d, seed=9)
    dev = torch.device("cuda", 0)
    qd, kd, vd, bd = (x.to(dev) for x in (q, k, v, beta))
    ref_out, ref_lse = fem.fem_fwd(qd, kd, vd, bd, causal=True)
    assert fem.workspace_bytes(B, H, T, d, True) == 256
    out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=dev)
    lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=dev)
    fem.fem_fwd_noalloc(qd, kd, vd, bd, causal=True, out=out, lse=lse)
    fem.check_device_error()
    assert torch.equal(out, ref_out) and torch.equal(lse, ref_lse)
    out_h, lse_h = fem.fem_fwd_host(q, k, v, beta, causal=True)
    assert torch.equal(out_h, ref_out.cpu()) and torch.equal(lse_h, ref_lse.cpu())
