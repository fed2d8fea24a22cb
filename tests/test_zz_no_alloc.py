"""fem_fwd_noalloc: the read without device allocation (needs a GB300).

Some callers may not allocate device memory while the read runs, e.g. a
plugin whose execute callback must not allocate, or a service that reserves
all device memory up front.  fem_fwd_noalloc serves them from a fixed 16 MiB
scratch array compiled into the library.  These tests call it through the C
ABI twice in a row (the scratch keeps the previous call's contents) and check
that each result equals fem_fwd's bit for bit (the same kernels run on the
same inputs), and check that a problem too large for the scratch is refused
before anything runs.  The file is named so that pytest collects it last.
"""
import pytest
import torch

from paper_2602_07160_gb300 import build, fem
from paper_2602_07160_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return fem.load()


@pytest.mark.parametrize("B,H,T,d,causal", [(1, 3, 300, 128, True), (2, 2, 197, 64, False)])
def test_noalloc_matches_fem_fwd_on_two_calls(B, H, T, d, causal):
    dev = torch.device("cuda", 0)
    q, k, v, beta = (x.to(dev) for x in W.make_custom(B, H, T, d, seed=T + d))
    ref_out, ref_lse = fem.fem_fwd(q, k, v, beta, causal=causal)
    torch.cuda.synchronize()
    for _ in range(2):
        out = torch.full(q.shape, float("nan"), dtype=torch.float32, device=dev)
        lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=dev)
        fem.fem_fwd_noalloc(q, k, v, beta, causal=causal, out=out, lse=lse)
        fem.check_device_error()
        assert torch.isfinite(out).all()
        assert torch.equal(out, ref_out), (out - ref_out).abs().max().item()
        assert torch.equal(lse, ref_lse)


def test_noalloc_refuses_too_large_problem():
    B, H, T, d = 4, 16, 8192, 128
    assert fem.workspace_bytes(B, H, T, d, True) > (16 << 20)
    dev = torch.device("cuda", 0)
    q = torch.zeros((B, H, T, d), dtype=torch.bfloat16, device=dev)
    beta = torch.ones((H, d), dtype=torch.float32, device=dev)
    out = torch.zeros((B, H, T, d), dtype=torch.float32, device=dev)
    with pytest.raises(fem.FemError) as e:
        fem.fem_fwd_noalloc(q, q, q, beta, causal=True, out=out, lse=False)
    assert e.value.status == 5  # FEM_ERR_NO_MEMORY
    assert torch.count_nonzero(out).item() == 0
