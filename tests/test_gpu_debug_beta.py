"""FEM_DEBUG=1: the entry points that take beta check it on the device (needs a GB300).

The flag is read once per process, so each case runs in a child interpreter
with FEM_DEBUG set: a negative, NaN or infinite beta is refused with
FEM_ERR_INVALID_ARG before anything else is enqueued, a valid beta reads as
usual, and without the flag the library does not look at beta's values.
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys, math, torch
sys.path.insert(0, {root!r})
from paper_2602_07160_gb300 import build, fem, workloads as W
build.build()
dev = torch.device("cuda", 0)
q, k, v, beta = (x.to(dev) for x in W.make_custom(1, 2, 200, {d}, seed=1))
qf, kf, vf = (x.float() for x in (q, k, v))
def refused(fn):
    try:
        fn()
    except fem.FemError as e:
        return e.status == 1
    return False
results = []
for bad in (-0.5, math.nan, math.inf):
    b2 = beta.clone()
    b2[1, 3] = bad
    results.append(refused(lambda: fem.fem_fwd(q, k, v, b2, causal=True)))
    results.append(refused(lambda: fem.fem_fwd_f32(qf, kf, vf, b2, causal=True)))
    results.append(refused(lambda: fem.fem_fwd_host(q.cpu(), k.cpu(), v.cpu(), b2.cpu(), causal=True)))
out, _ = fem.fem_fwd(q, k, v, beta, causal=True)
torch.cuda.synchronize()
results.append(bool(torch.isfinite(out).all()))
print("RESULT", all(results), results)
"""


@pytest.mark.parametrize("d", [64, 128])
def test_debug_mode_refuses_bad_beta(d):
    env = dict(os.environ, FEM_DEBUG="1")
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT, d=d)], env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    assert "RESULT True" in r.stdout, r.stdout[-2000:]
