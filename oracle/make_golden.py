"""Write tests/golden/bruteforce_tiny.json from the 50-digit brute force.

TEST INFRASTRUCTURE ONLY.  Calls nothing but ``oracle.bruteforce``: the stored
values are the read of Sec. 2.3 (Eq. "fem-free-energy-main") with the softmax
prior of App. C, evaluated in 50-digit arithmetic on tiny seeded inputs, so
the float64 C oracle can be checked on machines without mpmath.

    python -m oracle.make_golden
"""
from __future__ import annotations

import json
import os

import numpy as np

from oracle.bruteforce import fem_read_mp

OUT = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "tests", "golden",
                   "bruteforce_tiny.json")

# (seed, B, H, T, d, causal, beta values cycled over channels of each head)
CASES = [
    (0, 1, 2, 6, 3, True, [0.0, 1e-3, 0.5, 7.0, 1e3, 0.05]),
    (1, 1, 1, 5, 4, False, [1e-3, 2.0, 30.0, 0.0]),
    (2, 2, 1, 4, 2, True, [0.25, 100.0]),
]


def main():
    cases = []
    for seed, B, H, T, d, causal, bvals in CASES:
        r = np.random.default_rng(seed)
        q = r.standard_normal((B, H, T, d))
        k = r.standard_normal((B, H, T, d))
        v = r.standard_normal((B, H, T, d))
        beta = np.array([bvals[(h * d + j) % len(bvals)] for h in range(H) for j in range(d)]).reshape(H, d)
        out = np.empty((B, H, T, d), dtype=object)
        lse = np.empty((B, H, T), dtype=object)
        for b in range(B):
            for h in range(H):
                o, l = fem_read_mp(q[b, h].tolist(), k[b, h].tolist(), v[b, h].tolist(), beta[h].tolist(), causal)
                for t in range(T):
                    lse[b, h, t] = str(l[t])[:40]
                    for j in range(d):
                        out[b, h, t, j] = str(o[t][j])[:40]
        cases.append({
            "seed": seed, "causal": causal, "shape": [B, H, T, d],
            "q": q.tolist(), "k": k.tolist(), "v": v.tolist(), "beta": beta.tolist(),
            "out": out.reshape(-1, d).tolist(), "lse": lse.reshape(-1).tolist(),
        })
    doc = {
        "what": "Free Energy Mixer read, softmax prior, 50-digit mpmath brute force",
        "cite": "arXiv 2602.07160, Sec. 2.3 Eq. fem-free-energy-main; App. C Eq. softmax-prior",
        "writer": "python -m oracle.make_golden",
        "cases": cases,
    }
    os.makedirs(os.path.dirname(OUT), exist_ok=True)
    with open(OUT, "w") as f:
        json.dump(doc, f, indent=1)
    print(f"wrote {OUT}")


if __name__ == "__main__":
    main()
