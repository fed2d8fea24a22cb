"""50-digit brute force of the Free Energy Mixer read, for tiny inputs.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).  It pins the C oracle
from a different arrangement of the same definition: the prior p_t is formed
explicitly as a normalised softmax and the read is taken in the form of
Eq. "fem-free-energy-main" (Sec. 2.3),

    F_{t,j}(beta) = (1/beta) log sum_{i in M_t} p_t(i) exp(beta v_{i,j}),

instead of the difference of two log-sum-exps the C code evaluates.  Scores
are s_{t,i} = q_t . k_i / sqrt(d) (Sec. 1) over M_t = {0..t} (causal) or all
keys; beta = 0 is the prior mean (the beta -> 0 limit of Prop.
"app-baseline").  Pure-Python loops: only for T, d of a handful.
"""
from __future__ import annotations

import mpmath


def fem_read_mp(q, k, v, beta, causal: bool, dps: int = 50):
    """q, k, v: nested lists [T][d] of floats (one head); beta: list [d].

    Returns (out [T][d], lse [T]) as lists of mpmath.mpf."""
    with mpmath.workdps(dps):
        T, d = len(q), len(q[0])
        scale = 1 / mpmath.sqrt(d)
        out, lses = [], []
        for t in range(T):
            support = range(t + 1) if causal else range(T)
            s = [mpmath.fsum(mpmath.mpf(q[t][c]) * mpmath.mpf(k[i][c]) for c in range(d)) * scale
                 for i in support]
            w = [mpmath.exp(x) for x in s]
            z = mpmath.fsum(w)
            p = [x / z for x in w]
            lses.append(mpmath.log(z))
            row = []
            for j in range(d):
                b = mpmath.mpf(beta[j])
                vals = [mpmath.mpf(v[i][j]) for i in support]
                if b == 0:
                    row.append(mpmath.fsum(pi * vi for pi, vi in zip(p, vals)))
                else:
                    row.append(mpmath.log(mpmath.fsum(pi * mpmath.exp(b * vi) for pi, vi in zip(p, vals))) / b)
            out.append(row)
        return out, lses
