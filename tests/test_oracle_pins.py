"""The float64 oracle against what the paper and the mathematics fix (CPU only)."""
import numpy as np
import pytest

import oracle
from tests import oracle_pins


@pytest.fixture(scope="module")
def lib():
    return oracle.load()


@pytest.mark.parametrize("check", oracle_pins.ALL_CHECKS, ids=lambda c: c.__name__)
def test_pin(lib, check):
    check(lib)


def test_bruteforce_live(lib):
    """P8 with a fresh 50-digit evaluation (where mpmath is installed)."""
    pytest.importorskip("mpmath")
    from oracle.bruteforce import fem_read_mp

    r = np.random.default_rng(123)
    T, d = 7, 3
    q, k, v = (r.standard_normal((1, 1, T, d)) for _ in range(3))
    beta = np.array([[1e-3, 3.0, 250.0]])
    for causal in (True, False):
        out, lse = oracle.fem_read(q, k, v, beta, causal, lib=lib)
        mo, ml = fem_read_mp(q[0, 0].tolist(), k[0, 0].tolist(), v[0, 0].tolist(), beta[0].tolist(), causal)
        np.testing.assert_allclose(out[0, 0], np.array(mo, dtype=float), rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(lse[0, 0], np.array(ml, dtype=float), rtol=1e-13, atol=1e-13)


def test_rows_match_full(lib):
    """The sampled-row entry point returns the same rows as the full read."""
    r = np.random.default_rng(5)
    B, H, T, d = 2, 3, 17, 4
    q, k, v = (r.standard_normal((B, H, T, d)) for _ in range(3))
    beta = np.exp(r.uniform(-3, 3, size=(H, d)))
    for causal in (True, False):
        out, lse = oracle.fem_read(q, k, v, beta, causal, lib=lib)
        rows = r.choice(B * H * T, size=20, replace=False)
        o_r, l_r = oracle.fem_read_rows(q, k, v, beta, causal, rows, lib=lib)
        np.testing.assert_array_equal(o_r, out.reshape(-1, d)[rows])
        np.testing.assert_array_equal(l_r, lse.reshape(-1)[rows])


def test_rejects_negative_beta(lib):
    q = np.zeros((1, 1, 2, 2))
    with pytest.raises(ValueError):
        oracle.fem_read(q, q, q, np.array([[1.0, -1.0]]), True, lib=lib)
