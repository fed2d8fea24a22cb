"""The oracle's decode read is the last row of its causal read (CPU only)."""
import numpy as np

import oracle
from tests.oracle_pins import _inputs


def test_decode_is_the_last_causal_row():
    q, k, v, beta = _inputs(31, 2, 2, 11, 6, beta_lo=1e-3, beta_hi=50)
    beta[0, 1] = 0.0
    full, full_lse = oracle.fem_read(q, k, v, beta, True)
    out, lse = oracle.decode_read(q[:, :, -1, :], k, v, beta)
    assert np.array_equal(out, full[:, :, -1, :]) and np.array_equal(lse, full_lse[:, :, -1])


def test_decode_single_key_returns_its_value():
    """T = 1: the only key gets all the prior mass, so o = v_0 for every beta (P1)."""
    q, k, v, beta = _inputs(32, 1, 3, 1, 5)
    out, _ = oracle.decode_read(q[:, :, 0, :], k, v, beta)
    assert np.allclose(out, v[:, :, 0, :], rtol=0, atol=1e-12)
