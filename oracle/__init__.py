"""Float64 CPU oracle for the Free Energy Mixer forward read (softmax prior).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use this package; the library under
``paper_2602_07160_gb300`` never does, and the two share no code.

The arithmetic lives in ``fem_oracle.c`` (plain C99, double precision,
optionally OpenMP over rows).  This module compiles it with gcc and calls it
through ctypes.  ``bruteforce.py`` holds an independent 50-digit mpmath
statement of the same read used to pin the C code.

Definition followed (Sec. 2.3, Eq. "fem-free-energy-main"; App. C,
Eq. "softmax-prior"): o_{t,j} = (1/beta_j) log sum_{i in M_t} p_t(i)
exp(beta_j v_{i,j}) with p_t = softmax(q_t . k_i / sqrt(d)) over the masked
support M_t, beta_j = 0 meaning the prior mean; lse_t = LSE_i s_{t,i}.

``gated_read`` composes it into the two-level gated read of Sec. 3
("Two-Level Gated FEM"): out = g ((1 - lambda) mu + lambda Fmax), mu the
beta = 0 read and Fmax the read at beta_max.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fem_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB_PATH) -> str:
    """Compile the C oracle (gcc -O2, no fast-math, OpenMP when available)."""
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    os.makedirs(os.path.dirname(out), exist_ok=True)
    base = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fno-fast-math", src, "-o", out, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    return out


def load(path: str | None = None):
    """Build if needed and return the ctypes handle of the oracle library."""
    global _lib
    if path is not None:
        return _bind(ctypes.CDLL(path))
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
        return _lib


def _bind(lib):
    dp = ctypes.POINTER(ctypes.c_double)
    i64 = ctypes.c_int64
    lib.fem_oracle_fwd.argtypes = [dp, dp, dp, dp, i64, i64, i64, i64, ctypes.c_int, dp, dp, ctypes.c_int]
    lib.fem_oracle_fwd.restype = ctypes.c_int
    lib.fem_oracle_rows.argtypes = [dp, dp, dp, dp, i64, i64, i64, i64, ctypes.c_int,
                                    ctypes.POINTER(ctypes.c_int64), i64, dp, dp, ctypes.c_int]
    lib.fem_oracle_rows.restype = ctypes.c_int
    lib.fem_oracle_max_threads.argtypes = []
    lib.fem_oracle_max_threads.restype = ctypes.c_int
    return lib


def _f64(x) -> np.ndarray:
    if hasattr(x, "detach"):  # torch tensor: upcast its exact values
        x = x.detach().to("cpu").double().numpy()
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def max_threads(lib=None) -> int:
    return int((lib or load()).fem_oracle_max_threads())


def fem_read(q, k, v, beta, causal: bool, nthreads: int = 0, lib=None):
    """The whole read.  q, k, v: [B, H, T, d]; beta: [H, d].

    Returns (out [B, H, T, d], lse [B, H, T]) as float64 numpy arrays."""
    lib = lib or load()
    q, k, v, beta = _f64(q), _f64(k), _f64(v), _f64(beta)
    B, H, T, d = q.shape
    assert k.shape == q.shape and v.shape == q.shape and beta.shape == (H, d)
    out = np.empty((B, H, T, d), dtype=np.float64)
    lse = np.empty((B, H, T), dtype=np.float64)
    rc = lib.fem_oracle_fwd(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), B, H, T, d, int(bool(causal)),
                            _ptr(out), _ptr(lse), int(nthreads))
    if rc != 0:
        raise ValueError(f"fem_oracle_fwd failed with code {rc}")
    return out, lse


def fem_read_rows(q, k, v, beta, causal: bool, rows, nthreads: int = 0, lib=None):
    """Selected rows.  rows: flat indices (b*H + h)*T + t.

    Returns (out [n, d], lse [n]) as float64 numpy arrays."""
    lib = lib or load()
    q, k, v, beta = _f64(q), _f64(k), _f64(v), _f64(beta)
    B, H, T, d = q.shape
    rows = np.ascontiguousarray(np.asarray(rows, dtype=np.int64))
    out = np.empty((rows.size, d), dtype=np.float64)
    lse = np.empty((rows.size,), dtype=np.float64)
    rc = lib.fem_oracle_rows(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), B, H, T, d, int(bool(causal)),
                             rows.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), rows.size,
                             _ptr(out), _ptr(lse), int(nthreads))
    if rc != 0:
        raise ValueError(f"fem_oracle_rows failed with code {rc}")
    return out, lse


def gated_read(q, k, v, beta_max, lam, gate, causal: bool, nthreads: int = 0, lib=None):
    """Two-level gated read (Sec. 3, "Two-Level Gated FEM").

    The inner gate interpolates the prior mean mu_{t,j} = sum_i p_t(i) v_{i,j}
    (the beta = 0 read) and the high-temperature branch Fmax_{t,j} (the read at
    beta_max_j), Eq. "inner-gate-main"; the outer gate scales the result,
    Eq. "fem-two-gates-main":

        out = gate * ((1 - lam) * mu + lam * Fmax)

    q, k, v, lam, gate: [B, H, T, d]; beta_max: [H, d] (> 0).  lam and gate
    are taken as given (the activations that produce them are upstream).
    Returns (out [B, H, T, d], lse [B, H, T]) as float64 numpy arrays."""
    lam, gate, beta_max = _f64(lam), _f64(gate), _f64(beta_max)
    mu, lse = fem_read(q, k, v, np.zeros_like(beta_max), causal, nthreads=nthreads, lib=lib)
    fmax, _ = fem_read(q, k, v, beta_max, causal, nthreads=nthreads, lib=lib)
    return gate * ((1.0 - lam) * mu + lam * fmax), lse


def gated_read_rows(q, k, v, beta_max, lam, gate, causal: bool, rows, nthreads: int = 0, lib=None):
    """gated_read on selected rows (flat indices (b*H + h)*T + t): the same
    composition of the beta = 0 and beta_max reads of those rows.

    lam, gate: [B, H, T, d].  Returns (out [n, d], lse [n]) as float64 numpy arrays."""
    rows = np.ascontiguousarray(np.asarray(rows, dtype=np.int64))
    beta_max = _f64(beta_max)
    d = beta_max.shape[-1]
    lam = _f64(lam).reshape(-1, d)[rows]
    gate = _f64(gate).reshape(-1, d)[rows]
    mu, lse = fem_read_rows(q, k, v, np.zeros_like(beta_max), causal, rows, nthreads=nthreads, lib=lib)
    fmax, _ = fem_read_rows(q, k, v, beta_max, causal, rows, nthreads=nthreads, lib=lib)
    return gate * ((1.0 - lam) * mu + lam * fmax), lse


def decode_read(q, k, v, beta, nthreads: int = 0, lib=None):
    """Decode read: one query per (b, h) against a cache of T keys and values
    holding the query's own key and value, i.e. row T - 1 of the causal read
    (Sec. 2.3, Eq. "fem-free-energy-main") whose query row is q.

    q: [B, H, d]; k, v: [B, H, T, d]; beta: [H, d].
    Returns (out [B, H, d], lse [B, H]) as float64 numpy arrays."""
    q, k = _f64(q), _f64(k)
    B, H, T, d = k.shape
    assert q.shape == (B, H, d)
    qf = np.zeros((B, H, T, d))
    qf[:, :, T - 1, :] = q
    rows = np.arange(B * H, dtype=np.int64) * T + (T - 1)
    out, lse = fem_read_rows(qf, k, v, beta, True, rows, nthreads=nthreads, lib=lib)
    return out.reshape(B, H, d), lse.reshape(B, H)


def gla_read(qf, kf, v, logdecay, beta):
    """FEM read over a gated-linear-attention prior (App. "Gated Linear
    Attention (GLA) Prior", Eq. "gla-score-appendix"), float64, O(T^2) per head.

    qf, kf: [B, H, T, m] nonnegative features (the caller's ReLU(RoPE(.)) + eps);
    v: [B, H, T, d]; logdecay: [B, H, T], g_t <= 0; beta: [H, d].
    s_t(i) = K_{t,i} <qf_t, kf_i> for i <= t with K_{t,i} = exp(sum_{r=i+1..t} g_r),
    p_t = s_t / Z_t, o_{t,j} = (1/beta_j) log sum_i p_t(i) exp(beta_j v_{i,j})
    (beta_j = 0: sum_i p_t(i) v_{i,j}).
    Returns (out [B, H, T, d], log Z [B, H, T]) as float64 numpy arrays."""
    from scipy.special import logsumexp

    qf, kf, v, g, beta = (_f64(x) for x in (qf, kf, v, logdecay, beta))
    B, H, T, m = qf.shape
    d = v.shape[-1]
    out = np.empty((B, H, T, d))
    logz = np.empty((B, H, T))
    tri = np.tril(np.ones((T, T), dtype=bool))
    for b in range(B):
        for h in range(H):
            G = np.cumsum(g[b, h])  # G_t = sum_{r <= t} g_r, so log K_{t,i} = G_t - G_i
            with np.errstate(divide="ignore"):
                logs = (G[:, None] - G[None, :]) + np.log(qf[b, h] @ kf[b, h].T)
            logs = np.where(tri, logs, -np.inf)
            lz = logsumexp(logs, axis=1)
            logz[b, h] = lz
            logp = logs - lz[:, None]
            p = np.exp(logp)
            for j in range(d):
                bj = beta[h, j]
                if bj == 0.0:
                    out[b, h, :, j] = p @ v[b, h, :, j]
                else:
                    out[b, h, :, j] = logsumexp(logp + bj * v[b, h, None, :, j], axis=1) / bj
    return out, logz


def tdc_conv(s, u):
    """The time-decay conditioner's convolution (App. "Low-rank Convolution:
    Time-Decay Conditioner (TDC)", Eq. "tdc-conv") by its definition, float64,
    O(T^2) per channel: h_t = sum_{i<=t} exp(-(s_{i+1} + ... + s_t)) u_i.

    s, u: [B, T, Hc].  Returns h [B, T, Hc] as a float64 numpy array."""
    s, u = _f64(s), _f64(u)
    B, T, Hc = s.shape
    cs = np.cumsum(s, axis=1)  # cs_t = s_1 + ... + s_t, so the kernel is exp(-(cs_t - cs_i))
    h = np.empty((B, T, Hc))
    for t in range(T):
        kern = np.exp(-(cs[:, t : t + 1, :] - cs[:, : t + 1, :]))
        h[:, t, :] = (kern * u[:, : t + 1, :]).sum(axis=1)
    return h


def fem_backward(q, k, v, beta, dout, causal: bool):
    """Gradients of the read (float64 numpy), from the paper's derivatives:

      dF_{t,j}/dv_{i,j}  = q_{t,i,j}                       (Prop. "app-geom", Eq. "app-grad-hess")
      dF_{t,j}/ds_{t,i}  = (q_{t,i,j} - p_{t,i}) / beta_j  (Prop. "app-bounds" (iv), normalised logits)
      dF_{t,j}/dbeta_j   = KL(q_{t,.,j} || p_t) / beta_j^2 (Eq. "app-beta-deriv")

    with p_t = softmax(s_t), q_{t,.,j} proportional to p_t exp(beta_j v_{.,j}),
    s_{t,i} = q_t . k_i / sqrt(d), and at beta_j = 0 the limits
    (q - p)/beta -> p (v - mu) and KL/beta^2 -> Var_p(v)/2.  Chained through
    the scores: dQ = dS K / sqrt(d), dK = dS^T Q / sqrt(d) with
    dS_{t,i} = sum_j dout_{t,j} dF_{t,j}/ds_{t,i}.
    q, k, v, dout: [B, H, T, d]; beta: [H, d].
    Returns (dq, dk, dv [B, H, T, d], dbeta [H, d]) as float64 numpy arrays."""
    from scipy.special import logsumexp

    q, k, v, beta, dout = (_f64(x) for x in (q, k, v, beta, dout))
    B, H, T, d = q.shape
    dq, dk, dv = np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)
    dbeta = np.zeros((H, d))
    mask = np.tril(np.ones((T, T), dtype=bool)) if causal else np.ones((T, T), dtype=bool)
    for b in range(B):
        for h in range(H):
            s = (q[b, h] @ k[b, h].T) / np.sqrt(d)
            s = np.where(mask, s, -np.inf)
            lse = logsumexp(s, axis=1)
            p = np.exp(s - lse[:, None])
            dS = np.zeros((T, T))
            for j in range(d):
                bj, vj, gj = beta[h, j], v[b, h, :, j], dout[b, h, :, j]
                if bj == 0.0:
                    mu = p @ vj
                    qj = p
                    dsj = p * (vj[None, :] - mu[:, None])
                    kl_b2 = 0.5 * (p * (vj[None, :] - mu[:, None]) ** 2).sum(axis=1)
                else:
                    a = np.where(mask, s + bj * vj[None, :], -np.inf)
                    G = logsumexp(a, axis=1)
                    qj = np.exp(a - G[:, None])
                    dsj = (qj - p) / bj
                    with np.errstate(divide="ignore", invalid="ignore"):
                        kl = np.where(qj > 0, qj * (np.log(qj) - np.log(np.where(p > 0, p, 1.0))), 0.0).sum(axis=1)
                    kl_b2 = kl / bj**2
                dS += gj[:, None] * dsj
                dv[b, h, :, j] = qj.T @ gj
                dbeta[h, j] += gj @ kl_b2
            dq[b, h] = dS @ k[b, h] / np.sqrt(d)
            dk[b, h] = dS.T @ q[b, h] / np.sqrt(d)
    return dq, dk, dv, dbeta
