"""The C ABI library builds, loads and exports what include/fem.h declares (CPU only)."""
import ctypes
import os
import re

import pytest

from paper_2602_07160_gb300 import build, fem

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "fem.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(fem_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return fem.load()


def test_header_declares_the_boundary():
    names = _declared()
    assert names == sorted(fem.EXPORTS), names


def test_every_declared_symbol_is_exported(lib):
    raw = ctypes.CDLL(fem.library_path())
    for name in _declared():
        assert hasattr(raw, name), f"{name} missing from libfem.so"


def test_status_strings(lib):
    for code, name in fem.STATUS.items():
        assert lib.fem_status_str(code).decode() == name
    assert lib.fem_status_str(99).decode() == "FEM_ERR_UNKNOWN"


def test_workspace_bytes(lib):
    assert lib.fem_fwd_workspace_bytes(0, 1, 1, 64, 1) == 0
    assert lib.fem_fwd_workspace_bytes(1, 1, -3, 64, 1) == 0
    a = lib.fem_fwd_workspace_bytes(4, 16, 8192, 128, 1)
    b = lib.fem_fwd_workspace_bytes(4, 16, 8192, 128, 0)
    # both forms of the read keep the same arrays (the guard's fix-up list serves both)
    assert a == b > 0 and a % 256 == 0
    assert lib.fem_fwd_workspace_bytes(4, 16, 8192, 64, 1) < a


def _call(lib, fn, q=16, k=16, v=16, beta=16, out=16, lse=0, B=1, H=1, T=8, d=64, causal=1):
    p = lambda x: ctypes.c_void_p(x) if x else None  # noqa: E731  fake, never dereferenced
    return getattr(lib, fn)(p(q), p(k), p(v), p(beta), p(out), p(lse), B, H, T, d, causal, None)


@pytest.mark.parametrize("fn", ["fem_fwd", "fem_fwd_f32", "fem_fwd_host"])
def test_argument_errors_are_synchronous(lib, fn):
    """Invalid arguments are rejected on the host before any CUDA call."""
    assert _call(lib, fn, q=0) == 1
    assert _call(lib, fn, beta=0) == 1
    assert _call(lib, fn, out=0) == 1
    assert _call(lib, fn, B=0) == 1
    assert _call(lib, fn, T=-1) == 1
    assert _call(lib, fn, causal=2) == 1
    if fn != "fem_fwd_host":
        assert _call(lib, fn, q=24) == 1  # not 16-byte aligned


def test_unsupported_head_dim(lib):
    assert _call(lib, "fem_fwd", d=96) == 2
    assert _call(lib, "fem_fwd", d=8) == 2
    assert _call(lib, "fem_fwd_host", d=48) == 2
    assert _call(lib, "fem_fwd_f32", d=300) == 2


def test_small_head_dims_take_no_workspace(lib):
    """bf16 d in {16, 32} runs on CUDA cores: only the fix-up counters' 256 bytes."""
    lib.fem_fwd_workspace_bytes.restype = ctypes.c_size_t
    for d in (16, 32):
        assert lib.fem_fwd_workspace_bytes(4, 16, 8192, d, 1) == 256
    assert lib.fem_fwd_workspace_bytes(4, 16, 8192, 64, 1) > (1 << 20)


@pytest.mark.parametrize("fn", ["fem_fwd", "fem_fwd_host", "fem_fwd_noalloc"])
def test_sequence_beyond_the_tensor_core_limit_is_refused_synchronously(lib, fn):
    """T above 2^20 keys (the tensor-core kernel's bitmap of key tiles) is refused on the host
    with FEM_ERR_UNSUPPORTED before any CUDA call (the pointers are fakes)."""
    assert _call(lib, fn, T=(1 << 20) + 1) == 2


def test_workspace_variant_refuses_long_sequence_synchronously(lib):
    p = lambda x: ctypes.c_void_p(x) if x else None  # noqa: E731  fake, never dereferenced
    T = (1 << 20) + 1
    assert lib.fem_fwd_ws(p(16), p(16), p(16), p(16), p(16), None, 1, 1, T, 64, 1, p(256), 1 << 40, None) == 2


def test_binding_fails_loudly_without_library(tmp_path):
    with pytest.raises(RuntimeError):
        fem.load(str(tmp_path / "missing.so"))


def test_gated_argument_errors_are_synchronous(lib):
    """fem_fwd_gated rejects bad gates and head dimensions before any CUDA call."""
    p = lambda x: ctypes.c_void_p(x) if x else None  # noqa: E731  fake, never dereferenced
    f = lib.fem_fwd_gated
    ok = dict(q=16, k=16, v=16, b=16, lam=16, g=16, out=16)

    def call(d=64, **kw):
        a = dict(ok, **kw)
        return f(p(a["q"]), p(a["k"]), p(a["v"]), p(a["b"]), p(a["lam"]), p(a["g"]), p(a["out"]), None,
                 1, 1, 8, d, 1, None)

    assert call(lam=0) == 1
    assert call(g=0) == 1
    assert call(lam=24) == 1  # not 16-byte aligned
    assert call(b=0) == 1
    assert call(d=32) == 2
    assert f(p(16), p(16), p(16), p(16), p(16), p(16), p(16), None, 1, 1, (1 << 20) + 1, 64, 1, None) == 2


def test_decode_argument_errors_are_synchronous(lib):
    """fem_decode rejects bad pointers, sizes and head dimensions before any CUDA call."""
    p = lambda x: ctypes.c_void_p(x) if x else None  # noqa: E731  fake, never dereferenced
    f = lib.fem_decode
    assert f(None, p(16), p(16), p(16), p(16), None, 1, 1, 8, 64, None) == 1
    assert f(p(16), p(16), p(16), p(16), p(24), None, 1, 1, 8, 64, None) == 1
    assert f(p(16), p(16), p(16), p(16), p(16), None, 1, 1, 0, 64, None) == 1
    assert f(p(16), p(16), p(16), p(16), p(16), None, 1, 1, 8, 96, None) == 2


def test_gla_argument_errors_are_synchronous(lib):
    """fem_gla_fwd rejects bad pointers, sizes and feature widths before any CUDA call."""
    p = lambda x: ctypes.c_void_p(x) if x else None  # noqa: E731  fake, never dereferenced
    f = lib.fem_gla_fwd

    def call(qf=16, m=32, d=8, T=4):
        return f(p(qf), p(16), p(16), p(16), p(16), p(16), None, 1, 1, T, m, d, None)

    assert call(qf=0) == 1
    assert call(qf=8) == 1  # not 16-byte aligned
    assert call(T=0) == 1
    assert call(m=48) == 2
    assert call(d=200) == 2


def test_tdc_argument_errors_are_synchronous(lib):
    """fem_tdc_conv rejects bad pointers and sizes before any CUDA call."""
    p = lambda x: ctypes.c_void_p(x) if x else None  # noqa: E731  fake, never dereferenced
    f = lib.fem_tdc_conv
    assert f(None, p(16), p(16), 1, 8, 4, None) == 1
    assert f(p(16), p(16), p(18), 1, 8, 4, None) == 1
    assert f(p(16), p(16), p(16), 1, 0, 4, None) == 1


def test_backward_argument_errors_are_synchronous(lib):
    """fem_bwd_f32 rejects missing buffers and head dimensions before any CUDA call."""
    p = lambda x: ctypes.c_void_p(x) if x else None  # noqa: E731  fake, never dereferenced
    f = lib.fem_bwd_f32

    def call(lse=16, dq=16, d=64):
        return f(p(16), p(16), p(16), p(16), p(16), p(lse), p(16), p(dq), p(16), p(16), p(16), 1, 1, 8, d, 1, None)

    assert call(lse=0) == 1
    assert call(dq=0) == 1
    assert call(dq=8) == 1
    assert call(d=300) == 2


def test_wait_probe_argument_errors_are_synchronous(lib):
    """fem_probe_wait_timeout rejects a limit of 0 or above one second before any CUDA call."""
    assert lib.fem_probe_wait_timeout(0, None) == 1
    assert lib.fem_probe_wait_timeout(1_000_001, None) == 1
