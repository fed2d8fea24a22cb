"""Python binding of libfem.so (argument marshalling only).

Every function here checks shapes, dtypes and devices of torch tensors,
passes raw pointers and sizes to the C ABI of ``include/fem.h`` and raises on
a non-zero status.  All arithmetic of the read runs in the library's CUDA
kernels; there is no other implementation behind these names.  If the
library is not built, ``load()`` raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libfem.so")
_lock = threading.Lock()
_lib = None

STATUS = {0: "FEM_OK", 1: "FEM_ERR_INVALID_ARG", 2: "FEM_ERR_UNSUPPORTED", 3: "FEM_ERR_CUDA",
          4: "FEM_ERR_TIMEOUT", 5: "FEM_ERR_NO_MEMORY"}

EXPORTS = ["fem_fwd", "fem_fwd_ws", "fem_fwd_workspace_bytes", "fem_fwd_f32", "fem_fwd_host",
           "fem_check_device_error", "fem_last_fixup_rows", "fem_set_kernel_events", "fem_status_str",
           "fem_fwd_noalloc", "fem_fwd_gated", "fem_decode", "fem_gla_fwd", "fem_tdc_conv", "fem_bwd_f32",
           "fem_probe_wait_timeout", "fem_attn_fwd", "fem_gla_fwd_tc"]


class FemError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} returned {STATUS.get(status, status)}")
        self.status = status


def library_path() -> str:
    return _LIB_PATH


def load(path: str | None = None):
    """Load libfem.so (built by ``paper_2602_07160_gb300.build``) and bind its ABI."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or _LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is not built; run `python -m paper_2602_07160_gb300.build`")
        lib = ctypes.CDLL(p)
        vp, i, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        sig = [vp, vp, vp, vp, vp, vp, i, i, i, i, i]
        lib.fem_fwd.argtypes = sig + [vp]
        lib.fem_fwd_ws.argtypes = sig + [vp, sz, vp]
        lib.fem_fwd_f32.argtypes = sig + [vp]
        lib.fem_fwd_host.argtypes = sig + [vp]
        lib.fem_fwd_noalloc.argtypes = sig + [vp]
        lib.fem_fwd_noalloc.restype = i
        lib.fem_fwd_gated.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, i, i, i, i, i, vp]
        lib.fem_fwd_gated.restype = i
        lib.fem_decode.argtypes = [vp, vp, vp, vp, vp, vp, i, i, i, i, vp]
        lib.fem_decode.restype = i
        lib.fem_gla_fwd.argtypes = [vp, vp, vp, vp, vp, vp, vp, i, i, i, i, i, vp]
        lib.fem_gla_fwd.restype = i
        lib.fem_gla_fwd_tc.argtypes = [vp, vp, vp, vp, vp, vp, vp, i, i, i, i, i, vp]
        lib.fem_gla_fwd_tc.restype = i
        lib.fem_tdc_conv.argtypes = [vp, vp, vp, i, i, i, vp]
        lib.fem_tdc_conv.restype = i
        lib.fem_bwd_f32.argtypes = [vp] * 11 + [i, i, i, i, i, vp]
        lib.fem_bwd_f32.restype = i
        lib.fem_fwd_workspace_bytes.argtypes = [i, i, i, i, i]
        lib.fem_fwd_workspace_bytes.restype = sz
        lib.fem_check_device_error.argtypes = [vp]
        lib.fem_attn_fwd.argtypes = [vp, vp, vp, vp, vp, i, i, i, i, i, vp]
        lib.fem_attn_fwd.restype = i
        lib.fem_probe_wait_timeout.argtypes = [ctypes.c_uint, vp]
        lib.fem_probe_wait_timeout.restype = i
        lib.fem_last_fixup_rows.argtypes = [vp]
        lib.fem_set_kernel_events.argtypes = [vp, vp]
        lib.fem_set_kernel_events.restype = i
        lib.fem_status_str.argtypes = [i]
        lib.fem_status_str.restype = ctypes.c_char_p
        for name in ("fem_fwd", "fem_fwd_ws", "fem_fwd_f32", "fem_fwd_host", "fem_check_device_error",
                     "fem_last_fixup_rows"):
            getattr(lib, name).restype = i
        if path is None:
            _lib = lib
        return lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream, device):
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return ctypes.c_void_p(stream.cuda_stream)


def _check_qkvb(q, k, v, beta, dtype, device_type):
    if q.dim() != 4 or k.shape != q.shape or v.shape != q.shape:
        raise ValueError("q, k, v must share the shape [B, H, T, d]")
    B, H, T, d = q.shape
    if beta.shape != (H, d) or beta.dtype != torch.float32:
        raise ValueError("beta must be float32 [H, d]")
    for name, t in (("q", q), ("k", k), ("v", v), ("beta", beta)):
        if t.dtype != (torch.float32 if name == "beta" else dtype):
            raise ValueError(f"{name} has dtype {t.dtype}")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
        if t.device.type != device_type:
            raise ValueError(f"{name} must be on {device_type}")
    return B, H, T, d


def _outputs(q, out, lse, device):
    B, H, T, d = q.shape
    if out is None:
        out = torch.empty((B, H, T, d), dtype=torch.float32, device=device)
    if lse is None:
        lse = torch.empty((B, H, T), dtype=torch.float32, device=device)
    if out.shape != (B, H, T, d) or out.dtype != torch.float32 or not out.is_contiguous():
        raise ValueError("out must be contiguous float32 [B, H, T, d]")
    if lse is not False and (lse.shape != (B, H, T) or lse.dtype != torch.float32 or not lse.is_contiguous()):
        raise ValueError("lse must be contiguous float32 [B, H, T]")
    return out, lse


def fem_fwd(q, k, v, beta, causal: bool = True, out=None, lse=None, stream=None):
    """The read on bf16 CUDA tensors (tensor-core path).  Returns (out, lse).

    Pass ``lse=False`` to skip the log-normaliser output."""
    B, H, T, d = _check_qkvb(q, k, v, beta, torch.bfloat16, "cuda")
    out, lse = _outputs(q, out, lse, q.device)
    rc = load().fem_fwd(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), _ptr(out), None if lse is False else _ptr(lse),
                        B, H, T, d, int(bool(causal)), _stream(stream, q.device))
    if rc != 0:
        raise FemError("fem_fwd", rc)
    return out, (None if lse is False else lse)


def fem_attn_fwd(q, k, v, causal: bool = True, out=None, lse=None, stream=None):
    """Plain softmax attention on the same tensor-core kernel (the comparator; bf16 CUDA
    tensors).  Returns (out, lse)."""
    beta = torch.zeros((q.shape[1], q.shape[3]), dtype=torch.float32, device=q.device)  # shape check only
    B, H, T, d = _check_qkvb(q, k, v, beta, torch.bfloat16, "cuda")
    out, lse = _outputs(q, out, lse, q.device)
    rc = load().fem_attn_fwd(_ptr(q), _ptr(k), _ptr(v), _ptr(out), None if lse is False else _ptr(lse),
                             B, H, T, d, int(bool(causal)), _stream(stream, q.device))
    if rc != 0:
        raise FemError("fem_attn_fwd", rc)
    return out, (None if lse is False else lse)


def workspace_bytes(B: int, H: int, T: int, d: int, causal: bool = True) -> int:
    return int(load().fem_fwd_workspace_bytes(B, H, T, d, int(bool(causal))))


def fem_fwd_ws(q, k, v, beta, workspace, causal: bool = True, out=None, lse=None, stream=None):
    """fem_fwd with a caller-owned uint8 CUDA workspace of ``workspace_bytes()`` bytes."""
    B, H, T, d = _check_qkvb(q, k, v, beta, torch.bfloat16, "cuda")
    out, lse = _outputs(q, out, lse, q.device)
    rc = load().fem_fwd_ws(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), _ptr(out), None if lse is False else _ptr(lse),
                           B, H, T, d, int(bool(causal)), _ptr(workspace), workspace.numel() * workspace.element_size(),
                           _stream(stream, q.device))
    if rc != 0:
        raise FemError("fem_fwd_ws", rc)
    return out, (None if lse is False else lse)


def fem_fwd_gated(q, k, v, beta_max, lam, gate, causal: bool = True, out=None, lse=None, stream=None):
    """The two-level gated read on bf16 CUDA tensors: out = gate * ((1 - lam) mu + lam Fmax).

    lam and gate are float32 [B, H, T, d] (already activated); beta_max is float32 [H, d].
    Returns (out, lse)."""
    B, H, T, d = _check_qkvb(q, k, v, beta_max, torch.bfloat16, "cuda")
    for name, t in (("lam", lam), ("gate", gate)):
        if t.shape != q.shape or t.dtype != torch.float32 or not t.is_contiguous() or t.device != q.device:
            raise ValueError(f"{name} must be a contiguous float32 tensor shaped like q on its device")
    out, lse = _outputs(q, out, lse, q.device)
    rc = load().fem_fwd_gated(_ptr(q), _ptr(k), _ptr(v), _ptr(beta_max), _ptr(lam), _ptr(gate), _ptr(out),
                              None if lse is False else _ptr(lse), B, H, T, d, int(bool(causal)),
                              _stream(stream, q.device))
    if rc != 0:
        raise FemError("fem_fwd_gated", rc)
    return out, (None if lse is False else lse)


def fem_decode(q, k, v, beta, out=None, lse=None, stream=None):
    """Decode read on bf16 CUDA tensors: q [B, H, d] against the cache k, v [B, H, T, d].

    Returns (out [B, H, d] float32, lse [B, H] float32)."""
    if q.dim() != 3 or k.dim() != 4 or k.shape != v.shape or k.shape[:2] != q.shape[:2] or k.shape[3] != q.shape[2]:
        raise ValueError("q must be [B, H, d] and k, v [B, H, T, d]")
    B, H, T, d = k.shape
    for name, t in (("q", q), ("k", k), ("v", v)):
        if t.dtype != torch.bfloat16 or not t.is_contiguous() or t.device.type != "cuda":
            raise ValueError(f"{name} must be a contiguous bf16 CUDA tensor")
    if beta.shape != (H, d) or beta.dtype != torch.float32 or not beta.is_contiguous() or beta.device != q.device:
        raise ValueError("beta must be float32 [H, d] on q's device")
    if out is None:
        out = torch.empty((B, H, d), dtype=torch.float32, device=q.device)
    if lse is None:
        lse = torch.empty((B, H), dtype=torch.float32, device=q.device)
    rc = load().fem_decode(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), _ptr(out), None if lse is False else _ptr(lse),
                           B, H, T, d, _stream(stream, q.device))
    if rc != 0:
        raise FemError("fem_decode", rc)
    return out, (None if lse is False else lse)


def fem_gla_fwd_tc(qf, kf, v, logdecay, beta, out=None, logz=None, stream=None):
    """fem_gla_fwd chunked on the tensor cores (m = d = 64; bf16 operands, fp32 state)."""
    return fem_gla_fwd(qf, kf, v, logdecay, beta, out=out, logz=logz, stream=stream, _entry="fem_gla_fwd_tc")


def fem_gla_fwd(qf, kf, v, logdecay, beta, out=None, logz=None, stream=None, _entry="fem_gla_fwd"):
    """The read over a GLA prior on fp32 CUDA tensors.

    qf, kf: [B, H, T, m] nonnegative features; v: [B, H, T, d]; logdecay: [B, H, T] (<= 0);
    beta: [H, d].  Returns (out [B, H, T, d], logz [B, H, T])."""
    if qf.dim() != 4 or kf.shape != qf.shape or v.dim() != 4 or v.shape[:3] != qf.shape[:3]:
        raise ValueError("qf, kf must be [B, H, T, m] and v [B, H, T, d]")
    B, H, T, m = qf.shape
    d = v.shape[3]
    for name, t in (("qf", qf), ("kf", kf), ("v", v), ("logdecay", logdecay), ("beta", beta)):
        if t.dtype != torch.float32 or not t.is_contiguous() or t.device != qf.device or t.device.type != "cuda":
            raise ValueError(f"{name} must be a contiguous float32 CUDA tensor on qf's device")
    if logdecay.shape != (B, H, T) or beta.shape != (H, d):
        raise ValueError("logdecay must be [B, H, T] and beta [H, d]")
    if out is None:
        out = torch.empty((B, H, T, d), dtype=torch.float32, device=qf.device)
    if logz is None:
        logz = torch.empty((B, H, T), dtype=torch.float32, device=qf.device)
    rc = getattr(load(), _entry)(_ptr(qf), _ptr(kf), _ptr(v), _ptr(logdecay), _ptr(beta), _ptr(out),
                                 None if logz is False else _ptr(logz), B, H, T, m, d, _stream(stream, qf.device))
    if rc != 0:
        raise FemError(_entry, rc)
    return out, (None if logz is False else logz)


def fem_tdc_conv(s, u, out=None, stream=None):
    """The time-decay conditioner's convolution h_t = exp(-s_t) h_{t-1} + u_t on fp32
    CUDA tensors s, u of shape [B, T, Hc] (s >= 0).  Returns h."""
    if s.dim() != 3 or u.shape != s.shape:
        raise ValueError("s and u must share the shape [B, T, Hc]")
    for name, t in (("s", s), ("u", u)):
        if t.dtype != torch.float32 or not t.is_contiguous() or t.device.type != "cuda" or t.device != s.device:
            raise ValueError(f"{name} must be a contiguous float32 CUDA tensor on s's device")
    B, T, Hc = s.shape
    if out is None:
        out = torch.empty_like(s)
    rc = load().fem_tdc_conv(_ptr(s), _ptr(u), _ptr(out), B, T, Hc, _stream(stream, s.device))
    if rc != 0:
        raise FemError("fem_tdc_conv", rc)
    return out


def fem_bwd_f32(q, k, v, beta, out, lse, dout, causal: bool = True, stream=None):
    """Gradients of the fp32 read from its saved (out, lse) and the output cotangent dout.

    Returns (dq, dk, dv [B, H, T, d], dbeta [H, d] summed over batch and time)."""
    B, H, T, d = _check_qkvb(q, k, v, beta, torch.float32, "cuda")
    for name, t, shape in (("out", out, q.shape), ("dout", dout, q.shape), ("lse", lse, q.shape[:3])):
        if t.shape != shape or t.dtype != torch.float32 or not t.is_contiguous() or t.device != q.device:
            raise ValueError(f"{name} must be a contiguous float32 tensor of shape {tuple(shape)} on q's device")
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    dbeta = torch.empty_like(beta)
    rc = load().fem_bwd_f32(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), _ptr(out), _ptr(lse), _ptr(dout), _ptr(dq),
                            _ptr(dk), _ptr(dv), _ptr(dbeta), B, H, T, d, int(bool(causal)), _stream(stream, q.device))
    if rc != 0:
        raise FemError("fem_bwd_f32", rc)
    return dq, dk, dv, dbeta


def fem_fwd_f32(q, k, v, beta, causal: bool = True, out=None, lse=None, stream=None):
    """The read on fp32 CUDA tensors (CUDA-core path).  Returns (out, lse)."""
    B, H, T, d = _check_qkvb(q, k, v, beta, torch.float32, "cuda")
    out, lse = _outputs(q, out, lse, q.device)
    rc = load().fem_fwd_f32(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), _ptr(out), None if lse is False else _ptr(lse),
                            B, H, T, d, int(bool(causal)), _stream(stream, q.device))
    if rc != 0:
        raise FemError("fem_fwd_f32", rc)
    return out, (None if lse is False else lse)


def fem_fwd_host(q, k, v, beta, causal: bool = True, out=None, lse=None, stream=None, device=None):
    """The read on HOST (ideally pinned) bf16 tensors: copies in, computes, copies out."""
    B, H, T, d = _check_qkvb(q, k, v, beta, torch.bfloat16, "cpu")
    # outputs it allocates are pinned: copies into pageable memory do not overlap the read
    if out is None:
        out = torch.empty(q.shape, dtype=torch.float32).pin_memory()
    if lse is None:
        lse = torch.empty(q.shape[:3], dtype=torch.float32).pin_memory()
    out, lse = _outputs(q, out, lse, "cpu")
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    rc = load().fem_fwd_host(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), _ptr(out), None if lse is False else _ptr(lse),
                             B, H, T, d, int(bool(causal)), _stream(stream, dev))
    if rc != 0:
        raise FemError("fem_fwd_host", rc)
    return out, (None if lse is False else lse)


def fem_fwd_noalloc(q, k, v, beta, causal: bool = True, out=None, lse=None, stream=None):
    """fem_fwd without device allocation (the library's fixed 16 MiB scratch).

    For callers that may not allocate device memory during the read.  ``out``
    and ``lse`` should be passed preallocated by such callers.  Calls that
    overlap on the GPU share the scratch and race."""
    B, H, T, d = _check_qkvb(q, k, v, beta, torch.bfloat16, "cuda")
    out, lse = _outputs(q, out, lse, q.device)
    rc = load().fem_fwd_noalloc(_ptr(q), _ptr(k), _ptr(v), _ptr(beta), _ptr(out),
                                None if lse is False else _ptr(lse), B, H, T, d, int(bool(causal)),
                                _stream(stream, q.device))
    if rc != 0:
        raise FemError("fem_fwd_noalloc", rc)
    return out, (None if lse is False else lse)


def probe_wait_timeout(limit_us: int, stream=None, device=None):
    """Enqueue the library's wait probe: a bounded wait on an mbarrier nothing completes,
    which gives up after limit_us microseconds and records a timeout in the error word."""
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    rc = load().fem_probe_wait_timeout(int(limit_us), _stream(stream, dev))
    if rc != 0:
        raise FemError("fem_probe_wait_timeout", rc)


def check_device_error(stream=None, device=None):
    """Synchronise and raise FemError if a kernel gave up on a bounded wait."""
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    rc = load().fem_check_device_error(_stream(stream, dev))
    if rc != 0:
        raise FemError("fem_check_device_error", rc)


def set_kernel_events(start, stop):
    """Have the next bf16 read of this thread record torch CUDA events around its tensor-core kernel."""
    load().fem_set_kernel_events(ctypes.c_void_p(start.cuda_event), ctypes.c_void_p(stop.cuda_event))


def last_fixup_rows(stream=None, device=None) -> int:
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    return int(load().fem_last_fixup_rows(_stream(stream, dev)))
