"""Thin ctypes binding of the HLA C ABI (include/hla.h).

Every function has the name of the C entry point it calls and does argument
marshalling only: it checks tensor shapes/devices, takes raw pointers and the
current CUDA stream from PyTorch, and calls the library.  All arithmetic runs in
the CUDA kernels of ``libhla.so``.  If the library is missing the calls raise;
there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libhla.so")

HLA_OK, HLA_ERR_INVALID_ARGUMENT, HLA_ERR_UNSUPPORTED, HLA_ERR_CUDA, HLA_ERR_TIMEOUT, HLA_ERR_WORKSPACE = range(6)
HLA_F32, HLA_BF16 = 0, 1

# every symbol include/hla.h declares
EXPORTS = ("hla_status_string", "hla_last_error", "hla2_state_floats", "hla2_workspace_bytes", "hla2_forward",
           "hla2_forward_path", "hla2_step", "hla3_state_floats", "hla3_workspace_bytes", "hla3_forward",
           "hla3_forward_path", "hla2_backward_path",
           "hla2_forward_noalloc", "hla_poll_error_noalloc", "hla_poll_error", "hla2_sde_state_floats",
           "hla2_state_to_sde", "hla2_step_sde", "ahla_state_floats", "ahla_workspace_bytes", "ahla_forward",
           "ahla_step", "hla2_backward_workspace_bytes", "hla2_backward", "ahla_forward_path")

_lib = None


class HLAError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        detail = lib().hla_last_error().decode(errors="replace")
        super().__init__("%s: %s%s" % (where, hla_status_string(code), (" (" + detail + ")") if detail else ""))


def lib():
    """Load libhla.so (built by ``paper_2510_27258_gb300.build``); raise if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libhla.so is not built: run `python -c \"import __graft_entry__ as g; g.build()\"` "
                               "or `python paper_2510_27258_gb300/build.py`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i, f, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
        L.hla_status_string.argtypes = [i]
        L.hla_status_string.restype = ctypes.c_char_p
        L.hla_last_error.argtypes = []
        L.hla_last_error.restype = ctypes.c_char_p
        for name in ("hla2_state_floats", "hla3_state_floats"):
            getattr(L, name).argtypes = [i, i]
            getattr(L, name).restype = sz
        L.ahla_state_floats.argtypes = [i, i]
        L.ahla_state_floats.restype = sz
        L.ahla_forward.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, f, i, vp, vp, vp, sz, vp]
        L.ahla_forward.restype = i
        L.ahla_step.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, f, vp, vp]
        L.ahla_step.restype = i
        L.ahla_forward_path.argtypes = [i, i, i, i, i, i, i, i, i, i]
        L.ahla_forward_path.restype = i
        L.hla2_backward_path.argtypes = [i, i, i, i, i, i, i, i]
        L.hla2_backward_path.restype = i
        L.hla2_backward.argtypes = [vp, vp, vp, vp, vp, vp, vp, i, i, i, i, i, i, i, f, i, vp, sz, vp]
        L.hla2_backward.restype = i
        for name in ("hla2_workspace_bytes", "hla3_workspace_bytes", "ahla_workspace_bytes",
                     "hla2_backward_workspace_bytes"):
            getattr(L, name).argtypes = [i, i, i, i, i, i, i]
            getattr(L, name).restype = sz
        for name in ("hla2_forward", "hla3_forward"):
            getattr(L, name).argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, i, f, i, vp, vp, vp, sz, vp]
            getattr(L, name).restype = i
        L.hla2_forward_noalloc.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, i, f, i, vp, vp]
        L.hla2_forward_noalloc.restype = i
        for name in ("hla2_forward_path", "hla3_forward_path"):
            getattr(L, name).argtypes = [i, i, i, i, i, i, i, i, i, i, i, ctypes.POINTER(i)]
            getattr(L, name).restype = i
        L.hla2_step.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, f, vp, vp]
        L.hla2_step.restype = i
        L.hla_poll_error.argtypes = [vp, vp]
        L.hla_poll_error.restype = i
        L.hla_poll_error_noalloc.argtypes = [vp]
        L.hla_poll_error_noalloc.restype = i
        L.hla2_sde_state_floats.argtypes = [i, i]
        L.hla2_sde_state_floats.restype = sz
        L.hla2_state_to_sde.argtypes = [vp, vp, i, i, i, i, vp]
        L.hla2_state_to_sde.restype = i
        L.hla2_step_sde.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, f, vp, vp]
        L.hla2_step_sde.restype = i
        _lib = L
    return _lib


def hla_status_string(code: int) -> str:
    return lib().hla_status_string(int(code)).decode()


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return HLA_BF16
    if t.dtype == torch.float32:
        return HLA_F32
    raise TypeError("HLA tokens must be bfloat16 or float32, got %s" % t.dtype)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(code: int, where: str):
    if code != HLA_OK:
        raise HLAError(code, where)


def hla2_state_floats(d: int, dv: int) -> int:
    return int(lib().hla2_state_floats(d, dv))


def hla3_state_floats(d: int, dv: int) -> int:
    return int(lib().hla3_state_floats(d, dv))


def hla2_workspace_bytes(B, H, n, d, dv, chunk, dtype) -> int:
    code = dtype if isinstance(dtype, int) else (HLA_BF16 if dtype == torch.bfloat16 else HLA_F32)
    return int(lib().hla2_workspace_bytes(B, H, n, d, dv, chunk, code))


def hla3_workspace_bytes(B, H, n, d, dv, chunk, dtype) -> int:
    code = dtype if isinstance(dtype, int) else (HLA_BF16 if dtype == torch.bfloat16 else HLA_F32)
    return int(lib().hla3_workspace_bytes(B, H, n, d, dv, chunk, code))


def alloc_workspace(nbytes: int, device) -> torch.Tensor:
    """Caller-owned scratch for the forward calls (256-byte aligned by the allocator)."""
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def _forward(fn_name, ws_fn, q, k, v, out, masked, normalized, eps, chunk, state_in, state_out, workspace, stream):
    if q.dim() != 4:
        raise ValueError("q, k, v must be [B, H, n, d]")
    B, H, n, d = q.shape
    dv = v.shape[-1]
    if k.shape != q.shape or v.shape[:3] != q.shape[:3]:
        raise ValueError("shape mismatch: q %s k %s v %s" % (tuple(q.shape), tuple(k.shape), tuple(v.shape)))
    for t in (q, k, v):
        if not t.is_cuda or not t.is_contiguous() or t.dtype != q.dtype:
            raise ValueError("q, k, v must be contiguous CUDA tensors of one dtype")
    if out is None:
        out = torch.empty((B, H, n, dv), dtype=q.dtype, device=q.device)
    dt = _dtype_code(q)
    if workspace is None:
        workspace = alloc_workspace(ws_fn(B, H, n, d, dv, chunk, dt), q.device)
    code = getattr(lib(), fn_name)(_ptr(q), _ptr(k), _ptr(v), _ptr(out), dt, B, H, n, d, dv, int(masked),
                                   int(normalized), float(eps), int(chunk), _ptr(state_in), _ptr(state_out),
                                   _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream))
    _check(code, fn_name)
    return out


def hla2_forward(q, k, v, out=None, *, masked=True, normalized=False, eps=1e-6, chunk=128, state_in=None,
                 state_out=None, workspace=None, stream=None):
    """Second-order HLA forward (include/hla.h: hla2_forward). Returns ``out``."""
    return _forward("hla2_forward", hla2_workspace_bytes, q, k, v, out, masked, normalized, eps, chunk, state_in,
                    state_out, workspace, stream)


def hla3_forward(q, k, v, out=None, *, masked=True, normalized=False, eps=1e-6, chunk=32, state_in=None,
                 state_out=None, workspace=None, stream=None):
    """Third-order HLA forward (include/hla.h: hla3_forward). Returns ``out``."""
    return _forward("hla3_forward", hla3_workspace_bytes, q, k, v, out, masked, normalized, eps, chunk, state_in,
                    state_out, workspace, stream)


def hla2_forward_noalloc(q, k, v, out=None, *, masked=True, normalized=False, eps=1e-6, chunk=128, state_in=None,
                         stream=None):
    """hla2_forward without a workspace, for callers that cannot allocate device
    memory; the library's own 16 MiB device array serves as scratch (include/hla.h:
    hla2_forward_noalloc).  Returns ``out``."""
    B, H, n, d = q.shape
    dv = v.shape[-1]
    if out is None:
        out = torch.empty((B, H, n, dv), dtype=q.dtype, device=q.device)
    code = lib().hla2_forward_noalloc(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _dtype_code(q), B, H, n, d, dv,
                                      int(masked), int(normalized), float(eps), int(chunk), _ptr(state_in),
                                      _stream(stream))
    _check(code, "hla2_forward_noalloc")
    return out


def hla2_forward_path(B, H, n, d, dv, *, masked=True, normalized=False, chunk=128, dtype=torch.bfloat16,
                      has_state_in=False, has_state_out=False):
    """(path, launches) that hla2_forward takes: path 1 = fused tcgen05 kernel, 0 = generic, -1 = unsupported."""
    code = dtype if isinstance(dtype, int) else (HLA_BF16 if dtype == torch.bfloat16 else HLA_F32)
    n_launch = ctypes.c_int(0)
    path = lib().hla2_forward_path(B, H, n, d, dv, int(masked), int(normalized), int(chunk), code,
                                   int(has_state_in), int(has_state_out), ctypes.byref(n_launch))
    return int(path), int(n_launch.value)


def hla3_forward_path(B, H, n, d, dv, *, masked=True, normalized=False, chunk=32, dtype=torch.float32,
                      has_state_in=False, has_state_out=False):
    """(path, launches) that hla3_forward takes: path 2 = tensor-core kernels, 1 = chunk-parallel fp32
    kernels, 0 = serial kernel, -1 = unsupported."""
    code = dtype if isinstance(dtype, int) else (HLA_BF16 if dtype == torch.bfloat16 else HLA_F32)
    n_launch = ctypes.c_int(0)
    path = lib().hla3_forward_path(B, H, n, d, dv, int(masked), int(normalized), int(chunk), code,
                                   int(has_state_in), int(has_state_out), ctypes.byref(n_launch))
    return int(path), int(n_launch.value)


def hla2_step(q, k, v, state, out=None, *, masked=True, normalized=False, eps=1e-6, stream=None):
    """One decode step for every head (include/hla.h: hla2_step); ``state`` is updated in place.

    q, k: [B, H, d]; v: [B, H, dv]; state: fp32 [B, H, hla2_state_floats(d, dv)].
    """
    B, H, d = q.shape
    dv = v.shape[-1]
    if out is None:
        out = torch.empty((B, H, dv), dtype=q.dtype, device=q.device)
    if state.dtype != torch.float32 or not state.is_contiguous():
        raise ValueError("state must be contiguous float32")
    code = lib().hla2_step(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _dtype_code(q), B, H, d, dv, int(masked),
                           int(normalized), float(eps), _ptr(state), _stream(stream))
    _check(code, "hla2_step")
    return out


def hla2_backward_workspace_bytes(B, H, n, d, dv, chunk, dtype) -> int:
    code = dtype if isinstance(dtype, int) else (HLA_BF16 if dtype == torch.bfloat16 else HLA_F32)
    return int(lib().hla2_backward_workspace_bytes(B, H, n, d, dv, chunk, code))


def hla2_backward(q, k, v, dout, *, normalized=False, eps=1e-6, chunk=64, workspace=None, stream=None):
    """Gradients (dq, dk, dv) of sum(dout * out) for the masked second-order forward
    (include/hla.h: hla2_backward)."""
    B, H, n, d = q.shape
    dv = v.shape[-1]
    for t in (q, k, v, dout):
        if not t.is_cuda or not t.is_contiguous() or t.dtype != q.dtype:
            raise ValueError("q, k, v, dout must be contiguous CUDA tensors of one dtype")
    dt = _dtype_code(q)
    gq, gk, gv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    if workspace is None:
        workspace = alloc_workspace(hla2_backward_workspace_bytes(B, H, n, d, dv, chunk, dt), q.device)
    code = lib().hla2_backward(_ptr(q), _ptr(k), _ptr(v), _ptr(dout), _ptr(gq), _ptr(gk), _ptr(gv), dt, B, H, n, d,
                               dv, int(normalized), float(eps), int(chunk), _ptr(workspace),
                               workspace.numel() * workspace.element_size(), _stream(stream))
    _check(code, "hla2_backward")
    return gq, gk, gv


def ahla_state_floats(d: int, dv: int) -> int:
    return int(lib().ahla_state_floats(d, dv))


def ahla_workspace_bytes(B, H, n, d, dv, chunk, dtype) -> int:
    code = dtype if isinstance(dtype, int) else (HLA_BF16 if dtype == torch.bfloat16 else HLA_F32)
    return int(lib().ahla_workspace_bytes(B, H, n, d, dv, chunk, code))


def ahla_forward(q, k, v, out=None, *, normalized=False, eps=1e-6, chunk=64, state_in=None, state_out=None,
                 workspace=None, stream=None):
    """AHLA forward (include/hla.h: ahla_forward). Returns ``out``."""
    if q.dim() != 4:
        raise ValueError("q, k, v must be [B, H, n, d]")
    B, H, n, d = q.shape
    dv = v.shape[-1]
    for t in (q, k, v):
        if not t.is_cuda or not t.is_contiguous() or t.dtype != q.dtype:
            raise ValueError("q, k, v must be contiguous CUDA tensors of one dtype")
    if out is None:
        out = torch.empty((B, H, n, dv), dtype=q.dtype, device=q.device)
    dt = _dtype_code(q)
    if workspace is None:
        workspace = alloc_workspace(ahla_workspace_bytes(B, H, n, d, dv, chunk, dt), q.device)
    code = lib().ahla_forward(_ptr(q), _ptr(k), _ptr(v), _ptr(out), dt, B, H, n, d, dv, int(normalized), float(eps),
                              int(chunk), _ptr(state_in), _ptr(state_out), _ptr(workspace),
                              workspace.numel() * workspace.element_size(), _stream(stream))
    _check(code, "ahla_forward")
    return out


def hla2_backward_path(B, H, n, d, dv, *, normalized=False, chunk=64, dtype=torch.bfloat16) -> int:
    """1 if hla2_backward runs on the tensor cores for these arguments, 0 on the fp32 kernels, -1 unsupported."""
    code = dtype if isinstance(dtype, int) else (HLA_BF16 if dtype == torch.bfloat16 else HLA_F32)
    return int(lib().hla2_backward_path(B, H, n, d, dv, int(normalized), int(chunk), code))


def ahla_forward_path(B, H, n, d, dv, *, normalized=False, chunk=64, dtype=torch.bfloat16, has_state_in=False,
                      has_state_out=False) -> int:
    """1 if ahla_forward runs on the tensor cores for these arguments, 0 on the fp32 kernels, -1 unsupported."""
    code = dtype if isinstance(dtype, int) else (HLA_BF16 if dtype == torch.bfloat16 else HLA_F32)
    return int(lib().ahla_forward_path(B, H, n, d, dv, int(normalized), int(chunk), code, int(has_state_in),
                                       int(has_state_out)))


def ahla_step(q, k, v, state, out=None, *, normalized=False, eps=1e-6, stream=None):
    """One AHLA decode step for every head (include/hla.h: ahla_step); ``state`` is updated in place."""
    B, H, d = q.shape
    dv = v.shape[-1]
    if out is None:
        out = torch.empty((B, H, dv), dtype=q.dtype, device=q.device)
    if state.dtype != torch.float32 or not state.is_contiguous():
        raise ValueError("state must be contiguous float32")
    code = lib().ahla_step(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _dtype_code(q), B, H, d, dv, int(normalized),
                           float(eps), _ptr(state), _stream(stream))
    _check(code, "ahla_step")
    return out


def hla2_sde_state_floats(d: int, dv: int) -> int:
    return int(lib().hla2_sde_state_floats(d, dv))


def hla2_state_to_sde(state, d: int, dv: int, sde=None, *, stream=None):
    """(S, C, m, G, h) tuples [B, H, hla2_state_floats(d, dv)] -> (S, D, e) states
    [B, H, hla2_sde_state_floats(d, dv)] (include/hla.h: hla2_state_to_sde)."""
    B, H = state.shape[:2]
    if sde is None:
        sde = torch.empty((B, H, hla2_sde_state_floats(d, dv)), dtype=torch.float32, device=state.device)
    _check(lib().hla2_state_to_sde(_ptr(state), _ptr(sde), B, H, d, dv, _stream(stream)), "hla2_state_to_sde")
    return sde


def hla2_step_sde(q, k, v, sde, out=None, *, normalized=False, eps=1e-6, stream=None):
    """One decode step of the masked operator on (S, D, e) states, updated in place
    (include/hla.h: hla2_step_sde).  q, k: [B, H, d]; v: [B, H, dv]."""
    B, H, d = q.shape
    dv = v.shape[-1]
    if out is None:
        out = torch.empty((B, H, dv), dtype=q.dtype, device=q.device)
    if sde.dtype != torch.float32 or not sde.is_contiguous():
        raise ValueError("state must be contiguous float32")
    code = lib().hla2_step_sde(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _dtype_code(q), B, H, d, dv, int(normalized),
                               float(eps), _ptr(sde), _stream(stream))
    _check(code, "hla2_step_sde")
    return out


def hla_poll_error_noalloc(stream=None) -> int:
    """Synchronise and read the device-side error flag of the library's own scratch array, used by
    hla2_forward_noalloc (include/hla.h: hla_poll_error_noalloc)."""
    return int(lib().hla_poll_error_noalloc(_stream(stream)))


def hla_poll_error(workspace, stream=None) -> int:
    """Synchronise and read the device-side error flag of a workspace (include/hla.h: hla_poll_error)."""
    return int(lib().hla_poll_error(_ptr(workspace), _stream(stream)))
