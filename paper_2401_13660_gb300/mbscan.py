"""Python binding of libmbscan.so (argument marshalling only).

Each function has the name of the C entry point it calls (include/mbscan.h)
and takes torch CUDA tensors in place of device pointers. Every step of the
layer core runs in the library's kernels; this module only checks tensor
shapes/dtypes/devices, fills the C argument struct and forwards the call on
the current torch CUDA stream (or the stream given). There is no fallback: if
the library cannot be loaded, importing the functions raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

_lock = threading.Lock()
_lib = None

MB_OK, MB_ERR_INVALID_ARG, MB_ERR_UNSUPPORTED, MB_ERR_CUDA, MB_ERR_TIMEOUT = range(5)
MB_F32, MB_BF16 = 0, 1
_DTYPES = {torch.float32: MB_F32, torch.bfloat16: MB_BF16}


class MbError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {mb_status_string(status)}")


class mb_scan_args(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int64), ("seqlen", ctypes.c_int64),
        ("d_inner", ctypes.c_int64), ("d_state", ctypes.c_int64),
        ("dtype", ctypes.c_int32), ("bc_stride", ctypes.c_int32),
        ("x", ctypes.c_void_p), ("z", ctypes.c_void_p), ("dt", ctypes.c_void_p),
        ("B", ctypes.c_void_p), ("C", ctypes.c_void_p),
        ("A", ctypes.c_void_p), ("D", ctypes.c_void_p), ("dt_bias", ctypes.c_void_p),
        ("h0", ctypes.c_void_p), ("y", ctypes.c_void_p),
        ("dt_low", ctypes.c_void_p), ("W_dt", ctypes.c_void_p),
        ("dt_rank", ctypes.c_int32), ("dt_low_stride", ctypes.c_int32),
    ]


class mb_scan_grads(ctypes.Structure):
    _fields_ = [("dx", ctypes.c_void_p), ("dz", ctypes.c_void_p), ("ddt", ctypes.c_void_p),
                ("dB", ctypes.c_void_p), ("dC", ctypes.c_void_p), ("dA", ctypes.c_void_p),
                ("dD", ctypes.c_void_p), ("ddt_bias", ctypes.c_void_p), ("dh0", ctypes.c_void_p)]


MB_CKPT_STEPS = 16


def library_path() -> str:
    return _build.LIB


def load_library(build_if_needed: bool = True) -> ctypes.CDLL:
    """Load libmbscan.so (building it first if it is missing or stale)."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build() if build_if_needed else _build.LIB
            if not os.path.exists(path):
                raise RuntimeError(f"libmbscan.so not found at {path}; run build() first")
            lib = ctypes.CDLL(path)
            vp, i64, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_size_t
            ap = ctypes.POINTER(mb_scan_args)
            lib.mb_workspace_size.argtypes = [ap]
            lib.mb_workspace_size.restype = sz
            lib.mb_scan_prefill.argtypes = [ap, vp, vp, sz, vp]
            lib.mb_scan_verify.argtypes = [ap, vp, vp, sz, vp]
            lib.mb_rollback.argtypes = [vp, vp, vp, vp, i64, i64, i64, i64, vp, vp]
            lib.mb_step.argtypes = [ap, vp, vp, sz, vp]
            lib.mb_check.argtypes = [vp, vp, ctypes.POINTER(i64)]
            lib.mb_accept_topk.argtypes = [vp, ctypes.c_int32, vp, i64, i64, ctypes.c_int32, vp, vp]
            lib.mb_step_resume.argtypes = [ap, vp, vp, i64, vp, vp, sz, vp]
            lib.mb_scan_prefill_ckpt.argtypes = [ap, vp, vp, vp, sz, vp]
            lib.mb_rmsnorm.argtypes = [vp, vp, vp, ctypes.c_float, vp, i64, i64, ctypes.c_int32, vp]
            lib.mb_conv1d_step.argtypes = [vp, vp, vp, vp, vp, i64, i64, ctypes.c_int32, vp]
            lib.mb_scan_backward.argtypes = [ap, vp, vp, vp, ctypes.POINTER(mb_scan_grads), vp, sz, vp]
            lib.mb_selftest_timeout.argtypes = [vp, sz, i64, vp]
            lib.mb_scan_verify_resume.argtypes = [ap, vp, vp, i64, vp, vp, sz, vp]
            lib.mb_conv_xproj_workspace_size.argtypes = [i64, i64, ctypes.c_int32]
            lib.mb_conv_xproj_workspace_size.restype = sz
            lib.mb_conv_xproj.argtypes = [vp, vp, vp, vp, vp, vp, vp, i64, i64, ctypes.c_int32, ctypes.c_int32,
                                          vp, sz, vp]
            for f in ("mb_scan_prefill", "mb_scan_verify", "mb_rollback", "mb_step", "mb_check",
                      "mb_accept_topk", "mb_step_resume", "mb_scan_prefill_ckpt", "mb_scan_backward",
                      "mb_rmsnorm", "mb_conv1d_step", "mb_selftest_timeout", "mb_scan_verify_resume",
                      "mb_conv_xproj"):
                getattr(lib, f).restype = ctypes.c_int
            lib.mb_status_string.argtypes = [ctypes.c_int]
            lib.mb_status_string.restype = ctypes.c_char_p
            lib.mb_version.argtypes = []
            lib.mb_version.restype = ctypes.c_char_p
            _lib = lib
    return _lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _need(t, name, dtype=None, shape=None, device=None):
    if t is None:
        return
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name}: dtype {t.dtype}, expected {dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: shape {tuple(t.shape)}, expected {tuple(shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")


def _row_stride(name, t, batch, L, width, dtype, dev):
    """Row stride (elements) of t [batch, L, width]: width when contiguous,
    or S when t is a column block of wider rows (strides (L*S, S, 1))."""
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype or tuple(t.shape) != (batch, L, width) or t.device != dev:
        raise ValueError(f"{name}: {t.dtype} {tuple(t.shape)} on {t.device}, expected {dtype} "
                         f"{(batch, L, width)} on {dev}")
    if t.is_contiguous():
        return width
    sb, st, sn = t.stride()
    if sn != 1 or (L > 1 and sb != L * st) or st < width:
        raise ValueError(f"{name} must be contiguous or have strides (L*S, S, 1)")
    return st if L > 1 or batch == 1 else sb


def _bc_row_stride(B, C, batch, L, N, dtype, dev):
    """Row stride (elements) shared by B and C [batch, L, N]: N for
    contiguous tensors, or S when both are column blocks of wider rows
    (strides (L*S, S, 1))."""
    strides = {_row_stride(name, t, batch, L, N, dtype, dev) for name, t in (("B", B), ("C", C))}
    if len(strides) != 1:
        raise ValueError("B and C must share one row stride")
    return strides.pop()


def make_args(x, dt, B, C, A, y, *, z=None, D=None, dt_bias=None, h0=None, dt_low=None,
              W_dt=None) -> mb_scan_args:
    """Fill mb_scan_args from tensors. x, dt, z, y: [batch, L, d_inner];
    B, C: [batch, L, d_state] (all one dtype, fp32 or bf16), contiguous or
    column blocks of wider rows (strides (L*S, S, 1): bc_stride = S); A:
    [d_inner, d_state], D, dt_bias: [d_inner], h0: [batch, d_inner, d_state]
    (fp32). Fused Delta projection: dt = None, dt_low [batch, L, r] (contiguous
    or a column block of wider rows) and W_dt [d_inner, r]; the kernels then
    form dt = dt_low W_dt^T themselves."""
    if x.dtype not in _DTYPES:
        raise TypeError(f"unsupported input dtype {x.dtype}")
    batch, L, Dn = x.shape
    N = A.shape[1]
    dev = x.device
    if (dt is None) == (dt_low is None):
        raise ValueError("pass exactly one of dt and dt_low")
    if dt_low is not None and W_dt is None:
        raise ValueError("dt_low needs W_dt")
    for name, t in (("x", x), ("dt", dt), ("z", z), ("y", y)):
        _need(t, name, x.dtype, (batch, L, Dn), dev)
    S = _bc_row_stride(B, C, batch, L, N, x.dtype, dev)
    _need(A, "A", torch.float32, (Dn, N), dev)
    _need(D, "D", torch.float32, (Dn,), dev)
    _need(dt_bias, "dt_bias", torch.float32, (Dn,), dev)
    _need(h0, "h0", torch.float32, (batch, Dn, N), dev)
    a = mb_scan_args()
    a.batch, a.seqlen, a.d_inner, a.d_state = batch, L, Dn, N
    a.dtype = _DTYPES[x.dtype]
    a.bc_stride = 0 if S == N else S
    if dt_low is not None:
        r = W_dt.shape[1] if W_dt.dim() == 2 else -1
        _need(W_dt, "W_dt", x.dtype, (Dn, r), dev)
        S = _row_stride("dt_low", dt_low, batch, L, r, x.dtype, dev)
        a.dt_low, a.W_dt = dt_low.data_ptr(), W_dt.data_ptr()
        a.dt_rank = r
        a.dt_low_stride = 0 if S == r else S
    a.x, a.z, a.dt, a.B, a.C = (t.data_ptr() if t is not None else None for t in (x, z, dt, B, C))
    a.A, a.D, a.dt_bias, a.h0 = (t.data_ptr() if t is not None else None for t in (A, D, dt_bias, h0))
    a.y = y.data_ptr()
    return a


def _check(rc, where):
    if rc != MB_OK:
        raise MbError(rc, where)


def mb_status_string(status: int) -> str:
    return load_library().mb_status_string(int(status)).decode()


def mb_version() -> str:
    return load_library().mb_version().decode()


def mb_workspace_size(args: mb_scan_args) -> int:
    return int(load_library().mb_workspace_size(ctypes.byref(args)))


def new_workspace(args: mb_scan_args, device) -> torch.Tensor:
    """Zeroed workspace tensor for `args` (uint8, 256-byte aligned by torch)."""
    n = max(mb_workspace_size(args), 256)
    return torch.zeros(n, dtype=torch.uint8, device=device)


def mb_scan_prefill(x, dt, B, C, A, y, *, z=None, D=None, dt_bias=None, h0=None, h_last=None,
                    ws=None, stream=None, dt_low=None, W_dt=None):
    """Prefill scan: writes y and (if given) h_last [batch, d_inner, d_state].
    dt = None with dt_low, W_dt: the fused Delta projection (see make_args)."""
    a = make_args(x, dt, B, C, A, y, z=z, D=D, dt_bias=dt_bias, h0=h0, dt_low=dt_low, W_dt=W_dt)
    _need(h_last, "h_last", torch.float32, (a.batch, a.d_inner, a.d_state), x.device)
    if ws is None:
        ws = new_workspace(a, x.device)
    rc = load_library().mb_scan_prefill(ctypes.byref(a), _ptr(h_last), _ptr(ws), ws.numel(),
                                        _stream(stream))
    _check(rc, "mb_scan_prefill")
    return y, h_last


def mb_scan_verify(x, dt, B, C, A, y, h_all, *, z=None, D=None, dt_bias=None, h0=None, ws=None,
                   stream=None, dt_low=None, W_dt=None):
    """Verify scan of k = x.shape[1] drafted bytes: y and h_all [batch, k, d_inner, d_state]."""
    a = make_args(x, dt, B, C, A, y, z=z, D=D, dt_bias=dt_bias, h0=h0, dt_low=dt_low, W_dt=W_dt)
    _need(h_all, "h_all", torch.float32, (a.batch, a.seqlen, a.d_inner, a.d_state), x.device)
    if ws is None:
        ws = new_workspace(a, x.device)
    rc = load_library().mb_scan_verify(ctypes.byref(a), _ptr(h_all), _ptr(ws), ws.numel(),
                                       _stream(stream))
    _check(rc, "mb_scan_verify")
    return y, h_all


def mb_scan_verify_resume(x, dt, B, C, A, y, h_all, h_all_prev, accept, *, z=None, D=None, dt_bias=None,
                          h0=None, ws=None, stream=None, dt_low=None, W_dt=None):
    """Verify of k = x.shape[1] drafted bytes, stream s starting from h0[s]
    (zeros if None) when accept[s] == 0, else from h_all_prev[s, accept[s]-1]
    (the previous verify's per-position states, [batch, k_prev, d_inner,
    d_state]). A bad accept count is recorded in ws (mb_check) and that stream
    is left untouched."""
    a = make_args(x, dt, B, C, A, y, z=z, D=D, dt_bias=dt_bias, h0=h0, dt_low=dt_low, W_dt=W_dt)
    _need(h_all, "h_all", torch.float32, (a.batch, a.seqlen, a.d_inner, a.d_state), x.device)
    _need(h_all_prev, "h_all_prev", torch.float32, None, x.device)
    if h_all_prev.dim() != 4 or h_all_prev.shape[0] != a.batch or \
            tuple(h_all_prev.shape[2:]) != (a.d_inner, a.d_state):
        raise ValueError(f"h_all_prev: shape {tuple(h_all_prev.shape)}, expected [batch, k_prev, d_inner, d_state]")
    _need(accept, "accept", torch.int32, (a.batch,), x.device)
    if ws is None:
        ws = new_workspace(a, x.device)
    rc = load_library().mb_scan_verify_resume(ctypes.byref(a), _ptr(h_all_prev), _ptr(accept), h_all_prev.shape[1],
                                              _ptr(h_all), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "mb_scan_verify_resume")
    return y, h_all


def mb_rollback(h0, h_all, accept, h_out, *, ws=None, stream=None):
    """h_out[s] = h0[s] if accept[s] == 0 else h_all[s, accept[s]-1]."""
    batch, k, Dn, N = h_all.shape
    _need(h_all, "h_all", torch.float32)
    _need(h0, "h0", torch.float32, (batch, Dn, N), h_all.device)
    _need(h_out, "h_out", torch.float32, (batch, Dn, N), h_all.device)
    _need(accept, "accept", torch.int32, (batch,), h_all.device)
    rc = load_library().mb_rollback(_ptr(h0), _ptr(h_all), _ptr(accept), _ptr(h_out), batch, k,
                                    Dn, N, _ptr(ws), _stream(stream))
    _check(rc, "mb_rollback")
    return h_out


def mb_step(x, dt, B, C, A, y, state, *, z=None, D=None, dt_bias=None, ws=None, stream=None, dt_low=None,
            W_dt=None):
    """One decode step: x, dt, z, y [batch, 1, d_inner]; B, C [batch, 1, d_state];
    state [batch, d_inner, d_state] updated in place. ws (optional, >= 256
    bytes): status block where a timed-out wait is recorded (mb_check)."""
    a = make_args(x, dt, B, C, A, y, z=z, D=D, dt_bias=dt_bias, dt_low=dt_low, W_dt=W_dt)
    _need(state, "state", torch.float32, (a.batch, a.d_inner, a.d_state), x.device)
    _need(ws, "ws", torch.uint8, None, x.device)
    nbytes = 0 if ws is None else ws.numel()
    rc = load_library().mb_step(ctypes.byref(a), _ptr(state), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "mb_step")
    return y, state


def mb_scan_prefill_ckpt(x, dt, B, C, A, y, h_ckpt=None, *, z=None, D=None, dt_bias=None, h0=None,
                         h_last=None, ws=None, stream=None, dt_low=None, W_dt=None):
    """Training forward: prefill that also writes h_ckpt [batch, ceil(L / 16),
    d_inner, d_state], the state before every 16-step chunk (allocated when
    None). Returns (y, h_last, h_ckpt). (The fused Delta projection is not
    accepted here: MB_ERR_UNSUPPORTED.)"""
    a = make_args(x, dt, B, C, A, y, z=z, D=D, dt_bias=dt_bias, h0=h0, dt_low=dt_low, W_dt=W_dt)
    nch = (a.seqlen + MB_CKPT_STEPS - 1) // MB_CKPT_STEPS
    if h_ckpt is None:
        h_ckpt = torch.empty(a.batch, nch, a.d_inner, a.d_state, dtype=torch.float32, device=x.device)
    _need(h_ckpt, "h_ckpt", torch.float32, (a.batch, nch, a.d_inner, a.d_state), x.device)
    _need(h_last, "h_last", torch.float32, (a.batch, a.d_inner, a.d_state), x.device)
    if ws is None:
        ws = new_workspace(a, x.device)
    rc = load_library().mb_scan_prefill_ckpt(ctypes.byref(a), _ptr(h_last), _ptr(h_ckpt), _ptr(ws),
                                             ws.numel(), _stream(stream))
    _check(rc, "mb_scan_prefill_ckpt")
    return y, h_last, h_ckpt


def mb_scan_backward(x, dt, B, C, A, h_ckpt, dout, *, z=None, D=None, dt_bias=None, h0=None,
                     dh_last=None, grads=None, ws=None, stream=None):
    """Backward of the layer core. Returns a dict of gradients: dx, ddt, dz (or
    None) in the input dtype [batch, L, d_inner]; dB, dC fp32 [batch, L,
    d_state]; dA fp32 [d_inner, d_state]; dD, ddt_bias fp32 [d_inner]; dh0 fp32
    [batch, d_inner, d_state]. Tensors missing from `grads` are allocated."""
    if x.dtype not in _DTYPES:
        raise TypeError(f"unsupported input dtype {x.dtype}")
    batch, L, Dn = x.shape
    N = A.shape[1]
    dev = x.device
    a = make_args(x, dt, B, C, A, x, z=z, D=D, dt_bias=dt_bias, h0=h0)
    a.y = None
    nch = (L + MB_CKPT_STEPS - 1) // MB_CKPT_STEPS
    _need(h_ckpt, "h_ckpt", torch.float32, (batch, nch, Dn, N), dev)
    _need(dout, "dout", x.dtype, (batch, L, Dn), dev)
    _need(dh_last, "dh_last", torch.float32, (batch, Dn, N), dev)
    g = dict(grads or {})
    shapes = {"dx": ((batch, L, Dn), x.dtype), "ddt": ((batch, L, Dn), x.dtype),
              "dz": ((batch, L, Dn), x.dtype), "dB": ((batch, L, N), torch.float32),
              "dC": ((batch, L, N), torch.float32), "dA": ((Dn, N), torch.float32),
              "dD": ((Dn,), torch.float32), "ddt_bias": ((Dn,), torch.float32),
              "dh0": ((batch, Dn, N), torch.float32)}
    for k, (shp, dty) in shapes.items():
        if k == "dz" and z is None:
            g[k] = None
            continue
        if g.get(k) is None:
            g[k] = torch.empty(shp, dtype=dty, device=dev)
        _need(g[k], k, dty, shp, dev)
    st = mb_scan_grads(*(None if g[k] is None else g[k].data_ptr() for k in
                         ("dx", "dz", "ddt", "dB", "dC", "dA", "dD", "ddt_bias", "dh0")))
    if ws is None:
        ws = new_workspace(a, dev)
    rc = load_library().mb_scan_backward(ctypes.byref(a), _ptr(h_ckpt), _ptr(dout), _ptr(dh_last),
                                         ctypes.byref(st), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "mb_scan_backward")
    return g


def mb_rmsnorm(residual, w, out, *, add=None, eps=1e-5, stream=None):
    """residual [batch, width] fp32 += add (if given); out = residual * w /
    rms(residual), out and add in the input dtype (fp32 or bf16)."""
    if out.dtype not in _DTYPES:
        raise TypeError(f"unsupported dtype {out.dtype}")
    batch, width = residual.shape
    dev = residual.device
    _need(residual, "residual", torch.float32, (batch, width), dev)
    _need(w, "w", torch.float32, (width,), dev)
    _need(out, "out", out.dtype, (batch, width), dev)
    _need(add, "add", out.dtype, (batch, width), dev)
    rc = load_library().mb_rmsnorm(_ptr(add), _ptr(residual), _ptr(w), float(eps), _ptr(out), batch, width,
                                   _DTYPES[out.dtype], _stream(stream))
    _check(rc, "mb_rmsnorm")
    return out


def mb_conv1d_step(x, state, w, out, *, bias=None, stream=None):
    """One causal depthwise convolution step (kernel 4) with SiLU: x, out
    [batch, width]; state [batch, 3, width] (previous inputs, oldest first),
    updated in place; w [width, 4] fp32; bias [width] fp32."""
    if x.dtype not in _DTYPES:
        raise TypeError(f"unsupported dtype {x.dtype}")
    batch, width = x.shape
    dev = x.device
    _need(x, "x", x.dtype, (batch, width), dev)
    _need(state, "state", x.dtype, (batch, 3, width), dev)
    _need(w, "w", torch.float32, (width, 4), dev)
    _need(bias, "bias", torch.float32, (width,), dev)
    _need(out, "out", x.dtype, (batch, width), dev)
    rc = load_library().mb_conv1d_step(_ptr(x), _ptr(state), _ptr(w), _ptr(bias), _ptr(out), batch, width,
                                       _DTYPES[x.dtype], _stream(stream))
    _check(rc, "mb_conv1d_step")
    return out


def mb_conv_xproj_workspace_size(batch: int, width: int, n_out: int) -> int:
    """Workspace bytes mb_conv_xproj needs (0: shape not supported)."""
    return int(load_library().mb_conv_xproj_workspace_size(batch, width, n_out))


def mb_conv_xproj(x, state, w, W, xc, out, ws, *, bias=None, stream=None):
    """Convolution step fused with the x-projection: xc = silu(conv1d_step(x))
    as mb_conv1d_step (state [batch, 3, width] updated in place), then
    out = xc W^T. x, xc [batch, width], W [n_out, width], out [batch, n_out],
    all bf16; w [width, 4], bias [width] fp32; ws a uint8 workspace of
    mb_conv_xproj_workspace_size bytes."""
    batch, width = x.shape
    n_out = W.shape[0]
    dev, bf = x.device, torch.bfloat16
    _need(x, "x", bf, (batch, width), dev)
    _need(state, "state", bf, (batch, 3, width), dev)
    _need(w, "w", torch.float32, (width, 4), dev)
    _need(bias, "bias", torch.float32, (width,), dev)
    _need(W, "W", bf, (n_out, width), dev)
    _need(xc, "xc", bf, (batch, width), dev)
    _need(out, "out", bf, (batch, n_out), dev)
    _need(ws, "ws", torch.uint8, None, dev)
    rc = load_library().mb_conv_xproj(_ptr(x), _ptr(state), _ptr(w), _ptr(bias), _ptr(W), _ptr(xc), _ptr(out),
                                      batch, width, n_out, MB_BF16, _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "mb_conv_xproj")
    return out


def mb_step_resume(x, dt, B, C, A, y, h_all, accept, state, *, z=None, D=None, dt_bias=None, h0=None,
                   ws=None, stream=None, dt_low=None, W_dt=None):
    """One decode step from the state kept after accept[s] drafted bytes:
    h0[s] (zeros if None) when accept[s] == 0, else h_all[s, accept[s]-1].
    x, dt, z, y [batch, 1, d_inner]; B, C [batch, 1, d_state]; h_all [batch,
    k, d_inner, d_state]; accept [batch] int32; state [batch, d_inner,
    d_state] is written (it may be h0 itself)."""
    a = make_args(x, dt, B, C, A, y, z=z, D=D, dt_bias=dt_bias, h0=h0, dt_low=dt_low, W_dt=W_dt)
    _need(h_all, "h_all", torch.float32, None, x.device)
    if h_all.dim() != 4 or h_all.shape[0] != a.batch or tuple(h_all.shape[2:]) != (a.d_inner, a.d_state):
        raise ValueError(f"h_all: shape {tuple(h_all.shape)}, expected [batch, k, d_inner, d_state]")
    _need(accept, "accept", torch.int32, (a.batch,), x.device)
    _need(state, "state", torch.float32, (a.batch, a.d_inner, a.d_state), x.device)
    nbytes = 0 if ws is None else ws.numel()
    rc = load_library().mb_step_resume(ctypes.byref(a), _ptr(h_all), _ptr(accept), h_all.shape[1],
                                       _ptr(state), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "mb_step_resume")
    return y, state


def mb_accept_topk(logits, drafted, beta, accept=None, stream=None):
    """Accept counts of speculative decoding: logits [streams, k, 256] (fp32 or
    bf16), drafted [streams, k] uint8 -> accept [streams] int32."""
    if logits.dtype not in _DTYPES:
        raise TypeError(f"unsupported logits dtype {logits.dtype}")
    streams, k, v = logits.shape
    if v != 256:
        raise ValueError("logits must have 256 entries per position")
    _need(logits, "logits", logits.dtype)
    _need(drafted, "drafted", torch.uint8, (streams, k), logits.device)
    if accept is None:
        accept = torch.empty(streams, dtype=torch.int32, device=logits.device)
    _need(accept, "accept", torch.int32, (streams,), logits.device)
    rc = load_library().mb_accept_topk(_ptr(logits), _DTYPES[logits.dtype], _ptr(drafted), streams, k,
                                       int(beta), _ptr(accept), _stream(stream))
    _check(rc, "mb_accept_topk")
    return accept


def mb_selftest_timeout(ws, wait_cycles, stream=None):
    """Run the bounded-wait diagnostic: a kernel waits wait_cycles SM clocks on
    a barrier nothing arrives on and records MB_ERR_TIMEOUT in ws (read it with
    mb_check)."""
    _need(ws, "ws", torch.uint8)
    rc = load_library().mb_selftest_timeout(_ptr(ws), ws.numel(), int(wait_cycles), _stream(stream))
    _check(rc, "mb_selftest_timeout")


def mb_check(ws, stream=None):
    """Read and clear the workspace status block: (status, detail)."""
    detail = ctypes.c_int64(-1)
    rc = load_library().mb_check(_ptr(ws), _stream(stream), ctypes.byref(detail))
    return int(rc), int(detail.value)
