"""CPU checks of the C ABI: the library loads, exports every entry point that
include/mbscan.h declares, and rejects bad arguments on the host before any
launch (so these run without a GPU: no call below reaches the device)."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2401_13660_gb300 import mbscan as mb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mbscan.h")

FAKE = 1 << 40  # an aligned, never-dereferenced stand-in for a device address


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(mb_[a-z_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for f in ("mb_scan_prefill", "mb_scan_verify", "mb_rollback", "mb_step", "mb_workspace_size",
              "mb_check", "mb_status_string", "mb_version"):
        assert f in names


def test_library_exports_every_declared_symbol():
    lib = mb.load_library()
    for f in declared_functions():
        assert hasattr(lib, f), f
    out = subprocess.run(["nm", "-D", "--defined-only", mb.library_path()], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r" T (mb_[a-z_]+)$", out, flags=re.M))
    assert set(declared_functions()) <= exported


def test_status_strings_and_version():
    assert mb.mb_status_string(0) == "MB_OK"
    assert mb.mb_status_string(2) == "MB_ERR_UNSUPPORTED"
    assert mb.mb_status_string(99) == "MB_UNKNOWN_STATUS"
    assert "sm_103a" in mb.mb_version()


def _args(batch=2, L=8, Dn=64, N=16, dtype=mb.MB_BF16, **kw):
    a = mb.mb_scan_args()
    a.batch, a.seqlen, a.d_inner, a.d_state, a.dtype = batch, L, Dn, N, dtype
    base = FAKE
    for i, f in enumerate(("x", "z", "dt", "B", "C", "A", "D", "dt_bias", "h0", "y")):
        setattr(a, f, base + i * (1 << 32))
    for k, v in kw.items():
        setattr(a, k, v)
    return a


def _call(name, a, *extra):
    lib = mb.load_library()
    return getattr(lib, name)(ctypes.byref(a), *extra)


def _prefill(a, h_last=None, ws=FAKE + (200 << 32), ws_bytes=256):
    return _call("mb_scan_prefill", a, h_last, ws, ws_bytes, None)


def test_workspace_size():
    lib = mb.load_library()
    assert lib.mb_workspace_size(ctypes.byref(_args())) == 256
    assert lib.mb_workspace_size(ctypes.byref(_args(N=8))) == 0
    assert lib.mb_workspace_size(None) == 0


@pytest.mark.parametrize("bad, want", [
    (dict(N=8), mb.MB_ERR_UNSUPPORTED),
    (dict(Dn=60), mb.MB_ERR_UNSUPPORTED),
    (dict(dtype=7), mb.MB_ERR_INVALID_ARG),
    (dict(batch=-1), mb.MB_ERR_INVALID_ARG),
    (dict(L=-3), mb.MB_ERR_INVALID_ARG),
    (dict(x=None), mb.MB_ERR_INVALID_ARG),
    (dict(A=None), mb.MB_ERR_INVALID_ARG),
    (dict(y=None), mb.MB_ERR_INVALID_ARG),
    (dict(dt=FAKE + 8), mb.MB_ERR_INVALID_ARG),          # misaligned
    (dict(L=1 << 20, Dn=1 << 12, batch=1 << 10), mb.MB_ERR_INVALID_ARG),  # too many tokens
])
def test_prefill_rejects_bad_args(bad, want):
    kw = {}
    for k in ("batch", "L", "Dn", "N", "dtype"):
        if k in bad:
            kw[k] = bad.pop(k)
    a = _args(**kw)
    for k, v in bad.items():
        setattr(a, k, v)
    assert _prefill(a) == want


def test_prefill_rejects_aliasing_and_missing_workspace():
    a = _args()
    a.y = a.x + 64                                   # y overlaps x
    assert _prefill(a) == mb.MB_ERR_INVALID_ARG
    a = _args()
    assert _prefill(a, ws=None) == mb.MB_ERR_INVALID_ARG
    assert _prefill(a, ws_bytes=16) == mb.MB_ERR_INVALID_ARG
    assert _prefill(a, ws=FAKE + (200 << 32) + 16) == mb.MB_ERR_INVALID_ARG   # ws not 256-aligned
    assert _prefill(a, h_last=a.h0 + 16) == mb.MB_ERR_INVALID_ARG           # partial overlap with h0
    assert _prefill(a, h_last=a.y) == mb.MB_ERR_INVALID_ARG


def test_zero_sized_calls_launch_nothing():
    lib = mb.load_library()
    assert _prefill(_args(batch=0)) == mb.MB_OK
    assert _call("mb_scan_verify", _args(L=0), None, FAKE + (200 << 32), 256, None) == mb.MB_OK
    assert _call("mb_step", _args(batch=0, L=1), None, None, 0, None) == mb.MB_OK
    assert lib.mb_rollback(None, None, None, None, 0, 16, 64, 16, None, None) == mb.MB_OK


def test_verify_and_step_checks():
    a = _args(L=16)
    assert _call("mb_scan_verify", a, None, FAKE + (200 << 32), 256, None) == mb.MB_ERR_INVALID_ARG
    assert _call("mb_scan_verify", a, a.h0, FAKE + (200 << 32), 256, None) == mb.MB_ERR_INVALID_ARG
    s = _args(L=2)
    assert _call("mb_step", s, FAKE + (210 << 32), None, 0, None) == mb.MB_ERR_INVALID_ARG   # seqlen != 1
    s = _args(L=1)
    assert _call("mb_step", s, None, None, 0, None) == mb.MB_ERR_INVALID_ARG
    assert _call("mb_step", s, s.x, None, 0, None) == mb.MB_ERR_INVALID_ARG      # state aliases x
    st = FAKE + (210 << 32)
    assert _call("mb_step", s, st, FAKE + (200 << 32) + 16, 256, None) == mb.MB_ERR_INVALID_ARG  # ws not 256-aligned
    assert _call("mb_step", s, st, FAKE + (200 << 32), 128, None) == mb.MB_ERR_INVALID_ARG       # ws too small
    assert _call("mb_step", s, st, st, 256, None) == mb.MB_ERR_INVALID_ARG                       # ws inside state
    assert _call("mb_step", s, st, s.y, 256, None) == mb.MB_ERR_INVALID_ARG                      # ws overlaps y


def test_rollback_checks():
    lib = mb.load_library()
    h0, h_all, acc, out = FAKE, FAKE + (1 << 34), FAKE + (2 << 34), FAKE + (3 << 34)
    assert lib.mb_rollback(h0, h_all, acc, out, 4, 16, 64, 8, None, None) == mb.MB_ERR_UNSUPPORTED
    assert lib.mb_rollback(h0, h_all, None, out, 4, 16, 64, 16, None, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_rollback(h0, h_all, acc, h_all + 64, 4, 16, 64, 16, None, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_rollback(h0, h_all, acc + 2, out, 4, 16, 64, 16, None, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_rollback(h0, h_all, acc, out, -1, 16, 64, 16, None, None) == mb.MB_ERR_INVALID_ARG


def test_step_resume_checks():
    lib = mb.load_library()
    s = _args(L=1)
    h_all, acc, st, ws = FAKE + (20 << 32), FAKE + (24 << 32), FAKE + (28 << 32), FAKE + (32 << 32)

    def call(a=s, h=h_all, c=acc, k=16, out=st, w=ws, wb=256):
        return lib.mb_step_resume(ctypes.byref(a), h, c, k, out, w, wb, None)

    assert call(k=0) == mb.MB_ERR_INVALID_ARG                  # k >= 1
    assert call(h=None) == mb.MB_ERR_INVALID_ARG
    assert call(c=None) == mb.MB_ERR_INVALID_ARG
    assert call(c=acc + 2) == mb.MB_ERR_INVALID_ARG            # accept misaligned
    assert call(out=h_all + 64) == mb.MB_ERR_INVALID_ARG       # state inside h_all
    assert call(out=s.x) == mb.MB_ERR_INVALID_ARG              # state aliases x
    assert call(out=s.h0 + 64) == mb.MB_ERR_INVALID_ARG        # partial overlap with h0
    assert call(wb=16) == mb.MB_ERR_INVALID_ARG                # workspace too small
    assert call(a=_args(L=2)) == mb.MB_ERR_INVALID_ARG         # seqlen != 1
    assert call(a=_args(L=1, N=8)) == mb.MB_ERR_UNSUPPORTED
    assert call(a=_args(batch=0, L=1)) == mb.MB_OK             # nothing to do


def test_training_path_checks():
    lib = mb.load_library()
    a = _args(L=40)
    ck, ws = FAKE + (40 << 32), FAKE + (200 << 32)
    assert lib.mb_scan_prefill_ckpt(ctypes.byref(a), None, None, ws, 256, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_scan_prefill_ckpt(ctypes.byref(a), None, a.x, ws, 256, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_scan_prefill_ckpt(ctypes.byref(a), None, ck + 8, ws, 256, None) == mb.MB_ERR_INVALID_ARG

    def grads(**kw):
        base = FAKE + (60 << 32)
        g = mb.mb_scan_grads(*(base + i * (1 << 32) for i in range(9)))
        for k, v in kw.items():
            setattr(g, k, v)
        return g

    dout = FAKE + (50 << 32)

    def bwd(args=a, h=ck, o=dout, g=None):
        return lib.mb_scan_backward(ctypes.byref(args), h, o, None, ctypes.byref(g or grads()), ws, 256, None)

    b = _args(L=40, y=None)                                  # y is not needed by the backward
    assert bwd(args=b, h=None) == mb.MB_ERR_INVALID_ARG      # checkpoints required
    assert bwd(args=b, o=None) == mb.MB_ERR_INVALID_ARG      # dout required
    assert bwd(args=b, g=grads(dz=None)) == mb.MB_ERR_INVALID_ARG     # gate present, dz missing
    assert bwd(args=b, g=grads(dx=b.x)) == mb.MB_ERR_INVALID_ARG      # output aliases an input
    g2 = grads()
    g2.ddt = g2.dx + 64
    assert bwd(args=b, g=g2) == mb.MB_ERR_INVALID_ARG        # outputs overlap
    assert bwd(args=_args(L=40, N=8)) == mb.MB_ERR_UNSUPPORTED
    assert lib.mb_scan_backward(ctypes.byref(b), ck, dout, None, None, ws, 256, None) == mb.MB_ERR_INVALID_ARG
    # optional outputs left out (null) pass validation (the call then fails to launch: no GPU here)
    nz = _args(L=40, y=None, z=None)
    want_launch = (mb.MB_OK, mb.MB_ERR_CUDA)
    assert bwd(args=nz, g=grads(dz=None, dD=None, ddt_bias=None, dh0=None)) in want_launch


def test_block_kernel_checks():
    lib = mb.load_library()
    res, w, out, add = FAKE, FAKE + (1 << 32), FAKE + (2 << 32), FAKE + (3 << 32)
    f = ctypes.c_float(1e-5)
    assert lib.mb_rmsnorm(add, res, w, f, out, 4, 64, mb.MB_BF16, None) in (mb.MB_OK, mb.MB_ERR_CUDA)
    assert lib.mb_rmsnorm(add, res, w, f, out, 4, 60, mb.MB_BF16, None) == mb.MB_ERR_UNSUPPORTED
    assert lib.mb_rmsnorm(add, res, w, f, out, 4, 8200, mb.MB_BF16, None) in (mb.MB_OK, mb.MB_ERR_CUDA)
    assert lib.mb_rmsnorm(add, res, w, f, res + 64, 4, 64, mb.MB_BF16, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_rmsnorm(add, res, w, ctypes.c_float(-1.0), out, 4, 64, mb.MB_BF16, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_rmsnorm(add, None, w, f, out, 4, 64, mb.MB_BF16, None) == mb.MB_ERR_INVALID_ARG
    x, st, cw, cb, co = FAKE, FAKE + (1 << 32), FAKE + (2 << 32), FAKE + (3 << 32), FAKE + (4 << 32)
    assert lib.mb_conv1d_step(x, st, cw, cb, co, 4, 12, mb.MB_BF16, None) == mb.MB_ERR_UNSUPPORTED
    assert lib.mb_conv1d_step(x, st, cw, cb, st + 16, 4, 64, mb.MB_BF16, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_conv1d_step(x, x + 32, cw, cb, co, 4, 64, mb.MB_BF16, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_conv1d_step(x, st, None, cb, co, 4, 64, mb.MB_BF16, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_conv1d_step(x, st, cw, cb, co, 0, 64, mb.MB_BF16, None) == mb.MB_OK


def test_bc_stride_checks():
    a = _args(L=4)
    a.bc_stride = 12                                    # < d_state
    assert _prefill(a) == mb.MB_ERR_INVALID_ARG
    a.bc_stride = 20                                    # 40 bytes: not a multiple of 16 for bf16
    assert _prefill(a) == mb.MB_ERR_INVALID_ARG
    a = _args(L=4, dtype=mb.MB_F32)
    a.bc_stride = 20                                    # 80 bytes: fine for fp32
    assert _prefill(a) in (mb.MB_OK, mb.MB_ERR_CUDA)


def _fused(L=4, r=64, stride=0, **kw):
    """Arguments with the Delta projection in the kernel (dt = NULL)."""
    a = _args(L=L, **kw)
    a.dt = None
    a.dt_low, a.W_dt = FAKE + (20 << 32), FAKE + (21 << 32)
    a.dt_rank, a.dt_low_stride = r, stride
    return a


def test_fused_delta_checks():
    want_launch = (mb.MB_OK, mb.MB_ERR_CUDA)             # valid: the launch then fails without a GPU
    assert _prefill(_fused()) in want_launch
    assert _prefill(_fused(r=144, stride=176)) in want_launch      # column block of [dt_low | B | C]
    a = _fused()
    a.dt = FAKE + (2 << 32)                                          # both dt and dt_low
    assert _prefill(a) == mb.MB_ERR_INVALID_ARG
    assert _prefill(_fused(r=48)) == mb.MB_ERR_UNSUPPORTED           # below one 64-wide box
    assert _prefill(_fused(r=72)) == mb.MB_ERR_UNSUPPORTED           # not a multiple of 16
    assert _prefill(_fused(r=272)) == mb.MB_ERR_UNSUPPORTED          # above 256
    assert _prefill(_fused(dtype=mb.MB_F32)) == mb.MB_ERR_UNSUPPORTED
    assert _prefill(_fused(r=0)) == mb.MB_ERR_INVALID_ARG
    assert _prefill(_fused(stride=60)) == mb.MB_ERR_INVALID_ARG      # stride < rank
    assert _prefill(_fused(r=64, stride=68)) == mb.MB_ERR_INVALID_ARG   # rows not 16-byte aligned
    a = _fused()
    a.W_dt = None
    assert _prefill(a) == mb.MB_ERR_INVALID_ARG
    a = _fused()
    a.dt_low = a.dt_low + 8                                          # misaligned
    assert _prefill(a) == mb.MB_ERR_INVALID_ARG
    a = _fused()
    a.y = a.dt_low                                                   # y overlaps dt_low
    assert _prefill(a) == mb.MB_ERR_INVALID_ARG
    a = _fused()
    assert _prefill(a, h_last=a.W_dt) == mb.MB_ERR_INVALID_ARG      # h_last overlaps W_dt
    lib = mb.load_library()
    ws = FAKE + (200 << 32)
    assert lib.mb_scan_prefill_ckpt(ctypes.byref(_fused(L=40)), None, FAKE + (40 << 32), ws, 256,
                                    None) == mb.MB_ERR_UNSUPPORTED   # the training path takes dt
    s = _fused(L=1)
    assert _call("mb_step", s, FAKE + (210 << 32), None, 0, None) == mb.MB_ERR_UNSUPPORTED   # the step takes dt
    acc = FAKE + (220 << 32)
    assert lib.mb_step_resume(ctypes.byref(s), FAKE + (230 << 32), acc, 4, FAKE + (210 << 32), None, 0,
                              None) == mb.MB_ERR_UNSUPPORTED


def test_binding_rejects_cpu_shape_errors():
    import torch
    x = torch.zeros(1, 4, 8, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        mb.make_args(x, x, torch.zeros(1, 4, 16, dtype=torch.bfloat16),
                     torch.zeros(1, 4, 16, dtype=torch.bfloat16), torch.zeros(8, 16),
                     torch.zeros(1, 4, 9, dtype=torch.bfloat16))
    with pytest.raises(TypeError):
        mb.make_args(x.float(), x, x, x, torch.zeros(8, 16), x)
    B = torch.zeros(1, 4, 16, dtype=torch.bfloat16)
    with pytest.raises(ValueError):          # neither dt nor dt_low
        mb.make_args(x, None, B, B, torch.zeros(8, 16), x)
    with pytest.raises(ValueError):          # both
        mb.make_args(x, x, B, B, torch.zeros(8, 16), x, dt_low=torch.zeros(1, 4, 64, dtype=torch.bfloat16),
                     W_dt=torch.zeros(8, 64, dtype=torch.bfloat16))
    xdbl = torch.zeros(1, 4, 96, dtype=torch.bfloat16)
    a = mb.make_args(x, None, xdbl[:, :, 64:80], xdbl[:, :, 80:], torch.zeros(8, 16), x,
                     dt_low=xdbl[:, :, :64], W_dt=torch.zeros(8, 64, dtype=torch.bfloat16))
    assert (a.dt_rank, a.dt_low_stride, a.bc_stride, a.dt) == (64, 96, 96, None)


def test_selftest_timeout_checks():
    lib = mb.load_library()
    ws = FAKE + (200 << 32)
    assert lib.mb_selftest_timeout(None, 256, 1000, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_selftest_timeout(ws, 16, 1000, None) == mb.MB_ERR_INVALID_ARG        # too small
    assert lib.mb_selftest_timeout(ws + 16, 256, 1000, None) == mb.MB_ERR_INVALID_ARG   # not 256-aligned
    assert lib.mb_selftest_timeout(ws, 256, 0, None) == mb.MB_ERR_INVALID_ARG
    assert lib.mb_selftest_timeout(ws, 256, 5 * 10**9, None) == mb.MB_ERR_INVALID_ARG  # above the kernels' limit


def test_verify_resume_checks():
    lib = mb.load_library()
    a = _args(L=8)
    prev, acc, out, ws = FAKE + (30 << 32), FAKE + (31 << 32), FAKE + (32 << 32), FAKE + (200 << 32)
    call = lambda args=a, p=prev, c=acc, k=4, o=out, w=ws: lib.mb_scan_verify_resume(
        ctypes.byref(args), p, c, k, o, w, 256, None)
    assert call() in (mb.MB_OK, mb.MB_ERR_CUDA)               # valid (no GPU here)
    assert call(w=None) == mb.MB_ERR_INVALID_ARG              # the workspace receives bad counts
    assert call(k=0) == mb.MB_ERR_INVALID_ARG
    assert call(p=None) == mb.MB_ERR_INVALID_ARG
    assert call(c=acc + 2) == mb.MB_ERR_INVALID_ARG           # misaligned accept
    assert call(o=prev) == mb.MB_ERR_INVALID_ARG              # h_all overlaps h_all_prev
    assert call(o=a.x) == mb.MB_ERR_INVALID_ARG               # h_all overlaps an input
    b = _args(L=8)
    b.y = prev                                                # y overlaps h_all_prev
    assert call(args=b) == mb.MB_ERR_INVALID_ARG
    assert call(args=_args(batch=0, L=8)) == mb.MB_OK


def test_noalloc_prefill_host_checks():
    # mb_scan_prefill_noalloc applies mb_scan_prefill's argument and h_last
    # rules before it touches the GPU (here: before any CUDA call at all).
    lib = mb.load_library()
    f = lib.mb_scan_prefill_noalloc
    f.argtypes = [ctypes.POINTER(mb.mb_scan_args), ctypes.c_void_p, ctypes.c_void_p]
    f.restype = ctypes.c_int
    assert f(ctypes.byref(_args(batch=0)), None, None) == mb.MB_OK
    a = _fused()
    assert f(ctypes.byref(a), a.dt_low, None) == mb.MB_ERR_INVALID_ARG        # h_last overlaps dt_low
    assert f(ctypes.byref(a), a.W_dt, None) == mb.MB_ERR_INVALID_ARG          # h_last overlaps W_dt
    a = _args()
    assert f(ctypes.byref(a), a.h0 + 16, None) == mb.MB_ERR_INVALID_ARG       # partial overlap with h0
    assert f(ctypes.byref(a), a.B, None) == mb.MB_ERR_INVALID_ARG             # h_last overlaps B
    assert f(ctypes.byref(a), a.x + 4, None) == mb.MB_ERR_INVALID_ARG         # misaligned
    assert _prefill(_fused(), h_last=_fused().dt_low) == mb.MB_ERR_INVALID_ARG
    assert _prefill(_args(), h_last=_args().B) == mb.MB_ERR_INVALID_ARG
    # valid arguments: without a GPU the call then fails at its first CUDA call
    assert f(ctypes.byref(_args()), FAKE + (230 << 32), None) in (mb.MB_OK, mb.MB_ERR_CUDA)


def test_conv_xproj_host_checks():
    # mb_conv_xproj: shapes, dtype, alignment, workspace and aliasing are
    # checked on the host before any CUDA call.
    lib = mb.load_library()
    B, W_, n = 256, 4608, 176
    assert lib.mb_conv_xproj_workspace_size(B, W_, n) == 256 + (W_ // 128) * B * n * 4
    assert lib.mb_conv_xproj_workspace_size(B, 4600, n) == 0          # width % 128 != 0
    assert lib.mb_conv_xproj_workspace_size(B, W_, 168) == 0          # no kernel for this n_out
    need = lib.mb_conv_xproj_workspace_size(B, W_, n)
    p = {k: FAKE + (i << 32) for i, k in enumerate(("x", "st", "w", "b", "W", "xc", "out", "ws"), start=240)}

    def call(n_out=n, width=W_, batch=B, dtype=mb.MB_BF16, ws_bytes=need, **kw):
        q = dict(p, **kw)
        return lib.mb_conv_xproj(q["x"], q["st"], q["w"], q["b"], q["W"], q["xc"], q["out"], batch, width, n_out,
                                 dtype, q["ws"], ws_bytes, None)

    assert call() in (mb.MB_OK, mb.MB_ERR_CUDA)                     # valid (no GPU here)
    assert call(b=None) in (mb.MB_OK, mb.MB_ERR_CUDA)               # bias is optional
    assert call(batch=0) == mb.MB_OK                                # nothing to do
    assert call(n_out=168) == mb.MB_ERR_UNSUPPORTED
    assert call(width=4600) == mb.MB_ERR_UNSUPPORTED
    assert call(dtype=mb.MB_F32) == mb.MB_ERR_UNSUPPORTED
    assert call(batch=-1) == mb.MB_ERR_INVALID_ARG
    assert call(ws_bytes=need - 4) == mb.MB_ERR_INVALID_ARG         # workspace too small
    assert call(ws=p["ws"] + 16) == mb.MB_ERR_INVALID_ARG           # workspace not 256-byte aligned
    assert call(W=None) == mb.MB_ERR_INVALID_ARG
    assert call(x=p["x"] + 8) == mb.MB_ERR_INVALID_ARG              # misaligned
    assert call(xc=p["x"]) == mb.MB_ERR_INVALID_ARG                 # xc is x
    assert call(out=p["xc"]) == mb.MB_ERR_INVALID_ARG               # out is xc
    assert call(out=p["st"] + 4096) == mb.MB_ERR_INVALID_ARG        # out inside the window
    assert call(ws=p["W"]) == mb.MB_ERR_INVALID_ARG                 # workspace over W
    assert call(st=p["b"] - 256) == mb.MB_ERR_INVALID_ARG           # window runs into the bias

