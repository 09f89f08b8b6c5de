"""mb_scan_prefill_noalloc: the prefill for callers that cannot allocate device
memory (graph-recorded code, allocator-owned or real-time paths, plugins that
only get their input and output buffers). It must give the same results as
mb_scan_prefill with a caller workspace, call after call, although all its
calls share one library-owned scratch array per GPU.

This file is named so that pytest collects it last.
"""
import ctypes

import pytest
import torch

from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

from _parity import TOL, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _lib():
    lib = mb.load_library()
    f = lib.mb_scan_prefill_noalloc
    f.argtypes = [ctypes.POINTER(mb.mb_scan_args), ctypes.c_void_p, ctypes.c_void_p]
    f.restype = ctypes.c_int
    return lib


def _noalloc(lib, inp, stream):
    y = torch.empty_like(inp["x"])
    h_last = torch.empty(inp["x"].shape[0], inp["x"].shape[2], 16, device=DEV)
    args = mb.make_args(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"],
                        D=inp["D"], dt_bias=inp["dt_bias"], h0=inp["h0"])
    rc = lib.mb_scan_prefill_noalloc(ctypes.byref(args), ctypes.c_void_p(h_last.data_ptr()),
                                     ctypes.c_void_p(stream.cuda_stream))
    assert rc == mb.MB_OK, mb.mb_status_string(rc)
    return y, h_last


def _with_workspace(inp, stream):
    y = torch.empty_like(inp["x"])
    h_last = torch.empty(inp["x"].shape[0], inp["x"].shape[2], 16, device=DEV)
    mb.mb_scan_prefill(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=h_last, stream=stream)
    return y, h_last


@pytest.mark.parametrize("dtype, tol", [("bf16", TOL["bf16"]), ("f32", TOL["f32"])])
def test_noalloc_matches_prefill_twice(dtype, tol):
    lib = _lib()
    stream = torch.cuda.Stream(DEV)
    cases = [make_inputs(3, 100, 96, 16, dtype, "normal", seed=201, device=DEV),
             make_inputs(2, 47, 64, 16, dtype, "zeros", seed=202, device=DEV)]
    for inp in cases:                      # two calls in a row on the shared scratch
        with torch.cuda.stream(stream):
            y_ref, h_ref = _with_workspace(inp, stream)
            y, h = _noalloc(lib, inp, stream)
        stream.synchronize()
        assert rel_err(y, y_ref.double().cpu().numpy()) <= tol
        assert rel_err(h, h_ref.double().cpu().numpy()) <= tol


def test_noalloc_rejects_bad_arguments_before_launch():
    lib = _lib()
    inp = make_inputs(1, 8, 64, 16, "bf16", "zeros", seed=203, device=DEV)
    y = torch.empty_like(inp["x"])
    args = mb.make_args(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"],
                        D=inp["D"], dt_bias=inp["dt_bias"])
    args.d_state = 8
    assert lib.mb_scan_prefill_noalloc(ctypes.byref(args), None, None) == mb.MB_ERR_UNSUPPORTED
    args.d_state = 16
    args.y = args.x                         # output aliasing an input
    assert lib.mb_scan_prefill_noalloc(ctypes.byref(args), None, None) == mb.MB_ERR_INVALID_ARG
