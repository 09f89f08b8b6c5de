"""mb_scan_prefill_noalloc: the prefill for callers that cannot allocate device
memory (code under an allocator that owns all device memory, real-time paths
that must not allocate after start-up, plugins that only get their input and
output buffers). Its only scratch is a 256-byte array inside the library, one
per GPU, shared by every call; it holds the status block, not the segment
summaries of the time split, so every span runs unsplit. Its results must
therefore equal, bit for bit, those of mb_scan_prefill given a 256-byte
workspace, call after call, and match the fp64 oracle.

This file is named so that pytest collects it last.
"""
import ctypes

import pytest
import torch

from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

from _parity import TOL, TOL_STATE, oracle_channels, oracle_scan, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _lib():
    lib = mb.load_library()
    f = lib.mb_scan_prefill_noalloc
    f.argtypes = [ctypes.POINTER(mb.mb_scan_args), ctypes.c_void_p, ctypes.c_void_p]
    f.restype = ctypes.c_int
    return lib


def _dt_kw(inp):
    if inp.get("dt_low") is not None:
        return dict(dt=None, dt_low=inp["dt_low"], W_dt=inp["W_dt"])
    return dict(dt=inp["dt"])


def _noalloc(lib, inp, stream):
    y = torch.empty_like(inp["x"])
    h_last = torch.empty(inp["x"].shape[0], inp["x"].shape[2], 16, device=DEV)
    kw = _dt_kw(inp)
    args = mb.make_args(inp["x"], kw.pop("dt"), inp["B"], inp["C"], inp["A"], y, z=inp["z"],
                        D=inp["D"], dt_bias=inp["dt_bias"], h0=inp["h0"], **kw)
    rc = lib.mb_scan_prefill_noalloc(ctypes.byref(args), ctypes.c_void_p(h_last.data_ptr()),
                                     ctypes.c_void_p(stream.cuda_stream))
    assert rc == mb.MB_OK, mb.mb_status_string(rc)
    return y, h_last


def _with_workspace(inp, stream, ws_bytes=256):
    """mb_scan_prefill with a caller workspace of ws_bytes (256: unsplit)."""
    y = torch.empty_like(inp["x"])
    h_last = torch.empty(inp["x"].shape[0], inp["x"].shape[2], 16, device=DEV)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device=DEV)
    kw = _dt_kw(inp)
    mb.mb_scan_prefill(inp["x"], kw.pop("dt"), inp["B"], inp["C"], inp["A"], y, z=inp["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=h_last, ws=ws, stream=stream, **kw)
    return y, h_last, ws


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_noalloc_equals_prefill_twice(dtype):
    lib = _lib()
    stream = torch.cuda.Stream(DEV)
    cases = [make_inputs(3, 100, 96, 16, dtype, "normal", seed=201, device=DEV),
             make_inputs(2, 47, 64, 16, dtype, "zeros", seed=202, device=DEV)]
    for inp in cases:                      # two calls in a row on the shared scratch
        with torch.cuda.stream(stream):
            y_ref, h_ref, ws = _with_workspace(inp, stream)
            y, h = _noalloc(lib, inp, stream)
        stream.synchronize()
        assert mb.mb_check(ws, stream)[0] == mb.MB_OK
        assert torch.equal(y, y_ref) and torch.equal(h, h_ref)
        ry, rh, _ = oracle_scan(inp)
        assert rel_err(y, ry) <= TOL[dtype] and rel_err(h, rh) <= TOL_STATE[dtype]


def test_noalloc_single_prompt_runs_unsplit():
    # batch 1 x 8192 x 2048: few enough channels that mb_scan_prefill splits the
    # span over L when its workspace has room for the summaries. noalloc has
    # none, so it must equal the unsplit prefill bit for bit, and the split one
    # within the parity bars; sampled channels are checked against the oracle.
    lib = _lib()
    stream = torch.cuda.Stream(DEV)
    inp = make_inputs(1, 8192, 2048, 16, "bf16", "normal", seed=204, device=DEV)
    a = mb.make_args(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], torch.empty_like(inp["x"]),
                     z=inp["z"], h0=inp["h0"])
    split_bytes = mb.mb_workspace_size(a)
    assert split_bytes > 256                                   # this shape is split-eligible
    with torch.cuda.stream(stream):
        y_ref, h_ref, _ = _with_workspace(inp, stream)
        y_split, h_split, _ = _with_workspace(inp, stream, split_bytes)
        for _ in range(2):
            y, h = _noalloc(lib, inp, stream)
            stream.synchronize()
            assert torch.equal(y, y_ref) and torch.equal(h, h_ref)
    assert rel_err(y, y_split.double().cpu().numpy()) <= TOL["bf16"]
    assert rel_err(h, h_split.double().cpu().numpy()) <= TOL_STATE["bf16"]
    g = torch.Generator().manual_seed(5)
    chans = sorted(set(torch.randperm(2048, generator=g)[:48].tolist()) | {0, 2047})
    ry, rh, _ = oracle_channels(inp, [0], chans)
    c_t = torch.tensor(chans, device=DEV)
    assert rel_err(y[:, :, c_t], ry) <= TOL["bf16"] and rel_err(h[:, c_t], rh) <= TOL_STATE["bf16"]


def test_noalloc_fused_delta_projection():
    # Delta formed from dt_low W_dt^T inside the kernel (Eq. 3), twice in a row
    lib = _lib()
    stream = torch.cuda.Stream(DEV)
    for seed in (205, 206):
        inp = make_inputs(2, 70, 128, 16, "bf16", "normal", seed=seed, device=DEV, dt_rank=64)
        with torch.cuda.stream(stream):
            y_ref, h_ref, _ = _with_workspace(inp, stream)
            y, h = _noalloc(lib, inp, stream)
        stream.synchronize()
        assert torch.equal(y, y_ref) and torch.equal(h, h_ref)
        ry, rh, _ = oracle_scan(inp)
        assert rel_err(y, ry) <= TOL["bf16"] and rel_err(h, rh) <= TOL_STATE["bf16"]


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
