"""GPU parity with a general diagonal A. The workloads use Mamba's S4D-real
initialisation A[d, n] = -(n + 1), identical for every channel, so a kernel
that indexed A by the state alone (or by the wrong channel) would pass them.
Here A[d, n] = -exp(u), u uniform on [log 0.2, log 5] independently per
(d, n), as a trained Mamba's A = -exp(A_log) is, for every entry point that
reads A. Same error metric and bars as the other parity tests."""
import math

import pytest
import torch

from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

import oracle
from _parity import TOL, TOL_STATE, oracle_scan, rel_err, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _general(batch, L, Dn, dtype, h0, seed, **kw):
    inp = make_inputs(batch, L, Dn, 16, dtype, h0, seed=seed, device=DEV, **kw)
    g = torch.Generator(device=DEV).manual_seed(seed + 7)
    u = torch.rand(Dn, 16, device=DEV, generator=g) * (math.log(5.0) - math.log(0.2)) + math.log(0.2)
    inp["A"] = (-torch.exp(u)).contiguous()
    return inp


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_prefill_and_verify_general_a(dtype):
    inp = _general(3, 37, 8 * 67, dtype, "normal", 81)
    y = torch.empty_like(inp["x"])
    hl = torch.empty(3, 8 * 67, 16, device=DEV)
    mb.mb_scan_prefill(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=hl)
    ry, rh, rall = oracle_scan(inp, want_h_all=True)
    assert rel_err(y, ry) <= TOL[dtype] and rel_err(hl, rh) <= TOL_STATE[dtype]
    for L in (16, 37):   # single-chunk and multi-chunk verify spans
        sub = {k: (v[:, :L].contiguous() if k in ("x", "z", "dt", "B", "C") else v) for k, v in inp.items()}
        yv = torch.empty_like(sub["x"])
        h_all = torch.empty(3, L, 8 * 67, 16, device=DEV)
        mb.mb_scan_verify(sub["x"], sub["dt"], sub["B"], sub["C"], sub["A"], yv, h_all, z=sub["z"], D=sub["D"],
                          dt_bias=sub["dt_bias"], h0=sub["h0"])
        assert rel_err(yv, ry[:, :L]) <= TOL[dtype] and rel_err(h_all, rall[:, :L]) <= TOL_STATE[dtype]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_step_and_resume_general_a(dtype):
    inp = _general(5, 6, 8 * 67, dtype, "normal", 82)
    ry, _, rall = oracle_scan(inp, want_h_all=True)
    state = inp["h0"].clone()
    for t in range(3):   # three single-byte steps
        sl = slice(t, t + 1)
        y = torch.empty_like(inp["x"][:, sl])
        mb.mb_step(inp["x"][:, sl].contiguous(), inp["dt"][:, sl].contiguous(), inp["B"][:, sl].contiguous(),
                   inp["C"][:, sl].contiguous(), inp["A"], y, state, z=inp["z"][:, sl].contiguous(), D=inp["D"],
                   dt_bias=inp["dt_bias"])
        assert rel_err(y, ry[:, sl]) <= TOL[dtype]
    assert rel_err(state, rall[:, 2]) <= TOL_STATE[dtype]
    # resume: verify the first 5 bytes, keep a per-stream prefix, step byte 5 from it
    span = {k: (v[:, :5].contiguous() if k in ("x", "z", "dt", "B", "C") else v) for k, v in inp.items()}
    yv = torch.empty_like(span["x"])
    h_all = torch.empty(5, 5, 8 * 67, 16, device=DEV)
    mb.mb_scan_verify(span["x"], span["dt"], span["B"], span["C"], span["A"], yv, h_all, z=span["z"],
                      D=span["D"], dt_bias=span["dt_bias"], h0=span["h0"])
    acc = torch.tensor([0, 5, 2, 1, 4], dtype=torch.int32, device=DEV)
    nxt = {k: inp[k][:, 5:6].contiguous() for k in ("x", "z", "dt", "B", "C")}
    y = torch.empty_like(nxt["x"])
    out = torch.empty_like(inp["h0"])
    mb.mb_step_resume(nxt["x"], nxt["dt"], nxt["B"], nxt["C"], inp["A"], y, h_all, acc, out, z=nxt["z"],
                      D=inp["D"], dt_bias=inp["dt_bias"], h0=inp["h0"])
    for s, a in enumerate(acc.tolist()):   # oracle: one step from the kept state
        start = to_np(inp["h0"][s:s + 1]) if a == 0 else to_np(h_all[s:s + 1, a - 1])
        one = lambda k: to_np(nxt[k][s:s + 1])
        wy, wh, _ = oracle.scan(one("x"), one("dt"), one("B"), one("C"), to_np(inp["A"]), z=one("z"),
                                D=to_np(inp["D"]), dt_bias=to_np(inp["dt_bias"]), h0=start)
        assert rel_err(y[s:s + 1], wy) <= TOL[dtype] and rel_err(out[s:s + 1], wh) <= TOL_STATE[dtype]


def test_backward_general_a():
    inp = _general(2, 40, 96, "f32", "normal", 83)
    x = inp["x"]
    g = torch.Generator(device=DEV).manual_seed(84)
    dout = torch.randn(x.shape, device=DEV, generator=g)
    dhl = torch.randn(2, 96, 16, device=DEV, generator=g)
    y = torch.empty_like(x)
    _, _, ck = mb.mb_scan_prefill_ckpt(x, inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"], D=inp["D"],
                                       dt_bias=inp["dt_bias"], h0=inp["h0"])
    got = mb.mb_scan_backward(x, inp["dt"], inp["B"], inp["C"], inp["A"], ck, dout, z=inp["z"], D=inp["D"],
                              dt_bias=inp["dt_bias"], h0=inp["h0"], dh_last=dhl)
    want = oracle.scan_backward(to_np(x), to_np(inp["dt"]), to_np(inp["B"]), to_np(inp["C"]), to_np(inp["A"]),
                                to_np(dout), z=to_np(inp["z"]), D=to_np(inp["D"]), dt_bias=to_np(inp["dt_bias"]),
                                h0=to_np(inp["h0"]), dh_last=to_np(dhl))
    for k in ("dx", "ddt", "dz", "dh0"):
        assert rel_err(got[k], want[k]) <= 1e-4, k
    for k in ("dB", "dC", "dA", "dD", "ddt_bias"):
        assert rel_err(got[k], want[k]) <= 1e-3, k


def test_fused_delta_prefill_general_a():
    inp = _general(2, 40, 96, "bf16", "normal", 85, dt_rank=112)
    y = torch.empty_like(inp["x"])
    hl = torch.empty(2, 96, 16, device=DEV)
    mb.mb_scan_prefill(inp["x"], None, inp["B"], inp["C"], inp["A"], y, z=inp["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=hl, dt_low=inp["dt_low"], W_dt=inp["W_dt"])
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["bf16"] and rel_err(hl, rh) <= TOL_STATE["bf16"]
