"""GPU parity of the training path: mb_scan_prefill_ckpt (forward with state
checkpoints) and mb_scan_backward against the fp64 oracle (oracle.scan and
oracle.scan_backward, the latter pinned by finite differences).

Bars (err = max |g - r| / max(|r|, rms(r)) per tensor): fp32 inputs 1e-4 for
everything but the channel sums dB, dC, dA, dD, ddt_bias, whose fp32 atomic
accumulation over up to 2048 channels x 8192 steps is allowed 1e-3; bf16
inputs 2e-2 (the bf16 rounding of dx, ddt, dz dominates).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import WORKLOADS, make_inputs, workload_inputs

from _parity import rel_err, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
TOKEN_GRADS = ("dx", "ddt", "dz")
SUM_GRADS = ("dB", "dC", "dA", "dD", "ddt_bias")


def _bars(dtype):
    return (1e-4, 1e-3) if dtype == "f32" else (2e-2, 2e-2)


def _upstream(inp, seed, dh_last=True):
    g = torch.Generator(device=DEV).manual_seed(seed)
    x = inp["x"]
    dout = torch.randn(x.shape, device=DEV, generator=g).to(x.dtype)
    dhl = torch.randn(x.shape[0], x.shape[2], 16, device=DEV, generator=g) if dh_last else None
    return dout, dhl


def _gpu(inp, dout, dhl):
    x = inp["x"]
    y = torch.empty_like(x)
    _, _, ck = mb.mb_scan_prefill_ckpt(x, inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"],
                                       D=inp["D"], dt_bias=inp["dt_bias"], h0=inp["h0"])
    g = mb.mb_scan_backward(x, inp["dt"], inp["B"], inp["C"], inp["A"], ck, dout, z=inp["z"], D=inp["D"],
                            dt_bias=inp["dt_bias"], h0=inp["h0"], dh_last=dhl)
    return y, ck, g


def _oracle(inp, dout, dhl, chans=None, rows=None, nthreads=None):
    def sel(t, kind):
        if t is None:
            return None
        a = to_np(t)
        if rows is not None and kind in ("tok", "bc", "st"):
            a = a[rows]
        if chans is not None:
            if kind == "tok":
                a = a[:, :, chans]
            elif kind == "st":
                a = a[:, chans]
            elif kind == "par":
                a = a[chans]
        return a
    return oracle.scan_backward(sel(inp["x"], "tok"), sel(inp["dt"], "tok"), sel(inp["B"], "bc"),
                                sel(inp["C"], "bc"), sel(inp["A"], "par"), sel(dout, "tok"),
                                z=sel(inp["z"], "tok"), D=sel(inp["D"], "par"), dt_bias=sel(inp["dt_bias"], "par"),
                                h0=sel(inp["h0"], "st"), dh_last=sel(dhl, "st"), nthreads=nthreads)


@pytest.mark.parametrize("dtype, batch, L, Dn, h0", [("f32", 2, 40, 64, "normal"), ("bf16", 3, 64, 72, "normal"),
                                                     ("f32", 1, 16, 32, "zeros"), ("bf16", 2, 1, 40, "zeros"),
                                                     ("f32", 2, 33, 96, "normal")])
def test_checkpoints_are_the_forward_states(dtype, batch, L, Dn, h0):
    inp = make_inputs(batch, L, Dn, 16, dtype, h0, seed=L + Dn, device=DEV)
    x = inp["x"]
    y1, y2 = torch.empty_like(x), torch.empty_like(x)
    hl1 = torch.empty(batch, Dn, 16, device=DEV)
    hl2 = torch.empty_like(hl1)
    mb.mb_scan_prefill(x, inp["dt"], inp["B"], inp["C"], inp["A"], y1, z=inp["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=hl1)
    _, _, ck = mb.mb_scan_prefill_ckpt(x, inp["dt"], inp["B"], inp["C"], inp["A"], y2, z=inp["z"],
                                       D=inp["D"], dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=hl2)
    assert torch.equal(y1, y2) and torch.equal(hl1, hl2)   # same forward
    _, _, h_all = oracle.scan(x, inp["dt"], inp["B"], inp["C"], inp["A"], z=inp["z"], D=inp["D"],
                              dt_bias=inp["dt_bias"], h0=inp["h0"], want_h_all=True)
    start = to_np(inp["h0"]) if inp["h0"] is not None else np.zeros((batch, Dn, 16))
    want = np.stack([start] + [h_all[:, 16 * i - 1] for i in range(1, ck.shape[1])], axis=1)
    assert rel_err(ck, want) <= 1e-4


@pytest.mark.parametrize("dtype, batch, L, Dn, h0, gate, dh_last", [
    ("f32", 2, 40, 64, "normal", True, True),     # ragged last chunk
    ("bf16", 3, 64, 72, "normal", True, True),    # ragged channel tile
    ("f32", 1, 16, 32, "zeros", False, False),    # no gate, no h0, no dh_last
    ("f32", 2, 1, 40, "normal", True, True),      # one step
    ("bf16", 2, 49, 128, "zeros", True, False),
])
def test_backward_matches_oracle(dtype, batch, L, Dn, h0, gate, dh_last):
    inp = make_inputs(batch, L, Dn, 16, dtype, h0, seed=100 + L, device=DEV, gate=gate)
    dout, dhl = _upstream(inp, seed=L, dh_last=dh_last)
    _, _, got = _gpu(inp, dout, dhl)
    want = _oracle(inp, dout, dhl)
    tok_bar, sum_bar = _bars(dtype)
    for k in TOKEN_GRADS + ("dh0",):
        if want[k] is None:
            assert got[k] is None
            continue
        assert rel_err(got[k], want[k]) <= tok_bar, k
    for k in SUM_GRADS:
        assert rel_err(got[k], want[k]) <= sum_bar, k


def test_backward_empty_sequence_passes_the_state_gradient():
    inp = make_inputs(2, 0, 64, 16, "f32", "normal", seed=3, device=DEV)
    dout, dhl = _upstream(inp, seed=1)
    ck = torch.empty(2, 0, 64, 16, device=DEV)
    g = mb.mb_scan_backward(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], ck, dout, z=inp["z"],
                            D=inp["D"], dt_bias=inp["dt_bias"], h0=inp["h0"], dh_last=dhl)
    assert torch.equal(g["dh0"], dhl)
    assert torch.all(g["dA"] == 0) and torch.all(g["dD"] == 0) and torch.all(g["ddt_bias"] == 0)


@pytest.mark.parametrize("name", ["mambabyte353m_prefill_b8_L8192"])
def test_backward_full_size_sampled(name):
    w = WORKLOADS[name]
    inp = workload_inputs(w, DEV)
    dout, dhl = _upstream(inp, seed=5)
    _, _, got = _gpu(inp, dout, dhl)
    torch.cuda.synchronize()
    # per-channel outputs and the batch sums of dA, dD, ddt_bias on sampled channels
    chans = np.array([0, 1, 31, 32, 777, 1024, 2046, 2047])
    want = _oracle(inp, dout, dhl, chans=chans)
    tok_bar, sum_bar = _bars("bf16")
    for k in TOKEN_GRADS:
        assert rel_err(got[k][:, :, chans], want[k]) <= tok_bar, k
    assert rel_err(got["dh0"][:, chans], want["dh0"]) <= tok_bar
    for k in ("dA", "dD", "ddt_bias"):
        assert rel_err(got[k][chans], want[k]) <= sum_bar, k
    # the channel sums dB, dC of batch row 0 (all 2048 channels)
    row = _oracle(inp, dout, dhl, rows=[0])
    for k in ("dB", "dC"):
        assert rel_err(got[k][:1], row[k]) <= sum_bar, k
