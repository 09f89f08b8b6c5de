"""Helpers shared by the parity tests: the error metric and oracle calls on
the same seeded tensors that the CUDA path receives."""
import numpy as np
import torch

import oracle

# Tolerances on err = max |g - r| / max(|r|, rms(r)) per output tensor. TOL is
# the bar for y: 1e-4 with fp32 inputs, 2e-2 with bf16 inputs (y is rounded to
# bf16, 2^-9 relative, and inherits that rounding through D*x and the gate).
# TOL_STATE is the bar for the fp32 states (h_last, h_all, the stepped state):
# they are never rounded to bf16, so with bf16 inputs (widened exactly on both
# sides) only fp32 arithmetic separates them from the oracle (about 1e-5
# measured); 1e-3 still flags a state error 100x smaller than the y bar.
TOL = {"f32": 1e-4, "bf16": 2e-2}
TOL_STATE = {"f32": 1e-4, "bf16": 1e-3}


def rel_err(got, ref) -> float:
    """max_i |g_i - r_i| / max(|r_i|, rms(r)); 0 for empty tensors."""
    g = got.detach().cpu().double().numpy() if isinstance(got, torch.Tensor) else np.asarray(got, dtype=np.float64)
    r = np.asarray(ref, dtype=np.float64)
    assert g.shape == r.shape, (g.shape, r.shape)
    if r.size == 0:
        return 0.0
    rms = float(np.sqrt(np.mean(r * r)))
    floor = np.maximum(np.abs(r), rms if rms > 0 else 1e-30)
    return float(np.max(np.abs(g - r) / floor))


def to_np(t):
    return None if t is None else t.detach().cpu().double().numpy()


def oracle_dt(inp):
    """dt of an input dict: given, or formed from (dt_low, W_dt) by the oracle."""
    if inp.get("dt") is not None:
        return to_np(inp["dt"])
    return oracle.delta_projection(to_np(inp["dt_low"]), to_np(inp["W_dt"]))


def oracle_scan(inp, want_h_all=False, nthreads=None):
    """Oracle over a whole input dict from paper_2401_13660_gb300.inputs."""
    return oracle.scan(to_np(inp["x"]), oracle_dt(inp), to_np(inp["B"]), to_np(inp["C"]),
                       to_np(inp["A"]), z=to_np(inp.get("z")), D=to_np(inp.get("D")),
                       dt_bias=to_np(inp.get("dt_bias")), h0=to_np(inp.get("h0")),
                       want_h_all=want_h_all, nthreads=nthreads)


def oracle_channels(inp, rows, chans, nthreads=None):
    """Oracle on the sub-problem of batch rows `rows` and channels `chans`
    (channels are independent, so slicing them out is exact)."""
    rows = torch.as_tensor(rows)
    chans = torch.as_tensor(chans)

    def tok(t):
        return None if t is None else to_np(t.index_select(0, rows.to(t.device))[:, :, chans.to(t.device)])

    def bc(t):
        return to_np(t.index_select(0, rows.to(t.device)))

    h0 = inp.get("h0")
    h0s = None if h0 is None else to_np(h0.index_select(0, rows.to(h0.device))[:, chans.to(h0.device)])
    pick = lambda t: None if t is None else to_np(t[chans.to(t.device)])
    if inp.get("dt") is not None:
        dt = tok(inp["dt"])
    else:   # fused Delta projection: the selected rows of dt_low, the selected channels of W_dt
        dt = oracle.delta_projection(bc(inp["dt_low"]), to_np(inp["W_dt"][chans.to(inp["W_dt"].device)]))
    return oracle.scan(tok(inp["x"]), dt, bc(inp["B"]), bc(inp["C"]), pick(inp["A"]),
                       z=tok(inp.get("z")), D=pick(inp.get("D")), dt_bias=pick(inp.get("dt_bias")),
                       h0=h0s, nthreads=nthreads)
