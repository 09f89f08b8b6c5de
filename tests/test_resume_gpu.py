"""GPU parity of mb_step_resume, the decode step fused with the rollback of
speculative decoding (Algorithm 1): one step from h0[s] (accept 0) or
h_all[s, accept[s]-1]. Checked against the fp64 oracle's rollback followed by
its step, and bit for bit against mb_rollback followed by mb_step on the GPU
(the same arithmetic, so any indexing slip shows as a mismatch)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

from _parity import TOL, TOL_STATE, rel_err, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _problem(batch, k, Dn, dtype, h0="normal", seed=0):
    """A verify span of k drafted bytes (to produce h_all), accept counts that
    cover 0 and k, and the next byte's step inputs."""
    span = make_inputs(batch, k, Dn, 16, dtype, h0, seed=seed, device=DEV)
    nxt = make_inputs(batch, 1, Dn, 16, dtype, "zeros", seed=seed + 1, device=DEV)
    y = torch.empty_like(span["x"])
    h_all = torch.empty(batch, k, Dn, 16, device=DEV)
    mb.mb_scan_verify(span["x"], span["dt"], span["B"], span["C"], span["A"], y, h_all, z=span["z"],
                      D=span["D"], dt_bias=span["dt_bias"], h0=span["h0"])
    g = torch.Generator(device="cpu").manual_seed(seed + 2)
    acc = torch.randint(0, k + 1, (batch,), generator=g, dtype=torch.int32)
    acc[0] = 0
    if batch > 1:
        acc[1] = k
    return span, nxt, h_all, acc.to(DEV)


def _resume(span, nxt, h_all, acc, state, h0, ws=None):
    y = torch.empty_like(nxt["x"])
    mb.mb_step_resume(nxt["x"], nxt["dt"], nxt["B"], nxt["C"], span["A"], y, h_all, acc, state,
                      z=nxt["z"], D=span["D"], dt_bias=span["dt_bias"], h0=h0, ws=ws)
    return y


def _rollback_then_step(span, nxt, h_all, acc, h0):
    st = torch.empty(h_all.shape[0], h_all.shape[2], 16, device=DEV)
    mb.mb_rollback(h0 if h0 is not None else torch.zeros_like(st), h_all, acc, st)
    y = torch.empty_like(nxt["x"])
    mb.mb_step(nxt["x"], nxt["dt"], nxt["B"], nxt["C"], span["A"], y, st, z=nxt["z"], D=span["D"],
               dt_bias=span["dt_bias"])
    return y, st


def _oracle(span, nxt, h_all, acc, h0):
    start = oracle.rollback(to_np(h0), to_np(h_all), acc.cpu().numpy())
    y, h = oracle.step(start, to_np(nxt["x"][:, 0]), to_np(nxt["dt"][:, 0]), to_np(nxt["B"][:, 0]),
                       to_np(nxt["C"][:, 0]), to_np(span["A"]), z=to_np(nxt["z"][:, 0]),
                       D=to_np(span["D"]), dt_bias=to_np(span["dt_bias"]))
    return y, h


@pytest.mark.parametrize("dtype, batch, k, Dn", [("bf16", 32, 16, 2048), ("f32", 7, 5, 72),
                                                 ("bf16", 5, 1, 136)])
def test_resume_matches_oracle_and_rollback_then_step(dtype, batch, k, Dn):
    span, nxt, h_all, acc = _problem(batch, k, Dn, dtype)
    state = torch.full((batch, Dn, 16), float("nan"), device=DEV)
    y = _resume(span, nxt, h_all, acc, state, span["h0"])
    ry, rh = _oracle(span, nxt, h_all, acc, span["h0"])
    assert rel_err(y[:, 0], ry) <= TOL[dtype]
    assert rel_err(state, rh) <= TOL_STATE[dtype]
    y2, st2 = _rollback_then_step(span, nxt, h_all, acc, span["h0"])
    assert torch.equal(state, st2)
    assert torch.equal(y, y2)


def test_resume_in_place_over_the_cache_and_without_h0():
    span, nxt, h_all, acc = _problem(9, 4, 64, "f32", seed=5)
    cache = span["h0"].clone()
    _, want = _rollback_then_step(span, nxt, h_all, acc, span["h0"])
    _resume(span, nxt, h_all, acc, cache, cache)            # state aliases h0
    assert torch.equal(cache, want)
    # no cached state: accept 0 starts from zeros
    acc0 = torch.zeros_like(acc)
    state = torch.empty(9, 64, 16, device=DEV)
    y = _resume(span, nxt, h_all, acc0, state, None)
    ry, rh = _oracle(span, nxt, h_all, acc0, None)
    assert rel_err(state, rh) <= TOL_STATE["f32"] and rel_err(y[:, 0], ry) <= TOL["f32"]


def test_resume_bad_accept_is_reported_and_row_untouched():
    span, nxt, h_all, acc = _problem(6, 4, 64, "bf16", seed=9)
    acc[2] = 5          # > k
    acc[4] = -1
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    state = torch.full((6, 64, 16), 7.0, device=DEV)
    y = torch.full_like(nxt["x"], 3.0)
    mb.mb_step_resume(nxt["x"], nxt["dt"], nxt["B"], nxt["C"], span["A"], y, h_all, acc, state,
                      z=nxt["z"], D=span["D"], dt_bias=span["dt_bias"], h0=span["h0"], ws=ws)
    status, detail = mb.mb_check(ws)
    assert status == mb.MB_ERR_INVALID_ARG and detail in (2, 4)
    for s in (2, 4):
        assert torch.all(state[s] == 7.0) and torch.all(y[s] == 3.0)
    good = [s for s in range(6) if s not in (2, 4)]
    ry, rh = _oracle(span, nxt, h_all, torch.where(acc.cpu() < 0, 0, acc.cpu().clamp(max=4)).to(DEV),
                     span["h0"])
    assert rel_err(state[good], rh[good]) <= TOL_STATE["bf16"]
    assert rel_err(y[good, 0], ry[good]) <= TOL["bf16"]


# ------------------------------------------------------------------ verify resume
def _next_span(batch, k2, Dn, dtype, seed):
    return make_inputs(batch, k2, Dn, 16, dtype, "zeros", seed=seed, device=DEV)


@pytest.mark.parametrize("dtype, batch, k, k2, Dn, with_h0", [("bf16", 32, 16, 16, 2048, True),
                                                              ("f32", 7, 5, 19, 72, True),
                                                              ("bf16", 5, 3, 8, 8 * 67, False)])
def test_verify_resume_equals_rollback_then_verify(dtype, batch, k, k2, Dn, with_h0):
    """mb_scan_verify_resume is bit for bit mb_rollback then mb_scan_verify
    (the same scan from the same starting states), and matches the oracle."""
    span, _, h_all, acc = _problem(batch, k, Dn, dtype, h0="normal" if with_h0 else "zeros", seed=60 + k)
    h0 = span["h0"] if with_h0 else None
    nxt = _next_span(batch, k2, Dn, dtype, seed=70 + k2)
    y = torch.empty_like(nxt["x"])
    h_all2 = torch.empty(batch, k2, Dn, 16, device=DEV)
    mb.mb_scan_verify_resume(nxt["x"], nxt["dt"], nxt["B"], nxt["C"], span["A"], y, h_all2, h_all, acc,
                             z=nxt["z"], D=span["D"], dt_bias=span["dt_bias"], h0=h0)
    kept = torch.empty(batch, Dn, 16, device=DEV)
    mb.mb_rollback(h0 if h0 is not None else torch.zeros_like(kept), h_all, acc, kept)
    y_ref = torch.empty_like(nxt["x"])
    h_ref = torch.empty_like(h_all2)
    mb.mb_scan_verify(nxt["x"], nxt["dt"], nxt["B"], nxt["C"], span["A"], y_ref, h_ref, z=nxt["z"],
                      D=span["D"], dt_bias=span["dt_bias"], h0=kept)
    assert torch.equal(y, y_ref) and torch.equal(h_all2, h_ref)
    start = oracle.rollback(to_np(h0) if h0 is not None else np.zeros((batch, Dn, 16)), to_np(h_all),
                            acc.cpu().numpy())
    ry, _, rall = oracle.scan(to_np(nxt["x"]), to_np(nxt["dt"]), to_np(nxt["B"]), to_np(nxt["C"]),
                              to_np(span["A"]), z=to_np(nxt["z"]), D=to_np(span["D"]),
                              dt_bias=to_np(span["dt_bias"]), h0=start, want_h_all=True)
    assert rel_err(y, ry) <= TOL[dtype] and rel_err(h_all2, rall) <= TOL_STATE[dtype]


def test_verify_resume_bad_accept_is_reported_and_stream_untouched():
    span, _, h_all, acc = _problem(4, 6, 96, "f32", seed=81)
    nxt = _next_span(4, 8, 96, "f32", seed=82)
    acc[2] = 7                                    # > k_prev = 6
    y = torch.full_like(nxt["x"], 5.0)
    h_all2 = torch.full((4, 8, 96, 16), 5.0, device=DEV)
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    mb.mb_scan_verify_resume(nxt["x"], nxt["dt"], nxt["B"], nxt["C"], span["A"], y, h_all2, h_all, acc,
                             z=nxt["z"], D=span["D"], dt_bias=span["dt_bias"], h0=span["h0"], ws=ws)
    assert mb.mb_check(ws) == (mb.MB_ERR_INVALID_ARG, 2)
    assert torch.equal(y[2], torch.full_like(y[2], 5.0))
    assert torch.equal(h_all2[2], torch.full_like(h_all2[2], 5.0))
    assert not torch.equal(y[1], torch.full_like(y[1], 5.0))   # the other streams were scanned
