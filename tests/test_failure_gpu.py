"""Failure detection on the GPU without a fault: every device-side wait of
the library is bounded. A kernel made to wait on a barrier that nothing ever
arrives on gives up after its limit, records MB_ERR_TIMEOUT in the caller's
workspace and returns; the host reads the status, and the context keeps
working (a prefill on the same stream and workspace still matches the oracle)."""
import pytest
import torch

from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

from _parity import TOL, TOL_STATE, oracle_scan, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def test_bounded_wait_reports_timeout_and_context_survives():
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    limit = 2_000_000                                    # about 1 ms of SM clocks
    mb.mb_selftest_timeout(ws, limit)
    st, detail = mb.mb_check(ws)
    assert st == mb.MB_ERR_TIMEOUT
    assert limit < detail < 100 * limit                  # it waited out its limit, then returned
    assert mb.mb_check(ws) == (mb.MB_OK, -1)             # read and cleared
    inp = make_inputs(2, 40, 64, 16, "bf16", "normal", seed=71, device=DEV)
    y = torch.empty_like(inp["x"])
    hl = torch.empty(2, 64, 16, device=DEV)
    mb.mb_scan_prefill(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=hl, ws=ws)
    assert mb.mb_check(ws) == (mb.MB_OK, -1)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["bf16"] and rel_err(hl, rh) <= TOL_STATE["bf16"]


def test_step_status_channel():
    # The decode step takes an optional workspace where a timed-out wait of
    # its TMA ring would be recorded. A normal step leaves it clear, and the
    # workspace changes nothing in the results.
    inp = make_inputs(64, 1, 4608, 16, "bf16", "normal", seed=72, device=DEV)
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    st_a, st_b = inp["h0"].clone(), inp["h0"].clone()
    ya, yb = torch.empty_like(inp["x"]), torch.empty_like(inp["x"])
    kw = dict(z=inp["z"], D=inp["D"], dt_bias=inp["dt_bias"])
    for _ in range(2):
        mb.mb_step(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], ya, st_a, ws=ws, **kw)
        mb.mb_step(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], yb, st_b, **kw)
    assert mb.mb_check(ws) == (mb.MB_OK, -1)
    assert torch.equal(ya, yb) and torch.equal(st_a, st_b)
