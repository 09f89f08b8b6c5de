"""Maximum sizes the API accepts: batch * seqlen * d_inner up to 2^31 tokens
and batch * d_inner * 16 up to 2^31 state elements. At these sizes every
element offset is beyond 32-bit range, so a 32-bit product anywhere in the
index arithmetic shows up as a wrong channel or row. Sampled channels (the
first, the last and one in the middle of each checked row) are compared with
the oracle; the rest must be finite."""
import pytest
import torch

from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

from _parity import TOL, TOL_STATE, oracle_channels, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def test_prefill_at_the_token_limit():
    b, L, Dn = 1, 1 << 20, 2048          # exactly 2^31 tokens
    inp = make_inputs(b, L, Dn, 16, "bf16", "normal", seed=91, device=DEV)
    y = torch.empty_like(inp["x"])
    hl = torch.empty(b, Dn, 16, device=DEV)
    mb.mb_scan_prefill(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=hl)
    assert torch.isfinite(hl).all()
    chans = [0, 1031, Dn - 1]
    ry, rh, _ = oracle_channels(inp, [0], chans)
    c_t = torch.tensor(chans, device=DEV)
    assert rel_err(y[:, :, c_t], ry) <= TOL["bf16"]
    assert rel_err(hl[:, c_t], rh) <= TOL_STATE["bf16"]
    # the very last positions of the last channel
    assert rel_err(y[0, -64:, Dn - 1], ry[0, -64:, -1]) <= TOL["bf16"]
    del inp, y


def test_step_at_the_state_limit():
    b, Dn = 1 << 14, 8192                # 2^27 channels = 2^31 state elements
    inp = make_inputs(b, 1, Dn, 16, "bf16", "normal", seed=92, device=DEV)
    state = inp["h0"].clone()
    y = torch.empty_like(inp["x"])
    mb.mb_step(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, state, z=inp["z"], D=inp["D"],
               dt_bias=inp["dt_bias"])
    rows, chans = [0, 9000, b - 1], [0, 4097, Dn - 1]
    ry, rh, _ = oracle_channels(inp, rows, chans)
    r_t, c_t = torch.tensor(rows, device=DEV), torch.tensor(chans, device=DEV)
    assert rel_err(y.index_select(0, r_t)[:, :, c_t], ry) <= TOL["bf16"]
    assert rel_err(state.index_select(0, r_t)[:, c_t], rh) <= TOL_STATE["bf16"]
    untouched = inp["h0"][1:].ne(state[1:]).any(dim=2).float().mean()   # every row was stepped
    assert untouched > 0.99


def test_verify_and_rollback_beyond_32_bit_offsets():
    b, k, Dn = 4096, 16, 4096            # h_all: 2^32 floats (16 GB)
    inp = make_inputs(b, k, Dn, 16, "bf16", "normal", seed=93, device=DEV, accept=True)
    y = torch.empty_like(inp["x"])
    h_all = torch.empty(b, k, Dn, 16, device=DEV)
    mb.mb_scan_verify(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, h_all, z=inp["z"], D=inp["D"],
                      dt_bias=inp["dt_bias"], h0=inp["h0"])
    rows, chans = [0, 2049, b - 1], [0, 3001, Dn - 1]
    ry, _, _ = oracle_channels(inp, rows, chans)
    r_t, c_t = torch.tensor(rows, device=DEV), torch.tensor(chans, device=DEV)
    assert rel_err(y.index_select(0, r_t)[:, :, c_t], ry) <= TOL["bf16"]
    # per-position states of the last row: the oracle over its first j + 1 bytes
    for j in (0, k - 1):
        sub = {key: (v[:, :j + 1] if key in ("x", "z", "dt", "B", "C") else v) for key, v in inp.items()}
        _, rh, _ = oracle_channels(sub, [b - 1], chans)
        assert rel_err(h_all[b - 1:, j][:, c_t], rh) <= TOL_STATE["bf16"]
    h_out = torch.empty_like(inp["h0"])
    mb.mb_rollback(inp["h0"], h_all, inp["accept"], h_out)
    acc = inp["accept"].long()
    for s in rows:   # an index gather: bit-exact
        a = int(acc[s])
        want = inp["h0"][s] if a == 0 else h_all[s, a - 1]
        assert torch.equal(h_out[s], want)
