"""Time split of long prefill spans with few channels: when batch rows x
channel tiles fill less than half of the GPU, mb_scan_prefill (given the
workspace mb_workspace_size asks for) scans each segment of L from zero to
summarise it (end state, product of decays), then scans every segment from
the start state the summaries before it give (the associative operator of
Section 2). Results against the oracle, and against the unsplit kernel (a
256-byte workspace): the same sums in another association, so close but not
bit-identical."""
import pytest
import torch

from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

from _parity import TOL, TOL_STATE, oracle_channels, oracle_scan, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _prefill(inp, ws):
    y = torch.empty_like(inp["x"])
    hl = torch.empty(inp["x"].shape[0], inp["x"].shape[2], 16, device=DEV)
    mb.mb_scan_prefill(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp.get("z"), D=inp.get("D"),
                       dt_bias=inp.get("dt_bias"), h0=inp.get("h0"), h_last=hl, ws=ws)
    return y, hl


def _ws(inp, split=True):
    a = mb.make_args(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], torch.empty_like(inp["x"]), z=inp.get("z"))
    n = mb.mb_workspace_size(a) if split else 256
    return torch.zeros(max(n, 256), dtype=torch.uint8, device=DEV), n


@pytest.mark.parametrize("dtype, b, L, Dn, h0", [("f32", 1, 2000, 64, "normal"), ("f32", 2, 1237, 96, "zeros"),
                                                  ("f32", 1, 4099, 40, "normal"), ("bf16", 1, 2000, 64, "normal"),
                                                  ("bf16", 2, 1237, 96, "zeros"), ("bf16", 1, 4099, 40, "normal")])
def test_split_prefill_against_oracle(dtype, b, L, Dn, h0):
    inp = make_inputs(b, L, Dn, 16, dtype, h0, seed=L + Dn, device=DEV)
    ws, n = _ws(inp)
    assert n > 256   # these spans are split
    y, hl = _prefill(inp, ws)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL[dtype] and rel_err(hl, rh) <= TOL_STATE[dtype]
    assert mb.mb_check(ws) == (mb.MB_OK, -1)
    ws1, _ = _ws(inp, split=False)
    y1, hl1 = _prefill(inp, ws1)   # unsplit: the same values up to fp32 reassociation
    if dtype == "f32":
        torch.testing.assert_close(y, y1, rtol=1e-4, atol=1e-4)
    else:   # y is rounded to bf16: a reassociated fp32 value may round one step apart
        torch.testing.assert_close(y.float(), y1.float(), rtol=1e-2, atol=1e-2)
    torch.testing.assert_close(hl, hl1, rtol=1e-4, atol=1e-5)


def test_split_batch1_prompt_prefill_sampled():
    """One prompt of 8192 bytes at d_inner 2048 (64 channel tiles): split."""
    inp = make_inputs(1, 8192, 2048, 16, "bf16", "normal", seed=97, device=DEV)
    ws, n = _ws(inp)
    assert n > 256
    y, hl = _prefill(inp, ws)
    chans = [0, 31, 32, 1000, 2047]
    ry, rh, _ = oracle_channels(inp, [0], chans)
    c_t = torch.tensor(chans, device=DEV)
    assert rel_err(y[:, :, c_t], ry) <= TOL["bf16"] and rel_err(hl[:, c_t], rh) <= TOL_STATE["bf16"]
    ws1, _ = _ws(inp, split=False)
    y1, hl1 = _prefill(inp, ws1)
    assert rel_err(hl, hl1.double().cpu().numpy()) <= 1e-4
    assert (y.float() - y1.float()).abs().max().item() <= 0.02 * y1.float().abs().max().item()


def test_wide_spans_are_not_split():
    inp = make_inputs(8, 256, 2048, 16, "bf16", "zeros", seed=98, device=DEV)
    _, n = _ws(inp)
    assert n == 256   # 8 rows x 64 tiles already fill the GPU


def test_split_training_forward_checkpoints_and_backward():
    """The checkpointed forward splits the same way; its checkpoints (the
    state before every 16-step chunk) and the backward that reads them match
    the unsplit forward's."""
    inp = make_inputs(1, 1500, 64, 16, "f32", "normal", seed=99, device=DEV)
    x = inp["x"]
    out = {}
    for split in (True, False):
        ws, n = _ws(inp, split)
        assert (n > 256) == split
        y = torch.empty_like(x)
        hl = torch.empty(1, 64, 16, device=DEV)
        _, _, ck = mb.mb_scan_prefill_ckpt(x, inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"], D=inp["D"],
                                           dt_bias=inp["dt_bias"], h0=inp["h0"], h_last=hl, ws=ws)
        g = torch.Generator(device=DEV).manual_seed(5)
        dout = torch.randn(x.shape, device=DEV, generator=g)
        grads = mb.mb_scan_backward(x, inp["dt"], inp["B"], inp["C"], inp["A"], ck, dout, z=inp["z"], D=inp["D"],
                                    dt_bias=inp["dt_bias"], h0=inp["h0"])
        out[split] = (y, hl, ck, grads)
    y, hl, ck, gr = out[True]
    y1, hl1, ck1, gr1 = out[False]
    torch.testing.assert_close(ck, ck1, rtol=1e-4, atol=1e-5)
    torch.testing.assert_close(y, y1, rtol=1e-4, atol=1e-4)
    torch.testing.assert_close(hl, hl1, rtol=1e-4, atol=1e-5)
    for k in ("dx", "ddt", "dz", "dB", "dC", "dA", "dh0"):
        assert rel_err(gr[k], gr1[k].double().cpu().numpy()) <= 1e-3, k
