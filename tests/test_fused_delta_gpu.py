"""GPU parity of the fused low-rank Delta projection (Eq. 3: the timestep
before softplus is W_Delta (W_R x)): the prefill and verify kernels take
dt_low = W_R x [batch, L, r] and W_Delta [d_inner, r] and form the timestep
tile by tile on the tensor cores. The oracle forms dt as an fp64 matrix
product and runs the same fp64 scan. Same error metric and bf16 bar as the
other parity tests."""
import pytest
import torch

from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import WORKLOADS, make_inputs, workload_inputs

from _parity import TOL, TOL_STATE, oracle_channels, oracle_scan, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _prefill(inp, **kw):
    x = inp["x"]
    y = torch.empty_like(x)
    hl = torch.empty(x.shape[0], x.shape[2], 16, device=x.device)
    mb.mb_scan_prefill(x, None, kw.get("B", inp["B"]), kw.get("C", inp["C"]), inp["A"], y, z=inp.get("z"),
                       D=inp.get("D"), dt_bias=inp.get("dt_bias"), h0=inp.get("h0"), h_last=hl,
                       dt_low=kw.get("dt_low", inp["dt_low"]), W_dt=inp["W_dt"])
    return y, hl


def _verify(inp):
    x = inp["x"]
    y = torch.empty_like(x)
    h_all = torch.empty(x.shape[0], x.shape[1], x.shape[2], 16, device=x.device)
    mb.mb_scan_verify(x, None, inp["B"], inp["C"], inp["A"], y, h_all, z=inp.get("z"), D=inp.get("D"),
                      dt_bias=inp.get("dt_bias"), h0=inp.get("h0"), dt_low=inp["dt_low"], W_dt=inp["W_dt"])
    return y, h_all


@pytest.mark.parametrize("shape", [(2, 40, 64, 64), (3, 37, 8 * 67, 112), (1, 16, 96, 144),
                                   (2, 5, 64, 256), (1, 333, 128, 80), (2, 1, 32, 64)])
@pytest.mark.parametrize("h0", ["zeros", "normal"])
def test_fused_prefill_against_oracle(shape, h0):
    """Ragged spans (L not a multiple of the 16-step chunk), ragged channel
    tiles (536 channels), ranks that fill one to four 64-wide boxes, partly."""
    b, L, Dn, r = shape
    inp = make_inputs(b, L, Dn, 16, "bf16", h0, seed=61 + L + r, device=DEV, dt_rank=r)
    y, hl = _prefill(inp)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["bf16"]
    assert rel_err(hl, rh) <= TOL_STATE["bf16"]


def test_fused_prefill_without_gate_and_optionals():
    inp = make_inputs(2, 50, 48, 16, "bf16", "zeros", seed=62, device=DEV, gate=False, dt_rank=64)
    inp["D"] = None
    inp["dt_bias"] = None
    y, hl = _prefill(inp)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["bf16"] and rel_err(hl, rh) <= TOL_STATE["bf16"]


def test_fused_prefill_reads_the_x_projection_in_place():
    """dt_low, B and C as column blocks of one [dt_low | B | C] row per (b, t),
    the layout of a single x-projection GEMM's output."""
    b, L, Dn, r = 2, 70, 96, 112
    inp = make_inputs(b, L, Dn, 16, "bf16", "normal", seed=63, device=DEV, dt_rank=r)
    xdbl = torch.cat([inp["dt_low"], inp["B"], inp["C"]], dim=2).contiguous()
    y, hl = _prefill(inp, dt_low=xdbl[:, :, :r], B=xdbl[:, :, r:r + 16], C=xdbl[:, :, r + 16:])
    yc, hc = _prefill(inp)
    torch.testing.assert_close(y, yc, rtol=0, atol=0)
    torch.testing.assert_close(hl, hc, rtol=0, atol=0)


@pytest.mark.parametrize("name", ["mambabyte353m_prefill_fused_r64_b8_L8192",
                                  "mambabyte972m_prefill_fused_r112_b4_L8192"])
def test_fused_prefill_full_size_sampled(name):
    """Full-size launch; 2 rows x 66 sampled channels (first and last tiles
    included) over the whole span against the oracle."""
    w = WORKLOADS[name]
    inp = workload_inputs(w, DEV)
    y, hl = _prefill(inp)
    assert torch.isfinite(y.float()).all() and torch.isfinite(hl).all()
    g = torch.Generator().manual_seed(8)
    rows = sorted(torch.randperm(w.batch, generator=g)[:2].tolist())
    chans = sorted(set(torch.randperm(w.d_inner, generator=g)[:64].tolist()) | {0, w.d_inner - 1})
    ry, rh, _ = oracle_channels(inp, rows, chans)
    r_t, c_t = torch.tensor(rows, device=DEV), torch.tensor(chans, device=DEV)
    assert rel_err(y.index_select(0, r_t)[:, :, c_t], ry) <= TOL["bf16"]
    assert rel_err(hl.index_select(0, r_t)[:, c_t], rh) <= TOL_STATE["bf16"]


def test_fused_verify_full_size_and_rollback():
    w = WORKLOADS["verify_fused_r64_s32_k16_D2048"]
    inp = workload_inputs(w, DEV)
    y, h_all = _verify(inp)
    ry, _, rall = oracle_scan(inp, want_h_all=True)
    assert rel_err(y, ry) <= TOL["bf16"]
    assert rel_err(h_all, rall) <= TOL_STATE["bf16"]
    h_out = torch.empty_like(inp["h0"])
    mb.mb_rollback(inp["h0"], h_all, inp["accept"], h_out)
    acc = inp["accept"].long()
    want = torch.where((acc == 0)[:, None, None], inp["h0"],
                       h_all[torch.arange(w.batch, device=DEV), (acc - 1).clamp(min=0)])
    assert torch.equal(h_out, want)


@pytest.mark.parametrize("L", [5, 16, 40])
def test_fused_verify_matches_fused_prefill(L):
    """Single- and multi-chunk verify spans: y equals the fused prefill's and
    the last per-position state equals its h_last."""
    inp = make_inputs(3, L, 8 * 67, 16, "bf16", "normal", seed=64 + L, device=DEV, dt_rank=144)
    y, h_all = _verify(inp)
    ry, _, rall = oracle_scan(inp, want_h_all=True)
    assert rel_err(y, ry) <= TOL["bf16"] and rel_err(h_all, rall) <= TOL_STATE["bf16"]
    yp, hl = _prefill(inp)
    torch.testing.assert_close(y.float(), yp.float(), rtol=1e-2, atol=1e-2)   # one bf16 ulp
    torch.testing.assert_close(h_all[:, -1], hl, rtol=1e-5, atol=1e-6)


def test_fused_rejections_through_the_binding():
    inp = make_inputs(1, 8, 32, 16, "f32", "zeros", seed=65, device=DEV, dt_rank=64)
    with pytest.raises(mb.MbError) as e:                     # fp32: unsupported
        _prefill(inp)
    assert e.value.status == mb.MB_ERR_UNSUPPORTED
    inp = make_inputs(1, 8, 32, 16, "bf16", "zeros", seed=65, device=DEV, dt_rank=32)
    with pytest.raises(mb.MbError) as e:                     # rank below one 64-wide box
        _prefill(inp)
    assert e.value.status == mb.MB_ERR_UNSUPPORTED
