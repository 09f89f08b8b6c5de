"""B and C read with a row stride (bc_stride): the same problem with B, C as
column blocks of one wider [.., S] buffer must give bit-identical results to
contiguous B, C, for every entry point that reads them."""
import pytest
import torch

from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _strided(B, C, S=48, lead=8):
    """Copies of B, C [b, L, 16] placed at columns lead.. and lead+16.. of a
    [b, L, S] buffer (rows S elements apart)."""
    b, L, N = B.shape
    buf = torch.full((b, L, S), float("nan"), device=B.device, dtype=B.dtype)
    buf[:, :, lead:lead + N] = B
    buf[:, :, lead + N:lead + 2 * N] = C
    return buf[:, :, lead:lead + N], buf[:, :, lead + N:lead + 2 * N]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_prefill_verify_backward_with_strided_bc(dtype):
    inp = make_inputs(3, 40, 64, 16, dtype, "normal", seed=5, device=DEV)
    Bs, Cs = _strided(inp["B"], inp["C"])
    assert not Bs.is_contiguous()
    outs = []
    for B, C in ((inp["B"], inp["C"]), (Bs, Cs)):
        y = torch.empty_like(inp["x"])
        _, hl, ck = mb.mb_scan_prefill_ckpt(inp["x"], inp["dt"], B, C, inp["A"], y, z=inp["z"], D=inp["D"],
                                            dt_bias=inp["dt_bias"], h0=inp["h0"],
                                            h_last=torch.empty_like(inp["h0"]))
        yv = torch.empty_like(inp["x"])
        ha = torch.empty(3, 40, 64, 16, device=DEV)
        mb.mb_scan_verify(inp["x"], inp["dt"], B, C, inp["A"], yv, ha, z=inp["z"], D=inp["D"],
                          dt_bias=inp["dt_bias"], h0=inp["h0"])
        g = torch.Generator(device=DEV).manual_seed(1)
        dout = torch.randn(inp["x"].shape, device=DEV, generator=g).to(inp["x"].dtype)
        gr = mb.mb_scan_backward(inp["x"], inp["dt"], B, C, inp["A"], ck, dout, z=inp["z"], D=inp["D"],
                                 dt_bias=inp["dt_bias"], h0=inp["h0"])
        outs.append([y, hl, ck, yv, ha] + [gr[k] for k in ("dx", "ddt", "dz", "dh0")])
    for a, b in zip(*outs):
        assert torch.equal(a, b)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_step_and_resume_with_strided_bc(dtype):
    inp = make_inputs(6, 1, 128, 16, dtype, "normal", seed=6, device=DEV)
    Bs, Cs = _strided(inp["B"], inp["C"], S=40)
    res = []
    for B, C in ((inp["B"], inp["C"]), (Bs, Cs)):
        st = inp["h0"].clone()
        y = torch.empty_like(inp["x"])
        mb.mb_step(inp["x"], inp["dt"], B, C, inp["A"], y, st, z=inp["z"], D=inp["D"], dt_bias=inp["dt_bias"])
        h_all = torch.randn(6, 3, 128, 16, device=DEV, generator=torch.Generator(device=DEV).manual_seed(2))
        acc = torch.tensor([0, 1, 2, 3, 0, 3], dtype=torch.int32, device=DEV)
        st2 = torch.empty_like(st)
        y2 = torch.empty_like(y)
        mb.mb_step_resume(inp["x"], inp["dt"], B, C, inp["A"], y2, h_all, acc, st2, z=inp["z"], D=inp["D"],
                          dt_bias=inp["dt_bias"], h0=inp["h0"])
        res.append([st, y, st2, y2])
    for a, b in zip(*res):
        assert torch.equal(a, b)
