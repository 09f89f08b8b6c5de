"""GPU parity of mb_conv_xproj, the decode-step convolution fused with the
x-projection (Figure 6; Table 6 "Pre-SSM 1D convolution" and "Delta, B, C
from input x"), against the fp64 oracle (oracle.conv1d_step, then the product
with W in fp64).

xc must equal mb_conv1d_step's output bit for bit (the same arithmetic in
the same order) and the window must hold the inputs exactly. Each projected
value is checked on its own against a bound fixed by the arithmetic: it is
the fp32 sum of K bf16 products rounded once to bf16, so

    |out - r| <= 2^-8 |r| + K 2^-23 sum_k |a_k W_nk|

with r the exact product of the bf16 operands: half a bf16 ulp (2^-9
relative) for the final rounding and K unit roundoffs of fp32 (2^-24) for
any order of the sum, each taken twice over for slack."""
import numpy as np
import pytest
import torch

import oracle
from paper_2401_13660_gb300 import mbscan as mb

from _parity import rel_err, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
BF = torch.bfloat16


def _weights(width, n_out, seed):
    g = torch.Generator(device=DEV).manual_seed(seed)
    w = torch.rand(width, 4, device=DEV, generator=g) - 0.5
    bias = torch.rand(width, device=DEV, generator=g) - 0.5
    W = (torch.randn(n_out, width, device=DEV, generator=g) / width ** 0.5).to(BF)
    return g, w, bias, W


def _check_projection(out, xc, W):
    xc64, W64 = to_np(xc), to_np(W)
    r = xc64 @ W64.T
    mag = np.abs(xc64) @ np.abs(W64).T
    bound = 2.0 ** -8 * np.abs(r) + W64.shape[1] * 2.0 ** -23 * mag
    err = np.abs(to_np(out) - r)
    assert np.all(err <= bound), float(np.max(err / np.maximum(bound, 1e-300)))


@pytest.mark.parametrize("batch, width, n_out", [(4, 128, 40), (256, 4608, 176), (67, 2048, 96),
                                                 (1, 3584, 144), (130, 256, 176), (64, 384, 40)])
def test_conv_xproj_matches_oracle(batch, width, n_out):
    g, w, bias, W = _weights(width, n_out, batch + width + n_out)
    state = torch.zeros(batch, 3, width, device=DEV, dtype=BF)
    state_ref = state.clone()
    st_np = np.zeros((batch, 3, width))
    ws = torch.zeros(mb.mb_conv_xproj_workspace_size(batch, width, n_out), dtype=torch.uint8, device=DEV)
    for t in range(4):
        b = bias if t % 2 == 0 else None
        x = torch.randn(batch, width, device=DEV, generator=g).to(BF)
        xc = torch.empty_like(x)
        out = torch.full((batch, n_out), float("nan"), device=DEV, dtype=BF)
        mb.mb_conv_xproj(x, state, w, W, xc, out, ws, bias=b)
        xc_ref = torch.empty_like(x)
        mb.mb_conv1d_step(x, state_ref, w, xc_ref, bias=b)
        assert torch.equal(xc, xc_ref) and torch.equal(state, state_ref)
        xo, st_np = oracle.conv1d_step(st_np, to_np(x), to_np(w), None if b is None else to_np(b))
        assert np.array_equal(to_np(state), st_np)
        assert np.max(np.abs(to_np(xc) - xo)) <= 2.0 ** -8 * max(np.max(np.abs(xo)), 1e-30)
        _check_projection(out, xc, W)
    assert mb.mb_check(ws) == (mb.MB_OK, -1)


def test_conv_xproj_empty_batch_and_unsupported():
    _, w, bias, W = _weights(256, 40, 5)
    empty = torch.empty(0, 256, device=DEV, dtype=BF)
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    out = torch.empty(0, 40, device=DEV, dtype=BF)
    mb.mb_conv_xproj(empty, torch.empty(0, 3, 256, device=DEV, dtype=BF), w, W, torch.empty_like(empty), out, ws,
                     bias=bias)
    assert mb.mb_conv_xproj_workspace_size(4, 200, 40) == 0     # width not a multiple of 128
    assert mb.mb_conv_xproj_workspace_size(4, 256, 48) == 0     # n_out not one of the model shapes
    x = torch.zeros(4, 256, device=DEV, dtype=BF)
    with pytest.raises(mb.MbError):
        mb.mb_conv_xproj(x, torch.zeros(4, 3, 256, device=DEV, dtype=BF), w, W, x, torch.empty(4, 40, device=DEV,
                         dtype=BF), torch.zeros(4096, dtype=torch.uint8, device=DEV))   # xc is x


def test_conv_xproj_in_place_of_the_unfused_pair():
    # The decoder's shapes (48 x 2304 model, batch 256): the fused call and
    # mb_conv1d_step + a cuBLAS GEMM give the same xc and window bit for bit,
    # and projections that differ from an fp32 GEMM of the same operands by
    # the one bf16 rounding and the fp32 summation order.
    batch, width, n_out = 256, 4608, 176
    g, w, bias, W = _weights(width, n_out, 11)
    s0 = (torch.randn(batch, 3, width, device=DEV, generator=g)).to(BF)
    sa, sb = s0.clone(), s0.clone()
    x = torch.randn(batch, width, device=DEV, generator=g).to(BF)
    xa, xb = torch.empty_like(x), torch.empty_like(x)
    oa = torch.empty(batch, n_out, device=DEV, dtype=BF)
    ws = torch.zeros(mb.mb_conv_xproj_workspace_size(batch, width, n_out), dtype=torch.uint8, device=DEV)
    mb.mb_conv_xproj(x, sa, w, W, xa, oa, ws, bias=bias)
    mb.mb_conv1d_step(x, sb, w, xb, bias=bias)
    ob = xb.float() @ W.float().t()
    assert torch.equal(xa, xb) and torch.equal(sa, sb)
    assert rel_err(oa, to_np(ob)) <= 2.0 ** -7



@pytest.mark.parametrize("batch", [256, 4])
def test_back_to_back_calls_on_one_window(batch):
    """Consecutive mb_conv_xproj calls on the same convolution window with
    nothing in between (each call may start, and prefetch its window tiles
    into L2, while the previous one still writes them): eagerly and from a CUDA
    graph they equal bit for bit the same calls with a device synchronisation
    after each, and the window ends as the oracle's."""
    width, n_out, T = 4608, 176, 6
    g, w, bias, W = _weights(width, n_out, 21 + batch)
    xs = [torch.randn(batch, width, device=DEV, generator=g).to(BF) for _ in range(T)]
    s0 = torch.randn(batch, 3, width, device=DEV, generator=g).to(BF)
    xcs = [torch.empty_like(x) for x in xs]
    outs = [torch.empty(batch, n_out, device=DEV, dtype=BF) for _ in range(T)]
    ws = torch.zeros(mb.mb_conv_xproj_workspace_size(batch, width, n_out), dtype=torch.uint8, device=DEV)

    def run(state, sync):
        for x, xc, out in zip(xs, xcs, outs):
            mb.mb_conv_xproj(x, state, w, W, xc, out, ws, bias=bias)
            if sync:
                torch.cuda.synchronize()
        return [t.clone() for t in xcs + outs]

    st_sync = s0.clone()
    r_sync = run(st_sync, True)
    st_eager = s0.clone()
    r_eager = run(st_eager, False)
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        run(s0.clone(), False)   # warm-up outside the capture
    torch.cuda.current_stream().wait_stream(side)
    st_graph = s0.clone()
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gr):
        for x, xc, out in zip(xs, xcs, outs):
            mb.mb_conv_xproj(x, st_graph, w, W, xc, out, ws, bias=bias)
    gr.replay()
    torch.cuda.synchronize()
    r_graph = [t.clone() for t in xcs + outs]
    for a, b in zip(r_eager + r_graph, r_sync + r_sync):
        assert torch.equal(a, b)
    assert torch.equal(st_eager, st_sync) and torch.equal(st_graph, st_sync)
    st_np = to_np(s0)
    for x in xs:
        _, st_np = oracle.conv1d_step(st_np, to_np(x), to_np(w), to_np(bias))
    assert np.array_equal(to_np(st_sync), st_np)
    assert mb.mb_check(ws) == (mb.MB_OK, -1)
