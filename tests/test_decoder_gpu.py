"""GPU parity of the block kernels (mb_rmsnorm, mb_conv1d_step) and of the
whole recurrent decoder (paper_2401_13660_gb300.decoder) against the fp64
oracle (oracle.rmsnorm, oracle.conv1d_step, oracle.block_step; bf16 casts at
the tensor boundaries where the GPU path keeps bf16)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.decoder import CONFIGS, WEIGHT_KEYS, Decoder

from _parity import rel_err, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
DT = {"f32": torch.float32, "bf16": torch.bfloat16}


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("batch, width, with_add", [(4, 64, True), (256, 2304, True), (3, 8192, False),
                                                     (1, 8, True), (9, 12296, True)])
def test_rmsnorm_matches_oracle(dtype, batch, width, with_add):
    g = torch.Generator(device=DEV).manual_seed(width)
    res = torch.randn(batch, width, device=DEV, generator=g)
    add = torch.randn(batch, width, device=DEV, generator=g).to(DT[dtype]) if with_add else None
    w = torch.rand(width, device=DEV, generator=g) + 0.5
    out = torch.empty(batch, width, device=DEV, dtype=DT[dtype])
    r0 = res.clone()
    mb.mb_rmsnorm(res, w, out, add=add, eps=1e-5)
    rr, ro = oracle.rmsnorm(to_np(r0), to_np(w), 1e-5, None if add is None else to_np(add))
    assert rel_err(res, rr) <= 1e-6
    assert rel_err(out, ro) <= (1e-5 if dtype == "f32" else 1e-2)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("batch, width", [(4, 64), (256, 4608), (3, 8), (7, 136)])
def test_conv_step_matches_oracle(dtype, batch, width):
    g = torch.Generator(device=DEV).manual_seed(batch + width)
    state = torch.zeros(batch, 3, width, device=DEV, dtype=DT[dtype])
    w = torch.rand(width, 4, device=DEV, generator=g) - 0.5
    bias = torch.rand(width, device=DEV, generator=g) - 0.5
    st_ref = np.zeros((batch, 3, width))
    for t in range(5):
        x = torch.randn(batch, width, device=DEV, generator=g).to(DT[dtype])
        out = torch.empty_like(x)
        mb.mb_conv1d_step(x, state, w, out, bias=bias if t % 2 == 0 else None)
        ro, st_ref = oracle.conv1d_step(st_ref, to_np(x), to_np(w), to_np(bias) if t % 2 == 0 else None)
        assert rel_err(out, ro) <= (1e-5 if dtype == "f32" else 1e-2)
        assert np.array_equal(to_np(state), st_ref)   # the window holds the inputs exactly


def _oracle_decode(dec, tokens_seq):
    cfg = dec.cfg
    layers = [{k: to_np(L[k]) for k in WEIGHT_KEYS} for L in dec.layers]
    emb = to_np(dec.emb)
    normf = to_np(dec.norm_f)
    B = dec.batch
    ssm = [np.zeros((B, cfg.d_inner, cfg.d_state)) for _ in layers]
    conv = [np.zeros((B, 3, cfg.d_inner)) for _ in layers]
    outs = []
    for tok in tokens_seq:
        residual = emb[tok.cpu().numpy()]
        add = None
        for l, L in enumerate(layers):
            residual, add, ssm[l], conv[l] = oracle.block_step(L, residual, add, ssm[l], conv[l], eps=cfg.eps)
        residual, hf = oracle.rmsnorm(residual, normf, cfg.eps, add)
        outs.append(oracle.bf16_round(oracle.bf16_round(hf) @ emb.T))
    return outs, ssm, conv


@pytest.mark.parametrize("graph", [False, True])
def test_decoder_matches_oracle(graph):
    dec = Decoder(CONFIGS["tiny_2x64"], batch=4, device=DEV, seed=3)
    if graph:
        dec.capture()
    g = torch.Generator(device=DEV).manual_seed(9)
    seq = [torch.randint(0, 256, (4,), device=DEV, generator=g) for _ in range(4)]
    got = [dec.step(t).clone() for t in seq]
    torch.cuda.synchronize()
    want, ssm, conv = _oracle_decode(dec, seq)
    for gl, wl in zip(got, want):
        assert rel_err(gl, wl) <= 2e-2
    for l in range(dec.cfg.n_layers):
        assert rel_err(dec.ssm[l], ssm[l]) <= 2e-2
        assert rel_err(dec.conv[l], conv[l]) <= 2e-2


def test_graph_replay_equals_eager():
    a = Decoder(CONFIGS["tiny_2x64"], batch=8, device=DEV, seed=4)
    b = Decoder(CONFIGS["tiny_2x64"], batch=8, device=DEV, seed=4)
    b.capture()
    g = torch.Generator(device=DEV).manual_seed(2)
    for _ in range(3):
        t = torch.randint(0, 256, (8,), device=DEV, generator=g)
        assert torch.equal(a.step(t), b.step(t))
    for x, y in zip(a.ssm + a.conv, b.ssm + b.conv):
        assert torch.equal(x, y)
