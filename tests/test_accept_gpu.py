"""GPU parity of mb_accept_topk (integer result: bit-exact) and its use in the
speculative-decoding iteration: verify -> accept -> rollback."""
import numpy as np
import pytest
import torch

import oracle
from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import make_inputs

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("streams, k, beta", [(32, 16, 3), (7, 5, 1), (65, 33, 40), (4, 1, 256), (3, 0, 2)])
def test_accept_matches_oracle(dtype, streams, k, beta):
    g = torch.Generator(device=DEV).manual_seed(streams * 100 + k)
    logits = torch.randn(streams, k, 256, device=DEV, generator=g).to(dtype)
    if k:
        # make acceptance likely for a while: draft the argmax, then random bytes
        drafted = logits.float().argmax(dim=2).to(torch.uint8)
        noise = torch.randint(0, 256, (streams, k), device=DEV, generator=g).to(torch.uint8)
        switch = torch.rand(streams, k, device=DEV, generator=g) < 0.2
        drafted = torch.where(switch, noise, drafted)
    else:
        drafted = torch.empty(streams, 0, dtype=torch.uint8, device=DEV)
    acc = mb.mb_accept_topk(logits, drafted, beta)
    want = oracle.accept_topk(logits, drafted, beta)
    assert np.array_equal(acc.cpu().numpy(), want)


def test_verify_accept_rollback_resumes_from_accepted_prefix():
    """One speculative iteration on device: the kept state equals the state after
    the accepted drafted bytes (oracle prefix scan)."""
    streams, k, Dn = 16, 12, 64
    inp = make_inputs(streams, k, Dn, 16, "bf16", "normal", seed=77, device=DEV)
    y = torch.empty_like(inp["x"])
    h_all = torch.empty(streams, k, Dn, 16, device=DEV)
    mb.mb_scan_verify(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, h_all, z=inp["z"],
                      D=inp["D"], dt_bias=inp["dt_bias"], h0=inp["h0"])
    g = torch.Generator(device=DEV).manual_seed(5)
    logits = torch.randn(streams, k, 256, device=DEV, generator=g)
    drafted = torch.where(torch.rand(streams, k, device=DEV, generator=g) < 0.25,
                          torch.randint(0, 256, (streams, k), device=DEV, generator=g),
                          logits.argmax(dim=2)).to(torch.uint8)
    accept = mb.mb_accept_topk(logits, drafted, 2)
    kept = torch.empty_like(inp["h0"])
    mb.mb_rollback(inp["h0"], h_all, accept, kept)
    acc = accept.cpu().numpy()
    assert np.array_equal(acc, oracle.accept_topk(logits, drafted, 2))
    _, _, rall = oracle.scan(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], z=inp["z"], D=inp["D"],
                             dt_bias=inp["dt_bias"], h0=inp["h0"], want_h_all=True)
    want = oracle.rollback(inp["h0"], rall, acc)
    got = kept.cpu().double().numpy()
    rms = np.sqrt(np.mean(want ** 2))
    assert np.max(np.abs(got - want) / np.maximum(np.abs(want), rms)) <= 2e-2
