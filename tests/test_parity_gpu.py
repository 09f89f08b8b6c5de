"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on
the same seeded inputs, plus invariants that hold at any size.

Error metric and bars (tests/_parity.py): err = max |g - r| / max(|r|, rms(r))
per output tensor, <= 1e-4 for fp32 inputs and <= 2e-2 for bf16 inputs, with
the state carried in fp32 on the GPU. Index work (rollback) is bit-exact.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2401_13660_gb300 import mbscan as mb
from paper_2401_13660_gb300.inputs import WORKLOADS, make_inputs, torch_dtype, workload_inputs

from _parity import TOL, TOL_STATE, oracle_channels, oracle_scan, rel_err, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _prefill(inp, h_last=True):
    x = inp["x"]
    y = torch.empty_like(x)
    hl = torch.empty(x.shape[0], x.shape[2], 16, device=x.device) if h_last else None
    mb.mb_scan_prefill(x, inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp.get("z"),
                       D=inp.get("D"), dt_bias=inp.get("dt_bias"), h0=inp.get("h0"), h_last=hl)
    return y, hl


def _verify(inp):
    x = inp["x"]
    y = torch.empty_like(x)
    h_all = torch.empty(x.shape[0], x.shape[1], x.shape[2], 16, device=x.device)
    mb.mb_scan_verify(x, inp["dt"], inp["B"], inp["C"], inp["A"], y, h_all, z=inp.get("z"),
                      D=inp.get("D"), dt_bias=inp.get("dt_bias"), h0=inp.get("h0"))
    return y, h_all


def _step(inp, state, t):
    sl = slice(t, t + 1)
    x = inp["x"][:, sl].contiguous()
    y = torch.empty_like(x)
    z = inp["z"][:, sl].contiguous() if inp.get("z") is not None else None
    mb.mb_step(x, inp["dt"][:, sl].contiguous(), inp["B"][:, sl].contiguous(),
               inp["C"][:, sl].contiguous(), inp["A"], y, state, z=z, D=inp.get("D"),
               dt_bias=inp.get("dt_bias"))
    return y


# ------------------------------------------------------------------ prefill
def test_prefill_tiny_fp32_full():
    w = WORKLOADS["tiny_f32_b1_L256_D64"]
    inp = workload_inputs(w, DEV)
    y, hl = _prefill(inp)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["f32"]
    assert rel_err(hl, rh) <= TOL_STATE["f32"]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("shape", [(3, 37, 40), (2, 16, 32), (1, 1, 8), (2, 100, 72), (1, 333, 128)])
@pytest.mark.parametrize("h0", ["zeros", "normal"])
def test_prefill_ragged(dtype, shape, h0):
    b, L, Dn = shape
    inp = make_inputs(b, L, Dn, 16, dtype, h0, seed=11 + L + Dn, device=DEV)
    y, hl = _prefill(inp)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL[dtype]
    assert rel_err(hl, rh) <= TOL_STATE["f32" if dtype == "f32" else "bf16"]


def test_prefill_optional_operands_absent():
    inp = make_inputs(2, 50, 48, 16, "f32", "zeros", seed=5, device=DEV, gate=False)
    inp["D"] = None
    inp["dt_bias"] = None
    y, hl = _prefill(inp)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["f32"] and rel_err(hl, rh) <= TOL_STATE["f32"]
    y2, _ = _prefill(inp, h_last=False)
    torch.testing.assert_close(y2, y, rtol=0, atol=0)


def test_prefill_empty_sequence_passes_state():
    inp = make_inputs(2, 0, 32, 16, "bf16", "normal", seed=3, device=DEV)
    y, hl = _prefill(inp)
    assert y.numel() == 0
    torch.testing.assert_close(hl, inp["h0"], rtol=0, atol=0)


def test_prefill_h_last_in_place_over_h0():
    inp = make_inputs(2, 40, 64, 16, "f32", "normal", seed=9, device=DEV)
    _, rh, _ = oracle_scan(inp)
    h = inp["h0"].clone()
    y = torch.empty_like(inp["x"])
    mb.mb_scan_prefill(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, z=inp["z"],
                       D=inp["D"], dt_bias=inp["dt_bias"], h0=h, h_last=h)
    assert rel_err(h, rh) <= TOL_STATE["f32"]


@pytest.mark.parametrize("name", ["mambabyte353m_prefill_b8_L8192", "mambabyte972m_prefill_b4_L8192"])
def test_prefill_full_size_sampled(name):
    """Full-size launch (as timed in bench.py); 64 sampled channels x 2 rows
    over the whole 8192-byte span checked against the oracle."""
    w = WORKLOADS[name]
    inp = workload_inputs(w, DEV)
    y, hl = _prefill(inp)
    assert torch.isfinite(y.float()).all() and torch.isfinite(hl).all()
    g = torch.Generator().manual_seed(7)
    rows = sorted(torch.randperm(w.batch, generator=g)[:2].tolist())
    chans = sorted(torch.randperm(w.d_inner, generator=g)[:64].tolist())
    # always include the first and last channel tiles
    chans = sorted(set(chans) | {0, w.d_inner - 1})
    ry, rh, _ = oracle_channels(inp, rows, chans)
    r_t, c_t = torch.tensor(rows, device=DEV), torch.tensor(chans, device=DEV)
    gy = y.index_select(0, r_t)[:, :, c_t]
    gh = hl.index_select(0, r_t)[:, c_t]
    assert rel_err(gy, ry) <= TOL["bf16"]
    assert rel_err(gh, rh) <= TOL_STATE["bf16"]


def test_prefill_split_equals_one_scan():
    """Associativity (Section 2): scanning [0, L1) then [L1, L) from the carried
    state equals one scan over [0, L)."""
    inp = make_inputs(2, 300, 64, 16, "f32", "normal", seed=21, device=DEV)
    y, hl = _prefill(inp)
    L1 = 129
    a = {k: (v[:, :L1].contiguous() if k in ("x", "z", "dt", "B", "C") else v) for k, v in inp.items()}
    y1, h1 = _prefill(a)
    b = {k: (v[:, L1:].contiguous() if k in ("x", "z", "dt", "B", "C") else v) for k, v in inp.items()}
    b["h0"] = h1
    y2, h2 = _prefill(b)
    torch.testing.assert_close(torch.cat([y1, y2], 1), y, rtol=2e-5, atol=2e-5)
    torch.testing.assert_close(h2, hl, rtol=2e-5, atol=2e-5)


def test_prefill_delta_to_zero_keeps_state():
    inp = make_inputs(2, 64, 32, 16, "f32", "normal", seed=4, device=DEV)
    inp["dt"].fill_(-60.0)
    inp["dt_bias"].zero_()
    y, hl = _prefill(inp)
    torch.testing.assert_close(hl, inp["h0"], rtol=0, atol=0)
    ry, _, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["f32"]


def test_prefill_a_zero_linear_growth():
    b, L, Dn = 1, 64, 32
    inp = make_inputs(b, 1, Dn, 16, "f32", "normal", seed=8, device=DEV)
    rep = {k: inp[k].expand(b, L, -1).contiguous() for k in ("x", "z", "dt", "B", "C")}
    inp.update(rep)
    inp["A"] = torch.zeros_like(inp["A"])
    _, hl = _prefill(inp)
    delta = torch.nn.functional.softplus((inp["dt"][0, 0] + inp["dt_bias"]).double())
    want = inp["h0"][0].double() + L * (delta * inp["x"][0, 0].double())[:, None] * inp["B"][0, 0].double()[None]
    assert rel_err(hl[0], want.cpu().numpy()) <= TOL_STATE["f32"]


# ------------------------------------------------------------------ verify + rollback
def test_verify_full_size_against_oracle():
    w = WORKLOADS["verify_s32_k16_D2048"]
    inp = workload_inputs(w, DEV)
    y, h_all = _verify(inp)
    ry, rh, rall = oracle_scan(inp, want_h_all=True)
    assert rel_err(y, ry) <= TOL["bf16"]
    assert rel_err(h_all, rall) <= TOL_STATE["bf16"]
    # rollback at the seeded accept counts: an index gather, bit-exact
    h_out = torch.empty_like(inp["h0"])
    mb.mb_rollback(inp["h0"], h_all, inp["accept"], h_out)
    acc = inp["accept"].long()
    want = torch.where((acc == 0)[:, None, None], inp["h0"],
                       h_all[torch.arange(w.batch, device=DEV), (acc - 1).clamp(min=0)])
    assert torch.equal(h_out, want)
    ro = oracle.rollback(to_np(inp["h0"]), rall, to_np(inp["accept"]).astype(np.int32))
    assert rel_err(h_out, ro) <= TOL_STATE["bf16"]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_verify_matches_prefill_and_oracle_small(dtype):
    inp = make_inputs(5, 23, 40, 16, dtype, "normal", seed=31, device=DEV)
    y, h_all = _verify(inp)
    ry, _, rall = oracle_scan(inp, want_h_all=True)
    assert rel_err(y, ry) <= TOL[dtype] and rel_err(h_all, rall) <= TOL_STATE[dtype]
    yp, hl = _prefill(inp)
    if dtype == "f32":
        torch.testing.assert_close(y, yp, rtol=1e-5, atol=1e-5)
    torch.testing.assert_close(h_all[:, -1], hl, rtol=1e-5, atol=1e-6)


@pytest.mark.parametrize("dtype,L", [("bf16", 5), ("f32", 16), ("bf16", 1)])
def test_verify_single_chunk_ragged_stays_in_bounds(dtype, L):
    """Spans of at most one chunk stream every per-position state from the
    lanes' registers to h_all: positions past L and channels past d_inner
    (536 = 16 full 32-channel tiles + 24) must be skipped,
    so a sentinel tail after h_all stays untouched and every stream's rows
    match the oracle."""
    b, D = 3, 8 * 67
    inp = make_inputs(b, L, D, 16, dtype, "normal", seed=33, device=DEV)
    n = b * L * D * 16
    big = torch.full((n + 8192,), float("nan"), device=DEV)
    h_all = big[:n].view(b, L, D, 16)
    y = torch.empty_like(inp["x"])
    mb.mb_scan_verify(inp["x"], inp["dt"], inp["B"], inp["C"], inp["A"], y, h_all, z=inp.get("z"),
                      D=inp.get("D"), dt_bias=inp.get("dt_bias"), h0=inp.get("h0"))
    ry, _, rall = oracle_scan(inp, want_h_all=True)
    assert torch.isnan(big[n:]).all()
    assert rel_err(y, ry) <= TOL[dtype] and rel_err(h_all, rall) <= TOL_STATE[dtype]


def test_rollback_edges_and_alias():
    inp = make_inputs(6, 16, 32, 16, "f32", "normal", seed=41, device=DEV)
    _, h_all = _verify(inp)
    accept = torch.tensor([0, 16, 1, 8, 0, 15], dtype=torch.int32, device=DEV)
    h = inp["h0"].clone()
    mb.mb_rollback(h, h_all, accept, h)          # h_out aliases h0
    for s, a in enumerate(accept.tolist()):
        want = inp["h0"][s] if a == 0 else h_all[s, a - 1]
        assert torch.equal(h[s], want)
    # h0 = NULL means zeros for accept == 0
    out = torch.full_like(h, 7.0)
    mb.mb_rollback(None, h_all, accept, out)
    assert torch.equal(out[0], torch.zeros_like(out[0]))


def test_rollback_out_of_range_is_reported_not_faulted():
    inp = make_inputs(4, 8, 32, 16, "f32", "normal", seed=42, device=DEV)
    _, h_all = _verify(inp)
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    accept = torch.tensor([1, 2, 9, 0], dtype=torch.int32, device=DEV)   # 9 > k = 8
    out = torch.full_like(inp["h0"], 3.0)
    mb.mb_rollback(inp["h0"], h_all, accept, out, ws=ws)
    st, detail = mb.mb_check(ws)
    assert st == mb.MB_ERR_INVALID_ARG and detail == 2
    assert torch.equal(out[2], torch.full_like(out[2], 3.0))          # untouched
    assert torch.equal(out[0], h_all[0, 0])
    assert mb.mb_check(ws) == (mb.MB_OK, -1)                           # cleared


# ------------------------------------------------------------------ decode step
def test_step_full_size_one_layer():
    w = WORKLOADS["step_b256_D4608_x48"]
    inp = workload_inputs(w, DEV)
    state = inp["h0"].clone()
    y = _step(inp, state, 0)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["bf16"]
    assert rel_err(state, rh) <= TOL_STATE["bf16"]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_steps_equal_one_scan(dtype):
    """N single-byte steps equal one N-length scan (y and final state)."""
    inp = make_inputs(3, 12, 40, 16, dtype, "normal", seed=51, device=DEV)
    ry, rh, _ = oracle_scan(inp)
    state = inp["h0"].clone()
    ys = [_step(inp, state, t) for t in range(12)]
    assert rel_err(torch.cat(ys, 1), ry) <= TOL[dtype]
    assert rel_err(state, rh) <= TOL_STATE[dtype]
    _, hl = _prefill(inp)
    torch.testing.assert_close(state, hl, rtol=1e-5, atol=1e-6)


def test_step_ragged_channel_count():
    inp = make_inputs(3, 1, 8 * 67, 16, "bf16", "normal", seed=52, device=DEV)
    state = inp["h0"].clone()
    y = _step(inp, state, 0)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y, ry) <= TOL["bf16"] and rel_err(state, rh) <= TOL_STATE["bf16"]


def test_step_rows_independent_of_the_launch_shape():
    """The same rows stepped within grids of different shapes are bit-identical:
    256 rows x 2048 channels (512 tiles: a persistent grid at the resident
    limit), their first 32 rows (256 tiles: one wave spread at 2 CTAs per SM)
    and first 4 rows (32 tiles: 1 CTA per SM). Checked against the oracle too."""
    inp = make_inputs(256, 1, 2048, 16, "bf16", "normal", seed=53, device=DEV)
    outs = {}
    for rows in (256, 32, 4):
        sub = {k: (v[:rows].contiguous() if torch.is_tensor(v) and v.shape[0] == 256 else v) for k, v in inp.items()}
        state = sub["h0"].clone()
        outs[rows] = (_step(sub, state, 0), state)
    for rows in (32, 4):
        assert torch.equal(outs[rows][0], outs[256][0][:rows])
        assert torch.equal(outs[rows][1], outs[256][1][:rows])
    small = {k: (v[:4].contiguous() if torch.is_tensor(v) and v.shape[0] == 256 else v) for k, v in inp.items()}
    ry, rh, _ = oracle_scan(small)
    assert rel_err(outs[4][0], ry) <= TOL["bf16"] and rel_err(outs[4][1], rh) <= TOL_STATE["bf16"]


@pytest.mark.parametrize("rows", [256, 32, 4])
def test_back_to_back_steps_on_one_state(rows):
    """Consecutive mb_step launches on the same state with nothing in between:
    each step kernel may start (and prefetch its first tiles' state into L2)
    while the previous one still writes that state. 16 steps launched back to
    back, eagerly and from a CUDA graph, must equal bit for bit the same steps
    with a device synchronisation after each, and the oracle's 16-step scan.
    256 rows x 2048 channels fill the resident CTA slots; 32 and 4 rows leave
    slots free, so consecutive grids can be resident together."""
    L = 16
    inp = make_inputs(rows, L, 2048, 16, "bf16", "normal", seed=54 + rows, device=DEV)
    sl = lambda k, t: inp[k][:, t:t + 1].contiguous()
    steps = [dict(x=sl("x", t), dt=sl("dt", t), B=sl("B", t), C=sl("C", t), z=sl("z", t)) for t in range(L)]
    ys = [torch.empty_like(s["x"]) for s in steps]

    def run(state, sync):
        for s, y in zip(steps, ys):
            mb.mb_step(s["x"], s["dt"], s["B"], s["C"], inp["A"], y, state, z=s["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"])
            if sync:
                torch.cuda.synchronize()
        return torch.cat(ys, 1).clone()

    st_sync = inp["h0"].clone()
    y_sync = run(st_sync, True)
    st_eager = inp["h0"].clone()
    y_eager = run(st_eager, False)
    torch.cuda.synchronize()
    st_graph = inp["h0"].clone()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        run(inp["h0"].clone(), False)   # warm-up outside the capture
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for s, y in zip(steps, ys):
            mb.mb_step(s["x"], s["dt"], s["B"], s["C"], inp["A"], y, st_graph, z=s["z"], D=inp["D"],
                       dt_bias=inp["dt_bias"])
    g.replay()
    torch.cuda.synchronize()
    y_graph = torch.cat(ys, 1).clone()
    assert torch.equal(y_eager, y_sync) and torch.equal(st_eager, st_sync)
    assert torch.equal(y_graph, y_sync) and torch.equal(st_graph, st_sync)
    ry, rh, _ = oracle_scan(inp)
    assert rel_err(y_sync, ry) <= TOL["bf16"] and rel_err(st_sync, rh) <= TOL_STATE["bf16"]
