"""Pins for the fp64 oracle against what the paper and the mathematics fix.

None of these re-types the oracle's own loop. Each compares it with a
different route to the same number: the gated-RNN closed form of the
discretisation appendix, the Delta -> 0 limit stated there, linear state
growth when A = 0, the unrolled (non-recursive) solution of Eq. 2 written with
cumulative sums of Delta, and the associative operator of Section 2 folded in
random bracketings.
"""
import math

import numpy as np
import pytest

import oracle

RNG = np.random.default_rng(12345)


def _sig(v):
    return 1.0 / (1.0 + np.exp(-v))


def _rand_problem(batch, L, Dn, N, rng, a_scale=1.0):
    x = rng.standard_normal((batch, L, Dn))
    z = rng.standard_normal((batch, L, Dn))
    dt = rng.standard_normal((batch, L, Dn))
    B = rng.standard_normal((batch, L, N))
    C = rng.standard_normal((batch, L, N))
    A = -a_scale * rng.uniform(0.2, 3.0, (Dn, N))       # distinct per (d, n)
    D = rng.standard_normal(Dn)
    bias = rng.uniform(-3.0, 0.5, Dn)
    h0 = 0.3 * rng.standard_normal((batch, Dn, N))
    return dict(x=x, z=z, dt=dt, B=B, C=C, A=A, D=D, dt_bias=bias, h0=h0)


def _unrolled(p, b_rule=oracle.B_EULER):
    """Non-recursive solution of Eq. 2: h_t = exp(A S_t) h0 + sum_{s<=t}
    exp(A (S_t - S_s)) Bbar_s x_s, with S_t the running sum of Delta.
    Products of exp(Delta A) are taken as the exponential of a sum."""
    x, z, dt, B, C, A = p["x"], p["z"], p["dt"], p["B"], p["C"], p["A"]
    batch, L, Dn = x.shape
    N = A.shape[1]
    delta = np.logaddexp(0.0, dt + p["dt_bias"][None, None, :])   # softplus
    S = np.cumsum(delta, axis=1)                                    # [b, L, D]
    h_all = np.zeros((batch, L, Dn, N))
    for b in range(batch):
        for t in range(L):
            # [D, N]
            h = np.exp(A * S[b, t][:, None]) * (p["h0"][b] if p["h0"] is not None else 0.0)
            for s in range(t + 1):
                decay = np.exp(A * (S[b, t] - S[b, s])[:, None])
                if b_rule == oracle.B_EULER:
                    bbar = delta[b, s][:, None] * B[b, s][None, :]
                else:
                    bbar = np.expm1(A * delta[b, s][:, None]) / A * B[b, s][None, :]
                h = h + decay * bbar * x[b, s][:, None]
            h_all[b, t] = h
    yssm = np.einsum("btdn,btn->btd", h_all, C) + p["D"][None, None, :] * x
    y = yssm * z * _sig(z) if z is not None else yssm
    return y, h_all


@pytest.mark.parametrize("b_rule", [oracle.B_EULER, oracle.B_ZOH])
def test_unrolled_solution(b_rule):
    p = _rand_problem(2, 13, 3, 5, RNG)
    y, h_last, h_all = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], z=p["z"], D=p["D"],
                                   dt_bias=p["dt_bias"], h0=p["h0"], b_rule=b_rule,
                                   want_h_all=True)
    y_ref, h_ref = _unrolled(p, b_rule)
    np.testing.assert_allclose(h_all, h_ref, rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(h_last, h_ref[:, -1], rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(y, y_ref, rtol=1e-11, atol=1e-13)


def test_unrolled_solution_no_gate_no_h0():
    p = _rand_problem(1, 9, 4, 3, RNG)
    p["z"], p["h0"] = None, None
    y, h_last, _ = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], D=p["D"],
                               dt_bias=p["dt_bias"])
    y_ref, h_ref = _unrolled(p)
    np.testing.assert_allclose(y, y_ref, rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(h_last, h_ref[:, -1], rtol=1e-11, atol=1e-13)


def _gated_rnn_inputs(L, rng):
    v = rng.uniform(-6, 6, L)
    x = rng.standard_normal(L)
    h0 = rng.standard_normal()
    one = np.ones((1, L, 1))
    return v, x, h0, dict(x=x.reshape(1, L, 1), dt=v.reshape(1, L, 1), B=one, C=one,
                          A=np.array([[-1.0]]), h0=np.array([[[h0]]]))


def test_gated_rnn_zoh():
    """Discretisation appendix: A=-1, B=1, n=1 with ZOH gives
    Abar = 1 - sigmoid(v), Bbar = sigmoid(v): h = (1 - s) h + s x."""
    v, x, h0, p = _gated_rnn_inputs(40, RNG)
    y, h_last, h_all = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], h0=p["h0"],
                                   b_rule=oracle.B_ZOH, want_h_all=True)
    h, ref = h0, []
    for t in range(len(v)):
        s = 1.0 / (1.0 + math.exp(-v[t]))
        h = (1.0 - s) * h + s * x[t]
        ref.append(h)
    np.testing.assert_allclose(h_all[0, :, 0, 0], ref, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(y[0, :, 0], ref, rtol=1e-12, atol=1e-14)  # C=1, D=0, no gate


def test_gated_rnn_euler():
    """Same system with Mamba's Euler rule for B: Abar = 1/(1+e^v) = sigmoid(-v),
    Bbar = Delta = log(1+e^v)."""
    v, x, h0, p = _gated_rnn_inputs(40, RNG)
    y, _, h_all = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], h0=p["h0"],
                              want_h_all=True)
    h, ref = h0, []
    for t in range(len(v)):
        h = h / (1.0 + math.exp(v[t])) + math.log(1.0 + math.exp(v[t])) * x[t]
        ref.append(h)
    np.testing.assert_allclose(h_all[0, :, 0, 0], ref, rtol=1e-12, atol=1e-14)


def test_delta_to_zero_keeps_state():
    """Delta -> 0 ignores the input and keeps h (limit stated in the appendix):
    y_t = (C_t . h0 + D x_t) silu(z_t)."""
    p = _rand_problem(2, 7, 3, 4, RNG)
    p["dt"][:] = -60.0                 # softplus(-60) ~ 8.8e-27
    p["dt_bias"][:] = 0.0
    y, h_last, h_all = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], z=p["z"], D=p["D"],
                                   dt_bias=p["dt_bias"], h0=p["h0"], want_h_all=True)
    np.testing.assert_allclose(h_last, p["h0"], rtol=1e-20, atol=1e-24)
    ref = (np.einsum("bdn,btn->btd", p["h0"], p["C"]) + p["D"] * p["x"]) * p["z"] * _sig(p["z"])
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-14)


def test_a_zero_linear_growth():
    """A = 0 and constant inputs: Abar = 1, so h_t = h0 + t Delta B x (t = 1..L)
    and y_t = C . h_t + D x (Eq. 2 uses the updated state)."""
    L, Dn, N = 11, 3, 4
    rng = np.random.default_rng(7)
    xv, zv, dtv = rng.standard_normal(Dn), rng.standard_normal(Dn), rng.standard_normal(Dn)
    Bv, Cv = rng.standard_normal(N), rng.standard_normal(N)
    h0 = rng.standard_normal((1, Dn, N))
    Dk = rng.standard_normal(Dn)
    x = np.broadcast_to(xv, (1, L, Dn)).copy()
    z = np.broadcast_to(zv, (1, L, Dn)).copy()
    dt = np.broadcast_to(dtv, (1, L, Dn)).copy()
    B = np.broadcast_to(Bv, (1, L, N)).copy()
    C = np.broadcast_to(Cv, (1, L, N)).copy()
    y, h_last, h_all = oracle.scan(x, dt, B, C, np.zeros((Dn, N)), z=z, D=Dk, h0=h0,
                                   want_h_all=True)
    delta = np.logaddexp(0.0, dtv)
    t = np.arange(1, L + 1)[:, None, None]
    h_ref = h0[0][None] + t * (delta * xv)[None, :, None] * Bv[None, None, :]
    np.testing.assert_allclose(h_all[0], h_ref, rtol=1e-12, atol=1e-13)
    y_ref = (h_ref @ Cv + Dk * xv) * zv * _sig(zv)
    np.testing.assert_allclose(y[0], y_ref, rtol=1e-12, atol=1e-13)


def test_paper_operator_random_bracketing():
    """Section 2: e_k = (Abar_k, Bbar_k x_k) and e_j . e_k = (A_k A_j, A_k b_j + b_k)
    is associative; any bracketing of e_1 .. e_t applied to h0 gives h_t."""
    rng = np.random.default_rng(99)
    p = _rand_problem(1, 17, 2, 3, rng)
    _, _, h_all = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], z=p["z"], D=p["D"],
                              dt_bias=p["dt_bias"], h0=p["h0"], want_h_all=True)
    delta = np.logaddexp(0.0, p["dt"][0] + p["dt_bias"])             # [L, D]
    Ab = np.exp(delta[:, :, None] * p["A"][None])                      # [L, D, N]
    bb = delta[:, :, None] * p["B"][0][:, None, :] * p["x"][0][:, :, None]

    def op(ej, ek):
        return ek[0] * ej[0], ek[0] * ej[1] + ek[1]

    def fold(lo, hi):  # random split of [lo, hi)
        if hi - lo == 1:
            return Ab[lo], bb[lo]
        mid = int(rng.integers(lo + 1, hi))
        return op(fold(lo, mid), fold(mid, hi))

    for t in range(1, 18):
        Atot, btot = fold(0, t)
        np.testing.assert_allclose(Atot * p["h0"][0] + btot, h_all[0, t - 1], rtol=1e-11,
                                   atol=1e-13)


@pytest.mark.parametrize("split", [1, 5, 16, 31])
def test_split_scan_equals_one_scan(split):
    p = _rand_problem(2, 32, 3, 4, RNG)
    kw = dict(z=p["z"], D=p["D"], dt_bias=p["dt_bias"])
    y, h, _ = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], h0=p["h0"], **kw)
    sl1, sl2 = slice(0, split), slice(split, None)
    y1, h1, _ = oracle.scan(p["x"][:, sl1], p["dt"][:, sl1], p["B"][:, sl1], p["C"][:, sl1],
                            p["A"], h0=p["h0"], z=p["z"][:, sl1], D=p["D"], dt_bias=p["dt_bias"])
    y2, h2, _ = oracle.scan(p["x"][:, sl2], p["dt"][:, sl2], p["B"][:, sl2], p["C"][:, sl2],
                            p["A"], h0=h1, z=p["z"][:, sl2], D=p["D"], dt_bias=p["dt_bias"])
    np.testing.assert_allclose(np.concatenate([y1, y2], axis=1), y, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(h2, h, rtol=1e-13, atol=1e-15)


def test_steps_equal_one_scan():
    p = _rand_problem(3, 9, 4, 4, RNG)
    y, h, _ = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], z=p["z"], D=p["D"],
                          dt_bias=p["dt_bias"], h0=p["h0"])
    state = p["h0"].copy()
    for t in range(9):
        yt, state = oracle.step(state, p["x"][:, t], p["dt"][:, t], p["B"][:, t], p["C"][:, t],
                                p["A"], z=p["z"][:, t], D=p["D"], dt_bias=p["dt_bias"])
        np.testing.assert_allclose(yt, y[:, t], rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(state, h, rtol=1e-13, atol=1e-15)


def test_rollback_is_prefix_state():
    """Algorithm 1: after accepting a drafted bytes the verifier resumes from
    the state after those a bytes (h0 when a = 0)."""
    p = _rand_problem(5, 6, 3, 4, RNG)
    _, _, h_all = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], z=p["z"], D=p["D"],
                              dt_bias=p["dt_bias"], h0=p["h0"], want_h_all=True)
    _, h_ref = _unrolled(p)
    accept = np.array([0, 6, 3, 1, 5], dtype=np.int32)
    out = oracle.rollback(p["h0"], h_all, accept)
    for s, a in enumerate(accept):
        want = p["h0"][s] if a == 0 else h_ref[s, a - 1]
        np.testing.assert_allclose(out[s], want, rtol=1e-11, atol=1e-13)
    with pytest.raises(RuntimeError):
        oracle.rollback(p["h0"], h_all, np.array([0, 7, 0, 0, 0], dtype=np.int32))


def test_gate_and_skip_values():
    """C = 0 leaves y = D x silu(z); silu(1) = 1/(1 + 1/e), silu(0) = 0."""
    L, Dn, N = 3, 2, 4
    x = np.ones((1, L, Dn))
    z = np.array([[[1.0, 0.0], [-40.0, 40.0], [2.0, -1.0]]])
    D = np.array([1.0, 0.5])
    zeros = np.zeros((1, L, N))
    y, _, _ = oracle.scan(x, np.zeros((1, L, Dn)), zeros, zeros, -np.ones((Dn, N)), z=z, D=D)
    s1 = 1.0 / (1.0 + math.exp(-1.0))
    assert abs(y[0, 0, 0] - 0.7310585786300049) < 1e-15 and y[0, 0, 1] == 0.0
    assert abs(y[0, 1, 0] - (-40.0 / (1.0 + math.exp(40.0)))) < 1e-30
    assert abs(y[0, 1, 1] - 0.5 * 40.0) < 1e-12
    assert abs(y[0, 2, 0] - 2.0 / (1.0 + math.exp(-2.0))) < 1e-15
    assert abs(y[0, 2, 1] - 0.5 * (-1.0) * (1.0 - s1)) < 1e-15


def test_length_one_and_empty():
    p = _rand_problem(2, 1, 3, 4, RNG)
    y, h, _ = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], z=p["z"], D=p["D"],
                          dt_bias=p["dt_bias"], h0=p["h0"])
    delta = np.logaddexp(0.0, p["dt"][:, 0] + p["dt_bias"])          # [b, D]
    h1 = (np.exp(delta[:, :, None] * p["A"][None]) * p["h0"]
          + delta[:, :, None] * p["B"][:, 0][:, None, :] * p["x"][:, 0][:, :, None])
    np.testing.assert_allclose(h, h1, rtol=1e-13)
    # L = 0: nothing to scan, the state passes through unchanged.
    e = np.zeros((2, 0, 3))
    y0, h0out, _ = oracle.scan(e, e, np.zeros((2, 0, 4)), np.zeros((2, 0, 4)), p["A"],
                               h0=p["h0"])
    assert y0.shape == (2, 0, 3)
    np.testing.assert_array_equal(h0out, p["h0"])


def test_threads_do_not_change_results():
    p = _rand_problem(3, 50, 17, 16, RNG)
    kw = dict(z=p["z"], D=p["D"], dt_bias=p["dt_bias"], h0=p["h0"], want_h_all=True)
    r1 = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], nthreads=1, **kw)
    r4 = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], nthreads=4, **kw)
    for a, b in zip(r1, r4):
        np.testing.assert_array_equal(a, b)


def test_golden_fixture_and_hand_value():
    """tests/golden/tiny_scan.json holds oracle outputs on hand-written inputs
    (written by tests/golden/make_golden.py); its first output is also worked
    out here by hand, one operation at a time, from Eq. 2-3 and Table 6."""
    import json
    import os
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "tiny_scan.json")))
    a = {k: np.array(v, dtype=np.float64) for k, v in g["inputs"].items() if k != "accept"}
    y, h_last, h_all = oracle.scan(a["x"], a["dt"], a["B"], a["C"], a["A"], z=a["z"], D=a["D"],
                                   dt_bias=a["dt_bias"], h0=a["h0"], want_h_all=True)
    np.testing.assert_allclose(y, g["y"], rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(h_last, g["h_last"], rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(h_all, g["h_all"], rtol=1e-14, atol=1e-15)
    kept = oracle.rollback(a["h0"], h_all, np.array(g["inputs"]["accept"], dtype=np.int32))
    np.testing.assert_allclose(kept, g["rollback"], rtol=1e-14, atol=1e-15)
    # b = 0, t = 0, d = 0 by hand: dt + bias = -1, Delta = log(1 + e^-1).
    delta = math.log(1.0 + math.exp(-1.0))
    h_a = math.exp(-1.0 * delta) * 0.1 + delta * 1.0 * 0.5      # A=-1, B=1,    x=0.5
    h_b = math.exp(-2.0 * delta) * -0.2 + delta * -0.5 * 0.5    # A=-2, B=-0.5
    yssm = 0.5 * h_a + 1.0 * h_b + 1.0 * 0.5                    # C=(0.5, 1), D=1
    want = yssm * 1.0 / (1.0 + math.exp(-1.0))                  # z=1
    assert abs(g["y"][0][0][0] - want) < 1e-15
    assert abs(want - 0.3141092605981670) < 1e-15


# ---------------------------------------------------------------- Delta projection (Eq. 3)
def test_delta_projection_brute_force():
    """dt[b,t,d] = sum_k dt_low[b,t,k] W_dt[d,k], summed here term by term in
    plain Python on a tiny problem."""
    rng = np.random.default_rng(7)
    dl = rng.standard_normal((2, 3, 5))
    w = rng.standard_normal((4, 5))
    got = oracle.delta_projection(dl, w)
    assert got.shape == (2, 3, 4)
    for b in range(2):
        for t in range(3):
            for d in range(4):
                want = 0.0
                for k in range(5):
                    want += float(dl[b, t, k]) * float(w[d, k])
                assert abs(got[b, t, d] - want) <= 1e-12 * (1 + abs(want))


def test_delta_projection_selects_columns_and_is_linear():
    """One-hot rows of W_Delta pick single columns of W_R x exactly (a
    transposed operand would pick rows instead), and the map is linear in W."""
    rng = np.random.default_rng(8)
    dl = rng.standard_normal((3, 4, 6))
    pick = np.array([5, 0, 3, 3, 1, 2, 4])
    w = np.zeros((7, 6))
    w[np.arange(7), pick] = 1.0
    assert np.array_equal(oracle.delta_projection(dl, w), dl[:, :, pick])
    w1, w2 = rng.standard_normal((7, 6)), rng.standard_normal((7, 6))
    np.testing.assert_allclose(oracle.delta_projection(dl, 2.0 * w1 - w2),
                               2.0 * oracle.delta_projection(dl, w1) - oracle.delta_projection(dl, w2),
                               rtol=1e-12, atol=1e-12)


def test_scan_with_projected_delta_gated_rnn():
    """Through the scan: with N = 1, A = -1, B = C = 1, D = 0 and no gate, the
    recurrence is h_t = sigmoid(-v_t) h_{t-1} + softplus(v_t) x_t (the gated-RNN
    reading of the discretisation appendix) with v_t = dt_low[t] . W_dt[d]."""
    rng = np.random.default_rng(9)
    L, Dn, r = 12, 3, 4
    dl = rng.standard_normal((1, L, r))
    w = rng.standard_normal((Dn, r)) / 2.0
    x = rng.standard_normal((1, L, Dn))
    ones = np.ones((1, L, 1))
    y, hl, _ = oracle.scan(x, oracle.delta_projection(dl, w), ones, ones, -np.ones((Dn, 1)))
    for d in range(Dn):
        h = 0.0
        for t in range(L):
            v = float(dl[0, t] @ w[d])
            h = _sig(-v) * h + math.log1p(math.exp(v)) * x[0, t, d]
            assert abs(y[0, t, d] - h) <= 1e-12 * (1 + abs(h))
        assert abs(hl[0, d, 0] - h) <= 1e-12 * (1 + abs(h))
