"""Pins of the oracle's block functions (rmsnorm, conv1d_step, bf16_round, block_step)
against library routines and closed forms."""
import math

import numpy as np
import pytest

import oracle


def test_conv_steps_equal_the_causal_convolution():
    # Stepping the window from zeros over a sequence is the causal (zero
    # padded) convolution with the kernel reversed in time: np.convolve.
    r = np.random.default_rng(0)
    b, L, d = 2, 11, 5
    x = r.normal(size=(b, L, d))
    w = r.normal(size=(d, 4))
    bias = r.normal(size=d)
    state = np.zeros((b, 3, d))
    outs = []
    for t in range(L):
        o, state = oracle.conv1d_step(state, x[:, t], w, bias)
        outs.append(o)
    got = np.stack(outs, axis=1)
    want = np.empty_like(got)
    for bi in range(b):
        for di in range(d):
            full = np.convolve(x[bi, :, di], w[di, ::-1])[:L]
            want[bi, :, di] = oracle.silu(full + bias[di])
    assert np.allclose(got, want, rtol=1e-13, atol=1e-13)
    assert np.array_equal(state, x[:, -3:].transpose(0, 2, 1).transpose(0, 2, 1))


def test_silu_values():
    assert oracle.silu(0.0) == 0.0
    assert np.isclose(oracle.silu(1.0), 1.0 / (1.0 + np.exp(-1.0)), rtol=1e-15)


def test_rmsnorm_closed_forms():
    r = np.random.default_rng(1)
    x = r.normal(size=(3, 16))
    w = np.ones(16)
    res, out = oracle.rmsnorm(x, w, 0.0)
    assert np.array_equal(res, x)
    assert np.allclose(np.mean(out ** 2, axis=1), 1.0, rtol=1e-13)            # unit RMS
    _, out2 = oracle.rmsnorm(7.5 * x, w, 0.0)
    assert np.allclose(out, out2, rtol=1e-13)                                  # scale invariance
    c = np.full((1, 8), 3.0)
    _, oc = oracle.rmsnorm(c, 2 * np.ones(8), 1.0)
    assert np.allclose(oc, 2 * 3.0 / np.sqrt(9.0 + 1.0), rtol=1e-15)          # constant row
    add = r.normal(size=(3, 16))
    res3, _ = oracle.rmsnorm(x, w, 0.0, add)
    assert np.array_equal(res3, x + add)


@pytest.mark.parametrize("v, want", [(1.0, 1.0), (1.0078125, 1.0078125), (1.00390625, 1.0),
                                     (1.01171875, 1.015625), (1.001953125, 1.0), (1.005859375, 1.0078125),
                                     (-3.14159, -3.140625), (0.0, 0.0)])
def test_bf16_round_to_nearest_even(v, want):
    # bf16 keeps 8 significant bits (spacing 2^-7 at 1): 1 + 2^-7 is exact,
    # 1 + 2^-8 is a tie (to even: 1), 1 + 1.5 * 2^-7 is a tie (to even:
    # 1 + 2^-6), 1 + 0.75 * 2^-7 rounds up.
    assert oracle.bf16_round(np.array([v]))[0] == want


# ---------------------------------------------------------------------------
# The whole block step (Figure 6; Table 6 rows in order): a hand-worked layer.
#
# d_model 8, d_inner 8, d_state 2, dt_rank 1, with weights chosen so that
# every intermediate is a closed form of the inputs that the test writes out
# with index picks instead of matrix products:
#   rmsnorm:  eps 0 and residual + add = r with every |r_i| = 1, so rms(r) = 1
#             and the normalised row is r * norm_w;
#   W_in_x, W_in_z: cyclic shifts (x_i = h_{i+1}, z_i = 2 h_{i+3}); a
#             transposed product would shift the other way;
#   conv:     taps (1/4, 1/2, 3/4, 1), bias 1/10: xc = silu of the weighted
#             window;
#   W_dtlow, W_B, W_C: unit rows picking xc_1, (xc_2, xc_3), (xc_4, xc_5);
#   W_dt:     1/2 for every channel, so dt_d = xc_1 / 2;
#   A:        (-1, -2) in every channel, so by the discretisation appendix's
#             closed form exp(-softplus(v)) = 1 / (1 + e^v) the two decays are
#             s and s^2 with s = sigmoid(-v);
#   W_out:    a cyclic shift (out_i = g_{i+5}).
# ---------------------------------------------------------------------------
_NB = 8


def _shift(k, scale=1.0):
    """Matrix M with (M v)_i = scale * v_{(i + k) % 8}."""
    m = np.zeros((_NB, _NB))
    for i in range(_NB):
        m[i, (i + k) % _NB] = scale
    return m


def _unit_rows(*cols):
    m = np.zeros((len(cols), _NB))
    for r, c in enumerate(cols):
        m[r, c] = 1.0
    return m


def _hand_layer():
    return {
        "norm_w": np.arange(1, _NB + 1) / 4.0,
        "W_in_x": _shift(1), "W_in_z": _shift(3, 2.0),
        "conv_w": np.tile([0.25, 0.5, 0.75, 1.0], (_NB, 1)), "conv_b": np.full(_NB, 0.1),
        "W_dtlow": _unit_rows(1), "W_B": _unit_rows(2, 3), "W_C": _unit_rows(4, 5),
        "W_dt": np.full((_NB, 1), 0.5), "dt_bias": 0.1 * np.arange(_NB) - 0.3,
        "A": np.tile([-1.0, -2.0], (_NB, 1)), "D": np.full(_NB, 0.5),
        "W_out": _shift(5),
    }


def _hand_inputs(seed=7, batch=2):
    r = np.random.default_rng(seed)
    sign = np.where(r.random((batch, _NB)) < 0.5, -1.0, 1.0)
    add = np.round(r.normal(size=(batch, _NB)) * 8) / 8        # dyadic: residual + add is exact
    residual = sign - add
    ssm = r.normal(size=(batch, _NB, 2))
    conv = r.normal(size=(batch, 3, _NB))
    return sign, residual, add, ssm, conv


def _sig(v):
    return 1.0 / (1.0 + np.exp(-v))


def _hand_expected(sign, ssm, conv):
    """The block step worked out by hand for _hand_layer(), per batch row."""
    batch = sign.shape[0]
    out = np.empty((batch, _NB))
    ssm_new = np.empty_like(ssm)
    conv_new = np.empty_like(conv)
    bias = 0.1 * np.arange(_NB) - 0.3
    for b in range(batch):
        h = sign[b] * np.arange(1, _NB + 1) / 4.0
        x = np.array([h[(i + 1) % _NB] for i in range(_NB)])
        z = np.array([2.0 * h[(i + 3) % _NB] for i in range(_NB)])
        pre = 0.25 * conv[b, 0] + 0.5 * conv[b, 1] + 0.75 * conv[b, 2] + x + 0.1
        xc = pre * _sig(pre)
        g = np.empty(_NB)
        for d in range(_NB):
            v = 0.5 * xc[1] + bias[d]
            delta = math.log1p(math.exp(v))
            s = 1.0 / (1.0 + math.exp(v))                   # exp(-softplus(v))
            h0n = s * ssm[b, d, 0] + delta * xc[2] * xc[d]
            h1n = s * s * ssm[b, d, 1] + delta * xc[3] * xc[d]
            ssm_new[b, d] = (h0n, h1n)
            y = xc[4] * h0n + xc[5] * h1n + 0.5 * xc[d]
            g[d] = y * z[d] * _sig(z[d])
        out[b] = [g[(i + 5) % _NB] for i in range(_NB)]
        conv_new[b] = (conv[b, 1], conv[b, 2], x)
    return out, ssm_new, conv_new


def _block_err(fn):
    sign, residual, add, ssm, conv = _hand_inputs()
    r, out, ssm_new, conv_new = fn(_hand_layer(), residual, add, ssm, conv, eps=0.0, cast=lambda v: v)
    w_out, w_ssm, w_conv = _hand_expected(sign, ssm, conv)
    assert np.array_equal(r, sign)
    return max(float(np.max(np.abs(out - w_out))), float(np.max(np.abs(ssm_new - w_ssm))),
               float(np.max(np.abs(conv_new - w_conv))))


def test_block_step_hand_worked_layer():
    assert _block_err(oracle.block_step) < 1e-13


def _mutant(kind):
    """oracle.block_step with one planted wiring mistake."""
    def fn(layer, residual, add, ssm_state, conv_state, eps=1e-5, cast=oracle.bf16_round):
        r, h = oracle.rmsnorm(residual, layer["norm_w"], eps, add)
        x = cast(h @ layer["W_in_x"].T)
        z = cast(h @ layer["W_in_z"].T)
        if kind == "x_z_swapped":
            x, z = z, x
        if kind == "transposed_in_proj":
            x = cast(h @ layer["W_in_x"])
        xc, conv_state = oracle.conv1d_step(conv_state, x, layer["conv_w"], layer["conv_b"])
        xs = x if kind == "pre_conv_x_to_scan" else xc
        dtl = cast(xc @ (layer["W_B"][:1] if kind == "dt_low_from_B_rows" else layer["W_dtlow"]).T)
        Bm, Cm = cast(xc @ layer["W_B"].T), cast(xc @ layer["W_C"].T)
        if kind == "B_C_swapped":
            Bm, Cm = Cm, Bm
        dt = cast(dtl @ layer["W_dt"].T)
        zg = x if kind == "gate_with_x" else z
        y, ssm_state = oracle.step(ssm_state, x=xs, dt=dt, B=Bm, C=Cm, A=layer["A"], z=zg, D=layer["D"],
                                   dt_bias=layer["dt_bias"])
        out = cast(y @ layer["W_out"].T)
        if kind == "no_out_proj":
            out = cast(y)
        return r, out, ssm_state, conv_state
    return fn


@pytest.mark.parametrize("kind", ["none", "x_z_swapped", "transposed_in_proj", "pre_conv_x_to_scan",
                                  "dt_low_from_B_rows", "B_C_swapped", "gate_with_x", "no_out_proj"])
def test_block_step_pin_catches_wiring_mistakes(kind):
    # The unmutated copy passes the pin; every planted mistake fails it.
    err = _block_err(_mutant(kind))
    if kind == "none":
        assert err < 1e-13
    else:
        assert err > 1e-3, kind


def test_block_step_casts_where_the_gpu_keeps_bf16():
    # With bf16 rounding at the tensor boundaries the result moves by about
    # the bf16 spacing, never more than a few percent of the values here.
    sign, residual, add, ssm, conv = _hand_inputs(seed=9)
    _, out_c, ssm_c, _ = oracle.block_step(_hand_layer(), residual, add, ssm, conv, eps=0.0)
    w_out, w_ssm, _ = _hand_expected(sign, ssm, conv)
    assert np.max(np.abs(out_c - w_out)) <= 0.05 * np.max(np.abs(w_out))
    assert not np.array_equal(out_c, w_out)
    assert np.array_equal(oracle.bf16_round(out_c), out_c)      # out is a bf16 tensor
