"""Pins of the oracle's block functions (rmsnorm, conv1d_step, bf16_round)
against library routines and closed forms."""
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
