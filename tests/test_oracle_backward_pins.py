"""Pins of the fp64 backward oracle (oracle.scan_backward) against things other
than itself: the forward oracle (already pinned) through central finite
differences on tiny problems, and exact adjoint identities where the
objective is linear in an input.

Objective: J = sum(dout * out) + sum(dh_last * h_last), out and h_last from
the forward layer core (MambaByte Eq. 2-3, Table 6 output and gating).
"""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.filterwarnings("ignore")


def _problem(seed, batch=2, L=6, Dn=3, N=4, gate=True, h0=True, dh_last=True):
    r = np.random.default_rng(seed)
    p = dict(x=r.normal(size=(batch, L, Dn)), dt=r.normal(size=(batch, L, Dn)),
             B=r.normal(size=(batch, L, N)), C=r.normal(size=(batch, L, N)),
             A=-r.uniform(0.2, 2.0, size=(Dn, N)), D=r.normal(size=Dn), dt_bias=r.normal(size=Dn) - 1.0,
             z=r.normal(size=(batch, L, Dn)) if gate else None,
             h0=r.normal(size=(batch, Dn, N)) if h0 else None)
    up = dict(dout=r.normal(size=(batch, L, Dn)),
              dh_last=r.normal(size=(batch, Dn, N)) if dh_last else None)
    return p, up


def _J(p, up):
    y, h_last, _ = oracle.scan(p["x"], p["dt"], p["B"], p["C"], p["A"], z=p["z"], D=p["D"],
                               dt_bias=p["dt_bias"], h0=p["h0"], nthreads=1)
    J = float(np.sum(up["dout"] * y))
    if up["dh_last"] is not None:
        J += float(np.sum(up["dh_last"] * h_last))
    return J


def _grads(p, up):
    return oracle.scan_backward(p["x"], p["dt"], p["B"], p["C"], p["A"], up["dout"], z=p["z"], D=p["D"],
                                dt_bias=p["dt_bias"], h0=p["h0"], dh_last=up["dh_last"], nthreads=2)


GRAD_OF = {"x": "dx", "dt": "ddt", "B": "dB", "C": "dC", "A": "dA", "D": "dD", "dt_bias": "ddt_bias",
           "z": "dz", "h0": "dh0"}


@pytest.mark.parametrize("seed, kw", [(0, {}), (1, dict(gate=False)), (2, dict(h0=False, dh_last=False)),
                                      (3, dict(L=1, N=1)), (4, dict(batch=1, L=9, Dn=2, N=16))])
def test_every_gradient_matches_central_differences(seed, kw):
    p, up = _problem(seed, **kw)
    g = _grads(p, up)
    eps = 1e-6
    for name, gname in GRAD_OF.items():
        if p[name] is None:
            assert gname != "dz" or g["dz"] is None
            continue
        arr = p[name]
        num = np.empty_like(arr)
        for idx in np.ndindex(arr.shape):
            old = arr[idx]
            arr[idx] = old + eps
            jp = _J(p, up)
            arr[idx] = old - eps
            jm = _J(p, up)
            arr[idx] = old
            num[idx] = (jp - jm) / (2 * eps)
        scale = max(1.0, float(np.max(np.abs(num))))
        assert np.max(np.abs(g[gname] - num)) <= 2e-7 * scale, (name, np.max(np.abs(g[gname] - num)))


def test_adjoint_identity_is_exact_for_the_linear_inputs():
    # J is affine in x and in h0 (Delta, Abar do not depend on them), so a
    # perturbation of any size changes J by exactly <grad, perturbation>.
    p, up = _problem(7, batch=2, L=12, Dn=4, N=8)
    g = _grads(p, up)
    r = np.random.default_rng(8)
    J0 = _J(p, up)
    for name in ("x", "h0"):
        delta = r.normal(size=p[name].shape)
        q = dict(p)
        q[name] = p[name] + delta
        assert abs(_J(q, up) - J0 - float(np.sum(g[GRAD_OF[name]] * delta))) <= 1e-9 * (1 + abs(J0))


def test_state_gradient_is_the_product_of_decays():
    # dout = 0, dh_last = e: dJ/dh0[n] = prod_t Abar_t[n] * e[n] (Eq. 2 composed L times).
    p, up = _problem(11, batch=1, L=7, Dn=2, N=3)
    up["dout"] = np.zeros_like(up["dout"])
    e = np.ones_like(up["dh_last"])
    up["dh_last"] = e
    g = _grads(p, up)
    delta = np.log1p(np.exp(p["dt"][0] + p["dt_bias"]))          # [L, D]
    want = np.exp(np.einsum("td,dn->dn", delta, p["A"]))          # prod_t exp(Delta_t A)
    assert np.allclose(g["dh0"][0], want, rtol=1e-12, atol=0)
    # y does not enter J: no gradient reaches C, D or the gate
    assert np.all(g["dC"] == 0) and np.all(g["dD"] == 0) and np.all(g["dz"] == 0)


def test_thread_count_does_not_change_the_result_beyond_rounding():
    p, up = _problem(12, batch=3, L=20, Dn=9, N=16)
    a = oracle.scan_backward(p["x"], p["dt"], p["B"], p["C"], p["A"], up["dout"], z=p["z"], D=p["D"],
                             dt_bias=p["dt_bias"], h0=p["h0"], dh_last=up["dh_last"], nthreads=1)
    b = oracle.scan_backward(p["x"], p["dt"], p["B"], p["C"], p["A"], up["dout"], z=p["z"], D=p["D"],
                             dt_bias=p["dt_bias"], h0=p["h0"], dh_last=up["dh_last"], nthreads=4)
    for k in a:
        if a[k] is not None:
            assert np.allclose(a[k], b[k], rtol=1e-13, atol=1e-13), k
