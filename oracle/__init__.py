"""fp64 CPU oracle for the selective-scan layer core (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the benchmark's CPU
baseline leg may import this package. It shares no code with the CUDA library
and never imports it. The arithmetic lives in ``mb_oracle.c`` (plain C, fp64,
sequential in time); this module compiles it with gcc and marshals numpy
arrays to it.

Functions (MambaByte, Eq. 2-3, discretisation appendix, Table 6, Algorithm 1):

* ``scan``     - the layer core over a whole span: y, final state, and
                 optionally every per-position state (verify).
* ``delta_projection`` - the pre-softplus timestep of Eq. 3 from its low-rank
                 factor: W_Delta (W_R x), as an fp64 matrix product.
* ``step``     - one recurrent decode step (a scan of length 1).
* ``rollback`` - keep the state after ``accept`` drafted bytes.
* ``accept_topk`` - Algorithm 1's bifurcation: leading drafted bytes whose
                 rank in the verifier's distribution is within top-beta.
* ``scan_backward`` - every input gradient of J given dJ/dout and dJ/dh_last
                 (the training path), by the adjoint recurrence in fp64.
* ``rmsnorm``, ``conv1d_step``, ``block_step`` - the Mamba block around the
                 scan for recurrent decoding (Figure 6, Table 6): residual add
                 with RMS normalisation, one step of the causal depthwise
                 convolution with SiLU, and a whole block step (projections as
                 fp64 matrix products).

Inputs are widened exactly to float64 before the call (bf16 and fp32 values
are exactly representable in fp64).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mb_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libmb_oracle.so")
_lock = threading.Lock()
_lib = None

B_EULER, B_ZOH = 0, 1


def build(force: bool = False) -> str:
    """Compile mb_oracle.c into _build/libmb_oracle.so (gcc, OpenMP)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                    "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp, "-lm"],
                   check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            dp = ctypes.POINTER(ctypes.c_double)
            i64 = ctypes.c_int64
            lib.oracle_scan.argtypes = [i64, i64, i64, i64] + [dp] * 9 + [ctypes.c_int, dp, dp, dp,
                                                                         ctypes.c_int]
            lib.oracle_scan.restype = ctypes.c_int
            lib.oracle_rollback.argtypes = [i64, i64, i64, i64, dp, dp,
                                            ctypes.POINTER(ctypes.c_int32), dp]
            lib.oracle_rollback.restype = ctypes.c_int
            lib.oracle_scan_backward.argtypes = [i64, i64, i64, i64] + [dp] * 11 + [dp] * 9 + [ctypes.c_int]
            lib.oracle_scan_backward.restype = ctypes.c_int
            _lib = lib
    return _lib


def _f64(a):
    if a is None:
        return None
    if hasattr(a, "detach"):  # a torch tensor: widen exactly on the host
        a = a.detach().to("cpu").double().numpy()
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def default_threads() -> int:
    return os.cpu_count() or 1


def scan(x, dt, B, C, A, *, z=None, D=None, dt_bias=None, h0=None, b_rule=B_EULER,
         want_h_all=False, nthreads=None):
    """Run the layer core over [batch, L] and return (y, h_last, h_all or None).

    x, dt, z: [batch, L, D]; B, C: [batch, L, N]; A: [D, N]; D, dt_bias: [D];
    h0: [batch, D, N] or None (zeros). All outputs are float64.
    """
    x, dt, B, C, A = map(_f64, (x, dt, B, C, A))
    z, D, dt_bias, h0 = map(_f64, (z, D, dt_bias, h0))
    batch, L, Dn = x.shape
    N = A.shape[1]
    assert dt.shape == x.shape and B.shape == (batch, L, N) and C.shape == (batch, L, N)
    assert A.shape == (Dn, N)
    assert z is None or z.shape == x.shape
    assert h0 is None or h0.shape == (batch, Dn, N)
    y = np.empty((batch, L, Dn), dtype=np.float64)
    h_last = np.empty((batch, Dn, N), dtype=np.float64)
    h_all = np.empty((batch, L, Dn, N), dtype=np.float64) if want_h_all else None
    rc = _load().oracle_scan(batch, L, Dn, N, _ptr(x), _ptr(z), _ptr(dt), _ptr(B), _ptr(C),
                             _ptr(A), _ptr(D), _ptr(dt_bias), _ptr(h0), int(b_rule), _ptr(y),
                             _ptr(h_last), _ptr(h_all), int(nthreads or default_threads()))
    if rc != 0:
        raise RuntimeError(f"oracle_scan failed ({rc})")
    return y, h_last, h_all


def scan_backward(x, dt, B, C, A, dout, *, z=None, D=None, dt_bias=None, h0=None, dh_last=None,
                  nthreads=None):
    """Gradients of J, given dJ/dout [batch, L, D] and dJ/dh_last [batch, D, N]
    (None = 0), for the Euler-rule layer core. Returns a dict with dx, dz
    (None without a gate), ddt [batch, L, D]; dB, dC [batch, L, N]; dA [D, N];
    dD, ddt_bias [D]; dh0 [batch, D, N] (all float64)."""
    x, dt, B, C, A, dout = map(_f64, (x, dt, B, C, A, dout))
    z, D, dt_bias, h0, dh_last = map(_f64, (z, D, dt_bias, h0, dh_last))
    batch, L, Dn = x.shape
    N = A.shape[1]
    assert dt.shape == x.shape and dout.shape == x.shape
    assert B.shape == (batch, L, N) and C.shape == (batch, L, N) and A.shape == (Dn, N)
    g = {k: np.empty((batch, L, Dn)) for k in ("dx", "ddt")}
    g["dz"] = np.empty((batch, L, Dn)) if z is not None else None
    g["dB"] = np.empty((batch, L, N))
    g["dC"] = np.empty((batch, L, N))
    g["dA"] = np.empty((Dn, N))
    g["dD"] = np.empty(Dn)
    g["ddt_bias"] = np.empty(Dn)
    g["dh0"] = np.empty((batch, Dn, N))
    rc = _load().oracle_scan_backward(
        batch, L, Dn, N, _ptr(x), _ptr(z), _ptr(dt), _ptr(B), _ptr(C), _ptr(A), _ptr(D), _ptr(dt_bias),
        _ptr(h0), _ptr(dout), _ptr(dh_last), _ptr(g["dx"]), _ptr(g["dz"]), _ptr(g["ddt"]), _ptr(g["dB"]),
        _ptr(g["dC"]), _ptr(g["dA"]), _ptr(g["dD"]), _ptr(g["ddt_bias"]), _ptr(g["dh0"]),
        int(nthreads or default_threads()))
    if rc != 0:
        raise RuntimeError(f"oracle_scan_backward failed ({rc})")
    return g


def delta_projection(dt_low, W_dt):
    """Eq. 3: the timestep before softplus is W_Delta applied to the rank-r
    projection W_R x. dt_low [batch, L, r] holds W_R x, W_dt [d_inner, r] is
    W_Delta; returns dt [batch, L, d_inner] = sum_k dt_low[..., k] W_dt[d, k],
    in fp64."""
    dl = np.asarray(dt_low, dtype=np.float64)
    w = np.asarray(W_dt, dtype=np.float64)
    return np.matmul(dl, w.T)


def step(state, x, dt, B, C, A, *, z=None, D=None, dt_bias=None, b_rule=B_EULER, nthreads=None):
    """One recurrent decode step. x, dt, z: [batch, D]; B, C: [batch, N];
    state: [batch, D, N]. Returns (y [batch, D], new_state)."""
    x, dt, B, C, z = (None if a is None else _f64(a)[:, None] for a in (x, dt, B, C, z))
    y, h, _ = scan(x, dt, B, C, A, z=z, D=D, dt_bias=dt_bias, h0=state, b_rule=b_rule,
                   nthreads=nthreads)
    return y[:, 0], h


def rollback(h0, h_all, accept):
    """State kept after accept[s] drafted bytes: h0[s] if accept[s] == 0, else
    h_all[s, accept[s] - 1]. h_all: [batch, k, D, N]; h0: [batch, D, N] or None."""
    h_all = _f64(h_all)
    h0 = _f64(h0)
    batch, k, Dn, N = h_all.shape
    acc = np.ascontiguousarray(np.asarray(accept.cpu() if hasattr(accept, "cpu") else accept),
                               dtype=np.int32)
    out = np.empty((batch, Dn, N), dtype=np.float64)
    rc = _load().oracle_rollback(batch, k, Dn, N, _ptr(h0), _ptr(h_all),
                                 acc.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), _ptr(out))
    if rc != 0:
        raise RuntimeError("oracle_rollback: accept count out of [0, k]")
    return out


def accept_topk(logits, drafted, beta):
    """Accept count per stream (Algorithm 1, bifurcation position): the number
    of leading drafted bytes b_i with rank_{p_i}(b_i) <= beta, where
    rank(b) = 1 + #{v : score[v] > score[b]}. logits [streams, k, 256],
    drafted [streams, k]. Plain loops over streams and positions."""
    if hasattr(logits, "detach"):
        logits = logits.detach().to("cpu").double().numpy()
    if hasattr(drafted, "detach"):
        drafted = drafted.detach().to("cpu").numpy()
    logits = np.asarray(logits, dtype=np.float64)
    drafted = np.asarray(drafted)
    streams, k, _ = logits.shape
    out = np.empty(streams, dtype=np.int32)
    for s in range(streams):
        a = k
        for i in range(k):
            row = logits[s, i]
            rank = 1 + int(np.sum(row > row[int(drafted[s, i])]))
            if rank > beta:
                a = i
                break
        out[s] = a
    return out


def bf16_round(a):
    """Round float64 values to the nearest bfloat16 (ties to even), returned
    as float64: the value a bf16 tensor holds after a cast."""
    a = np.asarray(a, dtype=np.float64)
    f = a.astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    u = (u + 0x7FFF + lsb) & 0xFFFF0000
    out = u.astype(np.uint32).view(np.float32).astype(np.float64)
    return np.where(np.isfinite(f), out, f.astype(np.float64))


def rmsnorm(residual, w, eps, add=None):
    """Residual add and RMS normalisation that open a Mamba block:
    r = residual + add; out = r / sqrt(mean(r^2) + eps) * w (last axis).
    Returns (r, out)."""
    r = _f64(residual) + (0.0 if add is None else _f64(add))
    out = r / np.sqrt(np.mean(r * r, axis=-1, keepdims=True) + eps) * _f64(w)
    return r, out


def silu(v):
    v = np.asarray(v, dtype=np.float64)
    return v / (1.0 + np.exp(-v))


def conv1d_step(state, x, w, bias=None):
    """One decode step of the causal depthwise convolution (kernel 4) with
    SiLU. state [b, 3, d] holds the three previous inputs, oldest first;
    x [b, d]; w [d, 4] (w[:, 3] multiplies the current input); bias [d].
    Returns (out [b, d], new_state)."""
    state, x, w = _f64(state), _f64(x), _f64(w)
    acc = state[:, 0] * w[:, 0] + state[:, 1] * w[:, 1] + state[:, 2] * w[:, 2] + x * w[:, 3]
    if bias is not None:
        acc = acc + _f64(bias)
    return silu(acc), np.stack([state[:, 1], state[:, 2], x], axis=1)


def block_step(layer, residual, add, ssm_state, conv_state, eps=1e-5, cast=bf16_round):
    """One Mamba block for one decoded byte per stream (MambaByte's Mamba-1
    block, Figure 6; Table 6 rows). `layer` holds float64 weights: norm_w,
    W_in_x, W_in_z [d_inner, d_model], conv_w [d_inner, 4], conv_b, W_dtlow
    [r, d_inner], W_B, W_C [16, d_inner], W_dt [d_inner, r], dt_bias, A
    [d_inner, 16], D, W_out [d_model, d_inner]. residual [b, d_model] (fp32
    stream), add = the previous block's output or None. Tensors the GPU path
    keeps in the input dtype are passed through `cast` at the same points.
    Returns (residual, out, ssm_state, conv_state)."""
    r, h = rmsnorm(residual, layer["norm_w"], eps, add)
    h = cast(h)
    x = cast(h @ layer["W_in_x"].T)
    z = cast(h @ layer["W_in_z"].T)
    xc, conv_state = conv1d_step(conv_state, x, layer["conv_w"], layer["conv_b"])
    xc = cast(xc)
    dtl = cast(xc @ layer["W_dtlow"].T)
    Bm = cast(xc @ layer["W_B"].T)
    Cm = cast(xc @ layer["W_C"].T)
    dt = cast(dtl @ layer["W_dt"].T)
    y, ssm_state = step(ssm_state, x=xc, dt=dt, B=Bm, C=Cm, A=layer["A"], z=z, D=layer["D"],
                        dt_bias=layer["dt_bias"])
    out = cast(cast(y) @ layer["W_out"].T)
    return r, out, ssm_state, conv_state
