"""Seeded synthetic inputs for the selective-scan layer core.

This module only draws random tensors with the shapes and distributions of
MambaByte's layers (Table 5 hyper-parameters: n_state = 16, expansion e = 2,
d = 1024 / 1792 / 2304). It contains none of the layer core's arithmetic: the
CUDA path and the fp64 oracle both receive the tensors made here.

Recipe (per workload, one torch.Generator seeded with the workload's seed,
draws always in this order, always in fp32, rounded once to bf16 where the
workload is bf16):

* x, z, B, C ~ N(0, 1)
* dt (the raw pre-softplus timestep, "Delta_raw") ~ N(0, 1)
* D ~ N(0, 1)
* dt_bias[d] = inverse softplus of a target step Delta*_d drawn log-uniform on
  [0.01, 0.1], so that softplus(dt + dt_bias) has its median in 0.01..0.1
* A[d, n] = -(n + 1) (S4D-real initialisation of Mamba's diagonal A)
* h0 = 0, or ~ N(0, 0.1^2) for workloads that resume from a cached state
* accept (verify workloads) ~ uniform integers in [0, seqlen]
* fused Delta projection (dt_rank r > 0, drawn last): dt_low ~ N(0, 1)
  [batch, L, r] and W_dt ~ N(0, 1/r) [d_inner, r], so that dt_low W_dt^T is
  again ~ N(0, 1); dt itself is then dropped (the kernels form it)
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class Workload:
    """One selective-scan problem size, named by what it is."""
    name: str
    batch: int
    seqlen: int
    d_inner: int
    d_state: int
    dtype: str            # "f32" or "bf16": dtype of x, z, dt, B, C and y
    h0: str               # "zeros" or "normal"
    seed: int
    layers: int = 1       # distinct state/input sets (decode step over a layer stack)
    accept: bool = False  # draw per-stream accept counts (speculative verify)
    dt_rank: int = 0      # > 0: dt comes as the low-rank pair (dt_low, W_dt) of Eq. 3
    note: str = field(default="", compare=False)


WORKLOADS = {
    w.name: w
    for w in [
        Workload("tiny_f32_b1_L256_D64", 1, 256, 64, 16, "f32", "zeros", 0,
                 note="single fp32 layer, oracle-sized"),
        Workload("mambabyte353m_prefill_b8_L8192", 8, 8192, 2048, 16, "bf16", "zeros", 1,
                 note="MambaByte-353M layer (d=1024, e=2) prefill"),
        Workload("mambabyte972m_prefill_b4_L8192", 4, 8192, 3584, 16, "bf16", "normal", 2,
                 note="MambaByte-972M layer (d=1792, e=2) prefill from a given h0"),
        Workload("verify_s32_k16_D2048", 32, 16, 2048, 16, "bf16", "normal", 3, accept=True,
                 note="speculative verify of a 16-byte drafted span on 32 streams"),
        Workload("step_b256_D4608_x48", 256, 1, 4608, 16, "bf16", "normal", 4, layers=48,
                 note="MambaByte-1.6B (d=2304, e=2) batched decode step, 48 layers"),
        Workload("mambabyte353m_prefill_fused_r64_b8_L8192", 8, 8192, 2048, 16, "bf16", "zeros", 5,
                 dt_rank=64, note="MambaByte-353M layer prefill, Delta projection (r = d/16) in the kernel"),
        Workload("mambabyte972m_prefill_fused_r112_b4_L8192", 4, 8192, 3584, 16, "bf16", "normal", 6,
                 dt_rank=112, note="MambaByte-972M layer prefill, Delta projection (r = d/16) in the kernel"),
        Workload("verify_fused_r64_s32_k16_D2048", 32, 16, 2048, 16, "bf16", "normal", 7, accept=True,
                 dt_rank=64, note="speculative verify (353M layer), Delta projection in the kernel"),
    ]
}


def torch_dtype(dtype: str) -> torch.dtype:
    return {"f32": torch.float32, "bf16": torch.bfloat16}[dtype]


def _normal(gen, shape, device, std=1.0):
    t = torch.empty(shape, dtype=torch.float32, device=device)
    t.normal_(0.0, std, generator=gen)
    return t


def make_inputs(batch: int, seqlen: int, d_inner: int, d_state: int, dtype: str = "bf16",
                h0: str = "zeros", seed: int = 0, device="cpu", accept: bool = False,
                gate: bool = True, dt_rank: int = 0) -> dict:
    """Draw one problem. Returns a dict of contiguous torch tensors on `device`.

    Keys: x, z (None if gate=False), dt, B, C (input dtype); A [d_inner, d_state],
    D [d_inner], dt_bias [d_inner] (fp32); h0 [batch, d_inner, d_state] fp32 or
    None; accept [batch] int32 (only if accept=True). With dt_rank > 0, dt is
    None and dt_low [batch, L, dt_rank], W_dt [d_inner, dt_rank] (input dtype)
    are given instead.
    """
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    td = torch_dtype(dtype)
    tok = (batch, seqlen, d_inner)
    x = _normal(gen, tok, device).to(td)
    z = _normal(gen, tok, device).to(td)
    dt = _normal(gen, tok, device).to(td)
    B = _normal(gen, (batch, seqlen, d_state), device).to(td)
    C = _normal(gen, (batch, seqlen, d_state), device).to(td)
    D = _normal(gen, (d_inner,), device)
    u = torch.empty((d_inner,), dtype=torch.float64, device=device).uniform_(0.0, 1.0, generator=gen)
    lo, hi = math.log(0.01), math.log(0.1)
    target = torch.exp(lo + u * (hi - lo))                       # Delta* log-uniform on [0.01, 0.1]
    dt_bias = (target + torch.log(-torch.expm1(-target))).float()  # inverse softplus of Delta*
    A = -torch.arange(1, d_state + 1, dtype=torch.float32, device=device).repeat(d_inner, 1)
    out = dict(x=x, z=z if gate else None, dt=dt, B=B, C=C, A=A.contiguous(), D=D,
               dt_bias=dt_bias, h0=None)
    if h0 == "normal":
        out["h0"] = _normal(gen, (batch, d_inner, d_state), device, std=0.1)
    elif h0 != "zeros":
        raise ValueError(f"unknown h0 kind {h0!r}")
    if accept:
        out["accept"] = torch.randint(0, seqlen + 1, (batch,), generator=gen, device=device,
                                      dtype=torch.int64).to(torch.int32)
    if dt_rank > 0:
        out["dt_low"] = _normal(gen, (batch, seqlen, dt_rank), device).to(td)
        out["W_dt"] = _normal(gen, (d_inner, dt_rank), device, std=1.0 / math.sqrt(dt_rank)).to(td)
        out["dt"] = None
    return out


def workload_inputs(w: Workload, device="cpu", layer: int = 0) -> dict:
    """Inputs of one layer of a workload (layer > 0 reseeds so layers differ)."""
    return make_inputs(w.batch, w.seqlen, w.d_inner, w.d_state, w.dtype, w.h0,
                       seed=w.seed * 1000 + layer, device=device, accept=w.accept, dt_rank=w.dt_rank)
