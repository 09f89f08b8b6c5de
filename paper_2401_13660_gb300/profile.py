"""Launch one entry point on a named workload, for profilers and quick timing.

    python -m paper_2401_13660_gb300.profile --entry prefill \
        --workload mambabyte353m_prefill_b8_L8192 --iters 5

Inputs are drawn on the GPU with the seeded generator of `inputs`; each
iteration launches the entry point once through the C ABI on one stream.
Prints the mean device time per launch (CUDA events) and the algorithmic-byte
rate. For the decode step, `--layers` distinct state/input sets are cycled so
that the working set exceeds the 129 MB L2 (default 4 layers, 643 MB); the
fused convolution + x-projection of the decoder (`--entry conv_xproj`) needs
16 or more of its 8.8 MB window and weight sets for the same (48 in the model).
"""
from __future__ import annotations

import argparse
import json

import torch

from . import mbscan as mb
from .inputs import WORKLOADS, workload_inputs

N_STATE = 16


def algorithmic_bytes(entry: str, w, s_in: int) -> int:
    b, L, D, N = w.batch, w.seqlen, w.d_inner, N_STATE
    params = D * N * 4 + 2 * D * 4
    if entry in ("prefill", "verify"):
        rd = 3 * b * L * D * s_in + 2 * b * L * N * s_in + params
        if w.dt_rank:   # dt is formed in the kernel from dt_low [b, L, r] and W_dt [D, r]
            rd += (b * L * w.dt_rank + D * w.dt_rank - b * L * D) * s_in
        rd += b * D * N * 4 if (w.h0 != "zeros" or entry == "verify") else 0
        wr = b * L * D * s_in + (b * D * N * 4 if entry == "prefill" else b * L * D * N * 4)
        return rd + wr
    if entry == "rollback":
        return 2 * b * D * N * 4 + b * 4
    if entry == "step":
        return 2 * b * D * N * 4 + 3 * b * D * s_in + 2 * b * N * s_in + params + b * D * s_in
    if entry == "backward":
        nch = (L + 15) // 16
        rd = 4 * b * L * D * s_in + 2 * b * L * N * s_in + params + b * nch * D * N * 4
        rd += b * D * N * 4 if w.h0 != "zeros" else 0
        rd += b * D * N * 4   # dh_last
        wr = 3 * b * L * D * s_in + 2 * b * L * N * 4 + D * N * 4 + 2 * D * 4 + b * D * N * 4
        return rd + wr
    raise ValueError(entry)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--entry", choices=["prefill", "verify", "rollback", "step", "backward", "decode_model",
                                        "conv_xproj"], required=True)
    ap.add_argument("--workload", required=True,
                    help="a workload of inputs.WORKLOADS, or for --entry decode_model / conv_xproj a "
                         "decoder.CONFIGS name")
    ap.add_argument("--batch", type=int, default=256, help="streams of --entry decode_model / conv_xproj")
    ap.add_argument("--iters", type=int, default=5)
    ap.add_argument("--layers", type=int, default=4, help="state sets cycled by --entry step / conv_xproj")
    a = ap.parse_args()
    dev = torch.device("cuda:0")
    if a.entry == "decode_model":
        return decode_model(a, dev)
    if a.entry == "conv_xproj":
        return conv_xproj(a, dev)
    w = WORKLOADS[a.workload]
    mb.load_library()
    nsets = a.layers if a.entry == "step" else 1
    sets = []
    for layer in range(nsets):
        inp = workload_inputs(w, dev, layer=layer)
        x = inp["x"]
        inp["y"] = torch.empty_like(x)
        inp["ws"] = torch.zeros(256, dtype=torch.uint8, device=dev)
        if inp["h0"] is None and a.entry in ("verify", "rollback", "step"):
            inp["h0"] = torch.zeros(w.batch, w.d_inner, N_STATE, device=dev)
        if a.entry in ("prefill", "backward"):
            inp["h_last"] = torch.empty(w.batch, w.d_inner, N_STATE, device=dev)
        if a.entry in ("verify", "rollback"):
            inp["h_all"] = torch.empty(w.batch, w.seqlen, w.d_inner, N_STATE, device=dev)
            inp["h_out"] = torch.empty_like(inp["h0"])
            if "accept" not in inp:
                inp["accept"] = torch.randint(0, w.seqlen + 1, (w.batch,), device=dev,
                                              dtype=torch.int32)
        if a.entry == "step":
            for k in ("x", "z", "dt", "B", "C", "y"):
                inp[k] = inp[k][:, :1].contiguous()
            inp["state"] = inp["h0"].clone()
        sets.append(inp)
    if a.entry == "backward":   # the training forward provides the checkpoints
        s0 = sets[0]
        _, _, s0["h_ckpt"] = mb.mb_scan_prefill_ckpt(s0["x"], s0["dt"], s0["B"], s0["C"], s0["A"], s0["y"],
                                                     z=s0["z"], D=s0["D"], dt_bias=s0["dt_bias"], h0=s0["h0"],
                                                     h_last=s0["h_last"], ws=s0["ws"])
        gen = torch.Generator(device=dev).manual_seed(5)
        s0["dout"] = torch.randn(s0["x"].shape, device=dev, generator=gen).to(s0["x"].dtype)
        s0["dh_last"] = torch.randn(s0["h_last"].shape, device=dev, generator=gen)
        s0["grads"] = mb.mb_scan_backward(s0["x"], s0["dt"], s0["B"], s0["C"], s0["A"], s0["h_ckpt"],
                                          s0["dout"], z=s0["z"], D=s0["D"], dt_bias=s0["dt_bias"],
                                          h0=s0["h0"], dh_last=s0["dh_last"], ws=s0["ws"])
    if a.entry == "rollback":
        s0 = sets[0]
        mb.mb_scan_verify(s0["x"], s0["dt"], s0["B"], s0["C"], s0["A"], s0["y"], s0["h_all"],
                          z=s0["z"], D=s0["D"], dt_bias=s0["dt_bias"], h0=s0["h0"], ws=s0["ws"])

    stream = torch.cuda.Stream(dev)

    def launch(s):
        if a.entry == "prefill":
            mb.mb_scan_prefill(s["x"], s["dt"], s["B"], s["C"], s["A"], s["y"], z=s["z"], D=s["D"],
                               dt_bias=s["dt_bias"], h0=s["h0"], h_last=s["h_last"], ws=s["ws"],
                               stream=stream, dt_low=s.get("dt_low"), W_dt=s.get("W_dt"))
        elif a.entry == "verify":
            mb.mb_scan_verify(s["x"], s["dt"], s["B"], s["C"], s["A"], s["y"], s["h_all"], z=s["z"],
                              D=s["D"], dt_bias=s["dt_bias"], h0=s["h0"], ws=s["ws"], stream=stream,
                              dt_low=s.get("dt_low"), W_dt=s.get("W_dt"))
        elif a.entry == "rollback":
            mb.mb_rollback(s["h0"], s["h_all"], s["accept"], s["h_out"], ws=s["ws"], stream=stream)
        elif a.entry == "backward":
            mb.mb_scan_backward(s["x"], s["dt"], s["B"], s["C"], s["A"], s["h_ckpt"], s["dout"], z=s["z"],
                                D=s["D"], dt_bias=s["dt_bias"], h0=s["h0"], dh_last=s["dh_last"],
                                grads=s["grads"], ws=s["ws"], stream=stream)
        else:
            mb.mb_step(s["x"], s["dt"], s["B"], s["C"], s["A"], s["y"], s["state"], z=s["z"],
                       D=s["D"], dt_bias=s["dt_bias"], stream=stream)

    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    with torch.cuda.stream(stream):
        launch(sets[0])
        ev[0].record(stream)
        for i in range(a.iters):
            launch(sets[i % nsets])
        ev[1].record(stream)
    stream.synchronize()
    us = 1e3 * ev[0].elapsed_time(ev[1]) / max(a.iters, 1)
    nbytes = algorithmic_bytes(a.entry, w, 2 if w.dtype == "bf16" else 4)
    print(json.dumps({"entry": a.entry, "workload": w.name, "iters": a.iters, "us_per_launch": round(us, 3),
                      "algorithmic_bytes": nbytes, "GB/s": round(nbytes / (us * 1e-6) / 1e9, 1)}))


def decode_model(a, dev):
    """Whole-model decoding: capture the step's CUDA graph, replay it."""
    from .decoder import CONFIGS, Decoder

    dec = Decoder(CONFIGS[a.workload], batch=a.batch, device=dev, seed=1)
    dec.capture()
    tok = torch.randint(0, 256, (a.batch,), device=dev, generator=torch.Generator(device=dev).manual_seed(8))
    dec.step(tok)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev[0].record()
    for _ in range(a.iters):
        dec.step(tok)
    ev[1].record()
    torch.cuda.synchronize()
    ms = ev[0].elapsed_time(ev[1]) / max(a.iters, 1)
    nb = dec.bytes_per_step()
    print(json.dumps({"entry": "decode_model", "workload": a.workload, "batch": a.batch, "iters": a.iters,
                      "ms_per_step": round(ms, 4), "bytes_per_step": nb, "GB/s": round(nb / ms / 1e6, 1),
                      "generated_bytes_per_s": round(a.batch / (ms * 1e-3), 1)}))


def conv_xproj(a, dev):
    """The decoder's fused convolution step + x-projection (mb_conv_xproj,
    with its split-K reduction) at one layer's shapes: one CUDA graph of one
    launch per each of --layers distinct window and weight sets, replayed
    --iters times."""
    from .decoder import CONFIGS

    cfg = CONFIGS[a.workload]
    B, E, n_out = a.batch, cfg.d_inner, cfg.dt_rank + 2 * cfg.d_state
    g = torch.Generator(device=dev).manual_seed(3)
    bf = torch.bfloat16
    x = torch.randn(B, E, device=dev, generator=g).to(bf)
    sets = [dict(st=torch.randn(B, 3, E, device=dev, generator=g).to(bf),
                 w=torch.rand(E, 4, device=dev, generator=g) - 0.5, b=torch.rand(E, device=dev, generator=g) - 0.5,
                 W=(torch.randn(n_out, E, device=dev, generator=g) / E ** 0.5).to(bf)) for _ in range(a.layers)]
    xc = torch.empty(B, E, device=dev, dtype=bf)
    out = torch.empty(B, n_out, device=dev, dtype=bf)
    ws = torch.zeros(mb.mb_conv_xproj_workspace_size(B, E, n_out), dtype=torch.uint8, device=dev)
    def run_all():   # one launch per set, as the decoder's layers do
        for s in sets:
            mb.mb_conv_xproj(x, s["st"], s["w"], s["W"], xc, out, ws, bias=s["b"])

    stream = torch.cuda.Stream(dev)
    stream.wait_stream(torch.cuda.current_stream(dev))
    with torch.cuda.stream(stream):
        run_all()   # eager warm-up
    torch.cuda.current_stream(dev).wait_stream(stream)
    graph = torch.cuda.CUDAGraph()   # replayed, so that host launch costs stay out of the timing
    with torch.cuda.graph(graph):
        run_all()
    graph.replay()
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev[0].record()
    for _ in range(a.iters):
        graph.replay()
    ev[1].record()
    torch.cuda.synchronize()
    st, _ = mb.mb_check(ws)
    if st != mb.MB_OK:
        raise mb.MbError(st, "conv_xproj")
    us = 1e3 * ev[0].elapsed_time(ev[1]) / max(a.iters * a.layers, 1)
    # x read, window read and written, xc written, W and the convolution taps read, out written
    nbytes = B * E * 2 * (1 + 6 + 1) + n_out * E * 2 + E * 20 + B * n_out * 2
    print(json.dumps({"entry": "conv_xproj", "workload": a.workload, "batch": B, "n_out": n_out, "iters": a.iters,
                      "us_per_launch": round(us, 3), "algorithmic_bytes": nbytes,
                      "GB/s": round(nbytes / (us * 1e-6) / 1e9, 1)}))


if __name__ == "__main__":
    main()
