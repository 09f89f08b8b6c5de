"""CPU checks of bench.py's host logic: algorithmic byte counts, the
multi-rank timing reduction (two gloo ranks on 127.0.0.1) and the JSON line
of the oracle (reference) arm, alone and under torchrun with two ranks."""
import json
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench

ROOT_DIR = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_algorithmic_bytes_of_the_workloads():
    # Read + write bytes, each tensor once (prefill 353M-shaped, verify, rollback,
    # decode step per layer).
    assert sum(bench.bytes_prefill(8, 8192, 2048)) == 1_079_132_160
    assert sum(bench.bytes_prefill(4, 8192, 3584, h0=True)) == 943_714_304
    assert sum(bench.bytes_verify(32, 16, 2048)) == 79_872_000
    assert sum(bench.bytes_rollback(32, 2048)) == 8_388_736
    assert sum(bench.bytes_step(256, 4608)) == 160_780_288
    # backward: reads 4 token tensors, B, C, parameters, 512 checkpoints, dh_last;
    # writes 3 token tensors, dB, dC (fp32), dA, dD, ddt_bias, dh0
    rd, wr = bench.bytes_backward(8, 8192, 2048)
    st = 8 * 2048 * 16 * 4
    assert rd == 4 * 8 * 8192 * 2048 * 2 + 2 * 8 * 8192 * 16 * 2 + 2048 * 16 * 4 + 2 * 2048 * 4 + 512 * st + st
    assert wr == 3 * 8 * 8192 * 2048 * 2 + 2 * 8 * 8192 * 16 * 4 + 2048 * 16 * 4 + 2 * 2048 * 4 + st
    parts = bench.step_bytes()
    assert parts["step"] == 48 * 160_780_288


def test_sfu_roofline_of_the_scan():
    # Per element: one ex2 (1/32 clk/SM); per (b, t, d): softplus (ex2 + lg2)
    # and silu (ex2 + rcp) shared by 16 states -> (2/32 + 2/16) / 16.
    assert bench.sfu_clocks_per_element() == pytest.approx(1 / 32 + (2 / 32 + 2 / 16) / 16)
    r = bench.sfu_roofline(elements=2**31, seconds=1e-3, sms=152, sm_mhz=2000.0)
    assert r["peak"] == pytest.approx(152 * 2e9 / bench.sfu_clocks_per_element())
    assert r["achieved"] == pytest.approx(2**31 / 1e-3)
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"], rel=1e-3)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        out[rank] = bench.reduce_max(10.0 + rank, dist)
    finally:
        dist.destroy_process_group()


def test_reduce_max_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        assert dict(out) == {0: 11.0, 1: 11.0}


def test_reduce_max_single_process_is_identity():
    assert bench.reduce_max(3.5, None) == 3.5


def test_traffic_record_needs_matching_source(tmp_path, monkeypatch):
    (tmp_path / "profiles").mkdir()
    src = tmp_path / "paper_2401_13660_gb300" / "csrc"
    src.mkdir(parents=True)
    (src / "k.cu").write_text("kernel source v1\n")
    import hashlib
    sha = hashlib.sha256(b"kernel source v1\n").hexdigest()[:16]
    (tmp_path / "profiles" / "ncu_traffic.txt").write_text(
        f"kernel=my_kernel source=k.cu sha={sha} bytes_per_launch=1000\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_from_profiles("my_kernel") == 1000.0
    (src / "k.cu").write_text("kernel source v2\n")
    assert bench.traffic_from_profiles("my_kernel") is None
    assert bench.traffic_from_profiles("other") is None


def test_traffic_record_covers_every_listed_source(tmp_path, monkeypatch):
    (tmp_path / "profiles").mkdir()
    src = tmp_path / "paper_2401_13660_gb300" / "csrc"
    src.mkdir(parents=True)
    (src / "k.cu").write_text("kernel\n")
    (src / "h.cuh").write_text("header v1\n")
    import hashlib
    sha = hashlib.sha256(b"kernel\nheader v1\n").hexdigest()[:16]
    (tmp_path / "profiles" / "ncu_traffic.txt").write_text(
        f"kernel=my_kernel source=k.cu,h.cuh sha={sha} bytes_per_launch=500 scale=2\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_from_profiles("my_kernel") == 1000.0
    (src / "h.cuh").write_text("header v2\n")   # a header change also retires the record
    assert bench.traffic_from_profiles("my_kernel") is None
    (src / "h.cuh").unlink()
    assert bench.traffic_from_profiles("my_kernel") is None


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _reference_cmd():
    import sys
    return [sys.executable, os.path.join(ROOT_DIR, "bench.py"), "--impl", "reference", "--steps", "1",
            "--warmup", "3", "--ref-fraction", str(1 / 128)]


def test_reference_arm_prints_the_contract_line():
    """The oracle arm (no GPU) prints one JSON line with the contract's keys."""
    import subprocess
    r = subprocess.run(_reference_cmd(), capture_output=True, text=True, timeout=900, cwd=ROOT_DIR)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == "GB/s"
    assert d["value"] > 0 and d["steps"] == 1 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["higher_is_better"] is True and d["vs_baseline"] is None
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["e2e"]["value"] == d["value"] and d["config"]["workload"] == bench.WORKLOAD_NAME


def test_reference_arm_under_two_ranks_prints_once():
    """Under torchrun with 2 ranks, rank 0 alone runs and prints; both exit 0."""
    import subprocess
    import sys
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port())] + _reference_cmd()[1:] + ["--gpus", "2"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=900, cwd=ROOT_DIR)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.lstrip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0].strip())
    assert d["impl"] == "reference" and d["n_gpus"] == 2
