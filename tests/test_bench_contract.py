"""bench.py's host side, without a GPU: the reference arm's JSON line (the
oracle on the host's cores, as the benchmark contract specifies it) and the
single-buffer packing the end-to-end step copies with."""

import importlib.util
import json
import os
import subprocess
import sys

import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench_module():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_pack_views_share_one_aligned_buffer():
    b = _bench_module()
    q = torch.randn(3, 2, 5, 128).half()
    ctx = torch.tensor([7, 9, 0], dtype=torch.int32)
    meter = torch.rand(3, 2, 5)
    keep = torch.randint(0, 2, (30,), dtype=torch.uint8)
    buf, (q2, ctx2, meter2, keep2) = b._pack((q, ctx, meter, keep))
    for orig, view in ((q, q2), (ctx, ctx2), (meter, meter2), (keep, keep2)):
        assert torch.equal(orig, view) and view.shape == orig.shape and view.dtype == orig.dtype
        assert (view.data_ptr() - buf.data_ptr()) % 256 == 0
        assert buf.data_ptr() <= view.data_ptr() < buf.data_ptr() + buf.numel()
    ctx2[1] = 41                                  # a write through a view lands in the buffer
    off = ctx2.data_ptr() - buf.data_ptr()
    assert buf[off:off + 12].view(torch.int32).tolist() == [7, 41, 0]
    assert buf.numel() % 256 == 0


def test_reference_arm_prints_the_contract_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "1",
                        "--steps", "1", "--warmup", "3", "--cpu-budget", "0.5"],
                       capture_output=True, text=True, timeout=600, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [x for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert d["config"]["workload"].startswith("1L-8q2kv-S4096")


def test_reference_arm_under_torchrun_prints_one_line_from_rank_zero():
    """The launch the scaling run uses (one process per GPU under
    torch.distributed.run): rank 0 alone runs the oracle and prints the line,
    with n_gpus the world size; the other rank exits 0 without work."""
    import socket
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
                        "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
                        "--impl", "reference", "--gpus", "2", "--config", "1", "--steps", "1", "--warmup", "3",
                        "--cpu-budget", "0.5"],
                       capture_output=True, text=True, timeout=600, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [x for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0


def test_traffic_row_used_only_at_its_kernel_source(tmp_path, monkeypatch):
    """roofline.traffic comes from profiles/traffic.txt only for the decode
    source the row was captured at; any other source gives null."""
    import hashlib
    b = _bench_module()
    root = tmp_path
    (root / "paper_2607_28699_gb300" / "csrc").mkdir(parents=True)
    (root / "profiles").mkdir()
    src = root / "paper_2607_28699_gb300" / "csrc" / "decode_kernel.cu"
    src.write_bytes(b"// kernel A\n")
    sha = hashlib.sha256(b"// kernel A\n").hexdigest()[:16]
    (root / "profiles" / "traffic.txt").write_text(
        "# kernel  source_sha256_16  workload  bytes_per_launch\n"
        f"decode_kernel {sha} wl-a 123456\n"
        "decode_kernel 0000000000000000 wl-b 999\n")
    monkeypatch.setattr(b, "ROOT", str(root))
    assert b._traffic("wl-a") == 123456
    assert b._traffic("wl-b") is None and b._traffic("wl-c") is None
    src.write_bytes(b"// kernel B\n")          # the kernel changed since the capture
    assert b._traffic("wl-a") is None
