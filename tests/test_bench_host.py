"""Host-side pieces of bench.py, without a GPU.

* The multi-GPU path is replicas only: every rank serves its own sessions
  and the job's value is the summed bytes over the slowest rank's time. The
  reduction runs here on two gloo processes.
* The reference arm (the CPU oracle timed on the host cores) prints the
  contract's JSON line, and only rank 0 prints under a launcher.
"""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    total, e2e, kv = bench.reduce_over_ranks(10.0 + rank, 20.0 - rank, 1e9 * (rank + 1))
    out.put((rank, total, e2e, kv))
    dist.destroy_process_group()


def test_replica_reduction_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, total, e2e, kv in res:
        assert total == 11.0 and e2e == 20.0 and kv == 3e9


def test_replicas_draw_disjoint_sessions():
    sys.path.insert(0, ROOT)
    import bench
    import synth
    a = synth.session_lengths(bench.replica_seed(0, 0), 32, 8192, 32768)
    b = synth.session_lengths(bench.replica_seed(0, 1), 32, 8192, 32768)
    assert not np.array_equal(a, b)
    assert a.min() >= 8192 and a.max() <= 32768


def _run(args, env_extra=None):
    env = dict(os.environ)
    env.update(env_extra or {})
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                          env=env, capture_output=True, text=True, timeout=600)


def test_reference_arm_prints_contract_line():
    r = _run(["--impl", "reference", "--steps", "1", "--warmup", "3"])
    assert r.returncode == 0, r.stderr
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "cpu_baseline", "e2e", "config"):
        assert key in line
    assert line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0


def test_reference_arm_other_ranks_are_silent():
    r = _run(["--impl", "reference", "--steps", "1"], {"RANK": "1", "WORLD_SIZE": "2"})
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_traffic_record_goes_null_when_a_source_changes(tmp_path, monkeypatch):
    """roofline.traffic comes from the committed ncu record only while every
    kernel source it names still hashes to the captured value."""
    sys.path.insert(0, ROOT)
    import hashlib
    import bench
    src = tmp_path / "k.cu"
    src.write_text("kernel v1\n")
    (tmp_path / "profiles").mkdir()
    rec = tmp_path / "profiles" / bench.TRAFFIC_RECORD
    sha = hashlib.sha256(b"kernel v1\n").hexdigest()
    rec.write_text(f"# capture\nkernel: k\ndram_bytes_per_launch: 1234\nsha256 k.cu: {sha}\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.recorded_traffic() == 1234
    src.write_text("kernel v2\n")
    assert bench.recorded_traffic() is None
    rec.write_text("kernel: k\ndram_bytes_per_launch: 1234\n")   # no hashes: not trusted
    assert bench.recorded_traffic() is None


def test_cpu_unpack_baseline_reports_its_sample():
    """The resume metric's CPU baseline: the oracle's unpack on a bounded,
    stated sample, with the keys the bench line carries."""
    sys.path.insert(0, ROOT)
    import bench
    r = bench.cpu_unpack_baseline(0, tokens=64, budget_s=0.01)
    assert r["kind"] == "oracle" and r["cores"] == 1 and r["value"] > 0
    assert r["unit"] == "GB/s r+w" and "64-token image" in r["sample"]
