"""Host-side pieces of bench.py: the multi-rank reduction (gloo, world size 2)
and the reference arm's JSON line."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _rank(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    d = bench.Dist()
    mx = d.reduce(float(rank + 1), "max")
    sm = d.reduce(float(rank + 1), "sum")
    d.barrier()
    d.close()
    q.put((rank, mx, sm))


def test_two_rank_reduction_gloo():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + (os.getpid() % 2000)
    ps = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in ps)
    for p in ps:
        p.join(timeout=60)
    assert res == [(0, 2.0, 3.0), (1, 2.0, 3.0)]


def test_reference_arm_prints_one_json_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0", "--ref-tokens", "16"], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["e2e"]["h2d_bytes_per_step"] == 0
    assert d["cpu_baseline"]["kind"] == "oracle"


def test_captured_traffic_follows_the_source_hash(tmp_path):
    """The roofline's DRAM traffic comes from the traffic table only while the
    kernel source still has the hash recorded beside it and the workload is the
    one captured."""
    import hashlib
    import bench
    src = tmp_path / "kernel.cu"
    src.write_text("// kernel source\n")
    sha = hashlib.sha256(src.read_bytes()).hexdigest()
    table = tmp_path / "traffic.json"
    rec = {"source": os.path.relpath(str(src), ROOT), "sha256_prefix": sha[:16], "workload": "w B1",
           "bytes_per_launch": 123456, "summary": "s.md"}
    table.write_text(json.dumps({"my_kernel": rec}))
    assert bench.captured_traffic("my_kernel", "w B1", str(table))["bytes_per_launch"] == 123456
    assert bench.captured_traffic("other_kernel", "w B1", str(table)) is None
    assert bench.captured_traffic("my_kernel", "w B2", str(table)) is None
    src.write_text("// kernel source, changed\n")
    assert bench.captured_traffic("my_kernel", "w B1", str(table)) is None


def test_committed_traffic_table_is_well_formed():
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        t = json.load(f)
    for k, rec in t.items():
        if k.startswith("_"):
            continue
        assert set(rec) >= {"source", "sha256_prefix", "workload", "bytes_per_launch", "summary"}
        assert os.path.exists(os.path.join(ROOT, rec["source"])) and os.path.exists(os.path.join(ROOT, rec["summary"]))


def test_clock_record_counts_the_timed_region_apart():
    """The clock summary of nvidia-smi lines: the median SM clock under load,
    throttle reasons that were active, and the samples whose timestamps fall
    inside the timed region (with a 50 ms margin) counted apart."""
    import datetime
    import time

    sys.path.insert(0, ROOT)
    import bench
    now = time.time()

    def line(dt, sm, util, thermal="Not Active"):
        ts = datetime.datetime.fromtimestamp(now + dt).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
        return f"{ts}, 0, {sm}, 2070, 190.5, {util}, 0x0, Not Active, {thermal}, Not Active, Not Active\n"

    lines = [line(-0.40, 1980, 99), line(-0.20, 2070, 99), line(0.01, 2070, 99), line(0.30, 300, 0)]
    rec = bench.Clocks.summarize(lines, (now, now + 0.03))
    assert rec["samples"] == 4 and rec["samples_under_load"] == 3
    assert rec["sm_mhz"] == 2070.0 and rec["reasons"] == []
    assert rec["samples_in_timed_region"] == 1 and rec["sm_mhz_in_timed_region"] == 2070.0
    rec = bench.Clocks.summarize(lines + [line(0.02, 1500, 99, thermal="Active")], (now, now + 0.03))
    assert rec["reasons"] == ["hw_thermal_slowdown"] and rec["samples_in_timed_region"] == 2
    assert bench.Clocks.summarize(["garbage\n"]) is None
