"""bench.py end to end on a small workload: the JSON line keeps the benchmark contract.

Runs the DiT-XL/2 256 px workload (9.4 MB per step, L2 flushed between steps) with the
end-to-end leg and a short oracle baseline, and checks every key the contract names: the
headline metric, the roofline object, the host-buffer end-to-end figure, the CPU baseline,
the kernel-launch count and the clock record.
"""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_line_keeps_the_contract():
    p = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--workload", "c2i-256",
                        "--steps", "5", "--warmup", "3", "--no-sweep", "--no-extra",
                        "--cpu-seconds", "2"], capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stderr[-3000:]
    d = json.loads(p.stdout.strip().splitlines()[-1])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "roofline", "cpu_baseline", "e2e", "gpu_launches", "clocks"):
        assert key in d, key
    assert d["n_gpus"] == 1 and d["steps"] == 5 and d["warmup"] == 3
    assert d["value"] > 0 and d["unit"] == "GB/s" and d["higher_is_better"] is True
    assert d["config"]["workload"] == "c2i-256" and d["config"]["l2"].startswith("flushed")
    r = d["roofline"]
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["achieved"] > 0 and r["peak"] > 0
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"], abs=6e-5)   # 4 decimals
    assert r["traffic"] is None                    # the ncu record is for the video workload
    assert d["gpu_launches"] == 5                  # one forecast launch per step
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    c = d["cpu_baseline"]
    assert c["kind"] == "oracle" and c["cores"] >= 1 and c["value"] > 0 and c["sample"]
    if d["clocks"] is not None:
        assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(d["clocks"])


def test_end_to_end_leg_pipelines_a_capped_host_ring():
    # With less page-locked memory than one slot (a rank's share of a node's cap), the e2e
    # leg cycles layers through a ring of host buffers and still overlaps the copies: the
    # DiT-XL/2 512 px slot (28 layers of 18.9 MB) under a 0.2 GB cap is a ring of 10 layers,
    # moved in chunks of 5, a whole slot each way per step.
    p = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--workload", "c2i-512",
                        "--steps", "3", "--warmup", "3", "--no-sweep", "--no-extra",
                        "--no-cpu-baseline", "--no-clocks", "--e2e-host-cap-gb", "0.2"],
                       capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stderr[-3000:]
    e = json.loads(p.stdout.strip().splitlines()[-1])["e2e"]
    slot = 28 * 8 * 1024 * 1152 * 2
    assert e["h2d_bytes_per_step"] == slot and e["d2h_bytes_per_step"] == slot
    assert e["host_ring_layers"] == 10 and e["chunk_layers"] == 5 and e["overlapped"] is True
    assert e["host_buffer_bytes"] == 10 * slot // 28 and e["value"] > 0
