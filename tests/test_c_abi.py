"""The C ABI from plain C: tests/c/abi_client.c is compiled with gcc against
include/barycache.h and linked with libbarycache.so (and the oracle, for its checks)."""
import os
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def client(tmp_path_factory):
    import __graft_entry__
    import oracle
    libs = __graft_entry__.build_libraries()
    oracle.build()
    out = tmp_path_factory.mktemp("abi") / "abi_client"
    libdir = os.path.dirname(libs["libbarycache.so"])
    odir = os.path.join(ROOT, "oracle")
    cuda = "/usr/local/cuda/lib64"
    subprocess.check_call([
        "gcc", "-std=c11", "-O1", "-o", str(out), os.path.join(ROOT, "tests", "c", "abi_client.c"),
        "-I", os.path.join(ROOT, "include"),
        "-L", libdir, "-lbarycache", f"-Wl,-rpath,{libdir}",
        os.path.join(odir, "liboracle.so"), f"-Wl,-rpath,{odir}",
        "-L", cuda, "-lcudart", f"-Wl,-rpath,{cuda}", "-lm"])
    return str(out)


def test_c_client_host_calls(client):
    p = subprocess.run([client, "host"], capture_output=True, text=True, timeout=120)
    assert p.returncode == 0, p.stdout + p.stderr


@pytest.mark.gpu
def test_c_client_full_forecast_on_the_device(client):
    p = subprocess.run([client, "device"], capture_output=True, text=True, timeout=300)
    assert p.returncode == 0, p.stdout + p.stderr


@pytest.mark.gpu
def test_c_client_many_tensors_one_launch_each(client):
    # 2048 tensors pushed and forecast from plain C: one launch per call, every element
    # against the oracle, a planted NaN carried through
    p = subprocess.run([client, "manylayers"], capture_output=True, text=True, timeout=300)
    assert p.returncode == 0, p.stdout + p.stderr


@pytest.mark.gpu
def test_c_client_host_cost_mode_runs(client):
    # The timing mode reports one JSON line per cache size; the numbers are measurements,
    # so only their presence and sanity are checked here.
    import json
    p = subprocess.run([client, "hostcost"], capture_output=True, text=True, timeout=300)
    assert p.returncode == 0, p.stdout + p.stderr
    rows = [json.loads(l) for l in p.stdout.splitlines() if l.startswith("{")]
    assert [r["layers"] for r in rows] == [1, 4, 16, 64, 4096, 65536]
    small, large = rows[:4], rows[4:]
    assert all(0 < r["host_us_per_forecast"] < 1000 and r["memo_lookup_us"] > 0 for r in small)
    # thousands of tensors: the per-call work is linear in the tensor count, well under a
    # microsecond per tensor
    assert all(0 < r["host_ns_per_tensor_forecast"] < 200 and 0 < r["host_ns_per_tensor_push"] < 200
               for r in large)
