"""The launchers' tile counting on the CPU (no GPU): ``tests/c/tile_count.cpp`` is compiled
with g++ against the library's internal header and compares ``bc::TileCounter`` (a shift for
power-of-two tiles, a division otherwise) with the plain definition of the count."""
import os
import subprocess

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_tile_counts_match_the_definition(tmp_path):
    exe = tmp_path / "tile_count"
    subprocess.check_call([
        "g++", "-std=c++17", "-O2", "-o", str(exe), os.path.join(ROOT, "tests", "c", "tile_count.cpp"),
        "-I", os.path.join(ROOT, "include"),
        "-I", os.path.join(ROOT, "paper_2608_28670_gb300", "csrc")])
    p = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert p.returncode == 0, p.stdout + p.stderr
    assert "0 wrong" in p.stdout
