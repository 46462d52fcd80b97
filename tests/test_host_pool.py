"""The host staging thread pool (native code, CPU): every part of every run executes exactly
once and never after its run returned, over thousands of back-to-back runs."""
import os
import subprocess

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_pool_stress(tmp_path):
    exe = tmp_path / "pool_stress"
    subprocess.run(["g++", "-O2", "-std=c++17", "-pthread",
                    "-I", os.path.join(ROOT, "paper_2607_18957_gb300", "csrc"),
                    os.path.join(ROOT, "tests", "pool_stress.cpp"), "-o", str(exe)], check=True)
    r = subprocess.run([str(exe), "20000"], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
