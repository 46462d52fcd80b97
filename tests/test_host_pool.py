"""The host staging thread pool (native code, CPU): every part of every run executes exactly
once and never after its run returned, over thousands of back-to-back runs."""
import os
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_pool_stress(tmp_path):
    exe = tmp_path / "pool_stress"
    subprocess.run(["g++", "-O2", "-std=c++17", "-pthread",
                    "-I", os.path.join(ROOT, "paper_2607_18957_gb300", "csrc"),
                    os.path.join(ROOT, "tests", "pool_stress.cpp"), "-o", str(exe)], check=True)
    r = subprocess.run([str(exe), "20000"], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr


def test_pool_stress_under_thread_sanitizer(tmp_path):
    """The same stress run built with ThreadSanitizer: no data race between the caller, the
    workers and the job they share."""
    exe = tmp_path / "pool_stress_tsan"
    r = subprocess.run(["g++", "-O1", "-g", "-std=c++17", "-pthread", "-fsanitize=thread",
                        "-I", os.path.join(ROOT, "paper_2607_18957_gb300", "csrc"),
                        os.path.join(ROOT, "tests", "pool_stress.cpp"), "-o", str(exe)],
                       capture_output=True, text=True)
    if r.returncode != 0:
        pytest.skip("no ThreadSanitizer runtime for g++ here: " + r.stderr[-200:])
    r = subprocess.run([str(exe), "5000"], capture_output=True, text=True, timeout=300,
                       env={**os.environ, "TSAN_OPTIONS": "halt_on_error=1 exitcode=66"})
    if r.returncode != 0 and sanitizer_could_not_start(r.stderr):
        pytest.skip("the ThreadSanitizer runtime cannot start here: " + r.stderr[:200])
    assert r.returncode == 0, r.stdout + r.stderr[-3000:]


def sanitizer_could_not_start(stderr):
    """The sanitizer runtime failed before the program ran (ThreadSanitizer on a kernel whose
    address-space layout it does not support), as opposed to a report about the program."""
    return ("unexpected memory mapping" in stderr or "FATAL: ThreadSanitizer" in stderr
            or "Shadow memory range interleaves" in stderr)
