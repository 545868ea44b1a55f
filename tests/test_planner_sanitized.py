"""The host planner (planner.cpp) built with AddressSanitizer and
UndefinedBehaviorSanitizer and driven over random ragged layouts by
tests/planner_fuzz.cpp: chunk tables with and without tails, shard ranges,
on-chip grids and rounds.  The harness checks each result against its rule;
the sanitizers fail the run on any out-of-bounds access, leak or undefined
behaviour in the native code."""
import os
import shutil
import subprocess

import pytest

from conftest import ROOT

CSRC = os.path.join(ROOT, "paper_1904_00962_gb300", "csrc")


def test_planner_under_sanitizers(tmp_path):
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ not available")
    exe = tmp_path / "planner_fuzz"
    cmd = [gxx, "-std=c++17", "-O1", "-g", "-fno-omit-frame-pointer",
           "-fsanitize=address,undefined", "-fno-sanitize-recover=all",
           "-Wall", "-Wextra", "-Werror",
           "-I", os.path.join(ROOT, "include"), "-I", "/usr/local/cuda/include",
           "-I", CSRC, os.path.join(CSRC, "planner.cpp"),
           os.path.join(ROOT, "tests", "planner_fuzz.cpp"), "-o", str(exe)]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode and "sanitize" in res.stderr and "cannot find" in \
            res.stderr:
        pytest.skip("sanitizer runtime not available")
    assert res.returncode == 0, res.stderr
    run = subprocess.run([str(exe), "3000"], capture_output=True, text=True,
                         timeout=600,
                         env=dict(os.environ, ASAN_OPTIONS="detect_leaks=1"))
    assert run.returncode == 0, run.stderr[-4000:]
    assert run.stdout.strip() == "3000 layouts"
