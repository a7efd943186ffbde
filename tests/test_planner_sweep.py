"""The in-order schedule's units and reduction trees, checked on the CPU by
compiling the planner source with a C++ checker (tests/planner_check.cpp)."""
import os
import subprocess

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_30342_gb300", "csrc")


def test_sweep_schedule_is_consistent(tmp_path):
    exe = tmp_path / "planner_check"
    subprocess.run(["g++", "-std=c++17", "-O1", "-I", os.path.join(ROOT, "include"), "-I", CSRC,
                    os.path.join(ROOT, "tests", "planner_check.cpp"),
                    os.path.join(CSRC, "rikfad_planner.cpp"), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, timeout=300)
    assert out.returncode == 0 and out.stdout.strip().endswith("OK"), out.stdout + out.stderr
