"""The C ABI used from plain C: include/gar.h compiles as pedantic C99 and as C++, and a
C program linked against libgar.so (tests/c_abi_check.c, host-only calls) sees the same
plans, byte counts, schedule, error codes and cost model as the Python binding."""

import os
import shutil
import subprocess

import pytest

from paper_2004_09362_gb300 import gar

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INC = os.path.join(ROOT, "include")
pytestmark = pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")


def test_header_is_plain_c_and_cpp():
    hdr = os.path.join(INC, "gar.h")
    subprocess.run(["gcc", "-fsyntax-only", "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror",
                    "-x", "c", hdr], check=True)
    subprocess.run(["g++", "-fsyntax-only", "-std=c++11", "-Wall", "-Werror", "-x", "c++", hdr], check=True)


def test_c_program_matches_binding(tmp_path):
    lib_dir = os.path.dirname(gar.lib_path())
    exe = str(tmp_path / "c_abi_check")
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", INC, os.path.join(ROOT, "tests", "c_abi_check.c"),
                    "-L", lib_dir, "-lgar", f"-Wl,-rpath,{lib_dir}", "-o", exe], check=True)
    out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout.splitlines()
    cases = [(5, 1024, 3), (24, 16777216, gar.GAR_STEPS_BO), (127, 4194304, 7), (24, 1000, 22),
             (8, 100, gar.GAR_STEPS_RING)]
    for line, (P, n, steps) in zip(out, cases):
        plan = gar.gar_plan_create(P, n, "f32", "sum", steps)
        info = plan.info()
        ws, per_step, S = gar.gar_plan_bytes(plan)
        phase, partner, tx = gar.gar_plan_step(plan, 0)
        assert line == (f"P={P} S={S} K={info['K']} ws={ws} bytes={sum(per_step)} "
                        f"step0={phase},{partner},{len(tx)}")
    assert out[len(cases)].startswith("bad=-1 ") and out[len(cases)].endswith(" null=1")
    tau = gar.gar_cost_model(127, 7, 425.0, 1e-5, 1e-9, 1e-10)
    best = gar.gar_optimal_steps(127, 425.0, 1e-5, 1e-9, 1e-10)
    assert out[len(cases) + 1] == f"cost={tau:.6e} best={best}"
