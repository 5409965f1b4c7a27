"""The boundary is a C ABI: a C99 program including mone.h compiles with gcc (-pedantic,
warnings as errors), links libmone.so and gets the documented answers to calls that need
no GPU."""
import os
import shutil
import subprocess

import pytest

from paper_2608_17616_gb300 import build as mbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_c_program_links_and_calls_the_library(tmp_path):
    lib = mbuild.build()
    libdir = os.path.dirname(lib)
    exe = tmp_path / "c_abi_check"
    cmd = ["gcc", "-std=c99", "-pedantic", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"),
           os.path.join(ROOT, "tests", "c_abi_check.c"), "-o", str(exe), lib, f"-Wl,-rpath,{libdir}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and "c abi ok" in r.stdout, (r.returncode, r.stdout, r.stderr)
