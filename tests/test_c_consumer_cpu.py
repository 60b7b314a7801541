"""The C ABI from C: tests/c/consumer.c includes include/asap_moe.h, is
compiled as strict C11 with gcc, links libasap_moe.so and runs the pure-host
calls (config checks, workspace sizing, argument rejection) without a GPU."""
import os
import shutil
import subprocess

import pytest

from paper_2606_22541_gb300 import build as build_mod

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_c_program_uses_the_header_and_library(tmp_path):
    lib = build_mod.build()
    libdir = os.path.dirname(lib)
    exe = tmp_path / "consumer"
    cmd = ["gcc", "-std=c11", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", os.path.join(ROOT, "include"),
           os.path.join(ROOT, "tests", "c", "consumer.c"), "-o", str(exe), "-L", libdir, "-l:libasap_moe.so",
           "-Wl,-rpath," + libdir]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "0 failed checks" in r.stdout
