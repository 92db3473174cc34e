"""The boundary is a plain C ABI: a C11 program compiled by gcc against
include/mosa.h links libmosa.so and calls its host-only entry points (no
GPU needed)."""
import os
import shutil
import subprocess

import pytest

from paper_2505_00315_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_c_program_uses_the_abi(tmp_path):
    lib = libbuild.build()
    exe = tmp_path / "abi_consumer"
    src = os.path.join(ROOT, "tests", "c", "abi_consumer.c")
    subprocess.run(["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-pedantic",
                    "-I", os.path.join(ROOT, "include"), src, "-o", str(exe),
                    lib, f"-Wl,-rpath,{os.path.dirname(lib)}"], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stdout + out.stderr
    assert out.stdout.count("ok ") == 7
