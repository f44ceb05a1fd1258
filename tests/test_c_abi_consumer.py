"""A plain C99 consumer of libvcs (tests/c_abi/consumer.c): include/vcs.h compiles as strict C
and the calls that need no GPU (version, status strings, workspace sizes, host argument errors)
answer from C through the shared library (CPU only)."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2607_11185_gb300")
LIB = os.path.join(PKG, "libvcs.so")


def test_c_consumer(tmp_path):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    if not os.path.exists(LIB):
        from paper_2607_11185_gb300 import build
        build.build()
    exe = str(tmp_path / "consumer")
    cmd = [gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", os.path.join(ROOT, "include"),
           os.path.join(ROOT, "tests", "c_abi", "consumer.c"), "-L", PKG, "-lvcs", f"-Wl,-rpath,{PKG}", "-o", exe]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert r.stdout.count("ok ") == 8, r.stdout
