"""The C ABI from a plain C99 program: tests/c_client/lookup_client.c, built with gcc against include/lacache.h,
liblacache.so and the CUDA runtime, runs a lookup of exact duplicates, rejections and misses end to end."""
import os
import subprocess

import pytest

from paper_2608_01718_gb300 import build

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def test_c_client_looks_up_through_the_c_abi(tmp_path):
    lib = build.build()
    exe = str(tmp_path / "lookup_client")
    libdir = os.path.dirname(lib)
    cmd = ["gcc", "-std=c99", "-O2", "-Wall", "-Wextra", "-Werror", os.path.join(HERE, "c_client", "lookup_client.c"),
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(CUDA, "include"), "-L", libdir, "-llacache",
           "-L", os.path.join(CUDA, "lib64"), "-lcudart", "-lm", f"-Wl,-rpath,{libdir}",
           f"-Wl,-rpath,{os.path.join(CUDA, 'lib64')}", "-o", exe]
    res = subprocess.run(cmd, capture_output=True, text=True)
    assert res.returncode == 0, res.stderr
    run = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert run.returncode == 0 and run.stdout.strip() == "ok", run.stderr + run.stdout
