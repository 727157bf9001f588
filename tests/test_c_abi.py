"""A plain C program linked to libavits.so calls the C ABI (temporal score
and fused selection) and checks the results against host computations of its
own: the boundary works without the Python binding."""
import os
import shutil
import subprocess

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def test_c_caller(tmp_path):
    import paper_2608_17995_gb300 as av
    lib = av.build()
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    exe = str(tmp_path / "abi_caller")
    libdir = os.path.dirname(lib)
    subprocess.check_call([nvcc, "-x", "c", os.path.join(HERE, "c", "abi_caller.c"),
                           "-I" + os.path.join(ROOT, "include"), "-L" + libdir, "-lavits",
                           "-Xlinker", "-rpath=" + libdir, "-lm", "-o", exe])
    r = subprocess.run([exe], stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == "ok"
