"""The C ABI from a plain C11 program (tests/c_abi/estp_closed_forms.c): no Python
binding and no torch, only the CUDA runtime for device memory and the calls declared in
include/estp.h.  The program checks the whole path against closed forms (entropy of
equal, one-hot and tied logits; the importance of uniform causal attention; pooling with
equal weights; a zero length head), so it needs no oracle.

CPU: the program compiles with a C compiler in strict C11 mode and links against the
library, so the header is valid C and every entry point it calls is exported.
GPU: the program runs and every check holds."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c_abi", "estp_closed_forms.c")


def _cuda_home():
    home = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    return home if os.path.isdir(os.path.join(home, "include")) else None


def _build(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    cuda = _cuda_home()
    if cc is None or cuda is None:
        pytest.skip("no C compiler or CUDA toolkit headers")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_15592_gb300 as estp
    libdir = os.path.dirname(estp.LIB_PATH)
    cudalib = next((os.path.join(cuda, d) for d in ("lib64", "lib", "targets/sbsa-linux/lib",
                                                    "targets/x86_64-linux/lib")
                    if os.path.exists(os.path.join(cuda, d, "libcudart.so"))), None)
    if cudalib is None:
        pytest.skip("libcudart.so not found")
    exe = str(tmp_path / "estp_closed_forms")
    cmd = [cc, "-std=c11", "-O2", "-Wall", "-Wextra", "-pedantic", "-Werror", SRC,
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(cuda, "include"),
           "-L", libdir, "-lestp", "-L", cudalib, "-lcudart", "-lm",
           f"-Wl,-rpath,{libdir}", f"-Wl,-rpath,{cudalib}", "-o", exe]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    return exe


def test_c_program_compiles_and_links(tmp_path):
    assert os.path.exists(_build(tmp_path))


@pytest.mark.gpu
def test_c_program_closed_forms(tmp_path):
    exe = _build(tmp_path)
    r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert r.stdout.strip().endswith("OK")
