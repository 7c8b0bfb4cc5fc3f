"""A plain C program as the library's caller (tests/c/abi_parity.c): the
header compiles as C11, the program links against libspire and the CUDA
runtime, and on a GPU its verify and draft calls match the fp64 oracle that
is compiled into it."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c", "abi_parity.c")
ORACLE = os.path.join(ROOT, "oracle", "spire_oracle.c")


def _cuda_home():
    home = os.environ.get("CUDA_HOME") or "/usr/local/cuda"
    if not os.path.isfile(os.path.join(home, "include", "cuda_runtime_api.h")):
        pytest.skip("no CUDA toolkit headers")
    return home


@pytest.fixture(scope="module")
def program(tmp_path_factory):
    if not shutil.which("gcc"):
        pytest.skip("no gcc")
    import __graft_entry__
    __graft_entry__._load_build_module().build()
    from paper_2504_06419_gb300 import _lib
    home = _cuda_home()
    libdir = next((d for d in (os.path.join(home, "lib64"), os.path.join(home, "lib"))
                   if os.path.isdir(d)), None)
    out = str(tmp_path_factory.mktemp("cabi") / "abi_parity")
    cmd = ["gcc", "-std=c11", "-O2", "-Wall", "-Wextra", "-Werror", "-o", out, SRC, ORACLE,
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(home, "include"),
           "-L", libdir, "-lcudart", _lib.LIB_PATH,
           "-Wl,-rpath," + os.path.dirname(_lib.LIB_PATH), "-Wl,-rpath," + libdir,
           "-lm", "-lpthread"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return out


def test_c_program_compiles_and_links(program):
    assert os.access(program, os.X_OK)


@pytest.mark.gpu
def test_c_program_matches_the_oracle(program):
    r = subprocess.run([program], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert r.stdout.strip().endswith("ok"), r.stdout
