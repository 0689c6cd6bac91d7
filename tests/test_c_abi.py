"""The C ABI called from a plain C program (tests/c/test_abi.c), linked
against librefcache.so and, for the GPU case, the oracle's C library."""
import os
import subprocess

import pytest

import oracle
from paper_2608_21229_gb300 import build as cbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _compile(tmp_path):
    lib = cbuild.build()
    orc = oracle.build()
    cuda = cbuild.cuda_home()
    exe = str(tmp_path / "test_abi")
    cmd = ["gcc", "-O2", "-std=c11", os.path.join(ROOT, "tests", "c", "test_abi.c"),
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(cuda, "include"),
           "-L", os.path.dirname(lib), "-lrefcache", "-L", os.path.dirname(orc), "-loracle",
           "-L", os.path.join(cuda, "lib64"), "-lcudart", "-lm", "-fopenmp",
           f"-Wl,-rpath,{os.path.dirname(lib)}:{os.path.dirname(orc)}:{os.path.join(cuda, 'lib64')}",
           "-o", exe]
    subprocess.run(cmd, check=True)
    return exe


def test_c_program_host_checks(tmp_path):
    exe = _compile(tmp_path)
    r = subprocess.run([exe, "cpu"], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    assert "cpu ok" in r.stdout


@pytest.mark.gpu
def test_c_program_build_and_step_match_oracle(tmp_path):
    exe = _compile(tmp_path)
    r = subprocess.run([exe, "gpu"], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr + r.stdout
    assert "gpu d=64 ok" in r.stdout and "gpu d=128 ok" in r.stdout
