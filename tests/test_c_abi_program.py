"""A C program (tests/c/abi_smoke.c) calls libstride.so through
include/stride.h alone: it builds and links on the CPU, and on a GPU it
scores uniform-logit rows, checks the closed-form log-probs, the stop rule
and the loss, makes one restart choice, runs three decode steps, and sees
one column past the vocabulary limit refused."""
import shutil
import subprocess
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]


def _cuda_home() -> Path:
    nvcc = shutil.which("nvcc")
    return Path(nvcc).resolve().parents[1] if nvcc else Path("/usr/local/cuda")


def build_program(out: Path) -> Path:
    from paper_2609_14636_gb300 import _build

    lib = _build.build()
    cuda = _cuda_home()
    cmd = ["gcc", "-std=c99", "-Wall", "-Werror", "-I", str(ROOT / "include"), "-I", str(cuda / "include"),
           str(ROOT / "tests" / "c" / "abi_smoke.c"), "-L", str(lib.parent), "-lstride",
           "-L", str(cuda / "lib64"), "-lcudart", "-lm", f"-Wl,-rpath,{lib.parent}", f"-Wl,-rpath,{cuda / 'lib64'}",
           "-o", str(out)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return out


def test_c_program_builds(tmp_path):
    assert build_program(tmp_path / "abi_smoke").exists()


@pytest.mark.gpu
def test_c_program_runs(tmp_path):
    exe = build_program(tmp_path / "abi_smoke")
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "abi_smoke ok" in r.stdout
