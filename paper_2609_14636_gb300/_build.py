"""In-tree build of libstride.so for sm_103a (nvcc, no cmake).

Each .cu under csrc/ compiles to an object in parallel; the objects link into
paper_2609_14636_gb300/libstride.so against the shared CUDA runtime.  The
build is skipped when the library is newer than every source and header.
"""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor
from pathlib import Path

PKG = Path(__file__).resolve().parent
ROOT = PKG.parent
CSRC = PKG / "csrc"
INCLUDE = ROOT / "include"
BUILD = PKG / "_build"
LIB = PKG / "libstride.so"

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden", "-Xptxas", "-v",
              "-I", str(INCLUDE), "-I", str(CSRC)]


def nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    return cand


def sources() -> list[Path]:
    return sorted(CSRC.glob("*.cu"))


def _deps() -> list[Path]:
    return sources() + sorted(CSRC.glob("*.cuh")) + sorted(CSRC.glob("*.h")) + sorted(INCLUDE.glob("*.h"))


def up_to_date() -> bool:
    if not LIB.exists():
        return False
    t = LIB.stat().st_mtime
    return all(p.stat().st_mtime <= t for p in _deps())


def build(force: bool = False, verbose: bool = False, defines: tuple = (), lib: Path | None = None,
          build_dir: Path | None = None) -> Path:
    """Compile and link.  `defines` adds -D flags (tuning knobs of the
    kernels); `lib`/`build_dir` redirect the output (default: in-tree)."""
    out_lib = LIB if lib is None else Path(lib)
    bdir = BUILD if build_dir is None else Path(build_dir)
    if not force and lib is None and not defines and up_to_date():
        return LIB
    bdir.mkdir(parents=True, exist_ok=True)
    objs = []

    def compile_one(src: Path) -> tuple[Path, str]:
        obj = bdir / (src.stem + ".o")
        cmd = [nvcc(), *ARCH, *NVCC_FLAGS, *[f"-D{d}" for d in defines], "-c", str(src), "-o", str(obj)]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src.name}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stderr

    with ThreadPoolExecutor(max_workers=min(8, len(sources()))) as ex:
        results = list(ex.map(compile_one, sources()))
    log = []
    for obj, err in results:
        objs.append(obj)
        log.append(err)
    (bdir / "ptxas.log").write_text("\n".join(log))
    tmp = out_lib.with_name(out_lib.name + f".tmp{os.getpid()}")
    cmd = [nvcc(), *ARCH, "-shared", "-cudart", "shared", "-o", str(tmp), *map(str, objs)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, out_lib)
    if verbose:
        print("\n".join(log))
    return out_lib


if __name__ == "__main__":
    build(force=True, verbose=True)
    print(LIB)
