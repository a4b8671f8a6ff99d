"""The C-ABI library builds, loads and exports every symbol include/stride.h
declares.  No compute call is made (CPU only)."""
import ctypes
import re
import subprocess
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]


def declared_symbols():
    src = "\n".join(p.read_text() for p in sorted((ROOT / "include").glob("*.h")))
    return sorted(set(re.findall(r"STRIDE_API\s+[\w\s\*]+?\b(stride_\w+)\s*\(", src)))


def test_header_declares_entry_points():
    names = declared_symbols()
    for must in ("stride_score_batch", "stride_score_step", "stride_select_restart"):
        assert must in names


def test_library_exports_declared_symbols():
    from paper_2609_14636_gb300 import _build

    lib = _build.build()
    handle = ctypes.CDLL(str(lib))
    for name in declared_symbols():
        assert hasattr(handle, name), f"{name} is declared but not exported"
    nm = subprocess.run(["nm", "-D", "--defined-only", str(lib)], capture_output=True, text=True, check=True).stdout
    exported = {l.split()[-1] for l in nm.splitlines() if " T " in l}
    public = {s for s in exported if s.startswith("stride_")}
    assert public == set(declared_symbols()), (public, declared_symbols())


def test_host_only_calls():
    import paper_2609_14636_gb300 as stride

    assert stride.stride_abi_version() == 3
    assert stride.stride_score_batch_workspace_size(0) == 0
    assert stride.stride_score_batch_workspace_size(1000) >= 1000 * 68
    assert "INVALID_ARG" in stride.stride_status_string(1)


def test_header_compiles_as_c():
    pytest.importorskip("subprocess")
    r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-fsyntax-only", "-x", "c", "-I", str(ROOT / "include"), "-"],
                       input='#include "stride.h"\n#include "stride_selftest.h"\nint main(void){return sizeof(stride_scan_state)==80 && sizeof(stride_turn_stats)==40 ? 0 : 1;}\n',
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_max_vocab_constant_matches_header():
    import paper_2609_14636_gb300 as stride

    src = (ROOT / "include" / "stride.h").read_text()
    m = re.search(r"#define STRIDE_MAX_VOCAB \(1 << (\d+)\)", src)
    assert m and stride.MAX_VOCAB == 1 << int(m.group(1)) == 1 << 30
