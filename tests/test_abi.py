"""The C-ABI library loads and exports every entry point include/st.h declares
(no compute call: these run without a GPU)."""
import ctypes
import os
import re
import subprocess

from conftest import ROOT


def _declared():
    src = open(os.path.join(ROOT, "include", "st.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"ST_API\s+[\w\s\*]*?\b(st_\w+)\s*\(", src)))


def test_header_declares_the_method_calls():
    names = _declared()
    for n in ["st_fork", "st_append_kv", "st_decode_attn", "st_merge", "st_release",
              "st_pool_create", "st_workspace_bytes", "st_sync"]:
        assert n in names


def test_library_exports_every_declared_symbol(stlib):
    lib = ctypes.CDLL(stlib.LIB)
    for name in _declared():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", stlib.LIB], capture_output=True, text=True).stdout
    exported = {l.split()[-1] for l in out.splitlines() if " T " in l}
    assert set(_declared()) <= exported
    # nothing but the C ABI leaks out of the library
    assert all(s.startswith("st_") or s.startswith("_") for s in exported), exported


def test_workspace_bytes_and_config_validation(stlib):
    L = stlib.lib()
    good = stlib.StConfig(n_layers=2, n_q_heads=8, n_kv_heads=2, head_dim=64, page_size=16,
                          max_seqs=8, max_pages=64, max_decode_branches=5, max_splits=8,
                          n_blocks=128, seed=0)
    ws = L.st_workspace_bytes(ctypes.byref(good))
    assert ws > 5 * 2 * 8 * 8 * 65 * 4 and ws % 256 == 0
    for field, val in [("page_size", 32), ("head_dim", 96), ("n_kv_heads", 3), ("max_splits", 1),
                       ("max_splits", 33), ("n_blocks", 0), ("n_layers", 0)]:
        bad = stlib.StConfig.from_buffer_copy(good)
        setattr(bad, field, val)
        assert L.st_workspace_bytes(ctypes.byref(bad)) == 0, field


def test_status_strings(stlib):
    L = stlib.lib()
    for s in range(6):
        assert L.st_status_str(s)


def test_header_is_plain_c(tmp_path):
    """include/st.h is a C header (no C++ in the signatures): a C99 program
    that takes the address of every declared entry point compiles warning-free,
    and so does the same file as C++."""
    import shutil
    import pytest
    if not shutil.which("gcc"):
        pytest.skip("no C compiler")
    names = _declared()
    src = tmp_path / "use_st.c"
    src.write_text('#include "st.h"\n#include <stdio.h>\ntypedef void (*fn_t)(void);\nint main(void) {\n'
                   "  fn_t fns[] = {" + ", ".join(f"(fn_t)&{n}" for n in names) + "};\n"
                   '  printf("%d\\n", (int)(sizeof fns / sizeof fns[0]));\n  return 0;\n}\n')
    inc = os.path.join(ROOT, "include")
    for cmd in (["gcc", "-std=c99", "-Wall", "-Wextra", "-Wpedantic", "-Werror", "-fsyntax-only"],
                ["g++", "-std=c++17", "-Wall", "-Werror", "-fsyntax-only", "-x", "c++"]):
        r = subprocess.run(cmd + ["-I", inc, str(src)], capture_output=True, text=True)
        assert r.returncode == 0, r.stderr
