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


C_PROGRAM = r"""
#include <stdio.h>
#include "st.h"

#define CHECK(x) do { st_status s_ = (x); if (s_ != ST_OK) { \
  fprintf(stderr, "%s -> %s: %s\n", #x, st_status_str(s_), st_last_error(pool)); return 1; } } while (0)

static st_pool* pool;

static int dump(const char* what, st_seq s) {
  int32_t t[64]; int np = 0, nt = 0;
  CHECK(st_block_table(pool, s, t, 64, &np, &nt));
  printf("%s %d", what, nt);
  for (int i = 0; i < np; ++i) printf(" %d", t[i]);
  printf("\n");
  return 0;
}

int main(void) {
  st_config c = {0};
  c.n_layers = 2; c.n_q_heads = 8; c.n_kv_heads = 2; c.head_dim = 64; c.page_size = 16;
  c.max_seqs = 8; c.max_pages = 32; c.max_decode_branches = 8; c.max_splits = 4;
  c.n_blocks = 40; c.seed = 2608;
  if (st_pool_create(&c, NULL, NULL, NULL, -1, &pool) != ST_OK) return 2;
  st_seq main_seq, aux[4];
  CHECK(st_seq_create(pool, &main_seq));
  CHECK(st_append_kv(pool, &main_seq, 1, 37, NULL, NULL, NULL));
  CHECK(st_fork(pool, main_seq, 4, aux));
  st_seq two[2] = {aux[0], aux[2]};
  CHECK(st_append_kv(pool, two, 2, 5, NULL, NULL, NULL));
  CHECK(st_append_kv(pool, &aux[3], 1, 30, NULL, NULL, NULL));
  CHECK(st_release(pool, aux[1]));
  if (st_release(pool, aux[1]) != ST_ERR_INVALID) return 3;   /* stale handle */
  CHECK(st_merge(pool, main_seq, 20, NULL, NULL, NULL, NULL, NULL, NULL));
  if (dump("main", main_seq) || dump("a0", aux[0]) || dump("a2", aux[2]) || dump("a3", aux[3])) return 1;
  CHECK(st_release(pool, aux[2]));
  int32_t ref[40];
  CHECK(st_refcounts(pool, ref, 40));
  printf("ref");
  for (int i = 0; i < 40; ++i) printf(" %d", ref[i]);
  printf("\n");
  int32_t fl[40]; int64_t nf = 0;
  CHECK(st_free_list(pool, fl, 40, &nf));
  printf("free");
  for (int64_t i = 0; i < nf; ++i) printf(" %d", fl[i]);
  printf("\n");
  return st_pool_destroy(pool) == ST_OK ? 0 : 4;
}
"""


def test_c_program_drives_a_metadata_pool(stlib, tmp_path):
    """A plain C program built against include/st.h and linked with the
    library runs create -> append -> fork -> append (two branches, one
    copy-on-write each) -> release (and a stale second release) -> merge ->
    release on a metadata-only pool; its tables, refcounts and free list
    equal the oracle's for the same operations."""
    import shutil
    import pytest
    if not shutil.which("gcc"):
        pytest.skip("no C compiler")
    from oracle import pool as R
    src = tmp_path / "drive.c"
    src.write_text(C_PROGRAM)
    exe = tmp_path / "drive"
    libdir = os.path.dirname(stlib.LIB)
    r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src),
                        "-o", str(exe), stlib.LIB, "-Wl,-rpath," + libdir], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stderr
    got = {l.split()[0]: [int(x) for x in l.split()[1:]] for l in r.stdout.splitlines()}

    ref = R.RefPool(40, 2608)
    m = ref.create()
    ref.append([m], 37)
    aux = ref.fork(m, 4)
    ref.append([aux[0], aux[2]], 5)
    ref.append([aux[3]], 30)
    ref.release(aux[1])
    ref.merge(m, 20)
    for name, rid in (("main", m), ("a0", aux[0]), ("a2", aux[2]), ("a3", aux[3])):
        assert got[name] == [ref.seqs[rid].length] + ref.seqs[rid].table, name
    ref.release(aux[2])
    assert got["ref"] == ref.ref
    assert got["free"] == list(ref.free)
