"""C-ABI checks that need no GPU: the library builds, loads and exports every symbol
declared in include/*.h, and host-side argument checks reject bad calls before any
launch (no compute call is made here)."""

import ctypes
import glob
import os
import re
import subprocess

import pytest

from paper_2608_12913_gb300 import build as dcd_build
from paper_2608_12913_gb300 import dcd

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w\s\*]*?\b(dcd_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    dcd_build.build()
    return dcd.load()


def test_header_declares_the_entry_points():
    names = declared_functions()
    for required in ("dcd_verify_greedy", "dcd_verify_sample", "dcd_workspace_bytes", "dcd_score_rows",
                     "dcd_tree_walk", "dcd_get_device_error", "dcd_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    names = declared_functions()
    out = subprocess.run(["nm", "-D", "--defined-only", dcd_build.LIB], capture_output=True, text=True, check=True)
    exported = {line.split()[-1] for line in out.stdout.splitlines() if line.strip()}
    missing = [n for n in names if n not in exported]
    assert not missing, f"declared but not exported: {missing}"
    for n in names:
        assert hasattr(lib, n)


def test_library_is_built_for_sm_103a(lib):
    out = subprocess.run(["cuobjdump", "--list-elf", dcd_build.LIB], capture_output=True, text=True)
    if out.returncode != 0:
        pytest.skip("cuobjdump unavailable")
    assert "sm_103a" in out.stdout


def test_status_strings_and_version(lib):
    assert dcd.status_string(0) == "ok"
    assert "argument" in dcd.status_string(-1)
    assert "workspace" in dcd.status_string(-7)
    assert dcd.version() >= 10000


def test_workspace_bytes(lib):
    n = dcd.workspace_bytes(32, 60, 128256)
    assert n >= 256 + 32 * 60 * 32 and n % 256 == 0
    bad = dcd.make_shape(1, 0, 10, 0)
    assert lib.dcd_workspace_bytes(ctypes.byref(bad)) == 0
    bad = dcd.make_shape(1, 4, 10, 5)
    assert lib.dcd_workspace_bytes(ctypes.byref(bad)) == 0
    bad = dcd.make_shape(1, 4, 10, 0, ld=9)
    assert lib.dcd_workspace_bytes(ctypes.byref(bad)) == 0


def _fake(addr):
    return ctypes.c_void_p(addr)


def test_host_checks_reject_before_launch(lib):
    """Invalid calls return a negative status; the fake pointers are never dereferenced."""
    P = _fake(0x10000)
    sh = dcd.make_shape(2, 4, 100, dcd.DCD_BF16)
    ws_ok = _fake(0x100000)
    base = [P, P, P, P, P, None, P, P, P, None, None, None]
    # null shape
    assert lib.dcd_verify_greedy(None, *base, ws_ok, 1 << 20, None) == -1
    # null logits
    assert lib.dcd_verify_greedy(ctypes.byref(sh), None, *base[1:], ws_ok, 1 << 20, None) == -1
    # misaligned workspace / too small
    assert lib.dcd_verify_greedy(ctypes.byref(sh), *base, _fake(0x100010), 1 << 20, None) == -7
    assert lib.dcd_verify_greedy(ctypes.byref(sh), *base, ws_ok, 64, None) == -7
    # unsupported tree size
    big = dcd.make_shape(1, 2000, 100, dcd.DCD_BF16)
    assert lib.dcd_verify_greedy(ctypes.byref(big), *base, ws_ok, 1 << 30, None) == -3
    # sampled call without q or temperature
    assert lib.dcd_verify_sample(ctypes.byref(sh), P, P, None, P, P, P, None, P, 0, 0, P, P, P, None, None, None,
                                 None, ws_ok, 1 << 20, None) == -1
    assert lib.dcd_verify_sample(ctypes.byref(sh), P, P, P, P, P, P, None, None, 0, 0, P, P, P, None, None, None,
                                 None, ws_ok, 1 << 20, None) == -1
    # row stride shorter than the vocabulary
    bad = dcd.make_shape(2, 4, 100, dcd.DCD_BF16, ld=50)
    assert lib.dcd_verify_greedy(ctypes.byref(bad), *base, ws_ok, 1 << 20, None) == -1
    # invalid forced ring depth
    assert lib.dcd_score_rows_ex(ctypes.byref(sh), P, P, None, P, P, P, None, None, 0, 0, None, None, None, ws_ok,
                                 1 << 20, None, 1, 0, 0) == -1
    # negative poll limit
    assert lib.dcd_score_rows_ex(ctypes.byref(sh), P, P, None, P, P, P, None, None, 0, 0, None, None, None, ws_ok,
                                 1 << 20, None, 0, 0, -1) == -1
    # empty batch is a no-op
    empty = dcd.make_shape(0, 4, 100, dcd.DCD_BF16)
    assert lib.dcd_verify_greedy(ctypes.byref(empty), *base, ws_ok, 1 << 20, None) == 0
    # q staging: null pointers, a short row stride, an empty batch
    assert lib.dcd_upload_q_rows(ctypes.byref(sh), None, P, P, P, None) == -1
    assert lib.dcd_upload_q_rows(ctypes.byref(sh), P, P, None, P, None) == -1
    short = dcd.make_shape(2, 4, 100, dcd.DCD_BF16, ldq=50)
    assert lib.dcd_upload_q_rows(ctypes.byref(short), P, P, P, P, None) == -1
    assert lib.dcd_upload_q_rows(ctypes.byref(empty), P, P, P, P, None) == 0


def test_binding_refuses_cpu_tensors():
    import torch
    z = torch.zeros((6, 10))
    t = torch.zeros((1, 6), dtype=torch.int32)
    with pytest.raises(ValueError, match="CUDA"):
        dcd.dcd_verify_greedy(z, z, t, t, torch.zeros(1))


def test_fused_workspace_and_host_checks(lib):
    sh = dcd.make_shape(64, 60, 128256, dcd.DCD_BF16)
    n = lib.dcd_fused_workspace_bytes(ctypes.byref(sh))
    nvt = (128256 + 255) // 256
    assert n >= 256 + 3840 * (96 + 16) + 3840 * nvt * 16 and n % 256 == 0
    f32 = dcd.make_shape(2, 4, 100, dcd.DCD_F32)
    assert lib.dcd_fused_workspace_bytes(ctypes.byref(f32)) == 0
    P = _fake(0x10000)
    sh = dcd.make_shape(2, 4, 100, dcd.DCD_BF16)
    ws = _fake(0x100000)
    args = [P, 64, P, P, 64, P, P, P, P, P, P, P, None, None, None]
    # hidden size not a multiple of 8, misaligned matrix, small workspace: rejected before launch
    bad = list(args)
    bad[1] = 60
    assert lib.dcd_verify_fused_lmhead(ctypes.byref(sh), *bad, ws, 1 << 24, None) == -1
    bad = list(args)
    bad[0] = _fake(0x10008)
    assert lib.dcd_verify_fused_lmhead(ctypes.byref(sh), *bad, ws, 1 << 24, None) == -1
    assert lib.dcd_verify_fused_lmhead(ctypes.byref(sh), *args, ws, 64, None) == -7
    empty = dcd.make_shape(0, 4, 100, dcd.DCD_BF16)
    assert lib.dcd_verify_fused_lmhead(ctypes.byref(empty), *args, ws, 1 << 24, None) == 0


def test_diagnostics_workspace_and_host_checks(lib):
    sh = dcd.make_shape(32, 60, 128256, dcd.DCD_BF16)
    n = lib.dcd_diagnostics_workspace_bytes(ctypes.byref(sh))
    assert n == (1920 * ((128256 + 2047) // 2048) * 48 + 255) // 256 * 256
    bad = dcd.make_shape(2, 4, 100, dcd.DCD_BF16, ld=50)
    assert lib.dcd_diagnostics_workspace_bytes(ctypes.byref(bad)) == 0
    P = _fake(0x10000)
    ws = _fake(0x100000)
    sh = dcd.make_shape(2, 4, 100, dcd.DCD_BF16)
    # null logits or output, sibling flags, q with a short stride, bad workspace: rejected before launch
    assert lib.dcd_row_diagnostics(ctypes.byref(sh), None, P, None, None, None, None, None, None, P, ws, 1 << 20, None) == -1
    assert lib.dcd_row_diagnostics(ctypes.byref(sh), P, P, None, None, None, None, None, None, None, ws, 1 << 20, None) == -1
    flagged = dcd.make_shape(2, 4, 100, dcd.DCD_BF16, flags=dcd.DCD_SIBLINGS_DISTINCT)
    assert lib.dcd_row_diagnostics(ctypes.byref(flagged), P, P, None, None, None, None, None, None, P, ws, 1 << 20, None) == -1
    short_q = dcd.make_shape(2, 4, 100, dcd.DCD_BF16, ldq=99)
    assert lib.dcd_row_diagnostics(ctypes.byref(short_q), P, P, P, None, None, None, None, None, P, ws, 1 << 20, None) == -1
    assert lib.dcd_row_diagnostics(ctypes.byref(sh), P, P, None, None, None, None, None, None, P, _fake(0x100010), 1 << 20, None) == -7
    assert lib.dcd_row_diagnostics(ctypes.byref(sh), P, P, None, None, None, None, None, None, P, ws, 16, None) == -7
    empty = dcd.make_shape(0, 4, 100, dcd.DCD_BF16)
    assert lib.dcd_row_diagnostics(ctypes.byref(empty), P, P, None, None, None, None, None, None, P, ws, 1 << 20, None) == 0
    # cd_lse without alpha (the lemma needs both)
    assert lib.dcd_row_diagnostics(ctypes.byref(sh), P, P, None, None, P, None, None, None, P, ws, 1 << 20, None) == -1


def test_sampled_row_ranges_merges_adjacent_sequences():
    import torch
    from paper_2608_12913_gb300 import dcd
    t = torch.tensor([0.0, 1.0, 0.7, 0.0, 2.0])
    assert dcd.sampled_row_ranges(t, 4) == [(4, 12), (16, 20)]
    assert dcd.sampled_row_ranges(torch.zeros(3), 4) == []
    # with the tree: only nodes that have a child (node 0 of every sequence; node 1 in sequence 1;
    # node 2 in sequences 2 and 4)
    par = torch.tensor([[-1, 0, 0, 0], [-1, 0, 1, 1], [-1, 0, 0, 2], [-1, 0, 1, 2], [-1, 0, 0, 2]])
    assert dcd.sampled_row_ranges(t, 4, par) == [(4, 6), (8, 9), (10, 11), (16, 17), (18, 19)]


def test_header_is_plain_c(tmp_path):
    """include/dcd.h is a C header: a C99 translation unit using it compiles with -pedantic."""
    import shutil
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "use_dcd.c"
    src.write_text('#include "dcd.h"\n'
                   "int main(void) {\n"
                   "  dcd_shape s = {1, 6, 32000, DCD_F32, 0, 32000, 32000};\n"
                   "  return dcd_workspace_bytes(&s) == 0;\n"
                   "}\n")
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", inc, "-fsyntax-only",
                        str(src)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
