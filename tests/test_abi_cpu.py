"""The C-ABI library builds, loads and exports what include/sparoa.h declares (CPU only).

No compute runs here: only host-side entry points that touch no GPU
(status strings, occupancy sizing) and the error path of sparoa_create on a
machine without a usable device.
"""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sparoa.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2511_19457_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(sparoa_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for want in ["sparoa_op_stats", "sparoa_gemm", "sparoa_conv2d", "sparoa_run_graph",
                 "sparoa_create", "sparoa_destroy", "sparoa_status_str"]:
        assert want in names


def test_every_declared_symbol_is_exported(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_binding_covers_every_symbol():
    from paper_2511_19457_gb300 import sparoa
    assert sorted(sparoa.EXPORTED) == _declared()


def test_struct_layouts_match_header(tmp_path):
    """sizeof/offsetof in C (gcc on the header) equal the ctypes mirror."""
    from paper_2511_19457_gb300 import sparoa as sp
    prog = tmp_path / "layout.c"
    prog.write_text("""
#include <stdio.h>
#include <stddef.h>
#include "sparoa.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu %zu\\n", sizeof(sparoa_thresholds), sizeof(sparoa_stats),
         sizeof(sparoa_occupancy), sizeof(sparoa_epilogue), sizeof(sparoa_op), sizeof(sparoa_record));
  printf("%zu %zu %zu %zu\\n", offsetof(sparoa_op, weight), offsetof(sparoa_op, thr),
         offsetof(sparoa_stats, path), offsetof(sparoa_record, out_occ));
  return 0;
}
""")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(prog), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()
    sizes = [int(v) for v in out]
    assert sizes[:6] == [ctypes.sizeof(sp.Thresholds), ctypes.sizeof(sp.Stats),
                         ctypes.sizeof(sp.Occupancy), ctypes.sizeof(sp.Epilogue),
                         ctypes.sizeof(sp.Op), ctypes.sizeof(sp.Record)]
    assert sizes[6:] == [sp.Op.weight.offset, sp.Op.thr.offset, sp.Stats.path.offset,
                         sp.Record.out_occ.offset]


def test_host_only_entry_points(lib):
    lib.sparoa_status_str.restype = ctypes.c_char_p
    assert lib.sparoa_status_str(0) == b"ok"
    assert lib.sparoa_status_str(5) == b"device wait timed out"
    lib.sparoa_occupancy_bytes.restype = ctypes.c_uint64
    lib.sparoa_occupancy_bytes.argtypes = [ctypes.c_int64, ctypes.c_int64]
    # [25088, 64]: 16 + 64*4 + 1*4 (+pad) + 25088*8 + 196*2*4, 16-byte aligned pieces
    assert lib.sparoa_occupancy_bytes(25088, 64) == 16 + 256 + 16 + 25088 * 8 + 196 * 2 * 4
    assert lib.sparoa_occupancy_bytes(-1, 4) == 0


def test_create_rejects_bad_arguments(lib):
    lib.sparoa_create.restype = ctypes.c_int
    lib.sparoa_create.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p]
    assert lib.sparoa_create(None, 0, None) == 1          # INVALID_ARG
    h = ctypes.c_void_p()
    st = lib.sparoa_create(ctypes.byref(h), -1, None)
    assert st in (1, 4)                                  # bad device, or no CUDA device at all
    assert not h.value
