"""The C-ABI library builds, loads without a GPU and exports exactly the entry
points include/regmem.h declares (no compute calls here)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "regmem.h")


def declared():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"REGMEM_API[^;(]*?\b(regmem_\w+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib_path():
    from paper_2609_23286_gb300 import build
    return build.build()


def test_header_declares_entry_points():
    names = declared()
    for n in ("regmem_create", "regmem_attend_frame", "regmem_admit", "regmem_reset",
              "regmem_destroy", "regmem_set_frame", "regmem_frame_attention"):
        assert n in names


def test_library_exports_every_declared_symbol(lib_path):
    from paper_2609_23286_gb300 import regmem
    for path in (lib_path, regmem.CHECKED_LIB_PATH):  # the normal and the range-checked build
        out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True,
                             text=True, check=True).stdout
        exported = sorted(set(re.findall(r"\bT (regmem_\w+)", out)))
        assert exported == declared(), path


def test_library_loads_without_gpu_and_binding_covers_header(lib_path):
    from paper_2609_23286_gb300 import regmem
    lib = regmem.load(lib_path)
    for n in declared():
        assert hasattr(lib, n)
        assert n in regmem._SIGNATURES
        assert hasattr(regmem, n), f"binding lacks {n}"
    assert regmem.status_string(regmem.ERR_CAPACITY) == "REGMEM_ERR_CAPACITY"


def test_host_side_validation_without_gpu(lib_path):
    """Argument checks that need no device: bad create arguments, calls before
    set_frame, null handles."""
    from paper_2609_23286_gb300 import regmem
    lib = regmem.load(lib_path)
    h = ctypes.c_void_p()
    assert lib.regmem_create(ctypes.byref(h), 0, 1, 64, 1) == regmem.ERR_ARG
    assert lib.regmem_create(ctypes.byref(h), 1, 1, 96, 1) == regmem.ERR_UNSUPPORTED
    assert lib.regmem_create(None, 1, 1, 64, 1) == regmem.ERR_ARG
    handle = regmem.regmem_create(2, 4, 64, 3)
    try:
        assert lib.regmem_attend_frame(handle, 0, 16, 16, 16, 16, 16) == regmem.ERR_STATE
        assert "set_frame" in regmem.regmem_last_error(handle)
        assert lib.regmem_admit(handle, 0, 1, None) == regmem.ERR_STATE
        for call in (lib.regmem_attend_admit, lib.regmem_attend_admit_shared):
            assert call(handle, 0, 16, 16, 16, 16, 16, 1, None) == regmem.ERR_STATE  # before set_frame
        assert regmem.regmem_memory_len(handle, 1) == 0
        with pytest.raises(regmem.RegmemError):
            regmem.regmem_memory_len(handle, 2)
        fd = regmem.FrameDesc(70, 5, 8, 8, 2, 4, 0.0, 0)      # 70 != 5 + 64
        assert lib.regmem_set_frame(handle, ctypes.byref(fd)) == regmem.ERR_ARG
        assert lib.regmem_reset(handle) == 0
        assert lib.regmem_set_overlap(handle, 2) == regmem.ERR_ARG
        assert lib.regmem_set_overlap(handle, 1) == 0      # takes effect at the first attend
        assert lib.regmem_join(handle) == 0                 # no side work yet
        assert lib.regmem_set_overlap(handle, 0) == 0
    finally:
        regmem.regmem_destroy(handle)
    assert lib.regmem_reset(None) == regmem.ERR_ARG
    assert lib.regmem_set_overlap(None, 1) == regmem.ERR_ARG
    assert lib.regmem_join(None) == regmem.ERR_ARG
    assert lib.regmem_attend_admit_shared(None, 0, 16, 16, 16, 16, 16, 1, None) == regmem.ERR_ARG


def _c_struct_fields(name):
    """(type, field) pairs of a typedef struct in the header, in order."""
    src = open(HEADER).read()
    body = re.search(r"typedef struct %s \{(.*?)\} %s;" % (name, name), src, re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    return re.findall(r"\b(int32_t|int64_t|double|float)\s+(\w+)\s*;", body)


@pytest.mark.parametrize("cname, pyname", [("regmem_profile", "Profile"),
                                           ("regmem_frame_desc", "FrameDesc")])
def test_binding_structs_match_header(cname, pyname):
    """The ctypes mirrors of the header's structs have the same fields, in the
    same order, with the same C types (a mismatch would read garbage)."""
    from paper_2609_23286_gb300 import regmem
    ctype = {"int32_t": ctypes.c_int32, "int64_t": ctypes.c_int64, "double": ctypes.c_double,
             "float": ctypes.c_float}
    want = [(f, ctype[t]) for t, f in _c_struct_fields(cname)]
    got = [(f, t) for f, t in getattr(regmem, pyname)._fields_]
    assert got == want
