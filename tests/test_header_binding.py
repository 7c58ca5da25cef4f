"""The ctypes binding declares every entry point exactly as include/ee.h does
(CPU only): same parameter count, and for each parameter the same kind and
width -- a pointer, a 32-bit or 64-bit integer, a size_t, a float -- and the
same return type.  A mismatch here would pass garbage through the C ABI
without any compiler to notice it."""
import ctypes
import os
import re

import pytest

import paper_2506_02780_gb300 as E

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "ee.h")


def _strip_comments(src):
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    return re.sub(r"//[^\n]*", " ", src)


def _prototypes():
    src = _strip_comments(open(HEADER).read())
    out = {}
    for m in re.finditer(r"(ee_status|size_t|const\s+char\s*\*)\s*(ee_\w+)\s*\(([^)]*)\)\s*;", src):
        ret, name, params = m.group(1), m.group(2), m.group(3).strip()
        plist = [] if params in ("", "void") else [p.strip() for p in params.split(",")]
        out[name] = (re.sub(r"\s+", "", ret), plist)
    return out


def _kind_of_param(decl):
    """'ptr', 'i32', 'i64', 'size', 'f32' for one C parameter declaration."""
    if "*" in decl or "ee_stream_t" in decl:
        return "ptr"
    t = decl.split()
    base = t[-2] if len(t) >= 2 else t[0]
    return {"int32_t": "i32", "ee_status": "i32", "ee_verify_mode": "i32", "int64_t": "i64",
            "size_t": "size", "float": "f32"}[base]


def _kind_of_ctype(c):
    if c is ctypes.c_void_p or c is ctypes.c_char_p or (isinstance(c, type) and issubclass(c, ctypes._Pointer)):
        return "ptr"
    if c is ctypes.c_size_t:
        return "size"
    if c is ctypes.c_float:
        return "f32"
    if ctypes.sizeof(c) == 4:
        return "i32"
    if ctypes.sizeof(c) == 8:
        return "i64"
    raise AssertionError(c)


PROTOS = _prototypes()


def test_every_bound_entry_point_is_declared_and_every_declared_one_is_bound():
    assert set(PROTOS) == set(E._SIGS), (set(PROTOS) ^ set(E._SIGS))
    assert set(E.EXPORTS) == set(PROTOS)


@pytest.mark.parametrize("name", sorted(PROTOS))
def test_binding_signature_matches_header(name):
    ret, params = PROTOS[name]
    args, res = E._SIGS[name]
    assert len(args) == len(params), f"{name}: header has {len(params)} parameters, binding {len(args)}"
    for i, (decl, c) in enumerate(zip(params, args)):
        assert _kind_of_param(decl) == _kind_of_ctype(c), f"{name} parameter {i} '{decl}' bound as {c}"
    want = {"ee_status": "i32", "size_t": "size", "constchar*": "ptr"}[ret]
    assert _kind_of_ctype(res) == want, f"{name}: returns {ret}, bound as {res}"
