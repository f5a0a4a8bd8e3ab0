"""The C-ABI library builds, loads and exports every symbol include/sq.h
declares; the Python binding carries the same names.  No GPU needed: only
host-side calls that touch no device are made."""
import ctypes
import os
import re

import pytest

import paper_2602_22603_gb300 as sq
from paper_2602_22603_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sq.h")


def declared_functions():
    text = open(HEADER).read()
    return re.findall(r"^SQ_API\s+[\w\s\*]*?\b(sq_\w+)\s*\(", text, flags=re.M)


@pytest.fixture(scope="module")
def libsq():
    build.build_libsq()
    return ctypes.CDLL(build.LIBSQ)


def test_header_declares_the_six_calls_and_helpers():
    names = declared_functions()
    for call in ("sq_cache_create", "sq_append_kv", "sq_fork_aux", "sq_decode_attention",
                 "sq_evict_spans", "sq_release"):
        assert call in names
    assert len(names) == len(set(names))


def test_library_exports_every_declared_symbol(libsq):
    for name in declared_functions():
        assert hasattr(libsq, name), name


def test_binding_has_the_same_names():
    for name in declared_functions():
        assert callable(getattr(sq, name)), name


def test_host_only_calls(libsq):
    assert sq.strerror(sq.SQ_ERR_NO_PAGES) == "SQ_ERR_NO_PAGES"
    cfg = sq.make_config(32, 32, 8, 128, 64, 100)
    assert sq.sq_pool_bytes(cfg) == 32 * 100 * 2 * 8 * 64 * 128 * 2
    # geometries the kernels do not handle give 0 bytes
    assert sq.sq_pool_bytes(sq.make_config(1, 8, 2, 96, 16, 10)) == 0   # head dim 96
    assert sq.sq_pool_bytes(sq.make_config(1, 8, 2, 64, 12, 10)) == 0   # page size 12
    assert sq.sq_pool_bytes(sq.make_config(1, 64, 2, 64, 16, 10)) == 0  # group of 32
    assert sq.sq_pool_bytes(sq.make_config(1, 6, 4, 64, 16, 10)) == 0   # Hq % Hkv != 0


def test_null_cache_is_rejected(libsq):
    out = ctypes.c_int32()
    assert libsq.sq_seq_new(None, ctypes.byref(out)) == sq.SQ_ERR_BAD_HANDLE
    assert libsq.sq_cache_destroy(None) == sq.SQ_ERR_BAD_HANDLE


def test_binding_fails_loudly_without_the_library():
    # a fresh interpreter whose package points at a library that does not
    # exist: the first call raises instead of falling back to anything
    import subprocess
    import sys
    code = (
        "import paper_2602_22603_gb300 as sq\n"
        "sq.LIB_PATH = '/nonexistent/libsq.so'\n"
        "try:\n"
        "    sq.lib()\n"
        "except RuntimeError as e:\n"
        "    print('raised', 'libsq.so not found' in str(e))\n"
        "else:\n"
        "    print('loaded')\n")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300,
                       cwd=os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    assert r.stdout.strip() == "raised True", r.stdout + r.stderr


_CTYPES = {"int32_t": ctypes.c_int32, "int64_t": ctypes.c_int64, "uint32_t": ctypes.c_uint32,
           "float": ctypes.c_float, "void*": ctypes.c_void_p}


def header_struct(name):
    """Fields of `typedef struct { ... } name;` in include/sq.h, as (type, field)
    pairs in declaration order (one declaration per line; comments dropped)."""
    text = re.sub(r"/\*.*?\*/", " ", open(HEADER).read(), flags=re.S)
    m = re.search(r"typedef\s+struct\s*\{([^}]*)\}\s*" + name + r"\s*;", text)
    assert m, name
    out = []
    for decl in m.group(1).split(";"):
        decl = " ".join(decl.split())
        if not decl:
            continue
        mt = re.fullmatch(r"(\w+)\s*(\*?)\s*(\w+)", decl)
        assert mt, decl
        out.append((mt.group(1) + mt.group(2), mt.group(3)))
    return out


@pytest.mark.parametrize("c_name,py_struct", [("sq_config", sq.sq_config), ("sq_span", sq.sq_span),
                                               ("sq_stats_t", sq.sq_stats_t)])
def test_binding_structs_match_the_header(c_name, py_struct):
    """The binding's ctypes structures have the header's fields, in order and
    of the same types, so that a call that fills one (sq_stats copies the
    whole struct) never writes past the caller's buffer."""
    fields = header_struct(c_name)
    assert [f for _, f in fields] == [n for n, _ in py_struct._fields_]
    # the same field types in the same order give the same layout: ctypes lays
    # a Structure out by the platform's C rules
    for (ctype, fname), (_, pytype) in zip(fields, py_struct._fields_):
        assert ctypes.sizeof(_CTYPES[ctype]) == ctypes.sizeof(pytype), fname
        assert ctypes.alignment(_CTYPES[ctype]) == ctypes.alignment(pytype), fname


def _c_kind(decl):
    """Class of a C parameter or return type: ptr, i32, i64, f32 or size."""
    decl = " ".join(decl.replace("const", " ").split())
    if "*" in decl:
        return "ptr"
    base = decl.split()[0]
    return {"int": "i32", "int32_t": "i32", "sq_seq": "i32", "int64_t": "i64", "float": "f32",
            "size_t": "size"}[base]


def _py_kind(t):
    if t in (ctypes.c_void_p, ctypes.c_char_p) or hasattr(t, "_type_") and issubclass(
            t, ctypes._Pointer):
        return "ptr"
    if t in (ctypes.c_int32, ctypes.c_int):
        return "i32"
    if t is ctypes.c_int64:
        return "i64"
    if t is ctypes.c_float:
        return "f32"
    if t is ctypes.c_size_t:
        return "size"
    raise AssertionError(t)


def header_prototypes():
    text = re.sub(r"/\*.*?\*/", " ", open(HEADER).read(), flags=re.S)
    out = {}
    for m in re.finditer(r"^SQ_API\s+([\w\s\*]*?)\b(sq_\w+)\s*\(([^)]*)\)\s*;", text, flags=re.M):
        params = [p.strip() for p in m.group(3).split(",") if p.strip() and p.strip() != "void"]
        # drop each parameter's name: the type is everything before the last word
        types = [re.sub(r"\b\w+\s*$", "", p).strip() or p for p in params]
        out[m.group(2)] = (m.group(1).strip(), types)
    return out


def test_binding_signatures_match_the_header():
    """Every declared function has the binding's argument count, and each
    argument and the result the same class (pointer, 32/64-bit integer,
    float, size_t), so that ctypes marshals the call as C expects."""
    protos = header_prototypes()
    assert set(protos) == set(declared_functions())
    for name, (ret, params) in protos.items():
        res, args = sq._SIGS[name]
        assert len(args) == len(params), name
        assert _py_kind(res) == _c_kind(ret), name
        for i, (p, a) in enumerate(zip(params, args)):
            assert _c_kind(p) == _py_kind(a), (name, i, p)
