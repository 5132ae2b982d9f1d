"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every symbol include/lipcache.h declares, and rejects bad arguments before
touching a device."""
import ctypes as C
import os
import re
import subprocess

import pytest

from conftest import ROOT


@pytest.fixture(scope="module")
def lib():
    from paper_2608_13144_gb300.build import build
    build()
    from paper_2608_13144_gb300 import _lib
    return _lib.load()


def _declared_functions():
    text = open(os.path.join(ROOT, "include", "lipcache.h")).read()
    return sorted(set(re.findall(r"^\s*(?:lipcache_status|void|int64_t|const char\*)\s+(lipcache_\w+)\s*\(", text,
                                 re.M)))


def test_exports_every_declared_symbol(lib):
    from paper_2608_13144_gb300 import _lib
    declared = _declared_functions()
    assert declared, "no declarations parsed"
    assert sorted(_lib.EXPORTS) == declared
    out = subprocess.run(["nm", "-D", "--defined-only", _lib.LIB_PATH], capture_output=True, text=True).stdout
    exported = sorted(set(re.findall(r" T (lipcache_\w+)", out)))
    assert exported == declared
    for name in declared:
        assert hasattr(lib, name)


def test_no_gpu_runtime_dependency(lib):
    from paper_2608_13144_gb300 import _lib
    out = subprocess.run(["ldd", _lib.LIB_PATH], capture_output=True, text=True).stdout
    assert "libcuda.so" not in out and "libcudart" not in out


@pytest.mark.parametrize("args", [(0, 10, 100, 0), (16, 1, 100, 0), (16, 10, 0, 0), (16, 10, 100, 7),
                                  (2000, 10, 100, 0), (16, 5000, 100, 0), (16, 10, 1 << 40, 0)])
def test_create_rejects_bad_arguments(lib, args):
    h = C.c_void_p()
    st = lib.lipcache_create(*args, C.byref(h))
    assert st == 1  # E_INVALID, decided before any CUDA call
    assert not h.value
    assert lib.lipcache_last_error()


def test_null_handle_calls(lib):
    assert lib.lipcache_size(None) == 0
    lib.lipcache_destroy(None)
    assert lib.lipcache_set_head(None, None, None, None, None) == 1
    assert lib.lipcache_probe(None, None, 0, None, None, None, None) == 1
    assert lib.lipcache_insert(None, None, 0, None, 0, None, None, None, None) == 1
    n = C.c_int64(7)
    assert lib.lipcache_probe_writeback(None, None, 0, None, 0, None, None, None, None, C.byref(n), None) == 1
    assert n.value == 0
    nh, nc = C.c_int64(7), C.c_int64(7)
    assert lib.lipcache_consistency(None, None, 0, None, None, C.byref(nh), C.byref(nc), None) == 1
    assert nh.value == 0 and nc.value == 0
    ns = C.c_int64(7)
    assert lib.lipcache_insert_select(None, None, 0, None, 0, 1, 0, 0, None, None, C.byref(ns), None) == 1
    assert ns.value == 0
    assert lib.lipcache_set_radius_policy(None, 1, 1.0, None, None) == 1
    assert lib.lipcache_set_debug(None, 0) == 1
    assert lib.lipcache_read_entries(None, 0, 0, None, None, None, None, None) == 1
    assert lib.lipcache_read_head(None, None, None, None) == 1


def test_create_without_gpu_fails_cleanly(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    h = C.c_void_p()
    st = lib.lipcache_create(16, 10, 100, 0, C.byref(h))
    assert st in (6, 7)  # E_CUDA / E_NOMEM from the runtime
    assert not h.value


def test_numerics_constants():
    """The slack constants are bounded as the design states: the recheck
    deflation is far inside the 1e-5 decision band, and the screen slack is
    of order 2^-8 for the feature sizes of the workloads."""
    u = 2.0 ** -24
    for dpad in (32, 64, 128, 256, 1024):
        g = (dpad / 32 + 33) * u / (1 - (dpad / 32 + 33) * u)
        assert g < 5e-6
    assert abs((2 * (2 ** -9 + 2 ** -20 + 128 * 2 ** -22)) - 0.00397) < 1e-4


def test_info_struct_layout_matches_header(tmp_path):
    """The binding's ctypes mirror of lipcache_info has the C struct's fields,
    in order, at the same offsets and with the same size (a C program built
    against include/lipcache.h prints them)."""
    import ctypes
    import shutil
    import subprocess

    from paper_2608_13144_gb300 import _lib

    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    names = [f[0] for f in _lib.Info._fields_]
    src = tmp_path / "layout.c"
    body = "\n".join(f'  printf("{n} %zu\\n", offsetof(lipcache_info, {n}));' for n in names)
    src.write_text('#include <stddef.h>\n#include <stdio.h>\n#include "lipcache.h"\nint main(void) {\n'
                   f'{body}\n  printf("sizeof %zu\\n", sizeof(lipcache_info));\n  return 0;\n}}\n')
    exe = tmp_path / "layout"
    include = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.run([cc, "-I", include, str(src), "-o", str(exe)], check=True)
    out = dict(line.split() for line in subprocess.run([str(exe)], check=True, capture_output=True,
                                                       text=True).stdout.splitlines())
    for n in names:
        assert int(out[n]) == getattr(_lib.Info, n).offset, n
    assert int(out["sizeof"]) == ctypes.sizeof(_lib.Info)


def test_binding_signatures_match_header():
    """Every function the binding declares takes, in order, the argument kinds
    the header's prototype gives (pointer, int32, int64, double)."""
    import ctypes

    from paper_2608_13144_gb300 import _lib

    L = _lib.load()
    text = open(os.path.join(ROOT, "include", "lipcache.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    protos = {m.group(2): m.group(3) for m in re.finditer(
        r"(lipcache_status|int64_t|void|const char\s*\*)\s*(lipcache_\w+)\s*\(([^;]*?)\)\s*;", text, flags=re.S)}

    def c_kind(arg):
        arg = " ".join(arg.split())
        if "*" in arg or arg.startswith("lipcache_stream_t"):
            return "p"
        for t, k in (("int64_t", "i64"), ("int32_t", "i32"), ("double", "f64")):
            if arg.startswith(t) or arg.startswith("const " + t):
                return k
        raise AssertionError(f"unclassified argument {arg!r}")

    def py_kind(t):
        if t in (ctypes.c_void_p, ctypes.c_char_p) or (isinstance(t, type) and issubclass(t, ctypes._Pointer)):
            return "p"
        return {ctypes.c_int64: "i64", ctypes.c_int32: "i32", ctypes.c_double: "f64"}[t]

    checked = 0
    for name in _lib.EXPORTS:
        if name not in protos:
            continue
        args = [a for a in protos[name].split(",") if a.strip() and a.strip() != "void"]
        fn = getattr(L, name)
        assert fn.argtypes is not None, name
        assert [c_kind(a) for a in args] == [py_kind(t) for t in fn.argtypes], name
        checked += 1
    assert checked >= 20, checked


def test_every_declaration_cites_its_passage():
    """Each entry point's documentation (the text since the previous
    declaration) names the passage of the paper it implements, or says that it
    has none (options, instrumentation, test hooks)."""
    text = open(os.path.join(ROOT, "include", "lipcache.h")).read()
    decls = list(re.finditer(r"(?:lipcache_status|int64_t|void|const char\s*\*)\s*(lipcache_\w+)\s*\([^;]*\)\s*;", text))
    assert len(decls) >= 20
    cite = re.compile(r"Sec\.|Eqs?\.|Algorithm|Remark|Lemma|counterpart|not part of the method|Test hooks")
    prev = 0
    for m in decls:
        doc = text[prev:m.start()]
        assert cite.search(doc), m.group(1)
        prev = m.end()
