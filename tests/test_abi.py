"""Host-side checks of the C-ABI library (no GPU needed): it builds for
sm_103a, loads, exports every symbol include/bacon.h declares, and rejects
invalid arguments before touching the device."""

import ctypes
import os
import re
import threading

import pytest

from paper_2606_14782_gb300 import bacon, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return bacon.load()


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "bacon.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(bacon_[a-z_]+)\s*\(", text)))


def test_header_declares_the_binding_exports():
    assert declared_symbols() == sorted(bacon.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name


def test_default_params(lib):
    p = bacon.default_params()
    assert (p.r, p.m, p.rho, p.keep_window, p.use_E, p.use_L, p.use_T) == (5, 4, 2, 1, 1, 1, 1)
    assert p.gamma == 1.0 and abs(p.eps - 1e-8) < 1e-15
    assert p.max_seq_len == 16384 and p.max_requests == 4 and p.keep_scores == 0


@pytest.mark.parametrize("args,msg", [
    ((2, 4, 6, 64, 32, 7, 64), "multiple"),
    ((2, 4, 4, 96, 32, 7, 64), "head_dim"),
    ((2, 4, 4, 64, 32, 8, 64), "pool"),
    ((2, 4, 4, 64, 32, 7, 16), "budget"),
    ((0, 4, 4, 64, 32, 7, 64), "positive"),
    ((2, 4, 4, 64, 0, 7, 64), "window"),
])
def test_init_rejects_bad_shapes(lib, args, msg):
    h = ctypes.c_void_p()
    rc = lib.bacon_init(ctypes.byref(h), *args, None)
    assert rc == bacon.BACON_EINVAL
    assert msg in lib.bacon_last_error().decode()
    assert not h.value


def test_init_rejects_bad_params(lib):
    h = ctypes.c_void_p()
    for field, value in [("max_seq_len", 100000), ("max_requests", 0), ("r", -1),
                         ("max_requests", 1000)]:
        p = bacon.default_params(**{field: value})
        assert lib.bacon_init(ctypes.byref(h), 28, 4, 28, 128, 64, 7, 256,
                              ctypes.byref(p)) == bacon.BACON_EINVAL
    # G * W beyond the shared-memory bound of pass 2
    assert lib.bacon_init(ctypes.byref(h), 2, 1, 64, 128, 64, 7, 256,
                          None) == bacon.BACON_EUNSUPPORTED


def test_null_context_is_rejected(lib):
    assert lib.bacon_compress_all_layers(None, 1, None, None, None, 640, 64, None, None, None,
                                         None) == bacon.BACON_EINVAL
    assert lib.bacon_sync(None, None) == bacon.BACON_EINVAL
    assert lib.bacon_profile_enable(None, 1) == bacon.BACON_EINVAL


def test_last_error_is_per_thread(lib):
    h = ctypes.c_void_p()
    lib.bacon_init(ctypes.byref(h), 2, 4, 6, 64, 32, 7, 64, None)
    seen = {}

    def other():
        seen["msg"] = lib.bacon_last_error().decode()

    t = threading.Thread(target=other)
    t.start()
    t.join()
    assert seen["msg"] == ""
    assert "multiple" in lib.bacon_last_error().decode()


def test_product_path_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(bacon, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(bacon, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        bacon.load()


def test_struct_layouts_match_the_header(tmp_path):
    """ctypes mirrors of bacon_params and bacon_variant against the C layout."""
    import os
    import subprocess
    src = tmp_path / "layout.c"
    src.write_text(
        '#include <stdio.h>\n#include <stddef.h>\n#include "bacon.h"\n'
        "#define F(T, f) printf(#T \" \" #f \" %zu\\n\", offsetof(T, f));\n"
        "int main(void) {\n"
        '  printf("bacon_params size %zu\\n", sizeof(bacon_params));\n'
        '  printf("bacon_variant size %zu\\n", sizeof(bacon_variant));\n'
        + "".join(f"  F(bacon_params, {f})\n" for f, _ in bacon.Params._fields_)
        + "".join(f"  F(bacon_variant, {f})\n" for f, _ in bacon.Variant._fields_)
        + "  return 0;\n}\n")
    exe = tmp_path / "layout"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.run(["gcc", "-I", inc, str(src), "-o", str(exe)], check=True)
    got = {}
    for line in subprocess.run([str(exe)], check=True, capture_output=True,
                               text=True).stdout.splitlines():
        t, f, v = line.split()
        got[(t, f)] = int(v)
    for t, cls in (("bacon_params", bacon.Params), ("bacon_variant", bacon.Variant)):
        assert got[(t, "size")] == ctypes.sizeof(cls), t
        for f, _ in cls._fields_:
            assert got[(t, f)] == getattr(cls, f).offset, (t, f)


def test_sweep_rejects_null_context(lib):
    arr = (bacon.Variant * 1)()
    assert lib.bacon_sweep(None, 1, None, None, 640, 64, 1, arr, None, None,
                           None) == bacon.BACON_EINVAL
