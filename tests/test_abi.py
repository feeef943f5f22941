"""The C ABI without a GPU: the library loads, exports every declared entry
point, and rejects invalid arguments on the host before touching CUDA."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "lookme.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_16305_gb300 import build, lookme

    build.build()
    return lookme.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(lookme_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_four_calls():
    names = declared_functions()
    for n in ("lookme_table_create", "lookme_load_scenes", "lookme_lookup", "lookme_inject"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_the_header():
    from paper_2607_16305_gb300 import lookme

    assert sorted(lookme.EXPORTS) == declared_functions()


def test_desc_layout_matches_header():
    from paper_2607_16305_gb300 import lookme

    assert ctypes.sizeof(lookme.TableDesc) == 8 * 4 + 4 * 4 + 8 * 2


def _create(lib, **kw):
    from paper_2607_16305_gb300 import lookme

    d = dict(n_scenes=4, n_prims=8, d_key=16, d_value=16, dtype=0, residency=0, device=0, reserved0=0,
             max_tokens=0, stage_slots=0)
    d.update(kw)
    desc = lookme.TableDesc(**d)
    h = ctypes.c_void_p()
    st = lib.lookme_table_create(ctypes.byref(desc), ctypes.byref(h))
    return st, h, lib.lookme_last_error().decode()


@pytest.mark.parametrize("bad", [
    dict(n_scenes=0), dict(n_prims=0), dict(d_key=0), dict(d_value=0), dict(dtype=7), dict(residency=3),
    dict(reserved0=1), dict(d_key=12), dict(d_value=20, dtype=0), dict(d_key=6, dtype=1), dict(n_scenes=10**6),
    dict(n_prims=4096), dict(max_tokens=-1), dict(device=-1), dict(d_key=2048),
])
def test_create_rejects_bad_desc(lib, bad):
    from paper_2607_16305_gb300 import lookme

    st, h, msg = _create(lib, **bad)
    assert st == lookme.ERR_INVALID_ARG, (bad, st, msg)
    assert not h.value
    assert msg


def test_null_arguments(lib):
    from paper_2607_16305_gb300 import lookme

    assert lib.lookme_table_create(None, None) == lookme.ERR_INVALID_ARG
    h = ctypes.c_void_p()
    assert lib.lookme_table_create(None, ctypes.byref(h)) == lookme.ERR_INVALID_ARG
    assert lib.lookme_lookup(None, None, 0, 1, None, None, None, None, None) == lookme.ERR_INVALID_ARG
    assert lib.lookme_inject(None, None, None, None, 0, 1, None, None, 0, 0.5, None, 1, None, None,
                             None) == lookme.ERR_INVALID_ARG
    assert lib.lookme_load_scenes(None, 0, 1, None, None, None, None, 1, None) == lookme.ERR_INVALID_ARG
    assert lib.lookme_table_destroy(None) == lookme.OK
    assert lib.lookme_launch_count(None) == 0


def test_status_strings(lib):
    for s in range(7):
        assert lib.lookme_status_string(s)
    assert lib.lookme_kernel_name(4) == b"score"
    assert lib.lookme_kernel_name(99) == b"?"


def test_binding_fails_loudly_without_library(tmp_path):
    from paper_2607_16305_gb300 import lookme

    with pytest.raises(lookme.LookmeError):
        saved = lookme._lib
        lookme._lib = None
        try:
            lookme.load(str(tmp_path / "missing.so"))
        finally:
            lookme._lib = saved
