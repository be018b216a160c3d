"""Host-side checks of the C ABI: the library loads without a GPU, exports
every entry point include/*.h declares, and validates arguments on the host
before touching the device."""
import ctypes
import glob
import os
import re

import pytest

from paper_2608_15797_gb300 import kvr

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        for m in re.finditer(r"\b(kvr_[a-z0-9_]+)\s*\(", text):
            names.add(m.group(1))
    return sorted(names)


def test_every_declared_symbol_is_exported():
    names = _declared_functions()
    assert "kvr_decode_step" in names and "kvr_cache_create" in names
    for n in names:
        assert hasattr(kvr.lib, n), f"{n} declared in include/ but not exported"


def test_required_bytes_validates_descriptor():
    good = kvr.make_desc(2, 3, 4, 7, 128, 100)
    n = kvr.kvr_cache_required_bytes(good)
    # K and V slabs alone
    assert n >= 2 * 2 * 3 * 4 * 100 * 128 * 2
    for bad in (kvr.make_desc(0, 3, 4, 7, 128, 100),
                kvr.make_desc(2, 3, 4, 9, 128, 100),
                kvr.make_desc(2, 3, 4, 7, 96, 100),
                kvr.make_desc(2, 3, 4, 7, 128, 0),
                kvr.make_desc(2, 3, 4, 7, 128, 100, softmax_scale=-1.0)):
        assert kvr.kvr_cache_required_bytes(bad) == 0


def _create(desc, ptr, nbytes):
    h = ctypes.c_void_p()
    st = kvr.lib.kvr_cache_create(ctypes.byref(desc), ctypes.c_void_p(ptr),
                                  nbytes, None, ctypes.byref(h))
    return st, h


def test_create_rejects_bad_buffers_on_host():
    desc = kvr.make_desc(1, 1, 1, 1, 64, 8)
    need = kvr.kvr_cache_required_bytes(desc)
    st, h = _create(desc, 0, need)
    assert st == kvr.KVR_EINVAL and not h.value
    assert "null" in kvr.kvr_last_error()
    st, _ = _create(desc, 0x1000 + 8, need)
    assert st == kvr.KVR_EINVAL and "aligned" in kvr.kvr_last_error()
    st, _ = _create(desc, 0x1000, need - 1)
    assert st == kvr.KVR_ENOMEM
    bad = kvr.make_desc(1, 1, 1, 0, 64, 8)
    st, _ = _create(bad, 0x1000, need)
    assert st == kvr.KVR_EINVAL


def test_null_handle_is_rejected():
    assert kvr.lib.kvr_cache_load(None, 0, None, None, 0, 0, None) == kvr.KVR_EINVAL
    assert kvr.lib.kvr_decode_step(None, 0, 1, None, None, None, None, 1, 1,
                                   None) == kvr.KVR_EINVAL
    assert kvr.lib.kvr_evict_compact(None, 0, 1, 1, 1, None) == kvr.KVR_EINVAL
    assert kvr.lib.kvr_sync_status(None, None) == kvr.KVR_EINVAL


def test_missing_library_fails_loudly(tmp_path, monkeypatch):
    """The binding refuses to import without the compiled library."""
    import importlib.util
    src = os.path.join(ROOT, "paper_2608_15797_gb300", "kvr.py")
    pkg = tmp_path / "fakepkg"
    pkg.mkdir()
    (pkg / "kvr.py").write_text(open(src).read())
    spec = importlib.util.spec_from_file_location("fake_kvr", pkg / "kvr.py")
    mod = importlib.util.module_from_spec(spec)
    with pytest.raises(ImportError, match="libkvr.so not found"):
        spec.loader.exec_module(mod)


def test_entropy_descriptor_and_buffer_checks_on_host():
    """kvr_entropy_*: descriptors and buffers are validated on the host,
    before any device call."""
    good = kvr.kvr_entropy_desc(512, 152064, 12, 24, 7.0, 1.0, kvr.KVR_BF16)
    need = kvr.kvr_entropy_required_bytes(good)
    assert need >= 512 * 12 * 4  # the entropy ring at least
    for bad in (kvr.kvr_entropy_desc(0, 100, 12, 24, 7.0, 1.0, 0),
                kvr.kvr_entropy_desc(70000, 100, 12, 24, 7.0, 1.0, 0),
                kvr.kvr_entropy_desc(4, 100, 65, 24, 7.0, 1.0, 0),
                kvr.kvr_entropy_desc(4, 100, 12, 24, float("nan"), 1.0, 0),
                kvr.kvr_entropy_desc(4, 100, 12, 24, 7.0, 1.0, 3)):
        assert kvr.kvr_entropy_required_bytes(bad) == 0
    h = ctypes.c_void_p()
    st = kvr.lib.kvr_entropy_create(ctypes.byref(good), None, need, None,
                                    ctypes.byref(h))
    assert st == kvr.KVR_EINVAL and not h.value
    st = kvr.lib.kvr_entropy_create(ctypes.byref(good), ctypes.c_void_p(0x1000 + 8),
                                    need, None, ctypes.byref(h))
    assert st == kvr.KVR_EINVAL and "aligned" in kvr.kvr_last_error()
    st = kvr.lib.kvr_entropy_create(ctypes.byref(good), ctypes.c_void_p(0x1000),
                                    need - 1, None, ctypes.byref(h))
    assert st == kvr.KVR_ENOMEM


def test_host_step_rejects_null_buffers_on_host():
    """kvr_decode_step_host checks its host and staging pointers (and the
    handle) before it enqueues anything."""
    one = ctypes.c_void_p(16)
    st = kvr.lib.kvr_decode_step_host(None, 0, 1, None, one, one, one, one,
                                      one, one, one, 4, 1, None)
    assert st == kvr.KVR_EINVAL and "null host" in kvr.kvr_last_error()
    st = kvr.lib.kvr_decode_step_host(None, 0, 1, one, one, one, one, one,
                                      one, one, one, 4, 1, None)
    assert st == kvr.KVR_EINVAL and "null cache" in kvr.kvr_last_error()


def test_import_rejects_null_arguments_on_host():
    one = ctypes.c_void_p(16)
    st = kvr.lib.kvr_cache_import(None, 0, one, one, one, one, one, one, None)
    assert st == kvr.KVR_EINVAL and "null cache" in kvr.kvr_last_error()
