"""Host-only checks of the C ABI: the library loads, exports every declared
symbol, and rejects bad arguments before touching a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def kv():
    from paper_2607_05061_gb300 import build
    build.build()
    from paper_2607_05061_gb300 import kvpop
    return kvpop


def declared_functions():
    src = open(os.path.join(ROOT, "include", "kvpop.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(kvpop_[a-z_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("kvpop_init_cache", "kvpop_prefill_compress", "kvpop_decode_step", "kvpop_free"):
        assert required in names


def test_library_exports_every_declared_symbol(kv):
    lib = ctypes.CDLL(kv.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(declared_functions()) == set(kv.EXPORTED)


def test_status_strings(kv):
    for code in range(7):
        assert kv.kvpop_status_string(code)
    assert kv.kvpop_status_string(99) == b"unknown status"


def good_config(kv, **kw):
    base = dict(batch=1, n_kv_heads=2, q_per_kv=2, head_dim=64, budget_B=8, delay_D=2, n_sink=0,
                scorer_hidden=4, kv_dtype=kv.KVPOP_F32)
    base.update(kw)
    return kv.kvpop_config(**base)


@pytest.mark.parametrize("field,value", [
    ("batch", 0), ("n_kv_heads", 0), ("q_per_kv", 3), ("q_per_kv", 8), ("head_dim", 96),
    ("budget_B", 0), ("delay_D", 0), ("n_sink", -1), ("n_sink", 8), ("scorer_hidden", 0),
    ("scorer_hidden", 2048), ("kv_dtype", 7), ("batch", 100000)])
def test_init_rejects_bad_config(kv, field, value):
    cfg = good_config(kv, **{field: value})
    buf = (ctypes.c_float * 16)()
    sc = kv.kvpop_scorer(ctypes.addressof(buf), ctypes.addressof(buf), ctypes.addressof(buf),
                         ctypes.addressof(buf), None)
    h = ctypes.c_void_p(123)
    st = kv.kvpop_init_cache(ctypes.byref(cfg), ctypes.byref(sc), None, ctypes.byref(h))
    assert st == 1   # KVPOP_ERR_INVALID_ARG
    assert h.value is None


def test_init_rejects_missing_scorer(kv):
    cfg = good_config(kv)
    h = ctypes.c_void_p()
    assert kv.kvpop_init_cache(ctypes.byref(cfg), None, None, ctypes.byref(h)) == 1
    assert kv.kvpop_init_cache(None, None, None, ctypes.byref(h)) == 1
    assert kv.kvpop_init_cache(ctypes.byref(cfg), None, None, None) == 1


def test_free_null_and_foreign_handles(kv):
    assert kv.kvpop_free(None) == 0
    junk = (ctypes.c_uint64 * 64)()
    assert kv.kvpop_free(ctypes.addressof(junk)) == 1
    assert kv.kvpop_decode_step(ctypes.addressof(junk), None, None, None, None, None, None, None, None) == 1
    assert kv.kvpop_check(ctypes.addressof(junk), None) == 1


def test_alloc_fault_hook_is_callable(kv):
    kv.kvpop_debug_fail_alloc_after(0)
    kv.kvpop_debug_fail_alloc_after(-5)
