"""Host-only checks of the C ABI: the library loads, exports every declared
symbol, and rejects bad arguments before touching a GPU; the binding refuses to
import without the library, and the product package never reaches the oracle."""
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
    ("scorer_hidden", 2048), ("kv_dtype", 7), ("batch", 100000),
    ("batch", 6145)])                # 12290 pairs: one past the largest accepted 12288
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


def test_topk_and_prompt_attention_reject_bad_arguments(kv):
    """Argument checks of the cache-free prompt calls run before any CUDA call."""
    P = 0x1000                                   # 16-byte aligned dummy address, never dereferenced
    ws = kv.kvpop_topk_workspace_bytes(4, 100)
    assert ws >= 4 * 100 * 16
    assert kv.kvpop_topk_workspace_bytes(0, 100) == 0
    ok, bad, align = 0, 1, 2          # KVPOP_OK, KVPOP_ERR_INVALID_ARG, KVPOP_ERR_ALIGN
    cut = kv.kvpop_topk_cutoff
    assert cut(P, None, 0, 100, 0, 4, 8, P, P, None, P, ws, None) == ok          # nothing to do
    assert cut(P, None, 4, 100, 0, 0, 8, P, P, None, P, ws, None) == bad         # window 0
    assert cut(P, None, 4, 100, 0, 4, 0, P, P, None, P, ws, None) == bad         # k 0
    assert cut(P, None, 4, (1 << 18) + 1, 0, 4, 8, P, P, None, P, ws, None) == bad
    assert cut(P, None, 4, 100, 0, 4, 8, P, P, None, P, ws - 1, None) == bad     # workspace too small
    assert cut(None, None, 4, 100, 0, 4, 8, P, P, None, P, ws, None) == bad
    assert cut(P + 2, None, 4, 100, 0, 4, 8, P, P, None, P, ws, None) == align
    assert cut(P, None, 4, 100, 0, 4, 8, P, P, P + 2, P, ws, None) == align      # order 4-aligned
    assert cut(P, None, 4, 100, 0, 4, 8, P, P, None, P + 16, ws, None) == align  # workspace 256-aligned
    att = kv.kvpop_prompt_attention
    args = lambda **o: [o.get(n, v) for n, v in (
        ("Q", P), ("K", P), ("V", P), ("rank", P), ("tau", P), ("order", None), ("len", None),
        ("n", 2), ("H", 8),
        ("G", 4), ("d", 128), ("S", 64), ("s", 0), ("w", 16), ("k", 64), ("dt", kv.KVPOP_BF16),
        ("Y", P), ("lse", P), ("st", None))]
    assert att(*args(n=0)) == ok
    assert att(*args(d=96)) == bad
    assert att(*args(G=3)) == bad
    assert att(*args(w=0)) == bad
    assert att(*args(k=1 << 20)) == bad                 # key lists would not fit in shared memory
    assert att(*args(n=10000)) == bad                   # more than 65535 (sequence, head) rows
    assert att(*args(dt=7)) == bad
    assert att(*args(Y=None)) == bad
    assert att(*args(Q=P + 8)) == align
    assert att(*args(Y=P + 4)) == align
    assert att(*args(lse=P + 2)) == align
    assert att(*args(order=P + 2)) == align


def test_causal_lse_and_future_target_reject_bad_arguments(kv):
    P = 0x1000
    bad, align = 1, 2
    lse = kv.kvpop_causal_lse
    assert lse(P, P, None, 0, 8, 4, 128, 64, 1, P, None) == 0
    assert lse(P, P, None, 2, 8, 4, 96, 64, 1, P, None) == bad          # head_dim
    assert lse(P, P, None, 2, 8, 4, 128, 64, 5, P, None) == bad         # dtype
    assert lse(P, P, None, 2, 8, 4, 128, 64, 1, None, None) == bad
    assert lse(P + 8, P, None, 2, 8, 4, 128, 64, 1, P, None) == align
    ft = kv.kvpop_future_target
    args = lambda **o: [o.get(n, v) for n, v in (
        ("Q", P), ("K", P), ("lse", P), ("len", None), ("n", 2), ("H", 8), ("G", 4), ("d", 128),
        ("S", 64), ("w", 16), ("la", 0), ("dt", 1), ("logm", P), ("tgt", P), ("agg", 0), ("cn", 1),
        ("eps", 1e-6), ("st", None))]
    assert ft(*args(n=0)) == 0
    assert ft(*args(w=-1)) == bad
    assert ft(*args(la=-3)) == bad
    assert ft(*args(agg=2)) == bad
    assert ft(*args(cn=3)) == bad
    assert ft(*args(eps=-1.0)) == bad
    assert ft(*args(eps=float("nan"))) == bad
    assert ft(*args(eps=float("inf"))) == bad
    assert ft(*args(logm=None)) == bad
    assert ft(*args(G=3)) == bad
    assert ft(*args(lse=P + 2)) == align
    assert ft(*args(tgt=P + 1)) == align


def test_binding_fails_loudly_without_the_library(tmp_path):
    """A copy of the binding next to no libkvpop.so must refuse to import (no fallback)."""
    import importlib.util
    src = os.path.join(ROOT, "paper_2607_05061_gb300", "kvpop.py")
    dst = tmp_path / "kvpop.py"
    dst.write_text(open(src).read())
    spec = importlib.util.spec_from_file_location("kvpop_nolib", str(dst))
    mod = importlib.util.module_from_spec(spec)
    with pytest.raises(ImportError, match="libkvpop.so is missing"):
        spec.loader.exec_module(mod)


def test_product_package_never_reaches_the_oracle():
    """No file of the product package imports, loads or names the test oracle."""
    import re
    pkg = os.path.join(ROOT, "paper_2607_05061_gb300")
    pat = re.compile(r"\boracle\b")
    hits = []
    for dirpath, _, files in os.walk(pkg):
        if "_build" in dirpath or "__pycache__" in dirpath:
            continue
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                path = os.path.join(dirpath, f)
                for i, line in enumerate(open(path, encoding="utf-8"), 1):
                    if pat.search(line):
                        hits.append(f"{os.path.relpath(path, ROOT)}:{i}: {line.strip()}")
    assert not hits, "\n".join(hits)
