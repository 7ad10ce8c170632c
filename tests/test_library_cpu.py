"""The C-ABI library without a GPU: it builds, loads, exports every symbol the
header declares, and its host-side validation rejects bad arguments before
touching CUDA."""
import ctypes
import os
import re

import pytest

from paper_2511_18936_gb300 import swan

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "swan.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(swan.LIB_PATH):
        from paper_2511_18936_gb300 import build
        build.build()
    return swan.load_library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(swan_[a-z_]+)\s*\(", text)))


def test_header_declares_the_binding_list():
    assert declared_functions() == sorted(swan.EXPORTED)


def test_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    for s in range(9):
        assert lib.swan_status_string(s)
    assert lib.swan_status_string(99) == b"unknown status"


def _cfg(**kw):
    base = dict(num_layers=1, batch=1, n_q_heads=1, n_kv_heads=1, head_dim=128, k_store=64,
                buffer_cap=64, max_seq=1024, page_tokens=0, stream=None, value_format=0, k_store_v=0)
    base.update(kw)
    return swan.SwanConfig(*[base[f] for f, _ in swan.SwanConfig._fields_])


@pytest.mark.parametrize("kw,status", [
    (dict(head_dim=64), swan.ERR_UNSUPPORTED),
    (dict(n_q_heads=3, n_kv_heads=1), swan.ERR_UNSUPPORTED),
    (dict(n_q_heads=8, n_kv_heads=1), swan.ERR_UNSUPPORTED),
    (dict(n_q_heads=3, n_kv_heads=2), swan.ERR_INVALID_ARG),
    (dict(k_store=0), swan.ERR_INVALID_ARG),
    (dict(k_store=129), swan.ERR_INVALID_ARG),
    (dict(buffer_cap=-1), swan.ERR_INVALID_ARG),
    (dict(buffer_cap=5000), swan.ERR_INVALID_ARG),
    (dict(max_seq=0), swan.ERR_INVALID_ARG),
    (dict(page_tokens=48), swan.ERR_INVALID_ARG),
    (dict(page_tokens=96), swan.ERR_INVALID_ARG),
    (dict(page_tokens=8192), swan.ERR_INVALID_ARG),
    (dict(num_layers=0), swan.ERR_INVALID_ARG),
    (dict(batch=0), swan.ERR_INVALID_ARG),
    (dict(value_format=2), swan.ERR_INVALID_ARG),
    (dict(value_format=-1), swan.ERR_INVALID_ARG),
    (dict(k_store_v=129), swan.ERR_INVALID_ARG),
    (dict(k_store_v=-2), swan.ERR_INVALID_ARG),
])
def test_init_rejects_bad_config_without_cuda(lib, kw, status):
    h = ctypes.c_void_p(123)
    cfg = _cfg(**kw)
    r = lib.swan_init(ctypes.byref(h), ctypes.byref(cfg), ctypes.c_void_p(16), None)
    assert r == status, (kw, r, lib.swan_last_error())
    assert h.value is None
    assert lib.swan_last_error()


def test_null_arguments(lib):
    assert lib.swan_init(None, None, None, None) == swan.ERR_INVALID_ARG
    h = ctypes.c_void_p()
    cfg = _cfg()
    assert lib.swan_init(ctypes.byref(h), ctypes.byref(cfg), None, None) == swan.ERR_INVALID_ARG
    assert lib.swan_set_k(None, 4) == swan.ERR_INVALID_ARG
    assert lib.swan_set_kv(None, 4, 4) == swan.ERR_INVALID_ARG
    assert lib.swan_append(None, 0, None, None, 1) == swan.ERR_INVALID_ARG
    assert lib.swan_decode(None, 0, None, None) == swan.ERR_INVALID_ARG
    assert lib.swan_flush_buffer(None, 0) == swan.ERR_INVALID_ARG
    assert lib.swan_check(None) == swan.ERR_INVALID_ARG
    assert lib.swan_destroy(None) == swan.OK
    assert lib.swan_launch_count(None) == 0
