"""The C-ABI library without a GPU: it builds, loads, exports every symbol the
header declares, and its host-side validation rejects bad arguments before
touching CUDA."""
import ctypes
import os
import re

import pytest

from paper_2511_18936_gb300 import swan

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", h) for h in ("swan.h", "swan_basis.h")]


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(swan.LIB_PATH):
        from paper_2511_18936_gb300 import build
        build.build()
    return swan.load_library()


def declared_functions():
    names = set()
    for h in HEADERS:
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names |= set(re.findall(r"\b(swan_[a-z_]+)\s*\(", text))
    return sorted(names)


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
                buffer_cap=64, max_seq=1024, page_tokens=0, stream=None, value_format=0, k_store_v=0, pool_pages=0)
    base.update(kw)
    return swan.SwanConfig(*[base[f] for f, _ in swan.SwanConfig._fields_])


@pytest.mark.parametrize("kw,status", [
    (dict(head_dim=64), swan.ERR_UNSUPPORTED),
    (dict(n_q_heads=3, n_kv_heads=1), swan.ERR_UNSUPPORTED),
    (dict(n_q_heads=16, n_kv_heads=1), swan.ERR_UNSUPPORTED),
    (dict(n_q_heads=12, n_kv_heads=2), swan.ERR_UNSUPPORTED),
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
    (dict(pool_pages=-1), swan.ERR_INVALID_ARG),
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
    assert lib.swan_reset_sequence(None, 0) == swan.ERR_INVALID_ARG
    assert lib.swan_fork_sequence(None, 0, 1) == swan.ERR_INVALID_ARG
    assert lib.swan_append_varlen(None, 0, None, None, 1, None) == swan.ERR_INVALID_ARG
    assert lib.swan_query_lengths(None, 0, None, None) == swan.ERR_INVALID_ARG
    assert lib.swan_debug_export_seq(None, 0, 0, 1, None, 0) == swan.ERR_INVALID_ARG
    assert lib.swan_append(None, 0, None, None, 1) == swan.ERR_INVALID_ARG
    assert lib.swan_decode(None, 0, None, None) == swan.ERR_INVALID_ARG
    assert lib.swan_flush_buffer(None, 0) == swan.ERR_INVALID_ARG
    assert lib.swan_check(None) == swan.ERR_INVALID_ARG
    assert lib.swan_destroy(None) == swan.OK
    assert lib.swan_launch_count(None) == 0
    assert lib.swan_append_decode(None, 0, None, None, 1, None, None, None) == swan.ERR_INVALID_ARG
    assert lib.swan_debug_check_guards(None) == swan.ERR_INVALID_ARG


def test_fault_hook_arguments(lib):
    """The test hook validates its arguments; arming and disarming it needs no GPU."""
    assert lib.swan_debug_fail_after(0, 0) == swan.ERR_INVALID_ARG
    assert lib.swan_debug_fail_after(3, 0) == swan.ERR_INVALID_ARG
    assert lib.swan_debug_fail_after(swan.FAULT_ALLOC, -2) == swan.ERR_INVALID_ARG
    for kind in (swan.FAULT_ALLOC, swan.FAULT_LAUNCH):
        assert lib.swan_debug_fail_after(kind, 5) == swan.OK
        assert lib.swan_debug_fail_after(kind, -1) == swan.OK
    # a bad configuration is rejected before any allocation, so an armed
    # allocation fault stays armed and is then turned off
    assert lib.swan_debug_fail_after(swan.FAULT_ALLOC, 0) == swan.OK
    h = ctypes.c_void_p()
    cfg = _cfg(k_store=0)
    assert lib.swan_init(ctypes.byref(h), ctypes.byref(cfg), ctypes.c_void_p(4096), None) == swan.ERR_INVALID_ARG
    assert lib.swan_debug_fail_after(swan.FAULT_ALLOC, -1) == swan.OK


# ---------------------------------------------------------------------------
# Offline basis entry points: host-side validation (no launch happens)
# ---------------------------------------------------------------------------

def _vec(**kw):
    d = dict(data=4096, n_mats=2, group=1, count=100, stride_mat=12800, stride_group=0, stride_pos=128,
             stride_coord=1)
    d.update(kw)
    return swan.SwanVectors(**d)


@pytest.mark.parametrize("kw,needle", [
    (dict(data=0), "data is NULL"),
    (dict(data=4100), "16-byte aligned"),
    (dict(n_mats=0), "n_mats"),
    (dict(group=0), "group"),
    (dict(count=0), "count"),
    (dict(count=1 << 31), "count"),
    (dict(stride_pos=100), "stride_pos"),
    (dict(stride_coord=2, stride_pos=128), "either stride_coord or stride_pos"),
    (dict(stride_coord=100, stride_pos=1), "stride_coord"),
    (dict(group=2, stride_group=4), "stride_group"),
    (dict(stride_mat=0), "stride_mat"),
])
def test_basis_vectors_validation(lib, kw, needle):
    v = _vec(**kw)
    st = lib.swan_gram(ctypes.byref(v), ctypes.c_void_p(4096), 0, ctypes.c_void_p(1 << 20),
                       lib.swan_gram_workspace_bytes(2), None)
    assert st == swan.ERR_INVALID_ARG
    assert needle in lib.swan_last_error().decode()
    st = lib.swan_energy(ctypes.byref(v), ctypes.c_void_p(4096), ctypes.c_void_p(4096), 0, None)
    assert st == swan.ERR_INVALID_ARG


def test_basis_workspace_and_pointer_checks(lib):
    v = _vec()
    assert lib.swan_gram_workspace_bytes(0) == 0
    assert lib.swan_gram_workspace_bytes(1) == 320 * 65536 + 256
    assert lib.swan_gram_workspace_bytes(1000) == 1000 * 65536 + 256
    ws = lib.swan_gram_workspace_bytes(2)
    assert lib.swan_gram(ctypes.byref(v), None, 0, ctypes.c_void_p(1 << 20), ws, None) == swan.ERR_INVALID_ARG
    assert lib.swan_gram(ctypes.byref(v), ctypes.c_void_p(4096), 0, ctypes.c_void_p((1 << 20) + 16), ws,
                         None) == swan.ERR_INVALID_ARG
    assert lib.swan_gram(ctypes.byref(v), ctypes.c_void_p(4096), 0, ctypes.c_void_p(1 << 20), ws - 1,
                         None) == swan.ERR_INVALID_ARG
    assert "smaller" in lib.swan_last_error().decode()
    assert lib.swan_basis_eig(None, 1, ctypes.c_void_p(4096), None, None, None) == swan.ERR_INVALID_ARG
    assert lib.swan_basis_eig(ctypes.c_void_p(4096), 0, ctypes.c_void_p(4096), None, None,
                              None) == swan.ERR_INVALID_ARG
    assert lib.swan_basis_check(None, None) == swan.ERR_INVALID_ARG


def _noalloc_view(**over):
    """A well-formed no-allocation view over fake, aligned addresses (never
    dereferenced: every case below fails host validation first)."""
    base = dict(pages=0x10000, page_table=0x20000, num_pages=4, pages_per_unit=2, page_tokens=64,
                k_slots=64, k_active=64, buf_k=0x30000, buf_v=0x40000, buffer_cap=16, buf_start=0,
                buf_len=8, sparse_len=100, batch=1, n_q_heads=2, n_kv_heads=1, head_dim=128,
                R_qk=0x50000, R_vo_t=0x60000, value_format=0, k_slots_v=0, k_active_v=0)
    base.update(over)
    return swan.CacheView(**base)


@pytest.mark.parametrize("field,offset", [("pages", 8), ("page_table", 2), ("buf_k", 4), ("buf_v", 8),
                                          ("R_qk", 4), ("R_vo_t", 8)])
def test_noalloc_rejects_misaligned_view_pointers(lib, field, offset):
    v = _noalloc_view()
    setattr(v, field, getattr(v, field) + offset)
    assert lib.swan_decode_noalloc(ctypes.byref(v), 0x70000, 0x80000, None) == swan.ERR_INVALID_ARG
    assert b"misaligned" in lib.swan_last_error()


def test_noalloc_rejects_misaligned_q_and_out_and_oversize(lib):
    v = _noalloc_view()
    assert lib.swan_decode_noalloc(ctypes.byref(v), 0x70002, 0x80000, None) == swan.ERR_INVALID_ARG
    assert b"misaligned" in lib.swan_last_error()
    assert lib.swan_decode_noalloc(ctypes.byref(v), 0x70000, 0x80001, None) == swan.ERR_INVALID_ARG
    assert b"misaligned" in lib.swan_last_error()
    big = _noalloc_view(batch=600)
    assert lib.swan_decode_noalloc(ctypes.byref(big), 0x70000, 0x80000, None) == swan.ERR_INVALID_ARG
    assert b"static scratch" in lib.swan_last_error()
    assert lib.swan_decode_noalloc(None, 0x70000, 0x80000, None) == swan.ERR_INVALID_ARG


def test_starve_hook_arguments(lib):
    assert lib.swan_debug_starve_tc(-1) == swan.ERR_INVALID_ARG
    assert lib.swan_debug_starve_tc(999) == swan.ERR_INVALID_ARG
    assert lib.swan_debug_starve_tc(2_000_000_001) == swan.ERR_INVALID_ARG
    assert lib.swan_debug_starve_tc(1_000_000) == swan.OK
    assert lib.swan_debug_starve_tc(0) == swan.OK          # disarmed again
