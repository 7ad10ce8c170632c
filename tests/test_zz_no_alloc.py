"""swan_decode_noalloc on a GB300: against the oracle, and against swan_decode.

swan_decode_noalloc is for callers that cannot call cudaMalloc, such as a
serving engine that hands out all device memory from its own reserved pool
and must not see a hidden allocation.  It decodes over a cache in the
caller's own device memory and keeps its scratch in a fixed static device
array inside the library.

Two kinds of check, each over two calls in a row (the scratch keeps the last
call's contents, so the second call shows that nothing stale leaks in):

* the caller's cache is built here from the oracle's own state (its pruned
  indices and values, its dense buffer) in the page layout the header
  documents, and the output must match the oracle's decode within the
  attention tolerance: for G = 1, 2, 4, 8, fp16 and E4M3 values, equal and
  separate key/value keep counts, the >64-entry kernel variant, a
  buffer-only and an empty cache;
* the caller's cache is a copy of what a libswan context built, and the
  output must equal that context's swan_decode bit for bit (both size the
  grid with the same rule, so the same CTAs sum the same terms in the same
  order).

After every call the status word is read with swan_noalloc_check.  This file
is collected last so that a failure here comes after every other test.
"""
from __future__ import annotations

import ctypes

import numpy as np
import pytest

import oracle
from paper_2511_18936_gb300 import synth
from tests.helpers import TOL_OUT

pytestmark = pytest.mark.gpu

D = 128


def _slots(k):
    return -(-k // 8) * 8


def _e4m3_bytes(vals_fp16):
    """E4M3 bytes of fp16 values that are exact E4M3 numbers (the oracle's
    fp8 cache); an independent library cast, exact on such values."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(vals_fp16, np.float16).astype(np.float32))
    e = t.to(torch.float8_e4m3fn)
    assert torch.equal(e.float(), t), "values are not exact E4M3 numbers"
    return e.view(torch.uint8).numpy()


def build_pages(idx_k, val_k, idx_v, val_v, P, fp8, perm):
    """Lay per-unit sparse vectors out as the header's pages.

    idx_*, val_*: [units][L][k] in stored order (keys k_K, values k_V).
    Returns (pool [num_pages][page_bytes] uint8, table [units * ppu] int32,
    ppu, ks, vs).  Logical page g of unit u goes to physical page
    perm[u * ppu + g]."""
    units, L, kk = idx_k.shape
    kv = idx_v.shape[2]
    ks, vs = _slots(kk), _slots(kv)
    ppu = max(1, -(-L // P))
    Lp = ppu * P
    nblk = Lp // 32

    def pad(a, k_slots, dtype):
        out = np.zeros((units, Lp, k_slots), dtype)
        out[:, :L, :a.shape[2]] = a
        # [units][block][32 tok][chunk][8] -> [units][block][chunk][32 tok][8]
        return out.reshape(units, nblk, 32, k_slots // 8, 8).transpose(0, 1, 3, 2, 4)

    if fp8:
        def region(idx, val, k_slots):
            v8 = pad(_e4m3_bytes(val).reshape(val.shape), k_slots, np.uint8)
            i8 = pad(idx, k_slots, np.uint8)
            return np.concatenate([v8, i8], axis=-1).reshape(units, nblk, -1)   # 16-byte records
        blocks = np.concatenate([region(idx_k, val_k, ks), region(idx_v, val_v, vs)], axis=-1)
        assert blocks.shape[-1] == 64 * (ks + vs)
    else:
        def vals16(val, k_slots):
            return pad(np.asarray(val, np.float16).view(np.uint16), k_slots, np.uint16).reshape(
                units, nblk, -1).view(np.uint8)
        blocks = np.concatenate([vals16(val_k, ks), pad(idx_k, ks, np.uint8).reshape(units, nblk, -1),
                                 vals16(val_v, vs), pad(idx_v, vs, np.uint8).reshape(units, nblk, -1)],
                                axis=-1)
        assert blocks.shape[-1] == 96 * (ks + vs)
    logical = blocks.reshape(units * ppu, -1)
    pool = np.zeros_like(logical)
    pool[perm] = logical
    table = np.asarray(perm, np.int32)
    return pool, table, ppu, ks, vs


class CallerCache:
    """A cache held in caller-owned (torch) device memory, with a view."""

    def __init__(self, idx_k, val_k, idx_v, val_v, buf_k, buf_v, R, Rv, *, B, H_kv, G, P, cap, fp8,
                 seed=0):
        import torch
        dev = torch.device("cuda")
        units = B * H_kv
        L = idx_k.shape[1]
        nb = buf_k.shape[1]
        self.L, self.nb = L, nb
        self.perm = np.random.default_rng(seed).permutation(units * max(1, -(-L // P)))
        pool, table, ppu, ks, vs = build_pages(idx_k, val_k, idx_v, val_v, P, fp8, self.perm)
        self.start = 5 % cap if cap else 0
        ring_k = np.zeros((units, max(cap, 1), D), np.float16)
        ring_v = np.zeros((units, max(cap, 1), D), np.float16)
        for i in range(nb):
            ring_k[:, (self.start + i) % cap] = buf_k[:, i]
            ring_v[:, (self.start + i) % cap] = buf_v[:, i]
        self.t = dict(pool=torch.from_numpy(pool).to(dev), table=torch.from_numpy(table).to(dev),
                      rk=torch.from_numpy(ring_k).to(dev), rv=torch.from_numpy(ring_v).to(dev),
                      R=torch.from_numpy(np.ascontiguousarray(R, np.float32)).to(dev),
                      RvT=torch.from_numpy(np.ascontiguousarray(np.transpose(Rv, (0, 2, 1)), np.float32)).to(dev))
        self.geom = dict(num_pages=units * ppu, pages_per_unit=ppu, page_tokens=P, k_slots=ks, k_slots_v=vs,
                         buffer_cap=cap, batch=B, n_q_heads=H_kv * G, n_kv_heads=H_kv, fp8=fp8)

    def view(self, k_active, k_active_v, *, sparse=True):
        from paper_2511_18936_gb300 import swan
        g, t = self.geom, self.t
        return swan.CacheView(
            t["pool"].data_ptr() if sparse else 0, t["table"].data_ptr() if sparse else 0, g["num_pages"],
            g["pages_per_unit"], g["page_tokens"], g["k_slots"], k_active, t["rk"].data_ptr(),
            t["rv"].data_ptr(), g["buffer_cap"], self.start, self.nb, self.L if sparse else 0, g["batch"],
            g["n_q_heads"], g["n_kv_heads"], D, t["R"].data_ptr(), t["RvT"].data_ptr(),
            swan.VALUE_FORMATS["fp8_e4m3" if g["fp8"] else "fp16"], g["k_slots_v"], k_active_v)


def _decode(view, q_np):
    import torch

    from paper_2511_18936_gb300 import swan
    q = torch.from_numpy(q_np).cuda()
    out = torch.full_like(q, float("nan"))
    swan.decode_noalloc(view, q, out)
    swan.noalloc_check()              # synchronises; raises if the status word was set
    return out.float().cpu().numpy().astype(np.float64)


def _problem(B, H_kv, G, L, seed):
    R = synth.rotations(H_kv, D, seed=seed, workload=91, layer=0)
    Rv = synth.rotations(H_kv, D, seed=seed, workload=91, layer=0, tensor_id=synth.T_R_VO)
    k = synth.lowrank_kv(B, H_kv, L, D, seed, 91, 0, synth.T_K)
    v = synth.lowrank_kv(B, H_kv, L, D, seed, 91, 0, synth.T_V)
    q1 = synth.gaussian_fp16((B, H_kv * G, D), seed + 1, 91, 0, synth.T_Q)
    q2 = synth.gaussian_fp16((B, H_kv * G, D), seed + 2, 91, 0, synth.T_Q, scale=4.0)
    return R, Rv, k, v, q1, q2


# (G, values, k_K stored, k_V stored, second call's (k_K, k_V))
ORACLE_CASES = [
    (1, "fp16", 64, 64, (33, 33)),
    (2, "fp16", 60, 60, (29, 29)),
    (4, "fp16", 56, 56, (56, 17)),
    (1, "fp8_e4m3", 64, 64, (40, 40)),
    (4, "fp8_e4m3", 56, 56, (24, 56)),
    (2, "fp16", 64, 32, (48, 20)),
    (1, "fp8_e4m3", 48, 24, (48, 9)),
    (1, "fp16", 128, 128, (96, 96)),
    (4, "fp16", 128, 100, (72, 100)),
    (8, "fp16", 56, 56, (56, 21)),
    (8, "fp8_e4m3", 64, 40, (48, 40)),
]


@pytest.mark.parametrize("G,fmt,kk,kv,k2", ORACLE_CASES,
                         ids=[f"G{c[0]}-{c[1]}-k{c[2]}v{c[3]}" for c in ORACLE_CASES])
def test_noalloc_matches_oracle_twice(G, fmt, kk, kv, k2):
    B, H_kv, cap, P, L = 2, 2, 48, 64, 700
    R, Rv, k, v, q1, q2 = _problem(B, H_kv, G, L, seed=6 + G)
    ref = oracle.SwanOracle(R, Rv, batch=B, n_q_heads=H_kv * G, k_store=kk, buffer_cap=cap,
                            value_format=fmt, k_store_v=kv)
    ref.append(k[:, :, :333], v[:, :, :333])
    ref.append(k[:, :, 333:], v[:, :, 333:])
    units = B * H_kv
    Ls, nb = ref.sparse_len, ref.buffer_len
    assert Ls == L - cap and nb == cap
    cache = CallerCache(ref.sp_idx_k.reshape(units, Ls, kk), ref.sp_val_k.reshape(units, Ls, kk),
                        ref.sp_idx_v.reshape(units, Ls, kv), ref.sp_val_v.reshape(units, Ls, kv),
                        ref.buf_k.reshape(units, nb, D), ref.buf_v.reshape(units, nb, D), R, Rv,
                        B=B, H_kv=H_kv, G=G, P=P, cap=cap, fp8=fmt != "fp16", seed=G)
    for q, (ka, kav) in ((q1, (kk, kv)), (q2, k2)):
        ref.set_k(ka, kav)
        want = ref.decode(q)
        got = _decode(cache.view(ka, kav), q)
        err = np.abs(got - want).max()
        assert err <= TOL_OUT, (ka, kav, err)


def test_noalloc_buffer_only_and_empty_cache():
    B, H_kv, G, cap = 1, 2, 4, 64
    R, Rv, k, v, q1, q2 = _problem(B, H_kv, G, 40, seed=3)
    ref = oracle.SwanOracle(R, Rv, batch=B, n_q_heads=H_kv * G, k_store=32, buffer_cap=cap)
    ref.append(k, v)
    assert ref.sparse_len == 0 and ref.buffer_len == 40
    units = B * H_kv
    empty_idx = np.zeros((units, 0, 32), np.uint8)
    empty_val = np.zeros((units, 0, 32), np.float16)
    cache = CallerCache(empty_idx, empty_val, empty_idx, empty_val, ref.buf_k.reshape(units, 40, D),
                        ref.buf_v.reshape(units, 40, D), R, Rv, B=B, H_kv=H_kv, G=G, P=64, cap=cap, fp8=False)
    for q in (q1, q2):
        got = _decode(cache.view(32, 32, sparse=False), q)
        assert np.abs(got - ref.decode(q)).max() <= TOL_OUT
    cache.nb = 0                          # no token at all: the output is zero
    for q in (q1, q2):
        assert np.array_equal(_decode(cache.view(32, 32, sparse=False), q), np.zeros_like(q, np.float64))


# (G, values, k_K stored, k_V stored, runtime (k_K, k_V) of the two calls)
CONTEXT_CASES = [
    (2, "fp16", 60, 60, ((60, 60), (29, 29))),
    (1, "fp8_e4m3", 64, 32, ((64, 32), (40, 12))),
    (4, "fp16", 56, 56, ((56, 56), (30, 56))),
    (8, "fp16", 56, 48, ((56, 48), (17, 48))),
]


@pytest.mark.parametrize("G,fmt,kk,kv,ks", CONTEXT_CASES, ids=[f"G{c[0]}-{c[1]}" for c in CONTEXT_CASES])
def test_noalloc_equals_context_decode_bitwise(G, fmt, kk, kv, ks):
    import torch

    from paper_2511_18936_gb300 import swan

    dev = torch.device("cuda")
    B, H_kv, cap, P, L = 2, 2, 48, 64, 700
    R, Rv, k, v, q1, q2 = _problem(B, H_kv, G, L, seed=20 + G)
    ctx = swan.Context(torch.from_numpy(R)[None].to(dev), torch.from_numpy(Rv)[None].to(dev), num_layers=1,
                       batch=B, n_q_heads=H_kv * G, n_kv_heads=H_kv, k_store=kk, buffer_cap=cap, max_seq=L,
                       page_tokens=P, value_format=fmt, k_store_v=kv)
    kt, vt = torch.from_numpy(k).to(dev), torch.from_numpy(v).to(dev)
    ctx.append(0, kt[:, :, :333].contiguous(), vt[:, :, :333].contiguous())
    ctx.append(0, kt[:, :, 333:].contiguous(), vt[:, :, 333:].contiguous())
    info = ctx.query(0)
    units, Ls, nb = B * H_kv, info.sparse_len, info.buffer_len
    ik, vk = ctx.export_sparse(0, "k")
    iv, vv = ctx.export_sparse(0, "v")
    cache = CallerCache(ik.reshape(units, Ls, kk), vk.reshape(units, Ls, kk), iv.reshape(units, Ls, kv),
                        vv.reshape(units, Ls, kv), ctx.export_buffer(0, "k").reshape(units, nb, D),
                        ctx.export_buffer(0, "v").reshape(units, nb, D), R, Rv, B=B, H_kv=H_kv, G=G, P=P,
                        cap=cap, fp8=fmt != "fp16", seed=1)
    for q, (ka, kav) in zip((q1, q2), ks):
        ctx.set_k(ka, kav)
        want = ctx.decode(0, torch.from_numpy(q).to(dev)).float().cpu().numpy().astype(np.float64)
        got = _decode(cache.view(ka, kav), q)
        assert np.array_equal(got, want), (ka, kav, np.abs(got - want).max())
    ctx.check()
    ctx.check_guards()
    ctx.close()


def test_noalloc_rejects_misaligned_and_oversize_without_launching():
    import torch

    from paper_2511_18936_gb300 import swan

    B, H_kv, G = 1, 1, 2
    R, Rv, k, v, q1, _ = _problem(B, H_kv, G, 100, seed=4)
    ref = oracle.SwanOracle(R, Rv, batch=B, n_q_heads=G, k_store=16, buffer_cap=32)
    ref.append(k, v)
    cache = CallerCache(ref.sp_idx_k.reshape(1, 68, 16), ref.sp_val_k.reshape(1, 68, 16),
                        ref.sp_idx_v.reshape(1, 68, 16), ref.sp_val_v.reshape(1, 68, 16),
                        ref.buf_k.reshape(1, 32, D), ref.buf_v.reshape(1, 32, D), R, Rv,
                        B=B, H_kv=H_kv, G=G, P=64, cap=32, fp8=False)
    lib = swan.load_library()
    q = torch.from_numpy(q1).cuda()
    raw = torch.zeros(q.numel() + 8, dtype=torch.float16, device="cuda")
    sentinel = torch.full((q.numel() + 8,), 7.0, dtype=torch.float16, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    raw[1:1 + q.numel()] = q.flatten()
    cases = []
    bad = cache.view(16, 16)
    bad.pages += 8
    cases.append((bad, q.data_ptr(), sentinel.data_ptr()))
    bad = cache.view(16, 16)
    bad.buf_v += 2
    cases.append((bad, q.data_ptr(), sentinel.data_ptr()))
    cases.append((cache.view(16, 16), raw.data_ptr() + 2, sentinel.data_ptr()))      # q off by 2 bytes
    cases.append((cache.view(16, 16), q.data_ptr(), sentinel.data_ptr() + 1))        # out off by 1 byte
    for view, qp, op in cases:
        assert lib.swan_decode_noalloc(ctypes.byref(view), qp, op, stream) == swan.ERR_INVALID_ARG
        assert b"misaligned" in lib.swan_last_error()
    big = cache.view(16, 16)
    big.batch = 513                                  # 1026 query vectors > 1024
    assert lib.swan_decode_noalloc(ctypes.byref(big), q.data_ptr(), sentinel.data_ptr(), stream) == \
        swan.ERR_INVALID_ARG
    assert b"static scratch" in lib.swan_last_error()
    torch.cuda.synchronize()
    assert bool((sentinel == 7.0).all()), "a rejected call wrote its output"
    # the scratch is still usable afterwards
    got = _decode(cache.view(16, 16), q1)
    assert np.abs(got - ref.decode(q1)).max() <= TOL_OUT
