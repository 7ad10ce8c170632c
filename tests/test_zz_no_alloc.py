"""swan_decode_noalloc against swan_decode (needs a GB300).

swan_decode_noalloc serves callers that cannot call cudaMalloc: it decodes
over a cache held in the caller's own device memory and keeps its scratch in
a static device array inside the library.  Here the caller's memory is torch
tensors holding the same cache that a libswan context built (exported and
re-laid out by the test); the two entry points must agree, on two calls in a
row.  This file is collected last so that a failure here comes after every
other test has run.
"""
from __future__ import annotations

import numpy as np
import pytest

from paper_2511_18936_gb300 import synth
from tests.helpers import TOL_OUT

pytestmark = pytest.mark.gpu

D = 128


def _pages_from_export(idx_k, val_k, idx_v, val_v, P, k_slots, perm):
    """Lay exported sparse vectors out as pages (the layout the header
    documents: pages of P/32 blocks of 32 tokens); page slots follow the
    permutation ``perm``."""
    units, L, ks = idx_k.shape
    ppu = max(1, -(-L // P))
    page_bytes = P * k_slots * 6
    block_bytes = 192 * k_slots
    pool = np.zeros((units * ppu, page_bytes), np.uint8)
    table = np.empty(units * ppu, np.int32)
    for u in range(units):
        for pg in range(ppu):
            phys = perm[u * ppu + pg]
            table[u * ppu + pg] = phys
            for q in range(P // 32):
                blk = pool[phys, q * block_bytes:(q + 1) * block_bytes]
                t0 = pg * P + q * 32
                t1 = min(L, t0 + 32)
                if t1 <= t0:
                    continue
                for voff, idx, val in ((0, idx_k, val_k), (96 * k_slots, idx_v, val_v)):
                    ioff = voff + 64 * k_slots
                    vals = blk[voff:voff + 64 * k_slots].view(np.uint16).reshape(k_slots // 8, 32, 8)
                    inds = blk[ioff:ioff + 32 * k_slots].reshape(k_slots // 8, 32, 8)
                    for r in range(ks):
                        vals[r // 8, :t1 - t0, r % 8] = val[u, t0:t1, r].view(np.uint16)
                        inds[r // 8, :t1 - t0, r % 8] = idx[u, t0:t1, r]
    return pool, table, ppu


def test_decode_noalloc_matches_decode_twice():
    import torch

    from paper_2511_18936_gb300 import swan

    dev = torch.device("cuda")
    B, H, G, ks, cap, P, L = 2, 2, 2, 60, 48, 64, 700
    k_slots = 64
    R = synth.rotations(H, D, seed=5, workload=91, layer=0)
    Rv = synth.rotations(H, D, seed=5, workload=91, layer=0, tensor_id=synth.T_R_VO)
    k = synth.lowrank_kv(B, H, L, D, 6, 91, 0, synth.T_K)
    v = synth.lowrank_kv(B, H, L, D, 6, 91, 0, synth.T_V)
    q1 = torch.from_numpy(synth.gaussian_fp16((B, H * G, D), 7, 91, 0, synth.T_Q)).to(dev)
    q2 = torch.from_numpy(synth.gaussian_fp16((B, H * G, D), 8, 91, 0, synth.T_Q, scale=3.0)).to(dev)

    Rt, Rvt = torch.from_numpy(R)[None].to(dev), torch.from_numpy(Rv)[None].to(dev)
    ctx = swan.Context(Rt, Rvt, num_layers=1, batch=B, n_q_heads=H * G, n_kv_heads=H, k_store=ks,
                       buffer_cap=cap, max_seq=L, page_tokens=P)
    kt, vt = torch.from_numpy(k).to(dev), torch.from_numpy(v).to(dev)
    ctx.append(0, kt[:, :, :333].contiguous(), vt[:, :, :333].contiguous())
    ctx.append(0, kt[:, :, 333:].contiguous(), vt[:, :, 333:].contiguous())
    info = ctx.query(0)

    # the caller's copy of the cache, in caller-owned (torch) device memory
    units = B * H
    ik, vk = ctx.export_sparse(0, "k")
    iv, vv = ctx.export_sparse(0, "v")
    Ls = info.sparse_len
    ppu = max(1, -(-Ls // P))
    perm = np.random.default_rng(0).permutation(units * ppu)
    pool, table, ppu = _pages_from_export(ik.reshape(units, Ls, ks), vk.reshape(units, Ls, ks),
                                          iv.reshape(units, Ls, ks), vv.reshape(units, Ls, ks),
                                          P, k_slots, perm)
    nb = info.buffer_len
    start = 5
    ring_k = np.zeros((units, cap, D), np.float16)
    ring_v = np.zeros((units, cap, D), np.float16)
    bk = ctx.export_buffer(0, "k").reshape(units, nb, D)
    bv = ctx.export_buffer(0, "v").reshape(units, nb, D)
    for i in range(nb):
        ring_k[:, (start + i) % cap] = bk[:, i]
        ring_v[:, (start + i) % cap] = bv[:, i]
    t_pool = torch.from_numpy(pool).to(dev)
    t_table = torch.from_numpy(table).to(dev)
    t_rk, t_rv = torch.from_numpy(ring_k).to(dev), torch.from_numpy(ring_v).to(dev)
    t_R = torch.from_numpy(R).to(dev).contiguous()
    t_RvoT = torch.from_numpy(np.ascontiguousarray(Rv.transpose(0, 2, 1))).to(dev)

    def view(k_active):
        return swan.CacheView(t_pool.data_ptr(), t_table.data_ptr(), units * ppu, ppu, P, k_slots,
                              k_active, t_rk.data_ptr(), t_rv.data_ptr(), cap, start, nb, Ls,
                              B, H * G, H, D, t_R.data_ptr(), t_RvoT.data_ptr())

    # two calls in a row, each checked against the context's own decode
    for q, k_active in ((q1, ks), (q2, 29)):
        ctx.set_k(k_active)
        want = ctx.decode(0, q)
        got = torch.empty_like(q)
        swan.decode_noalloc(view(k_active), q, got)
        torch.cuda.synchronize()
        err = (got.float() - want.float()).abs().max().item()
        assert err <= TOL_OUT, err
    ctx.check()
    ctx.check_guards()
    ctx.close()

    # sizes beyond the static scratch are rejected with a clear error
    big = view(ks)
    big.batch = 512
    with pytest.raises(swan.SwanError) as e:
        swan.decode_noalloc(big, torch.empty((512, H * G, D), dtype=torch.float16, device=dev),
                            torch.empty((512, H * G, D), dtype=torch.float16, device=dev))
    assert e.value.status == swan.ERR_INVALID_ARG and "static scratch" in str(e.value)
