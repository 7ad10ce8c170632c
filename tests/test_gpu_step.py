"""swan_append_decode, one call per serving step: the same bits as
swan_append_varlen followed by swan_decode, within tolerance of the ragged
oracle, in two launches for a decode-step append (needs a GB300)."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2511_18936_gb300 import synth
from tests.helpers import TOL_OUT

pytestmark = pytest.mark.gpu

D = 128


def _contexts(R, Rv, **kw):
    import torch

    from paper_2511_18936_gb300 import swan
    dev = torch.device("cuda")
    Rt = torch.from_numpy(np.asarray(R, np.float32))[None].to(dev).contiguous()
    Rvt = torch.from_numpy(np.asarray(Rv, np.float32))[None].to(dev).contiguous()
    return swan.Context(Rt, Rvt, num_layers=1, **kw), swan.Context(Rt, Rvt, num_layers=1, **kw)


def _steps(B, T_list, ragged, seed):
    """Per step: (T, n_new or None).  Decode steps (T = 1, some rows idle when
    ragged), an empty step, and one bulk step that takes the separate
    rotation launch."""
    gen = np.random.default_rng(seed)
    out = []
    for T in T_list:
        n = None
        if ragged:
            n = [int(x) for x in gen.integers(0, T + 1, size=B)]
            n[0] = T
        out.append((T, n))
    return out


@pytest.mark.parametrize("G,fmt,ragged,cap", [(1, "fp16", False, 8), (2, "fp16", True, 8),
                                              (4, "fp8_e4m3", False, 4), (1, "fp16", True, 0),
                                              (2, "fp8_e4m3", True, 16), (8, "fp16", True, 8)])
def test_append_decode_equals_append_then_decode(G, fmt, ragged, cap):
    import torch

    B, H_kv, k_store = 3, 2, 48
    Hq = H_kv * G
    seed = 100 + 10 * G + cap
    R = synth.rotations(H_kv, D, seed=seed, workload=96, layer=0, tensor_id=synth.T_R_QK)
    Rv = synth.rotations(H_kv, D, seed=seed, workload=96, layer=0, tensor_id=synth.T_R_VO)
    T_list = [90] + [1] * 14 + [0, 1, 40, 1, 1]  # B * 90 > 256: the bulk path
    steps = _steps(B, T_list, ragged, seed)
    max_seq = sum(T_list) + 1
    kw = dict(batch=B, n_q_heads=Hq, n_kv_heads=H_kv, k_store=k_store, buffer_cap=cap, max_seq=max_seq,
              value_format=fmt, k_store_v=32)
    fused, split = _contexts(R, Rv, **kw)
    ref = oracle.RaggedOracle(R, Rv, batch=B, n_q_heads=Hq, k_store=k_store, buffer_cap=cap, value_format=fmt,
                              k_store_v=32)
    dev = torch.device("cuda")
    for i, (T, n_new) in enumerate(steps):
        k = synth.lowrank_kv(B, H_kv, max(T, 1), D, seed, 96, i, synth.T_K)[:, :, :T].copy()
        v = synth.lowrank_kv(B, H_kv, max(T, 1), D, seed, 96, i, synth.T_V)[:, :, :T].copy()
        q = synth.gaussian_fp16((B, Hq, D), seed, 96, i, synth.T_Q)
        tk = torch.from_numpy(k).to(dev) if T else torch.empty((B, H_kv, 0, D), dtype=torch.float16, device=dev)
        tv = torch.from_numpy(v).to(dev) if T else torch.empty((B, H_kv, 0, D), dtype=torch.float16, device=dev)
        tq = torch.from_numpy(q).to(dev)
        got = fused.append_decode(0, tk, tv, tq, T=T, n_new=n_new)
        split.append(0, tk, tv, T, n_new=n_new)
        want = split.decode(0, tq)
        torch.cuda.synchronize()
        assert torch.equal(got, want), i
        assert fused.lengths(0) == split.lengths(0), i
        if T:
            ref.append(k, v, n_new)
        o = ref.decode(q)
        assert np.abs(got.float().cpu().numpy() - o).max() <= TOL_OUT, i
    assert list(fused.lengths(0)[0]) == ref.sparse_lens
    for b in range(B):
        for which in ("k", "v"):
            assert np.array_equal(fused.export_buffer_seq(0, b, which), split.export_buffer_seq(0, b, which))
            fi, fv = fused.export_sparse_seq(0, b, which)
            si, sv = split.export_sparse_seq(0, b, which)
            assert np.array_equal(fi, si) and np.array_equal(fv, sv)
    fused.check()
    split.check()
    fused.check_guards()
    split.check_guards()
    fused.close()
    split.close()


def test_append_decode_launches_and_errors():
    """A decode step is two launches (fused append + rotation, decode); the
    bulk path is three or more.  A bad q or out, or a capacity error, leaves
    the cache and `out` unchanged."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, H, cap = 2, 4, 4
    R = synth.rotations(H, D, seed=5, workload=96, layer=1, tensor_id=synth.T_R_QK)
    fused, _ = _contexts(R, R, batch=B, n_q_heads=H, n_kv_heads=H, k_store=64, buffer_cap=cap, max_seq=140)
    dev = torch.device("cuda")
    k = torch.from_numpy(synth.lowrank_kv(B, H, 130, D, 5, 96, 1, synth.T_K)).to(dev)
    v = torch.from_numpy(synth.lowrank_kv(B, H, 130, D, 5, 96, 1, synth.T_V)).to(dev)
    q = torch.from_numpy(synth.gaussian_fp16((B, H, D), 5, 96, 1, synth.T_Q)).to(dev)
    out = torch.zeros_like(q)
    n0 = fused.launch_count()
    fused.append_decode(0, k[:, :, :1].contiguous(), v[:, :, :1].contiguous(), q, out)
    assert fused.launch_count() - n0 == 2
    n0 = fused.launch_count()
    fused.append_decode(0, k, v, q, out)  # B * 130 > 256 vectors: the bulk append
    assert fused.launch_count() - n0 >= 3
    torch.cuda.synchronize()
    before = fused.lengths(0)
    snap = out.clone()
    lib = swan.load_library()
    k1, v1 = k[:, :, :1].contiguous(), v[:, :, :1].contiguous()
    # q == NULL, out overlapping q
    assert lib.swan_append_decode(fused._h, 0, k1.data_ptr(), v1.data_ptr(), 1, None, None,
                                  out.data_ptr()) == swan.ERR_INVALID_ARG
    assert lib.swan_append_decode(fused._h, 0, k1.data_ptr(), v1.data_ptr(), 1, None, q.data_ptr(),
                                  q.data_ptr()) == swan.ERR_INVALID_ARG
    # 131 + 10 tokens > max_seq 140
    k10, v10 = k[:, :, :10].contiguous(), v[:, :, :10].contiguous()
    assert lib.swan_append_decode(fused._h, 0, k10.data_ptr(), v10.data_ptr(), 10, None, q.data_ptr(),
                                  out.data_ptr()) == swan.ERR_CAPACITY
    torch.cuda.synchronize()
    assert fused.lengths(0) == before
    assert torch.equal(out, snap)
    fused.check()
    fused.close()


def test_documented_usage_matches_the_oracle():
    """The flow the README shows (prefill, decode, a fused serving step, a
    smaller runtime k), on layer 1 of a two-layer GQA context, against the
    oracle fed the same operations."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, Hq, Hkv, cap = 2, 4, 2, 16
    R = np.stack([synth.rotations(Hkv, D, seed=9, workload=98, layer=l) for l in range(2)])
    dev = torch.device("cuda")
    ctx = swan.Context(torch.from_numpy(R).to(dev), num_layers=2, batch=B, n_q_heads=Hq, n_kv_heads=Hkv,
                       k_store=64, buffer_cap=cap, max_seq=512)
    ref = oracle.SwanOracle(R[1], None, batch=B, n_q_heads=Hq, k_store=64, buffer_cap=cap)
    k = synth.lowrank_kv(B, Hkv, 300, D, 9, 98, 1, synth.T_K)
    v = synth.lowrank_kv(B, Hkv, 300, D, 9, 98, 1, synth.T_V)
    q = synth.gaussian_fp16((B, Hq, D), 9, 98, 1, synth.T_Q)
    tq = torch.from_numpy(q).to(dev)
    ctx.append(1, torch.from_numpy(k).to(dev), torch.from_numpy(v).to(dev))
    ref.append(k, v)
    outs = [(ctx.decode(1, tq), ref.decode(q))]
    k1 = synth.lowrank_kv(B, Hkv, 1, D, 9, 98, 2, synth.T_K)
    v1 = synth.lowrank_kv(B, Hkv, 1, D, 9, 98, 2, synth.T_V)
    outs.append((ctx.append_decode(1, torch.from_numpy(k1).to(dev), torch.from_numpy(v1).to(dev), tq), None))
    ref.append(k1, v1)
    outs[-1] = (outs[-1][0], ref.decode(q))
    ctx.set_k(48)
    ref.set_k(48)
    outs.append((ctx.decode(1, tq), ref.decode(q)))
    ctx.check()
    ctx.check_guards()
    for got, want in outs:
        assert np.abs(got.float().cpu().numpy() - want).max() <= TOL_OUT
    assert ctx.lengths(0) == ([0] * B, [0] * B)  # the other layer is untouched
    ctx.close()
