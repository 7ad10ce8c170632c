"""CUDA path vs the CPU oracle, through the C ABI (needs a GB300)."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2511_18936_gb300 import synth
from tests.helpers import TOL_OUT, check_topk_near_ties, fp16_ulp_distance, run_ops

pytestmark = pytest.mark.gpu

D = 128


def _rot(H, seed, tensor_id=synth.T_R_QK):
    return synth.rotations(H, D, seed=seed, workload=90, layer=0, tensor_id=tensor_id)


def _kv(B, H, T, seed, offset=0):
    k = synth.lowrank_kv(B, H, T, D, seed, 90, 0, synth.T_K, offset)
    v = synth.lowrank_kv(B, H, T, D, seed, 90, 0, synth.T_V, offset)
    return k, v


def _q(B, Hq, seed, scale=1.0):
    return synth.gaussian_fp16((B, Hq, D), seed, 90, 0, synth.T_Q, scale=scale)


def _tricky_vectors(n, seed):
    """fp16 vectors with many exact magnitude ties, +-0 and wide ranges."""
    g = np.random.default_rng(seed)
    x = g.integers(-4, 5, size=(n, D)).astype(np.float16)
    x[::3] = (g.standard_normal((x[::3].shape[0], D)) * 30).astype(np.float16)
    x[1::5, ::7] = np.float16(-0.0)
    x[2::7] = np.float16(1.5)  # all equal magnitudes
    return x


# ---------------------------------------------------------------------------
# Pruning: bit-exact on identical rotated inputs (R = I on both sides)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("k_store,cap,P", [(64, 5, 128), (60, 0, 32), (128, 64, 64), (1, 3, 32),
                                           (8, 200, 256), (56, 128, 128)])
def test_prune_bitexact_on_identical_rotated_inputs(k_store, cap, P):
    B, H = 2, 3
    eye = np.broadcast_to(np.eye(D, dtype=np.float32), (H, D, D)).copy()
    # oracle-side rotation with a real R, rounded to fp16: the "already rotated"
    # inputs that both sides receive (R = I keeps them exact on the GPU)
    R = _rot(H, 1)
    kraw, vraw = _kv(B, H, 301, seed=2)
    k16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", kraw.astype(np.float64), R.astype(np.float64)))
    v16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", vraw.astype(np.float64), R.astype(np.float64)))
    k16[0, 0, :40] = _tricky_vectors(40, 3)
    v16[1, 2, :40] = _tricky_vectors(40, 4)
    splits = [0, 37, 38, 138, 139, 301]
    ops = []
    for a, b in zip(splits[:-1], splits[1:]):
        ops.append(("append", k16[:, :, a:b].copy(), v16[:, :, a:b].copy()))
    ops.append(("flush",))
    ctx, ref, _ = run_ops(ops, eye, None, B=B, H_kv=H, G=1, k_store=k_store, cap=cap, page_tokens=P)
    for which, ri, rv in (("k", ref.sp_idx_k, ref.sp_val_k), ("v", ref.sp_idx_v, ref.sp_val_v)):
        gi, gv = ctx.export_sparse(0, which)
        assert np.array_equal(gi, ri), which
        assert np.array_equal(gv.view(np.uint16), rv.view(np.uint16)), which
    ctx.close()


@pytest.mark.parametrize("k_store,k_store_v,fmt,cap", [(64, 64, "fp16", 5), (128, 40, "fp16", 0),
                                                      (40, 128, "fp8_e4m3", 16), (8, 64, "fp8_e4m3", 3),
                                                      (65, 63, "fp16", 7)])
def test_bulk_prune_bitexact_on_tricky_vectors(k_store, k_store_v, fmt, cap):
    """The bulk append (batch x T > 256 vectors: tensor-core rotation, register
    sorting networks, two lanes per vector) on vectors with many exact
    magnitude ties, +-0, all-equal magnitudes and values beyond the E4M3
    range, in every tile of the append including the ragged last one; keep
    counts on both sides of 64 (the top-half and the full-sort paths) and not
    multiples of 8 (padded chunks)."""
    B, H, T = 2, 3, 300
    eye = np.broadcast_to(np.eye(D, dtype=np.float32), (H, D, D)).copy()
    R = _rot(H, 7)
    kraw, vraw = _kv(B, H, T, seed=8)
    k16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", kraw.astype(np.float64), R.astype(np.float64)))
    v16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", vraw.astype(np.float64), R.astype(np.float64)))
    for i, (b, h, t0) in enumerate([(0, 0, 0), (1, 2, 130), (0, 1, 260), (1, 0, 90)]):
        k16[b, h, t0:t0 + 40] = _tricky_vectors(40, 20 + i)
        v16[b, (h + 1) % H, t0:t0 + 40] = _tricky_vectors(40, 30 + i) * np.float16(20)
    ops = [("append", k16, v16), ("flush",)]
    ctx, ref, _ = run_ops(ops, eye, None, B=B, H_kv=H, G=1, k_store=k_store, cap=cap, value_format=fmt,
                          k_store_v=k_store_v)
    for which, ri, rv in (("k", ref.sp_idx_k, ref.sp_val_k), ("v", ref.sp_idx_v, ref.sp_val_v)):
        gi, gv = ctx.export_sparse(0, which)
        assert np.array_equal(gi, ri), which
        assert np.array_equal(gv.view(np.uint16), rv.view(np.uint16)), which
    ctx.check()
    ctx.check_guards()
    ctx.close()


def test_buffer_contents_bitexact_on_identical_inputs():
    B, H = 1, 2
    eye = np.broadcast_to(np.eye(D, dtype=np.float32), (H, D, D)).copy()
    k16 = _tricky_vectors(2 * 50, 5).reshape(1, 2, 50, D)
    v16 = _tricky_vectors(2 * 50, 6).reshape(1, 2, 50, D)
    ops = [("append", k16[:, :, :7].copy(), v16[:, :, :7].copy()),
           ("append", k16[:, :, 7:30].copy(), v16[:, :, 7:30].copy()),
           ("append", k16[:, :, 30:].copy(), v16[:, :, 30:].copy())]
    ctx, ref, _ = run_ops(ops, eye, None, B=B, H_kv=H, G=1, k_store=16, cap=24)
    assert np.array_equal(ctx.export_buffer(0, "k").view(np.uint16), ref.buf_k.view(np.uint16))
    assert np.array_equal(ctx.export_buffer(0, "v").view(np.uint16), ref.buf_v.view(np.uint16))
    ctx.close()


# ---------------------------------------------------------------------------
# Rotation: fp32 arithmetic on the GPU vs fp64 in the oracle, both rounded
# to fp16; they differ only where the fp32 error straddles a rounding point
# ---------------------------------------------------------------------------

def test_rotation_within_fp32_error_bound():
    B, H = 2, 4
    R, Rv = _rot(H, 7), _rot(H, 7, synth.T_R_VO)
    k, v = _kv(B, H, 300, seed=8)
    ops = [("append", k, v)]
    ctx, ref, _ = run_ops(ops, R, Rv, B=B, H_kv=H, G=1, k_store=64, cap=300)
    for which, want, x, Rm in (("k", ref.buf_k, k, R), ("v", ref.buf_v, v, Rv)):
        got = ctx.export_buffer(0, which)
        y64 = np.einsum("bhti,hij->bhtj", x.astype(np.float64), Rm.astype(np.float64))
        # fp32 dot of 128 terms: |y32 - y64| <= 128 * 2^-24 * sum_i |x_i R_ij|;
        # then one fp16 rounding: half an fp16 ulp
        bound = 128 * 2.0 ** -24 * np.einsum("bhti,hij->bhtj", np.abs(x.astype(np.float64)),
                                             np.abs(Rm.astype(np.float64)))
        half_ulp = 0.5 * np.spacing(np.abs(got)).astype(np.float64)
        err = np.abs(got.astype(np.float64) - y64)
        assert (err <= half_ulp + bound).all(), (which, (err - half_ulp - bound).max())
        dist = fp16_ulp_distance(got, want)
        assert (dist > 0).mean() < 0.01, (which, (dist > 0).mean())
    ctx.close()


def test_direct_and_buffered_pruning_agree():
    """Tokens pruned straight from the append and tokens pruned later from
    the ring are the same function of the same fp16 vector."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, H, T = 2, 2, 333
    R = _rot(H, 9)
    k, v = _kv(B, H, T, seed=10)
    Rt = torch.from_numpy(R)[None].cuda()
    a = swan.Context(Rt, num_layers=1, batch=B, n_q_heads=H, n_kv_heads=H, k_store=48,
                     buffer_cap=0, max_seq=T)
    b = swan.Context(Rt, num_layers=1, batch=B, n_q_heads=H, n_kv_heads=H, k_store=48,
                     buffer_cap=T, max_seq=T)
    kt, vt = torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda()
    a.append(0, kt, vt)
    b.append(0, kt, vt)
    b.flush(0)
    for which in ("k", "v"):
        ia, va = a.export_sparse(0, which)
        ib, vb = b.export_sparse(0, which)
        assert np.array_equal(ia, ib) and np.array_equal(va.view(np.uint16), vb.view(np.uint16))
    a.close()
    b.close()


def test_small_and_bulk_append_paths_agree():
    """One bulk append of T tokens per sequence (tensor-core rotation) and the
    same tokens appended one per call (CUDA-core rotation, evicting one
    buffered vector each time) hold the same tokens in the same places; the
    two fp32 rotations round to the same fp16 vector except within an ulp,
    so entries agree except at near-ties (and both are valid top-k)."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, H, T, cap, ks = 4, 2, 150, 40, 40
    R, Rv = _rot(H, 13), _rot(H, 13, synth.T_R_VO)
    k, v = _kv(B, H, T, seed=14)
    Rt, Rvt = torch.from_numpy(R)[None].cuda(), torch.from_numpy(Rv)[None].cuda()
    kw = dict(num_layers=1, batch=B, n_q_heads=H, n_kv_heads=H, k_store=ks, buffer_cap=cap,
              max_seq=T, page_tokens=32)
    a = swan.Context(Rt, Rvt, **kw)
    b = swan.Context(Rt, Rvt, **kw)
    kt, vt = torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda()
    a.append(0, kt, vt)
    for t in range(T):
        b.append(0, kt[:, :, t:t + 1].contiguous(), vt[:, :, t:t + 1].contiguous())
    for which, x, Rm in (("k", k, R), ("v", v, Rv)):
        y64 = np.einsum("bhti,hij->bhtj", x.astype(np.float64), Rm.astype(np.float64))
        ia, va = a.export_sparse(0, which)
        ib, vb = b.export_sparse(0, which)
        n_sp = T - cap
        assert ia.shape == ib.shape == (B, H, n_sp, ks)
        for idx, vals in ((ia, va), (ib, vb)):
            check_topk_near_ties(y64[:, :, :n_sp], idx, vals, ks)
        assert (ia == ib).all(-1).mean() > 0.97
        # the buffered vectors: both within the fp32-dot bound of the exact
        # rotation (then one fp16 rounding), and nearly all identical
        ba, bb = a.export_buffer(0, which), b.export_buffer(0, which)
        xb = x[:, :, n_sp:].astype(np.float64)
        bound = 128 * 2.0 ** -24 * np.einsum("bhti,hij->bhtj", np.abs(xb), np.abs(Rm.astype(np.float64)))
        for got in (ba, bb):
            half_ulp = 0.5 * np.spacing(np.abs(got)).astype(np.float64)
            assert (np.abs(got.astype(np.float64) - y64[:, :, n_sp:]) <= half_ulp + bound).all()
        assert (ba.view(np.uint16) != bb.view(np.uint16)).mean() < 0.01
    a.check()
    b.check()
    a.close()
    b.close()


def test_index_parity_end_to_end_with_near_tie_exemption():
    B, H = 2, 2
    R, Rv = _rot(H, 11), _rot(H, 11, synth.T_R_VO)
    k, v = _kv(B, H, 500, seed=12)
    ops = [("append", k[:, :, :200].copy(), v[:, :, :200].copy()),
           ("append", k[:, :, 200:].copy(), v[:, :, 200:].copy()), ("flush",)]
    ctx, ref, _ = run_ops(ops, R, Rv, B=B, H_kv=H, G=1, k_store=64, cap=32)
    for which, x, Rm, ri in (("k", k, R, ref.sp_idx_k), ("v", v, Rv, ref.sp_idx_v)):
        gi, gv = ctx.export_sparse(0, which)
        y64 = np.einsum("bhti,hij->bhtj", x.astype(np.float64), Rm.astype(np.float64))
        check_topk_near_ties(y64, gi, gv, 64)
        same = (gi == ri).all(-1).mean()
        assert same > 0.97, (which, same)
    ctx.close()


# ---------------------------------------------------------------------------
# Decode: outputs within 2e-3 of the oracle at every keep level
# ---------------------------------------------------------------------------

DECODE_CASES = [
    # B, H_kv, G, L_total, cap, k_store, k_actives, page_tokens
    (1, 1, 1, 1088, 64, 64, (64, 32, 1), 0),        # the 1-head latency shape
    (2, 2, 1, 1000, 64, 64, (64, 57), 128),         # one unit over many CTAs
    (4, 8, 1, 2050, 128, 64, (64,), 128),           # CTAs spanning units
    (2, 2, 4, 1500, 128, 56, (56, 48, 13), 64),     # GQA G = 4
    (2, 4, 2, 777, 16, 60, (60, 7), 32),            # G = 2, ragged everything
    (1, 2, 1, 700, 128, 128, (128, 96, 64, 48, 32), 128),  # runtime k sweep
    (3, 2, 4, 300, 0, 24, (24, 5), 32),             # no buffer at all
    (2, 2, 8, 1300, 64, 56, (56, 40, 3), 64),       # GQA G = 8 (two 16-byte q' gathers)
    (1, 2, 8, 600, 32, 128, (128, 80), 32),         # G = 8, more than 64 entries read
    (2, 1, 8, 40, 64, 32, (32, 9), 32),             # G = 8, dense buffer only
    (1, 2, 8, 333, 0, 40, (40, 17), 32),            # G = 8, no buffer at all
]


@pytest.mark.parametrize("B,H,G,L,cap,ks,kas,P", DECODE_CASES)
def test_decode_matches_oracle(B, H, G, L, cap, ks, kas, P):
    R, Rv = _rot(H, 20 + L), _rot(H, 20 + L, synth.T_R_VO)
    k, v = _kv(B, H, L, seed=L)
    q = _q(B, H * G, seed=L)
    qp = _q(B, H * G, seed=L + 1, scale=4.0)  # peaked scores
    cut = max(1, L // 3)
    ops = [("append", k[:, :, :cut].copy(), v[:, :, :cut].copy()), ("decode", q),
           ("append", k[:, :, cut:].copy(), v[:, :, cut:].copy())]
    for ka in kas:
        ops += [("set_k", ka), ("decode", q), ("decode", qp)]
    ctx, ref, outs = run_ops(ops, R, Rv, B=B, H_kv=H, G=G, k_store=ks, cap=cap, page_tokens=P)
    for got, want in outs:
        err = np.abs(got - want).max()
        assert err <= TOL_OUT, err
    ctx.close()


def test_decode_kernel_on_identical_cache_is_fp16_exact():
    """With R = I and oracle-rotated inputs both sides hold the same cache;
    the only differences left are fp32 vs fp64 arithmetic and the final fp16
    rounding: at most one fp16 ulp."""
    B, H, G = 2, 2, 2
    eye = np.broadcast_to(np.eye(D, dtype=np.float32), (H, D, D)).copy()
    R = _rot(H, 31)
    k, v = _kv(B, H, 900, seed=32)
    k16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", k.astype(np.float64), R.astype(np.float64)))
    v16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", v.astype(np.float64), R.astype(np.float64)))
    q = _q(B, H * G, seed=33, scale=3.0)
    ops = [("append", k16, v16), ("decode", q), ("set_k", 29), ("decode", q)]
    ctx, ref, outs = run_ops(ops, eye, None, B=B, H_kv=H, G=G, k_store=64, cap=100)
    for got, want in outs:
        assert fp16_ulp_distance(got.astype(np.float16), want.astype(np.float16)).max() <= 1
    ctx.close()


def test_k_prefix_equals_fresh_cache():
    """Decoding a k_store = 128 cache at k_active = k' gives the same result as
    a cache built with k_store = k' (exact re-pruning at runtime)."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, H = 2, 2
    R = _rot(H, 41)
    k, v = _kv(B, H, 600, seed=42)
    q = torch.from_numpy(_q(B, H, seed=43)).cuda()
    Rt = torch.from_numpy(R)[None].cuda()
    kt, vt = torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda()
    big = swan.Context(Rt, num_layers=1, batch=B, n_q_heads=H, n_kv_heads=H, k_store=128,
                       buffer_cap=64, max_seq=600)
    big.append(0, kt, vt)
    for ka in (32, 48, 64, 96):
        fresh = swan.Context(Rt, num_layers=1, batch=B, n_q_heads=H, n_kv_heads=H, k_store=ka,
                             buffer_cap=64, max_seq=600)
        fresh.append(0, kt, vt)
        big.set_k(ka)
        a = big.decode(0, q)
        b = fresh.decode(0, q)
        torch.cuda.synchronize()
        assert torch.equal(a, b), ka
        fresh.close()
    big.close()


def test_k_equals_d_is_dense_attention():
    """k = d: SWAN equals ordinary attention on the unrotated inputs up to the
    fp16 storage of the rotated cache (Lemmas 1 and 2)."""
    B, H = 1, 2
    R, Rv = _rot(H, 51), _rot(H, 51, synth.T_R_VO)
    k, v = _kv(B, H, 400, seed=52)
    q = _q(B, H, seed=53)
    ops = [("append", k, v), ("decode", q)]
    ctx, ref, outs = run_ops(ops, R, Rv, B=B, H_kv=H, G=1, k_store=128, cap=100)
    got = outs[0][0]
    for h in range(H):
        dense = oracle.dense_attention(q[0, h], k[0, h], v[0, h])
        assert np.abs(got[0, h] - dense).max() <= TOL_OUT
    ctx.close()


# ---------------------------------------------------------------------------
# Edge cases
# ---------------------------------------------------------------------------

def test_empty_cache_decodes_to_zero():
    import torch

    from paper_2511_18936_gb300 import swan
    R = torch.from_numpy(_rot(2, 60))[None].cuda()
    ctx = swan.Context(R, num_layers=1, batch=2, n_q_heads=4, n_kv_heads=2, k_store=64,
                       buffer_cap=8, max_seq=64)
    q = torch.from_numpy(_q(2, 4, seed=61)).cuda()
    out = ctx.decode(0, q)
    torch.cuda.synchronize()
    assert torch.count_nonzero(out).item() == 0
    ctx.close()


def test_single_token_and_buffer_only_and_sparse_only():
    B, H = 1, 1
    R = _rot(H, 70)
    k, v = _kv(B, H, 40, seed=71)
    q = _q(B, H, seed=72)
    ops = [("append", k[:, :, :1].copy(), v[:, :, :1].copy()), ("decode", q),   # one token, buffer
           ("flush",), ("decode", q),                                            # one token, sparse
           ("append", k[:, :, 1:].copy(), v[:, :, 1:].copy()), ("decode", q),   # both
           ("flush",), ("decode", q)]
    ctx, ref, outs = run_ops(ops, R, None, B=B, H_kv=H, G=1, k_store=64, cap=16)
    for got, want in outs:
        assert np.abs(got - want).max() <= TOL_OUT
    ctx.close()


def test_capacity_error_leaves_state_unchanged():
    import torch

    from paper_2511_18936_gb300 import swan
    R = torch.from_numpy(_rot(1, 80))[None].cuda()
    ctx = swan.Context(R, num_layers=1, batch=1, n_q_heads=1, n_kv_heads=1, k_store=16,
                       buffer_cap=4, max_seq=50)
    k, v = _kv(1, 1, 60, seed=81)
    kt, vt = torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda()
    ctx.append(0, kt[:, :, :45].contiguous(), vt[:, :, :45].contiguous())
    before = (ctx.query(0).sparse_len, ctx.query(0).buffer_len)
    with pytest.raises(swan.SwanError) as e:
        ctx.append(0, kt[:, :, 45:].contiguous(), vt[:, :, 45:].contiguous())
    assert e.value.status == swan.ERR_CAPACITY
    assert (ctx.query(0).sparse_len, ctx.query(0).buffer_len) == before
    with pytest.raises(swan.SwanError):
        ctx.set_k(17)
    with pytest.raises(swan.SwanError):
        ctx.decode(1, torch.zeros(1, 1, D, dtype=torch.float16, device="cuda"))
    ctx.check()
    ctx.check_guards()
    ctx.close()


def test_multi_layer_state_is_independent():
    import torch

    from paper_2511_18936_gb300 import swan
    B, H, Lyr = 2, 2, 3
    R = np.stack([_rot(H, 90 + l) for l in range(Lyr)])
    Rt = torch.from_numpy(R).cuda()
    ctx = swan.Context(Rt, num_layers=Lyr, batch=B, n_q_heads=H, n_kv_heads=H, k_store=32,
                       buffer_cap=16, max_seq=300)
    q = _q(B, H, seed=95)
    for l in range(Lyr):
        k, v = _kv(B, H, 100 + 50 * l, seed=96 + l)
        ref = oracle.SwanOracle(R[l], batch=B, n_q_heads=H, k_store=32, buffer_cap=16)
        ref.append(k, v)
        ctx.append(l, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda())
        if l == 1:
            ref.flush()
            ctx.flush(l)
        got = ctx.decode(l, torch.from_numpy(q).cuda()).float().cpu().numpy()
        assert np.abs(got - ref.decode(q)).max() <= TOL_OUT
    ctx.check()
    ctx.check_guards()
    ctx.close()


# ---------------------------------------------------------------------------
# 8-bit (E4M3) kept values (Section 4.3, Section 5.1)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("k_store,cap,P", [(64, 5, 128), (60, 0, 32), (128, 64, 64), (56, 128, 128)])
def test_fp8_prune_bitexact_on_identical_rotated_inputs(k_store, cap, P):
    B, H = 2, 3
    eye = np.broadcast_to(np.eye(D, dtype=np.float32), (H, D, D)).copy()
    R = _rot(H, 101)
    kraw, vraw = _kv(B, H, 301, seed=102)
    k16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", kraw.astype(np.float64), R.astype(np.float64)))
    v16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", vraw.astype(np.float64), R.astype(np.float64)))
    k16[0, 0, :40] = _tricky_vectors(40, 103)          # ties, +-0, values beyond 448
    v16[1, 2, :40] = _tricky_vectors(40, 104) * np.float16(20)
    ops = [("append", k16[:, :, :37].copy(), v16[:, :, :37].copy()),
           ("append", k16[:, :, 37:38].copy(), v16[:, :, 37:38].copy()),
           ("append", k16[:, :, 38:].copy(), v16[:, :, 38:].copy()), ("flush",)]
    ctx, ref, _ = run_ops(ops, eye, None, B=B, H_kv=H, G=1, k_store=k_store, cap=cap, page_tokens=P,
                          value_format="fp8_e4m3")
    assert ctx.query(0).value_format == 1
    for which, ri, rv in (("k", ref.sp_idx_k, ref.sp_val_k), ("v", ref.sp_idx_v, ref.sp_val_v)):
        gi, gv = ctx.export_sparse(0, which)
        assert np.array_equal(gi, ri), which
        assert np.array_equal(gv.view(np.uint16), rv.view(np.uint16)), which
    ctx.close()


FP8_DECODE_CASES = [
    # B, H_kv, G, L_total, cap, k_store, k_actives, page_tokens
    (2, 2, 1, 1000, 64, 64, (64, 57, 16), 128),
    (4, 8, 1, 2050, 128, 64, (64,), 128),
    (2, 2, 4, 1500, 128, 56, (56, 13), 64),
    (2, 4, 2, 777, 16, 60, (60, 7), 32),
    (1, 2, 1, 700, 128, 128, (128, 96, 32), 128),
    (2, 2, 8, 1300, 64, 56, (56, 11), 64),
]


@pytest.mark.parametrize("B,H,G,L,cap,ks,kas,P", FP8_DECODE_CASES)
def test_fp8_decode_matches_oracle(B, H, G, L, cap, ks, kas, P):
    R, Rv = _rot(H, 120 + L), _rot(H, 120 + L, synth.T_R_VO)
    k, v = _kv(B, H, L, seed=L + 7)
    q = _q(B, H * G, seed=L + 8)
    qp = _q(B, H * G, seed=L + 9, scale=4.0)
    cut = max(1, L // 3)
    ops = [("append", k[:, :, :cut].copy(), v[:, :, :cut].copy()), ("decode", q),
           ("append", k[:, :, cut:].copy(), v[:, :, cut:].copy())]
    for ka in kas:
        ops += [("set_k", ka), ("decode", q), ("decode", qp)]
    ctx, ref, outs = run_ops(ops, R, Rv, B=B, H_kv=H, G=G, k_store=ks, cap=cap, page_tokens=P,
                             value_format="fp8_e4m3")
    for got, want in outs:
        err = np.abs(got - want).max()
        assert err <= TOL_OUT, err
    ctx.close()


# ---------------------------------------------------------------------------
# Separate keep counts for keys and values (Appendix, ablation on key and
# value pruning ratios)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("fmt", ["fp16", "fp8_e4m3"])
@pytest.mark.parametrize("k_store,k_store_v,cap,P", [(40, 24, 5, 64), (16, 96, 0, 32), (128, 8, 64, 128),
                                                     (3, 61, 20, 32)])
def test_asymmetric_prune_bitexact_on_identical_rotated_inputs(fmt, k_store, k_store_v, cap, P):
    B, H = 2, 3
    eye = np.broadcast_to(np.eye(D, dtype=np.float32), (H, D, D)).copy()
    R = _rot(H, 141)
    kraw, vraw = _kv(B, H, 301, seed=142)
    k16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", kraw.astype(np.float64), R.astype(np.float64)))
    v16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", vraw.astype(np.float64), R.astype(np.float64)))
    k16[0, 0, :40] = _tricky_vectors(40, 143)
    v16[1, 2, :40] = _tricky_vectors(40, 144)
    ops = [("append", k16[:, :, :37].copy(), v16[:, :, :37].copy()),
           ("append", k16[:, :, 37:38].copy(), v16[:, :, 37:38].copy()),
           ("append", k16[:, :, 38:].copy(), v16[:, :, 38:].copy()), ("flush",)]
    ctx, ref, _ = run_ops(ops, eye, None, B=B, H_kv=H, G=1, k_store=k_store, cap=cap, page_tokens=P,
                          value_format=fmt, k_store_v=k_store_v)
    info = ctx.query(0)
    assert (info.k_store, info.k_store_v, info.k_active, info.k_active_v) == (k_store, k_store_v,
                                                                              k_store, k_store_v)
    for which, ri, rv in (("k", ref.sp_idx_k, ref.sp_val_k), ("v", ref.sp_idx_v, ref.sp_val_v)):
        gi, gv = ctx.export_sparse(0, which)
        assert gi.shape[-1] == (k_store if which == "k" else k_store_v)
        assert np.array_equal(gi, ri), which
        assert np.array_equal(gv.view(np.uint16), rv.view(np.uint16)), which
    ctx.close()


ASYM_DECODE_CASES = [
    # B, H_kv, G, L_total, cap, k_store, k_store_v, [(k_active, k_active_v)], page_tokens, fmt
    (2, 2, 1, 1000, 64, 64, 32, [(64, 32), (32, 32), (17, 9)], 128, "fp16"),
    (2, 2, 1, 1000, 64, 32, 96, [(32, 96), (8, 64), (32, 1)], 64, "fp16"),
    (2, 4, 2, 777, 16, 60, 20, [(60, 20), (7, 13)], 32, "fp16"),
    (2, 2, 4, 1500, 128, 24, 72, [(24, 72), (24, 40)], 64, "fp16"),
    (2, 2, 1, 1000, 64, 64, 32, [(64, 32), (40, 5)], 128, "fp8_e4m3"),
    (2, 2, 4, 900, 32, 96, 16, [(96, 16), (65, 16)], 32, "fp8_e4m3"),
    (2, 2, 8, 1100, 32, 40, 80, [(40, 80), (33, 71)], 64, "fp16"),
    # G = 8 with at most 64 entries read: scores from the key tile on the tensor cores
    (2, 2, 8, 1100, 32, 56, 24, [(56, 24), (13, 17)], 64, "fp16"),
    (2, 2, 8, 900, 16, 24, 56, [(24, 56), (9, 56)], 32, "fp8_e4m3"),
]


@pytest.mark.parametrize("B,H,G,L,cap,ks,ksv,kas,P,fmt", ASYM_DECODE_CASES)
def test_asymmetric_decode_matches_oracle(B, H, G, L, cap, ks, ksv, kas, P, fmt):
    R, Rv = _rot(H, 150 + L), _rot(H, 150 + L, synth.T_R_VO)
    k, v = _kv(B, H, L, seed=L + 11)
    q = _q(B, H * G, seed=L + 12)
    qp = _q(B, H * G, seed=L + 13, scale=4.0)
    cut = max(1, L // 3)
    ops = [("append", k[:, :, :cut].copy(), v[:, :, :cut].copy()), ("decode", q),
           ("append", k[:, :, cut:].copy(), v[:, :, cut:].copy())]
    for ka, kav in kas:
        ops += [("set_kv", ka, kav), ("decode", q), ("decode", qp)]
    ops += [("set_k", ks), ("decode", q)]   # set_k clamps the value count at k_store_v
    ctx, ref, outs = run_ops(ops, R, Rv, B=B, H_kv=H, G=G, k_store=ks, cap=cap, page_tokens=P,
                             value_format=fmt, k_store_v=ksv)
    assert ctx.query(0).k_active_v == min(ks, ksv)
    for got, want in outs:
        err = np.abs(got - want).max()
        assert err <= TOL_OUT, err
    ctx.close()


def test_runtime_value_prefix_equals_stored_split():
    """A symmetric k_store = 128 cache decoded at (k, k_v) gives the result of
    a cache stored with k_store = k, k_store_v = k_v: both keep the same
    leading entries of each vector."""
    import torch

    from paper_2511_18936_gb300 import swan
    dev = torch.device("cuda")
    B, H, G, L, cap = 2, 2, 2, 900, 64
    R = _rot(H, 160)
    k, v = _kv(B, H, L, seed=161)
    q = torch.from_numpy(_q(B, H * G, seed=162, scale=2.0)).to(dev)
    Rt = torch.from_numpy(R)[None].to(dev)
    kt, vt = torch.from_numpy(k).to(dev), torch.from_numpy(v).to(dev)
    full = swan.Context(Rt, num_layers=1, batch=B, n_q_heads=H * G, n_kv_heads=H, k_store=128,
                        buffer_cap=cap, max_seq=L)
    full.append(0, kt, vt)
    for ka, kav in ((48, 16), (16, 48), (64, 64)):
        split = swan.Context(Rt, num_layers=1, batch=B, n_q_heads=H * G, n_kv_heads=H, k_store=ka,
                             k_store_v=kav, buffer_cap=cap, max_seq=L)
        split.append(0, kt, vt)
        full.set_k(ka, kav)
        a = full.decode(0, q).float()
        b = split.decode(0, q).float()
        torch.cuda.synchronize()
        assert (a - b).abs().max().item() <= 1e-3, (ka, kav)
        split.check()
        split.close()
    full.check()
    full.close()


@pytest.mark.parametrize("G,fmt", [(1, "fp16"), (4, "fp8_e4m3")])
def test_maximum_buffer_page_and_keep_sizes(G, fmt):
    """The largest sizes the header allows for the dense buffer (4096 tokens)
    and a page (4096 tokens, 128 blocks), with every coordinate stored
    (k_store 128) and read back at k 128 and below: 128 buffer groups per
    unit, a sparse history over two pages, both kernel families."""
    B, H, cap, P, ks = 1, 2, 4096, 4096, 128
    L = cap + 4500
    R, Rv = _rot(H, 140 + G), _rot(H, 140 + G, synth.T_R_VO)
    k, v = _kv(B, H, L, seed=141)
    q = _q(B, H * G, seed=142, scale=2.0)
    ops = [("append", k[:, :, :5000].copy(), v[:, :, :5000].copy()), ("decode", q),
           ("append", k[:, :, 5000:].copy(), v[:, :, 5000:].copy()), ("decode", q),
           ("set_k", 100), ("decode", q), ("flush",), ("decode", q)]
    ctx, ref, outs = run_ops(ops, R, Rv, B=B, H_kv=H, G=G, k_store=ks, cap=cap, page_tokens=P,
                             value_format=fmt)
    for got, want in outs:
        assert np.abs(got - want).max() <= TOL_OUT
    ctx.close()
