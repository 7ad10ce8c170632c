"""Rows of different lengths and the shared page pool (swan_append_varlen,
swan_reset_sequence, pool_pages) against the ragged oracle (needs a GB300)."""
from __future__ import annotations

import copy

import numpy as np
import pytest

import oracle
from paper_2511_18936_gb300 import synth
from tests.helpers import TOL_OUT

pytestmark = pytest.mark.gpu

D = 128


def _rot(H, seed, tensor_id=synth.T_R_QK):
    return synth.rotations(H, D, seed=seed, workload=95, layer=0, tensor_id=tensor_id)


def _kv(B, H, T, seed):
    return (synth.lowrank_kv(B, H, T, D, seed, 95, 0, synth.T_K),
            synth.lowrank_kv(B, H, T, D, seed, 95, 0, synth.T_V))


def _q(B, Hq, seed, scale=1.0):
    return synth.gaussian_fp16((B, Hq, D), seed, 95, 0, synth.T_Q, scale=scale)


def run_ragged(ops, R, Rv, *, B, H_kv, G, k_store, cap, max_seq, page_tokens=0, value_format="fp16",
               k_store_v=None, pool_pages=0):
    """Replay ragged ops on the ragged oracle and a libswan context.
    ops: ("append", k, v, n_new | None) | ("flush",) | ("reset", b) |
    ("fork", src, dst) | ("set_k", k[, k_v]) | ("decode", q).  Lengths are compared after every
    op, outputs after every decode."""
    import torch

    from paper_2511_18936_gb300 import swan
    dev = torch.device("cuda")
    ref = oracle.RaggedOracle(R, Rv, batch=B, n_q_heads=H_kv * G, k_store=k_store, buffer_cap=cap,
                              value_format=value_format, k_store_v=k_store_v)
    Rt = torch.from_numpy(np.asarray(R, np.float32))[None].to(dev).contiguous()
    Rvt = None if Rv is None else torch.from_numpy(np.asarray(Rv, np.float32))[None].to(dev).contiguous()
    ctx = swan.Context(Rt, Rvt, num_layers=1, batch=B, n_q_heads=H_kv * G, n_kv_heads=H_kv, k_store=k_store,
                       buffer_cap=cap, max_seq=max_seq, page_tokens=page_tokens, value_format=value_format,
                       k_store_v=k_store_v or 0, pool_pages=pool_pages)
    worst = 0.0
    for op in ops:
        if op[0] == "append":
            ref.append(op[1], op[2], op[3])
            ctx.append(0, torch.from_numpy(op[1]).to(dev), torch.from_numpy(op[2]).to(dev), n_new=op[3])
        elif op[0] == "flush":
            ref.flush()
            ctx.flush(0)
        elif op[0] == "reset":
            ref.reset(op[1])
            ctx.reset_sequence(op[1])
        elif op[0] == "fork":  # the oracle's row dst becomes a copy of row src
            ref.rows[op[2]] = copy.deepcopy(ref.rows[op[1]])
            ctx.fork_sequence(op[1], op[2])
        elif op[0] == "set_k":
            ref.set_k(*op[1:])
            ctx.set_k(*op[1:])
        elif op[0] == "decode":
            want = ref.decode(op[1])
            got = ctx.decode(0, torch.from_numpy(op[1]).to(dev)).float().cpu().numpy()
            err = float(np.abs(got - want).max())
            worst = max(worst, err)
            assert err <= TOL_OUT, err
        else:
            raise ValueError(op)
        sp, bf = ctx.lengths(0)
        assert sp == ref.sparse_lens and bf == ref.buffer_lens, (op[0], sp, ref.sparse_lens, bf, ref.buffer_lens)
    ctx.check()
    ctx.check_guards()
    return ctx, ref, worst


RAGGED_CASES = [
    # B, H_kv, G, cap, k_store, k_store_v, P, fmt
    (5, 2, 1, 64, 64, None, 128, "fp16"),
    (4, 2, 4, 32, 56, 24, 64, "fp16"),
    (3, 2, 2, 16, 40, None, 32, "fp8_e4m3"),
    (6, 1, 1, 0, 24, None, 32, "fp16"),       # no buffer
]


@pytest.mark.parametrize("B,H,G,cap,ks,ksv,P,fmt", RAGGED_CASES)
def test_ragged_rows_match_oracle(B, H, G, cap, ks, ksv, P, fmt):
    R, Rv = _rot(H, 10 + B), _rot(H, 10 + B, synth.T_R_VO)
    T0 = 1500
    k, v = _kv(B, H, T0 + 400, seed=B)
    lens = [0, 1, 33, 700, 1500, 64][:B]
    q, qp = _q(B, H * G, seed=B), _q(B, H * G, seed=B + 1, scale=4.0)
    ops = [("append", k[:, :, :T0].copy(), v[:, :, :T0].copy(), lens), ("decode", q), ("decode", qp)]
    t = T0
    # decode steps where only some rows take a token (small-append path)
    for step in range(3):
        n_new = [(b + step) % 2 for b in range(B)]
        ops += [("append", k[:, :, t:t + 1].copy(), v[:, :, t:t + 1].copy(), n_new), ("decode", q)]
        t += 1
    # a ragged bulk append (prune of evicted buffer rows + rotation launch)
    ops += [("append", k[:, :, t:t + 200].copy(), v[:, :, t:t + 200].copy(), [200, 0, 150, 7, 199, 1][:B]),
            ("decode", qp), ("set_k", max(1, ks // 2)), ("decode", q), ("set_k", ks)]
    t += 200
    # a finished request leaves, a new one arrives in its row
    ops += [("reset", 2 % B), ("decode", q),
            ("append", k[:, :, t:t + 90].copy(), v[:, :, t:t + 90].copy(), [0, 0, 90, 0, 0, 0][:B]),
            ("decode", q), ("flush",), ("decode", qp)]
    ctx, ref, worst = run_ragged(ops, R, Rv, B=B, H_kv=H, G=G, k_store=ks, cap=cap, max_seq=T0 + 400,
                                 page_tokens=P, value_format=fmt, k_store_v=ksv)
    assert ctx.query(0).uniform == 0
    ctx.close()


def test_ragged_prune_bitexact_per_row():
    """R = I and oracle-rotated inputs: every row's sparse history and buffer
    are bit-identical to the oracle's, row by row."""
    B, H = 3, 2
    eye = np.broadcast_to(np.eye(D, dtype=np.float32), (H, D, D)).copy()
    R = _rot(H, 40)
    kraw, vraw = _kv(B, H, 400, seed=41)
    k16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", kraw.astype(np.float64), R.astype(np.float64)))
    v16 = oracle.to_fp16(np.einsum("bhti,hij->bhtj", vraw.astype(np.float64), R.astype(np.float64)))
    ops = [("append", k16[:, :, :300].copy(), v16[:, :, :300].copy(), [300, 5, 129]),
           ("append", k16[:, :, 300:301].copy(), v16[:, :, 300:301].copy(), [1, 0, 1]),
           ("append", k16[:, :, 301:400].copy(), v16[:, :, 301:400].copy(), [99, 60, 0])]
    ctx, ref, _ = run_ragged(ops, eye, None, B=B, H_kv=H, G=1, k_store=48, cap=20, max_seq=400, page_tokens=32)
    for b in range(B):
        row = ref.rows[b]
        for which, ri, rv in (("k", row.sp_idx_k, row.sp_val_k), ("v", row.sp_idx_v, row.sp_val_v)):
            gi, gv = ctx.export_sparse_seq(0, b, which)
            assert np.array_equal(gi, ri[0]), (b, which)
            assert np.array_equal(gv.view(np.uint16), rv[0].view(np.uint16)), (b, which)
        assert np.array_equal(ctx.export_buffer_seq(0, b, "k").view(np.uint16), row.buf_k[0].view(np.uint16))
    from paper_2511_18936_gb300 import swan
    with pytest.raises(swan.SwanError):
        ctx.export_sparse(0, "k")  # rows differ: whole-batch export refuses
    ctx.close()


def test_uniform_batch_keeps_the_uniform_path():
    """Equal appends keep every row equal: the uniform kernels run (no ragged
    table) and results match the batched oracle."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, H = 2, 2
    R = _rot(H, 50)
    k, v = _kv(B, H, 300, seed=51)
    q = _q(B, H, seed=52)
    ctx = swan.Context(torch.from_numpy(R)[None].cuda(), num_layers=1, batch=B, n_q_heads=H, n_kv_heads=H,
                       k_store=32, buffer_cap=16, max_seq=300)
    ctx.append(0, torch.from_numpy(k[:, :, :200]).cuda(), torch.from_numpy(v[:, :, :200]).cuda(), n_new=[200, 200])
    assert ctx.query(0).uniform == 1
    ref = oracle.SwanOracle(R, batch=B, n_q_heads=H, k_store=32, buffer_cap=16)
    ref.append(k[:, :, :200], v[:, :, :200])
    got = ctx.decode(0, torch.from_numpy(q).cuda()).float().cpu().numpy()
    assert np.abs(got - ref.decode(q)).max() <= TOL_OUT
    ctx.close()


def test_page_pool_shared_by_rows():
    """A pool smaller than batch x max_seq: rows take pages as they grow, an
    append that would exhaust the pool fails with CAPACITY and changes
    nothing, a reset returns the row's pages, and reused (dirty) pages decode
    correctly."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, H, G, P, cap, ks = 3, 2, 2, 64, 16, 40
    R, Rv = _rot(H, 60), _rot(H, 60, synth.T_R_VO)
    k, v = _kv(B, H, 2000, seed=61)
    q = _q(B, H * G, seed=62)
    pool = 2 * H * 8 + 4  # room for two rows of 8 pages per head, plus 4 pages
    ops = [("append", k[:, :, :500].copy(), v[:, :, :500].copy(), [500, 0, 300]), ("decode", q)]
    ctx, ref, _ = run_ragged(ops, R, Rv, B=B, H_kv=H, G=G, k_store=ks, cap=cap, max_seq=2000, page_tokens=P,
                             pool_pages=pool)
    info = ctx.query(0)
    # row 0: 484 sparse tokens -> 8 pages per head; row 2: 284 -> 5 pages per head
    assert info.pool_pages == pool and info.free_pages == pool - H * (8 + 5)
    dev = torch.device("cuda")
    big_k, big_v = torch.from_numpy(k[:, :, 500:1500].copy()).to(dev), torch.from_numpy(v[:, :, 500:1500].copy()).to(dev)
    before = ctx.lengths(0)
    with pytest.raises(swan.SwanError) as e:
        ctx.append(0, big_k, big_v, n_new=[0, 1000, 0])
    assert e.value.status == swan.ERR_CAPACITY
    assert ctx.lengths(0) == before and ctx.query(0).free_pages == info.free_pages
    # free row 0 and give its pages to row 1
    ctx.reset_sequence(0)
    ref.reset(0)
    assert ctx.query(0).free_pages == info.free_pages + H * 8
    ctx.append(0, big_k[:, :, :600].contiguous(), big_v[:, :, :600].contiguous(), n_new=[0, 600, 0])
    ref.append(k[:, :, 500:1100], v[:, :, 500:1100], [0, 600, 0])
    got = ctx.decode(0, torch.from_numpy(q).to(dev)).float().cpu().numpy()
    assert np.abs(got - ref.decode(q)).max() <= TOL_OUT
    ctx.flush(0)
    ref.flush()
    got = ctx.decode(0, torch.from_numpy(q).to(dev)).float().cpu().numpy()
    assert np.abs(got - ref.decode(q)).max() <= TOL_OUT
    assert ctx.lengths(0) == (ref.sparse_lens, ref.buffer_lens)
    ctx.check()
    ctx.check_guards()
    ctx.close()


def test_bulk_append_tiles_and_alignment():
    """Bulk appends whose token count leaves a partial 128-vector tile (T = 129
    and T = 255 per row, rows taking different counts), then a decode; and a
    misaligned input is refused before anything changes."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, H, G = 3, 2, 2
    R, Rv = _rot(H, 70), _rot(H, 70, synth.T_R_VO)
    k, v = _kv(B, H, 400, seed=71)
    q = _q(B, H * G, seed=72)
    ops = [("append", k[:, :, :129].copy(), v[:, :, :129].copy(), [129, 128, 1]), ("decode", q),
           ("append", k[:, :, 129:384].copy(), v[:, :, 129:384].copy(), [255, 0, 200]), ("decode", q)]
    ctx, ref, _ = run_ragged(ops, R, Rv, B=B, H_kv=H, G=G, k_store=48, cap=16, max_seq=400, page_tokens=64)
    before = ctx.lengths(0)
    buf = torch.from_numpy(np.concatenate([k[:, :, 384:], k[:, :, 384:]], axis=2)).cuda()
    mis = buf.view(-1)[1:1 + B * H * 8 * D].view(B, H, 8, D)  # 2-byte offset
    with pytest.raises(swan.SwanError) as e:
        ctx.append(0, mis, mis)
    assert e.value.status == swan.ERR_INVALID_ARG and "aligned" in str(e.value)
    assert ctx.lengths(0) == before
    ctx.check()
    ctx.check_guards()
    ctx.close()


def test_ragged_fp8_separate_counts_and_pool():
    """Everything at once: rows of different lengths, E4M3 values, keys and
    values keeping different counts, a shared page pool, grouped-query heads."""
    B, H, G, P = 4, 2, 4, 32
    R, Rv = _rot(H, 80), _rot(H, 80, synth.T_R_VO)
    k, v = _kv(B, H, 900, seed=81)
    q = _q(B, H * G, seed=82, scale=2.0)
    pool = H * (900 // P + 2) * 3
    ops = [("append", k[:, :, :600].copy(), v[:, :, :600].copy(), [600, 17, 0, 333]), ("decode", q),
           ("set_k", 40, 12), ("decode", q),
           ("append", k[:, :, 600:601].copy(), v[:, :, 600:601].copy(), [1, 1, 0, 1]), ("decode", q),
           ("reset", 0), ("append", k[:, :, 601:900].copy(), v[:, :, 601:900].copy(), [299, 0, 299, 0]),
           ("decode", q), ("flush",), ("decode", q)]
    ctx, ref, _ = run_ragged(ops, R, Rv, B=B, H_kv=H, G=G, k_store=40, cap=24, max_seq=900, page_tokens=P,
                             value_format="fp8_e4m3", k_store_v=24, pool_pages=pool)
    ctx.close()


FORK_CASES = [
    # B, H_kv, G, cap, k_store, P, fmt
    (3, 2, 2, 32, 48, 64, "fp16"),
    (3, 2, 1, 16, 64, 32, "fp8_e4m3"),
    (4, 2, 8, 24, 56, 64, "fp16"),
]


@pytest.mark.parametrize("B,H,G,cap,ks,P,fmt", FORK_CASES)
def test_fork_sequence_matches_oracle(B, H, G, cap, ks, P, fmt):
    """Forked rows (swan_fork_sequence) against the oracle: the fork shares
    the source's pages and copies its buffer, then both rows take different
    tokens (the first appends write into the shared, partly filled last
    page: copy on write), a fork onto a row that already holds tokens, a
    flush, a reset and a second fork of a fork."""
    R, Rv = _rot(H, 90 + G), _rot(H, 90 + G, synth.T_R_VO)
    k, v = _kv(B, H, 1400, seed=91 + G)
    q = _q(B, H * G, seed=92, scale=2.0)
    n0 = [300] + [0] * (B - 2) + [150]
    ops = [("append", k[:, :, :300].copy(), v[:, :, :300].copy(), n0), ("decode", q),
           ("fork", 0, 1), ("decode", q),
           ("append", k[:, :, 300:337].copy(), v[:, :, 300:337].copy(), [37, 21] + [5] * (B - 2)), ("decode", q),
           ("append", k[:, :, 337:338].copy(), v[:, :, 337:338].copy(), [1] * B), ("decode", q),
           ("fork", 1, B - 1), ("decode", q),
           ("append", k[:, :, 338:700].copy(), v[:, :, 338:700].copy(), [362, 0] + [100] * (B - 2)), ("decode", q),
           ("flush",), ("decode", q),
           ("fork", B - 1, 0), ("reset", 1), ("decode", q),
           ("append", k[:, :, 700:1300].copy(), v[:, :, 700:1300].copy(), [600, 300] + [77] * (B - 2)),
           ("decode", q)]
    pool = H * B * (1400 // P + 3)
    ctx, ref, _ = run_ragged(ops, R, Rv, B=B, H_kv=H, G=G, k_store=ks, cap=cap, max_seq=1400, page_tokens=P,
                             value_format=fmt, pool_pages=pool)
    for b in range(B):
        ctx.reset_sequence(b)
    info = ctx.query(0)
    assert info.free_pages == info.pool_pages  # every page back once no row holds it
    ctx.close()


def test_fork_shares_pages_and_isolates_rows():
    """Page accounting and isolation: a fork takes no page until a row
    writes into a shared page; the copy leaves the other row's output
    bit for bit unchanged; forking needs a pool and two different rows."""
    import torch

    from paper_2511_18936_gb300 import swan
    B, H, G, P, cap = 2, 2, 2, 64, 16
    R, Rv = _rot(H, 97), _rot(H, 97, synth.T_R_VO)
    k, v = _kv(B, H, 600, seed=98)
    q = torch.from_numpy(_q(B, H * G, seed=99)).cuda()
    ctx = swan.Context(torch.from_numpy(R)[None].cuda(), torch.from_numpy(Rv)[None].cuda(), num_layers=1,
                       batch=B, n_q_heads=H * G, n_kv_heads=H, k_store=32, buffer_cap=cap, max_seq=600,
                       page_tokens=P, pool_pages=64)
    kt, vt = torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda()
    ctx.append(0, kt[:, :, :216].contiguous(), vt[:, :, :216].contiguous(), n_new=[216, 0])
    free0 = ctx.query(0).free_pages                      # row 0: 200 sparse tokens, 4 pages a head
    assert free0 == 64 - H * 4
    ctx.fork_sequence(0, 1)
    assert ctx.query(0).free_pages == free0              # shared, nothing copied yet
    qq = torch.cat([q[:1], q[:1]])                       # the same query for both rows
    out = ctx.decode(0, qq).float().cpu().numpy()
    assert np.abs(out[0] - out[1]).max() <= TOL_OUT      # the same history (CTA splits may differ)
    ctx.append(0, kt[:, :, 216:220].contiguous(), vt[:, :, 216:220].contiguous(), n_new=[4, 0])
    assert ctx.query(0).free_pages == free0 - H          # row 0 copied its shared last page
    ctx.append(0, kt[:, :, 220:224].contiguous(), vt[:, :, 220:224].contiguous(), n_new=[0, 4])
    assert ctx.query(0).free_pages == free0 - H          # row 1 was the last holder: no copy
    assert ctx.lengths(0) == ([204, 204], [16, 16])
    ctx.reset_sequence(0)
    ctx.reset_sequence(1)
    assert ctx.query(0).free_pages == 64
    for a, b in ((0, 0), (0, 2), (-1, 1)):
        with pytest.raises(swan.SwanError) as e:
            ctx.fork_sequence(a, b)
        assert e.value.status == swan.ERR_INVALID_ARG
    ctx.check()
    ctx.check_guards()
    ctx.close()
    plain = swan.Context(torch.from_numpy(R)[None].cuda(), num_layers=1, batch=2, n_q_heads=H, n_kv_heads=H,
                         k_store=32, buffer_cap=cap, max_seq=600)
    with pytest.raises(swan.SwanError) as e:
        plain.fork_sequence(0, 1)
    assert e.value.status == swan.ERR_UNSUPPORTED
    plain.close()
