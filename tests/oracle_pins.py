"""Pins that tie the oracle to facts fixed by the paper or by mathematics.

Each ``pin_*`` takes the oracle module as its argument so that the same pins
can be run against deliberately broken copies of the oracle
(``test_oracle_mutants.py``): every plausible mistake must fail one of them.
"""
from __future__ import annotations

import itertools
import math
import os

import numpy as np
import torch

from paper_2511_18936_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _small_problem(seed, B=2, H_kv=2, G=1, d=16, L=40):
    gen = np.random.default_rng(seed)
    R = np.stack([synth.random_orthogonal(d, gen) for _ in range(H_kv)])
    Rv = np.stack([synth.random_orthogonal(d, gen) for _ in range(H_kv)])
    k = (gen.standard_normal((B, H_kv, L, d))).astype(np.float16)
    v = (gen.standard_normal((B, H_kv, L, d))).astype(np.float16)
    q = (gen.standard_normal((B, H_kv * G, d))).astype(np.float16)
    return R, Rv, k, v, q


# -- P1: rotation (Lemma 1 premise: P^T P = I; row-vector convention) ------

def pin_rotation_orthogonal(o):
    R = synth.rotations(4, 128, seed=0, workload=0, layer=0)
    for h in range(4):
        err = np.abs(R[h].astype(np.float64).T @ R[h].astype(np.float64) - np.eye(128)).max()
        assert err < 1e-6, err
    x = np.random.default_rng(1).standard_normal((5, 128))
    y = o.rotate(x, R[0])
    assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1), rtol=1e-6)
    assert np.allclose(o.rotate_back(y, R[0]), x, atol=1e-6)


def pin_rotation_orientation(o):
    """A permutation matrix fixes the orientation: with ``x_hat = x P`` and
    ``P[i, pi(i)] = 1``, ``x_hat[pi(i)] = x[i]`` (Section 4.2 row vectors)."""
    d = 8
    pi = np.array([3, 0, 6, 1, 7, 2, 5, 4])
    P = np.zeros((d, d))
    P[np.arange(d), pi] = 1.0
    x = np.arange(1, d + 1, dtype=np.float64)
    y = o.rotate(x, P)
    assert np.array_equal(y[pi], x), (y, x)
    # the cache state machine must use the same orientation
    st = o.SwanOracle(P[None], batch=1, n_q_heads=1, k_store=3, buffer_cap=0)
    kx = np.array([0.5, -4.0, 1.0, 8.0, -2.0, 0.25, 3.0, -0.125], np.float16)
    st.append(kx[None, None, None, :], kx[None, None, None, :])
    want_src = [3, 1, 6]  # |8|, |-4|, |3| at source coordinates
    want_idx = pi[want_src]
    assert st.sp_idx_k[0, 0, 0].tolist() == want_idx.tolist(), st.sp_idx_k[0, 0, 0]
    assert st.sp_val_k[0, 0, 0].tolist() == [8.0, -4.0, 3.0]


# -- P3: top-k pruning against brute force on d = 8 -----------------------

def pin_prune_bruteforce(o):
    gen = np.random.default_rng(7)
    d = 8
    for trial in range(60):
        # small integer magnitudes force many ties, incl. +0 / -0
        x = gen.integers(-3, 4, size=d).astype(np.float16)
        if trial % 3 == 0:
            x = gen.standard_normal(d).astype(np.float16)
        if trial % 5 == 0:
            x[gen.integers(0, d)] = np.float16(-0.0)
        for k in range(1, d + 1):
            idx, vals = o.prune(x, k)
            energy = lambda S: float(sum(float(x[j]) ** 2 for j in S))
            best = max(energy(S) for S in itertools.combinations(range(d), k))
            maximisers = [S for S in itertools.combinations(range(d), k) if energy(S) == best]
            # chosen set: a maximiser, and among maximisers the lowest indices
            assert sorted(idx.tolist()) == list(min(maximisers)), (x, k, idx)
            # stored order: decreasing magnitude, ties by increasing index
            keys = [(-abs(float(x[j])), int(j)) for j in idx]
            assert keys == sorted(keys), (x, k, idx)
            assert np.array_equal(vals.view(np.uint16), x[idx.astype(int)].view(np.uint16))


# -- P2 / Lemmas 1-2: k = d and exact rotation reproduce dense attention --

def pin_k_equals_d_is_dense(o):
    for G, b_cap in ((1, 5), (2, 0), (1, 100)):
        R, Rv, k, v, q = _small_problem(11 + G + b_cap, G=G)
        B, H_kv, L, d = k.shape
        st = o.SwanOracle(R, Rv, batch=B, n_q_heads=H_kv * G, k_store=d, buffer_cap=b_cap,
                          round_rotated=False)
        st.append(k[:, :, :17], v[:, :, :17])
        st.append(k[:, :, 17:], v[:, :, 17:])
        out = st.decode(q)
        for b in range(B):
            for hq in range(H_kv * G):
                ref = o.dense_attention(q[b, hq], k[b, hq // G], v[b, hq // G])
                assert np.abs(out[b, hq] - ref).max() < 1e-12
        # with the fp16 storage rounding the error stays at the fp16 level
        st16 = o.SwanOracle(R, Rv, batch=B, n_q_heads=H_kv * G, k_store=d, buffer_cap=b_cap)
        st16.append(k, v)
        out16 = st16.decode(q)
        ref = np.stack([np.stack([o.dense_attention(q[b, hq], k[b, hq // G], v[b, hq // G])
                                  for hq in range(H_kv * G)]) for b in range(B)])
        assert np.abs(out16 - ref).max() < 2e-3


# -- P4: decompression-free == dense attention over zero-filled vectors ---

def pin_decompression_free(o):
    R, Rv, k, v, q = _small_problem(23, B=1, H_kv=2, G=2, d=32, L=50)
    B, H_kv, L, d = k.shape
    for k_store, b_cap in ((7, 9), (16, 0), (31, 64)):
        st = o.SwanOracle(R, Rv, batch=B, n_q_heads=H_kv * 2, k_store=k_store, buffer_cap=b_cap)
        st.append(k, v)
        out = st.decode(q)
        for hq in range(H_kv * 2):
            h = hq // 2
            Kd = np.concatenate([o.densify(st.sp_idx_k[0, h], st.sp_val_k[0, h], d),
                                 st.buf_k[0, h].astype(np.float64)])
            Vd = np.concatenate([o.densify(st.sp_idx_v[0, h], st.sp_val_v[0, h], d),
                                 st.buf_v[0, h].astype(np.float64)])
            qh = torch.from_numpy(q[0, hq].astype(np.float64) @ R[h].astype(np.float64))
            ref = torch.nn.functional.scaled_dot_product_attention(
                qh[None, None, None], torch.from_numpy(Kd)[None, None],
                torch.from_numpy(Vd)[None, None])[0, 0, 0].numpy()
            ref = ref @ Rv[h].astype(np.float64).T
            assert np.abs(out[0, hq] - ref).max() < 1e-12, (k_store, b_cap, hq)


# -- P5: buffer semantics (Algorithm 1 eviction; b >= L and b = 0) --------

def pin_buffer_semantics(o):
    R, Rv, k, v, q = _small_problem(31, B=1, H_kv=1, d=16, L=12)
    d = 16
    # no eviction when the buffer is large enough: every vector stays dense
    st = o.SwanOracle(R, Rv, batch=1, n_q_heads=1, k_store=4, buffer_cap=12)
    st.append(k, v)
    assert st.sparse_len == 0 and st.buffer_len == 12
    kh = (k[0, 0].astype(np.float64) @ R[0].astype(np.float64)).astype(np.float16)
    vh = (v[0, 0].astype(np.float64) @ Rv[0].astype(np.float64)).astype(np.float16)
    ref = o.dense_attention(q[0, 0].astype(np.float64) @ R[0].astype(np.float64), kh, vh)
    assert np.abs(st.decode(q)[0, 0] - ref @ Rv[0].astype(np.float64).T).max() < 1e-12
    # b = 0: everything is sparse; and token-by-token appends equal one bulk append
    for b_cap in (0, 3, 5):
        bulk = o.SwanOracle(R, Rv, batch=1, n_q_heads=1, k_store=5, buffer_cap=b_cap)
        bulk.append(k, v)
        step = o.SwanOracle(R, Rv, batch=1, n_q_heads=1, k_store=5, buffer_cap=b_cap)
        for t in range(12):
            step.append(k[:, :, t:t + 1], v[:, :, t:t + 1])
            # Algorithm 1: the buffer never holds more than b after an append
            assert step.buffer_len == min(t + 1, b_cap)
        assert bulk.sparse_len == 12 - b_cap and bulk.buffer_len == b_cap
        for a in ("sp_idx_k", "sp_val_k", "sp_idx_v", "sp_val_v", "buf_k", "buf_v"):
            assert np.array_equal(getattr(bulk, a), getattr(step, a)), a
        # FIFO: the sparse entries are the OLDEST tokens, pruned one by one
        for t in range(12 - b_cap):
            ik, vk = o.prune(kh[t], 5)
            assert np.array_equal(bulk.sp_idx_k[0, 0, t], ik)
            assert np.array_equal(bulk.sp_val_k[0, 0, t].view(np.uint16), vk.view(np.uint16))
            iv, vv = o.prune(vh[t], 5)
            assert np.array_equal(bulk.sp_idx_v[0, 0, t], iv)
        # and the buffer holds the newest ones, oldest first
        assert np.array_equal(bulk.buf_k[0, 0].view(np.uint16), kh[12 - b_cap:].view(np.uint16))
    # flush empties the buffer into the sparse history
    st.flush()
    assert st.buffer_len == 0 and st.sparse_len == 12


# -- P6: split combine equals the unsplit softmax -------------------------

def pin_split_combine(o):
    gen = np.random.default_rng(5)
    s = gen.standard_normal(97) * 4
    V = gen.standard_normal((97, 16))
    e = np.exp(s - s.max())
    ref = (e / e.sum()) @ V
    for cuts in ([50], [0, 13, 13, 60, 96], list(range(1, 97, 7))):
        edges = [0] + cuts + [97]
        parts = [o.partial_state(s[a:b], V[a:b]) for a, b in zip(edges[:-1], edges[1:])]
        assert np.abs(o.combine_partials(parts) - ref).max() < 1e-12
    # a single partial is the plain softmax
    assert np.abs(o.combine_partials([o.partial_state(s, V)]) - ref).max() < 1e-12


# -- P7: a smaller runtime k is exact re-pruning --------------------------

def pin_k_prefix(o):
    R, Rv, k, v, q = _small_problem(41, B=1, H_kv=2, G=2, d=32, L=30)
    big = o.SwanOracle(R, Rv, batch=1, n_q_heads=4, k_store=32, buffer_cap=4)
    big.append(k, v)
    for ka in (1, 5, 16, 31, 32):
        fresh = o.SwanOracle(R, Rv, batch=1, n_q_heads=4, k_store=ka, buffer_cap=4)
        fresh.append(k, v)
        big.set_k(ka)
        assert np.array_equal(big.decode(q), fresh.decode(q)), ka


# -- GQA grouping (Section 4.1.1) ----------------------------------------

def pin_gqa_mapping(o):
    R, Rv, k, v, q = _small_problem(53, B=1, H_kv=2, G=3, d=16, L=20)
    st = o.SwanOracle(R, Rv, batch=1, n_q_heads=6, k_store=16, buffer_cap=3, round_rotated=False)
    st.append(k, v)
    out = st.decode(q)
    for hq in range(6):
        ref = o.dense_attention(q[0, hq], k[0, hq // 3], v[0, hq // 3])
        assert np.abs(out[0, hq] - ref).max() < 1e-12
    # the per-unit entry point agrees with the batched one
    assert np.abs(st.decode_unit(q[0, 4], 0, 4) - out[0, 4]).max() < 1e-15


# -- P8: byte and FLOP formulas with the paper's worked numbers -----------

def _golden_rows(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


def pin_formulas(o):
    for d, k, b, want in _golden_rows("break_even.txt"):
        got = o.break_even_length(int(d), int(k), int(b))
        assert round(got) == int(want), (d, k, b, got, want)
        # the break-even point is where the FLOP counts meet
        L = math.ceil(got + 1e-9)
        assert o.flops_swan(L, int(d), int(k), int(b)) < o.flops_standard(L, int(d))
        assert o.flops_swan(L - 1, int(d), int(k), int(b)) >= o.flops_standard(L - 1, int(d))
    for row in _golden_rows("memory_formula.txt"):
        if row[0] == "dense":
            assert o.dense_vector_bytes(int(row[1])) == int(row[2])
        elif row[0] == "fp16_memory_break_even_k":
            kmax = max(k for k in range(1, 129) if o.sparse_vector_bytes(k) < o.dense_vector_bytes(128))
            assert kmax == int(row[1])
            assert kmax / 128 < 0.66 <= (kmax + 1) / 128
        else:
            assert o.sparse_vector_bytes(int(row[0]), value_bytes=int(row[1])) == int(row[2])
    assert abs(o.compression_ratio(64, 128) - 194 / 256) < 1e-15


# -- 8-bit value rounding (E4M3) against torch's float8_e4m3fn ------------

def pin_e4m3_rounding(o):
    h = np.arange(65536, dtype=np.uint16).view(np.float16)
    h = h[np.isfinite(h)].astype(np.float64)
    got = o.to_e4m3(h)
    inr = np.abs(h) < 464.0  # torch turns |x| >= 480 into NaN instead of saturating
    ref = torch.from_numpy(h[inr].astype(np.float32)).to(torch.float8_e4m3fn).double().numpy()
    assert np.array_equal(got[inr], ref)
    assert np.all(np.abs(got[~inr]) == 448.0) and np.array_equal(np.sign(got[~inr]), np.sign(h[~inr]))
    # every E4M3 value is its own rounding; ties go to the even neighbour
    assert np.array_equal(o.to_e4m3(got), got)
    assert o.to_e4m3(1.0625) == 1.0 and o.to_e4m3(1.1875) == 1.25 and o.to_e4m3(2.0 ** -10) == 0.0


def pin_fp8_cache_is_rounded_sparse_cache(o):
    """The fp8 cache holds the same indices as the fp16 cache (selection on
    the fp16 vector) with the kept values rounded to E4M3; decoding it equals
    dense attention on the zero-filled rounded vectors."""
    R, Rv, k, v, q = _small_problem(61, B=1, H_kv=1, d=32, L=40)
    a = o.SwanOracle(R, Rv, batch=1, n_q_heads=1, k_store=12, buffer_cap=5)
    b = o.SwanOracle(R, Rv, batch=1, n_q_heads=1, k_store=12, buffer_cap=5, value_format="fp8_e4m3")
    a.append(k, v)
    b.append(k, v)
    assert np.array_equal(a.sp_idx_k, b.sp_idx_k) and np.array_equal(a.sp_idx_v, b.sp_idx_v)
    assert np.array_equal(b.sp_val_k.astype(np.float64), o.to_e4m3(a.sp_val_k.astype(np.float64)))
    assert np.array_equal(a.buf_k.view(np.uint16), b.buf_k.view(np.uint16))
    Kd = np.concatenate([o.densify(b.sp_idx_k[0, 0], b.sp_val_k[0, 0], 32), b.buf_k[0, 0].astype(np.float64)])
    Vd = np.concatenate([o.densify(b.sp_idx_v[0, 0], b.sp_val_v[0, 0], 32), b.buf_v[0, 0].astype(np.float64)])
    qh = q[0, 0].astype(np.float64) @ R[0].astype(np.float64)
    ref = o.dense_attention(qh, Kd, Vd) @ Rv[0].astype(np.float64).T
    assert np.abs(b.decode(q)[0, 0] - ref).max() < 1e-12


# -- asymmetric keep counts for keys and values (appendix ablation) --------

def pin_asymmetric_keep_counts(o):
    """Keys keep k_K entries and values k_V: decoding equals dense attention
    on keys zero-filled at k_K and values zero-filled at k_V; a runtime split
    on a symmetric cache equals a cache stored with that split."""
    R, Rv, k, v, q = _small_problem(71, B=1, H_kv=1, d=32, L=30)
    st = o.SwanOracle(R, Rv, batch=1, n_q_heads=1, k_store=9, k_store_v=20, buffer_cap=4)
    st.append(k, v)
    assert st.sp_idx_k.shape[-1] == 9 and st.sp_idx_v.shape[-1] == 20
    kh = (k[0, 0].astype(np.float64) @ R[0].astype(np.float64)).astype(np.float16)
    vh = (v[0, 0].astype(np.float64) @ Rv[0].astype(np.float64)).astype(np.float16)
    ik, vk = o.prune(kh[:26], 9)
    iv, vv = o.prune(vh[:26], 20)
    Kd = np.concatenate([o.densify(ik, vk, 32), kh[26:].astype(np.float64)])
    Vd = np.concatenate([o.densify(iv, vv, 32), vh[26:].astype(np.float64)])
    qh = q[0, 0].astype(np.float64) @ R[0].astype(np.float64)
    ref = o.dense_attention(qh, Kd, Vd) @ Rv[0].astype(np.float64).T
    assert np.abs(st.decode(q)[0, 0] - ref).max() < 1e-12
    big = o.SwanOracle(R, Rv, batch=1, n_q_heads=1, k_store=32, buffer_cap=4)
    big.append(k, v)
    big.set_k(9, 20)
    assert np.array_equal(big.decode(q), st.decode(q))


ALL_PINS = [pin_rotation_orthogonal, pin_rotation_orientation, pin_prune_bruteforce,
            pin_k_equals_d_is_dense, pin_decompression_free, pin_buffer_semantics,
            pin_split_combine, pin_k_prefix, pin_gqa_mapping, pin_formulas, pin_e4m3_rounding,
            pin_fp8_cache_is_rounded_sparse_cache, pin_asymmetric_keep_counts]


# -- Offline basis (Section 4.1); each takes the basis oracle module ---------

def _orthonormal_columns(m, n, gen):
    q, _ = np.linalg.qr(gen.standard_normal((m, n)))
    return q


def pin_basis_recovers_planted_svd(b):
    """S = U diag(sigma) W^T with known factors: the basis is W (columns, in
    order of decreasing sigma, up to the sign rule) and the singular values
    are sigma."""
    gen = np.random.default_rng(101)
    d, m = 16, 60
    W = synth.random_orthogonal(d, gen)
    U = _orthonormal_columns(m, d, gen)
    sigma = 2.0 ** -(np.arange(d) / 2.0)
    P, s = b.principal_basis(U @ np.diag(sigma) @ W.T)
    assert P.shape == (d, d)
    assert np.allclose(s, sigma, atol=1e-12)
    for j in range(d):
        assert abs(abs(P[:, j] @ W[:, j]) - 1.0) < 1e-10, j
        lead = int(np.argmax(np.abs(P[:, j])))
        assert P[lead, j] > 0, j
    assert np.allclose(P.T @ P, np.eye(d), atol=1e-12)


def pin_basis_ky_fan_maximum(b):
    """For every k the first k basis vectors keep the most energy of any
    k-dimensional orthonormal set (Ky Fan): sum_{j<k} |S p_j|^2 equals the sum
    of the k largest eigenvalues of S^T S and no random basis beats it."""
    gen = np.random.default_rng(102)
    S = gen.standard_normal((200, 12)) * np.linspace(3.0, 0.2, 12)[None, :] @ synth.random_orthogonal(12, gen)
    P, _ = b.principal_basis(S)
    lam = np.sort(np.linalg.eigvalsh(b.gram(S)))[::-1]
    kept = np.cumsum(np.sum((S @ P) ** 2, axis=0))
    assert np.allclose(kept, np.cumsum(lam), rtol=1e-10)
    for _ in range(20):
        Qr = synth.random_orthogonal(12, gen)
        other = np.cumsum(np.sum((S @ Qr) ** 2, axis=0))
        assert (other <= kept * (1 + 1e-12)).all()


def pin_gram_planted_factors(b):
    """gram(S) is S^T S, whose eigenvectors are SVD(S)_V (Section 4.1.2):
    for S = U diag(sigma) W^T with orthonormal U, W it equals
    W diag(sigma^2) W^T, and for any S it is the sum over the rows s_r of the
    outer products s_r^T s_r (brute force, every row counted once)."""
    gen = np.random.default_rng(106)
    d, m = 12, 40
    W = synth.random_orthogonal(d, gen)
    U = _orthonormal_columns(m, d, gen)
    sigma = np.linspace(3.0, 0.25, d)
    G = b.gram(U @ np.diag(sigma) @ W.T)
    assert G.shape == (d, d)
    assert np.allclose(G, W @ np.diag(sigma ** 2) @ W.T, atol=1e-12)
    S = gen.standard_normal((7, 5)) * np.array([1.0, 2.0, 0.5, 4.0, 1.5])
    S[0] *= 9.0                       # a dropped first or last row shows
    S[-1] *= 7.0
    brute = np.zeros((5, 5))
    for r in range(S.shape[0]):
        for i in range(5):
            for j in range(5):
                brute[i, j] += S[r, i] * S[r, j]
    assert np.allclose(b.gram(S), brute, atol=1e-12)
    assert b.gram(S).dtype == np.float64


def _planted_groups(gen, n_kv, G, n, d, d_model, r):
    """Per kv head j four planted r-dimensional subspaces: the query heads
    jG..jG+G-1 live in span(Bq[j]), key head j in span(Bk[j]), value head j
    in span(Bv[j]) and the columns of the W_O slices of those query heads in
    span(Bw[j])."""
    Bq, Bk, Bv, Bw = ([_orthonormal_columns(d, r, gen) for _ in range(n_kv)] for _ in range(4))
    Q = np.stack([gen.standard_normal((n, r)) @ Bq[h // G].T for h in range(n_kv * G)])
    K = np.stack([gen.standard_normal((n, r)) @ Bk[j].T for j in range(n_kv)])
    V = np.stack([gen.standard_normal((n, r)) @ Bv[j].T for j in range(n_kv)])
    W_O = np.concatenate([Bw[h // G] @ gen.standard_normal((r, d_model)) for h in range(n_kv * G)])
    return Bq, Bk, Bv, Bw, Q, K, V, W_O


def pin_joint_matrices_group_heads(b):
    """Section 4.1.1 grouping and Section 4.1.2 concatenation: with query
    heads jG..jG+G-1, key head j, value head j and the W_O slices of those
    query heads each in their own planted r-dimensional subspace, the first
    2r basis vectors of S_QK[j] span exactly span(Bq[j], Bk[j]) and those of
    S_VO[j] span(Bv[j], Bw[j]); a wrong grouping or a dropped part leaves a
    different span."""
    gen = np.random.default_rng(103)
    n_kv, G, n, d, d_model, r = 3, 2, 40, 16, 24, 3
    Bq, Bk, Bv, Bw, Q, K, V, W_O = _planted_groups(gen, n_kv, G, n, d, d_model, r)
    sqk = b.joint_qk(Q, K, G)
    svo = b.joint_vo(V, W_O, G)
    assert len(sqk) == n_kv and len(svo) == n_kv
    for j in range(n_kv):
        assert sqk[j].shape == ((G + 1) * n, d)
        assert svo[j].shape == (n + G * d_model, d)
        for S, B in ((sqk[j], np.hstack([Bq[j], Bk[j]])), (svo[j], np.hstack([Bv[j], Bw[j]]))):
            P, sigma = b.principal_basis(S)
            B, _ = np.linalg.qr(B)
            assert np.linalg.norm(B.T @ P[:, :2 * r]) ** 2 > 2 * r - 1e-9, j
            assert sigma[2 * r] < 1e-9 * sigma[0]


def pin_energy_curve_bruteforce(b):
    """E[k] is the sum over vectors of the best k-subset of squared rotated
    coordinates (brute force over all subsets, d = 8); E[0] = 0 and E[d] is
    the total energy (P orthogonal)."""
    gen = np.random.default_rng(104)
    d = 8
    X = gen.standard_normal((30, d)) * np.array([3, 1, 0.5, 2, 0.1, 1, 4, 0.3])
    P = synth.random_orthogonal(d, gen)
    E = b.energy_curve(X, P)
    Y = X @ P
    for k in range(d + 1):
        best = 0.0
        for y in Y:
            best += max((sum(y[list(c)] ** 2) for c in itertools.combinations(range(d), k)), default=0.0)
        assert abs(E[k] - best) < 1e-9 * max(1.0, best), k
    assert E[0] == 0.0 and abs(E[d] - np.sum(X * X)) < 1e-9


def pin_energy_planted_rank(b):
    """Vectors in the span of the first r columns of an orthogonal W keep all
    their energy at k = r with P = W, and with the principal basis of the
    vectors themselves; a random basis keeps less."""
    gen = np.random.default_rng(105)
    d, r = 16, 4
    W = synth.random_orthogonal(d, gen)
    X = gen.standard_normal((50, r)) @ W[:, :r].T
    for P in (W, b.principal_basis(X)[0]):
        E = b.energy_curve(X, P)
        assert abs(E[r] - E[d]) < 1e-9 * E[d]
    assert b.energy_curve(X, synth.random_orthogonal(d, gen))[r] < 0.99 * np.sum(X * X)


BASIS_PINS = [pin_basis_recovers_planted_svd, pin_basis_ky_fan_maximum, pin_gram_planted_factors,
              pin_joint_matrices_group_heads, pin_energy_curve_bruteforce, pin_energy_planted_rank]


def pin_ragged_rows_are_independent(o):
    """A batch of rows of different lengths: with equal appends the ragged
    state machine equals the batched one bitwise, row b's outputs depend only
    on row b's own tokens, and a reset row equals a fresh cache fed only what
    came after the reset."""
    R, Rv, k, v, q = _small_problem(61, B=3, H_kv=2, G=2, d=16, L=30)
    bat = o.SwanOracle(R, Rv, batch=3, n_q_heads=4, k_store=5, buffer_cap=4)
    rag = o.RaggedOracle(R, Rv, batch=3, n_q_heads=4, k_store=5, buffer_cap=4)
    bat.append(k[:, :, :20], v[:, :, :20])
    rag.append(k[:, :, :20], v[:, :, :20])
    assert np.array_equal(bat.decode(q), rag.decode(q))
    rag.append(k[:, :, 20:30], v[:, :, 20:30], n_new=[10, 0, 3])
    assert rag.sparse_lens == [26, 16, 19] and rag.buffer_lens == [4, 4, 4]
    solo = o.SwanOracle(R, Rv, batch=1, n_q_heads=4, k_store=5, buffer_cap=4)
    solo.append(k[2:3, :, :23], v[2:3, :, :23])
    assert np.array_equal(rag.decode(q)[2], solo.decode(q[2:3])[0])
    rag.reset(1)
    assert np.array_equal(rag.decode(q)[1], np.zeros((4, 16)))
    rag.append(k[:, :, 25:30], v[:, :, 25:30], n_new=[0, 5, 0])
    fresh = o.SwanOracle(R, Rv, batch=1, n_q_heads=4, k_store=5, buffer_cap=4)
    fresh.append(k[1:2, :, 25:30], v[1:2, :, 25:30])
    assert np.array_equal(rag.decode(q)[1], fresh.decode(q[1:2])[0])


ALL_PINS.append(pin_ragged_rows_are_independent)
