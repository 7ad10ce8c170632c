"""Offline basis construction on the GPU (swan_gram, swan_basis_eig,
swan_energy) against the CPU basis oracle (needs a GB300)."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2511_18936_gb300 import synth

pytestmark = pytest.mark.gpu

D = 128
bo = oracle.basis_oracle


def _gram_tol(S):
    """Summation bound for S^T S: 2^-14 * sum_r |s_ri| |s_rj|.  The products
    are exact; each CTA sums at most 1024 of them per entry in fp32 at these
    sizes (gamma_1024 = 2^-14) and the partials are added in fp64."""
    A = np.abs(np.asarray(S, np.float64))
    return 2.0 ** -14 * (A.T @ A) + 1e-30


def _cal(n_kv, G, n, d_model, seed):
    return synth.calibration(n_kv, G, n, D, d_model, seed=seed, workload=60, layer=0)


@pytest.mark.parametrize("n_kv,G,n,d_model", [(2, 2, 1000, 200), (1, 1, 1, 8), (3, 4, 65, 64),
                                              (1, 8, 4097, 136)])
def test_gram_matches_oracle(n_kv, G, n, d_model):
    import torch

    from paper_2511_18936_gb300 import swan
    Q, K, V, W_O = _cal(n_kv, G, n, d_model, seed=n)
    dev = torch.device("cuda")
    tq, tk, tv, tw = (torch.from_numpy(a).to(dev) for a in (Q, K, V, W_O))
    qk = swan.Gram(n_kv).add(swan.rows_of(tq, G), accumulate=False).add(swan.rows_of(tk))
    vo = swan.Gram(n_kv).add(swan.rows_of(tv), accumulate=False).add(swan.columns_of(tw, G))
    qk.check()
    vo.check()
    for g, S_list in ((qk.gram, bo.joint_qk(Q, K, G)), (vo.gram, bo.joint_vo(V, W_O, G))):
        got = g.double().cpu().numpy()
        for j, S in enumerate(S_list):
            want = bo.gram(S)
            assert (np.abs(got[j] - want) <= _gram_tol(S)).all(), j


def test_gram_token_major_layout_and_determinism():
    """Q stored token-major ([n][N_q][d], strides instead of a copy) gives the
    same Gram matrices, bit for bit, run after run."""
    import torch

    from paper_2511_18936_gb300 import swan
    n_kv, G, n = 2, 4, 3000
    Q, K, _, _ = _cal(n_kv, G, n, 64, seed=7)
    dev = torch.device("cuda")
    tq = torch.from_numpy(Q).to(dev)
    tq_tm = tq.transpose(0, 1).contiguous()  # [n][N_q][d]
    a = swan.Gram(n_kv).add(swan.rows_of(tq, G), accumulate=False).gram.clone()
    v = swan.SwanVectors(tq_tm.data_ptr(), n_kv, G, n, G * D, D, n_kv * G * D, 1)
    g2 = swan.Gram(n_kv)
    b = g2.add(v, accumulate=False).gram.clone()
    c = g2.add(v, accumulate=False).gram.clone()
    g2.check()
    torch.cuda.synchronize()
    assert torch.equal(b, c)
    S = [Q[j * G:(j + 1) * G].reshape(-1, D).astype(np.float64) for j in range(n_kv)]
    for j in range(n_kv):
        tol = _gram_tol(S[j])
        assert (np.abs(a[j].double().cpu().numpy() - bo.gram(S[j])) <= tol).all()
        assert (np.abs(b[j].double().cpu().numpy() - bo.gram(S[j])) <= tol).all()


def test_eig_matches_oracle_basis():
    import torch

    from paper_2511_18936_gb300 import swan
    n_kv, G, n, d_model = 2, 2, 2048, 256
    Q, K, V, W_O = _cal(n_kv, G, n, d_model, seed=11)
    dev = torch.device("cuda")
    tq, tk, tv, tw = (torch.from_numpy(a).to(dev) for a in (Q, K, V, W_O))
    grams = [swan.Gram(n_kv).add(swan.rows_of(tq, G), False).add(swan.rows_of(tk)),
             swan.Gram(n_kv).add(swan.rows_of(tv), False).add(swan.columns_of(tw, G))]
    for g, S_list in zip(grams, (bo.joint_qk(Q, K, G), bo.joint_vo(V, W_O, G))):
        R, lam, sweeps = swan.basis_eig(g.gram)
        R64 = R.double().cpu().numpy()
        lam64 = lam.double().cpu().numpy()
        assert (sweeps.cpu().numpy() > 0).all()
        for j, S in enumerate(S_list):
            P, sigma = bo.principal_basis(S)
            C = bo.gram(S)
            lmax = sigma[0] ** 2
            assert np.abs(lam64[j] - sigma ** 2).max() <= 1e-5 * lmax
            assert np.abs(R64[j].T @ R64[j] - np.eye(D)).max() <= 2e-6
            resid = np.linalg.norm(C @ R64[j] - R64[j] * lam64[j][None, :], axis=0)
            assert resid.max() <= 2e-5 * lmax
            # well-separated leading directions match the oracle's, signs included
            gaps = np.minimum(np.abs(np.diff(sigma ** 2, prepend=np.inf)), np.abs(np.diff(sigma ** 2, append=-np.inf)))
            for r in np.nonzero(gaps > 1e-2 * lmax)[0]:
                assert R64[j][:, r] @ P[:, r] > 1 - 1e-6, (j, r)


def test_eig_degenerate_inputs():
    """A zero Gram matrix and a diagonal one: no rotation is needed; the basis
    is a signed permutation ordering the diagonal decreasingly."""
    import torch

    from paper_2511_18936_gb300 import swan
    g = torch.zeros((2, D, D), dtype=torch.float32, device="cuda")
    diag = torch.from_numpy(np.random.default_rng(3).permutation(D).astype(np.float32) + 1.0)
    g[1] = torch.diag(diag).cuda()
    R, lam, sweeps = swan.basis_eig(g)
    R, lam = R.cpu().numpy(), lam.cpu().numpy()
    assert (sweeps.cpu().numpy() == 1).all()
    assert np.array_equal(R[0], np.eye(D, dtype=np.float32))
    assert np.array_equal(lam[1], np.sort(diag.numpy())[::-1])
    order = np.argsort(-diag.numpy(), kind="stable")
    assert np.array_equal(R[1], np.eye(D, dtype=np.float32)[:, order])


@pytest.mark.parametrize("layout", ["rows", "cols"])
def test_energy_matches_oracle(layout):
    import torch

    from paper_2511_18936_gb300 import swan
    n_kv, G, n, d_model = 2, 2, 777, 296
    Q, K, V, W_O = _cal(n_kv, G, n, d_model, seed=13)
    gen = np.random.default_rng(13)
    R = np.stack([synth.random_orthogonal(D, gen) for _ in range(n_kv)]).astype(np.float32)
    dev = torch.device("cuda")
    tR = torch.from_numpy(R).to(dev)
    if layout == "rows":
        t = torch.from_numpy(Q).to(dev)
        E = swan.energy(swan.rows_of(t, G), tR).cpu().numpy()
        sets = [Q[j * G:(j + 1) * G].reshape(-1, D) for j in range(n_kv)]
    else:
        t = torch.from_numpy(W_O).to(dev)
        E = swan.energy(swan.columns_of(t, G), tR).cpu().numpy()
        sets = [np.concatenate([W_O[h * D:(h + 1) * D].T for h in range(j * G, (j + 1) * G)]) for j in range(n_kv)]
    for j in range(n_kv):
        want = bo.energy_curve(sets[j], R[j])
        assert E[j][0] == 0.0
        assert np.abs(E[j] - want).max() <= 1e-5 * want[-1], j
    # accumulate adds a second pass
    E2 = swan.energy(swan.rows_of(torch.from_numpy(Q).to(dev), G) if layout == "rows"
                     else swan.columns_of(torch.from_numpy(W_O).to(dev), G), tR,
                     out=torch.from_numpy(E).to(dev), accumulate=True).cpu().numpy()
    assert np.allclose(E2, 2 * E, rtol=1e-12)


def test_data_driven_basis_keeps_more_energy_and_plugs_into_decode():
    """The GPU basis of a calibration set keeps more energy at k = 32, 64
    than a random basis on held-out keys and values, and a context built with
    it decodes within tolerance of the oracle fed the same matrices."""
    import torch

    from paper_2511_18936_gb300 import swan
    from tests.helpers import TOL_OUT
    n_kv, G, n, d_model = 2, 2, 4096, 512
    Q, K, V, W_O = _cal(n_kv, G, n, d_model, seed=17)
    dev = torch.device("cuda")
    tq, tk, tv, tw = (torch.from_numpy(a).to(dev) for a in (Q, K, V, W_O))
    g_qk = swan.Gram(n_kv).add(swan.rows_of(tq[:, :n // 2].contiguous(), G), False) \
        .add(swan.rows_of(tk[:, :n // 2].contiguous()))
    g_vo = swan.Gram(n_kv).add(swan.rows_of(tv[:, :n // 2].contiguous()), False).add(swan.columns_of(tw, G))
    R_qk, _, _ = swan.basis_eig(g_qk.gram)
    R_vo, _, _ = swan.basis_eig(g_vo.gram)
    gen = np.random.default_rng(17)
    R_rand = torch.from_numpy(np.stack([synth.random_orthogonal(D, gen) for _ in range(n_kv)])
                              .astype(np.float32)).to(dev)
    held_k = swan.rows_of(tk[:, n // 2:].contiguous())
    held_v = swan.rows_of(tv[:, n // 2:].contiguous())
    for held, R in ((held_k, R_qk), (held_v, R_vo)):
        e_data = swan.energy(held, R).cpu().numpy()
        e_rand = swan.energy(held, R_rand).cpu().numpy()
        for j in range(n_kv):
            for k in (32, 64):
                assert e_data[j][k] / e_data[j][D] > e_rand[j][k] / e_rand[j][D] + 0.05, (j, k)
    # the constructed basis as the cache rotation
    from tests.helpers import run_ops
    kk = K[None, :, n // 2:n // 2 + 300].copy()
    vv = V[None, :, n // 2:n // 2 + 300].copy()
    q = synth.gaussian_fp16((1, n_kv * G, D), 17, 60, 0, synth.T_Q)
    ops = [("append", kk, vv), ("decode", q), ("set_k", 32), ("decode", q)]
    ctx, ref, outs = run_ops(ops, R_qk.cpu().numpy(), R_vo.cpu().numpy(), B=1, H_kv=n_kv, G=G, k_store=64,
                             cap=32)
    for got, want in outs:
        assert np.abs(got - want).max() <= TOL_OUT
    ctx.close()
