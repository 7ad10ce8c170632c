"""CPU fp64 oracle for SWAN's offline basis construction (test infrastructure only).

Like ``swan_oracle``, this file is the reference the CUDA path is checked
against; only the test-suite, ``__graft_entry__.smoke()`` and the CPU legs of
``bench.py`` may import it, and it shares no code with the library.

It restates Section 4.1 of "SWAN: Sparse Winnowed Attention" (arXiv
2511.18936) in float64 with NumPy primitives:

* Section 4.1.1: for each kv head ``j`` the query heads ``jG .. jG+G-1``
  (``G = N_q / N_kv``) are grouped with it; the output-projection matrix
  ``W_O`` (``[N_q d_h][d_model]``) is sliced into per-head ``[d_h][d_model]``
  blocks that are grouped the same way.
* Section 4.1.2: two joint matrices per kv head, concatenated along the
  sequence (row) dimension, ``S_QK = Concat(Q_grouped, K)`` and
  ``S_VO = Concat(V, W_O_grouped^T)``; the projection is the matrix of right
  singular vectors of the joint matrix, ordered by decreasing singular value.
* The measure reported for a basis is the energy that per-vector top-k
  pruning (Algorithm 1) keeps: ``E[k] = sum over vectors of the k largest
  squared coordinates of x P``; ``E[d]`` is the total energy (``P``
  orthogonal).

Readings where the paper is silent (each listed in the design notes):

* A singular vector is defined up to sign; the sign is fixed so that the
  coordinate of largest magnitude of each basis vector is positive (the
  lowest such coordinate on an exact tie).
* ``W_O_grouped^T`` contributes one row per (query head of the group,
  column of ``W_O``): the ``d_model`` columns of each head's slice.
* The energy measure sums over vectors (the share of the total energy of a
  set that the pruned vectors keep), not a mean of per-vector shares.

Parity status: every function below is pinned in ``tests/oracle_pins.py``
(planted singular vectors, the Ky Fan maximum property, the Gram matrix of
planted factors and by brute force over rows, planted per-group
subspaces for both joint matrices, brute-force top-k energy on d = 8).
"""
from __future__ import annotations

import numpy as np


def joint_qk(Q, K, group: int):
    """Section 4.1.2: ``S_QK[j] = Concat(Q[jG..jG+G-1] (all tokens), K[j])``.

    Q: ``[N_q][n][d]``, K: ``[N_kv][n][d]`` -> list of ``[(G+1) n][d]`` fp64.
    """
    Q = np.asarray(Q, np.float64)
    K = np.asarray(K, np.float64)
    n_kv, n, d = K.shape
    assert Q.shape[0] == n_kv * group
    out = []
    for j in range(n_kv):
        q_rows = Q[j * group:(j + 1) * group].reshape(group * Q.shape[1], d)
        out.append(np.concatenate([q_rows, K[j]], axis=0))
    return out


def joint_vo(V, W_O, group: int):
    """Section 4.1.2: ``S_VO[j] = Concat(V[j], W_O_grouped[j]^T)``.

    V: ``[N_kv][n][d]``; W_O: ``[N_q d][d_model]``, head h's slice is rows
    ``h d .. h d + d - 1``; its transpose contributes ``d_model`` rows.
    """
    V = np.asarray(V, np.float64)
    W_O = np.asarray(W_O, np.float64)
    n_kv, n, d = V.shape
    out = []
    for j in range(n_kv):
        parts = [V[j]]
        for g in range(group):
            h = j * group + g
            parts.append(W_O[h * d:(h + 1) * d, :].T)
        out.append(np.concatenate(parts, axis=0))
    return out


def fix_signs(P):
    """Make the largest-magnitude coordinate of every column positive."""
    P = np.array(P, np.float64, copy=True)
    lead = np.argmax(np.abs(P), axis=0)
    s = np.sign(P[lead, np.arange(P.shape[1])])
    s[s == 0] = 1.0
    return P * s[None, :]


def principal_basis(S):
    """Section 4.1.2: ``P = SVD(S)_V``, columns ordered by decreasing singular
    value, signs fixed.  Returns ``(P [d][d], sigma [d])``."""
    S = np.asarray(S, np.float64)
    _, sigma, vt = np.linalg.svd(S, full_matrices=False)
    P = vt.T
    if P.shape[1] < S.shape[1]:
        raise ValueError("fewer rows than columns: the basis is not determined")
    return fix_signs(P), sigma


def gram(S):
    """``S^T S`` in fp64 (the matrix whose eigenvectors are ``SVD(S)_V``)."""
    S = np.asarray(S, np.float64)
    return S.T @ S


def energy_curve(X, P):
    """Energy kept by per-vector magnitude top-k after rotating by ``P``.

    X: ``[m][d]`` row vectors; returns ``E [d + 1]`` with ``E[k]`` the sum over
    the rows of the ``k`` largest squared coordinates of ``x P``.
    """
    Y = np.asarray(X, np.float64) @ np.asarray(P, np.float64)
    sq = np.sort(Y * Y, axis=1)[:, ::-1]
    E = np.zeros(Y.shape[1] + 1)
    E[1:] = np.cumsum(sq.sum(axis=0))
    return E
