"""Seeded synthetic inputs shaped like the SWAN decode workloads.

This module only draws random numbers.  It holds none of SWAN's arithmetic
(no rotation of cache vectors, no pruning, no attention): it produces the
inputs that both the CUDA path and the CPU oracle consume.

Recipe (the paper's workloads are Llama-2-7B / Llama-3-8B activations,
Section 6; no weights or datasets are used here, these stand in for them):

* Low-rank key/value vectors: for each (batch, kv-head) unit,
  ``X = Z diag(sigma) W^T`` with ``Z ~ N(0, 1)`` of shape ``[L, d]``, ``W`` a
  random orthogonal matrix and ``sigma_i ∝ 1/i`` normalised so that
  ``sum sigma_i^2 = d`` (so ``E|x|^2 = d``).  Cast to fp16.
* Queries ``q ~ N(0, 1)`` in fp16 (optionally scaled, "peaked").
* The rotation ``R`` per (layer, kv-head): ``Q`` of the QR factorisation of a
  seeded Gaussian ``d x d`` matrix, column signs fixed so that the diagonal of
  the triangular factor is positive, cast to fp32 (the paper's random
  orthogonal projection ablation, Appendix, "Random Projection").
* Plain Gaussian K/V/q for the 32-layer stack workload.
* Calibration sets for the offline basis (Section 4.1): per kv head ``j``
  two random orthogonal bases ``W_qk[j]`` and ``W_vo[j]``; the G query heads
  of the group and the key head draw ``Z diag(sigma) W_qk[j]^T`` (queries
  with the flatter spectrum ``sigma_i ∝ i^-1/2``, keys with ``∝ 1/i``), the
  value head ``Z diag(sigma) W_vo[j]^T``, and the output-projection slice of
  each query head of the group is ``W_vo[j] diag(tau) Y`` (``tau_i ∝ i^-1/2``,
  ``Y`` Gaussian ``d x d_model`` scaled by ``d_model^-1/2``), so that the
  columns of every slice share the value basis of their kv head.

Seeds: ``numpy.random.SeedSequence([seed, workload, layer, tensor_id])``.
Large workloads are drawn on the GPU with a seeded ``torch.Generator`` (the
same recipe, a different stream of random numbers); a test that compares the
CUDA path with the oracle hands both sides the very same arrays.
"""
from __future__ import annotations

import numpy as np

# tensor ids inside a SeedSequence
T_R_QK, T_R_VO, T_K, T_V, T_Q, T_KBASIS, T_VBASIS, T_NEWK, T_NEWV = range(9)
# calibration activations and weights for the offline basis
T_CAL_Q, T_CAL_K, T_CAL_V, T_CAL_WO, T_QK_BASIS, T_VO_BASIS = range(9, 15)


def seed_seq(seed: int, workload: int, layer: int, tensor_id: int, *extra: int):
    return np.random.SeedSequence([seed, workload, layer, tensor_id, *extra])


def rng(seed: int, workload: int, layer: int, tensor_id: int, *extra: int):
    return np.random.default_rng(seed_seq(seed, workload, layer, tensor_id, *extra))


def random_orthogonal(d: int, gen: np.random.Generator) -> np.ndarray:
    """Haar-like random orthogonal matrix (fp64), sign-fixed QR of a Gaussian."""
    g = gen.standard_normal((d, d))
    q, r = np.linalg.qr(g)
    s = np.sign(np.diag(r))
    s[s == 0] = 1.0
    return q * s[None, :]


def rotations(n_kv_heads: int, d: int, seed: int, workload: int, layer: int,
              tensor_id: int = T_R_QK) -> np.ndarray:
    """Per-kv-head random orthogonal matrices, fp32 ``[n_kv_heads][d][d]``."""
    out = np.empty((n_kv_heads, d, d), np.float32)
    for h in range(n_kv_heads):
        out[h] = random_orthogonal(d, rng(seed, workload, layer, tensor_id, h)).astype(np.float32)
    return out


def power_law_sigma(d: int) -> np.ndarray:
    """sigma_i ∝ 1/i (i = 1..d), normalised so that sum sigma_i^2 = d."""
    s = 1.0 / np.arange(1, d + 1, dtype=np.float64)
    return s * np.sqrt(d / np.sum(s * s))


def lowrank_vectors(n: int, d: int, gen: np.random.Generator,
                    basis: np.ndarray | None = None) -> np.ndarray:
    """``n`` vectors with a power-law singular spectrum, fp16 ``[n][d]``."""
    if basis is None:
        basis = random_orthogonal(d, gen)
    z = gen.standard_normal((n, d))
    x = (z * power_law_sigma(d)[None, :]) @ basis.T
    return x.astype(np.float16)


def lowrank_kv(batch: int, n_kv_heads: int, n_tokens: int, d: int, seed: int,
               workload: int, layer: int, tensor_id: int, token_offset: int = 0):
    """fp16 ``[batch][n_kv_heads][n_tokens][d]`` low-rank keys (or values).

    The basis of each (batch, head) unit is fixed by (seed, workload, layer,
    tensor_id, b, h); the Gaussian factor additionally by ``token_offset`` so
    that successive calls extend the same unit with fresh tokens.
    """
    basis_id = T_KBASIS if tensor_id in (T_K, T_NEWK) else T_VBASIS
    out = np.empty((batch, n_kv_heads, n_tokens, d), np.float16)
    for b in range(batch):
        for h in range(n_kv_heads):
            w = random_orthogonal(d, rng(seed, workload, layer, basis_id, b, h))
            g = rng(seed, workload, layer, tensor_id, b, h, token_offset)
            out[b, h] = lowrank_vectors(n_tokens, d, g, basis=w)
    return out


def gaussian_fp16(shape, seed: int, workload: int, layer: int, tensor_id: int,
                  *extra: int, scale: float = 1.0) -> np.ndarray:
    g = rng(seed, workload, layer, tensor_id, *extra)
    return (g.standard_normal(shape) * scale).astype(np.float16)


# --------------------------------------------------------------------------
# Device-side generation for the full-size workloads (inputs of several GB).
# --------------------------------------------------------------------------

def torch_lowrank_kv(batch: int, n_kv_heads: int, n_tokens: int, d: int, seed: int,
                     tensor_id: int, device, out=None, chunk_tokens: int = 4096):
    """Same recipe as :func:`lowrank_kv`, drawn on ``device`` with torch.

    Returns fp16 ``[batch][n_kv_heads][n_tokens][d]``.  The orthogonal bases
    are drawn on the host (small) and moved to the device.
    """
    import torch
    units = batch * n_kv_heads
    basis_id = T_KBASIS if tensor_id in (T_K, T_NEWK) else T_VBASIS
    bases = np.empty((units, d, d), np.float32)
    for u in range(units):
        bases[u] = random_orthogonal(d, rng(seed, 1000, 0, basis_id, u))
    wt = torch.from_numpy(bases).to(device).transpose(1, 2).contiguous()  # W^T
    sigma = torch.from_numpy(power_law_sigma(d).astype(np.float32)).to(device)
    if out is None:
        out = torch.empty((batch, n_kv_heads, n_tokens, d), dtype=torch.float16, device=device)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed_seq(seed, 1000, 0, tensor_id).generate_state(1)[0]))
    flat = out.view(units, n_tokens, d)
    for t0 in range(0, n_tokens, chunk_tokens):
        t1 = min(n_tokens, t0 + chunk_tokens)
        z = torch.randn((units, t1 - t0, d), generator=gen, device=device, dtype=torch.float32)
        flat[:, t0:t1] = torch.bmm(z * sigma, wt).to(torch.float16)
    return out


def torch_gaussian_fp16(shape, seed: int, tensor_id: int, device, scale: float = 1.0,
                        *extra: int):
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed_seq(seed, 2000, 0, tensor_id, *extra).generate_state(1)[0]))
    x = torch.randn(shape, generator=gen, device=device, dtype=torch.float32) * scale
    return x.to(torch.float16)


def spectrum(d: int, power: float) -> np.ndarray:
    """sigma_i ∝ i^-power (i = 1..d), normalised so that sum sigma_i^2 = d."""
    s = np.arange(1, d + 1, dtype=np.float64) ** -power
    return s * np.sqrt(d / np.sum(s * s))


def calibration(n_kv_heads: int, group: int, n_tokens: int, d: int, d_model: int, seed: int,
                workload: int, layer: int):
    """Host calibration set: fp16 ``Q [n_kv_heads*group][n_tokens][d]``,
    ``K, V [n_kv_heads][n_tokens][d]``, ``W_O [n_kv_heads*group*d][d_model]``."""
    H_q = n_kv_heads * group
    Q = np.empty((H_q, n_tokens, d), np.float16)
    K = np.empty((n_kv_heads, n_tokens, d), np.float16)
    V = np.empty((n_kv_heads, n_tokens, d), np.float16)
    W_O = np.empty((H_q * d, d_model), np.float16)
    s_flat, s_steep = spectrum(d, 0.5), spectrum(d, 1.0)
    for j in range(n_kv_heads):
        w_qk = random_orthogonal(d, rng(seed, workload, layer, T_QK_BASIS, j))
        w_vo = random_orthogonal(d, rng(seed, workload, layer, T_VO_BASIS, j))
        for g in range(group):
            h = j * group + g
            z = rng(seed, workload, layer, T_CAL_Q, h).standard_normal((n_tokens, d))
            Q[h] = ((z * s_flat) @ w_qk.T).astype(np.float16)
            y = rng(seed, workload, layer, T_CAL_WO, h).standard_normal((d, d_model)) / np.sqrt(d_model)
            W_O[h * d:(h + 1) * d] = ((w_vo * s_flat[None, :]) @ y).astype(np.float16)
        z = rng(seed, workload, layer, T_CAL_K, j).standard_normal((n_tokens, d))
        K[j] = ((z * s_steep) @ w_qk.T).astype(np.float16)
        z = rng(seed, workload, layer, T_CAL_V, j).standard_normal((n_tokens, d))
        V[j] = ((z * s_steep) @ w_vo.T).astype(np.float16)
    return Q, K, V, W_O


def torch_calibration(n_kv_heads: int, group: int, n_tokens: int, d: int, d_model: int, seed: int,
                      device, chunk_tokens: int = 8192):
    """Same recipe as :func:`calibration`, drawn on ``device`` (large sets)."""
    import torch
    H_q = n_kv_heads * group
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed_seq(seed, 3000, 0, T_CAL_Q).generate_state(1)[0]))
    s_flat = torch.from_numpy(spectrum(d, 0.5).astype(np.float32)).to(device)
    s_steep = torch.from_numpy(spectrum(d, 1.0).astype(np.float32)).to(device)
    w_qk = torch.from_numpy(np.stack([random_orthogonal(d, rng(seed, 3000, 0, T_QK_BASIS, j))
                                      for j in range(n_kv_heads)]).astype(np.float32)).to(device)
    w_vo = torch.from_numpy(np.stack([random_orthogonal(d, rng(seed, 3000, 0, T_VO_BASIS, j))
                                      for j in range(n_kv_heads)]).astype(np.float32)).to(device)
    Q = torch.empty((H_q, n_tokens, d), dtype=torch.float16, device=device)
    K = torch.empty((n_kv_heads, n_tokens, d), dtype=torch.float16, device=device)
    V = torch.empty((n_kv_heads, n_tokens, d), dtype=torch.float16, device=device)
    wq_t = w_qk.repeat_interleave(group, 0).transpose(1, 2).contiguous()
    for t0 in range(0, n_tokens, chunk_tokens):
        t1 = min(n_tokens, t0 + chunk_tokens)
        z = torch.randn((H_q, t1 - t0, d), generator=gen, device=device)
        Q[:, t0:t1] = torch.bmm(z * s_flat, wq_t).to(torch.float16)
        z = torch.randn((n_kv_heads, t1 - t0, d), generator=gen, device=device)
        K[:, t0:t1] = torch.bmm(z * s_steep, w_qk.transpose(1, 2)).to(torch.float16)
        z = torch.randn((n_kv_heads, t1 - t0, d), generator=gen, device=device)
        V[:, t0:t1] = torch.bmm(z * s_steep, w_vo.transpose(1, 2)).to(torch.float16)
    y = torch.randn((H_q, d, d_model), generator=gen, device=device) / float(np.sqrt(d_model))
    W_O = torch.bmm(w_vo.repeat_interleave(group, 0) * s_flat[None, None, :], y)
    return Q, K, V, W_O.reshape(H_q * d, d_model).to(torch.float16)
