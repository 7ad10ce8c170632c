"""CPU fp64 oracle for SWAN decode attention (test infrastructure only).

This file is the reference against which the CUDA path is checked.  Only the
test-suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import it; the library never calls it and has no CPU
fallback.  It shares no code with the CUDA path.

It restates the method of "SWAN: Sparse Winnowed Attention" (arXiv
2511.18936) step by step, in float64, with NumPy primitives (matmul, stable
argsort, gather, bincount) standing in for single steps:

* Section 4.2 and Algorithm 1: queries and keys are rotated by the orthogonal
  ``P_QK`` after RoPE, values arrive rotated by ``P_VO`` (row vectors:
  ``x_hat = x P``).  Here both rotations are applied explicitly to the
  unrotated inputs.
* Algorithm 1 and Section 4.3: a hybrid cache, a dense FIFO buffer of the
  ``b`` most recent rotated vectors, and a sparse history; when the buffer
  holds more than ``b`` vectors the oldest is popped, pruned to its top-k
  coordinates by magnitude (separately for the key and the value), and
  appended to the sparse history.
* Section 5.1: a sparse vector is stored as its kept values (fp16) and their
  coordinate indices (8-bit).
* Algorithm 1 and Section 3.2: the decode output is
  ``softmax(q_hat K_cache^T / sqrt(d_h)) V_cache`` over the concatenation of
  the sparse history and the buffer, computed on the sparse entries directly
  (gather for the scores, scatter-add for the values), with no reconstruction.
* Appendix A.1, Lemma 2: the per-head output is rotated back by ``P_VO^T``
  (the paper folds this into ``W_O``; the library returns it explicitly).

Readings where the paper is silent (each listed in the design notes):

* The stored representation of a rotated vector is its fp16 rounding (round
  to nearest even), and the top-k choice is made on that fp16 vector.
* Ties in magnitude go to the lower coordinate index.
* Kept entries are stored in decreasing magnitude order, so a smaller
  runtime keep count is a prefix of a larger one.
* The score scale is ``1/sqrt(d_h)`` with the full head dimension.
* With 8-bit values (Section 4.3, Section 5.1) the format is E4M3, the kept
  entries are chosen on the fp16 vector and then rounded to nearest even,
  saturating to +-448; the dense buffer stays fp16.
* The rotated query is not rounded.
* Query head ``h`` attends to kv head ``h // G`` (the reshape of Section
  4.1.1 groups consecutive query heads).
* An append of ``T`` tokens at once evicts, oldest first, every vector beyond
  the ``b`` most recent, exactly as ``T`` single appends would.

Parity status: every function below has a pin in ``tests/oracle_pins.py`` (run by
``tests/test_oracle_pins.py``).
The paper prints no worked example of an attention output at ``k < d`` with a
buffer; that general case is pinned by the decompression-free equivalence
(attention on the pruned cache equals PyTorch's scaled-dot-product attention
on the zero-filled rotated vectors followed by the buffer, rotated back:
agreement to 1e-12 at several keep counts and buffer sizes), with the
sparse entries pinned by a brute-force top-k, and by the special cases
k = d (dense attention), no pruning, the k-prefix property and the split
combine.
"""
from __future__ import annotations

import math

import numpy as np


# ---------------------------------------------------------------------------
# Rotation (Section 4.2, Algorithm 1)
# ---------------------------------------------------------------------------

def rotate(x, R) -> np.ndarray:
    """``x_hat = x R`` for row vectors ``x[..., d]`` (Section 4.2), in fp64."""
    return np.asarray(x, np.float64) @ np.asarray(R, np.float64)


def rotate_back(o_hat, R) -> np.ndarray:
    """``o = o_hat R^T`` (Appendix A.1, Lemma 2: ``P_VO P_VO^T = I``)."""
    return np.asarray(o_hat, np.float64) @ np.asarray(R, np.float64).T


def to_fp16(y) -> np.ndarray:
    """Round fp64 to fp16, round-to-nearest-even (NumPy rounds correctly)."""
    return np.asarray(y, np.float64).astype(np.float16)


# ---------------------------------------------------------------------------
# Magnitude top-k pruning (Algorithm 1, Section 4.3)
# ---------------------------------------------------------------------------

def prune(x16, k: int):
    """Top-``k`` coordinates of each vector by magnitude.

    ``x16[..., d]`` fp16.  Returns ``(idx uint8 [..., k], vals fp16 [..., k])``
    in decreasing magnitude order, ties to the lower index (stable sort).
    """
    x16 = np.asarray(x16, np.float16)
    d = x16.shape[-1]
    if not (1 <= k <= d):
        raise ValueError("k out of range")
    mag = np.abs(x16.astype(np.float64))
    order = np.argsort(-mag, axis=-1, kind="stable")[..., :k]
    vals = np.take_along_axis(x16, order, axis=-1)
    return order.astype(np.uint8), vals


def to_e4m3(x) -> np.ndarray:
    """Round to the 8-bit float E4M3 (1 sign, 4 exponent bits with bias 7,
    3 mantissa bits, no infinities; largest finite value 448, subnormal
    spacing 2^-9), round-to-nearest-even, saturating to +-448.  Returns the
    rounded values as fp64.  (Section 4.3 and Section 5.1 store the kept
    values as 8-bit floats; the format is E4M3.)"""
    x = np.asarray(x, np.float64)
    a = np.abs(x)
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -30)))
    e = np.maximum(e, -6.0)                    # below 2^-6 the spacing stays 2^-9
    q = np.exp2(e - 3.0)                       # spacing of the binade: 3 mantissa bits
    r = np.minimum(np.round(a / q) * q, 448.0)  # np.round: halves to even
    return np.copysign(r, x)


def densify(idx, vals, d: int) -> np.ndarray:
    """Zero-filled dense fp64 form of sparse vectors (used by pins only)."""
    idx = np.asarray(idx)
    out = np.zeros(idx.shape[:-1] + (d,), np.float64)
    np.put_along_axis(out, idx.astype(np.int64), np.asarray(vals, np.float64), axis=-1)
    return out


# ---------------------------------------------------------------------------
# Attention
# ---------------------------------------------------------------------------

def dense_attention(q, K, V) -> np.ndarray:
    """Textbook single-query attention ``softmax(q K^T / sqrt(d)) V``
    (Section 3, Section 3.2), fp64.  ``q[d]``, ``K[L, d]``, ``V[L, d]``."""
    q = np.asarray(q, np.float64)
    K = np.asarray(K, np.float64)
    V = np.asarray(V, np.float64)
    s = K @ q / math.sqrt(q.shape[-1])
    s = s - s.max()
    p = np.exp(s)
    return (p / p.sum()) @ V


def sparse_scores(q_hat, idx, vals) -> np.ndarray:
    """``s_t = sum_j q_hat[idx[t, j]] * vals[t, j]`` (the sparse-dense
    mat-vec of Algorithm 1 and Section 4.3)."""
    q_hat = np.asarray(q_hat, np.float64)
    return np.sum(q_hat[np.asarray(idx, np.int64)] * np.asarray(vals, np.float64), axis=-1)


def sparse_value_sum(p, idx, vals, d: int) -> np.ndarray:
    """``o[j] = sum_t sum_e p[t] * vals[t, e] * [idx[t, e] == j]`` (the sparse
    part of the value product), as a scatter-add."""
    idx = np.asarray(idx, np.int64)
    w = np.asarray(p, np.float64)[:, None] * np.asarray(vals, np.float64)
    return np.bincount(idx.ravel(), weights=w.ravel(), minlength=d)


def swan_attend_unit(q_hat, sp_idx, sp_vals_k, sp_idx_v, sp_vals_v, buf_k, buf_v,
                     k_active: int, d: int, k_active_v: int | None = None):
    """Attention of one rotated query over one unit's hybrid cache.

    Algorithm 1: ``S = q_hat Concat(K_sparse, K_buffer)^T``,
    ``o_hat = softmax(S / sqrt(d_h)) Concat(V_sparse, V_buffer)``; the sparse
    keys use their first ``k_active`` stored entries, the sparse values their
    first ``k_active_v`` (default: the same; the appendix ablation varies the
    two).  Returns ``(o_hat, scores)`` with the scores already divided by
    ``sqrt(d)``.
    """
    ka = k_active
    kv = k_active if k_active_v is None else k_active_v
    s_sp = sparse_scores(q_hat, sp_idx[:, :ka], sp_vals_k[:, :ka])
    s_bf = np.asarray(buf_k, np.float64) @ np.asarray(q_hat, np.float64)
    s = np.concatenate([s_sp, s_bf]) / math.sqrt(d)
    if s.size == 0:
        return np.zeros(d), s
    m = s.max()
    e = np.exp(s - m)
    p = e / e.sum()
    n_sp = s_sp.shape[0]
    o = sparse_value_sum(p[:n_sp], sp_idx_v[:, :kv], sp_vals_v[:, :kv], d)
    o = o + p[n_sp:] @ np.asarray(buf_v, np.float64)
    return o, s


def partial_state(scores, values):
    """Flash-style partial ``(m, l, acc)`` of a block of scores and their value
    rows: ``m = max s``, ``l = sum exp(s - m)``, ``acc = sum exp(s - m) v``."""
    s = np.asarray(scores, np.float64)
    if s.size == 0:
        return -np.inf, 0.0, np.zeros(np.asarray(values).shape[-1])
    m = s.max()
    e = np.exp(s - m)
    return m, e.sum(), e @ np.asarray(values, np.float64)


def combine_partials(parts):
    """Log-sum-exp merge of split partials (the split-K combine):
    ``m = max m_s``, ``l = sum l_s e^{m_s - m}``, ``acc = sum acc_s e^{m_s - m}``,
    result ``acc / l``."""
    ms = np.array([p[0] for p in parts], np.float64)
    m = ms.max()
    w = np.where(np.isfinite(ms), np.exp(ms - m), 0.0)
    l = sum(wi * p[1] for wi, p in zip(w, parts))
    acc = sum(wi * np.asarray(p[2], np.float64) for wi, p in zip(w, parts))
    return acc / l


# ---------------------------------------------------------------------------
# The hybrid cache as a state machine (Algorithm 1, Section 4.3)
# ---------------------------------------------------------------------------

class SwanOracle:
    """One layer's hybrid cache for ``batch`` sequences of equal length.

    ``R_qk``, ``R_vo``: ``[n_kv_heads][d][d]`` (fp32 or fp64); ``R_vo=None``
    uses ``R_qk`` for both.  ``round_rotated=False`` keeps the rotated vectors
    in fp64 (used only to check the lossless-rotation lemmas).
    """

    def __init__(self, R_qk, R_vo=None, *, batch: int, n_q_heads: int, k_store: int,
                 buffer_cap: int, round_rotated: bool = True, value_format: str = "fp16",
                 k_store_v: int | None = None):
        self.R_qk = np.asarray(R_qk, np.float64)
        self.R_vo = self.R_qk if R_vo is None else np.asarray(R_vo, np.float64)
        self.H_kv, self.d, _ = self.R_qk.shape
        self.B = batch
        self.H_q = n_q_heads
        if self.H_q % self.H_kv:
            raise ValueError("n_q_heads must be a multiple of n_kv_heads")
        self.G = self.H_q // self.H_kv
        k_store_v = k_store if k_store_v is None else k_store_v
        if not (1 <= k_store <= self.d) or not (1 <= k_store_v <= self.d):
            raise ValueError("k_store out of range")
        self.k_store = k_store      # keys
        self.k_store_v = k_store_v  # values
        self.k_active = k_store
        self.k_active_v = k_store_v
        self.b = buffer_cap
        self.round = round_rotated
        if value_format not in ("fp16", "fp8_e4m3"):
            raise ValueError("value_format must be fp16 or fp8_e4m3")
        self.fp8 = value_format == "fp8_e4m3"
        vdt = np.float16 if round_rotated else np.float64
        self.buf_k = np.zeros((self.B, self.H_kv, 0, self.d), vdt)
        self.buf_v = np.zeros((self.B, self.H_kv, 0, self.d), vdt)
        self.sp_idx_k = np.zeros((self.B, self.H_kv, 0, k_store), np.uint8)
        self.sp_val_k = np.zeros((self.B, self.H_kv, 0, k_store), vdt)
        self.sp_idx_v = np.zeros((self.B, self.H_kv, 0, k_store_v), np.uint8)
        self.sp_val_v = np.zeros((self.B, self.H_kv, 0, k_store_v), vdt)

    # -- Section 4.2 / Algorithm 1: rotate the incoming key and value -------
    def _rotate_store(self, x, R):
        y = np.einsum("bhti,hij->bhtj", np.asarray(x, np.float64), R)
        return to_fp16(y) if self.round else y

    def _prune(self, x, k: int):
        if self.round:
            idx, vals = prune(x, k)
            if self.fp8:
                # the kept fp16 values are stored as E4M3 (exact in fp16)
                vals = to_e4m3(vals.astype(np.float64)).astype(np.float16)
            return idx, vals
        # fp64 variant (lemma checks only): same rule on the fp64 vector
        mag = np.abs(x)
        order = np.argsort(-mag, axis=-1, kind="stable")[..., :k]
        return order.astype(np.uint8), np.take_along_axis(x, order, axis=-1)

    def _move_to_sparse(self, n: int):
        """Pop the ``n`` oldest buffered vectors, prune them (K and V
        separately) and append them to the sparse history."""
        if n <= 0:
            return
        ik, vk = self._prune(self.buf_k[:, :, :n], self.k_store)
        iv, vv = self._prune(self.buf_v[:, :, :n], self.k_store_v)
        self.sp_idx_k = np.concatenate([self.sp_idx_k, ik], axis=2)
        self.sp_val_k = np.concatenate([self.sp_val_k, vk], axis=2)
        self.sp_idx_v = np.concatenate([self.sp_idx_v, iv], axis=2)
        self.sp_val_v = np.concatenate([self.sp_val_v, vv], axis=2)
        self.buf_k = self.buf_k[:, :, n:]
        self.buf_v = self.buf_v[:, :, n:]

    def append(self, k, v):
        """Append ``T`` tokens ``k, v [batch][n_kv_heads][T][d]`` (unrotated);
        evict oldest-first while the buffer holds more than ``b`` vectors."""
        k_hat = self._rotate_store(k, self.R_qk)
        v_hat = self._rotate_store(v, self.R_vo)
        self.buf_k = np.concatenate([self.buf_k, k_hat], axis=2)
        self.buf_v = np.concatenate([self.buf_v, v_hat], axis=2)
        self._move_to_sparse(self.buf_k.shape[2] - self.b)

    def flush(self):
        """Move every buffered vector to the sparse history."""
        self._move_to_sparse(self.buf_k.shape[2])

    def set_k(self, k_active: int, k_active_v: int | None = None):
        """Runtime keep counts for keys and values (values default to
        ``min(k_active, k_store_v)``)."""
        if k_active_v is None:
            k_active_v = min(k_active, self.k_store_v)
        if not (1 <= k_active <= self.k_store) or not (1 <= k_active_v <= self.k_store_v):
            raise ValueError("k_active out of range")
        self.k_active = k_active
        self.k_active_v = k_active_v

    @property
    def sparse_len(self) -> int:
        return self.sp_idx_k.shape[2]

    @property
    def buffer_len(self) -> int:
        return self.buf_k.shape[2]

    def decode(self, q, return_rotated: bool = False):
        """``q [batch][n_q_heads][d]`` (unrotated, post-RoPE) -> fp64 output
        ``[batch][n_q_heads][d]`` in the original (unrotated) value basis."""
        q = np.asarray(q, np.float64)
        out = np.zeros((self.B, self.H_q, self.d))
        o_hat_all = np.zeros_like(out)
        for b in range(self.B):
            for hq in range(self.H_q):
                h = hq // self.G
                q_hat = q[b, hq] @ self.R_qk[h]
                o_hat, _ = swan_attend_unit(
                    q_hat, self.sp_idx_k[b, h], self.sp_val_k[b, h],
                    self.sp_idx_v[b, h], self.sp_val_v[b, h],
                    self.buf_k[b, h], self.buf_v[b, h], self.k_active, self.d, self.k_active_v)
                o_hat_all[b, hq] = o_hat
                out[b, hq] = rotate_back(o_hat, self.R_vo[h])
        return (out, o_hat_all) if return_rotated else out

    def decode_unit(self, q_vec, b: int, hq: int):
        """Output of a single (batch, query-head) pair; cheap sampling."""
        h = hq // self.G
        q_hat = np.asarray(q_vec, np.float64) @ self.R_qk[h]
        o_hat, _ = swan_attend_unit(
            q_hat, self.sp_idx_k[b, h], self.sp_val_k[b, h],
            self.sp_idx_v[b, h], self.sp_val_v[b, h],
            self.buf_k[b, h], self.buf_v[b, h], self.k_active, self.d, self.k_active_v)
        return rotate_back(o_hat, self.R_vo[h])


class RaggedOracle:
    """A batch whose sequences (rows) differ in length: one single-row
    ``SwanOracle`` per row, each following Algorithm 1 on its own tokens.
    ``append(k, v, n_new)`` gives row b the first ``n_new[b]`` of the ``T``
    tokens ``k[b, :, :T]``; ``reset(b)`` empties row b.  An empty row decodes
    to zeros."""

    def __init__(self, R_qk, R_vo=None, *, batch: int, n_q_heads: int, k_store: int, buffer_cap: int,
                 value_format: str = "fp16", k_store_v: int | None = None):
        self._args = dict(batch=1, n_q_heads=n_q_heads, k_store=k_store, buffer_cap=buffer_cap,
                          value_format=value_format, k_store_v=k_store_v)
        self._R = (R_qk, R_vo)
        self.rows = [SwanOracle(R_qk, R_vo, **self._args) for _ in range(batch)]
        self.k_active, self.k_active_v = k_store, k_store if k_store_v is None else k_store_v

    def append(self, k_new, v_new, n_new=None):
        T = k_new.shape[2]
        for b, row in enumerate(self.rows):
            n = T if n_new is None else int(n_new[b])
            if n:
                row.append(k_new[b:b + 1, :, :n], v_new[b:b + 1, :, :n])

    def flush(self):
        for row in self.rows:
            row.flush()

    def reset(self, b: int):
        self.rows[b] = SwanOracle(*self._R, **self._args)
        self.rows[b].set_k(self.k_active, self.k_active_v)

    def set_k(self, k_active: int, k_active_v: int | None = None):
        for row in self.rows:
            row.set_k(k_active, k_active_v)
        self.k_active, self.k_active_v = self.rows[0].k_active, self.rows[0].k_active_v

    def decode(self, q):
        return np.concatenate([row.decode(q[b:b + 1]) for b, row in enumerate(self.rows)])

    @property
    def sparse_lens(self):
        return [row.sparse_len for row in self.rows]

    @property
    def buffer_lens(self):
        return [row.buffer_len for row in self.rows]


# ---------------------------------------------------------------------------
# Byte and FLOP accounting (Section 5, Appendix "Derivation of Computational
# Complexity")
# ---------------------------------------------------------------------------

def sparse_vector_bytes(k: int, value_bytes: int = 2, index_bytes: int = 1,
                        offset_bytes: int = 2) -> int:
    """Section 5.1: ``k (sizeof(value) + sizeof(index)) + 2``; fp16 gives
    ``3k + 2``, fp8 values give ``2k + 2``."""
    return k * (value_bytes + index_bytes) + offset_bytes


def dense_vector_bytes(d: int, value_bytes: int = 2) -> int:
    """Section 5.1: a dense fp16 vector takes ``2 d`` bytes."""
    return d * value_bytes


def compression_ratio(k: int, d: int, value_bytes: int = 2) -> float:
    """Section 5.1: sparse bytes over dense bytes."""
    return sparse_vector_bytes(k, value_bytes) / dense_vector_bytes(d)


def flops_standard(L: int, d: int) -> int:
    """Appendix, standard attention per head per decode step: ``4 L d``."""
    return 4 * L * d


def flops_swan(L: int, d: int, k: int, b: int) -> int:
    """Appendix, SWAN per head per decode step:
    ``4 d^2 + 4 (L - b) k + 4 b d``."""
    return 4 * d * d + 4 * (L - b) * k + 4 * b * d


def break_even_length(d: int, k: int, b: int) -> float:
    """Eq. (break-even), Section 5.2: SWAN is cheaper once
    ``L > d^2 / (d - k) + b`` (requires ``k < d``)."""
    if k >= d:
        raise ValueError("break-even needs k < d")
    return d * d / (d - k) + b
