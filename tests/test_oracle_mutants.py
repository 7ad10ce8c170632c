"""Plant plausible mistakes in a copy of the oracle; each must fail a pin.

The mutant is the oracle's own source with one small textual change, loaded as
a separate module on the CPU; the real oracle is never modified.
"""
import importlib.util
import os
import sys
import types

import pytest

from tests.oracle_pins import ALL_PINS, BASIS_PINS

ORACLE_DIR = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle")
SRC = os.path.join(ORACLE_DIR, "swan_oracle.py")
BASIS_SRC = os.path.join(ORACLE_DIR, "basis_oracle.py")

# (name, original text, mutated text, count of occurrences to replace)
MUTANTS = [
    ("transposed_R_for_cache",
     'np.einsum("bhti,hij->bhtj"', 'np.einsum("bhti,hji->bhtj"', 1),
    ("transposed_R_for_query",
     "q_hat = q[b, hq] @ self.R_qk[h]", "q_hat = q[b, hq] @ self.R_qk[h].T", 1),
    ("rotate_back_without_transpose",
     "@ np.asarray(R, np.float64).T", "@ np.asarray(R, np.float64)", 1),
    ("prune_smallest",
     'np.argsort(-mag, axis=-1, kind="stable")[..., :k]\n    vals',
     'np.argsort(mag, axis=-1, kind="stable")[..., :k]\n    vals', 1),
    ("prune_signed_not_magnitude",
     "mag = np.abs(x16.astype(np.float64))", "mag = x16.astype(np.float64)", 1),
    ("prune_ties_to_higher_index",
     'order = np.argsort(-mag, axis=-1, kind="stable")[..., :k]\n    vals',
     'order = (mag.shape[-1] - 1 - np.argsort(-mag[..., ::-1], axis=-1, kind="stable"))[..., :k]\n    vals', 1),
    ("scale_sqrt_k",
     "s = np.concatenate([s_sp, s_bf]) / math.sqrt(d)",
     "s = np.concatenate([s_sp, s_bf]) / math.sqrt(ka)", 1),
    ("dropped_buffer_values",
     "o = o + p[n_sp:] @ np.asarray(buf_v, np.float64)", "o = o", 1),
    ("value_sum_without_weights",
     "w = np.asarray(p, np.float64)[:, None] * np.asarray(vals, np.float64)",
     "w = np.asarray(vals, np.float64) + 0 * np.asarray(p)[:, None]", 1),
    ("key_indices_used_for_values",
     "o = sparse_value_sum(p[:n_sp], sp_idx_v[:, :kv]", "o = sparse_value_sum(p[:n_sp], sp_idx[:, :kv]", 1),
    ("combine_wrong_sign",
     "np.exp(ms - m)", "np.exp(m - ms)", 1),
    ("evict_newest",
     "ik, vk = self._prune(self.buf_k[:, :, :n], self.k_store)",
     "ik, vk = self._prune(self.buf_k[:, :, -n:], self.k_store)", 1),
    ("keys_pruned_with_the_value_count",
     "ik, vk = self._prune(self.buf_k[:, :, :n], self.k_store)",
     "ik, vk = self._prune(self.buf_k[:, :, :n], self.k_store_v)", 1),
    ("values_use_the_key_keep_count",
     "kv = k_active if k_active_v is None else k_active_v", "kv = k_active", 1),
    ("gqa_modulo_mapping",
     "h = hq // self.G\n                q_hat", "h = hq % self.H_kv\n                q_hat", 1),
    ("no_fp16_storage",
     "return to_fp16(y) if self.round else y", "return y", 1),
    ("break_even_without_buffer",
     "return d * d / (d - k) + b", "return d * d / (d - k)", 1),
    ("bytes_without_offset",
     "return k * (value_bytes + index_bytes) + offset_bytes",
     "return k * (value_bytes + index_bytes)", 1),
    ("e4m3_two_mantissa_bits",
     "q = np.exp2(e - 3.0)", "q = np.exp2(e - 2.0)", 1),
    ("e4m3_no_saturation",
     "r = np.minimum(np.round(a / q) * q, 448.0)", "r = np.round(a / q) * q", 1),
    ("e4m3_no_subnormals",
     "e = np.maximum(e, -6.0)", "e = np.maximum(e, -30.0)", 1),
    ("fp8_values_not_rounded",
     "vals = to_e4m3(vals.astype(np.float64)).astype(np.float16)", "vals = vals", 1),
    ("ragged_append_ignores_counts",
     "n = T if n_new is None else int(n_new[b])", "n = T", 1),
    ("runtime_k_ignored",
     "s_sp = sparse_scores(q_hat, sp_idx[:, :ka], sp_vals_k[:, :ka])",
     "s_sp = sparse_scores(q_hat, sp_idx, sp_vals_k)", 1),
]


BASIS_MUTANTS = [
    ("basis_rows_of_vt", "P = vt.T\n", "P = vt\n", 1),
    ("basis_ascending", "P = vt.T\n", "P = vt.T[:, ::-1]\n", 1),
    ("basis_no_sign_rule", "return fix_signs(P), sigma", "return P * np.sign(P[0])[None, :], sigma", 1),
    ("qk_grouped_by_modulo",
     "q_rows = Q[j * group:(j + 1) * group]", "q_rows = Q[j::n_kv]", 1),
    ("vo_slice_rows_not_columns", "parts.append(W_O[h * d:(h + 1) * d, :].T)",
     "parts.append(W_O[h * d:(h + 1) * d, :d].T)", 1),
    ("vo_values_dropped", "parts = [V[j]]", "parts = [0 * V[j]]", 1),
    ("gram_transposed", "return S.T @ S", "return S @ S.T", 1),
    ("gram_drops_first_row", "return S.T @ S", "return S[1:].T @ S[1:]", 1),
    ("gram_drops_last_row", "return S.T @ S", "return S[:-1].T @ S[:-1]", 1),
    ("gram_diagonal_only", "return S.T @ S", "return np.diag(np.sum(S * S, axis=0))", 1),
    ("energy_smallest_first", "sq = np.sort(Y * Y, axis=1)[:, ::-1]", "sq = np.sort(Y * Y, axis=1)", 1),
    ("energy_unsquared", "sq = np.sort(Y * Y, axis=1)[:, ::-1]", "sq = np.sort(np.abs(Y), axis=1)[:, ::-1]", 1),
    ("energy_unrotated", "Y = np.asarray(X, np.float64) @ np.asarray(P, np.float64)",
     "Y = np.asarray(X, np.float64) + 0 * np.asarray(P)[0, 0]", 1),
]


def _load_mutant(name, old, new, count, src_path=SRC):
    src = open(src_path).read()
    assert src.count(old) == count, (name, src.count(old))
    mod = types.ModuleType("oracle_mutant_" + name)
    mod.__file__ = src_path
    sys.modules[mod.__name__] = mod
    exec(compile(src.replace(old, new), src_path, "exec"), mod.__dict__)
    return mod


def _caught(mod, pins):
    failed = []
    for pin in pins:
        try:
            pin(mod)
        except Exception as e:  # noqa: BLE001 - any failure counts as caught
            failed.append((pin.__name__, type(e).__name__))
    return failed


@pytest.mark.parametrize("name,old,new,count", BASIS_MUTANTS, ids=[m[0] for m in BASIS_MUTANTS])
def test_basis_mutant_is_caught(name, old, new, count):
    mod = _load_mutant(name, old, new, count, BASIS_SRC)
    assert _caught(mod, BASIS_PINS), f"mutant {name} passed every pin"


@pytest.mark.parametrize("name,old,new,count", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(name, old, new, count):
    mod = _load_mutant(name, old, new, count)
    failed = []
    for pin in ALL_PINS:
        try:
            pin(mod)
        except Exception as e:  # noqa: BLE001 - any failure counts as caught
            failed.append((pin.__name__, type(e).__name__))
    assert failed, f"mutant {name} passed every pin"
