"""Drive the oracle and the CUDA path through the same op log; comparison
utilities for the parity tests."""
from __future__ import annotations

import numpy as np

import oracle

TOL_OUT = 2e-3  # max-abs tolerance on attention outputs (fp16 storage, fp32 accumulate)


def run_ops(ops, R, Rv, *, B, H_kv, G, k_store, cap, max_seq=None, page_tokens=0,
            check_each=True, value_format="fp16", k_store_v=None):
    """Replay ``ops`` on the oracle and on a libswan context.

    ops: ("append", k, v) | ("flush",) | ("set_k", k) | ("set_kv", k, k_v) |
    ("decode", q); all arrays fp16 NumPy.  Returns (ctx, ref, [(gpu_out, ref_out), ...]).
    """
    import torch

    from paper_2511_18936_gb300 import swan

    dev = torch.device("cuda")
    if max_seq is None:
        max_seq = sum(op[1].shape[2] for op in ops if op[0] == "append") or 1
    ref = oracle.SwanOracle(R, Rv, batch=B, n_q_heads=H_kv * G, k_store=k_store, buffer_cap=cap,
                            value_format=value_format, k_store_v=k_store_v)
    Rt = torch.from_numpy(np.asarray(R, np.float32))[None].to(dev).contiguous()
    Rvt = None if Rv is None else torch.from_numpy(np.asarray(Rv, np.float32))[None].to(dev).contiguous()
    ctx = swan.Context(Rt, Rvt, num_layers=1, batch=B, n_q_heads=H_kv * G, n_kv_heads=H_kv,
                       k_store=k_store, buffer_cap=cap, max_seq=max_seq, page_tokens=page_tokens,
                       value_format=value_format, k_store_v=k_store_v or 0)
    outs = []
    for op in ops:
        if op[0] == "append":
            ref.append(op[1], op[2])
            ctx.append(0, torch.from_numpy(op[1]).to(dev), torch.from_numpy(op[2]).to(dev))
        elif op[0] == "flush":
            ref.flush()
            ctx.flush(0)
        elif op[0] == "set_k":
            ref.set_k(op[1])
            ctx.set_k(op[1])
        elif op[0] == "set_kv":
            ref.set_k(op[1], op[2])
            ctx.set_k(op[1], op[2])
        elif op[0] == "decode":
            want = ref.decode(op[1])
            got = ctx.decode(0, torch.from_numpy(op[1]).to(dev))
            torch.cuda.synchronize()
            outs.append((got.float().cpu().numpy().astype(np.float64), want))
        else:
            raise ValueError(op)
        if check_each:
            info = ctx.query(0)
            assert info.sparse_len == ref.sparse_len, (info.sparse_len, ref.sparse_len)
            assert info.buffer_len == ref.buffer_len, (info.buffer_len, ref.buffer_len)
    ctx.check()
    ctx.check_guards()
    return ctx, ref, outs


def fp16_ulp_distance(a, b) -> np.ndarray:
    """Distance in units in the last place between fp16 arrays (sign-aware)."""
    def ordered(x):
        u = np.asarray(x, np.float16).view(np.uint16).astype(np.int64)
        return np.where(u & 0x8000, -(u & 0x7FFF), u)
    return np.abs(ordered(a) - ordered(b))


def check_topk_near_ties(y64, idx, vals, k):
    """Validate a GPU-pruned vector set against the fp64 rotated vectors
    ``y64`` (the oracle's, before rounding) allowing near-ties: every kept
    coordinate is at least as large as every dropped one, and the stored order
    is non-increasing, up to max(1e-3, 2^-9 |y|); kept values are within one
    fp16 ulp of round(y)."""
    y64 = np.asarray(y64, np.float64).reshape(-1, y64.shape[-1])
    idx = np.asarray(idx).reshape(-1, idx.shape[-1])[:, :k].astype(np.int64)
    vals = np.asarray(vals).reshape(-1, vals.shape[-1])[:, :k]
    N, d = y64.shape
    ay = np.abs(y64)
    kept = np.zeros((N, d), bool)
    np.put_along_axis(kept, idx, True, axis=1)
    assert (kept.sum(1) == k).all(), "duplicate indices"
    ak = np.take_along_axis(ay, idx, axis=1)
    min_kept = ak.min(1)
    if k < d:
        max_drop = np.where(kept, -np.inf, ay).max(1)
        tol = np.maximum(1e-3, 2.0 ** -9 * np.maximum(min_kept, max_drop))
        bad = min_kept < max_drop - tol
        assert not bad.any(), f"{bad.sum()} vectors keep a clearly smaller coordinate"
    tol_o = np.maximum(1e-3, 2.0 ** -9 * ak[:, :-1])
    assert (ak[:, :-1] >= ak[:, 1:] - tol_o).all(), "stored order not by decreasing magnitude"
    want_vals = np.take_along_axis(y64, idx, axis=1).astype(np.float16)
    assert fp16_ulp_distance(vals, want_vals).max() <= 1, "values differ by more than one fp16 ulp"
