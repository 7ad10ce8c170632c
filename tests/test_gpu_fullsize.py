"""Full-size workloads on the GPU, checked against the oracle on sampled
(batch, head) units (needs a GB300).

Each test builds the whole cache through the C ABI exactly as bench.py does
(one prefill append, then decode steps), and recomputes a few sampled units
with the CPU oracle from host copies of the very same inputs.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2511_18936_gb300 import synth
from tests.helpers import TOL_OUT, check_topk_near_ties

pytestmark = pytest.mark.gpu

D = 128


def _layer_case(B, H_q, H_kv, L_s, n_b, k_store, k_actives, samples, seed=0, steps=2,
                value_format="fp16", q_scale=1.0):
    """Prefill L_s + n_b tokens, then `steps` decode steps (append one token +
    decode at every k in k_actives); compare sampled units with the oracle."""
    import torch

    from paper_2511_18936_gb300 import swan
    dev = torch.device("cuda")
    G = H_q // H_kv
    R = synth.rotations(H_kv, D, seed=seed, workload=1, layer=0)
    ctx = swan.Context(torch.from_numpy(R)[None].to(dev), num_layers=1, batch=B, n_q_heads=H_q,
                       n_kv_heads=H_kv, k_store=k_store, buffer_cap=n_b, max_seq=L_s + n_b + steps,
                       value_format=value_format)
    kk = synth.torch_lowrank_kv(B, H_kv, L_s + n_b + steps, D, seed, synth.T_K, dev)
    vv = synth.torch_lowrank_kv(B, H_kv, L_s + n_b + steps, D, seed, synth.T_V, dev)
    ctx.append(0, kk[:, :, :L_s + n_b].contiguous(), vv[:, :, :L_s + n_b].contiguous())
    qs = synth.torch_gaussian_fp16((steps, B, H_q, D), seed, synth.T_Q, dev, q_scale)
    refs = {}
    for b, h in samples:
        st = oracle.SwanOracle(R[h:h + 1], batch=1, n_q_heads=G, k_store=k_store, buffer_cap=n_b,
                               value_format=value_format)
        st.append(kk[b:b + 1, h:h + 1, :L_s + n_b].cpu().numpy(), vv[b:b + 1, h:h + 1, :L_s + n_b].cpu().numpy())
        refs[(b, h)] = st
    worst = 0.0
    for i in range(steps):
        t = L_s + n_b + i
        ctx.append(0, kk[:, :, t:t + 1].contiguous(), vv[:, :, t:t + 1].contiguous())
        for (b, h), st in refs.items():
            st.append(kk[b:b + 1, h:h + 1, t:t + 1].cpu().numpy(), vv[b:b + 1, h:h + 1, t:t + 1].cpu().numpy())
        q_host = qs[i].cpu().numpy()
        for ka in k_actives:
            ctx.set_k(ka)
            out = ctx.decode(0, qs[i]).float().cpu().numpy()
            for (b, h), st in refs.items():
                st.set_k(ka)
                want = st.decode(q_host[b:b + 1, h * G:(h + 1) * G])[0]
                err = float(np.abs(out[b, h * G:(h + 1) * G] - want).max())
                worst = max(worst, err)
                assert err <= TOL_OUT, (i, ka, b, h, err)
    info = ctx.query(0)
    assert info.sparse_len == L_s + steps and info.buffer_len == n_b
    ctx.check()
    ctx.check_guards()
    ctx.close()
    return worst


def test_llama2_layer_32k_sampled():
    _layer_case(B=16, H_q=32, H_kv=32, L_s=32768, n_b=128, k_store=64, k_actives=(64,),
                samples=[(0, 0), (7, 19), (15, 31)])


def test_llama2_layer_32k_fp8_values_sampled():
    _layer_case(B=16, H_q=32, H_kv=32, L_s=32768, n_b=128, k_store=64, k_actives=(64,),
                samples=[(1, 2), (14, 29)], value_format="fp8_e4m3")


def test_gqa_131k_sampled():
    _layer_case(B=4, H_q=32, H_kv=8, L_s=130944, n_b=128, k_store=56, k_actives=(56,),
                samples=[(0, 0), (3, 7)])


@pytest.mark.parametrize("fmt", ["fp16", "fp8_e4m3"])
def test_gqa_131k_peaked_queries_sampled(fmt):
    """Queries scaled by 4 (peaked softmax) on the 131k GQA layer: the
    regime where the score precision (q' gathers) shows most."""
    _layer_case(B=4, H_q=32, H_kv=8, L_s=130944, n_b=128, k_store=56, k_actives=(56,),
                samples=[(1, 3)], seed=1, q_scale=4.0, value_format=fmt)


@pytest.mark.parametrize("seed,q_scale", [(0, 1.0), (1, 4.0)])
def test_gqa_g8_32k_sampled(seed, q_scale):
    """Eight query heads per kv head (a 64-query, 8-kv-head layer) at 32k
    context: the two-gather q' path and the two-product value path, split
    over many CTAs, with ordinary and peaked (x4) queries."""
    _layer_case(B=2, H_q=64, H_kv=8, L_s=32640, n_b=128, k_store=56, k_actives=(56, 24),
                samples=[(0, 0), (1, 7)], seed=seed, q_scale=q_scale)


def test_ksweep_32k_sampled_and_dense_at_k128():
    _layer_case(B=16, H_q=32, H_kv=32, L_s=32768, n_b=128, k_store=128,
                k_actives=(32, 48, 64, 96, 128), samples=[(2, 5), (11, 30)], steps=1)


def test_ksweep_k128_equals_dense_attention():
    """k_active = d on the 32k shape: SWAN equals dense attention on the
    unrotated inputs up to the fp16 storage of the rotated vectors."""
    import torch

    from paper_2511_18936_gb300 import swan
    dev = torch.device("cuda")
    B, H, L = 16, 32, 32768 + 128
    R = synth.rotations(H, D, seed=3, workload=1, layer=0)
    ctx = swan.Context(torch.from_numpy(R)[None].to(dev), num_layers=1, batch=B, n_q_heads=H,
                       n_kv_heads=H, k_store=128, buffer_cap=128, max_seq=L)
    kk = synth.torch_lowrank_kv(B, H, L, D, 3, synth.T_K, dev)
    vv = synth.torch_lowrank_kv(B, H, L, D, 3, synth.T_V, dev)
    ctx.append(0, kk, vv)
    q = synth.torch_gaussian_fp16((B, H, D), 3, synth.T_Q, dev)
    out = ctx.decode(0, q).float().cpu().numpy()
    qh = q.cpu().numpy()
    for b, h in ((0, 0), (9, 21), (15, 31)):
        dense = oracle.dense_attention(qh[b, h], kk[b, h].cpu().numpy(), vv[b, h].cpu().numpy())
        err = float(np.abs(out[b, h] - dense).max())
        assert err <= TOL_OUT, (b, h, err)
    ctx.close()


def test_stack_32_layers_prefix_and_flush_schedule_sampled():
    """32 layers, batch 8, 8192-token prefix compressed by one append per
    layer, then 256 decode steps appending one token per layer with every
    buffer flushed after each 128 steps; sampled (layer, step, unit) outputs
    against an oracle replay of the same op log, and the sampled units'
    packed caches after the prefix against the fp64 rotation."""
    import torch

    from paper_2511_18936_gb300 import swan
    dev = torch.device("cuda")
    Lyr, B, H, pre, cap, k, steps = 32, 8, 32, 8192, 128, 64, 256
    sample_layers, sample_steps = (0, 31), (0, 127, 128, 255)
    sample_units = [(0, 0), (5, 17)]
    R = np.stack([synth.rotations(H, D, seed=0, workload=4, layer=l) for l in range(Lyr)])
    ctx = swan.Context(torch.from_numpy(R).to(dev), num_layers=Lyr, batch=B, n_q_heads=H,
                       n_kv_heads=H, k_store=k, buffer_cap=cap, max_seq=pre + steps)
    kn = synth.torch_gaussian_fp16((Lyr, steps, B, H, 1, D), 0, synth.T_NEWK, dev)
    vn = synth.torch_gaussian_fp16((Lyr, steps, B, H, 1, D), 0, synth.T_NEWV, dev)
    qs = synth.torch_gaussian_fp16((Lyr, steps, B, H, D), 0, synth.T_Q, dev)
    refs = {}
    for l in range(Lyr):
        kk = synth.torch_gaussian_fp16((B, H, pre, D), 0, synth.T_K, dev, 1.0, l)
        vv = synth.torch_gaussian_fp16((B, H, pre, D), 0, synth.T_V, dev, 1.0, l)
        ctx.append(l, kk, vv)
        ctx.flush(l)
        if l in sample_layers:
            for b, h in sample_units:
                st = oracle.SwanOracle(R[l, h:h + 1], batch=1, n_q_heads=1, k_store=k, buffer_cap=cap)
                st.append(kk[b:b + 1, h:h + 1].cpu().numpy(), vv[b:b + 1, h:h + 1].cpu().numpy())
                st.flush()
                refs[(l, b, h)] = st
                # the packed cache the bulk append left, against the fp64
                # rotation of the same vectors (near-ties allowed)
                for which, x in (("k", kk), ("v", vv)):
                    gi, gv = ctx.export_sparse_seq(l, b, which)
                    y64 = x[b, h].cpu().numpy().astype(np.float64) @ R[l, h].astype(np.float64)
                    check_topk_near_ties(y64, gi[h], gv[h], k)
        del kk, vv
    knh, vnh, qsh = kn.cpu().numpy(), vn.cpu().numpy(), qs.cpu().numpy()
    outs = torch.empty((Lyr, B, H, D), dtype=torch.float16, device=dev)
    for i in range(steps):
        for l in range(Lyr):
            ctx.append(l, kn[l, i], vn[l, i], 1)
            ctx.decode(l, qs[l, i], outs[l])
        if i in sample_steps:
            got = outs.float().cpu().numpy()
        for (l, b, h), st in refs.items():
            st.append(knh[l, i, b:b + 1, h:h + 1], vnh[l, i, b:b + 1, h:h + 1])
            if i in sample_steps:
                want = st.decode(qsh[l, i, b:b + 1, h:h + 1])[0, 0]
                err = float(np.abs(got[l, b, h] - want).max())
                assert err <= TOL_OUT, (l, i, b, h, err)
        if (i + 1) % 128 == 0:
            ctx.flush(-1)
            for st in refs.values():
                st.flush()
    for l in range(Lyr):
        info = ctx.query(l)
        assert info.sparse_len == pre + steps and info.buffer_len == 0
    ctx.check()
    ctx.check_guards()
    ctx.close()
