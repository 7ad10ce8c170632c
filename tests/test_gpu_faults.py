"""Failures made on the host and the guard regions around device buffers
(needs a GB300).  swan_debug_fail_after fails an allocation or a launch in
the library without calling CUDA, so no GPU fault is ever caused: the tests
check the documented outcomes (NOMEM with nothing left allocated; CUDA, then
STATE for every later call, on a poisoned context; other contexts
unaffected)."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2511_18936_gb300 import synth
from tests.helpers import TOL_OUT, run_ops

pytestmark = pytest.mark.gpu

D = 128


def _ctx(**kw):
    import torch

    from paper_2511_18936_gb300 import swan
    H = kw.pop("H", 4)
    R = torch.from_numpy(synth.rotations(H, D, seed=3, workload=97, layer=0))[None].cuda()
    args = dict(num_layers=1, batch=2, n_q_heads=H, n_kv_heads=H, k_store=64, buffer_cap=16, max_seq=4096)
    args.update(kw)
    return swan.Context(R, **args)


def test_every_allocation_failure_frees_the_rest():
    import torch

    from paper_2511_18936_gb300 import swan
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    fired = 0
    try:
        for i in range(64):
            swan.debug_fail_after(swan.FAULT_ALLOC, i)
            try:
                ctx = _ctx(max_seq=65536)  # a pool of ~100 MB: a leak would show
            except swan.SwanError as e:
                assert e.status == swan.ERR_NOMEM and "injected" in str(e)
                torch.cuda.synchronize()
                assert abs(torch.cuda.mem_get_info()[0] - free0) < (4 << 20), i
                fired += 1
                continue
            ctx.close()  # i is past the last allocation: nothing was injected
            break
        else:
            pytest.fail("swan_init made more than 64 allocations")
    finally:
        swan.debug_fail_after(swan.FAULT_ALLOC, -1)
    assert fired >= 10  # every buffer of the context was tried


@pytest.mark.parametrize("when", [0, 1, 2])
def test_launch_failure_poisons_only_its_context(when):
    """The (when+1)-th launch after arming fails: the call returns CUDA, every
    later call on that context returns STATE, destroy works, and another
    context on the same device computes correctly."""
    import torch

    from paper_2511_18936_gb300 import swan
    ctx = _ctx()
    dev = torch.device("cuda")
    k = torch.from_numpy(synth.lowrank_kv(2, 4, 40, D, 3, 97, 0, synth.T_K)).to(dev)
    v = torch.from_numpy(synth.lowrank_kv(2, 4, 40, D, 3, 97, 0, synth.T_V)).to(dev)
    q = torch.from_numpy(synth.gaussian_fp16((2, 4, D), 3, 97, 0, synth.T_Q)).to(dev)
    ctx.append(0, k, v)
    ctx.decode(0, q)
    torch.cuda.synchronize()
    swan.debug_fail_after(swan.FAULT_LAUNCH, when)
    try:
        statuses = []
        for _ in range(3):  # append_decode: two launches per call; the third call sees the poison
            try:
                ctx.append_decode(0, k[:, :, :1].contiguous(), v[:, :, :1].contiguous(), q)
                statuses.append(swan.OK)
            except swan.SwanError as e:
                statuses.append(e.status)
    finally:
        swan.debug_fail_after(swan.FAULT_LAUNCH, -1)
    first_bad = statuses.index(swan.ERR_CUDA)
    assert first_bad == when // 2
    assert all(s == swan.ERR_STATE for s in statuses[first_bad + 1:])
    with pytest.raises(swan.SwanError) as e:
        ctx.decode(0, q)
    assert e.value.status == swan.ERR_STATE
    with pytest.raises(swan.SwanError) as e:
        ctx.check()
    assert e.value.status == swan.ERR_STATE
    ctx.close()
    # a fresh context is unaffected
    kk = synth.lowrank_kv(1, 2, 70, D, 4, 97, 1, synth.T_K)
    vv = synth.lowrank_kv(1, 2, 70, D, 4, 97, 1, synth.T_V)
    qq = synth.gaussian_fp16((1, 2, D), 4, 97, 1, synth.T_Q)
    R = synth.rotations(2, D, seed=4, workload=97, layer=1)
    ctx2, _, outs = run_ops([("append", kk, vv), ("decode", qq)], R, None, B=1, H_kv=2, G=1, k_store=48, cap=8)
    for got, want in outs:
        assert np.abs(got - want).max() <= TOL_OUT
    ctx2.close()


def test_guards_hold_across_paths():
    """Every kind of write the library does (bulk and decode-step appends with
    eviction, flushes, a shared page pool handing out its last pages, GQA and
    E4M3 decodes, ragged rows, a reset) leaves all guard regions intact."""
    import torch

    from paper_2511_18936_gb300 import swan
    dev = torch.device("cuda")
    for fmt, H_q, H_kv in (("fp16", 4, 4), ("fp8_e4m3", 8, 2)):
        R = torch.from_numpy(synth.rotations(H_kv, D, seed=5, workload=97, layer=2))[None].to(dev)
        B, cap, P = 3, 8, 32
        max_seq = 300
        pages = B * H_kv * ((max_seq + P - 1) // P)  # exactly enough pages
        ctx = swan.Context(R, num_layers=1, batch=B, n_q_heads=H_q, n_kv_heads=H_kv, k_store=40, buffer_cap=cap,
                           max_seq=max_seq, page_tokens=P, value_format=fmt, k_store_v=24, pool_pages=pages)
        q = torch.from_numpy(synth.gaussian_fp16((B, H_q, D), 5, 97, 2, synth.T_Q)).to(dev)
        for i, (T, n_new) in enumerate(((100, None), (90, [90, 10, 0]), (1, None), (1, [1, 0, 1]), (5, None))):
            k = torch.from_numpy(synth.lowrank_kv(B, H_kv, T, D, 5, 97, 10 + i, synth.T_K)).to(dev)
            v = torch.from_numpy(synth.lowrank_kv(B, H_kv, T, D, 5, 97, 10 + i, synth.T_V)).to(dev)
            ctx.append_decode(0, k, v, q, T=T, n_new=n_new)
        ctx.flush(0)
        ctx.decode(0, q)
        ctx.reset_sequence(1)
        ctx.decode(0, q)
        ctx.check()
        ctx.check_guards()
        ctx.close()


def test_bulk_append_wait_runs_out_and_reports_timeout():
    """A bounded barrier wait of the tensor-core bulk append runs out: with
    swan_debug_starve_tc the next such launch issues no copies, so its MMA
    thread's wait on the tile barrier (armed, but with no producer) gives up
    after 1 ms.  Nothing is left in flight; swan_check reports
    DEVICE_TIMEOUT, and a fresh context on the same device then appends and
    decodes correctly."""
    import time

    import torch

    from paper_2511_18936_gb300 import swan
    dev = torch.device("cuda")
    ctx = _ctx(H=2)
    k = torch.from_numpy(synth.lowrank_kv(2, 2, 300, D, 6, 97, 3, synth.T_K)).to(dev)
    v = torch.from_numpy(synth.lowrank_kv(2, 2, 300, D, 6, 97, 3, synth.T_V)).to(dev)
    torch.cuda.synchronize()
    swan.debug_starve_tc(1_000_000)
    try:
        t0 = time.perf_counter()
        ctx.append(0, k, v)              # 600 vectors: the tensor-core path
        with pytest.raises(swan.SwanError) as e:
            ctx.check()
        elapsed = time.perf_counter() - t0
    finally:
        swan.debug_starve_tc(0)
    assert e.value.status == swan.ERR_DEVICE_TIMEOUT, e.value
    assert elapsed < 1.5, elapsed        # the 1 ms limit, not the default 2 s
    ctx.check()                          # the word was cleared; nothing else fired
    ctx.close()
    kk = synth.lowrank_kv(2, 2, 300, D, 6, 97, 4, synth.T_K)
    vv = synth.lowrank_kv(2, 2, 300, D, 6, 97, 4, synth.T_V)
    qq = synth.gaussian_fp16((2, 2, D), 6, 97, 4, synth.T_Q)
    R = synth.rotations(2, D, seed=6, workload=97, layer=4)
    ctx2, _, outs = run_ops([("append", kk, vv), ("decode", qq)], R, None, B=2, H_kv=2, G=1, k_store=48, cap=16)
    for got, want in outs:
        assert np.abs(got - want).max() <= TOL_OUT
    ctx2.close()


def test_gram_wait_runs_out_and_reports_timeout():
    """The same for the Gram kernel of the offline basis: starved, every CTA's
    MMA thread gives up after 1 ms, swan_basis_check reports DEVICE_TIMEOUT
    (and clears it), and the next accumulation is correct again."""
    import torch

    from paper_2511_18936_gb300 import swan
    n_kv, G, n = 2, 2, 700
    Q, K, _, _ = synth.calibration(n_kv, G, n, D, 64, seed=9, workload=60, layer=0)
    dev = torch.device("cuda")
    tq, tk = torch.from_numpy(Q).to(dev), torch.from_numpy(K).to(dev)
    g = swan.Gram(n_kv)
    swan.debug_starve_tc(1_000_000)
    try:
        g.add(swan.rows_of(tq, G), accumulate=False)
        with pytest.raises(swan.SwanError) as e:
            g.check()
    finally:
        swan.debug_starve_tc(0)
    assert e.value.status == swan.ERR_DEVICE_TIMEOUT, e.value
    g.check()
    g.add(swan.rows_of(tq, G), accumulate=False).add(swan.rows_of(tk))
    g.check()
    got = g.gram.double().cpu().numpy()
    for j, S in enumerate(oracle.basis_oracle.joint_qk(Q, K, G)):
        A = np.abs(S)
        assert (np.abs(got[j] - oracle.basis_oracle.gram(S)) <= 2.0 ** -14 * (A.T @ A) + 1e-30).all(), j
