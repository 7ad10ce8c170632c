"""SWAN decode benchmark on one GB300 (or N replicas, one per GPU).

One step = one pass of the whole hot path (Algorithm 1 for one token): append
one new key/value per sequence (rotate, insert into the dense buffer, evict
the oldest buffered vector and prune it into the sparse cache) and one decode
attention over the hybrid cache (rotate q, sparse + dense scores, online
softmax, value scatter, split combine, rotate-back).

Default workload: a Llama-2-7B-shaped attention layer at 32k context: batch
16, 32 MHA heads, head_dim 128, 32768 sparse tokens + 128 dense buffer tokens,
keep k = 64, synthetic low-rank keys/values (sigma_i ∝ 1/i), per-head random
orthogonal R.  Metric: decode KV-tokens/s (token-head records attended per
second) and HBM GB/s over the algorithmic bytes.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl swan|reference]
  python bench.py --workload gqa-131k   # Llama-3-8B GQA layer, 131072 ctx
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

for _v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

D = 128
WORKLOADS = {
    "latency-1k": dict(B=1, H_q=1, H_kv=1, L_s=1024, n_b=64, k=64, k_store=64, l2_flush=True,
                       desc="one head, batch 1, d 128, 1024 sparse + 64 dense-buffer tokens, k 64 "
                            "(L2-resident: latency)"),
    "llama2-7b-layer-32k": dict(B=16, H_q=32, H_kv=32, L_s=32768, n_b=128, k=64, k_store=64,
                                desc="Llama-2-7B-shaped layer: batch 16, 32 MHA heads, d 128, "
                                     "32768 sparse + 128 dense-buffer tokens, k 64"),
    "gqa-131k": dict(B=4, H_q=32, H_kv=8, L_s=130944, n_b=128, k=56, k_store=56,
                     desc="Llama-3-8B-shaped GQA layer: batch 4, 32 q / 8 kv heads, d 128, "
                          "130944 sparse + 128 dense-buffer tokens (131072 ctx), k 56"),
    "gqa8-32k": dict(B=4, H_q=64, H_kv=8, L_s=32640, n_b=128, k=56, k_store=56,
                     desc="GQA layer with 8 query heads per kv head (64 q / 8 kv heads, d 128, the "
                          "attention shape of a Llama-3-70B layer): batch 4, 32640 sparse + 128 "
                          "dense-buffer tokens (32768 ctx), k 56"),
    "ksweep-32k": dict(B=16, H_q=32, H_kv=32, L_s=32768, n_b=128, k=64, k_store=128,
                       desc="Llama-2-7B-shaped layer at 32k with k_store 128, decoded at a runtime "
                            "keep count k (--k-active)"),
    "stack-32x8k": dict(kind="stack", B=8, H_q=32, H_kv=32, layers=32, prefix=8192, n_b=128,
                        flush_every=128, max_steps=256, k=64, k_store=64,
                        desc="32-layer Llama-2-7B-shaped KV stack, batch 8, 8192-token prefix "
                             "compressed by one append per layer, decode steps appending one token "
                             "per layer, buffers flushed every 128 steps, k 64"),
    "ragged-serve-32": dict(kind="ragged", B=32, H_q=32, H_kv=32, n_b=128, k=64, k_store=64,
                            len_lo=1024, len_hi=65536, P=128, L_s=8192,
                            desc="serving batch of 32 Llama-2-7B-shaped sequences (32 MHA heads, d 128) "
                                 "whose contexts are drawn log-uniformly from 1024 to 65536 tokens (seeded), "
                                 "k 64, 128-token buffers; the pages come from one shared pool sized to "
                                 "the contexts (not to 32 x the longest)"),
    "basis-llama3-8b": dict(kind="basis", n_kv=8, G=4, n=65536, d_model=4096,
                            desc="offline basis (Section 4.1) for one Llama-3-8B-shaped layer: 32 q / 8 kv "
                                 "heads, d 128, d_model 4096; one step accumulates S_QK^T S_QK and "
                                 "S_VO^T S_VO over a calibration batch of 65536 tokens (Q, K, V and the "
                                 "W_O columns); the eigensolver runs once after the batches"),
}
METRIC = "decode-attention KV-tokens/s and achieved HBM GB/s (% of 8 TB/s) at 32k ctx"
BASIS_METRIC = "offline-basis calibration vectors/s (Gram accumulation on the tensor cores)"
NOMINAL_HBM_GBS = 8000.0


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return None


def decode_kernel_traffic(workload: str, values: str = "fp16", variant: str = ""):
    """DRAM bytes per decode-kernel launch from the committed ncu summary, if
    it was taken on the current kernel sources (every `<file> sha256[:16]`
    line of the summary must match that file now; else None)."""
    text = None
    suffix = ("" if values == "fp16" else "-fp8") + variant
    for name in (f"decode_kernel_{workload}{suffix}.md", f"decode_ws_kernel_{workload}{suffix}.md",
                 f"decode_mma_kernel_{workload}{suffix}.md"):
        try:
            text = open(os.path.join(ROOT, "profiles", name)).read()
            break
        except OSError:
            continue
    if text is None:
        return None
    hashes = re.findall(r"([\w.]+\.cuh) sha256\[:16\]:\s*([0-9a-f]{16})", text)
    m_tr = re.search(r"dram bytes per launch:\s*([0-9.eE+]+)", text)
    if not hashes or not m_tr:
        return None
    for fname, want in hashes:
        src = os.path.join(ROOT, "paper_2511_18936_gb300", "csrc", fname)
        try:
            digest = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        except OSError:
            return None
        if digest != want:
            return None
    return float(m_tr.group(1))


class ClockSampler:
    """nvidia-smi samples of SM clocks and throttle reasons during a region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        rows = []
        for ln in (self.out or "").splitlines():
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------------
# CPU baseline: the oracle as it stands, on a bounded sample of the workload
# ---------------------------------------------------------------------------

def oracle_sample(wl, n_units: int, seed: int = 0, first_unit: int = 0):
    """Prepare the compressed state of ``n_units`` (batch, kv-head) units of
    the workload on the host (untimed) and return a step function that runs
    one oracle step (append one token, decode every query head of the unit)."""
    import oracle
    from paper_2511_18936_gb300 import synth
    G = wl["H_q"] // wl["H_kv"]
    L_s = wl.get("L_s", wl.get("prefix"))
    L = L_s + wl["n_b"]
    states = []
    compress_s = 0.0
    for u in range(first_unit, first_unit + n_units):
        R = synth.rotations(1, D, seed=seed, workload=7, layer=0, tensor_id=synth.T_R_QK, )
        k = synth.lowrank_kv(1, 1, L + 64, D, seed, 7, u, synth.T_K)
        v = synth.lowrank_kv(1, 1, L + 64, D, seed, 7, u, synth.T_V)
        st = oracle.SwanOracle(R, batch=1, n_q_heads=G, k_store=wl["k_store"], buffer_cap=wl["n_b"],
                               value_format=wl["values"], k_store_v=wl["k_store_v"])
        t0 = time.perf_counter()
        st.append(k[:, :, :L_s], v[:, :, :L_s])
        st.flush()
        st.append(k[:, :, L_s:L], v[:, :, L_s:L])
        compress_s += time.perf_counter() - t0
        st.set_k(wl["k"], wl["k_v"])
        q = synth.gaussian_fp16((1, G, D), seed, 7, u, synth.T_Q)
        states.append((st, k[:, :, L:], v[:, :, L:], q))
    step_no = [0]

    def step():
        i = step_no[0] % 64
        step_no[0] += 1
        tokens = 0
        for st, kn, vn, q in states:
            st.append(kn[:, :, i:i + 1], vn[:, :, i:i + 1])
            st.decode(q)
            tokens += st.sparse_len + st.buffer_len
        return tokens
    # the compress step of the preparation: token-heads (a key and a value
    # vector each) rotated, pruned or buffered, per second
    step.compress = {"value": n_units * L / compress_s, "unit": "token-heads/s",
                     "sample": f"{n_units} unit(s) x {L} tokens (append {L_s}, flush, append {wl['n_b']}), "
                               f"{compress_s:.2f} s, NumPy fp64 single thread"}
    return step


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def _oracle_worker(wl, unit, warmup, steps, budget_s, barrier, results):
    """One host core: one (batch, kv-head) unit of the workload in the oracle
    (single-threaded NumPy), prepared untimed; then, between two barriers
    shared with every other core, `steps` oracle steps (or steps until
    `budget_s` has passed)."""
    step = oracle_sample(wl, 1, first_unit=unit)
    for _ in range(warmup):
        step()
    tokens, n = 0, 0
    barrier.wait()
    t0 = time.perf_counter()
    while (n < steps) if steps else (time.perf_counter() - t0 < budget_s):
        tokens += step()
        n += 1
    barrier.wait()
    results.put((tokens, n, step.compress["value"]))


def oracle_all_cores(wl, warmup: int = 1, steps: int = 0, budget_s: float = 15.0):
    """The oracle as it stands on every host core: one single-threaded oracle
    process per core, each on its own (batch, kv-head) unit of the workload
    (the units are independent), all timed together between two barriers.
    Processes are started with `spawn` (safe after CUDA has been used)."""
    import multiprocessing as mp
    n = host_cores()
    ctx = mp.get_context("spawn")
    barrier = ctx.Barrier(n + 1)
    results = ctx.Queue()
    procs = [ctx.Process(target=_oracle_worker, args=(wl, u, warmup, steps, budget_s, barrier, results),
                         daemon=True) for u in range(n)]
    for p in procs:
        p.start()
    try:
        barrier.wait(timeout=600)
        t0 = time.perf_counter()
        barrier.wait(timeout=600)
        wall = time.perf_counter() - t0
        got = [results.get(timeout=60) for _ in procs]
    finally:
        for p in procs:
            p.join(timeout=30)
            if p.is_alive():
                p.terminate()
    tokens = sum(g[0] for g in got)
    return {"value": tokens / wall, "unit": "KV-tokens/s", "cores": n, "kind": "oracle",
            "seconds": wall, "steps_per_core": [g[1] for g in got],
            "compress_per_core": statistics.mean(g[2] for g in got),
            "sample": f"{n} of {wl['B'] * wl['H_kv']} (batch, kv-head) units of the same workload "
                      f"({wl['H_q'] // wl['H_kv']} query heads each), one single-threaded NumPy fp64 oracle "
                      f"process per host core, each step append 1 token + decode, {wall:.1f} s"}


def basis_oracle_step(wl, n_tokens: int, seed: int = 0):
    """One oracle step of the basis workload on a bounded sample: the joint
    matrices of one kv head over ``n_tokens`` tokens and their SVD basis.
    Returns (step function, vectors per step)."""
    import oracle
    from paper_2511_18936_gb300 import synth
    G, d_model = wl["G"], wl["d_model"]
    Q, K, V, W_O = synth.calibration(1, G, n_tokens, D, d_model, seed=seed, workload=8, layer=0)
    bo = oracle.basis_oracle

    def step():
        bo.principal_basis(bo.joint_qk(Q, K, G)[0])
        bo.principal_basis(bo.joint_vo(V, W_O, G)[0])
    return step, (G + 2) * n_tokens + G * d_model


def run_reference(args, wl, rank: int):
    if rank != 0:
        return None
    if wl.get("kind") == "basis":
        return run_reference_basis(args, wl)
    # one thread: two units stepped in turn
    n_units = min(2, wl["B"] * wl["H_kv"])
    t0 = time.perf_counter()
    step = oracle_sample(wl, n_units)
    prep = time.perf_counter() - t0
    for _ in range(args.warmup):
        step()
    times, toks = [], 0
    for _ in range(args.steps):
        t = time.perf_counter()
        toks += step()
        times.append(time.perf_counter() - t)
    total1 = sum(times)
    single = {"value": toks / total1, "unit": "KV-tokens/s", "cores": 1, "kind": "oracle",
              "ms_per_step": 1e3 * total1 / args.steps,
              "sample": f"{n_units} of {wl['B'] * wl['H_kv']} (batch, kv-head) units of the workload, "
                        f"{wl['H_q'] // wl['H_kv']} query heads each, one thread; one step = append 1 token + "
                        f"decode; state preparation {prep:.1f} s outside the steps"}
    # every host core: one unit per core, all stepped at once (the line's value)
    allc = oracle_all_cores(wl, warmup=args.warmup, steps=args.steps)
    value = allc["value"]
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "KV-tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * allc["seconds"] / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.workload, "desc": wl["desc"],
                       "parallelism": f"host CPU, {allc['cores']} cores (one oracle process per core)"},
            "cpu_baseline": {"value": value, "unit": "KV-tokens/s", "cores": allc["cores"], "kind": "oracle",
                             "sample": allc["sample"] + f"; {args.steps} steps per core after {args.warmup} "
                                                        "untimed"},
            "single_thread": single,
            "e2e": {"value": value, "unit": "KV-tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "compress": step.compress}
    return line


def run_reference_basis(args, wl):
    n_tok = 8192
    step, vecs = basis_oracle_step(wl, n_tok)
    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    total = time.perf_counter() - t0
    value = vecs * args.steps / total
    sample = (f"1 of {wl['n_kv']} kv heads, {n_tok} of {wl['n']} calibration tokens: the joint matrices "
              f"S_QK and S_VO and their SVD bases (NumPy fp64)")
    return {"impl": "reference", "metric": BASIS_METRIC, "value": value, "unit": "vectors/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * total / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.workload, "desc": wl["desc"], "parallelism": "none (host CPU)"},
            "cpu_baseline": {"value": value, "unit": "vectors/s", "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "vectors/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def cpu_baseline_basis(wl, budget_s: float = 15.0):
    n_tok = 16384
    step, vecs = basis_oracle_step(wl, n_tok)
    step()
    t0 = time.perf_counter()
    n = 0
    while time.perf_counter() - t0 < budget_s:
        step()
        n += 1
    dt = time.perf_counter() - t0
    return {"value": vecs * n / dt, "unit": "vectors/s", "cores": 1, "kind": "oracle",
            "sample": f"1 of {wl['n_kv']} kv heads, {n_tok} calibration tokens, joint matrices + SVD "
                      f"basis (NumPy fp64, one thread), {n} steps in {dt:.1f} s"}


def gram_kernel_traffic(workload: str):
    """DRAM bytes per Gram launch from the committed ncu summary, if it was
    taken on the current kernel source (else None)."""
    src = os.path.join(ROOT, "paper_2511_18936_gb300", "csrc", "basis.cu")
    digest = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    try:
        text = open(os.path.join(ROOT, "profiles", f"gram_kernel_{workload}.md")).read()
    except OSError:
        return None
    m_src = re.search(r"basis\.cu sha256\[:16\]:\s*([0-9a-f]{16})", text)
    m_tr = re.search(r"dram bytes per launch:\s*([0-9.eE+]+)", text)
    if not m_src or not m_tr or m_src.group(1) != digest:
        return None
    return float(m_tr.group(1))


def run_basis(args, wl, rank: int, world: int, local_rank: int):
    """The offline-basis workload: Gram accumulation of the joint matrices
    over calibration batches on the tensor cores (the data-parallel part),
    the eigensolver timed once."""
    import torch

    from paper_2511_18936_gb300 import swan, synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    n_kv, G, n, d_model = wl["n_kv"], wl["G"], wl["n"], wl["d_model"]
    stream = torch.cuda.Stream(dev)
    with torch.cuda.stream(stream):
        Q, K, V, W_O = synth.torch_calibration(n_kv, G, n, D, d_model, seed=args.seed + rank, device=dev)
        gq, gv = swan.Gram(n_kv, dev, stream), swan.Gram(n_kv, dev, stream)
    stream.synchronize()
    parts = [("Q", gq, swan.rows_of(Q, G)), ("K", gq, swan.rows_of(K)), ("V", gv, swan.rows_of(V)),
             ("W_O", gv, swan.columns_of(W_O, G))]
    vecs = n_kv * G * n + 2 * n_kv * n + n_kv * G * d_model
    part_bytes = {"Q": Q.numel() * 2, "K": K.numel() * 2, "V": V.numel() * 2, "W_O": W_O.numel() * 2}

    def step():
        for name, g, v in parts:
            g.add(v, accumulate=True)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    stream.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local_rank) as clk:
        with torch.cuda.stream(stream):
            ev0.record(stream)
            for _ in range(args.steps):
                step()
            ev1.record(stream)
        stream.synchronize()
    ms = ev0.elapsed_time(ev1)
    if world > 1:
        torch.distributed.barrier()
    gq.check()
    gv.check()

    # per-part times (memset + Gram kernel + split reduction) in a second region
    part_ms = {}
    with torch.cuda.stream(stream):
        for name, g, v in parts:
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(args.steps):
                g.add(v, accumulate=True)
            b.record(stream)
            stream.synchronize()
            part_ms[name] = a.elapsed_time(b) / args.steps
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        both = torch.cat([gq.gram, gv.gram])  # one launch, one CTA per matrix
        a.record(stream)
        R_all, _, sw_all = swan.basis_eig(both, stream)
        b.record(stream)
    stream.synchronize()
    eig_ms = a.elapsed_time(b)

    # the energy that top-k pruning keeps (Section 4.1.2's purpose, without a
    # model): bases from the first half of the batch, measured on the held-out
    # second half, against a random orthogonal basis
    half = n // 2
    with torch.cuda.stream(stream):
        h_qk, h_vo = swan.Gram(n_kv, dev, stream), swan.Gram(n_kv, dev, stream)
        h_qk.add(swan.rows_of(Q[:, :half].contiguous(), G), False).add(swan.rows_of(K[:, :half].contiguous()))
        h_vo.add(swan.rows_of(V[:, :half].contiguous()), False).add(swan.columns_of(W_O, G))
        R_h, _, _ = swan.basis_eig(torch.cat([h_qk.gram, h_vo.gram]), stream)
        gen = np.random.default_rng(args.seed + 7)
        R_rand = torch.from_numpy(np.stack([synth.random_orthogonal(D, gen) for _ in range(n_kv)])
                                  .astype(np.float32)).to(dev)
        energy_kept = {}
        for name, held, R_data in (("K", K, R_h[:n_kv]), ("V", V, R_h[n_kv:])):
            rows = swan.rows_of(held[:, half:].contiguous())
            e_d = swan.energy(rows, R_data.contiguous(), stream=stream).sum(0)
            e_r = swan.energy(rows, R_rand, stream=stream).sum(0)
            energy_kept[name] = {f"k{k}": {"data_basis": float(e_d[k] / e_d[D]), "random_basis": float(e_r[k] / e_r[D])}
                                 for k in (16, 32, 56, 64, 96)}
    stream.synchronize()

    # end to end: Q, K, V of the batch copied from pinned host memory every
    # step, the Gram matrices read back
    host = [t.cpu().pin_memory() for t in (Q, K, V)]
    dev_in = [torch.empty_like(t) for t in (Q, K, V)]
    e2e_parts = [(gq, swan.rows_of(dev_in[0], G)), (gq, swan.rows_of(dev_in[1])), (gv, swan.rows_of(dev_in[2])),
                 (gv, swan.columns_of(W_O, G))]
    host_out = [torch.empty_like(g.gram, device="cpu").pin_memory() for g in (gq, gv)]

    def e2e_step():
        with torch.cuda.stream(stream):
            for d, h in zip(dev_in, host):
                d.copy_(h, non_blocking=True)
            for g, v in e2e_parts:
                g.add(v, accumulate=True)
            for ho, g in zip(host_out, (gq, gv)):
                ho.copy_(g.gram, non_blocking=True)
        stream.synchronize()

    e2e_step()
    t0 = time.perf_counter()
    for _ in range(args.e2e_steps):
        e2e_step()
    e2e_s = time.perf_counter() - t0

    value, e2e_value, t_max = aggregate_ranks(vecs * args.steps, ms, vecs * args.e2e_steps, e2e_s, world, dev)
    peaks = measured_peaks()
    peak = float(peaks["hbm_gbs"]) if peaks else 6800.0
    q_s = part_ms["Q"] / 1e3
    achieved = part_bytes["Q"] / q_s / 1e9
    tflops = part_bytes["Q"] / 256 * 2 * D * D / q_s / 1e12
    tpeak = float(peaks["bf16_tflops"]) if peaks and "bf16_tflops" in peaks else 1900.0
    line = {
        "metric": BASIS_METRIC, "value": value, "unit": "vectors/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_max / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16 x f16 -> f32",
        "data": "synthetic calibration set (seeded per-head principal bases, power-law spectra)",
        "config": {"workload": args.workload, "desc": wl["desc"], "n_kv_heads": n_kv, "group": G,
                   "tokens_per_batch": n, "d_model": d_model,
                   "l2": f"inputs larger than L2: {sum(part_bytes.values()) / 1e9:.2f} GB read per step, no flush",
                   "parallelism": f"replicas x{world} (independent batches per GPU)" if world > 1
                   else "single GPU"},
        "roofline": {"kernel": "gram (Q part: memset + gram_kernel + split reduction)", "bound": "hbm",
                     "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                     "peak_source": "MEASURED_PEAKS.json hbm_gbs (measured copy)" if peaks else "fallback 6.8 TB/s",
                     "alg_bytes_per_launch": part_bytes["Q"], "avg_launch_ms": part_ms["Q"],
                     "tensor_tflops": tflops, "tensor_frac_of_bf16_peak": tflops / tpeak,
                     "traffic": gram_kernel_traffic(args.workload)},
        "parts_ms_per_step": part_ms,
        "eig_ms_16_matrices": eig_ms,
        "eig_sweeps": sw_all.tolist(),
        "energy_kept": {"held_out": f"{n - half} tokens per kv head (bases from the other {half})",
                        **energy_kept},
        "gpu_launches": 2 * len(parts) * args.steps,
        "e2e": {"value": e2e_value, "unit": "vectors/s",
                "h2d_bytes_per_step": sum(t.numel() * t.element_size() for t in host),
                "d2h_bytes_per_step": sum(t.numel() * t.element_size() for t in host_out),
                "steps": args.e2e_steps},
        "clocks": clk.summary(),
    }
    return line


def cpu_baseline_leg(wl, budget_s: float = 15.0):
    """The oracle on every host core (the reported figure) and on one thread."""
    step = oracle_sample(wl, 1)
    step()
    t0 = time.perf_counter()
    toks, n = 0, 0
    while time.perf_counter() - t0 < budget_s:
        toks += step()
        n += 1
    dt = time.perf_counter() - t0
    single = {"value": toks / dt, "unit": "KV-tokens/s", "cores": 1, "kind": "oracle",
              "sample": f"1 of {wl['B'] * wl['H_kv']} (batch, kv-head) units of the same workload "
                        f"({wl['H_q'] // wl['H_kv']} query heads), {n} steps of append 1 token + decode, "
                        f"{dt:.1f} s, NumPy fp64 single thread",
              "compress": step.compress}
    line = oracle_all_cores(wl, budget_s=budget_s)
    line["single_thread"] = single
    line["compress"] = step.compress
    return line


# ---------------------------------------------------------------------------
# The CUDA path
# ---------------------------------------------------------------------------

def aggregate_ranks(kv_tokens: float, ms: float, e2e_tokens: float, e2e_s: float, world: int,
                    device=None):
    """Whole-job throughput over ``world`` replicas: every rank processed the
    same number of tokens; the job time is the slowest rank's (MAX over
    ranks).  Returns (value, e2e_value, max_ms)."""
    t_max, e2e_max = ms, e2e_s
    if world > 1:
        import torch
        tt = torch.tensor([ms, e2e_s], dtype=torch.float64, device=device)
        torch.distributed.all_reduce(tt, op=torch.distributed.ReduceOp.MAX)
        t_max, e2e_max = float(tt[0]), float(tt[1])
    return world * kv_tokens / (t_max / 1e3), world * e2e_tokens / e2e_max, t_max


class LayerRun:
    """One attention layer (the 1-head, 32k, GQA-131k and k-sweep workloads):
    prefill the context in one append, then per step append one token per
    sequence (the buffer is full, so one vector is evicted and pruned) and
    decode."""

    def __init__(self, wl, dev, stream, seed, steps_total):
        import torch

        from paper_2511_18936_gb300 import swan, synth
        self.wl = wl
        B, H_q, H_kv, L_s, n_b = wl["B"], wl["H_q"], wl["H_kv"], wl["L_s"], wl["n_b"]
        self.layers = 1
        self.max_seq = L_s + n_b + steps_total + 8
        with torch.cuda.stream(stream):
            R = torch.from_numpy(synth.rotations(H_kv, D, seed=seed, workload=1, layer=0))[None].to(dev)
            self.ctx = swan.Context(R, num_layers=1, batch=B, n_q_heads=H_q, n_kv_heads=H_kv,
                                    k_store=wl["k_store"], buffer_cap=n_b, max_seq=self.max_seq,
                                    stream=stream, value_format=wl["values"], k_store_v=wl["k_store_v"])
            kk = synth.torch_lowrank_kv(B, H_kv, L_s + n_b, D, seed, synth.T_K, dev)
            vv = synth.torch_lowrank_kv(B, H_kv, L_s + n_b, D, seed, synth.T_V, dev)
            # the prefill (one bulk append: rotate, prune L_s tokens, buffer n_b),
            # timed on the stream
            ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            ev0.record(stream)
            self.ctx.append(0, kk, vv)
            ev1.record(stream)
            del kk, vv
            k_new = synth.torch_lowrank_kv(B, H_kv, steps_total, D, seed, synth.T_NEWK, dev)
            v_new = synth.torch_lowrank_kv(B, H_kv, steps_total, D, seed, synth.T_NEWV, dev)
            self.k_steps = [k_new[:, :, i:i + 1].contiguous() for i in range(steps_total)]
            self.v_steps = [v_new[:, :, i:i + 1].contiguous() for i in range(steps_total)]
            del k_new, v_new
            self.qs = synth.torch_gaussian_fp16((steps_total, B, H_q, D), seed, synth.T_Q, dev)
            self.out = torch.empty((B, H_q, D), dtype=torch.float16, device=dev)
            self.ctx.set_k(wl["k"], wl["k_v"])
        stream.synchronize()
        self.prefill_ms = ev0.elapsed_time(ev1)
        self.ctx.check()

    def step(self, i):
        self.ctx.append_decode(0, self.k_steps[i], self.v_steps[i], self.qs[i], self.out, 1)

    def context_after(self, i):
        """(sparse, buffer) tokens attended by the decode of step i."""
        wl = self.wl
        return wl["L_s"] + i + 1, wl["n_b"]

    def host_inputs(self, i):
        return [self.k_steps[i], self.v_steps[i], self.qs[i]]

    def step_with(self, dev_inputs):
        dk, dv, dq = dev_inputs
        self.ctx.append_decode(0, dk, dv, dq, self.out, 1)
        return [self.out]


class RaggedRun(LayerRun):
    """A batch of sequences of different lengths sharing one page pool:
    prefilled in 2048-token chunks with per-row counts, then per step one
    token appended to every row and one decode."""

    def __init__(self, wl, dev, stream, seed, steps_total):
        import torch

        from paper_2511_18936_gb300 import swan, synth
        self.wl = wl
        B, H_q, H_kv, n_b, P = wl["B"], wl["H_q"], wl["H_kv"], wl["n_b"], wl["P"]
        gen = np.random.default_rng(synth.seed_seq(seed, 6, 0, 0))
        lo, hi = np.log(wl["len_lo"]), np.log(wl["len_hi"])
        self.lens = [int(x) for x in np.exp(gen.uniform(lo, hi, size=B)).round()]
        self.layers = 1
        self.max_seq = max(self.lens) + steps_total + 8
        sparse_max = [max(0, L + steps_total - n_b) for L in self.lens]
        pool = H_kv * sum((s + P - 1) // P for s in sparse_max) + B * H_kv
        self.pool_pages = pool
        with torch.cuda.stream(stream):
            R = torch.from_numpy(synth.rotations(H_kv, D, seed=seed, workload=1, layer=0))[None].to(dev)
            self.ctx = swan.Context(R, num_layers=1, batch=B, n_q_heads=H_q, n_kv_heads=H_kv,
                                    k_store=wl["k_store"], buffer_cap=n_b, max_seq=self.max_seq, page_tokens=P,
                                    stream=stream, value_format=wl["values"], k_store_v=wl["k_store_v"],
                                    pool_pages=pool)
            chunk = 2048
            for ci, t0 in enumerate(range(0, max(self.lens), chunk)):
                n_new = [max(0, min(chunk, L - t0)) for L in self.lens]
                kk = synth.torch_lowrank_kv(B, H_kv, chunk, D, seed * 1000 + ci, synth.T_K, dev)
                vv = synth.torch_lowrank_kv(B, H_kv, chunk, D, seed * 1000 + ci, synth.T_V, dev)
                self.ctx.append(0, kk, vv, chunk, n_new=n_new)
                del kk, vv
            k_new = synth.torch_lowrank_kv(B, H_kv, steps_total, D, seed, synth.T_NEWK, dev)
            v_new = synth.torch_lowrank_kv(B, H_kv, steps_total, D, seed, synth.T_NEWV, dev)
            self.k_steps = [k_new[:, :, i:i + 1].contiguous() for i in range(steps_total)]
            self.v_steps = [v_new[:, :, i:i + 1].contiguous() for i in range(steps_total)]
            del k_new, v_new
            self.qs = synth.torch_gaussian_fp16((steps_total, B, H_q, D), seed, synth.T_Q, dev)
            self.out = torch.empty((B, H_q, D), dtype=torch.float16, device=dev)
            self.ctx.set_k(wl["k"], wl["k_v"])
        stream.synchronize()
        self.ctx.check()
        self.page_bytes = self.ctx.query(0).page_bytes

    def rows_after(self, i):
        """Per-row (sparse, buffer) tokens attended by the decode of step i."""
        n_b = self.wl["n_b"]
        out = []
        for L in self.lens:
            tot = L + i + 1
            out.append((max(0, tot - n_b), min(tot, n_b)))
        return out

    def context_after(self, i):
        rows = self.rows_after(i)
        return (sum(sp for sp, _ in rows) / len(rows), sum(bf for _, bf in rows) / len(rows))


class StackRun:
    """A 32-layer KV stack: the prefix of every layer compressed by one
    append (timed separately), flushed, then decode steps that append one
    token per layer and decode it, with every layer's buffer flushed after
    each 128 steps."""

    def __init__(self, wl, dev, stream, seed, steps_total):
        import torch

        from paper_2511_18936_gb300 import swan, synth
        self.wl = wl
        B, H, Lyr, pre, cap = wl["B"], wl["H_q"], wl["layers"], wl["prefix"], wl["n_b"]
        self.layers = Lyr
        self.max_seq = pre + steps_total + 8
        self.flush_every = wl["flush_every"]
        R = np.stack([synth.rotations(H, D, seed=seed, workload=4, layer=l) for l in range(Lyr)])
        with torch.cuda.stream(stream):
            Rt = torch.from_numpy(R).to(dev)
            self.ctx = swan.Context(Rt, num_layers=Lyr, batch=B, n_q_heads=H, n_kv_heads=H,
                                    k_store=wl["k_store"], buffer_cap=cap, max_seq=self.max_seq,
                                    stream=stream, value_format=wl["values"], k_store_v=wl["k_store_v"])
            self.ctx.set_k(wl["k"], wl["k_v"])
        stream.synchronize()
        # prefix: one append per layer (plain Gaussian K/V), timed on the stream
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        self.prefix_ms = 0.0
        for l in range(Lyr):
            with torch.cuda.stream(stream):
                kk = synth.torch_gaussian_fp16((B, H, pre, D), seed, synth.T_K, dev, 1.0, l)
                vv = synth.torch_gaussian_fp16((B, H, pre, D), seed, synth.T_V, dev, 1.0, l)
                ev0.record(stream)
                self.ctx.append(l, kk, vv)
                self.ctx.flush(l)
                ev1.record(stream)
            stream.synchronize()
            self.prefix_ms += ev0.elapsed_time(ev1)
            del kk, vv
        with torch.cuda.stream(stream):
            kn = synth.torch_gaussian_fp16((Lyr, steps_total, B, H, 1, D), seed, synth.T_NEWK, dev)
            vn = synth.torch_gaussian_fp16((Lyr, steps_total, B, H, 1, D), seed, synth.T_NEWV, dev)
            self.kn, self.vn = kn, vn
            self.qs = synth.torch_gaussian_fp16((Lyr, steps_total, B, H, D), seed, synth.T_Q, dev)
            self.out = torch.empty((Lyr, B, H, D), dtype=torch.float16, device=dev)
        stream.synchronize()
        self.ctx.check()

    def _flush_due(self, i):
        return (i + 1) % self.flush_every == 0

    def step(self, i):
        for l in range(self.layers):
            self.ctx.append_decode(l, self.kn[l, i], self.vn[l, i], self.qs[l, i], self.out[l], 1)
        if self._flush_due(i):
            self.ctx.flush(-1)

    def context_after(self, i):
        # the buffer holds the tokens appended since the last flush
        in_buf = i % self.flush_every + 1
        return self.wl["prefix"] + i + 1 - in_buf, in_buf

    def host_inputs(self, i):
        return [self.kn[:, i], self.vn[:, i], self.qs[:, i]]

    def step_with(self, dev_inputs):
        dk, dv, dq = dev_inputs
        i = self._e2e_i
        for l in range(self.layers):
            self.ctx.append_decode(l, dk[l], dv[l], dq[l], self.out[l], 1)
        if self._flush_due(i):
            self.ctx.flush(-1)
        return [self.out]


def run_swan(args, wl, rank: int, world: int, local_rank: int):
    import torch

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    B, H_q, H_kv, k = wl["B"], wl["H_q"], wl["H_kv"], wl["k"]
    steps_total = args.warmup + 2 * args.steps + 2 * args.e2e_steps
    stream = torch.cuda.Stream(dev)
    seed = args.seed + rank
    kind = wl.get("kind", "layer")
    if kind == "stack" and steps_total > wl["max_steps"]:
        raise SystemExit(f"the stack workload runs at most {wl['max_steps']} decode steps")
    run = {"stack": StackRun, "ragged": RaggedRun}.get(kind, LayerRun)(wl, dev, stream, seed, steps_total)
    ctx = run.ctx
    flush_l2 = wl.get("l2_flush", False)
    l2_buf = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev) if flush_l2 else None

    for i in range(args.warmup):
        run.step(i)
    stream.synchronize()

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    def timed(step_range):
        """CUDA-event time of the steps on the context's stream (ms)."""
        if not flush_l2:
            ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            ev0.record(stream)
            for i in step_range:
                run.step(i)
            ev1.record(stream)
            stream.synchronize()
            return ev0.elapsed_time(ev1)
        # L2-resident workload: flush L2 (write 512 MB) before every timed step
        total = 0.0
        for i in step_range:
            with torch.cuda.stream(stream):
                l2_buf.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            run.step(i)
            e1.record(stream)
            stream.synchronize()
            total += e0.elapsed_time(e1)
        return total

    # ---- timed region: inputs resident in HBM -----------------------------
    steps = range(args.warmup, args.warmup + args.steps)
    launches0 = ctx.launch_count()
    barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local_rank) as clk:
        ms = timed(steps)
    barrier()
    torch.cuda.synchronize(dev)
    launches = ctx.launch_count() - launches0

    # ---- per-kernel CUDA-event times over a second timed region of the same
    # length (events between launches would hide the launch overlap above)
    ksteps = range(args.warmup + args.steps, args.warmup + 2 * args.steps)
    ctx.timing_enable(True)
    torch.cuda.synchronize(dev)
    timed(ksteps)
    kt = ctx.timing_read()
    ctx.timing_enable(False)

    # ---- end to end: pinned host inputs, H2D copies and the D2H read inside -
    e2e_steps = args.e2e_steps
    base = args.warmup + 2 * args.steps
    host = [[t.cpu().pin_memory() for t in run.host_inputs(base + i)] for i in range(2 * e2e_steps)]
    dev_in = [torch.empty_like(t, device=dev) for t in host[0]]
    host_out = [torch.empty_like(run.out, device="cpu").pin_memory()]

    def e2e_step(i):
        run._e2e_i = base + i
        with torch.cuda.stream(stream):
            for d, h in zip(dev_in, host[i]):
                d.copy_(h, non_blocking=True)
            outs = run.step_with(dev_in)
            for ho, o in zip(host_out, outs):
                ho.copy_(o, non_blocking=True)
        stream.synchronize()

    for i in range(e2e_steps):  # warm-up of the copy path
        e2e_step(i)
    barrier()
    t0 = time.perf_counter()
    e2e_tokens = 0
    for i in range(e2e_steps, 2 * e2e_steps):
        e2e_step(i)
        sp, bf = run.context_after(base + i)
        e2e_tokens += B * H_kv * (sp + bf) * run.layers
    e2e_s = time.perf_counter() - t0
    barrier()
    h2d = sum(t.numel() * t.element_size() for t in host[0])
    d2h = sum(t.numel() * t.element_size() for t in host_out)

    # ---- aggregate over ranks ----------------------------------------------
    ctxs = [run.context_after(i) for i in steps]
    kv_tokens = sum(B * H_kv * (sp + bf) * run.layers for sp, bf in ctxs)
    value, e2e_value, t_max = aggregate_ranks(kv_tokens, ms, e2e_tokens, e2e_s, world, dev)

    dec_ms, dec_n = kt["decode"]
    avg_dec_s = dec_ms / 1e3 / max(dec_n, 1)
    kctxs = [run.context_after(i) for i in ksteps]  # the region the kernels were timed on
    sp_mean = statistics.mean(sp for sp, _ in kctxs)
    bf_mean = statistics.mean(bf for _, bf in kctxs)
    # algorithmic bytes of one decode-kernel launch (one layer): per (sparse
    # token, kv head) (value + index bytes) * (k + k_v) (6k with fp16 values
    # and k_v = k, 4k with 8-bit values); per (buffer token, kv head) 2 * 2 * d
    sp_bytes = (2 if wl["values"] == "fp8_e4m3" else 3) * (k + wl["k_v"])
    alg_decode = B * H_kv * (sp_mean * sp_bytes + bf_mean * 4 * D)
    achieved = alg_decode / avg_dec_s / 1e9
    peaks = measured_peaks()
    peak = float(peaks["hbm_gbs"]) if peaks else 6800.0
    step_s = t_max / 1e3 / args.steps
    sp_step = statistics.mean(sp for sp, _ in ctxs)
    bf_step = statistics.mean(bf for _, bf in ctxs)
    alg_decode_step = B * H_kv * (sp_step * sp_bytes + bf_step * 4 * D)
    # whole-step algorithmic bytes per layer: decode reads + q/out (fp16) + R
    # (fp32, once per kv head, query and value rotations) + the append's new
    # vectors (fp16 in, fp16 to the buffer)
    alg_step = run.layers * (alg_decode_step + 2 * B * H_q * D * 2 + 2 * H_kv * D * D * 4
                             + B * H_kv * 2 * D * 2 * 2)
    l2_note = ("L2 flushed (512 MB written) before every timed step" if flush_l2 else
               f"inputs larger than L2: {alg_decode * run.layers / 1e9:.2f} GB read per step, no flush")
    cfg = {"workload": args.workload, "desc": wl["desc"], "batch": B, "n_q_heads": H_q,
           "n_kv_heads": H_kv, "layers": run.layers, "sparse_tokens": wl.get("L_s", wl.get("prefix")),
           "buffer_tokens": wl["n_b"], "k": k, "k_store": wl["k_store"],
           "k_v": wl["k_v"], "k_store_v": wl["k_store_v"],
           "storage": ("e4m3" if wl["values"] == "fp8_e4m3" else "fp16")
                      + " values + uint8 indices (sparse), fp16 (buffer)", "l2": l2_note,
           "parallelism": f"replicas x{world} (independent batches per GPU)" if world > 1
           else "single GPU"}
    if kind == "ragged":
        pb = run.page_bytes
        cfg["sparse_tokens"] = None
        cfg["context_lengths"] = {"min": min(run.lens), "mean": statistics.mean(run.lens), "max": max(run.lens)}
        cfg["pool_gb"] = run.pool_pages * pb / 1e9
        cfg["full_reservation_gb"] = B * H_kv * ((run.max_seq + wl["P"] - 1) // wl["P"]) * pb / 1e9
    line = {
        "metric": METRIC, "value": value, "unit": "KV-tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": t_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded low-rank K/V, Gaussian q, random orthogonal R)"
                if kind != "stack" else "synthetic (seeded Gaussian q/K/V, random orthogonal R)",
        "config": cfg,
        "hbm_gbs_step": alg_step / step_s / 1e9,
        "pct_of_8tbs_step": 100.0 * alg_step / step_s / 1e9 / NOMINAL_HBM_GBS,
        "roofline": {"kernel": "decode", "bound": "hbm", "achieved": achieved, "peak": peak,
                     "unit": "GB/s", "frac": achieved / peak,
                     "peak_source": "MEASURED_PEAKS.json hbm_gbs (measured copy)" if peaks
                     else "fallback 6.8 TB/s",
                     "pct_of_8tbs": 100.0 * achieved / NOMINAL_HBM_GBS,
                     "alg_bytes_per_launch": alg_decode, "avg_launch_ms": avg_dec_s * 1e3,
                     "traffic": decode_kernel_traffic(
                         args.workload, wl["values"],
                         ("" if wl["k_store_v"] == wl["k_store"] else f"-ksv{wl['k_store_v']}")
                         + (f"-k{k}" if args.workload == "ksweep-32k" else ""))},
        "kernels_ms_per_step": {name: v[0] / args.steps for name, v in kt.items() if v[1]},
        "kernels_timed": "second timed region of the same length, CUDA events around every launch",
        "gpu_launches": launches,
        "e2e": {"value": e2e_value, "unit": "KV-tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": e2e_steps},
        "clocks": clk.summary(),
    }
    if kind == "stack":
        line["prefix_ms"] = run.prefix_ms
        line["prefix_tokens_per_s"] = wl["layers"] * B * H_kv * wl["prefix"] / (run.prefix_ms / 1e3)
    elif type(run) is LayerRun:
        # the compress step of the prefill: token-heads (a key and a value
        # vector each) rotated, pruned or buffered, per second
        line["prefill_ms"] = run.prefill_ms
        line["prefill_tokens_per_s"] = B * H_kv * (wl["L_s"] + wl["n_b"]) / (run.prefill_ms / 1e3)
    ctx.check()
    ctx.close()
    return line


# Every other configuration of the benchmark, run after the headline line in
# the default invocation (one GPU) with bounded steps: (label, workload,
# make_workload overrides).  The k sweep re-prunes one k_store 128 cache at
# each runtime keep count.
SUB_WORKLOADS = [
    ("latency-1k", "latency-1k", {}),
    ("gqa-131k", "gqa-131k", {}),
    ("gqa-131k-e4m3", "gqa-131k", {"values": "fp8_e4m3"}),
    ("gqa8-32k", "gqa8-32k", {}),
    ("llama2-7b-layer-32k-e4m3", "llama2-7b-layer-32k", {"values": "fp8_e4m3"}),
    ("llama2-7b-layer-32k-kv64-32", "llama2-7b-layer-32k", {"k_store_v": 32}),
    *[(f"ksweep-32k-k{k}", "ksweep-32k", {"k_active": k}) for k in (32, 48, 64, 96, 128)],
    ("ragged-serve-32", "ragged-serve-32", {}),
    ("stack-32x8k", "stack-32x8k", {}),
    ("basis-llama3-8b", "basis-llama3-8b", {}),
]


def summarize(line):
    """The per-workload figures of a bench line (for the workloads object)."""
    rf = line["roofline"]
    out = {"desc": line["config"]["desc"], "value": line["value"], "unit": line["unit"],
           "ms_per_step": line["ms_per_step"], "steps": line["steps"], "warmup": line["warmup"],
           "gpu_launches": line["gpu_launches"], "e2e": line["e2e"], "clocks": line["clocks"],
           "l2": line["config"].get("l2"),
           "roofline": {k: rf.get(k) for k in ("kernel", "bound", "achieved", "peak", "unit", "frac", "pct_of_8tbs",
                                               "alg_bytes_per_launch", "avg_launch_ms", "traffic",
                                               "tensor_tflops") if k in rf}}
    if "alg_bytes_per_launch" in rf and rf.get("pct_of_8tbs") is not None and "L2 flushed" not in out["l2"]:
        # the time the decode launch would take at 70 % of the nominal 8 TB/s
        out["launch_ms_at_70pct_of_8tbs"] = rf["alg_bytes_per_launch"] / (0.7 * NOMINAL_HBM_GBS * 1e9) * 1e3
    for key in ("prefill_ms", "prefill_tokens_per_s", "prefix_ms", "prefix_tokens_per_s", "eig_ms_16_matrices"):
        if key in line:
            out[key] = line[key]
    return out


def run_workloads(args, rank: int, world: int, local_rank: int):
    """Run every configuration of SUB_WORKLOADS with bounded steps; a failure
    is recorded (and the others still run)."""
    import argparse as _ap
    import gc

    import torch
    res = {}
    for label, name, over in SUB_WORKLOADS:
        sub = _ap.Namespace(**vars(args))
        sub.workload = name
        sub.warmup = 3
        sub.steps = 20 if name == "latency-1k" else 10
        sub.e2e_steps = 5
        try:
            wl = make_workload(name, **over)
            line = (run_basis if wl.get("kind") == "basis" else run_swan)(sub, wl, rank, world, local_rank)
            res[label] = summarize(line)
        except Exception as e:  # noqa: BLE001 - recorded in the line, the rest still runs
            res[label] = {"error": f"{type(e).__name__}: {e}"[:300]}
        gc.collect()
        torch.cuda.empty_cache()
    return res


def make_workload(name: str, values: str = "fp16", batch: int = 0, k_active: int = 0, tokens: int = 0,
                  k_store_v: int = 0, k_active_v: int = 0):
    """The workload dict of ``name`` with the command line's overrides
    applied (ValueError on an out-of-range keep count)."""
    wl = dict(WORKLOADS[name])
    wl["values"] = values
    if values != "fp16":
        wl["desc"] += f" ({values} values)"
    if batch:
        wl["B"] = batch
        wl["desc"] += f" (batch overridden to {batch})"
    if k_active:
        if not 1 <= k_active <= wl["k_store"]:
            raise ValueError(f"--k-active must be in [1, {wl['k_store']}]")
        wl["k"] = k_active
        wl["desc"] += f" (k_active {k_active})"
    if wl.get("kind") == "basis":
        wl["k_store_v"] = wl["k_v"] = None
        if tokens:
            wl["n"] = tokens
            wl["desc"] += f" (tokens per batch overridden to {tokens})"
        return wl
    # value keep counts of the decode workloads
    wl["k_store_v"] = k_store_v or wl["k_store"]
    if not 1 <= wl["k_store_v"] <= D:
        raise ValueError(f"--k-store-v must be in [1, {D}]")
    if k_store_v:
        wl["desc"] += f" (k_store_v {wl['k_store_v']})"
    wl["k_v"] = min(wl["k"], wl["k_store_v"])
    if k_active_v:
        if not 1 <= k_active_v <= wl["k_store_v"]:
            raise ValueError(f"--k-active-v must be in [1, {wl['k_store_v']}]")
        wl["k_v"] = k_active_v
        wl["desc"] += f" (k_active_v {k_active_v})"
    return wl


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="swan", choices=["swan", "reference"])
    ap.add_argument("--workload", default="llama2-7b-layer-32k", choices=sorted(WORKLOADS))
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the other configurations the default run adds as 'workloads'")
    ap.add_argument("--batch", type=int, default=0,
                    help="override the workload's batch (smaller cases for profiling)")
    ap.add_argument("--values", default="fp16", choices=["fp16", "fp8_e4m3"],
                    help="kept sparse values as fp16 (3k bytes per vector) or E4M3 (2k)")
    ap.add_argument("--k-active", type=int, default=0,
                    help="runtime keep count (ksweep-32k: 32, 48, 64, 96 or 128)")
    ap.add_argument("--tokens", type=int, default=0,
                    help="basis workload: calibration tokens per batch (smaller cases for profiling)")
    ap.add_argument("--k-store-v", type=int, default=0,
                    help="value entries stored per vector (default: as for keys)")
    ap.add_argument("--k-active-v", type=int, default=0,
                    help="runtime value keep count (default: min(k_active, k_store_v))")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    try:
        wl = make_workload(args.workload, args.values, args.batch, args.k_active, args.tokens, args.k_store_v,
                           args.k_active_v)
    except ValueError as e:
        ap.error(str(e))

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        line = run_reference(args, wl, rank)
        if line is not None:
            print(json.dumps(line), flush=True)
        return

    if world > 1:
        import torch
        torch.distributed.init_process_group("nccl")
    basis = wl.get("kind") == "basis"
    line = (run_basis if basis else run_swan)(args, wl, rank, world, local_rank)
    if world == 1 and not args.no_workloads and args.workload == "llama2-7b-layer-32k" and \
            wl["desc"] == WORKLOADS[args.workload]["desc"]:
        line["workloads"] = run_workloads(args, rank, world, local_rank)
    if rank == 0:
        if not args.no_cpu_baseline and world == 1:
            line["cpu_baseline"] = cpu_baseline_basis(wl) if basis else cpu_baseline_leg(wl)
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
