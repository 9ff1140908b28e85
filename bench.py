#!/usr/bin/env python3
"""Benchmark of the block-hybrid decoding hot path on GB300.

One step = one denoising step of block-hybrid attention over the active block
of every request followed by the commit of that block into the per-request
states (hybrid_block_attn_commit, one launch): every stage of Section 3.1's
per-block computation, for the batch-64 ragged-prefix GQA workload by default.
The same step as two separate launches (hybrid_block_attn, then
hybrid_commit_block) is timed afterwards for context.

Metric: active-block tokens per second = n_req * B * steps / time.

Timing: CUDA events on the launching stream; W untimed warm-up steps, then
exactly K timed steps bracketed by a barrier and torch.cuda.synchronize();
L2 is defeated by rotating through independent buffer sets whose total size is
more than 4x the L2.  With --gpus N (launched by torchrun) every rank runs its
own independent batch (weak scaling, no collective on the data path) and the
slowest rank's time is used.

--impl reference times the fp64 CPU oracle instead (host cores, bounded
sample per step), printing the same JSON line with "impl": "reference".
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import re
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "active-block tokens/sec per denoising step at batch 64; HBM GB/s vs GB300 peak"
FALLBACK_HBM_GBS = 6800.0


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------
def dist_info():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(value: float, ws: int, device=None) -> float:
    """Max of a float over all ranks (identity for a single process)."""
    if ws <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def rank_workload(wl, rank: int):
    """The batch rank `rank` draws: every rank has its own independent requests
    (weak scaling; no data is exchanged between ranks)."""
    return wl.with_(seed=wl.seed + 1000 * rank) if rank else wl


def barrier(ws: int):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            return json.load(fh), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


_COMMENT = re.compile(r"//[^\n]*|/\*.*?\*/", re.S)


def source_sha(paths):
    """Hash of the kernel's sources with comments and whitespace removed, so a
    recorded capture stays valid across comment-only edits and no longer."""
    h = hashlib.sha256()
    for p in paths:
        with open(os.path.join(ROOT, p), encoding="utf-8") as fh:
            code = _COMMENT.sub(" ", fh.read())
        h.update(" ".join(code.split()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str):
    """Per-launch DRAM bytes from a committed ncu summary, or None if absent or
    taken on a different build of the kernel's source."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as fh:
            rec = json.load(fh).get(kernel)
    except (OSError, ValueError):
        return None
    if not rec or rec.get("workload") != workload:
        return None
    if rec.get("source_sha") != source_sha(rec.get("sources", [])):
        return None
    return rec.get("bytes_per_launch")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 50 ms."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, bus_id: str | None):
        self.samples = []   # (t, sm_mhz, max_mhz, reasons)
        self.proc = None
        self.bus_id = bus_id
        self.thread = None

    def start(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50"]
        if self.bus_id:
            cmd += ["-i", self.bus_id]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm, mx = float(parts[1]), float(parts[2])
            except ValueError:
                continue
            reasons = [n for n, v in zip(self.REASONS, parts[5:9]) if v.lower() == "active"]
            self.samples.append((time.time(), sm, mx, reasons))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=5)

    def summary(self, t0, t1):
        inside = [s for s in self.samples if t0 <= s[0] <= t1]
        window = "timed region"
        if not inside:
            inside = [s for s in self.samples if t0 - 2.0 <= s[0] <= t1 + 0.5]
            window = "timed region +-2 s (timed region shorter than the 50 ms sampling period)"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "window": "no nvidia-smi samples"}
        reasons = sorted({r for s in inside for r in s[3]})
        return {"sm_mhz": float(np.median([s[1] for s in inside])),
                "sm_max_mhz": float(max(s[2] for s in inside)),
                "reasons": reasons, "samples": len(inside), "window": window}


def bus_id_of(torch, dev):
    try:
        p = torch.cuda.get_device_properties(dev)
        return f"{p.pci_domain_id:08X}:{p.pci_bus_id:02X}:{p.pci_device_id:02X}.0"
    except Exception:  # noqa: BLE001
        return None


# ---------------------------------------------------------------------------
# algorithmic bytes (per launch) of the two kernels
# ---------------------------------------------------------------------------
def algorithmic_bytes(wl, io_bytes):
    n, B, Hq, Hkv, d, F = wl.n_req, wl.B, wl.Hq, wl.Hkv, wl.d, wl.F
    q = n * B * Hq * d * io_bytes
    kv = n * B * Hkv * d * io_bytes
    state = n * Hkv * (2 * F * d + 2 * F) * 4
    w = Hkv * d * F * io_bytes
    attn = q + q + 2 * kv + state + w + Hq * 4 + n * 8          # Q, O, K, V, (S, z), W, alpha, ptrs
    commit = 2 * kv + 2 * state + w + n * 8                      # K, V, read+write (S, z), W, ptrs
    fused = q + q + 2 * kv + 2 * state + w + Hq * 4 + n * 8     # one pass: state read once, written once
    return {"attn": attn, "commit": commit, "fused": fused, "q": q, "kv": kv, "state": state}


# ---------------------------------------------------------------------------
# CPU oracle baseline
# ---------------------------------------------------------------------------
def oracle_sample_step(wl, orc, n_sample, tag, W64, alpha64):
    """One oracle step (block attention + commit) on n_sample requests."""
    import torch
    from paper_2608_06628_gb300 import workloads as wk
    Q, K, V = wk.block_qkv(wl, tag, "cpu", n_req=n_sample)
    Q64, K64, V64 = (t.to(torch.float64).numpy() for t in (Q, K, V))
    S, z = orc.empty_state(n_sample, wl.Hkv, wl.d, wl.F)
    t0 = time.perf_counter()
    orc.block_attn(Q64, K64, V64, W64, alpha64, S, z)
    orc.commit(K64, V64, W64, S, z)
    return time.perf_counter() - t0


def cpu_baseline(wl, budget_s=12.0):
    """Time the oracle as it stands on the host cores: whole-batch-shaped steps
    of the workload (n_sample requests each), repeated for about budget_s."""
    import oracle
    from paper_2608_06628_gb300 import workloads as wk
    orc = oracle.load()
    cores = oracle.default_threads()
    W, alpha = wk.params(wl)
    W64 = W.double().numpy()
    alpha64 = alpha.double().numpy()
    n_sample = min(wl.n_req, 16)
    t_one = oracle_sample_step(wl, orc, n_sample, "cpu-probe", W64, alpha64)
    reps = max(1, min(10000, int(budget_s / max(t_one, 1e-6))))
    tot = 0.0
    for i in range(reps):
        tot += oracle_sample_step(wl, orc, n_sample, ("cpu", i), W64, alpha64)
    tokens = reps * n_sample * wl.B
    return {"value": tokens / tot, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{reps} steps x {n_sample} of {wl.n_req} requests (block attention + commit, "
                      f"fp64 C oracle, {cores} threads), {tot:.1f} s"}


def small_config_context(dev, warmup=5, iters=20):
    """Context for the two small configurations (not part of the value): the
    per-call device time of the call the tests make on them, replayed from a CUDA
    graph and launched directly (median of iters after warmup); the oracle's
    one-thread time for the same call is in the CPU-baseline leg.  c1 (fp32, one
    request) is latency-bound and uses one buffer set; c2 rotates enough sets that
    each call misses L2."""
    import torch
    from paper_2608_06628_gb300 import hybrid as H
    from paper_2608_06628_gb300 import workloads as wk
    from paper_2608_06628_gb300.state_pool import StatePool
    out = {}
    for wl, fused in ((wk.C1, False), (wk.C2, True)):
        cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
        W, alpha = wk.params(wl, device=dev)
        io_bytes = 2 if wl.io_dtype == torch.bfloat16 else 4
        ab = algorithmic_bytes(wl, io_bytes)
        l2 = torch.cuda.get_device_properties(dev).L2_cache_size
        per_set = ab["q"] * 2 + ab["kv"] * 2 + ab["state"]
        n_sets = 1 if not fused else max(2, math.ceil(4 * l2 / per_set) + 1)
        plen = wk.prefix_lengths(wl)
        pool0 = StatePool(cfg, wl.n_req, dev)
        H.hybrid_state_init(cfg, pool0.all_ptrs(), wl.n_req)
        for b in range(int(plen.max()) // wl.B):
            reqs = np.nonzero(plen > b * wl.B)[0]
            K, V = wk.prefix_kv(wl, b, dev, n_req=len(reqs))
            H.hybrid_commit_block(cfg, K, V, wl.B, W, pool0.ptr_array(reqs.tolist()), len(reqs))
        H.hybrid_check()
        sets = []
        for i in range(n_sets):
            pool = pool0 if i == 0 else StatePool(cfg, wl.n_req, dev)
            if i:
                pool.slab.copy_(pool0.slab)
            Q, K, V = wk.block_qkv(wl, ("ctx", i), dev)
            sets.append(dict(pool=pool, ptrs=pool.all_ptrs(), Q=Q, K=K, V=V, O=torch.empty_like(Q)))
        fn = H.hybrid_block_attn_commit if fused else H.hybrid_block_attn
        stream = torch.cuda.current_stream(dev)

        def call(s, st):
            fn(cfg, s["Q"], s["K"], s["V"], W, alpha, s["ptrs"], wl.n_req, s["O"], st, check=False)

        for i in range(warmup):
            call(sets[i % n_sets], stream.cuda_stream)
        H.hybrid_check()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(iters)]
        for i in range(iters):
            evs[i][0].record(stream)
            call(sets[i % n_sets], stream.cuda_stream)
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        direct = sorted(a.elapsed_time(b) for a, b in evs)[iters // 2]
        side = torch.cuda.Stream(dev)
        side.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            for i in range(iters):
                call(sets[i % n_sets], side.cuda_stream)
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        a_, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a_.record(stream)
        g.replay()
        b_.record(stream)
        torch.cuda.synchronize()
        graph_ms = a_.elapsed_time(b_) / iters
        status = H.hybrid_check(check=False)
        if status != H.HYBRID_OK:
            raise SystemExit(f"device error in the small-config context: {H.hybrid_status_str(status)}")
        nbytes = ab["fused"] if fused else ab["attn"]
        out[wl.name] = {"call": fn.__name__, "graph_us": graph_ms * 1e3, "direct_us_median": direct * 1e3,
                        "algorithmic_bytes": nbytes, "buffer_sets": n_sets,
                        "tokens_per_s_graph": wl.n_req * wl.B / (graph_ms * 1e-3)}
    return out


def large_config_context(dev, warmup=3, iters=15, n_req=None):
    """Context for the two other large configurations (not part of the value):
    the per-call device time of the step (hybrid_block_attn) and of the block
    commit (hybrid_commit_block, B tokens), replayed from a CUDA graph of iters
    calls over the rotating buffer sets (graph_us, the figure the fraction of HBM
    is taken from) and launched directly (direct_us_median, which for a call of a
    few tens of microseconds also holds the host's launch latency).  c4 is one
    layer of the decode loop (32 requests, MHA);
    its state fits in L2, so it rotates enough buffer sets that each call misses
    L2.  c5 (256 requests, F = 256) holds a 1.08 GB state and uses one set.  The
    kernels' cost does not depend on the state's values: states start empty.
    n_req, if given, replaces both configurations' request count (a smaller case
    of the same kernels, e.g. for a profiler capture)."""
    import torch
    from paper_2608_06628_gb300 import hybrid as H
    from paper_2608_06628_gb300 import workloads as wk
    from paper_2608_06628_gb300.state_pool import StatePool
    peaks, _ = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    out = {}
    for wl in (wk.C4, wk.C5):
        if n_req is not None:
            wl = dataclasses.replace(wl, n_req=n_req)
        cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
        W, alpha = wk.params(wl, device=dev)
        ab = algorithmic_bytes(wl, 2 if wl.io_dtype == torch.bfloat16 else 4)
        l2 = torch.cuda.get_device_properties(dev).L2_cache_size
        per_set = ab["q"] * 2 + ab["kv"] * 2 + ab["state"]
        n_sets = 1 if per_set > 4 * l2 else math.ceil(4 * l2 / per_set) + 1
        sets = []
        for i in range(n_sets):
            pool = StatePool(cfg, wl.n_req, dev)
            ptrs = pool.all_ptrs()
            H.hybrid_state_init(cfg, ptrs, wl.n_req)
            Q, K, V = wk.block_qkv(wl, ("large", i), dev)
            sets.append(dict(pool=pool, ptrs=ptrs, Q=Q, K=K, V=V, O=torch.empty_like(Q)))
        stream = torch.cuda.current_stream(dev)
        calls = {
            "step": lambda s, st: H.hybrid_block_attn(cfg, s["Q"], s["K"], s["V"], W, alpha, s["ptrs"], wl.n_req,
                                                      s["O"], st.cuda_stream, check=False),
            "commit": lambda s, st: H.hybrid_commit_block(cfg, s["K"], s["V"], wl.B, W, s["ptrs"], wl.n_req,
                                                          st.cuda_stream, check=False),
        }
        res = {"buffer_sets": n_sets}
        side = torch.cuda.Stream(dev)
        for name, fn in calls.items():
            for i in range(warmup):
                fn(sets[i % n_sets], stream)
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(iters)]
            for i, (a_, b_) in enumerate(evs):
                a_.record(stream)
                fn(sets[i % n_sets], stream)
                b_.record(stream)
            torch.cuda.synchronize()
            direct = sorted(a_.elapsed_time(b_) for a_, b_ in evs)[iters // 2] * 1e3
            side.wait_stream(stream)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side):
                for i in range(iters):
                    fn(sets[i % n_sets], side)
            torch.cuda.synchronize()
            g.replay()
            torch.cuda.synchronize()
            a_, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a_.record(stream)
            g.replay()
            b_.record(stream)
            torch.cuda.synchronize()
            us = a_.elapsed_time(b_) * 1e3 / iters
            del g
            nbytes = ab["attn"] if name == "step" else ab["commit"]
            res[name] = {"graph_us": us, "direct_us_median": direct, "algorithmic_bytes": nbytes,
                         "GBps": nbytes / us / 1e3, "frac_of_measured_hbm": nbytes / us / 1e3 / hbm}
        status = H.hybrid_check(check=False)
        if status != H.HYBRID_OK:
            raise SystemExit(f"device error in the large-config context: {H.hybrid_status_str(status)}")
        out[wl.name] = res
        del sets
        torch.cuda.empty_cache()
    return out


def small_config_oracle():
    """The oracle's one-thread time for the call small_config_context times on
    c1 and c2 (its cost does not depend on the state's values: empty states)."""
    import torch
    import oracle
    from paper_2608_06628_gb300 import workloads as wk
    orc = oracle.load()
    out = {}
    for wl, fused in ((wk.C1, False), (wk.C2, True)):
        Wc, alc = wk.params(wl)
        W64, al64 = Wc.double().numpy(), alc.double().numpy()
        Q, K, V = wk.block_qkv(wl, "ctx-oracle", "cpu")
        Q64, K64, V64 = (t.to(torch.float64).numpy() for t in (Q, K, V))
        S, z = orc.empty_state(wl.n_req, wl.Hkv, wl.d, wl.F)
        t0 = time.perf_counter()
        orc.block_attn(Q64, K64, V64, W64, al64, S, z, n_threads=1)
        if fused:
            orc.commit(K64, V64, W64, S, z, n_threads=1)
        out[wl.name] = {"oracle_1thread_us": (time.perf_counter() - t0) * 1e6}
    return out


def train_flops(wl):
    """Dense-contraction flops of one training forward and backward (Stage 1) on
    the workload, per (sequence, state head, block) unit times the units:
    forward  Q W, Q K^T, P V, phi(Q) [S | z], K W, phi(K)^T [V | 1];
    backward Q W, Q K^T, dO V^T, S dN, phi(Q)^T [dN | dD], K W, R v, and
    dW = sum x du^T over the G B query rows and B key rows."""
    G, B, d, F = wl.Hq // wl.Hkv, wl.B, wl.d, wl.F
    rq = G * B
    fwd = rq * 2 * d * F + 2 * rq * B * d * 2 + rq * 2 * F * (d + 1) * 2 + B * 2 * d * F + B * 2 * F * (d + 1) * 2
    bwd = (rq * 2 * d * F + 2 * rq * B * d * 2 + rq * 2 * F * d * 2 + rq * 2 * F * (d + 1) * 2
           + B * 2 * d * F + B * 2 * F * d * 2 + (rq + B) * d * F * 2)
    units = wl.n_req * wl.Hkv * (wl.seq_len // wl.B)
    return fwd * units, bwd * units


def train_context(dev, warmup=2, iters=5):
    """Context (not part of the value): the training form of Stage 1 attention
    transfer on the 8 x 2048-token batch (hybrid_train_forward, then
    hybrid_train_backward), median device time of iters pairs after warmup."""
    import torch
    from paper_2608_06628_gb300 import hybrid as H
    from paper_2608_06628_gb300 import workloads as wk
    wl = wk.T1
    Q, K, V, dO = wk.train_batch(wl, device=dev)
    W, alpha = wk.params(wl, 0, dev)
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    n, L = wl.n_req, wl.seq_len
    nb = H.hybrid_train_workspace_bytes(cfg, n, L)
    ws = torch.empty(nb + 1024, dtype=torch.uint8, device=dev)
    ptr = (ws.data_ptr() + 1023) & ~1023
    O = torch.empty_like(Q)
    dW = torch.empty(W.shape, dtype=torch.float32, device=dev)
    da = torch.empty(wl.Hq, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    st = stream.cuda_stream

    def fwd():
        H.hybrid_train_forward(cfg, Q, K, V, W, alpha, n, L, O, ptr, nb, st, check=False)

    def bwd():
        H.hybrid_train_backward(cfg, Q, K, V, W, alpha, dO, n, L, ptr, nb, dW, da, st, check=False)

    for _ in range(warmup):
        fwd()
        bwd()
    H.hybrid_check()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(iters)]
    for e in ev:
        e[0].record(stream)
        fwd()
        e[1].record(stream)
        bwd()
        e[2].record(stream)
    torch.cuda.synchronize()
    status = H.hybrid_check(check=False)
    if status != H.HYBRID_OK:
        raise SystemExit(f"device error in the training context: {H.hybrid_status_str(status)}")
    tf = sorted(e[0].elapsed_time(e[1]) for e in ev)[iters // 2] * 1e-3
    tb = sorted(e[1].elapsed_time(e[2]) for e in ev)[iters // 2] * 1e-3
    ff, fb = train_flops(wl)
    peaks, _ = measured_peaks()
    bf16 = float(peaks.get("bf16_tflops", 1900.0))
    del ws
    return {"workload": wl.name, "calls": "hybrid_train_forward + hybrid_train_backward",
            "tokens": n * L, "fwd_us": tf * 1e6, "bwd_us": tb * 1e6,
            "tokens_per_s": n * L / (tf + tb), "workspace_bytes": nb,
            "fwd_TFLOPs": ff / tf / 1e12, "bwd_TFLOPs": fb / tb / 1e12,
            "frac_bf16_peak": (ff + fb) / (tf + tb) / 1e12 / bf16}


def train_oracle_sample(seq_len=1024):
    """The oracle's training forward and backward on one sequence of seq_len
    tokens of the training batch's shape (all host threads)."""
    import oracle
    from paper_2608_06628_gb300 import workloads as wk
    orc = oracle.load()
    wl = wk.T1
    Q, K, V, dO = wk.train_batch(wl, tag="oracle", n_seq=1, seq_len=seq_len)
    W, alpha = wk.params(wl)
    args = [t.double().numpy() for t in (Q, K, V, W, alpha)]
    t0 = time.perf_counter()
    orc.train_forward(*args, wl.B)
    orc.train_backward(*args, dO.double().numpy(), wl.B)
    t = time.perf_counter() - t0
    return {"tokens_per_s": seq_len / t, "sample": f"1 sequence x {seq_len} tokens of {wl.name}, "
            f"forward + backward, {oracle.default_threads()} threads (units: {wl.Hkv} state heads)", "s": t}


def prefill_context(dev, wl, T=4096, warmup=2, iters=5):
    """Context (not part of the value): one prompt prefill of T tokens into every
    request's state at the workload's shape (hybrid_commit_block with n_tok = T),
    median device time of iters calls after warmup.  Traffic is K + V + the state
    read and written once; flops are U_k^T = W^T K^T (2FdT per unit) and
    dS^T = V^T phi(K)^T (4FdT per unit)."""
    import torch
    from paper_2608_06628_gb300 import hybrid as H
    from paper_2608_06628_gb300 import workloads as wk
    from paper_2608_06628_gb300.state_pool import StatePool
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    W, _ = wk.params(wl, device=dev)
    pool = StatePool(cfg, wl.n_req, dev)
    ptrs = pool.all_ptrs()
    H.hybrid_state_init(cfg, ptrs, wl.n_req)
    g = torch.Generator(device=dev).manual_seed(4096)
    shape = (wl.n_req, T, wl.Hkv, wl.d)
    K = torch.randn(shape, generator=g, device=dev, dtype=torch.float32).to(wl.io_dtype)
    V = torch.randn(shape, generator=g, device=dev, dtype=torch.float32).to(wl.io_dtype)
    stream = torch.cuda.current_stream(dev)
    for _ in range(warmup):
        H.hybrid_commit_block(cfg, K, V, T, W, ptrs, wl.n_req, stream.cuda_stream, check=False)
    H.hybrid_check()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(iters)]
    for a_, b_ in evs:
        a_.record(stream)
        H.hybrid_commit_block(cfg, K, V, T, W, ptrs, wl.n_req, stream.cuda_stream, check=False)
        b_.record(stream)
    torch.cuda.synchronize()
    status = H.hybrid_check(check=False)
    if status != H.HYBRID_OK:
        raise SystemExit(f"device error in the prefill context: {H.hybrid_status_str(status)}")
    ms = sorted(a_.elapsed_time(b_) for a_, b_ in evs)[iters // 2]
    io = K.element_size()
    units = wl.n_req * wl.Hkv
    nbytes = 2 * K.numel() * io + 2 * units * (2 * wl.F * wl.d + 2 * wl.F) * 4 + wl.Hkv * wl.d * wl.F * io
    flops = 6.0 * wl.F * wl.d * T * units
    peaks, _ = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    bf16 = float(peaks.get("bf16_tflops", 1900.0))
    del K, V
    out = {"call": "hybrid_commit_block", "tokens_per_request": T, "us": ms * 1e3,
           "algorithmic_bytes": nbytes, "GBps": nbytes / (ms * 1e-3) / 1e9,
           "frac_hbm": nbytes / (ms * 1e-3) / 1e9 / hbm,
           "TFLOPs": flops / (ms * 1e-3) / 1e12, "frac_bf16_peak": flops / (ms * 1e-3) / 1e12 / bf16,
           "prompt_tokens_per_s": wl.n_req * T / (ms * 1e-3)}
    # the same requests with ragged prompt lengths, seeded U{1, ..., 2T - 1}, packed
    # token-major (hybrid_commit_ragged); same bytes per token and per state
    lens = np.random.default_rng(4097).integers(1, 2 * T, size=wl.n_req)
    offs = np.concatenate([[0], np.cumsum(lens)]).tolist()
    total = int(offs[-1])
    Kr = torch.randn((total, wl.Hkv, wl.d), generator=g, device=dev, dtype=torch.float32).to(wl.io_dtype)
    Vr = torch.randn((total, wl.Hkv, wl.d), generator=g, device=dev, dtype=torch.float32).to(wl.io_dtype)
    for _ in range(warmup):
        H.hybrid_commit_ragged(cfg, Kr, Vr, offs, W, ptrs, wl.n_req, stream.cuda_stream, check=False)
    for a_, b_ in evs:
        a_.record(stream)
        H.hybrid_commit_ragged(cfg, Kr, Vr, offs, W, ptrs, wl.n_req, stream.cuda_stream, check=False)
        b_.record(stream)
    torch.cuda.synchronize()
    status = H.hybrid_check(check=False)
    if status != H.HYBRID_OK:
        raise SystemExit(f"device error in the ragged prefill context: {H.hybrid_status_str(status)}")
    ms_r = sorted(a_.elapsed_time(b_) for a_, b_ in evs)[iters // 2]
    nbytes_r = 2 * Kr.numel() * io + 2 * units * (2 * wl.F * wl.d + 2 * wl.F) * 4 + wl.Hkv * wl.d * wl.F * io
    out["ragged"] = {"call": "hybrid_commit_ragged", "tokens_per_request": f"U{{1..{2 * T - 1}}} (seeded)",
                     "tokens": total, "us": ms_r * 1e3, "algorithmic_bytes": nbytes_r,
                     "GBps": nbytes_r / (ms_r * 1e-3) / 1e9, "frac_hbm": nbytes_r / (ms_r * 1e-3) / 1e9 / hbm,
                     "prompt_tokens_per_s": total / (ms_r * 1e-3)}
    del Kr, Vr
    return out


# ---------------------------------------------------------------------------
# reference arm: the oracle, timed step by step
# ---------------------------------------------------------------------------
def run_reference(args, wl):
    ws, rank, _ = dist_info()
    if rank != 0:
        return 0
    import oracle
    from paper_2608_06628_gb300 import workloads as wk
    orc = oracle.load()
    cores = oracle.default_threads()
    W, alpha = wk.params(wl)
    W64, alpha64 = W.double().numpy(), alpha.double().numpy()
    t_probe = oracle_sample_step(wl, orc, 1, "ref-probe", W64, alpha64)
    total_budget = 120.0
    n_sample = int(max(1, min(wl.n_req, total_budget / max(1, args.steps + args.warmup) / max(t_probe, 1e-6))))
    for i in range(args.warmup):
        oracle_sample_step(wl, orc, n_sample, ("ref-warm", i), W64, alpha64)
    tot = 0.0
    for i in range(args.steps):
        tot += oracle_sample_step(wl, orc, n_sample, ("ref", i), W64, alpha64)
    value = args.steps * n_sample * wl.B / tot
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(wl, None),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": f"each step: {n_sample} of {wl.n_req} requests, block attention + commit, "
                                   f"fp64 C oracle on {cores} host threads"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def workload_config(wl, l2_note):
    cfg = {"workload": wl.name, "n_req": wl.n_req, "block_size": wl.B, "n_q_heads": wl.Hq,
           "n_kv_heads": wl.Hkv, "head_dim": wl.d, "feat_dim": wl.F,
           "prefix": (f"ragged U{{{wl.prefix_min}..{wl.prefix_max}}} step {wl.B}"
                      if wl.prefix_min != wl.prefix_max else f"{wl.prefix_min}"),
           "k_scale": wl.k_scale, "io_dtype": str(wl.io_dtype).replace("torch.", ""),
           "state_dtype": "float32",
           "step": "hybrid_block_attn_commit: one denoising step and the commit of its block, one launch"}
    if l2_note:
        cfg["l2"] = l2_note
    return cfg


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
def run_hybrid(args, wl):
    import torch
    ws, rank, local = dist_info()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device(f"cuda:{local}" if ws > 1 else "cuda:0")
    torch.cuda.set_device(dev)

    from paper_2608_06628_gb300 import build
    build.build()
    from paper_2608_06628_gb300 import hybrid as H
    from paper_2608_06628_gb300 import workloads as wk
    from paper_2608_06628_gb300.state_pool import StatePool

    # each rank draws its own independent batch (weak scaling)
    wl = rank_workload(wl, rank)
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    W, alpha = wk.params(wl, device=dev)
    io_bytes = 2 if wl.io_dtype == torch.bfloat16 else 4
    ab = algorithmic_bytes(wl, io_bytes)
    per_set = ab["q"] * 2 + ab["kv"] * 2 + ab["state"]
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    n_sets = max(2, math.ceil(4 * l2 / per_set) + 1)

    # states of set 0: ragged prefixes built by block commits
    plen = wk.prefix_lengths(wl)
    pool0 = StatePool(cfg, wl.n_req, dev)
    H.hybrid_state_init(cfg, pool0.all_ptrs(), wl.n_req)
    for b in range(int(plen.max()) // wl.B):
        reqs = np.nonzero(plen > b * wl.B)[0]
        K, V = wk.prefix_kv(wl, b, dev, n_req=len(reqs))
        H.hybrid_commit_block(cfg, K, V, wl.B, W, pool0.ptr_array(reqs.tolist()), len(reqs))
    H.hybrid_check()
    sets = []
    for i in range(n_sets):
        pool = pool0 if i == 0 else StatePool(cfg, wl.n_req, dev)
        if i:
            pool.slab.copy_(pool0.slab)
        Q, K, V = wk.block_qkv(wl, ("bench", i), dev)
        sets.append(dict(pool=pool, ptrs=pool.all_ptrs(), Q=Q, K=K, V=V, O=torch.empty_like(Q)))
    torch.cuda.synchronize()

    stream = torch.cuda.current_stream(dev)
    sh = stream.cuda_stream

    def step(s):
        H.hybrid_block_attn_commit(cfg, s["Q"], s["K"], s["V"], W, alpha, s["ptrs"], wl.n_req, s["O"], sh,
                                   check=False)

    def timed(fn, n, first=0):
        """n calls of fn(set) with CUDA events around each, on the launching stream."""
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        for i in range(n):
            s = sets[(first + i) % n_sets]
            evs[i][0].record(stream)
            fn(s)
            evs[i][1].record(stream)
        return evs

    clocks = ClockSampler(bus_id_of(torch, dev))
    clocks.start()
    time.sleep(0.3)
    for i in range(args.warmup):
        step(sets[i % n_sets])
    H.hybrid_check(sh)

    # The timed steps are replayed from CUDA graphs (how a serving loop issues
    # its decode steps), so per-call host overhead does not starve the GPU:
    # one graph holds one step per buffer set, a second one the remainder.
    K_ = args.steps
    side = torch.cuda.Stream(dev)
    side.wait_stream(stream)

    def capture(n_steps):
        if n_steps == 0:
            return None
        g_ = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_, stream=side):
            for i in range(n_steps):
                s = sets[i % n_sets]
                H.hybrid_block_attn_commit(cfg, s["Q"], s["K"], s["V"], W, alpha, s["ptrs"], wl.n_req, s["O"],
                                           side.cuda_stream, check=False)
        return g_

    g_full, g_rem = capture(n_sets), capture(K_ % n_sets)
    torch.cuda.synchronize()
    for _ in range(2):
        g_full.replay()
    torch.cuda.synchronize()
    barrier(ws)
    torch.cuda.synchronize()
    t_wall0 = time.time()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(K_ // n_sets):
        g_full.replay()
    if g_rem is not None:
        g_rem.replay()
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier(ws)
    t_wall1 = time.time()
    status = H.hybrid_check(sh, check=False)
    if status != H.HYBRID_OK:
        raise SystemExit(f"device error during the timed region: {H.hybrid_status_str(status)}")
    elapsed_ms = ev0.elapsed_time(ev1)
    fused_ms = elapsed_ms / K_
    elapsed_ms = max_over_ranks(elapsed_ms, ws, dev)

    # the same steps launched one call at a time from Python (context)
    evs = timed(step, min(K_, 500))
    torch.cuda.synchronize()
    direct_ms = (evs[0][0].elapsed_time(evs[-1][1])) / len(evs)

    # context (not part of the value): the step split into its two separate
    # launches, each replayed from a CUDA graph like the timed steps
    def attn_only(s, st):
        H.hybrid_block_attn(cfg, s["Q"], s["K"], s["V"], W, alpha, s["ptrs"], wl.n_req, s["O"], st, check=False)

    def commit_only(s, st):
        H.hybrid_commit_block(cfg, s["K"], s["V"], wl.B, W, s["ptrs"], wl.n_req, st, check=False)

    def graph_ms(fn, n_rep=max(1, min(K_, 200) // n_sets)):
        g_ = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_, stream=side):
            for i in range(n_sets):
                fn(sets[i], side.cuda_stream)
        torch.cuda.synchronize()
        g_.replay()
        torch.cuda.synchronize()
        a_, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a_.record(stream)
        for _ in range(n_rep):
            g_.replay()
        b_.record(stream)
        torch.cuda.synchronize()
        return a_.elapsed_time(b_) / (n_rep * n_sets)

    attn_ms = graph_ms(attn_only)
    commit_ms = graph_ms(commit_only)

    # end to end through the public API: every step copies its inputs in from
    # pinned host memory and reads its output back.  As a serving loop would, the
    # steps are pipelined over three streams (copy in, compute, copy out) so the
    # next step's inputs and the previous step's output move while a step runs;
    # the sequence is captured once in a CUDA graph and replayed.
    # a step's Q, K and V sit back to back in one pinned host buffer and one
    # device buffer, so each step's input is one copy
    q0, k0, v0 = sets[0]["Q"], sets[0]["K"], sets[0]["V"]
    nq, nk = q0.numel(), k0.numel()
    hQKV = torch.cat([q0.reshape(-1), k0.reshape(-1), v0.reshape(-1)]).cpu().pin_memory()
    hO = [torch.empty(q0.shape, dtype=q0.dtype).pin_memory() for _ in range(2)]

    def split_qkv(buf):
        return dict(Q=buf[:nq].view(q0.shape), K=buf[nq:nq + nk].view(k0.shape), V=buf[nq + nk:].view(v0.shape))

    e2e_bufs = [torch.empty_like(hQKV, device=dev) for _ in sets]
    e2e_sets = [dict(s, **split_qkv(b)) for s, b in zip(sets, e2e_bufs)]
    # a replay starts with the pipeline empty and ends by draining it (its first copy in and
    # its last copy out overlap nothing), so one graph holds many steps
    n_e2e = 8 * n_sets
    cin, cout = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    g_e2e = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_e2e, stream=side):
        cin.wait_stream(side)
        cout.wait_stream(side)
        ev_in = [torch.cuda.Event() for _ in range(n_e2e)]
        ev_done = [torch.cuda.Event() for _ in range(n_e2e)]
        ev_out = [torch.cuda.Event() for _ in range(n_e2e)]
        for i in range(n_e2e):
            s = e2e_sets[i % n_sets]
            if i >= n_sets:
                cin.wait_event(ev_out[i - n_sets])   # the set's previous step has finished with it
            with torch.cuda.stream(cin):
                e2e_bufs[i % n_sets].copy_(hQKV, non_blocking=True)
            ev_in[i].record(cin)
            side.wait_event(ev_in[i])
            H.hybrid_block_attn_commit(cfg, s["Q"], s["K"], s["V"], W, alpha, s["ptrs"], wl.n_req, s["O"],
                                       side.cuda_stream, check=False)
            ev_done[i].record(side)
            cout.wait_event(ev_done[i])
            with torch.cuda.stream(cout):
                hO[i % 2].copy_(s["O"], non_blocking=True)
            ev_out[i].record(cout)
        side.wait_stream(cin)
        side.wait_stream(cout)
    torch.cuda.synchronize()
    reps = max(1, K_ // n_e2e)
    for _ in range(max(1, args.warmup // n_e2e)):
        g_e2e.replay()
    barrier(ws)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        g_e2e.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(ws)
    clocks.stop()
    status = H.hybrid_check(sh, check=False)
    if status != H.HYBRID_OK:
        raise SystemExit(f"device error in the end-to-end steps: {H.hybrid_status_str(status)}")
    e2e_steps = reps * n_e2e
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), ws, dev)

    if rank != 0:
        return 0
    tokens = wl.n_req * wl.B * K_ * ws
    value = tokens / (elapsed_ms * 1e-3)
    peaks, peak_kind = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    kname = "hybrid_block_attn_commit"
    achieved = ab["fused"] / (fused_ms * 1e-3) / 1e9

    def kinfo(nbytes, ms):
        return {"us_per_launch": ms * 1e3, "bytes": nbytes, "GBps": nbytes / (ms * 1e-3) / 1e9,
                "frac_hbm": nbytes / (ms * 1e-3) / 1e9 / hbm}

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": ws, "steps": K_,
        "warmup": args.warmup, "ms_per_step": elapsed_ms / K_, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if wl.io_dtype == torch.bfloat16 else "f32",
        "data": "synthetic (seeded N(0,1) activations, random-init W ~ N(0,1/d), alpha ~ U(0,1))",
        "config": workload_config(wl, f"{n_sets} rotating buffer sets of {per_set / 1e6:.1f} MB "
                                      f"(> 4x the {l2 / 1e6:.0f} MB L2)"),
        "roofline": {"bound": "hbm", "kernel": kname, "achieved": achieved, "peak": hbm,
                     "peak_kind": f"{peak_kind} (HBM copy, MEASURED_PEAKS hbm_gbs)" if peak_kind == "measured"
                     else "fallback 6.8 TB/s", "unit": "GB/s", "frac": achieved / hbm,
                     "traffic": recorded_traffic(kname, wl.name),
                     "algorithmic_bytes_per_launch": ab["fused"]},
        # the step alone (the attention-only launches of the denoising steps that do
        # not commit), timed the same way in its own graph of the rotating sets
        "roofline_step": {"bound": "hbm", "kernel": "hybrid_block_attn",
                          "achieved": ab["attn"] / (attn_ms * 1e-3) / 1e9, "peak": hbm,
                          "unit": "GB/s", "frac": ab["attn"] / (attn_ms * 1e-3) / 1e9 / hbm,
                          "traffic": recorded_traffic("hybrid_block_attn", wl.name),
                          "algorithmic_bytes_per_launch": ab["attn"], "us_per_launch": attn_ms * 1e3},
        "timing": "K steps replayed from CUDA graphs (one launch per step); "
                  f"direct Python launches: {direct_ms * 1e3:.1f} us/step",
        "kernels": {
            "hybrid_block_attn_commit (timed step)": kinfo(ab["fused"], fused_ms),
            "hybrid_block_attn (context)": kinfo(ab["attn"], attn_ms),
            "hybrid_commit_block (context)": kinfo(ab["commit"], commit_ms),
        },
        "e2e": {"value": wl.n_req * wl.B * e2e_steps * ws / (e2e_ms * 1e-3), "unit": "tokens/s",
                "steps": e2e_steps, "pipelined": "copy-in / step / copy-out on three streams, graph-replayed",
                "h2d_bytes_per_step": int(hQKV.numel() * hQKV.element_size()),
                "d2h_bytes_per_step": int(hO[0].numel() * hO[0].element_size())},
        "gpu_launches": K_,
        "clocks": clocks.summary(t_wall0, t_wall1),
    }
    if not args.no_small_configs and ws == 1:
        line["small_configs"] = small_config_context(dev)
        line["large_configs"] = large_config_context(dev)
        line["prefill_context"] = prefill_context(dev, wl)
        line["train_context"] = train_context(dev)
    if not args.no_cpu_baseline and ws == 1:
        line["cpu_baseline"] = cpu_baseline(wl)
        if not args.no_small_configs:
            line["cpu_baseline"]["contexts"] = {"small_configs": small_config_oracle(),
                                                "train": train_oracle_sample()}
    print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", choices=("hybrid", "reference"), default="hybrid")
    ap.add_argument("--config", default="c3_bf16_b64_gqa_ragged")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-small-configs", action="store_true",
                    help="skip the context timings (c1/c2, c4/c5, prefill, training form)")
    ap.add_argument("--n-req", type=int, default=None,
                    help="with --context large: requests per configuration (default: the configs' own)")
    ap.add_argument("--context", choices=("train", "prefill", "small", "large"),
                    help="time only this context on cuda:0 and print its JSON object")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    from paper_2608_06628_gb300 import workloads as wk
    wl = wk.CONFIGS[args.config]
    if args.context:
        import torch
        from paper_2608_06628_gb300 import build
        build.build()
        dev = torch.device("cuda", 0)
        torch.cuda.set_device(dev)
        fn = {"train": lambda: train_context(dev), "prefill": lambda: prefill_context(dev, wl),
              "small": lambda: small_config_context(dev), "large": lambda: large_config_context(dev, n_req=args.n_req)}[args.context]
        print(json.dumps({"context": args.context, **fn()}), flush=True)
        return 0
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_hybrid(args, wl)


if __name__ == "__main__":
    sys.exit(main())
