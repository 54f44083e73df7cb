#!/usr/bin/env python3
"""Retrieve throughput of the MemAttention memory hot path on GB300.

One step = one retrieval pass (score -> two relation hops -> top-k -> page
resolve) of a batch of 256 bf16 queries against the N=1,048,576-chunk,
d=1024 synthetic store (gmm1m recipe: 4096-component Zipf(1.1) mixture,
32-neighbour power-law relation graph, 64 chunks per page, clustered
placement), k=32, alpha=0.5.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

N>1 runs under torch.distributed.run: every rank runs an independent
replica of the store on its own GPU (queries are independent; there is no
collective on the data path); timing is the max over ranks and `value`
counts the queries of all ranks.  `--impl reference` times the CPU oracle
(plain single-threaded fp64 C) on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "retrieve queries/sec at N=1M chunks, d=1024, B=256; % of roofline"
WORKLOAD = ("gmm1m: N=1048576 chunks, d=1024 bf16, 4096-component Zipf(1.1) mixture, 32-neighbour "
            "power-law relation graph (nnz 33554432), B=256 queries, hops=2, alpha=0.5, k=32, "
            "64 chunks/page, clustered placement")
SCOPED_METRIC = ("namespace-scoped retrieve queries/sec at N=1M chunks, d=1024, B=256, "
                 "SortByTime")
SCOPED_WORKLOAD = ("gmm1m store with 64 namespaces (chunk tag = mixture component mod 64), each "
                   "query scoped to a seeded namespace, hops=2, alpha=0.5, k=32, results in "
                   "chronological (chunk ID) order, clustered placement")
DENSE_METRIC = "Dense-only retrieve queries/sec at N=1M chunks, d=1024, B=256, top-p 5, no hops"
DENSE_WORKLOAD = ("gmm1m store (N=1048576, d=1024 bf16), B=256 queries, k=5, hops=0 "
                  "(embedding similarity only), 64 chunks/page, clustered placement")
MEMORY_METRIC = ("Memory Manager requests/sec (co-retrieval counts, relocation, block compaction) "
                 "at N=1M chunks, batches of 256 top-5 requests")
MEMORY_WORKLOAD = ("gmm1m store (N=1048576, d=1024 bf16, 64 chunks/page) in random placement (the "
                   "append-only log); trace of Dense-only top-5 retrievals, queries = one of 4096 "
                   "anchor chunks drawn with Zipf(1.1) popularity + N(0,(0.05/sqrt d)^2) noise; per "
                   "step relocate(S, tau_assoc=0.7) then compact(theta=0.75, tau_assoc=0.7)")


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops", 1895.6), "measured"
    return 6800.0, 1900.0, "fallback"


def algorithmic_bytes(n, d, b, nnz, hops, k):
    """Bytes a retrieval pass must move at least once (E once, the graph once
    per hop, the fp32 score slab written by the score pass and, per hop, each
    input slab read once and the output written once except the last hop's,
    which feeds the top-k directly), plus queries, page table and outputs."""
    slab = n * b * 4
    graph = (n + 1) * 8 + nnz * 4 + nnz * 4
    passes = 1 + (2 * hops if hops > 0 else 1)          # u write; per hop read in + write/ u read
    return dict(emb=n * d * 2, graph=graph * hops, slab=slab * passes,
                small=b * d * 2 + n * 4 + b * k * 16 + b * 4)


def hop_bytes(n, b, nnz):
    """One propagation hop: graph once + two slab passes (hop 1 reads u and
    writes s1; the last hop reads s^(H-1) and u and writes nothing)."""
    return (n + 1) * 8 + nnz * 8 + 2 * n * b * 4


# DRAM bytes of one full propagation hop on this workload (the first hop:
# hub segments 3.795 GB read + 0.361 GB written, then hub sums + rows kept
# whole 5.948 + 1.060 GB), from an ncu capture of
# `bench.py --steps 2 --warmup 1 --no-cpu-baseline` with the
# dram__bytes_read/write counters.  Set to None when the hop kernels change
# until they are captured again.
HOP_DRAM_BYTES = 11.16e9
# DRAM bytes of the score GEMM (E read once, the u slab written once; 2.148 +
# 1.035 GB) from the same kind of capture, taken on the current epilogue (u's
# row extremes, Z's column sums per warp).  None once that kernel changes.
SCORE_DRAM_BYTES = 3.183e9
# distinct query batches the retrieval steps rotate through
QUERY_POOL = 8
# timed steps of the hop_path record (the hops always run)
HOP_PATH_STEPS = 40


def score_bytes(n, d, b):
    return n * d * 2 + n * b * 4 + b * d * 2


class Clocks:
    """nvidia-smi sampled during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, dev):
        self.dev = dev
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.dev)], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                self.out = ""

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def cpu_baseline(wl, placement, n_queries, rng_seed=0, weights=None, k=None, hops=None,
                 ns_of=None, q_ns=None, sort_by_time=False):
    """The oracle retrieving n_queries of the batch against the full store on
    one host thread (the relation weights, which the GPU store computes at
    append time, are computed once beforehand)."""
    import oracle
    hops = wl.hops if hops is None else hops
    w = (weights if weights is not None else oracle.row_softmax(wl.row_ptr, wl.aff)) if hops else None
    rows = np.random.default_rng(rng_seed).choice(wl.n_queries, size=n_queries, replace=False)
    t0 = time.perf_counter()
    oracle.retrieve(wl.emb, wl.queries[rows], wl.row_ptr if hops else None,
                    wl.col if hops else None, w, tau=wl.tau, alpha=wl.alpha, hops=hops,
                    k=wl.k if k is None else k, page_of=wl.page_of[placement], ns_of=ns_of,
                    q_ns=None if q_ns is None else q_ns[rows], sort_by_time=sort_by_time)
    dt = time.perf_counter() - t0
    return dict(value=n_queries / dt, unit="queries/s", cores=1, kind="oracle",
                sample=f"{n_queries} of the {wl.n_queries} queries against the full store, "
                       f"one thread",
                seconds=dt)


def max_over_ranks(values, device=None):
    """Max of each value over all ranks of the default process group (the
    slowest rank sets the job's time); identity when not distributed."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def job_throughput(units_per_rank, world, ms):
    """Whole-job throughput: the units every rank processed over the max time."""
    return units_per_rank * world / (ms * 1e-3)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    import synth
    wl = synth.workload(2, scale=args.scale, placements=("clustered",))
    w = oracle.row_softmax(wl.row_ptr, wl.aff)
    workload = WORKLOAD if args.scale == 1.0 else f"{WORKLOAD} scaled by {args.scale}"
    per_step = 1
    times = []
    for i in range(args.warmup + args.steps):
        r = cpu_baseline(wl, "clustered", per_step, rng_seed=i, weights=w)
        if i >= args.warmup:
            times.append(r["seconds"])
    tot = sum(times)
    value = per_step * len(times) / tot
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "queries/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * tot / len(times), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload, "sample": f"{per_step} query per step"},
        "cpu_baseline": {"value": value, "unit": "queries/s", "cores": 1, "kind": "oracle",
                         "sample": f"{per_step} query of 256 per step, whole store, one thread"},
        "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_update(args):
    """Relation update: each step appends the 4096 new chunks of the update
    workload again and links them to every prior chunk (cosine GEMM of
    4096 x N_prior x 1024, top-32, reciprocal CSR insert, weights and the
    in-edge transpose rebuilt).  Prior chunks grow by 4096 per step."""
    import torch
    import synth
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_05708_gb300 import MemStore
    wl = synth.workload(3, scale=args.scale)
    n_new = wl.new_emb.shape[0]
    total = args.warmup + args.steps
    store = MemStore.from_arrays(wl.emb, wl.page_of["clustered"], wl.row_ptr, wl.col, wl.aff,
                                 capacity=wl.n + n_new * total, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau, relation_scale=wl.relation_scale)
    new = torch.from_numpy(np.ascontiguousarray(wl.new_emb).view(np.int16)).cuda()
    st = torch.cuda.Stream()
    times, flops = [], []
    store.set_profiling(True)
    with Clocks(0) as clk:
        for i in range(total):
            first = store.append_chunks(new, stream=st)
            torch.cuda.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(st)
            store.update_relations(first, n_new, wl.top_m, True, stream=st)
            e1.record(st)
            torch.cuda.synchronize()
            if i >= args.warmup:
                times.append(e0.elapsed_time(e1))
                flops.append(2.0 * n_new * first * wl.dim)
            elif i == args.warmup - 1:
                store.phase_times()
    phases = store.phase_times()
    hbm, bf16, kind = peaks()
    ms = sum(times) / len(times)
    fl = sum(flops) / len(flops)
    relate_ms = phases["relate"][0] / len(times)
    line = {
        "metric": "relation update ms per 4096 new chunks (N=1M, d=1024, M=32); % of bf16 tensor peak",
        "value": ms, "unit": "ms/update", "higher_is_better": False, "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": f"update: gmm1m store + {n_new} new chunks, top-{wl.top_m}, reciprocal"
                   + ("" if args.scale == 1.0 else f", scaled by {args.scale}")},
        "roofline": {"bound": "tensor", "achieved": fl / (relate_ms * 1e-3) / 1e12, "peak": bf16,
                     "unit": "TFLOP/s", "frac": fl / (relate_ms * 1e-3) / 1e12 / bf16,
                     "traffic": None, "kernel": "relation GEMM + top-M (relate phase)",
                     "peak_kind": kind},
        "phases_ms_per_step": {p: phases[p][0] / len(times)
                               for p in ("relate", "graph", "csr_insert", "transpose", "hub_plan")},
        "tensor_frac_of_whole_update": fl / (ms * 1e-3) / 1e12 / bf16,
        "clocks": clk.summary(),
    }
    print(json.dumps(line), flush=True)
    store.close()
    return 0


def run_delete(args):
    """Chunk deletion: each step deletes 1024 fresh random chunks of the
    gmm1m store (tombstones, edges into and out of them dropped from the CSR
    and the transpose, rows re-softmaxed, hub plan rebuilt).  Bytes moved per
    call: both edge lists read, flagged and compacted once."""
    import torch
    import synth
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_05708_gb300 import MemStore
    wl = synth.workload(2, scale=args.scale)
    store = MemStore.from_arrays(wl.emb, wl.page_of["clustered"], wl.row_ptr, wl.col, wl.aff,
                                 capacity=wl.n, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau)
    total = args.warmup + args.steps
    order = np.random.default_rng(5).permutation(wl.n)[:1024 * total]
    st = torch.cuda.Stream()
    times = []
    with Clocks(0) as clk:
        for i in range(total):
            ids = torch.from_numpy(order[i * 1024:(i + 1) * 1024].astype(np.int64)).cuda()
            torch.cuda.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(st)
            store.delete(ids, stream=st)
            e1.record(st)
            torch.cuda.synchronize()
            if i >= args.warmup:
                times.append(e0.elapsed_time(e1))
    ms = sum(times) / len(times)
    n_rows, nnz = store.size()
    hbm, _, kind = peaks()
    # per call: out CSR (col+aff read, flags, scan, compacted write) and the
    # same for the transpose, plus the row softmax over the CSR
    moved = nnz * (4 + 4 + 8 + 8 + 8 + 4 + 4) * 2 + nnz * 12
    line = {
        "metric": "delete ms per 1024 chunks (N=1M, nnz 33.5M)", "value": ms, "unit": "ms/delete",
        "higher_is_better": False, "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "gmm1m store, 1024 random chunks deleted per step"
                   + ("" if args.scale == 1.0 else f", scaled by {args.scale}")},
        "roofline": {"bound": "hbm", "achieved": moved / (ms * 1e-3) / 1e9, "peak": hbm,
                     "unit": "GB/s", "frac": moved / (ms * 1e-3) / 1e9 / hbm, "traffic": None,
                     "kernel": "whole delete call", "peak_kind": kind},
        "edges_left": nnz,
        "clocks": clk.summary(),
    }
    print(json.dumps(line), flush=True)
    store.close()
    return 0


def _numpy_top5(wl, q_bf16, block=65536):
    """Top-5 chunk IDs by dot product, plain numpy fp32 (input preparation of
    the CPU sample; ties broken arbitrarily, which timing does not mind)."""
    import synth
    q = synth.bf16_to_f32(q_bf16)
    best_v = np.full((q.shape[0], 5), -np.inf, np.float32)
    best_i = np.zeros((q.shape[0], 5), np.int64)
    for r0 in range(0, wl.n, block):
        e = synth.bf16_to_f32(wl.emb[r0:r0 + block])
        d = q @ e.T
        part = np.argpartition(-d, 5, axis=1)[:, :5]
        v = np.take_along_axis(d, part, axis=1)
        cv = np.concatenate([best_v, v], axis=1)
        ci = np.concatenate([best_i, part + r0], axis=1)
        top = np.argpartition(-cv, 5, axis=1)[:, :5]
        best_v = np.take_along_axis(cv, top, axis=1)
        best_i = np.take_along_axis(ci, top, axis=1)
    return best_i


def run_memory(args):
    """The Memory Manager (co-retrieval statistics, relocation of associated
    chunks, block compaction) fed by the retrieval it serves: every step
    takes one batch of 256 Dense-only top-5 request sets of a replayed trace
    and runs relocate + compact on the gmm1m directory.  Reports pages per
    request over the trace before and after, and space / write
    amplification."""
    import torch
    import synth
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_05708_gb300 import MemStore
    wl = synth.workload(2, scale=args.scale)
    B, K, W = 256, args.steps, args.warmup
    T = W + 2 * K
    Q = synth.request_trace(wl, T * B, n_topics=max(64, wl.n // 256))
    cpu = None
    if not args.no_cpu_baseline:
        from oracle.memory_manager import MemoryManager
        n_b = 4
        S_cpu = _numpy_top5(wl, Q[:n_b * B])
        mm = MemoryManager(wl.page_of["random"], wl.chunks_per_page)
        t0 = time.perf_counter()
        for b in range(n_b):
            mm.relocate(S_cpu[b * B:(b + 1) * B], 0.7)
            mm.compact(0.75, 0.7)
        t = time.perf_counter() - t0
        cpu = {"value": n_b * B / t, "unit": "requests/s", "cores": 1, "kind": "oracle",
               "sample": f"first {n_b} batches of 256 requests on the fresh 1M-chunk directory "
                         "(request sets from a numpy fp32 top-5, untimed)"}
    store = MemStore.from_arrays(wl.emb, wl.page_of["random"], wl.row_ptr, wl.col, wl.aff,
                                 capacity=wl.n, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau)
    st = torch.cuda.Stream()
    q_dev = torch.from_numpy(Q.view(np.int16)).cuda()
    S = torch.empty((T, B, 5), dtype=torch.int64, device="cuda")
    sc = torch.empty((B, 5), dtype=torch.float32, device="cuda")
    pg = torch.empty((B, 5), dtype=torch.int32, device="cuda")
    npg = torch.empty((T, B), dtype=torch.int32, device="cuda")

    def replay():
        for b in range(T):
            store.retrieve(q_dev[b * B:(b + 1) * B], 5, wl.alpha, 0, S[b], sc, pg, npg[b],
                           stream=st)
        torch.cuda.synchronize()
        return npg.float().mean().item()

    before = replay()

    def step(b):
        store.relocate(S[b], 0.7, stream=st)
        store.compact_pages(0.75, 0.7, stream=st)

    for b in range(W):
        step(b)
    torch.cuda.synchronize()
    store.set_profiling(True)
    store.phase_times()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    with Clocks(0) as clk:
        ev0.record(st)
        for b in range(W, W + K):
            step(b)
        ev1.record(st)
        torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1) / K
    phases = store.phase_times()
    store.set_profiling(False)
    # end to end: request sets from pinned host memory, page accounting read back
    S_host = S[W + K:].cpu().pin_memory()
    s_dev = torch.empty((B, 5), dtype=torch.int64, device="cuda")
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for i in range(K):
        with torch.cuda.stream(st):
            s_dev.copy_(S_host[i], non_blocking=True)
        store.relocate(s_dev, 0.7, stream=st)
        store.compact_pages(0.75, 0.7, stream=st)
        stats = store.page_stats()
    e1.record(st)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1) / K
    after = replay()
    stats = store.page_stats()
    n_pages = stats["pages_in_use"]
    hbm, _, kind = peaks()
    rel_ms, rel_l = phases["relocate"]
    cmp_ms, cmp_l = phases["compact"]
    # compaction: every page's two counters and every chunk's page and
    # tombstone read once (the directory scan that finds what moves)
    cmp_bytes = n_pages * 8 + wl.n * 8
    achieved = cmp_bytes / (cmp_ms / K * 1e-3) / 1e9
    line = {
        "metric": MEMORY_METRIC, "value": B * 1000.0 / ms, "unit": "requests/s",
        "n_gpus": 1, "steps": K, "warmup": W, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int32", "data": "synthetic",
        "config": {"workload": MEMORY_WORKLOAD
                   + ("" if args.scale == 1.0 else f", scaled by {args.scale}"),
                   "l2": "directory and tables stay resident; the step's work is latency-bound"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm, "traffic": None,
                     "kernel": "whole compaction call", "peak_kind": kind},
        "phases_ms_per_step": {"relocate": rel_ms / K, "compact": cmp_ms / K},
        "pages_per_request": {"before": before, "after": after},
        "space_amplification": stats["slots_total"] / max(1, stats["slots_live"]),
        "write_amplification": stats["chunk_writes"] / max(1, stats["appended"]),
        "e2e": {"value": B * 1000.0 / e2e_ms, "unit": "requests/s",
                "h2d_bytes_per_step": B * 5 * 8, "d2h_bytes_per_step": 5 * 8},
        "gpu_launches": int(rel_l + cmp_l),
        "cpu_baseline": cpu,
        "clocks": clk.summary(),
    }
    print(json.dumps(line), flush=True)
    store.close()
    return 0


def run_streams(args):
    """4M-chunk store, 1024 queries issued as 8 streams of 128 in a seeded
    arrival order; aggregate queries/s over all streams."""
    import torch
    import synth
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_05708_gb300 import MemStore
    wl = synth.workload(4, scale=args.scale)
    store = MemStore.from_arrays(wl.emb, wl.page_of[args.placement], wl.row_ptr, wl.col, wl.aff,
                                 capacity=wl.n, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau)
    per = wl.n_queries // wl.streams
    streams = [torch.cuda.Stream() for _ in range(wl.streams)]
    qs = [torch.from_numpy(np.ascontiguousarray(wl.queries[i * per:(i + 1) * per]).view(np.int16)).cuda()
          for i in range(wl.streams)]
    outs = [(torch.empty((per, wl.k), dtype=torch.int64, device="cuda"),
             torch.empty((per, wl.k), dtype=torch.float32, device="cuda"),
             torch.empty((per, wl.k), dtype=torch.int32, device="cuda"),
             torch.empty((per,), dtype=torch.int32, device="cuda")) for _ in range(wl.streams)]

    def step():
        for i in wl.stream_order:
            store.retrieve(qs[i], wl.k, wl.alpha, wl.hops, *outs[i], stream=streams[i])

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    main = torch.cuda.current_stream()
    with Clocks(0) as clk:
        t0.record(main)
        for s in streams:
            s.wait_stream(main)
        for _ in range(args.steps):
            step()
        for s in streams:
            main.wait_stream(s)
        t1.record(main)
        torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / args.steps
    store.sync()
    pages = {}
    for kind in wl.page_of:
        po = wl.page_of[kind]
        sel = np.concatenate([o[0].cpu().numpy() for o in outs])
        pages[kind] = float(np.mean([len(set(po[r].tolist())) for r in sel]))
    ab = algorithmic_bytes(wl.n, wl.dim, per, wl.nnz, wl.hops, wl.k)
    hbm, bf16, kind = peaks()
    line = {
        "metric": "retrieve queries/sec at N=4M chunks, d=768, 8 streams x 128 queries",
        "value": wl.n_queries / (ms * 1e-3), "unit": "queries/s", "higher_is_better": True,
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "gmm4m: N=4194304 chunks, d=768, 16384-component Zipf(1.1) mixture, "
                   "32-neighbour power-law graph, 8 streams x 128 queries (seeded arrival), "
                   f"hops=2, alpha=0.4, k=64, 64 chunks/page, {args.placement} placement"
                   + ("" if args.scale == 1.0 else f", scaled by {args.scale}")},
        "pass_roofline": {"algorithmic_bytes_per_call": sum(ab.values()),
                          "ideal_ms_all_calls": wl.streams * sum(ab.values()) / (hbm * 1e9) * 1e3},
        "pages_per_query": pages,
        "clocks": clk.summary(),
    }
    print(json.dumps(line), flush=True)
    store.close()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default: 400 for retrieve and dense, 100 for scoped and "
                         "the reference arm, 5 for update, 20 for streams and memory, 10 for "
                         "delete)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--cpu-queries", type=int, default=8)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-hop-path", action="store_true",
                    help="skip the retrieve workload's hop_path record (the same retrieval "
                         "with the hops always run)")
    ap.add_argument("--placement", default="clustered")
    ap.add_argument("--scale", type=float, default=1.0,
                    help="shrink N (profiling captures of a smaller case); 1.0 = the benchmark")
    ap.add_argument("--workload", default="retrieve",
                    choices=["retrieve", "update", "streams", "dense", "scoped", "delete",
                             "memory"],
                    help="retrieve: the benchmark; update: relation update of 4096 new chunks "
                         "on the 1M-chunk store; streams: 4M-chunk store, 8 streams x 128 "
                         "queries; dense: the Dense-only form (k=5, no hops) on the 1M store; "
                         "scoped: namespace-scoped retrieval with SortByTime on the 1M store; "
                         "delete: 1024 chunks deleted per step from the 1M store; memory: "
                         "relocation + block compaction of 256 top-5 requests per step")
    args = ap.parse_args()
    if args.steps is None and args.impl == "reference":
        args.steps = 100          # one oracle query per step, ~1 s each
    if args.steps is None:
        args.steps = {"retrieve": 400, "update": 5, "streams": 20, "dense": 400,
                      "scoped": 100, "delete": 10, "memory": 20}[args.workload]
    if args.impl == "reference":
        return run_reference(args)
    if args.workload == "update":
        return run_update(args)
    if args.workload == "streams":
        return run_streams(args)
    if args.workload == "delete":
        return run_delete(args)
    if args.workload == "memory":
        return run_memory(args)
    if args.workload == "dense":
        return run_retrieve(args, k=5, hops=0, metric=DENSE_METRIC, workload=DENSE_WORKLOAD)
    if args.workload == "scoped":
        return run_retrieve(args, metric=SCOPED_METRIC, workload=SCOPED_WORKLOAD, scoped=True)
    return run_retrieve(args, hop_path=not args.no_hop_path)


def run_retrieve(args, k=None, hops=None, metric=METRIC, workload=WORKLOAD, scoped=False,
                 hop_path=False):
    """The retrieval pass on the gmm1m store (k / hops override the
    configuration: the Dense-only form uses k = 5, hops = 0; `scoped` tags
    chunks by component mod 64 and scopes each query to a namespace, with
    results in chronological order)."""
    import torch
    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = local if ws > 1 else 0
    torch.cuda.set_device(dev)

    import synth
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_05708_gb300 import MemStore

    t_gen = time.perf_counter()
    wl = synth.workload(2, scale=args.scale)
    t_gen = time.perf_counter() - t_gen
    ns_of = q_ns_host = None
    if scoped:
        ns_of = (wl.component % 64).astype(np.int32)
        q_ns_host = np.random.default_rng(64).integers(0, 64, wl.n_queries).astype(np.int32)
    cpu = None
    if rank == 0 and not args.no_cpu_baseline and ws == 1:
        cpu = cpu_baseline(wl, args.placement, args.cpu_queries, k=k, hops=hops, ns_of=ns_of,
                           q_ns=q_ns_host, sort_by_time=scoped)

    store = MemStore.from_arrays(wl.emb, wl.page_of[args.placement], wl.row_ptr, wl.col, wl.aff,
                                 capacity=wl.n, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau, device=dev)
    B = wl.n_queries
    k = wl.k if k is None else k
    hops = wl.hops if hops is None else hops
    st = torch.cuda.Stream(device=dev)
    # a rotating pool of distinct seeded query batches (the workload's own
    # batch first): step i retrieves batch i mod POOL
    batches = [wl.queries] + synth.query_batches(wl, QUERY_POOL - 1)
    q_pool = torch.from_numpy(np.stack(batches).view(np.int16)).to(f"cuda:{dev}")
    q_dev = torch.empty_like(q_pool[0])
    ids = torch.empty((B, k), dtype=torch.int64, device=f"cuda:{dev}")
    scores = torch.empty((B, k), dtype=torch.float32, device=f"cuda:{dev}")
    pages = torch.empty((B, k), dtype=torch.int32, device=f"cuda:{dev}")
    npages = torch.empty((B,), dtype=torch.int32, device=f"cuda:{dev}")

    q_ns = None
    if scoped:
        store.set_namespace(0, torch.from_numpy(ns_of).to(f"cuda:{dev}"))
        q_ns = torch.from_numpy(q_ns_host).to(f"cuda:{dev}")

    def step(i, q=None, target=None):
        (target or store).retrieve(q_pool[i % QUERY_POOL] if q is None else q, k, wl.alpha, hops,
                                   ids, scores, pages, npages, stream=st, q_ns=q_ns,
                                   sort_by_time=scoped)

    def barrier():
        torch.cuda.synchronize(dev)
        if ws > 1:
            torch.distributed.barrier()

    with torch.cuda.stream(st):
        for i in range(args.warmup):
            step(i)
    store.sync(stream=st)
    # ---- timed region (device-resident inputs)
    store.set_profiling(True)
    store.phase_times()                       # reset
    barrier()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    with Clocks(dev) as clk:
        ev0.record(st)
        for i in range(args.steps):
            step(i)
        ev1.record(st)
        barrier()
    store.sync(stream=st)
    ms = ev0.elapsed_time(ev1)
    phases = store.phase_times()
    store.set_profiling(False)
    # page counts of this placement and of the other
    npg_clustered = npages.float().mean().item()

    # ---- end-to-end: host query buffer in, host results out, via the public API
    q_host = torch.from_numpy(np.stack(batches).view(np.int16)).pin_memory()
    outs_host = [torch.empty((B, k), dtype=torch.int64).pin_memory(),
                 torch.empty((B, k), dtype=torch.float32).pin_memory(),
                 torch.empty((B, k), dtype=torch.int32).pin_memory(),
                 torch.empty((B,), dtype=torch.int32).pin_memory()]

    def e2e_step(i):
        with torch.cuda.stream(st):
            q_dev.copy_(q_host[i % QUERY_POOL], non_blocking=True)
            step(i, q=q_dev)
            for h, d in zip(outs_host, (ids, scores, pages, npages)):
                h.copy_(d, non_blocking=True)

    for i in range(args.warmup):
        e2e_step(i)
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for i in range(args.steps):
        e2e_step(i)
    e1.record(st)
    barrier()
    ms_e2e = e0.elapsed_time(e1)
    store.sync(stream=st)
    h2d = q_host[0].numel() * 2
    d2h = sum(t.numel() * t.element_size() for t in outs_host)

    # max over ranks
    ms, ms_e2e = max_over_ranks([ms, ms_e2e], device=f"cuda:{dev}" if ws > 1 else None)

    hbm, bf16, peak_kind = peaks()
    ab = algorithmic_bytes(wl.n, wl.dim, B, wl.nnz, hops, k)
    total_ab = sum(ab.values())
    per_step_ms = ms / args.steps
    # dominant phase.  "propagate" holds the hops before the last (full
    # hops); the last hop ("last_hop") skips the rows whose bound stays
    # below the top-k floor, so its bytes are not a full hop's.
    retr = ("score", "propagate", "last_hop", "bound", "select")
    full_hops = hops - 1 if phases["last_hop"][0] > 0 else hops
    dom = max(("score", "propagate", "select"), key=lambda p: phases[p][0])
    dom_ms, dom_launches = phases[dom]
    if dom == "propagate":
        per_launch_bytes = hop_bytes(wl.n, 256, wl.nnz)
        units = args.steps * max(1, full_hops)
        what = "full propagation hop (graph once + two slab passes)"
    elif dom == "score":
        per_launch_bytes = score_bytes(wl.n, wl.dim, 256)
        units = args.steps
        what = "score pass (E read once + u slab written once)"
    else:
        per_launch_bytes = wl.n * 256 * 4
        units = args.steps
        what = "selection pass (final slab read once)"
    dom_avg_ms = dom_ms / units
    achieved = per_launch_bytes / (dom_avg_ms * 1e-3) / 1e9
    # which propagation ran: the hops, or (two hops, every row that can reach
    # the top-k among the reach candidates) the candidates' scores from u
    if hops >= 1 and phases["propagate"][1] == 0 and phases["last_hop"][1] > 0:
        moved = wl.n * wl.dim * 2 + 2 * wl.n * 256 * 4 + wl.n * 64 * 2 * 2
        path_note = {"propagation": "two-hop scores of the top-k candidates from graph-only "
                                    "reach coefficients, one tensor-core pass over u (no hop run)",
                     "bytes_moved_per_step": moved,
                     "note": "pass_roofline counts full hops (five slab passes); this path "
                             "reads E, writes u and reads u and 64 coefficient rows per store "
                             "row (bf16 hi + lo; 128 when a flagged candidate is at slot 64 or "
                             "above)"}
    else:
        moved = total_ab
        path_note = {"propagation": "hops (the last one skips rows below the top-k floor)",
                     "bytes_moved_per_step": moved}
    path_note["call_hbm_frac"] = moved / (per_step_ms * 1e-3) / 1e9 / hbm
    line = {
        "metric": metric,
        "value": job_throughput(B * args.steps, ws, ms),
        "unit": "queries/s",
        "n_gpus": ws,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": per_step_ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": workload if args.scale == 1.0 else f"{workload} scaled by {args.scale}",
                   "l2": "inputs larger than L2 (E 2.1 GB, score slabs 1.07 GB "
                   "each), no flush", "placement": args.placement,
                   "queries": f"{QUERY_POOL} distinct seeded batches of {B}, step i takes batch "
                              f"i mod {QUERY_POOL}",
                   "parallelism": "replicas" if ws > 1 else "single GPU"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm,
                     "traffic": (None if args.scale != 1.0 else
                                 HOP_DRAM_BYTES if dom == "propagate" else
                                 SCORE_DRAM_BYTES if dom == "score" else None),
                     "kernel": dom, "what": what, "peak_kind": peak_kind},
        "pass_roofline": {"algorithmic_bytes": total_ab,
                          "ideal_ms": total_ab / (hbm * 1e9) * 1e3,
                          "frac": (total_ab / (hbm * 1e9) * 1e3) / per_step_ms,
                          "flops": 2.0 * wl.n * B * wl.dim,
                          "peak_tflops_bf16": bf16},
        "phases_ms_per_step": {p: phases[p][0] / args.steps for p in retr},
        "path": path_note,
        "e2e": {"value": job_throughput(B * args.steps, ws, ms_e2e), "unit": "queries/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": int(sum(v[1] for v in phases.values())),
        "pages_per_query": {args.placement: npg_clustered},
        "clocks": clk.summary(),
        "gen_seconds": t_gen,
    }
    if cpu is not None:
        line["cpu_baseline"] = {k2: cpu[k2] for k2 in ("value", "unit", "cores", "kind", "sample")}
    # the other placement's page count (same selected IDs, different page table)
    other = "random" if args.placement == "clustered" else "clustered"
    if other in wl.page_of:
        po = wl.page_of[other]
        sel = ids.cpu().numpy()
        line["pages_per_query"][other] = float(np.mean([len(set(po[r].tolist())) for r in sel]))
    store.close()
    if hop_path and hops >= 1 and not scoped and args.scale == 1.0:
        line["hop_path"] = time_hop_path(args, wl, step, st, barrier, dev, ws, B, hbm, peak_kind)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()
    return 0


def time_hop_path(args, wl, step, st, barrier, dev, ws, B, hbm, peak_kind):
    """The same retrieval with the hops always run (a store created with
    AKASHIC_REACH=0), timed the same way over the same rotating batches:
    its queries/s, and the full hop's roofline (graph once + two slab
    passes per hop against the hop phase's event-timed duration) with its
    ncu DRAM bytes."""
    import torch
    from paper_2607_05708_gb300 import MemStore
    old = os.environ.get("AKASHIC_REACH")
    os.environ["AKASHIC_REACH"] = "0"
    try:
        store = MemStore.from_arrays(wl.emb, wl.page_of[args.placement], wl.row_ptr, wl.col,
                                     wl.aff, capacity=wl.n, chunks_per_page=wl.chunks_per_page,
                                     temperature=wl.tau, device=dev)
    finally:
        if old is None:
            del os.environ["AKASHIC_REACH"]
        else:
            os.environ["AKASHIC_REACH"] = old
    steps = max(1, min(args.steps, HOP_PATH_STEPS))
    with torch.cuda.stream(st):
        for i in range(args.warmup):
            step(i, target=store)
    store.sync(stream=st)
    store.set_profiling(True)
    store.phase_times()
    barrier()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(st)
    for i in range(steps):
        step(i, target=store)
    ev1.record(st)
    barrier()
    store.sync(stream=st)
    ms = ev0.elapsed_time(ev1)
    phases = store.phase_times()
    store.close()
    ms = max_over_ranks([ms], device=f"cuda:{dev}" if ws > 1 else None)[0]
    hop_ms = phases["propagate"][0] / steps
    per_hop = hop_bytes(wl.n, 256, wl.nnz)
    achieved = per_hop / (hop_ms * 1e-3) / 1e9
    return {
        "value": job_throughput(B * steps, ws, ms), "unit": "queries/s", "steps": steps,
        "ms_per_step": ms / steps,
        "phases_ms_per_step": {p: phases[p][0] / steps
                               for p in ("score", "propagate", "last_hop", "bound", "select")},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm, "traffic": HOP_DRAM_BYTES,
                     "kernel": "propagate", "what": "full propagation hop (graph once + two "
                     "slab passes), k_hop_segs + k_hop_rows", "peak_kind": peak_kind},
        "note": "the same store and batches with AKASHIC_REACH=0: the first hop runs in full, "
                "the last skips rows whose bound stays below the top-k floor",
    }


if __name__ == "__main__":
    sys.exit(main())
