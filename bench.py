#!/usr/bin/env python
"""Benchmark of the DoPR online scoring pass on GB300.

One step = one dopr_score call over one batch of the workload: Q queries'
candidate lists (default 20 queries x 100 candidates = 2,000 pairs of the
Qwen3-8B, m = 64, Zipf(1.1) workload).  Steps walk through the workload's
200 queries; with --gpus N every rank scores its own batches (pairs are
independent: weak scaling, no data-path collective).

Printed JSON line (rank 0):
  value      scored pairs/s, inputs resident in HBM (io_on_device = 1), max over ranks
  e2e        same metric through the C ABI with pinned host buffers (H2D of the
             batch and D2H of its scores inside the timed region)
  roofline   dominant kernel (the tcgen05 projection GEMM family): algorithmic
             FLOPs / CUDA-event time of its launches in the timed region, vs
             the measured sustained bf16 peak
  kernels    the same accounting for every kernel family
  cpu_baseline  the fp64 oracle timed on a bounded sample on the host cores
  --impl reference  times the oracle alone (the reference arm of this workload)
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "scored query-doc pairs/sec at 1 GB300 (Qwen3-8B shape, m=64); p50 batch latency"
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e data-sheet bandwidth, printed beside the measured-peak fractions


# Short numbers for the measured workloads: 0 the 2-layer Qwen3-0.6B-width case, 1 Qwen3-0.6B,
# 2 Qwen3-4B with long queries, 3 Qwen3-8B with Zipf reuse and mixed prefix lengths, 3' the same
# Qwen3-8B pairs with m = 64 throughout (the default), 4 those pairs scored uncompressed.
CONFIG_WORKLOADS = {"0": "qwen3-0.6b-2l", "1": "qwen3-0.6b", "2": "qwen3-4b", "3": "qwen3-8b-zipf",
                    "3'": "qwen3-8b-m64", "4": "qwen3-8b-fulldoc"}


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["dopr", "reference"], default="dopr")
    ap.add_argument("--workload", default="qwen3-8b-m64")
    ap.add_argument("--config", choices=sorted(CONFIG_WORKLOADS), default=None,
                    help="select the workload by configuration number (overrides --workload)")
    ap.add_argument("--queries-per-step", type=int, default=20)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-seconds", type=float, default=120.0,
                    help="bound on the oracle time of the CPU-baseline sample (8 length-stratified pairs)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--latency-queries", type=int, default=10)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the bounded measurement of every configuration after the headline")
    ap.add_argument("--reuse", action="store_true",
                    help="amortised cost under document reuse (T_off, T_full, T_online, Speedup(r)) instead of the bench")
    args = ap.parse_args(argv)
    if args.config is not None:
        args.workload = CONFIG_WORKLOADS[args.config]
    return args


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        p = json.load(open(path))
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"],
                "bf16_tflops_sustained": p.get("bf16_tflops_sustained", p["bf16_tflops"]), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# ------------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""
    FIELDS = "index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown," \
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown," \
             "clocks_event_reasons.sw_power_cap"

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.lines = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# -------------------------------------------------------------- workload

def build_pairs(wl, seed):
    from paper_2609_03311_gb300 import synth

    pairs = synth.make_workload_pairs(wl, seed=seed)
    if wl.fulldoc_tokens:
        # uncompressed pointwise scoring: [doc tokens ; query] per pair, no prefix
        qo, qt, docs = pairs["q_offsets"], pairs["q_tokens"], pairs["doc_ids"]
        cache = {}
        seqs = []
        for p in range(len(docs)):
            d = int(docs[p])
            if d not in cache:
                cache[d] = synth.make_fulldoc_tokens(wl, d, seed=seed)
            seqs.append(np.concatenate([cache[d], qt[qo[p]:qo[p + 1]]]))
        pairs["q_offsets"] = np.concatenate([[0], np.cumsum([len(s) for s in seqs])]).astype(np.int32)
        pairs["q_tokens"] = np.concatenate(seqs).astype(np.int32)
    return pairs


def slice_pairs(pairs, p0, p1):
    qo = pairs["q_offsets"]
    return {"q_offsets": (qo[p0:p1 + 1] - qo[p0]).astype(np.int32),
            "q_tokens": pairs["q_tokens"][qo[p0]:qo[p1]].astype(np.int32),
            "doc_ids": pairs["doc_ids"][p0:p1].astype(np.int64)}


def oracle_sample(wl, w_host, doc_m, pairs, idx, seed, deadline_s, gen_device):
    """Score pairs idx[0], idx[1], ... with the oracle until deadline_s of oracle
    time is used (at least one pair).  The prefix states are drawn and copied to
    the host before the clock starts; only the oracle's scoring is timed.
    Returns (scores dict, seconds, threads); the scored pairs' token count is
    in oracle_sample.tokens after the call."""
    import oracle
    from paper_2609_03311_gb300 import synth

    s = wl.model
    om = oracle.OracleModel(oracle.Shape(s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn,
                                         s.vocab, s.rope_theta, s.rms_eps, s.score_token_id), w_host)
    got = {}
    secs = 0.0
    oracle_sample.tokens = 0
    for p in idx:
        d = int(pairs["doc_ids"][p])
        m = int(doc_m[d])
        # the same draw the store received (same seed, same generator device), moved to the host untimed
        k, v = synth.make_prefix(s, m, d, seed=seed, device=gen_device)
        kv = [(k.cpu(), v.cpu())]
        one = slice_pairs(pairs, p, p + 1)
        t0 = time.perf_counter()
        got[int(p)] = float(om.score_pairs(one["q_offsets"], one["q_tokens"], [0], kv)[0])
        secs += time.perf_counter() - t0
        oracle_sample.tokens += len(one["q_tokens"]) + 1
        if secs >= deadline_s:
            break
    return got, secs, oracle.num_threads()


def stratified_pairs(wl, pairs, n_queries, n):
    """A length-stratified sample of n pairs from the first n_queries queries'
    candidate lists: the queries at n evenly spaced quantiles of query length
    (shortest and longest included), the first candidate of each."""
    per_q = wl.docs_per_query
    lens = np.diff(pairs["q_offsets"])[::per_q][:n_queries]
    order = np.argsort(lens, kind="stable")
    picks = sorted(set(int(order[round(i * (len(order) - 1) / max(n - 1, 1))]) for i in range(n)))
    return [q * per_q for q in picks]


CPU_SAMPLE_PAIRS = 8  # the oracle's timed sample (the GPU arm's cpu_baseline and the reference arm)
L2_FLUSH_BYTES = 512 << 20  # four times the 129 MB L2


def streamed_bytes_per_step(wl):
    """Bytes of fp16 projection matrices one step reads (every layer's QKV, O,
    gate/up and down) -- the input that does not depend on the batch."""
    m = wl.model
    qkv = m.hidden * (m.n_q_heads + 2 * m.n_kv_heads) * m.head_dim
    o = m.n_q_heads * m.head_dim * m.hidden
    mlp = 3 * m.hidden * m.ffn
    return 2 * m.n_layers * (qkv + o + mlp)


def shard_batch(rank, world, step, n_batches):
    """Index of the batch that `rank` scores at `step`.  The ranks of one step
    take consecutive batches, so no two ranks score the same pairs in a step
    while the step count times the world size stays within the workload."""
    return (rank + step * world) % n_batches


def reduce_over_ranks(dist, x, op, device):
    """Scalar all-reduce ("max" or "sum") over the ranks; the identity at world size 1.
    The tensor lives on the GPU for NCCL and on the host for gloo."""
    if dist is None:
        return x
    import torch

    t = torch.tensor([x], dtype=torch.float64, device=device if dist.get_backend() == "nccl" else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def setup(wl, seed, device, need_host_weights):
    """Random-init model and prefix store on `device`; optional host copy of
    the weights for the oracle."""
    import torch

    from paper_2609_03311_gb300 import dopr, synth

    s = wl.model
    w = synth.make_weights(s, seed=seed, device=device, norms="ones")
    max_pos = max(wl.m_choices) + wl.fulldoc_tokens + wl.qlen_max + 2
    cfg = dopr.make_config(s, max_position=max(1024, max_pos))
    model = dopr.Model(cfg, w)
    w_host = None
    if need_host_weights:
        w_host = {k: (v.cpu() if isinstance(v, torch.Tensor) else [t.cpu() for t in v]) for k, v in w.items()}
    del w
    torch.cuda.empty_cache()
    store, doc_m = make_store(cfg, wl, seed, device)
    return cfg, model, store, doc_m, w_host


def make_store(cfg, wl, seed, device):
    """The workload's prefix store (every document, drawn on `device`)."""
    import torch

    from paper_2609_03311_gb300 import dopr, synth

    doc_m = synth.doc_prefix_lengths(wl, seed=seed)
    pool = sum(dopr.prefix_bytes(cfg, int(m)) for m in doc_m) + (1 << 20)
    store = dopr.Store(cfg, wl.n_docs - 1, pool)
    for d in range(wl.n_docs):
        k, v = synth.make_prefix(wl.model, int(doc_m[d]), d, seed=seed, device=device)
        store.put(d, k, v)
    torch.cuda.synchronize()
    return store, doc_m


def gemm_traffic_record():
    """ncu-measured DRAM traffic of the projection GEMMs as a multiple of their
    algorithmic bytes, valid only for the kernel source it was captured from
    (else None)."""
    path = os.path.join(ROOT, "profiles", "gemm_traffic.json")
    if not os.path.exists(path):
        return None
    rec = json.load(open(path))
    src = open(os.path.join(ROOT, "paper_2609_03311_gb300", "csrc", "k_gemm.cu"), "rb").read()
    if rec.get("k_gemm_sha256") != hashlib.sha256(src).hexdigest():
        return None
    return rec


def kernel_table(prof, steps, peaks):
    """Per kernel family: launches and ms per step, share of kernel time, achieved
    TFLOP/s and GB/s on algorithmic work, and the roofline fraction (the slower of
    FLOPs at the sustained tensor peak and bytes at the HBM peak, over the time)."""
    tot_ms = sum(v["time_ms"] for v in prof.values()) or 1e-9
    kernels = {}
    for name, v in prof.items():
        if v["launches"] == 0:
            continue
        t_s = v["time_ms"] / 1e3
        ent = {"launches_per_step": v["launches"] / steps, "ms_per_step": v["time_ms"] / steps,
               "share": v["time_ms"] / tot_ms}
        if t_s > 0:
            tf = v["flops"] / t_s / 1e12
            gbs = v["bytes"] / t_s / 1e9
            t_roof = max(v["flops"] / (peaks["bf16_tflops_sustained"] * 1e12), v["bytes"] / (peaks["hbm_gbs"] * 1e9))
            ent.update({"tflops": tf, "gbs": gbs, "roofline_frac": t_roof / t_s,
                        "gbs_frac_of_nominal_hbm": gbs / NOMINAL_HBM_GBS})
        kernels[name] = ent
    return kernels


# Queries per step of each configuration's measurement in the default run (the headline's
# 20; 32 for the launch-bound 2-layer model; 10 for the long 4B queries; 2 for the 512-token
# uncompressed documents), and the bounded step counts it uses.
CONFIG_QUERIES = {"0": 32, "1": 20, "2": 10, "3": 20, "4": 2}
CONFIG_WARMUP, CONFIG_STEPS = 2, 3


def time_workload(model, store, wl, pairs, Q, steps, warmup, dev, gpu_index):
    """Steps of Q queries' candidate lists through dopr_score with device-resident inputs
    (L2 flushed between steps when the streamed weights fit in it); CUDA-event time,
    clocks sampled meanwhile, per-kernel accounting."""
    import torch

    from paper_2609_03311_gb300 import dopr

    per_q = wl.docs_per_query
    n_batches = max(1, wl.n_queries // Q)
    batches = []
    for b in range(n_batches):
        sl = slice_pairs(pairs, b * Q * per_q, (b + 1) * Q * per_q)
        batches.append((torch.tensor(sl["q_offsets"], device=dev), torch.tensor(sl["q_tokens"], device=dev),
                        torch.tensor(sl["doc_ids"], device=dev)))
    for i in range(warmup):
        dopr.score(model, store, *batches[i % n_batches])
    stream_bytes = streamed_bytes_per_step(wl)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev) if stream_bytes < L2_FLUSH_BYTES else None
    stream = torch.cuda.current_stream(dev)
    torch.cuda.synchronize()
    dopr.profile_enable(model, True)
    clocks = ClockSampler(gpu_index)
    clocks.start()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * steps)]
    n_pairs = 0
    for i in range(steps):
        if flush is not None:
            flush.zero_()
        b = batches[(warmup + i) % n_batches]
        ev[2 * i].record(stream)
        dopr.score(model, store, *b)
        ev[2 * i + 1].record(stream)
        n_pairs += b[2].numel()
    torch.cuda.synchronize()
    clk = clocks.stop()
    prof = dopr.profile_read(model)
    dopr.profile_enable(model, False)
    step_ms = [ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(steps)]
    total_ms = sum(step_ms) if flush is not None else ev[0].elapsed_time(ev[-1])
    peaks = measured_peaks()
    kernels = kernel_table(prof, steps, peaks)
    gemm = [f for f in ("gemm_qkv", "gemm_o", "gemm_gate_up", "gemm_down") if f in prof]
    g_ms = sum(prof[f]["time_ms"] for f in gemm)
    g_tf = sum(prof[f]["flops"] for f in gemm) / (g_ms / 1e3) / 1e12 if g_ms > 0 else None
    return {"workload": wl.name, "pairs_per_s": n_pairs / (total_ms / 1e3), "ms_per_step": statistics.mean(step_ms),
            "p50_batch_ms": statistics.median(step_ms), "pairs_per_step": Q * per_q, "steps": steps,
            "warmup": warmup, "clocks": clk,
            "roofline_frac": {k: round(v["roofline_frac"], 4) for k, v in kernels.items() if "roofline_frac" in v},
            "share": {k: round(v["share"], 4) for k, v in kernels.items()},
            "gemm_tflops": g_tf,
            "gemm_frac_of_sustained": g_tf / peaks["bf16_tflops_sustained"] if g_tf else None,
            "l2": "flushed between steps" if flush is not None else "inputs larger than L2"}


def run_configs(args, dev, gpu_index, headline, model8=None, cfg8=None):
    """Every configuration once after the headline, with bounded step counts: pairs/s,
    clocks and per-kernel roofline fractions; for the uncompressed arm (4) also the
    speed-up of DoPR (m = 64: the headline's pairs) over it and the doc-side K/V ratio.
    `model8`, the headline's Qwen3-8B model when it is one, serves configurations 3 and
    4 and is closed here."""
    import torch

    from paper_2609_03311_gb300 import dopr, synth

    out = {}
    for key in ("3", "4", "2", "1", "0"):  # the 8B arms first, while the headline's model is resident
        wl = synth.WORKLOADS[CONFIG_WORKLOADS[key]]
        t0 = time.perf_counter()
        if model8 is not None and wl.model.name == "qwen3-8b":
            model, own = model8, False
            store, _ = make_store(cfg8, wl, args.seed, dev)
        else:
            if model8 is not None:  # the 8B arms are done: free the headline's model
                model8.close()
                model8 = None
                torch.cuda.empty_cache()
            _, model, store, _, _ = setup(wl, args.seed, dev, False)
            own = True
        pairs = build_pairs(wl, args.seed)
        r = time_workload(model, store, wl, pairs, min(CONFIG_QUERIES[key], wl.n_queries), CONFIG_STEPS,
                          CONFIG_WARMUP, dev, gpu_index)
        r["setup_and_run_s"] = round(time.perf_counter() - t0, 1)
        store.close()
        if own:
            model.close()
        torch.cuda.empty_cache()
        out[key] = r
    if headline.get("workload") == "qwen3-8b-m64":
        c8 = dopr.make_config(synth.MODELS["qwen3-8b"])
        out["4"]["dopr_m64_pairs_per_s"] = headline["value"]
        out["4"]["speedup_dopr_over_uncompressed"] = headline["value"] / out["4"]["pairs_per_s"]
        out["4"]["doc_kv_bytes_ratio"] = dopr.prefix_bytes(c8, 512) / dopr.prefix_bytes(c8, 64)
    if model8 is not None:
        model8.close()
    return out


# ------------------------------------------------------------------ arms

def run_dopr(args, rank, world, local_rank, dist):
    import torch

    from paper_2609_03311_gb300 import dopr, synth

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    wl = synth.WORKLOADS[args.workload]
    want_cpu = (not args.no_cpu_baseline) and rank == 0 and world == 1
    cfg, model, store, doc_m, w_host = setup(wl, args.seed, dev, want_cpu)
    pairs = build_pairs(wl, args.seed)
    per_q = wl.docs_per_query
    Q = max(1, min(args.queries_per_step, wl.n_queries))
    n_batches = wl.n_queries // Q
    batches = []
    for b in range(n_batches):
        sl = slice_pairs(pairs, b * Q * per_q, (b + 1) * Q * per_q)
        sl["dev"] = (torch.tensor(sl["q_offsets"], device=dev), torch.tensor(sl["q_tokens"], device=dev),
                     torch.tensor(sl["doc_ids"], device=dev))
        sl["pin"] = (torch.tensor(sl["q_offsets"]).pin_memory(), torch.tensor(sl["q_tokens"]).pin_memory(),
                     torch.tensor(sl["doc_ids"]).pin_memory())
        sl["first_pair"] = b * Q * per_q
        batches.append(sl)
    stream = torch.cuda.current_stream(dev)

    def batch_for(step):
        return batches[shard_batch(rank, world, step, n_batches)]

    def step_dev(b):
        qo, qt, di = b["dev"]
        return dopr.score(model, store, qo, qt, di)

    def barrier():
        if dist is not None:
            dist.barrier()

    def max_over_ranks(x):
        return reduce_over_ranks(dist, x, "max", dev)

    def sum_over_ranks(x):
        return reduce_over_ranks(dist, x, "sum", dev)

    for i in range(args.warmup):
        step_dev(batch_for(i))
    # A step streams every layer's projection matrices and the batch's prefixes from
    # HBM; where those fit in L2 (129 MB), each timed step starts from a flushed L2.
    stream_bytes = streamed_bytes_per_step(wl)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev) if stream_bytes < L2_FLUSH_BYTES else None
    torch.cuda.synchronize()

    # ---------------- timed region: device-resident inputs
    dopr.profile_enable(model, True)
    clocks = ClockSampler(local_rank)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * args.steps)]
    pairs_done = 0
    outs = []
    for i in range(args.steps):
        if flush is not None:
            flush.zero_()  # outside the events: evicts the previous step's weights from L2
        b = batch_for(args.warmup + i)
        ev[2 * i].record(stream)
        outs.append((b, step_dev(b)))
        ev[2 * i + 1].record(stream)
        pairs_done += len(b["doc_ids"])
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    prof = dopr.profile_read(model)
    dopr.profile_enable(model, False)
    step_ms = [ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(args.steps)]
    # back to back without a flush the steps are contiguous, so the sum is the span
    total_ms = max_over_ranks(sum(step_ms) if flush is not None else ev[0].elapsed_time(ev[-1]))
    all_pairs = sum_over_ranks(pairs_done)
    value = all_pairs / (total_ms / 1e3)

    # ---------------- e2e: pinned host buffers through the C ABI
    e2e = None
    if not args.no_e2e:
        out_pin = torch.empty(Q * per_q, dtype=torch.float32).pin_memory()
        barrier()
        torch.cuda.synchronize()
        ee = [torch.cuda.Event(enable_timing=True) for _ in range(2 * args.steps)]
        h2d = d2h = 0
        for i in range(args.steps):
            if flush is not None:
                flush.zero_()
            b = batch_for(args.warmup + i)
            qo, qt, di = b["pin"]
            n = len(b["doc_ids"])
            ee[2 * i].record(stream)
            dopr.score(model, store, qo, qt, di, out=out_pin[:n])
            ee[2 * i + 1].record(stream)
            h2d += qo.numel() * 4 + qt.numel() * 4 + di.numel() * 8
            d2h += n * 4
        torch.cuda.synchronize()
        barrier()
        e_steps = [ee[2 * i].elapsed_time(ee[2 * i + 1]) for i in range(args.steps)]
        e_ms = max_over_ranks(sum(e_steps) if flush is not None else ee[0].elapsed_time(ee[-1]))
        e2e = {"value": all_pairs / (e_ms / 1e3), "unit": "pairs/s", "h2d_bytes_per_step": h2d // args.steps,
               "d2h_bytes_per_step": d2h // args.steps}

    # ---------------- per-query latency (one call per query's candidate list)
    lat = []
    for qi in range(min(args.latency_queries, wl.n_queries)):
        sl = slice_pairs(pairs, qi * per_q, (qi + 1) * per_q)
        qo, qt, di = (torch.tensor(sl["q_offsets"], device=dev), torch.tensor(sl["q_tokens"], device=dev),
                      torch.tensor(sl["doc_ids"], device=dev))
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        dopr.score(model, store, qo, qt, di)
        torch.cuda.synchronize()
        lat.append((time.perf_counter() - t0) * 1e3)
    lat_sorted = sorted(lat[1:] if len(lat) > 1 else lat)

    # ---------------- roofline accounting from the live CUDA-event timing
    peaks = measured_peaks()
    gemm_fams = ["gemm_qkv", "gemm_o", "gemm_gate_up", "gemm_down"]
    tot_ms = sum(v["time_ms"] for v in prof.values()) or 1e-9
    g_ms = sum(prof[f]["time_ms"] for f in gemm_fams)
    g_flops = sum(prof[f]["flops"] for f in gemm_fams)
    g_launch = sum(prof[f]["launches"] for f in gemm_fams)
    g_bytes = sum(prof[f]["bytes"] for f in gemm_fams)
    achieved = g_flops / (g_ms / 1e3) / 1e12 if g_ms > 0 else None
    traffic = gemm_traffic_record()
    roofline = {"bound": "tensor", "kernel": "k_gemm_pair (QKV/O/gate-up/down projections on CTA pairs)",
                "achieved": achieved, "peak": peaks["bf16_tflops_sustained"], "unit": "TFLOP/s",
                "frac": (achieved / peaks["bf16_tflops_sustained"]) if achieved else None,
                "peak_source": f"{peaks['source']} sustained bf16 (kernel timed inside a long step)",
                "traffic": (traffic["traffic_over_algorithmic"] * g_bytes / max(g_launch, 1) if traffic else None),
                "algorithmic_flops_per_launch": g_flops / max(g_launch, 1),
                "algorithmic_bytes_per_launch": g_bytes / max(g_launch, 1),
                "share_of_step": g_ms / tot_ms}
    kernels = kernel_table(prof, args.steps, peaks)
    gpu_launches = sum(v["launches"] for v in prof.values())

    # ---------------- CPU baseline: the oracle on a bounded sample, rank 0, N = 1
    cpu = parity = None
    if want_cpu:
        # the oracle on a length-stratified sample of the workload's first batch (the same
        # pairs as the reference arm), compared with the GPU scores of that batch
        b0 = batches[0]
        gpu_scores = step_dev(b0).cpu().numpy()
        idx = stratified_pairs(wl, pairs, Q, CPU_SAMPLE_PAIRS)
        got, secs, threads = oracle_sample(wl, w_host, doc_m, pairs, idx, args.seed, args.cpu_seconds, dev)
        toks = oracle_sample.tokens
        lens = [int(pairs["q_offsets"][p + 1] - pairs["q_offsets"][p]) for p in got]
        cpu = {"value": len(got) / secs, "unit": "pairs/s", "cores": threads, "kind": "oracle",
               "tokens_per_s": toks / secs,
               "sample": f"{len(got)} pair(s), one per query at evenly spaced length quantiles of the first "
                         f"batch (query lengths {lens}), fp64 C oracle, {secs:.1f} s of scoring (prefix draws "
                         f"and host copies untimed)"}
        diffs = [abs(float(gpu_scores[p - b0["first_pair"]]) - s) for p, s in got.items()]
        parity = {"pairs": len(diffs), "max_abs_diff": max(diffs), "tolerance": 3e-2,
                  "oracle_scores": [round(s, 5) for s in got.values()]}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "pairs/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": statistics.mean(step_ms),
            "p50_batch_ms": statistics.median(step_ms), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f16",
            "data": "synthetic: seeded random-init bf16 weights N(0,0.02), N(0,1) prefix K/V, uniform token ids",
            "config": {"workload": wl.name,
                       "decoder": f"{wl.model.name}: {wl.model.n_layers} layers, hidden {wl.model.hidden}, "
                                f"{wl.model.n_q_heads}/{wl.model.n_kv_heads} heads, head_dim 128, ffn {wl.model.ffn}",
                       "docs": wl.n_docs, "m": list(wl.m_choices), "fulldoc_tokens": wl.fulldoc_tokens,
                       "pairs_per_step": Q * per_q, "queries_per_step": Q, "query_len": [wl.qlen_min, wl.qlen_max],
                       "candidates": "Zipf(%.1f)" % wl.zipf_s if wl.zipf_s else "uniform",
                       "parallelism": f"replicas x{world} (pairs sharded by query)",
                       "l2": (f"L2 flushed between timed steps ({L2_FLUSH_BYTES >> 20} MiB written outside the "
                              f"events); {stream_bytes / 1e9:.2f} GB streamed per step" if flush is not None else
                              f"inputs larger than L2 ({stream_bytes / 1e9:.2f} GB of weights streamed per step)")},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": gpu_launches,
            "clocks": clk,
            "latency": {"per_query_pairs": per_q, "p50_ms": lat_sorted[len(lat_sorted) // 2] if lat_sorted else None,
                        "p90_ms": lat_sorted[int(0.9 * (len(lat_sorted) - 1))] if lat_sorted else None},
            "kernels": kernels, "parity": parity,
        }
        if not args.no_configs and world == 1:
            # every configuration, bounded, after the headline (its store freed; its model
            # reused by the other Qwen3-8B arms, else freed too)
            store.close()
            reuse = wl.model.name == "qwen3-8b"
            if not reuse:
                model.close()
            torch.cuda.empty_cache()
            line["configs"] = run_configs(args, dev, local_rank, {"workload": wl.name, "value": value},
                                          model if reuse else None, cfg)
        print(json.dumps(line))


def run_reuse(args):
    """Controlled cross-query reuse (the paper's amortised speedup): one document
    scored for r queries costs r * T_full uncompressed and T_off + r * T_online with
    DoPR, Speedup(r) = r T_full / (T_off + r T_online).  Measured on the workload's
    model: T_online per pair on its compressed prefixes, T_full per pair on
    [document tokens ; query ; t_score] with no prefix, and T_off per document =
    the key token selection over its tokens (a document-only pass and the
    salience ranking) + the prefix build over its m selected representations."""
    import torch

    from paper_2609_03311_gb300 import dopr, synth

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wl = synth.WORKLOADS[args.workload]
    full_wl = synth.WORKLOADS["qwen3-8b-fulldoc"] if wl.model.name == "qwen3-8b" else wl
    n_doc_tokens = full_wl.fulldoc_tokens or 512
    cfg, model, store, doc_m, _ = setup(wl, args.seed, dev, False)
    s = wl.model
    empty = dopr.Store(cfg, wl.n_docs - 1, 1 << 16)  # every document with m = 0
    for d in range(wl.n_docs):
        z = torch.zeros((s.n_layers, 0, s.n_kv_heads, s.head_dim), dtype=torch.bfloat16)
        empty.put(d, z, z)
    pairs = synth.make_workload_pairs(wl, seed=args.seed)
    per_q = wl.docs_per_query

    def timed(fn, reps):
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        return statistics.median(ts)

    def dev_batch(b):
        return (torch.tensor(b["q_offsets"], device=dev), torch.tensor(b["q_tokens"], device=dev),
                torch.tensor(b["doc_ids"], device=dev))

    # T_online: 20 queries' candidate lists against the compressed prefixes
    n_on = 20 * per_q
    on = dev_batch(slice_pairs(pairs, 0, n_on))
    t_online = timed(lambda: dopr.score(model, store, *on), args.steps) / n_on
    # T_full: 2 queries' lists as [document tokens ; query]
    n_full = 2 * per_q
    full_pairs = build_pairs(full_wl, args.seed) if full_wl is not wl else None
    if full_pairs is None:
        raise SystemExit("--reuse needs the 8B workload family")
    fb = dev_batch(slice_pairs(full_pairs, 0, n_full))
    t_full = timed(lambda: dopr.score(model, empty, *fb), max(1, args.steps // 2)) / n_full
    # T_off: the offline construction of 100 documents -- key token selection (a
    # document-only pass over their tokens, Sec. 3.2.1; p left open by the paper:
    # the column mean) and the prefix build over the selected representations
    docs = np.arange(100, dtype=np.int64)
    toks = [synth.make_fulldoc_tokens(full_wl, int(d), seed=args.seed) for d in docs]
    qo = np.concatenate([[0], np.cumsum([len(t) for t in toks])]).astype(np.int32)
    all_toks = np.concatenate(toks)
    m = int(doc_m[0])
    sel = {}

    def select():
        sel["pos"], sel["x"], _ = dopr.select_prefix_inputs(model, qo, all_toks, m, 1 << 30)

    t_doc = timed(select, args.steps) / len(docs)
    bstore = dopr.Store(cfg, len(docs) - 1, len(docs) * dopr.prefix_bytes(cfg, m))
    x = sel["x"].reshape(-1, s.hidden).to(dev)
    offs = np.arange(0, m * len(docs) + 1, m, dtype=np.int32)
    t_build = timed(lambda: dopr.build_prefixes(model, bstore, docs, offs, x), args.steps) / len(docs)
    t_off = t_doc + t_build
    rs = [1, 2, 4, 8, 16, 32, 64, 128]
    print(json.dumps({
        "metric": "amortised speedup under document reuse, r T_full / (T_off + r T_online)", "unit": "x",
        "config": {"workload": wl.name, "decoder": s.name, "m": m, "document_tokens": n_doc_tokens,
                   "online_pairs": n_on, "full_pairs": n_full, "offline_documents": len(docs)},
        "t_online_ms_per_pair": t_online, "t_full_ms_per_pair": t_full,
        "t_off_ms_per_doc": t_off, "t_off_parts_ms": {"key_token_selection": t_doc, "prefix_build": t_build},
        "speedup": {str(r): r * t_full / (t_off + r * t_online) for r in rs},
        "speedup_limit": t_full / t_online, "data": "synthetic", "dtype": "f16",
    }))


def run_reference(args, rank, world):
    """The oracle alone, on the host cores, on bounded samples of the workload."""
    if rank != 0:
        return
    import torch

    from paper_2609_03311_gb300 import synth

    wl = synth.WORKLOADS[args.workload]
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    w = synth.make_weights(wl.model, seed=args.seed, device=dev, norms="ones")
    w_host = {k: (v.cpu() if isinstance(v, torch.Tensor) else [t.cpu() for t in v]) for k, v in w.items()}
    del w
    doc_m = synth.doc_prefix_lengths(wl, seed=args.seed)
    pairs = build_pairs(wl, args.seed)
    n_total = args.warmup + args.steps
    # one pair per step, cycling through the GPU arm's length-stratified sample
    sample = stratified_pairs(wl, pairs, min(args.queries_per_step, wl.n_queries), CPU_SAMPLE_PAIRS)
    for i in range(args.warmup):
        oracle_sample(wl, w_host, doc_m, pairs, [sample[i % len(sample)]], args.seed, 0.0, dev)
    done, secs, toks, threads = 0, 0.0, 0, 1
    for i in range(args.steps):
        got, t, threads = oracle_sample(wl, w_host, doc_m, pairs, [sample[(args.warmup + i) % len(sample)]],
                                        args.seed, 0.0, dev)
        done += len(got)
        secs += t
        toks += oracle_sample.tokens
    value = done / secs
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "pairs/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic: seeded random-init bf16 weights, N(0,1) prefix K/V, uniform token ids",
        "config": {"workload": wl.name, "pairs_per_step": 1, "steps_total": n_total},
        "cpu_baseline": {"value": value, "unit": "pairs/s", "cores": threads, "kind": "oracle",
                         "tokens_per_s": toks / secs,
                         "sample": f"{done} pair(s), one per step, cycling through {len(sample)} pairs at evenly "
                                   f"spaced query-length quantiles of the first batch; fp64 C oracle, scoring "
                                   f"timed alone"},
        "e2e": {"value": value, "unit": "pairs/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def main():
    args = parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch
        import torch.distributed as tdist

        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local_rank)
        tdist.init_process_group(backend=backend)
        dist = tdist
    if args.reuse:
        run_reuse(args)
    elif args.impl == "reference":
        run_reference(args, rank, world)
    else:
        run_dopr(args, rank, world, local_rank, dist)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
