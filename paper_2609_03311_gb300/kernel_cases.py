"""Stand-alone kernel cases for profiling (ncu) and quick timing.

    python -m paper_2609_03311_gb300.kernel_cases projections --model qwen3-8b --m 24576
        the four projection GEMMs of one decoder layer at M = m tokens
        (QKV / O +residual / gate-up +SwiGLU / down +residual), each once per rep
    python -m paper_2609_03311_gb300.kernel_cases score --workload qwen3-8b-m64 --layers 2 --pairs 2000
        a scoring pass of the workload's first `pairs` pairs through a model cut
        to `layers` layers (keeps the device footprint to a few GB)

Each case prints CUDA-event times; run under ncu with -k to capture one kernel.
"""
from __future__ import annotations

import argparse
import json

import numpy as np
import torch

from . import dopr, synth


def projections(args):
    s = synth.MODELS[args.model]
    H, F = s.hidden, s.ffn
    qkv = (s.n_q_heads + 2 * s.n_kv_heads) * s.head_dim
    o = s.n_q_heads * s.head_dim
    M = args.m
    g = torch.Generator(device="cuda").manual_seed(0)

    def rnd(r, c, std):
        return (std * torch.randn(r, c, device="cuda", generator=g)).to(torch.float16)

    cases = [("qkv", rnd(M, H, 1.0), rnd(qkv, H, 0.02), dopr.EPI_STORE),
             ("o", rnd(M, o, 1.0), rnd(H, o, 0.02), dopr.EPI_RESID_ADD),
             ("gate_up", rnd(M, H, 1.0), rnd(2 * F, H, 0.02), dopr.EPI_SWIGLU),
             ("down", rnd(M, F, 1.0), rnd(H, F, 0.02), dopr.EPI_RESID_ADD)]
    out = {}
    for name, A, B, epi in cases:
        res = None
        ms = []
        for _ in range(args.reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            if epi == dopr.EPI_RESID_ADD:
                res = torch.zeros(M, B.shape[0], device="cuda")
            e0.record()
            dopr.gemm(A, B, epi, out=res)
            e1.record()
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
        flops = 2.0 * M * B.shape[0] * A.shape[1]
        out[name] = {"M": M, "N": B.shape[0], "K": A.shape[1], "ms": min(ms), "tflops": flops / min(ms) / 1e9}
    print(json.dumps(out))


def score(args):
    wl = synth.WORKLOADS[args.workload]
    s = wl.model.with_layers(args.layers)
    w = synth.make_weights(s, seed=0, device="cuda")
    cfg = dopr.make_config(s, max_position=1024)
    model = dopr.Model(cfg, w)
    del w
    doc_m = synth.doc_prefix_lengths(wl)
    store = dopr.Store(cfg, wl.n_docs - 1, sum(dopr.prefix_bytes(cfg, int(m)) for m in doc_m) + (1 << 20))
    for d in range(wl.n_docs):
        store.put(d, *synth.make_prefix(s, int(doc_m[d]), d, device="cuda"))
    pairs = synth.make_workload_pairs(wl)
    n = min(args.pairs, len(pairs["doc_ids"]))
    qo = torch.tensor(pairs["q_offsets"][:n + 1], device="cuda")
    qt = torch.tensor(pairs["q_tokens"][:int(pairs["q_offsets"][n])], device="cuda")
    di = torch.tensor(pairs["doc_ids"][:n], device="cuda")
    for _ in range(args.reps):
        dopr.profile_enable(model, True)
        dopr.score(model, store, qo, qt, di)
        torch.cuda.synchronize()
        prof = dopr.profile_read(model)
    print(json.dumps({k: v for k, v in prof.items() if v["launches"]}))


def main():
    ap = argparse.ArgumentParser()
    sub = ap.add_subparsers(dest="case", required=True)
    p = sub.add_parser("projections")
    p.add_argument("--model", default="qwen3-8b")
    p.add_argument("--m", type=int, default=24576)
    p.add_argument("--reps", type=int, default=1)
    p = sub.add_parser("score")
    p.add_argument("--workload", default="qwen3-8b-m64")
    p.add_argument("--layers", type=int, default=2)
    p.add_argument("--pairs", type=int, default=2000)
    p.add_argument("--reps", type=int, default=2)
    args = ap.parse_args()
    {"projections": projections, "score": score}[args.case](args)


if __name__ == "__main__":
    main()
