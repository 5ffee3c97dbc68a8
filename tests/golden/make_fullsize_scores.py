"""Write the stored oracle scores of the full-size parity cases.

Calls only the fp64 oracle (``oracle/``) and the seeded input generators
(``paper_2609_03311_gb300.synth``, which hold none of the scoring
arithmetic).  Inputs are drawn with ``portable=True`` (float64 host draws,
rounded to bf16), so the GPU test that reads these files rebuilds the very
same bytes on its own host; a fingerprint of every input tensor is stored
beside the scores and checked there first.

Cases (seed 0, the bench's first batch of each workload = queries 0..19):
  qwen3-8b-m64   the complete 100-candidate list of the batch's median-length query
  qwen3-8b-zipf  the complete 100-candidate list of the batch's longest query
                 (prefix lengths 32..256)
  qwen3-4b       the first 24 candidates of the batch's longest query
                 (a BRIGHT-like query of >= 200 tokens)

    python tests/golden/make_fullsize_scores.py [case ...]

Each case is written to tests/golden/fullsize_<case>.json (and resumes from a
partial file of the same case).  This takes tens of minutes of CPU per case.
"""
from __future__ import annotations

import hashlib
import json
import os
import sys
import time

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2609_03311_gb300 import synth  # noqa: E402

SEED = 0
BATCH_QUERIES = 20  # the bench's default step: 20 queries' candidate lists
CASES = {
    "qwen3-8b-m64": {"pick": "median", "n_cand": None},
    "qwen3-8b-zipf": {"pick": "longest", "n_cand": None},
    "qwen3-4b": {"pick": "longest", "n_cand": 24},
}


def fingerprint(t: torch.Tensor) -> str:
    """sha256 over a tensor's shape and bf16 bytes (every element)."""
    h = hashlib.sha256(str(tuple(t.shape)).encode())
    h.update(memoryview(np.ascontiguousarray(t.contiguous().view(torch.int16).numpy())))
    return h.hexdigest()[:32]


def weights_fingerprint(w: dict) -> str:
    """Digest of every weight tensor's fingerprint, in name order (hashed in threads)."""
    from concurrent.futures import ThreadPoolExecutor

    ts = [t for k in sorted(w) for t in (w[k] if isinstance(w[k], list) else [w[k]])]
    with ThreadPoolExecutor(max_workers=max(1, min(32, os.cpu_count() or 1))) as ex:
        fps = list(ex.map(fingerprint, ts))
    h = hashlib.sha256()
    for f in fps:
        h.update(f.encode())
    return h.hexdigest()[:32]


def case_pairs(name: str):
    """Pair indices (into the workload's pair list) of the case, and the query index."""
    wl = synth.WORKLOADS[name]
    pairs = synth.make_workload_pairs(wl, seed=SEED)
    k = wl.docs_per_query
    lens = np.diff(pairs["q_offsets"])[::k][:BATCH_QUERIES]  # one length per query of the first batch
    if CASES[name]["pick"] == "longest":
        q = int(np.argmax(lens))
    else:
        q = int(np.argsort(lens, kind="stable")[len(lens) // 2])
    n = CASES[name]["n_cand"] or k
    return pairs, q, list(range(q * k, q * k + n))


def oshape(s):
    return oracle.Shape(s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn, s.vocab, s.rope_theta,
                        s.rms_eps, s.score_token_id)


def run(name: str, block: int = 8):
    wl = synth.WORKLOADS[name]
    s = wl.model
    out_path = os.path.join(HERE, f"fullsize_{name}.json")
    pairs, q, idx = case_pairs(name)
    doc_m = synth.doc_prefix_lengths(wl, seed=SEED)
    rec = {"workload": name, "seed": SEED, "generator": "synth portable (float64 host draws -> bf16)",
           "batch_queries": BATCH_QUERIES, "query": q, "pairs": idx,
           "doc_ids": [int(pairs["doc_ids"][p]) for p in idx],
           "m": [int(doc_m[int(pairs["doc_ids"][p])]) for p in idx],
           "query_len": int(pairs["q_offsets"][idx[0] + 1] - pairs["q_offsets"][idx[0]]),
           "scores": {}, "prefix_fingerprint": {}}
    if os.path.exists(out_path):
        old = json.load(open(out_path))
        if old.get("pairs") == idx:
            rec["scores"] = old.get("scores", {})
            rec["prefix_fingerprint"] = old.get("prefix_fingerprint", {})
    t0 = time.time()
    w = synth.make_weights(s, seed=SEED, device="cpu", norms="ones", portable=True)
    rec["weights_fingerprint"] = weights_fingerprint(w)
    print(f"{name}: weights drawn in {time.time() - t0:.0f} s; query {q} (len {rec['query_len']}), "
          f"{len(idx)} pairs, {oracle.num_threads()} threads", flush=True)
    om = oracle.OracleModel(oshape(s), w)
    todo = [p for p in idx if str(p) not in rec["scores"]]
    for b in range(0, len(todo), block):
        part = todo[b:b + block]
        t1 = time.time()
        docs, qo, qt, pd = [], [0], [], []
        for i, p in enumerate(part):
            d = int(pairs["doc_ids"][p])
            k, v = synth.make_prefix(s, int(doc_m[d]), d, seed=SEED, portable=True)
            rec["prefix_fingerprint"][str(d)] = hashlib.sha256(
                (fingerprint(k) + fingerprint(v)).encode()).hexdigest()[:32]
            docs.append((k, v))
            a, e = pairs["q_offsets"][p], pairs["q_offsets"][p + 1]
            qt.append(pairs["q_tokens"][a:e])
            qo.append(qo[-1] + e - a)
            pd.append(i)
        sc = om.score_pairs(np.asarray(qo, np.int32), np.concatenate(qt).astype(np.int32), pd, docs)
        for p, x in zip(part, sc):
            rec["scores"][str(p)] = float(x)
        rec["oracle_seconds"] = rec.get("oracle_seconds", 0.0) + time.time() - t1
        json.dump(rec, open(out_path + ".tmp", "w"), indent=1)
        os.replace(out_path + ".tmp", out_path)
        print(f"  {len(rec['scores'])}/{len(idx)} pairs, {time.time() - t1:.0f} s for {len(part)}", flush=True)
    rec["complete"] = len(rec["scores"]) == len(idx)
    json.dump(rec, open(out_path + ".tmp", "w"), indent=1)
    os.replace(out_path + ".tmp", out_path)


if __name__ == "__main__":
    for c in (sys.argv[1:] or list(CASES)):
        run(c)
