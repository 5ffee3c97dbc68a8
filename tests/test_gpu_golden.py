"""Full-size parity against stored oracle scores.

tests/golden/fullsize_<workload>.json holds fp64 oracle scores that
tests/golden/make_fullsize_scores.py computed on a host (oracle only) for:
the complete 100-candidate list of one Qwen3-8B query (m = 64), the complete
list of the longest first-batch query of the Zipf workload (m 32..256), and
24 candidates of the longest first-batch Qwen3-4B query (>= 200 tokens).
Here the same bytes are rebuilt (portable host draws; their fingerprints must
match the stored ones), the bench's first batch (20 queries' candidate lists)
is scored in one dopr_score call, and every stored pair must be within 3e-2
of its oracle score, with the top-10 order of the oracle kept wherever the
oracle's adjacent gap exceeds 0.1 (Sec. 3.1 pointwise scores, Sec. 4.4
ranking).
"""
import json
import os
import sys
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

from paper_2609_03311_gb300 import dopr, synth

pytestmark = pytest.mark.gpu
TOL = 3e-2
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
sys.path.insert(0, GOLDEN)
import make_fullsize_scores as mk  # noqa: E402  (fingerprints and the case definitions)


def _load(name):
    rec = json.load(open(os.path.join(GOLDEN, f"fullsize_{name}.json")))
    assert rec.get("complete"), f"{name}: stored scores incomplete"
    return rec


_MODELS = {}


def _model(shape):
    """Portable weights of `shape` (seed 0) on the host, fingerprinted, and the device model."""
    if shape.name not in _MODELS:
        for k in list(_MODELS):  # one full-size model resident at a time
            _MODELS.pop(k)[1].close()
        w = synth.make_weights(shape, seed=mk.SEED, device="cpu", norms="ones", portable=True)
        fp = mk.weights_fingerprint(w)
        cfg = dopr.make_config(shape, max_position=1024)
        _MODELS[shape.name] = (cfg, dopr.Model(cfg, w), fp)
        del w
    return _MODELS[shape.name]


@pytest.mark.parametrize("name", ["qwen3-8b-m64", "qwen3-8b-zipf", "qwen3-4b"])
def test_full_size_scores_match_stored_oracle(name):
    rec = _load(name)
    wl = synth.WORKLOADS[name]
    s = wl.model
    cfg, model, wfp = _model(s)
    assert wfp == rec["weights_fingerprint"], "the host generator did not rebuild the stored weights"
    pairs, q, idx = mk.case_pairs(name)
    assert idx == rec["pairs"] and q == rec["query"]
    per_q = wl.docs_per_query
    n = mk.BATCH_QUERIES * per_q
    qo = pairs["q_offsets"][:n + 1].astype(np.int32)
    qt = pairs["q_tokens"][:qo[-1]].astype(np.int32)
    di = pairs["doc_ids"][:n].astype(np.int64)
    doc_m = synth.doc_prefix_lengths(wl, seed=mk.SEED)
    docs = sorted(set(int(d) for d in di))
    store = dopr.Store(cfg, wl.n_docs - 1, sum(dopr.prefix_bytes(cfg, int(doc_m[d])) for d in docs) + (1 << 20))

    def draw(d):
        return d, synth.make_prefix(s, int(doc_m[d]), d, seed=mk.SEED, portable=True)

    golden_docs = set(rec["doc_ids"])
    with ThreadPoolExecutor(max_workers=max(1, min(32, os.cpu_count() or 1))) as ex:
        for d, (k, v) in ex.map(draw, docs):
            if d in golden_docs:
                got_fp = mk.hashlib.sha256((mk.fingerprint(k) + mk.fingerprint(v)).encode()).hexdigest()[:32]
                assert got_fp == rec["prefix_fingerprint"][str(d)], f"doc {d}: prefix bytes differ"
            store.put(d, k, v)
    dev = torch.device("cuda")
    got = dopr.score(model, store, torch.tensor(qo, device=dev), torch.tensor(qt, device=dev),
                     torch.tensor(di, device=dev)).cpu().numpy()
    store.close()
    ref = np.array([rec["scores"][str(p)] for p in idx])
    g = got[idx].astype(np.float64)
    d = np.abs(g - ref)
    print(f"{name}: {len(idx)} pairs, |score - oracle| max {d.max():.4f} p99 {np.quantile(d, 0.99):.4f} "
          f"mean {d.mean():.4f}")
    assert np.all(np.isfinite(g))
    assert d.max() <= TOL, (float(d.max()), int(idx[int(np.argmax(d))]))
    order = np.argsort(-ref, kind="stable")[:10]
    for a, c in zip(order[:-1], order[1:]):
        if ref[a] - ref[c] > 0.1:
            assert g[a] > g[c], (int(idx[a]), int(idx[c]))


def teardown_module(module):
    for k in list(_MODELS):
        _MODELS.pop(k)[1].close()
