"""The optional MLP scoring head (Sec. 3.2.3) on the GPU against the fp64
oracle: scores within 3e-2 for each activation, and the yes/no rows again
once the head is removed."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_03311_gb300 import dopr, synth

pytestmark = pytest.mark.gpu
TOL = 3e-2
SHAPE = synth.ModelShape("head-g4", n_layers=2, hidden=512, n_q_heads=8, n_kv_heads=2, head_dim=128, ffn=640,
                         vocab=777)


def _head(d, H, seed, act):
    rng = np.random.default_rng(seed)
    bf = lambda a: torch.tensor(a, dtype=torch.float32).to(torch.bfloat16)
    return {"w1": bf(rng.normal(0, 0.05, size=(d, H))), "b1": bf(rng.normal(0, 0.1, size=d)),
            "w2": bf(rng.normal(0, 0.1, size=d)), "b2": 0.25, "act": act}


@pytest.mark.parametrize("act", [0, 1, 2, 3])
def test_mlp_head_scores_match_oracle(act):
    s = SHAPE
    w = synth.make_weights(s, seed=51, norms="random")
    cfg = dopr.make_config(s, max_position=1024)
    model = dopr.Model(cfg, w)
    om = oracle.OracleModel(oracle.Shape(s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn,
                                         s.vocab, s.rope_theta, s.rms_eps, s.score_token_id), w)
    doc_m = {0: 0, 1: 40, 2: 64}
    store = dopr.Store(cfg, 2, sum(dopr.prefix_bytes(cfg, m) for m in doc_m.values()) + 4096)
    docs = {}
    for d, m in doc_m.items():
        k, v = synth.make_prefix(s, m, d, seed=51)
        store.put(d, k, v)
        docs[d] = (oracle.bf16_to_f64(k), oracle.bf16_to_f64(v))
    head = _head(96, s.hidden, 51 + act, act)
    dopr.set_mlp_head(model, head)
    rng = np.random.default_rng(51)
    n = 10
    di = rng.integers(0, 3, size=n).astype(np.int64)
    ql = rng.integers(0, 20, size=n)
    qo = np.concatenate([[0], np.cumsum(ql)]).astype(np.int32)
    qt = rng.integers(0, s.vocab, size=int(qo[-1])).astype(np.int32)
    got = dopr.score(model, store, qo, qt, di).numpy()
    ref = []
    for p in range(n):
        ids = np.concatenate([qt[qo[p]:qo[p + 1]], [s.score_token_id]])
        m = doc_m[int(di[p])]
        k, v = docs[int(di[p])]
        h = om.forward(om.embed(ids), m, k if m else None, v if m else None)["h"]
        ref.append(om.mlp_head(h[-1], head))
    assert np.max(np.abs(got - np.array(ref))) <= TOL, np.max(np.abs(got - np.array(ref)))
    # removing the head gives the yes/no rows back
    dopr.set_mlp_head(model, None)
    got2 = dopr.score(model, store, qo, qt, di).numpy()
    keys = sorted(doc_m)
    ref2 = om.score_pairs(qo, qt, [keys.index(int(d)) for d in di], [docs[d] for d in keys])
    assert np.max(np.abs(got2 - ref2)) <= TOL
    model.close()
    store.close()
