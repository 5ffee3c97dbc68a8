"""Offline prefix construction on the GPU (dopr_build_prefixes) against the
fp64 oracle (Sec. 3.3; Sec. 3.4 footnote: the stored states are the
multi-layer keys/values of forwarding the selected representations as prefix
inputs).

Bars:
  * stored K/V, element by element, within 2e-2 + 2e-2 |ref| of the oracle's
    causal pass over the same bf16 vectors -- the stored values are fp16
    (2^-11 relative) computed from fp16 operands with fp32 accumulation over a
    few layers, a few 1e-3 relative in all; the margin covers the rotated and
    normalised keys of magnitude up to ~4;
  * scores against GPU-built prefixes within 3e-2 of the oracle scoring
    against oracle-built prefixes;
  * one batch or one document at a time: identical stored bytes.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_03311_gb300 import dopr, synth

pytestmark = pytest.mark.gpu
TOL = 3e-2

SHAPE = synth.ModelShape("build-g4", n_layers=3, hidden=512, n_q_heads=8, n_kv_heads=2, head_dim=128, ffn=640,
                         vocab=777)
SHAPE_G2 = synth.ModelShape("build-g2", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=128, ffn=384,
                            vocab=1000)
DOC_M = {3: 1, 5: 7, 8: 64, 9: 130, 12: 256, 14: 33}


def oshape(s):
    return oracle.Shape(s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn, s.vocab, s.rope_theta,
                        s.rms_eps, s.score_token_id)


class BuildRig:
    def __init__(self, shape, doc_m, seed):
        self.shape = shape
        self.w = synth.make_weights(shape, seed=seed, norms="random")
        self.cfg = dopr.make_config(shape, max_position=1024)
        self.model = dopr.Model(self.cfg, self.w)
        self.doc_m = doc_m
        self.ids, self.offs, self.x = synth.make_doc_representations(shape, doc_m, seed=seed)
        self.om = oracle.OracleModel(oshape(shape), self.w)

    def store(self, extra=0):
        pool = sum(dopr.prefix_bytes(self.cfg, m) for m in self.doc_m.values()) + extra
        return dopr.Store(self.cfg, max(self.doc_m) + 1, max(pool, 256))

    def oracle_kv(self, d):
        i = list(self.ids).index(d)
        xd = oracle.bf16_to_f64(self.x[self.offs[i]:self.offs[i + 1]])
        out = self.om.forward(xd, 0, want_kv=True)
        return out["k"], out["v"]  # [L, m, Hkv, D]


@pytest.mark.parametrize("shape", [SHAPE, SHAPE_G2], ids=["g4", "g2"])
def test_built_keys_values_match_oracle(shape):
    rig = BuildRig(shape, DOC_M, seed=31)
    store = rig.store()
    dopr.build_prefixes(rig.model, store, rig.ids, rig.offs, rig.x.cuda())
    worst = 0.0
    for d, m in DOC_M.items():
        rk, rv = rig.oracle_kv(d)
        for l in range(shape.n_layers):
            k, v = store.read_layer(d, l, m)
            for got, ref in ((k, rk[l]), (v, rv[l])):
                err = np.abs(got.astype(np.float64) - ref)
                assert np.all(err <= 2e-2 + 2e-2 * np.abs(ref)), (d, l, float(err.max()))
                worst = max(worst, float(err.max()))
    assert worst > 0.0  # the comparison saw real data


def test_scores_against_built_prefixes_match_oracle():
    rig = BuildRig(SHAPE, DOC_M, seed=32)
    store = rig.store()
    dopr.build_prefixes(rig.model, store, rig.ids, rig.offs, rig.x)  # host input path
    rng = np.random.default_rng(32)
    docs = np.asarray(sorted(DOC_M), np.int64)
    n = 24
    di = rng.choice(docs, size=n)
    lens = rng.integers(0, 40, size=n)
    qo = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    qt = rng.integers(0, SHAPE.vocab, size=int(qo[-1])).astype(np.int32)
    got = dopr.score(rig.model, store, qo, qt, di).numpy()
    kv = {d: rig.oracle_kv(d) for d in DOC_M}
    keys = sorted(DOC_M)
    ref = rig.om.score_pairs(qo, qt, [keys.index(int(d)) for d in di], [kv[d] for d in keys])
    assert np.max(np.abs(got - ref)) <= TOL, np.max(np.abs(got - ref))


def test_one_batch_equals_one_document_at_a_time():
    rig = BuildRig(SHAPE, DOC_M, seed=33)
    a, b = rig.store(), rig.store()
    dopr.build_prefixes(rig.model, a, rig.ids, rig.offs, rig.x.cuda())
    for i, d in enumerate(rig.ids):
        dopr.build_prefixes(rig.model, b, [d], np.array([0, rig.offs[i + 1] - rig.offs[i]], np.int32),
                            rig.x[rig.offs[i]:rig.offs[i + 1]].cuda())
    for d, m in DOC_M.items():
        for l in range(SHAPE.n_layers):
            ka, va = a.read_layer(d, l, m)
            kb, vb = b.read_layer(d, l, m)
            np.testing.assert_array_equal(ka.view(np.uint16), kb.view(np.uint16))
            np.testing.assert_array_equal(va.view(np.uint16), vb.view(np.uint16))


def test_build_errors_and_empty_prefix():
    rig = BuildRig(SHAPE_G2, {2: 5, 4: 0}, seed=34)
    store = rig.store()
    x = rig.x.cuda()
    with pytest.raises(dopr.DoprError) as ei:  # a doc id twice
        dopr.build_prefixes(rig.model, store, [2, 2], np.array([0, 2, 5], np.int32), x)
    assert ei.value.status == dopr.ERR_INVALID_ARG
    big = torch.zeros((257, SHAPE_G2.hidden), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(dopr.DoprError) as ei:  # m above 256
        dopr.build_prefixes(rig.model, store, [2], np.array([0, 257], np.int32), big)
    assert ei.value.status == dopr.ERR_INVALID_ARG
    dopr.build_prefixes(rig.model, store, rig.ids, rig.offs, x)
    with pytest.raises(dopr.DoprError) as ei:  # rebuilt with another m
        dopr.build_prefixes(rig.model, store, [2], np.array([0, 4], np.int32), x[:4])
    assert ei.value.status == dopr.ERR_INVALID_ARG
    tiny = dopr.Store(rig.cfg, 8, dopr.prefix_bytes(rig.cfg, 5) - 256)
    with pytest.raises(dopr.DoprError) as ei:  # pool too small
        dopr.build_prefixes(rig.model, tiny, [2], np.array([0, 5], np.int32), x[:5])
    assert ei.value.status == dopr.ERR_OUT_OF_MEMORY
    # doc 4 has m = 0: its pass is the query-only forward
    q = np.arange(9, dtype=np.int32)
    got = dopr.score(rig.model, store, np.array([0, 9], np.int32), q, np.array([4], np.int64)).numpy()[0]
    full = rig.om.forward(rig.om.embed(np.concatenate([q, [SHAPE_G2.score_token_id]])), 0)["h"]
    assert abs(got - rig.om.score_head(full[-1])) <= TOL
