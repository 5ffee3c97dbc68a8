"""The fp16 operand range of the scoring path.

The tensor cores take fp16 operands (three more mantissa bits than the
paper's bf16, Tab. 7, but a range that ends at 65,504).  Values outside that
range must never turn into a silent inf/NaN score: weights that do not fit
are refused when they are put, and every kernel that writes an fp16 operand
(the normed activations, q/k/v, the SwiGLU output, the attention output) or a
score flags a value that is not finite or exceeds 65,504, which the call
reports as DOPR_ERR_RANGE.  Heavy-tailed but representable inputs (large norm
gains, outlier residual channels, a few large weights) either match the
oracle within 3e-2 or fail with that status.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_03311_gb300 import dopr, synth

pytestmark = pytest.mark.gpu
TOL = 3e-2

SHAPE = synth.ModelShape("range", n_layers=3, hidden=512, n_q_heads=8, n_kv_heads=2, head_dim=128, ffn=640,
                         vocab=500)


def _oshape(s):
    return oracle.Shape(s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn, s.vocab, s.rope_theta,
                        s.rms_eps, s.score_token_id)


def _bf16(x):
    return torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)


def _heavy_weights(seed):
    """Trained-checkpoint-like magnitudes: norm gains 10..50, four residual channels
    of the embedding at 1e3..1e4, and a few entries of every projection at 1..4."""
    s = SHAPE
    w = synth.make_weights(s, seed=seed, norms="random")
    rng = np.random.default_rng(seed)
    for key in ("attn_norm", "mlp_norm"):
        w[key] = [_bf16(rng.uniform(10, 50, size=s.hidden)) for _ in range(s.n_layers)]
    emb = w["embed"].float().numpy().copy()
    ch = rng.choice(s.hidden, size=4, replace=False)
    emb[:, ch] = rng.choice([-1.0, 1.0], size=(s.vocab, 4)) * rng.uniform(1e3, 1e4, size=(s.vocab, 4))
    w["embed"] = _bf16(emb)
    for key in ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down"):
        mats = []
        for m in w[key]:
            a = m.float().numpy().copy()
            idx = rng.choice(a.size, size=8, replace=False)
            a.flat[idx] = rng.choice([-1.0, 1.0], size=8) * rng.uniform(1, 4, size=8)
            mats.append(_bf16(a))
        w[key] = mats
    return w


def _rig(w, doc_m, seed):
    cfg = dopr.make_config(SHAPE, max_position=1024)
    model = dopr.Model(cfg, w)
    store = dopr.Store(cfg, max(doc_m), sum(dopr.prefix_bytes(cfg, m) for m in doc_m.values()) + (1 << 16))
    docs = {}
    for d, m in doc_m.items():
        k, v = synth.make_prefix(SHAPE, m, d, seed=seed)
        store.put(d, k, v)
        docs[d] = (k, v)
    return cfg, model, store, docs


def _pairs(n, doc_m, seed):
    rng = np.random.default_rng(seed)
    lens = rng.integers(0, 40, size=n)
    qo = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    qt = rng.integers(0, SHAPE.vocab, size=int(qo[-1])).astype(np.int32)
    di = rng.choice(sorted(doc_m), size=n).astype(np.int64)
    return qo, qt, di


@pytest.mark.parametrize("bad", [1.0e5, -7.0e4, float("inf"), float("nan")])
@pytest.mark.parametrize("key", ["wq", "w_down"])
def test_weight_outside_fp16_range_is_refused(key, bad):
    w = synth.make_weights(SHAPE, seed=5)
    a = w[key][1].float().clone()
    a[3, 7] = bad
    w[key][1] = a.to(torch.bfloat16)
    with pytest.raises(dopr.DoprError) as ei:
        dopr.Model(dopr.make_config(SHAPE, max_position=1024), w)
    assert ei.value.status == dopr.ERR_INVALID_ARG and "fp16" in str(ei.value)


def test_heavy_tailed_inputs_match_oracle_or_fail_cleanly():
    seed = 11
    doc_m = {0: 0, 1: 17, 2: 64, 3: 130}
    w = _heavy_weights(seed)
    cfg, model, store, docs = _rig(w, doc_m, seed)
    qo, qt, di = _pairs(24, doc_m, seed)
    try:
        got = dopr.score(model, store, qo, qt, di).numpy()
    except dopr.DoprError as e:
        assert e.status == dopr.ERR_RANGE, str(e)
        got = None
    if got is not None:
        assert np.all(np.isfinite(got))
        om = oracle.OracleModel(_oshape(SHAPE), w)
        keys = sorted(doc_m)
        ref = om.score_pairs(qo, qt, [keys.index(int(d)) for d in di], [docs[d] for d in keys])
        assert np.max(np.abs(got - ref)) <= TOL, float(np.max(np.abs(got - ref)))
    model.close()
    store.close()


def test_operand_overflow_is_reported_not_returned():
    # An MLP-norm gain of 6e4 makes the normed operand r * g * rs exceed fp16's range
    # for every entry with |r * rs| > 1.1: the call must fail with DOPR_ERR_RANGE and
    # leave the caller's scores untouched.
    seed = 12
    doc_m = {0: 8, 1: 64}
    w = synth.make_weights(SHAPE, seed=seed, norms="random")
    w["mlp_norm"][0] = _bf16(np.full(SHAPE.hidden, 6.0e4))
    cfg, model, store, docs = _rig(w, doc_m, seed)
    qo, qt, di = _pairs(10, doc_m, seed)
    out = torch.full((10,), -3.0, dtype=torch.float32, device="cuda")
    with pytest.raises(dopr.DoprError) as ei:
        dopr.score(model, store, torch.tensor(qo, device="cuda"), torch.tensor(qt, device="cuda"),
                   torch.tensor(di, device="cuda"), out=out)
    assert ei.value.status == dopr.ERR_RANGE
    # the same model with representable gains still scores (the error word is per call)
    w["mlp_norm"][0] = _bf16(np.full(SHAPE.hidden, 1.5))
    model2 = dopr.Model(cfg, w)
    got = dopr.score(model2, store, qo, qt, di).numpy()
    assert np.all(np.isfinite(got))
    for x in (model, model2, store):
        x.close()
