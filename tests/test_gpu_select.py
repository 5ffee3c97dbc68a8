"""Attention-based key token selection on the GPU (dopr_select_prefix_inputs)
against the fp64 oracle (Sec. 3.2.1, applied offline as in Sec. 3.3).

The GPU recomputes the last layer's attention weights in fp32 from its fp16
q and k, so the salience u agrees with the oracle's fp64 values within
2e-3 + 5e-2 |u| (logit errors of ~1e-2 from fp16 operands move softmax
weights by about that fraction).  The ranking is a decision taken in each
side's own precision, so the selected positions are checked for validity:
no unselected token's oracle salience exceeds a selected one's by more than
the tolerance, and where the oracle's K-th and (K+1)-th values are further
apart than twice the tolerance the sets are identical.  The returned states
match the oracle's final-norm states at those positions within
3e-2 + 3e-2 |ref| (bf16 output, fp16 pass).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_03311_gb300 import dopr, synth

pytestmark = pytest.mark.gpu
TOL = 3e-2

SHAPE = synth.ModelShape("sel-g4", n_layers=3, hidden=512, n_q_heads=8, n_kv_heads=2, head_dim=128, ffn=640,
                         vocab=777)
SHAPE_G2 = synth.ModelShape("sel-g2", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=128, ffn=384,
                            vocab=1000)


def oshape(s):
    return oracle.Shape(s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn, s.vocab, s.rope_theta,
                        s.rms_eps, s.score_token_id)


def _docs(shape, lens, seed):
    rng = np.random.default_rng(seed)
    toks = [rng.integers(0, shape.vocab, size=n).astype(np.int32) for n in lens]
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    return off, np.concatenate(toks), toks


def _u_tol(u):
    return 2e-3 + 5e-2 * np.abs(u)


@pytest.mark.parametrize("shape,top_p", [(SHAPE, 4), (SHAPE, 10 ** 6), (SHAPE_G2, 1)], ids=["g4-p4", "g4-mean", "g2-p1"])
def test_salience_positions_and_states_match_oracle(shape, top_p):
    w = synth.make_weights(shape, seed=41, norms="random")
    model = dopr.Model(dopr.make_config(shape, max_position=4096), w)
    om = oracle.OracleModel(oshape(shape), w)
    lens = [1, 5, 64, 200, 300]
    K = 24
    off, tok, docs = _docs(shape, lens, seed=41)
    pos, x, u = dopr.select_prefix_inputs(model, off, tok, K, top_p)
    g = oracle.bf16_to_f64(w["final_norm"])
    for d, ids in enumerate(docs):
        n = len(ids)
        xo = om.embed(ids)
        out = om.forward(xo, 0, want_probs=True)
        ref_u = oracle.salience(out["probs"], top_p)
        got_u = u[off[d]:off[d + 1]].astype(np.float64)
        assert np.all(np.abs(got_u - ref_u) <= _u_tol(ref_u)), (d, float(np.max(np.abs(got_u - ref_u))))
        k = min(K, n)
        sel = pos[d, :k]
        assert np.all(pos[d, k:] == -1) and np.all(np.diff(sel) > 0)
        tol = _u_tol(ref_u).max()
        rest = np.setdiff1d(np.arange(n), sel)
        if len(rest):
            assert ref_u[rest].max() <= ref_u[sel].min() + 2 * tol, d
        srt = np.sort(ref_u)[::-1]
        if k < n and srt[k - 1] - srt[k] > 2 * tol:
            np.testing.assert_array_equal(sel, oracle.select_topk(ref_u, K))
        want = np.stack([oracle.rmsnorm(out["h"][i], g, shape.rms_eps) for i in sel])
        got = oracle.bf16_to_f64(x[d, :k])
        assert np.all(np.abs(got - want) <= TOL + TOL * np.abs(want)), (d, float(np.max(np.abs(got - want))))
        assert np.all(oracle.bf16_to_f64(x[d, k:]) == 0.0)
    model.close()


def test_selection_at_the_document_length_limit():
    # a 2,048-token document (the longest the selection accepts) next to a short one
    shape = SHAPE_G2
    w = synth.make_weights(shape, seed=44, norms="random")
    model = dopr.Model(dopr.make_config(shape, max_position=4096), w)
    om = oracle.OracleModel(oshape(shape), w)
    lens = [2048, 3]
    K = 64
    off, tok, docs = _docs(shape, lens, seed=44)
    pos, x, u = dopr.select_prefix_inputs(model, off, tok, K, 10 ** 6)
    for d, ids in enumerate(docs):
        out = om.forward(om.embed(ids), 0, want_probs=True)
        ref_u = oracle.salience(out["probs"], 10 ** 6)
        got_u = u[off[d]:off[d + 1]].astype(np.float64)
        assert np.all(np.abs(got_u - ref_u) <= _u_tol(ref_u)), (d, float(np.max(np.abs(got_u - ref_u))))
        k = min(K, len(ids))
        sel = pos[d, :k]
        assert np.all(np.diff(sel) > 0) and np.all(pos[d, k:] == -1)
        rest = np.setdiff1d(np.arange(len(ids)), sel)
        if len(rest):
            assert ref_u[rest].max() <= ref_u[sel].min() + 2 * _u_tol(ref_u).max()
    model.close()


def test_select_build_score_pipeline_matches_oracle():
    # offline selection -> prefix build -> online scoring, on both sides from the same positions
    shape = SHAPE
    w = synth.make_weights(shape, seed=42, norms="random")
    cfg = dopr.make_config(shape, max_position=4096)
    model = dopr.Model(cfg, w)
    om = oracle.OracleModel(oshape(shape), w)
    lens = [120, 37, 260]
    K = 16
    off, tok, docs = _docs(shape, lens, seed=42)
    pos, x, _ = dopr.select_prefix_inputs(model, off, tok, K, 8)
    store = dopr.Store(cfg, len(lens) - 1, len(lens) * dopr.prefix_bytes(cfg, K))
    dopr.build_prefixes(model, store, np.arange(len(lens)), np.arange(0, K * len(lens) + 1, K, dtype=np.int32),
                        x.reshape(-1, shape.hidden))
    rng = np.random.default_rng(42)
    di = rng.integers(0, len(lens), size=12).astype(np.int64)
    ql = rng.integers(0, 30, size=12)
    qo = np.concatenate([[0], np.cumsum(ql)]).astype(np.int32)
    qt = rng.integers(0, shape.vocab, size=int(qo[-1])).astype(np.int32)
    got = dopr.score(model, store, qo, qt, di).numpy()
    g = oracle.bf16_to_f64(w["final_norm"])
    kv = []
    for d, ids in enumerate(docs):
        h = om.forward(om.embed(ids), 0)["h"]
        c = np.stack([oracle.rmsnorm(h[i], g, shape.rms_eps) for i in pos[d]])
        # the GPU hands bf16 representations to the builder: the oracle builds from the same rounding
        c = oracle.bf16_to_f64(torch.tensor(c, dtype=torch.float32).to(torch.bfloat16))
        o = om.forward(c, 0, want_kv=True)
        kv.append((o["k"], o["v"]))
    ref = om.score_pairs(qo, qt, [int(d) for d in di], kv)
    assert np.max(np.abs(got - ref)) <= TOL, np.max(np.abs(got - ref))
    model.close()
    store.close()


def test_select_errors():
    shape = SHAPE_G2
    model = dopr.Model(dopr.make_config(shape, max_position=4096), synth.make_weights(shape, seed=43))
    for off, tok, K, p in ((np.array([0, 0], np.int32), np.zeros(0, np.int32), 4, 1),        # empty document
                           (np.array([0, 2049], np.int32), np.zeros(2049, np.int32), 4, 1),  # too long
                           (np.array([0, 3], np.int32), np.array([1, 2, 5000], np.int32), 4, 1),  # bad token
                           (np.array([0, 3], np.int32), np.array([1, 2, 3], np.int32), 0, 1),  # top_k 0
                           (np.array([0, 3], np.int32), np.array([1, 2, 3], np.int32), 4, 0)):  # top_p 0
        with pytest.raises(dopr.DoprError) as ei:
            dopr.select_prefix_inputs(model, off, tok, K, p)
        assert ei.value.status == dopr.ERR_INVALID_ARG
    model.close()


def test_selection_workspace_is_reused_across_calls():
    # The n^2 attention matrices, salience, positions and states live in a
    # workspace of the model that grows on demand and is kept.  A long call,
    # shorter ones after it (a larger, stale workspace) and a longer one again
    # (growth) must each return exactly what a fresh model returns.
    shape = SHAPE_G2
    w = synth.make_weights(shape, seed=45, norms="random")
    cfg = dopr.make_config(shape, max_position=4096)
    model = dopr.Model(cfg, w)
    calls = [([300, 200, 17], 24, 4), ([5, 1], 8, 10 ** 6), ([64], 64, 2), ([900, 3, 512], 32, 1)]
    for i, (lens, K, p) in enumerate(calls):
        off, tok, _ = _docs(shape, lens, seed=45 + i)
        got = dopr.select_prefix_inputs(model, off, tok, K, p)
        fresh = dopr.Model(cfg, w)
        want = dopr.select_prefix_inputs(fresh, off, tok, K, p)
        fresh.close()
        np.testing.assert_array_equal(got[0], want[0], err_msg=f"call {i}: positions")
        assert torch.equal(got[1].view(torch.int16), want[1].view(torch.int16)), f"call {i}: states"
        np.testing.assert_array_equal(got[2], want[2], err_msg=f"call {i}: salience")
    model.close()
