"""Pins of the fp64 oracle against things other than itself.

Each check ties one part of the oracle to a library routine, a closed form,
an independent formulation or an invariant that the paper's formulation
fixes (DoPR Sec. 3.1 and Sec. 3.4), so that a dropped term, a wrong sign, a
wrong index or a transposed operand in the oracle fails at least one test.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from oracle import OracleModel, Shape, bf16_to_f64
from paper_2609_03311_gb300 import synth

TINY = synth.ModelShape("tiny", n_layers=2, hidden=64, n_q_heads=4, n_kv_heads=2, head_dim=16,
                        ffn=96, vocab=50, rope_theta=1e4, rms_eps=1e-6)


def oracle_shape(s: synth.ModelShape) -> Shape:
    return Shape(s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn, s.vocab,
                 s.rope_theta, s.rms_eps, s.score_token_id)


def tiny_model(seed=0, zero=(), shape=TINY, std=0.2):
    w = synth.make_weights(shape, seed=seed, norms="random", std=std, zero=zero)
    return OracleModel(oracle_shape(shape), w), w


def f64(t):
    return bf16_to_f64(t) if t.dtype == torch.bfloat16 else np.asarray(t, dtype=np.float64)


# ---------------------------------------------------------------- single ops

def test_bf16_widening_exact(oracle_lib):
    cases = {0x3F80: 1.0, 0xC000: -2.0, 0x0000: 0.0, 0x3E80: 0.25, 0x4049: 3.140625,
             0x7F80: math.inf, 0x0001: 2.0 ** -133}
    for bits, val in cases.items():
        assert oracle_lib.oracle_bf16_to_f64(bits) == val


def test_rmsnorm_matches_torch_rms_norm():
    rng = np.random.default_rng(1)
    for n in (1, 7, 128, 1024):
        x = rng.normal(size=n) * rng.uniform(0.01, 10)
        g = 1 + 0.3 * rng.normal(size=n)
        ref = F.rms_norm(torch.tensor(x), (n,), weight=torch.tensor(g), eps=1e-6).numpy()
        np.testing.assert_allclose(oracle.rmsnorm(x, g, 1e-6), ref, rtol=1e-13, atol=1e-15)


def test_rmsnorm_constant_vector_closed_form():
    # x = c * 1  =>  mean(x^2) = c^2  =>  y = g * c / sqrt(c^2 + eps)
    for c in (3.0, -0.5, 1e-4):
        n, eps = 16, 1e-6
        g = np.linspace(0.5, 2.0, n)
        y = oracle.rmsnorm(np.full(n, c), g, eps)
        np.testing.assert_allclose(y, g * c / math.sqrt(c * c + eps), rtol=1e-14)


def test_rope_matches_complex_rotation():
    # Rotate-half RoPE == multiplying z_i = x_i + i x_{i+D/2} by exp(i pos theta^(-2i/D)).
    rng = np.random.default_rng(2)
    for D, theta in ((16, 1e4), (128, 1e6)):
        for pos in (0, 1, 5, 63, 300):
            x = rng.normal(size=D)
            half = D // 2
            z = x[:half] + 1j * x[half:]
            freq = theta ** (-2.0 * np.arange(half) / D)
            w = z * np.exp(1j * pos * freq)
            ref = np.concatenate([w.real, w.imag])
            np.testing.assert_allclose(oracle.rope(x, pos, theta), ref, rtol=1e-12, atol=1e-12)


def test_rope_relative_position_property():
    # <R(a) q, R(b) k> depends only on a - b; pos 0 is the identity; norms are kept.
    rng = np.random.default_rng(3)
    q, k = rng.normal(size=128), rng.normal(size=128)
    d0 = oracle.rope(q, 70, 1e6) @ oracle.rope(k, 64, 1e6)
    d1 = oracle.rope(q, 6, 1e6) @ oracle.rope(k, 0, 1e6)
    assert abs(d0 - d1) < 1e-9
    np.testing.assert_array_equal(oracle.rope(q, 0, 1e6), q)
    assert abs(np.linalg.norm(oracle.rope(q, 123, 1e6)) - np.linalg.norm(q)) < 1e-12


def test_attend_matches_sdpa():
    rng = np.random.default_rng(4)
    for n, D in ((1, 16), (9, 16), (200, 128)):
        q, K, V = rng.normal(size=D), rng.normal(size=(n, D)), rng.normal(size=(n, D))
        scale = 1 / math.sqrt(D)
        ref = F.scaled_dot_product_attention(torch.tensor(q)[None, None, None], torch.tensor(K)[None, None],
                                             torch.tensor(V)[None, None], scale=scale)[0, 0, 0].numpy()
        np.testing.assert_allclose(oracle.attend(q, K, V, scale), ref, rtol=1e-12, atol=1e-13)


def test_silu_matches_torch():
    for x in (-20.0, -1.5, 0.0, 0.3, 7.0):
        assert abs(oracle.silu(x) - F.silu(torch.tensor(x, dtype=torch.float64)).item()) < 1e-15


# ----------------------------------------------- whole model vs library ops

def torch_forward(w, s: synth.ModelShape, x0, pos0, pk=None, pv=None):
    """Independent composition from torch library routines (F.linear,
    F.rms_norm, complex-number RoPE, SDPA with GQA).  Returns h [T,H] and
    per-layer attention outputs [L,T,Hq*D]."""
    H, Hq, Hkv, D = s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim
    t = lambda a: torch.tensor(f64(a))
    x = torch.tensor(x0)
    T = x.shape[0]
    m = 0 if pk is None else pk.shape[1]
    half = D // 2
    freq = s.rope_theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / D)
    ang = torch.arange(pos0, pos0 + T, dtype=torch.float64)[:, None] * freq[None]
    rot = torch.polar(torch.ones_like(ang), ang)  # [T, half]

    def rope(v):  # v [T, heads, D]
        z = torch.complex(v[..., :half], v[..., half:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    # mask[t, key]: prefix keys always visible, own keys causal
    mask = torch.ones(T, m + T, dtype=torch.bool)
    mask[:, m:] = torch.tril(torch.ones(T, T, dtype=torch.bool))
    attn_all = []
    for l in range(s.n_layers):
        xn = F.rms_norm(x, (H,), weight=t(w["attn_norm"][l]), eps=s.rms_eps)
        q = F.linear(xn, t(w["wq"][l])).view(T, Hq, D)
        k = F.linear(xn, t(w["wk"][l])).view(T, Hkv, D)
        v = F.linear(xn, t(w["wv"][l])).view(T, Hkv, D)
        q = rope(F.rms_norm(q, (D,), weight=t(w["q_norm"][l]), eps=s.rms_eps))
        k = rope(F.rms_norm(k, (D,), weight=t(w["k_norm"][l]), eps=s.rms_eps))
        if m:
            k = torch.cat([torch.tensor(pk[l]), k], 0)
            v = torch.cat([torch.tensor(pv[l]), v], 0)
        o = F.scaled_dot_product_attention(q.transpose(0, 1)[None], k.transpose(0, 1)[None],
                                           v.transpose(0, 1)[None], attn_mask=mask, enable_gqa=True,
                                           scale=1 / math.sqrt(D))[0].transpose(0, 1).reshape(T, Hq * D)
        attn_all.append(o)
        x = x + F.linear(o, t(w["wo"][l]))
        xn = F.rms_norm(x, (H,), weight=t(w["mlp_norm"][l]), eps=s.rms_eps)
        x = x + F.linear(F.silu(F.linear(xn, t(w["w_gate"][l]))) * F.linear(xn, t(w["w_up"][l])),
                         t(w["w_down"][l]))
    return x.numpy(), torch.stack(attn_all).numpy()


def test_forward_matches_torch_composition_with_prefix():
    om, w = tiny_model(seed=5)
    rng = np.random.default_rng(5)
    m, T = 6, 5
    pk = rng.normal(size=(TINY.n_layers, m, TINY.n_kv_heads, TINY.head_dim))
    pv = rng.normal(size=(TINY.n_layers, m, TINY.n_kv_heads, TINY.head_dim))
    x0 = om.embed(rng.integers(0, TINY.vocab, size=T))
    got = om.forward(x0, m, pk, pv, want_attn=True)
    h_ref, attn_ref = torch_forward(w, TINY, x0, m, pk, pv)
    np.testing.assert_allclose(got["attn"], attn_ref, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(got["h"], h_ref, rtol=1e-10, atol=1e-12)


def test_gqa_mapping_single_key():
    # m = 0 and a single online token: attention output of q head h is the
    # value of kv head floor(h / G) (contiguous head groups).
    om, w = tiny_model(seed=6)
    x0 = om.embed([TINY.score_token_id])
    out = om.forward(x0, 0, want_kv=True, want_attn=True)
    G = TINY.n_q_heads // TINY.n_kv_heads
    D = TINY.head_dim
    for l in range(TINY.n_layers):
        for h in range(TINY.n_q_heads):
            np.testing.assert_allclose(out["attn"][l, 0, h * D:(h + 1) * D], out["v"][l, 0, h // G], rtol=1e-13)
    # and the mapping is not the interleaved one (kv head h % Hkv)
    assert not np.allclose(out["attn"][0, 0, 1 * D:2 * D], out["v"][0, 0, 1])


def test_uniform_attention_when_wq_zero():
    # W_q = 0 => q = 0 after QK-norm => every visible key has equal weight =>
    # attention output is the mean of the m prefix values and online values 0..t.
    om, w = tiny_model(seed=7, zero=("wq",))
    rng = np.random.default_rng(7)
    m, T = 4, 6
    pk = rng.normal(size=(TINY.n_layers, m, TINY.n_kv_heads, TINY.head_dim))
    pv = rng.normal(size=(TINY.n_layers, m, TINY.n_kv_heads, TINY.head_dim))
    x0 = om.embed(rng.integers(0, TINY.vocab, size=T))
    out = om.forward(x0, m, pk, pv, want_kv=True, want_attn=True)
    G, D = TINY.n_q_heads // TINY.n_kv_heads, TINY.head_dim
    for l in range(TINY.n_layers):
        for t in range(T):
            for h in range(TINY.n_q_heads):
                vals = np.concatenate([pv[l, :, h // G], out["v"][l, :t + 1, h // G]], 0)
                assert vals.shape[0] == m + t + 1
                np.testing.assert_allclose(out["attn"][l, t, h * D:(h + 1) * D], vals.mean(0), rtol=1e-12, atol=1e-14)


def test_score_closed_form_when_block_outputs_zero():
    # W_o = W_down = 0 => every block adds 0 to the residual => h_last = E[t_score]
    # => score = <W_s[yes] - W_s[no], RMSNorm(E[t_score]) * g_final>, whatever q and d are.
    om, w = tiny_model(seed=8, zero=("wo", "w_down"))
    rng = np.random.default_rng(8)
    e = f64(w["embed"][TINY.score_token_id])
    hn = F.rms_norm(torch.tensor(e), (TINY.hidden,), weight=torch.tensor(f64(w["final_norm"])), eps=TINY.rms_eps)
    ws = torch.tensor(f64(w["score_head"]))
    expect = float((ws[0] - ws[1]) @ hn)
    docs = [tuple(rng.normal(size=(2, TINY.n_layers, m, TINY.n_kv_heads, TINY.head_dim))) for m in (0, 3, 9)]
    pairs = synth.random_pairs(6, len(docs), 0, 7, TINY.vocab, seed=8)
    s = om.score_pairs(pairs["q_offsets"], pairs["q_tokens"], pairs["doc_ids"], docs)
    np.testing.assert_allclose(s, expect, rtol=1e-12)


def test_score_is_yes_minus_no():
    # Swapping the two head rows negates every score; zeroing the "no" row
    # leaves the plain "yes" logit.
    om, w = tiny_model(seed=9)
    h = np.random.default_rng(9).normal(size=TINY.hidden)
    s = om.score_head(h)
    w2 = dict(w)
    w2["score_head"] = w["score_head"].flip(0).contiguous()
    om2 = OracleModel(oracle_shape(TINY), w2)
    assert om2.score_head(h) == pytest.approx(-s, rel=1e-14)
    w3 = dict(w)
    w3["score_head"] = torch.stack([w["score_head"][0], torch.zeros_like(w["score_head"][1])])
    om3 = OracleModel(oracle_shape(TINY), w3)
    hn = F.rms_norm(torch.tensor(h), (TINY.hidden,), weight=torch.tensor(f64(w["final_norm"])), eps=TINY.rms_eps)
    assert om3.score_head(h) == pytest.approx(float(torch.tensor(f64(w["score_head"][0])) @ hn), rel=1e-13)


# --------------------------------------------------------------- invariants

def test_prefix_states_reproduce_full_forward():
    # Prefix consistency: running the decoder over m prefix tokens and storing
    # each layer's (normed, rotated) keys and values, then scoring [q ; t_score]
    # at positions m.., equals one causal pass over [prefix ; q ; t_score].
    om, w = tiny_model(seed=10)
    rng = np.random.default_rng(10)
    for m, L in ((5, 4), (1, 0), (12, 9)):
        ptoks = rng.integers(0, TINY.vocab, size=m)
        qtoks = rng.integers(0, TINY.vocab, size=L)
        full_ids = np.concatenate([ptoks, qtoks, [TINY.score_token_id]])
        full = om.forward(om.embed(full_ids), 0)["h"]
        s_full = om.score_head(full[-1])
        pre = om.forward(om.embed(ptoks), 0, want_kv=True)
        s = om.score_pairs([0, L], qtoks, [0], [(pre["k"], pre["v"])])[0]
        assert abs(s - s_full) <= 1e-9 * max(1.0, abs(s_full))
        # the online hidden states agree too, row by row
        on = om.forward(om.embed(np.concatenate([qtoks, [TINY.score_token_id]])), m, pre["k"], pre["v"])["h"]
        np.testing.assert_allclose(on, full[m:], rtol=1e-9, atol=1e-12)


def test_empty_prefix_is_query_only_forward():
    om, w = tiny_model(seed=11)
    rng = np.random.default_rng(11)
    q = rng.integers(0, TINY.vocab, size=7)
    ids = np.concatenate([q, [TINY.score_token_id]])
    h = om.forward(om.embed(ids), 0)["h"]
    s = om.score_pairs([0, 7], q, [0], [(np.zeros((TINY.n_layers, 0, 2, 16)), np.zeros((TINY.n_layers, 0, 2, 16)))])
    assert s[0] == om.score_head(h[-1])
    h_ref, _ = torch_forward(w, TINY, om.embed(ids), 0)
    np.testing.assert_allclose(h, h_ref, rtol=1e-10, atol=1e-12)


def test_scores_invariant_to_batch_order_and_doc_sharing():
    om, w = tiny_model(seed=12)
    rng = np.random.default_rng(12)
    docs = [tuple(synth.make_prefix(TINY, m, d, seed=12)) for d, m in enumerate((3, 0, 8, 5))]
    pairs = synth.random_pairs(10, len(docs), 0, 6, TINY.vocab, seed=12)
    s = om.score_pairs(pairs["q_offsets"], pairs["q_tokens"], pairs["doc_ids"], docs)
    # permute the pairs
    perm = rng.permutation(10)
    qo, qt = pairs["q_offsets"], pairs["q_tokens"]
    lens = np.diff(qo)[perm]
    qo2 = np.concatenate([[0], np.cumsum(lens)])
    qt2 = np.concatenate([qt[qo[p]:qo[p + 1]] for p in perm])
    s2 = om.score_pairs(qo2, qt2, pairs["doc_ids"][perm], docs)
    np.testing.assert_array_equal(s2, s[perm])
    # give every pair its own copy of its document: no sharing, same scores
    own = [docs[d] for d in pairs["doc_ids"]]
    s3 = om.score_pairs(qo, qt, np.arange(10), own)
    np.testing.assert_array_equal(s3, s)
    # duplicate pairs score identically
    s4 = om.score_pairs(np.concatenate([qo, qo[1:] + qo[-1]]), np.concatenate([qt, qt]),
                        np.concatenate([pairs["doc_ids"]] * 2), docs)
    np.testing.assert_array_equal(s4[:10], s4[10:])


def test_bf16_prefix_widened_exactly():
    om, w = tiny_model(seed=13)
    k, v = synth.make_prefix(TINY, 4, 0, seed=13)
    s_bf = om.score_pairs([0, 2], [1, 2], [0], [(k, v)])
    s_64 = om.score_pairs([0, 2], [1, 2], [0], [(bf16_to_f64(k), bf16_to_f64(v))])
    assert s_bf[0] == s_64[0]


# -------------------------------------------------------------- batch plan

def test_pack_plan_against_python_stable_sort():
    rng = np.random.default_rng(14)
    for n in (0, 1, 17, 300):
        lens = rng.integers(0, 9, size=n)
        qo = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        qt = rng.integers(0, 1000, size=int(qo[-1])).astype(np.int32)
        docs = rng.integers(0, 7, size=n) * 1000003  # sparse, large ids
        m_of_doc = {d: int(rng.integers(0, 5)) for d in set(docs.tolist())}
        pm = np.asarray([m_of_doc[d] for d in docs], np.int32)
        plan = oracle.pack_plan(qo, qt, docs, pm, 999)
        perm = sorted(range(n), key=lambda p: docs[p])  # Python's sort is stable
        np.testing.assert_array_equal(plan["perm"], perm)
        off = 0
        for s, p in enumerate(perm):
            assert plan["tok_off"][s] == off
            L = lens[p]
            for j in range(L + 1):
                assert plan["tok_pos"][off + j] == pm[p] + j
                assert plan["tok_id"][off + j] == (qt[qo[p] + j] if j < L else 999)
                assert plan["tok_pair"][off + j] == s
            off += L + 1
        assert plan["tok_off"][n] == off


# --------------------------------------------- key token selection (Sec. 3.2.1)

def test_salience_hand_worked_matrix():
    # column i's causal entries are rows i..n-1; u_i = mean of the top-p of them
    A = np.array([[1.0, 0.0, 0.0, 0.0],
                  [0.25, 0.75, 0.0, 0.0],
                  [0.5, 0.2, 0.3, 0.0],
                  [0.1, 0.6, 0.1, 0.2]])
    np.testing.assert_allclose(oracle.salience(A, 1), [1.0, 0.75, 0.3, 0.2], rtol=0, atol=1e-15)
    np.testing.assert_allclose(oracle.salience(A, 2), [0.75, 0.675, 0.2, 0.2], rtol=0, atol=1e-15)
    np.testing.assert_allclose(oracle.salience(A, 4), [1.85 / 4, 1.55 / 3, 0.4 / 2, 0.2], rtol=0, atol=1e-15)
    np.testing.assert_allclose(oracle.salience(A, 100), oracle.salience(A, 4), rtol=0, atol=0)


def test_select_topk_against_brute_force_with_ties():
    rng = np.random.default_rng(3)
    for n, K in ((1, 1), (7, 3), (40, 40), (40, 55), (200, 16)):
        u = rng.integers(0, 6, size=n).astype(np.float64) / 5.0  # many exact ties
        want = sorted(sorted(range(n), key=lambda i: (-u[i], i))[:min(K, n)])
        np.testing.assert_array_equal(oracle.select_topk(u, K), want)


def test_attention_weights_uniform_when_wq_zero():
    # W_q = 0 => every causal key of token t weighs 1/(t+1) in every head, so the
    # head-averaged matrix is A[t][i] = 1/(t+1) for i <= t; column i's top-p are
    # 1/(i+1) .. 1/(i+k), k = min(p, n - i).
    om, w = tiny_model(seed=8, zero=("wq",))
    rng = np.random.default_rng(8)
    n = 9
    out = om.forward(om.embed(rng.integers(0, TINY.vocab, size=n)), 0, want_probs=True)
    want = np.tril(np.ones((n, n))) / np.arange(1, n + 1)[:, None]
    np.testing.assert_allclose(out["probs"], want, rtol=1e-13, atol=1e-15)
    for p in (1, 3, n):
        u = oracle.salience(out["probs"], p)
        for i in range(n):
            k = min(p, n - i)
            assert abs(u[i] - np.mean(1.0 / np.arange(i + 1, i + k + 1))) <= 1e-13


def test_attention_weights_rows_causal_and_consistent_with_outputs():
    # rows sum to 1, nothing above the diagonal (beyond the prefix); with one kv head
    # the head-averaged weights applied to the last layer's values give the mean of
    # the heads' attention outputs (oracle_attend's own path).
    shape = synth.ModelShape("tiny-kv1", n_layers=2, hidden=64, n_q_heads=4, n_kv_heads=1, head_dim=16, ffn=96,
                             vocab=50, rope_theta=1e4, rms_eps=1e-6)
    om, _ = tiny_model(seed=9, shape=shape)
    rng = np.random.default_rng(9)
    m, T = 3, 8
    pk = rng.normal(size=(shape.n_layers, m, 1, shape.head_dim))
    pv = rng.normal(size=(shape.n_layers, m, 1, shape.head_dim))
    out = om.forward(om.embed(rng.integers(0, shape.vocab, size=T)), m, pk, pv, want_kv=True, want_attn=True,
                     want_probs=True)
    P = out["probs"]
    np.testing.assert_allclose(P.sum(1), 1.0, rtol=0, atol=1e-13)
    for t in range(T):
        assert np.all(P[t, m + t + 1:] == 0.0)
    L, D = shape.n_layers - 1, shape.head_dim
    V = np.concatenate([pv[L, :, 0], out["v"][L, :, 0]], 0)  # [m + T, D]
    head_mean = out["attn"][L].reshape(T, shape.n_q_heads, D).mean(1)
    np.testing.assert_allclose(P @ V, head_mean, rtol=1e-11, atol=1e-13)


# ------------------------------------------------------- MLP scoring head (Sec. 3.2.3)

def _mlp_head(d, H, seed, act, std=0.05):
    rng = np.random.default_rng(seed)
    bf = lambda a: torch.tensor(a, dtype=torch.float32).to(torch.bfloat16)
    return {"w1": bf(rng.normal(0, std, size=(d, H))), "b1": bf(rng.normal(0, 0.1, size=d)),
            "w2": bf(rng.normal(0, 0.1, size=d)), "b2": 0.25, "act": act}


@pytest.mark.parametrize("act", [0, 1, 2, 3])
def test_mlp_head_matches_torch_composition(act):
    om, w = tiny_model(seed=12)
    head = _mlp_head(24, TINY.hidden, 12, act)
    h = np.random.default_rng(12).normal(size=TINY.hidden)
    hn = F.rms_norm(torch.tensor(h), (TINY.hidden,), torch.tensor(f64(w["final_norm"])), eps=TINY.rms_eps)
    z = torch.tensor(f64(head["w1"])) @ hn + torch.tensor(f64(head["b1"]))
    a = [torch.relu, lambda x: F.gelu(x, approximate="none"), F.silu, torch.tanh][act](z)
    want = float(torch.tensor(f64(head["w2"])) @ a + head["b2"])
    assert abs(om.mlp_head(h, head) - want) <= 1e-12 * max(1.0, abs(want))


def test_mlp_head_identity_closed_form():
    # W1 = I, b1 = 0, ReLU, w2 = 1, b2 = 0: the sum of the positive normed components
    om, w = tiny_model(seed=13)
    H = TINY.hidden
    eye = torch.eye(H, dtype=torch.bfloat16)
    head = {"w1": eye, "b1": torch.zeros(H, dtype=torch.bfloat16), "w2": torch.ones(H, dtype=torch.bfloat16),
            "b2": 0.0, "act": 0}
    h = np.random.default_rng(13).normal(size=H)
    g = f64(w["final_norm"])
    hn = h / math.sqrt(np.mean(h * h) + TINY.rms_eps) * g
    assert abs(om.mlp_head(h, head) - np.sum(np.maximum(hn, 0.0))) <= 1e-12
