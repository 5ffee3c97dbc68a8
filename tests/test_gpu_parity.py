"""GPU parity: the CUDA scoring path (through the C ABI) against the fp64
oracle on identical seeded inputs.

Bars: |score - oracle| <= 3e-2 absolute; packing plan (pair order, token
offsets, positions, ids) bit-exact; top-10 order per query identical wherever
the oracle's adjacent score gap exceeds 0.1.  The projection kernel alone is
checked against a plain fp64 reference of the same product.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_03311_gb300 import dopr, synth

pytestmark = pytest.mark.gpu
TOL = 3e-2


def oshape(s):
    return oracle.Shape(s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.ffn, s.vocab, s.rope_theta,
                        s.rms_eps, s.score_token_id)


class Rig:
    """Model + store on the GPU and the oracle over the same bytes."""

    def __init__(self, shape, doc_m: dict, seed=0, norms="random", std=0.02, max_doc_id=None, max_position=2048):
        self.shape = shape
        self.w = synth.make_weights(shape, seed=seed, norms=norms, std=std)
        self.cfg = dopr.make_config(shape, max_position=max_position)
        self.model = dopr.Model(self.cfg, self.w)
        pool = sum(dopr.prefix_bytes(self.cfg, m) for m in doc_m.values()) + (1 << 16)
        self.store = dopr.Store(self.cfg, max_doc_id if max_doc_id is not None else max(doc_m), pool)
        self.docs = {}
        for d, m in doc_m.items():
            k, v = synth.make_prefix(shape, m, d, seed=seed)
            self.store.put(d, k, v)
            self.docs[d] = (k, v)
        self.om = oracle.OracleModel(oshape(shape), self.w)

    def score(self, pairs):
        return dopr.score(self.model, self.store, pairs["q_offsets"], pairs["q_tokens"], pairs["doc_ids"]).numpy()

    def oracle(self, pairs, idx=None):
        qo, qt, di = pairs["q_offsets"], pairs["q_tokens"], pairs["doc_ids"]
        if idx is not None:
            lens = np.diff(qo)[idx]
            qt = np.concatenate([qt[qo[p]:qo[p + 1]] for p in idx]) if len(idx) else qt[:0]
            qo = np.concatenate([[0], np.cumsum(lens)])
            di = di[idx]
        keys = sorted(set(int(d) for d in di))
        local = {d: i for i, d in enumerate(keys)}
        return self.om.score_pairs(qo, qt, [local[int(d)] for d in di], [self.docs[d] for d in keys])


SMALL_G2 = synth.ModelShape("small-g2", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=128, ffn=384,
                            vocab=1000)
SMALL_G4 = synth.ModelShape("small-g4", n_layers=3, hidden=512, n_q_heads=8, n_kv_heads=2, head_dim=128, ffn=640,
                            vocab=777)


# ------------------------------------------------------------------ GEMM

def _ref_gemm(A, B):
    return (A.double() @ B.double().T)


@pytest.mark.parametrize("M,N,K", [(1, 256, 64), (127, 256, 128), (128, 512, 64), (300, 768, 1024),
                                   (1000, 1024, 512), (2085, 1536, 2048)])
def test_gemm_store_f16(M, N, K):
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.float16)
    B = (0.05 * torch.randn(N, K, device="cuda", generator=g)).to(torch.float16)
    out = dopr.gemm(A, B, dopr.EPI_STORE)
    torch.cuda.synchronize()
    ref = _ref_gemm(A, B)
    err = (out.double() - ref).abs()
    assert torch.all(err <= ref.abs() * 2 ** -10 + 1e-4 * ref.abs().max()), float(err.max())


@pytest.mark.parametrize("M,N,K", [(5, 256, 64), (333, 512, 512), (1500, 1024, 1536)])
def test_gemm_residual_add(M, N, K):
    g = torch.Generator(device="cuda").manual_seed(M + 1)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.float16)
    B = (0.05 * torch.randn(N, K, device="cuda", generator=g)).to(torch.float16)
    R = torch.randn(M, N, device="cuda", generator=g)
    ref = _ref_gemm(A, B) + R.double()
    out = dopr.gemm(A, B, dopr.EPI_RESID_ADD, out=R.clone())
    torch.cuda.synchronize()
    scale = (A.double().abs() @ B.double().abs().T) + R.double().abs()
    assert torch.all((out.double() - ref).abs() <= 1e-5 * scale + 1e-6)


@pytest.mark.parametrize("M,N,K", [(77, 256, 128), (640, 768, 1024)])
def test_gemm_swiglu(M, N, K):
    g = torch.Generator(device="cuda").manual_seed(N + K)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.float16)
    B = (0.05 * torch.randn(N, K, device="cuda", generator=g)).to(torch.float16)
    out = dopr.gemm(A, B, dopr.EPI_SWIGLU)
    torch.cuda.synchronize()
    C = _ref_gemm(A, B)
    blocks = C.view(M, N // 256, 2, 128)
    gate, up = blocks[:, :, 0, :].reshape(M, N // 2), blocks[:, :, 1, :].reshape(M, N // 2)
    ref = torch.nn.functional.silu(gate) * up
    err = (out.double() - ref).abs()
    assert torch.all(err <= ref.abs() * 2 ** -9 + 1e-4 * ref.abs().max()), float(err.max())


# ------------------------------------------------------------ packing plan

def test_pack_plan_bit_exact_against_oracle():
    doc_m = {3: 0, 17: 5, 256: 64, 4000: 1, 4095: 256, 100: 33}
    rig = Rig(SMALL_G2, doc_m, seed=3, max_doc_id=4095)
    rng = np.random.default_rng(3)
    for n in (1, 7, 33, 500):
        lens = rng.integers(0, 50, size=n)
        qo = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        qt = rng.integers(0, SMALL_G2.vocab, size=int(qo[-1])).astype(np.int32)
        docs = rng.choice(list(doc_m), size=n).astype(np.int64)
        got = dopr.pack_plan(rig.model, rig.store, qo, qt, docs)
        ref = oracle.pack_plan(qo, qt, docs, [doc_m[int(d)] for d in docs], SMALL_G2.score_token_id)
        for key in ("perm", "tok_off", "tok_pos", "tok_id", "tok_pair"):
            np.testing.assert_array_equal(got[key], ref[key], err_msg=key)


# ------------------------------------------------------------------ scores

@pytest.mark.parametrize("shape", [SMALL_G2, SMALL_G4], ids=["G2", "G4"])
def test_scores_match_oracle_ragged(shape):
    doc_m = {0: 0, 1: 1, 2: 63, 3: 64, 4: 65, 5: 200, 6: 256, 7: 17}
    rig = Rig(shape, doc_m, seed=5)
    pairs = synth.random_pairs(40, len(doc_m), 0, 150, shape.vocab, seed=5)
    got = rig.score(pairs)
    ref = rig.oracle(pairs)
    assert np.all(np.isfinite(got))
    assert np.max(np.abs(got - ref)) <= TOL, np.max(np.abs(got - ref))


@pytest.mark.parametrize("shape", [SMALL_G2, SMALL_G4], ids=["G2", "G4"])
@pytest.mark.parametrize("doc_m", [{0: 0, 1: 1, 2: 17, 3: 63, 4: 64}, {0: 65, 1: 100, 2: 128, 3: 3}],
                         ids=["mpad64", "mpad128"])
def test_scores_match_oracle_short_prefixes_long_queries(shape, doc_m):
    # Prefixes of at most 128 rows with queries up to 160 tokens: pairs whose
    # own keys fit the attention kernel's resident buffer share batches, the
    # longer ones stream their keys in chunks; both must match the oracle.
    rig = Rig(shape, doc_m, seed=15)
    pairs = synth.random_pairs(48, len(doc_m), 0, 160, shape.vocab, seed=15)
    got = rig.score(pairs)
    ref = rig.oracle(pairs)
    assert np.all(np.isfinite(got))
    assert np.max(np.abs(got - ref)) <= TOL, np.max(np.abs(got - ref))


def test_empty_queries_and_empty_prefix():
    rig = Rig(SMALL_G2, {0: 0, 1: 8}, seed=6)
    pairs = {"q_offsets": np.array([0, 0, 0, 3, 3], np.int32), "q_tokens": np.array([5, 6, 7], np.int32),
             "doc_ids": np.array([0, 1, 0, 1], np.int64)}
    got, ref = rig.score(pairs), rig.oracle(pairs)
    assert np.max(np.abs(got - ref)) <= TOL


def test_qwen3_06b_width_two_layer_workload():
    # 2-layer Qwen3-0.6B-width model, 64 docs (m = 64), 32 queries x 8 docs, 24-token queries.
    wl = synth.WORKLOADS["qwen3-0.6b-2l"]
    doc_m = {d: 64 for d in range(wl.n_docs)}
    rig = Rig(wl.model, doc_m, seed=0, norms="ones")
    pairs = synth.make_workload_pairs(wl, seed=0)
    got = rig.score(pairs)
    ref = rig.oracle(pairs)
    assert np.max(np.abs(got - ref)) <= TOL, np.max(np.abs(got - ref))
    # top-10 order per query wherever the oracle's adjacent gap > 0.1
    q = pairs["query_of_pair"]
    for qi in np.unique(q):
        idx = np.where(q == qi)[0]
        order = idx[np.argsort(-ref[idx], kind="stable")][:10]
        for a, b in zip(order[:-1], order[1:]):
            if ref[a] - ref[b] > 0.1:
                assert got[a] > got[b], (qi, a, b)


def test_batch_order_and_chunking_do_not_change_scores():
    rig = Rig(SMALL_G4, {0: 64, 1: 3, 2: 128, 3: 0}, seed=7)
    pairs = synth.random_pairs(64, 4, 0, 80, SMALL_G4.vocab, seed=7)
    base = rig.score(pairs)
    rng = np.random.default_rng(7)
    perm = rng.permutation(64)
    qo, qt = pairs["q_offsets"], pairs["q_tokens"]
    lens = np.diff(qo)[perm]
    p2 = {"q_offsets": np.concatenate([[0], np.cumsum(lens)]).astype(np.int32),
          "q_tokens": np.concatenate([qt[qo[p]:qo[p + 1]] for p in perm]).astype(np.int32),
          "doc_ids": pairs["doc_ids"][perm]}
    np.testing.assert_array_equal(rig.score(p2), base[perm])
    # one pair at a time
    singles = np.array([rig.score({"q_offsets": np.array([0, qo[p + 1] - qo[p]], np.int32),
                                   "q_tokens": qt[qo[p]:qo[p + 1]], "doc_ids": pairs["doc_ids"][p:p + 1]})[0]
                        for p in range(8)])
    np.testing.assert_array_equal(singles, base[:8])


def test_rows_split_between_short_and_long_tiles_are_batch_invariant():
    # Prefixes of 100-200 keys with queries of 20-250 tokens: a long pair's early tiles fit
    # the tensor-core kernel's 256 key columns and its later ones take the long-tile kernel,
    # and which tile (so which kernel) a row lands in depends on the other pairs of its
    # document in the batch.  The rows' results must not.
    rig = Rig(SMALL_G4, {0: 128, 1: 100, 2: 200}, seed=12)
    pairs = synth.random_pairs(24, 3, 20, 250, SMALL_G4.vocab, seed=12)
    qo, qt, di = pairs["q_offsets"], pairs["q_tokens"], pairs["doc_ids"]
    lens = np.diff(qo)
    assert lens.max() + 128 > 256 and lens.min() + 100 < 256
    base = rig.score(pairs)
    idx = sorted({int(np.argmax(lens)), int(np.argmin(lens)), 3})
    ref = rig.oracle(pairs, idx)
    assert np.max(np.abs(base[idx] - ref)) <= TOL, np.max(np.abs(base[idx] - ref))

    def sub(sel):
        return {"q_offsets": np.concatenate([[0], np.cumsum(lens[sel])]).astype(np.int32),
                "q_tokens": np.concatenate([qt[qo[p]:qo[p + 1]] for p in sel]).astype(np.int32),
                "doc_ids": di[sel]}

    perm = np.random.default_rng(12).permutation(24)
    np.testing.assert_array_equal(rig.score(sub(perm)), base[perm])
    odd = np.arange(1, 24, 2)
    np.testing.assert_array_equal(rig.score(sub(odd)), base[odd])
    for p in (int(np.argmax(lens)), 0, 7):
        np.testing.assert_array_equal(rig.score(sub(np.array([p]))), base[p:p + 1])


def test_device_io_matches_host_io():
    rig = Rig(SMALL_G2, {0: 64, 1: 100}, seed=8)
    pairs = synth.random_pairs(30, 2, 0, 40, SMALL_G2.vocab, seed=8)
    host = rig.score(pairs)
    dev = dopr.score(rig.model, rig.store, torch.tensor(pairs["q_offsets"], device="cuda"),
                     torch.tensor(pairs["q_tokens"], device="cuda"), torch.tensor(pairs["doc_ids"], device="cuda"))
    torch.cuda.synchronize()
    np.testing.assert_array_equal(dev.cpu().numpy(), host)


def test_multi_chunk_batch_matches_small_batches_and_oracle():
    # more packed tokens than one chunk holds -> several chunks, groups split across them
    shape = SMALL_G2
    rig = Rig(shape, {d: (d * 37) % 257 for d in range(12)}, seed=9)
    pairs = synth.random_pairs(900, 12, 20, 60, shape.vocab, seed=9)
    assert int(pairs["q_offsets"][-1]) + 900 > 32768
    big = rig.score(pairs)
    idx = np.random.default_rng(9).choice(900, size=24, replace=False)
    ref = rig.oracle(pairs, idx)
    assert np.max(np.abs(big[idx] - ref)) <= TOL
    qo, qt, di = pairs["q_offsets"], pairs["q_tokens"], pairs["doc_ids"]
    small = rig.score({"q_offsets": qo[:101] - qo[0], "q_tokens": qt[:qo[100]], "doc_ids": di[:100]})
    np.testing.assert_array_equal(small, big[:100])


def test_long_online_sequence_without_prefix():
    # [512 doc tokens ; query ; score token] at positions 0.. with m = 0: the
    # uncompressed pointwise form (Eq. 1) through the same engine.
    rig = Rig(SMALL_G4, {0: 0}, seed=10)
    rng = np.random.default_rng(10)
    qts = [rng.integers(0, SMALL_G4.vocab, size=L).astype(np.int32) for L in (575, 300, 513)]
    pairs = {"q_offsets": np.concatenate([[0], np.cumsum([len(t) for t in qts])]).astype(np.int32),
             "q_tokens": np.concatenate(qts), "doc_ids": np.zeros(3, np.int64)}
    got, ref = rig.score(pairs), rig.oracle(pairs)
    assert np.max(np.abs(got - ref)) <= TOL, np.max(np.abs(got - ref))


@pytest.mark.parametrize("doc_len", [1024, 2048])
def test_full_document_pointwise_scoring_at_the_document_budgets(doc_len):
    # The uncompressed comparison at the paper's longest document budgets (Tab. 8: up to
    # 2,048 tokens): [doc_len document tokens ; query ; score token] per pair with m = 0,
    # several pairs sharing one document's text as the uncompressed run scores them.
    rig = Rig(SMALL_G4, {0: 0}, seed=13, max_position=4096)
    rng = np.random.default_rng(13 + doc_len)
    doc = rng.integers(0, SMALL_G4.vocab, size=doc_len).astype(np.int32)
    qts = [np.concatenate([doc, rng.integers(0, SMALL_G4.vocab, size=L).astype(np.int32)]) for L in (8, 37, 64)]
    pairs = {"q_offsets": np.concatenate([[0], np.cumsum([len(t) for t in qts])]).astype(np.int32),
             "q_tokens": np.concatenate(qts), "doc_ids": np.zeros(len(qts), np.int64)}
    got, ref = rig.score(pairs), rig.oracle(pairs)
    assert np.max(np.abs(got - ref)) <= TOL, np.max(np.abs(got - ref))


def test_prefix_built_by_forward_pass_reproduces_full_forward():
    # Sec. 3.4 footnote: stored states are the per-layer K/V of forwarding the
    # prefix inputs.  Build them with the oracle, store them in bf16, and the
    # GPU score of [q ; t_score] must match one causal pass over [prefix ; q ; t_score].
    shape = SMALL_G4
    rig = Rig(shape, {}, seed=11, max_doc_id=4)
    rng = np.random.default_rng(11)
    m, L = 40, 12
    ptoks = rng.integers(0, shape.vocab, size=m)
    pre = rig.om.forward(rig.om.embed(ptoks), 0, want_kv=True)
    k = torch.tensor(pre["k"], dtype=torch.float32).to(torch.bfloat16)
    v = torch.tensor(pre["v"], dtype=torch.float32).to(torch.bfloat16)
    store = dopr.Store(rig.cfg, 4, dopr.prefix_bytes(rig.cfg, m))
    store.put(2, k, v)
    q = rng.integers(0, shape.vocab, size=L).astype(np.int32)
    got = dopr.score(rig.model, store, np.array([0, L], np.int32), q, np.array([2], np.int64)).numpy()[0]
    full = rig.om.forward(rig.om.embed(np.concatenate([ptoks, q, [shape.score_token_id]])), 0)["h"]
    assert abs(got - rig.om.score_head(full[-1])) <= TOL


# ------------------------------------------------------------------ errors

def test_error_paths_leave_outputs_untouched():
    shape = SMALL_G2
    rig = Rig(shape, {0: 8, 1: 8}, seed=12, max_doc_id=9)
    k, v = synth.make_prefix(shape, 8, 5, seed=12)
    rig.store.put_layer(5, 0, k[0], v[0])  # doc 5 stored for layer 0 only
    qo, qt = np.array([0, 2], np.int32), np.array([1, 2], np.int32)
    out = torch.full((1,), 123.0)

    def status(doc, tokens=qt):
        try:
            dopr.score(rig.model, rig.store, qo, tokens, np.array([doc], np.int64), out=out)
            return dopr.OK
        except dopr.DoprError as e:
            return e.status

    assert status(3) == dopr.ERR_UNKNOWN_DOC
    assert status(10) == dopr.ERR_UNKNOWN_DOC
    assert status(5) == dopr.ERR_INCOMPLETE
    assert status(0, np.array([1, shape.vocab], np.int32)) == dopr.ERR_INVALID_ARG
    assert float(out[0]) == 123.0
    # device-side validation of device inputs
    with pytest.raises(dopr.DoprError) as ei:
        dopr.score(rig.model, rig.store, torch.tensor(qo, device="cuda"), torch.tensor(qt, device="cuda"),
                   torch.tensor([3], dtype=torch.int64, device="cuda"))
    assert ei.value.status == dopr.ERR_UNKNOWN_DOC
    with pytest.raises(dopr.DoprError) as ei:
        dopr.score(rig.model, rig.store, torch.tensor(qo, device="cuda"),
                   torch.tensor([1, -4], dtype=torch.int32, device="cuda"),
                   torch.tensor([0], dtype=torch.int64, device="cuda"))
    assert ei.value.status == dopr.ERR_INVALID_ARG
    # store misuse
    k2, v2 = synth.make_prefix(shape, 9, 0, seed=12)
    with pytest.raises(dopr.DoprError) as ei:
        rig.store.put_layer(0, 0, k2[0], v2[0])  # m differs from the first put
    assert ei.value.status == dopr.ERR_INVALID_ARG
    k3, v3 = synth.make_prefix(shape, 257, 0, seed=12)
    with pytest.raises(dopr.DoprError) as ei:
        rig.store.put_layer(7, 0, k3[0], v3[0])
    assert ei.value.status == dopr.ERR_INVALID_ARG
    tiny = dopr.Store(rig.cfg, 3, dopr.prefix_bytes(rig.cfg, 8))
    tiny.put(0, *synth.make_prefix(shape, 8, 0, seed=12))
    with pytest.raises(dopr.DoprError) as ei:
        tiny.put(1, *synth.make_prefix(shape, 8, 1, seed=12))
    assert ei.value.status == dopr.ERR_OUT_OF_MEMORY
    # the good path still works after all of that
    good = rig.score({"q_offsets": qo, "q_tokens": qt, "doc_ids": np.array([1], np.int64)})
    ref = rig.oracle({"q_offsets": qo, "q_tokens": qt, "doc_ids": np.array([1], np.int64)})
    assert abs(good[0] - ref[0]) <= TOL


def test_incomplete_model_rejected():
    cfg = dopr.make_config(SMALL_G2)
    model = dopr.Model(cfg)
    store = dopr.Store(cfg, 1, dopr.prefix_bytes(cfg, 4))
    store.put(0, *synth.make_prefix(SMALL_G2, 4, 0))
    with pytest.raises(dopr.DoprError) as ei:
        dopr.score(model, store, np.array([0, 1], np.int32), np.array([3], np.int32), np.array([0], np.int64))
    assert ei.value.status == dopr.ERR_INCOMPLETE


def test_bounded_wait_gives_up_and_context_survives():
    import time

    t0 = time.time()
    assert dopr.wait_timeout_probe(200) == dopr.ERR_TIMEOUT
    assert time.time() - t0 < 30
    A = torch.randn(128, 64, device="cuda").to(torch.float16)
    B = torch.randn(256, 64, device="cuda").to(torch.float16)
    out = dopr.gemm(A, B)
    torch.cuda.synchronize()
    assert torch.allclose(out.float(), (A.float() @ B.float().T), rtol=1e-2, atol=1e-1)
