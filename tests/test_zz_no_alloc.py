"""The allocation-free packing entry point (dopr_pack_order_noalloc).

It serves callers that cannot allocate device memory while they score
(their GPU memory belongs to another allocator, or cudaMalloc would stall a
latency-critical loop).  Its results must equal those of the regular packer
entry point, call after call, although every call reuses one scratch array
compiled into the library.  This file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_03311_gb300 import dopr, synth

pytestmark = pytest.mark.gpu

SHAPE = synth.ModelShape("noalloc", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=128, ffn=384,
                         vocab=1000)


@pytest.fixture(scope="module")
def rig():
    cfg = dopr.make_config(SHAPE, max_position=1024)
    model = dopr.Model(cfg, synth.make_weights(SHAPE, seed=21))
    doc_m = {2: 0, 9: 7, 40: 64, 500: 130, 131071: 256}
    store = dopr.Store(cfg, 131071, sum(dopr.prefix_bytes(cfg, m) for m in doc_m.values()))
    for d, m in doc_m.items():
        store.put(d, *synth.make_prefix(SHAPE, m, d, seed=21))
    return cfg, model, store, doc_m


def _batch(doc_m, n, seed):
    rng = np.random.default_rng(seed)
    lens = rng.integers(0, 60, size=n)
    qo = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    qt = rng.integers(0, SHAPE.vocab, size=int(qo[-1])).astype(np.int32)
    docs = rng.choice(list(doc_m), size=n).astype(np.int64)
    return qo, qt, docs


def _noalloc(store, qo, docs):
    n = len(docs)
    perm = torch.full((max(n, 1),), -7, dtype=torch.int32, device="cuda")
    tok_off = torch.full((n + 1,), -7, dtype=torch.int32, device="cuda")
    dopr.pack_order_noalloc(store, torch.tensor(qo, device="cuda"), torch.tensor(docs, device="cuda"), perm, tok_off)
    return perm[:n].cpu().numpy(), tok_off.cpu().numpy()


def test_noalloc_matches_regular_packer_on_consecutive_calls(rig):
    cfg, model, store, doc_m = rig
    # two calls in a row with different batches, then the first batch again:
    # leftover scratch contents of a previous call must not leak into the next
    for n, seed in ((700, 1), (33, 2), (700, 1), (1, 3)):
        qo, qt, docs = _batch(doc_m, n, seed)
        ref = dopr.pack_plan(model, store, qo, qt, docs)
        # the oracle's plan (stable sort by document, packed offsets) fixes both
        want = oracle.pack_plan(qo, qt, docs, [doc_m[int(d)] for d in docs], SHAPE.score_token_id)
        perm, tok_off = _noalloc(store, qo, docs)
        np.testing.assert_array_equal(perm, want["perm"])
        np.testing.assert_array_equal(tok_off, want["tok_off"])
        np.testing.assert_array_equal(perm, ref["perm"])
        np.testing.assert_array_equal(tok_off, ref["tok_off"])


def test_noalloc_limits_and_errors(rig):
    cfg, model, store, doc_m = rig
    qo = torch.zeros(32769 + 1, dtype=torch.int32, device="cuda")
    docs = torch.full((32769,), 2, dtype=torch.int64, device="cuda")
    out = torch.zeros(32770, dtype=torch.int32, device="cuda")
    with pytest.raises(dopr.DoprError) as ei:
        dopr.pack_order_noalloc(store, qo, docs, out[:32769], out)
    assert ei.value.status == dopr.ERR_UNSUPPORTED and "32768" in str(ei.value)
    big = dopr.Store(cfg, 131072, 1 << 16)
    with pytest.raises(dopr.DoprError) as ei:
        dopr.pack_order_noalloc(big, qo[:2], docs[:1], out[:1], out[:2])
    assert ei.value.status == dopr.ERR_UNSUPPORTED
    with pytest.raises(dopr.DoprError) as ei:
        dopr.pack_order_noalloc(store, torch.tensor([0, 3], dtype=torch.int32, device="cuda"),
                                torch.tensor([5], dtype=torch.int64, device="cuda"), out[:1], out[:2])
    assert ei.value.status == dopr.ERR_UNKNOWN_DOC
    # short caller buffers are refused by the binding before anything is launched
    qo3 = torch.tensor([0, 1, 2, 3], dtype=torch.int32, device="cuda")
    d3 = torch.full((3,), 2, dtype=torch.int64, device="cuda")
    o3 = torch.full((4,), -7, dtype=torch.int32, device="cuda")
    for args in ((qo3, d3[:2], o3[:3], o3), (qo3, d3, o3[:2], o3), (qo3, d3, o3[:3], o3[:3])):
        with pytest.raises(ValueError):
            dopr.pack_order_noalloc(store, *args)
    assert torch.all(o3 == -7)
    # still correct after the failed calls
    qo2, qt2, docs2 = _batch(doc_m, 50, 4)
    want = oracle.pack_plan(qo2, qt2, docs2, [doc_m[int(d)] for d in docs2], SHAPE.score_token_id)
    perm, tok_off = _noalloc(store, qo2, docs2)
    np.testing.assert_array_equal(perm, want["perm"])
    np.testing.assert_array_equal(tok_off, want["tok_off"])
