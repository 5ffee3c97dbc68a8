"""The synthetic workloads match their stated recipe (host only, no GPU).

The measured configurations stand in for the paper's TREC DL / BEIR / BRIGHT
candidate lists with seeded synthetic data of the same shapes; these checks
pin that recipe: pair and query counts, query lengths, candidate lists of
distinct documents, per-document prefix lengths, the Zipf(1.1) reuse of the
skewed workloads, the uncompressed comparison's document text, and that every
draw is reproducible from its seed.
"""
import numpy as np
import pytest

import bench
from paper_2609_03311_gb300 import synth


@pytest.mark.parametrize("name", sorted(synth.WORKLOADS))
def test_pairs_follow_the_recipe(name):
    wl = synth.WORKLOADS[name]
    pairs = synth.make_workload_pairs(wl, seed=0)
    n, k = wl.n_pairs, wl.docs_per_query
    assert len(pairs["doc_ids"]) == n and len(pairs["q_offsets"]) == n + 1
    qlen = np.diff(pairs["q_offsets"])
    assert qlen.min() >= wl.qlen_min and qlen.max() <= wl.qlen_max
    assert pairs["q_tokens"].min() >= 0 and pairs["q_tokens"].max() < wl.model.vocab
    qid = pairs["query_of_pair"]
    assert np.array_equal(qid, np.repeat(np.arange(wl.n_queries), k))
    for q in range(wl.n_queries):
        sel = slice(q * k, (q + 1) * k)
        docs = pairs["doc_ids"][sel]
        assert len(set(docs.tolist())) == k  # a candidate list has no repeated document
        assert docs.min() >= 0 and docs.max() < wl.n_docs
        assert len(set(qlen[sel].tolist())) == 1  # one query text per list
        qo, qt = pairs["q_offsets"], pairs["q_tokens"]
        toks = [tuple(qt[qo[p]:qo[p + 1]]) for p in range(sel.start, sel.stop)]
        assert len(set(toks)) == 1
    # seeded: the same seed gives the same bytes, another seed other draws
    again = synth.make_workload_pairs(wl, seed=0)
    for key in ("q_offsets", "q_tokens", "doc_ids"):
        np.testing.assert_array_equal(again[key], pairs[key])
    other = synth.make_workload_pairs(wl, seed=1)
    assert not np.array_equal(other["doc_ids"], pairs["doc_ids"])


@pytest.mark.parametrize("name", sorted(synth.WORKLOADS))
def test_prefix_lengths_follow_the_recipe(name):
    wl = synth.WORKLOADS[name]
    m = synth.doc_prefix_lengths(wl, seed=0)
    assert len(m) == wl.n_docs and set(m.tolist()) <= set(wl.m_choices)
    if len(wl.m_choices) > 1:  # drawn uniformly: every choice is well represented
        counts = np.array([(m == c).sum() for c in wl.m_choices])
        assert counts.min() > 0.15 * wl.n_docs
    np.testing.assert_array_equal(synth.doc_prefix_lengths(wl, seed=0), m)


def test_zipf_workload_reuses_popular_documents():
    wl = synth.WORKLOADS["qwen3-8b-zipf"]
    docs = synth.make_workload_pairs(wl, seed=0)["doc_ids"]
    counts = np.bincount(docs, minlength=wl.n_docs)
    # Zipf(1.1) candidate weights: the most popular documents recur across most queries'
    # lists, while a uniform draw of 100 of 1,000 documents would put each in about 10 %
    top = np.sort(counts)[::-1]
    assert top[0] >= 0.9 * wl.n_queries
    assert top[:10].mean() > 5 * counts.mean()
    # the headline (m = 64) and the uncompressed workloads score exactly the same pairs
    for other in ("qwen3-8b-m64", "qwen3-8b-fulldoc"):
        o = synth.make_workload_pairs(synth.WORKLOADS[other], seed=0)
        ref = synth.make_workload_pairs(wl, seed=0)
        for key in ("q_offsets", "q_tokens", "doc_ids"):
            np.testing.assert_array_equal(o[key], ref[key])


def test_uncompressed_run_prepends_the_fixed_document_text():
    wl = synth.WORKLOADS["qwen3-8b-fulldoc"]
    base = synth.make_workload_pairs(wl, seed=0)
    full = bench.build_pairs(wl, 0)
    for p in (0, 1, 137):
        d = int(base["doc_ids"][p])
        doc = synth.make_fulldoc_tokens(wl, d, seed=0)
        assert len(doc) == 512
        seq = full["q_tokens"][full["q_offsets"][p]:full["q_offsets"][p + 1]]
        q = base["q_tokens"][base["q_offsets"][p]:base["q_offsets"][p + 1]]
        np.testing.assert_array_equal(seq, np.concatenate([doc, q]))
    # the same document's text is the same in every pair that names it
    d0 = int(base["doc_ids"][0])
    same = np.where(base["doc_ids"] == d0)[0]
    for p in same[:3]:
        seq = full["q_tokens"][full["q_offsets"][p]:full["q_offsets"][p] + 512]
        np.testing.assert_array_equal(seq, synth.make_fulldoc_tokens(wl, d0, seed=0))
