"""Seeded synthetic inputs for the DoPR online scoring pass.

This module only draws random numbers: decoder weights, stored prefix
states, queries and (query, document) pair lists.  It holds none of the
scoring arithmetic.  The same drawn bytes feed both the GPU library and the
fp64 oracle, so both sides always see identical inputs.

Recipe (shapes follow the Qwen3 backbones the paper uses, Sec. 4.1):
  * matrices N(0, 0.02) in fp32, rounded to bf16 (round-to-nearest-even);
  * norm gains 1.0 ("ones") or 1 + N(0, 0.1) ("random", used by tests so the
    gains are exercised);
  * stored prefix K and V N(0, 1) bf16.  A RoPE rotation of an isotropic
    Gaussian pair is again isotropic Gaussian, so these draws have the
    distribution of keys rotated at positions 0..m-1; no rotation is applied
    here because this module contains none of the method's arithmetic;
  * token ids uniform in [0, vocab); the score token is vocab - 1;
  * candidate lists: each query draws distinct documents, uniformly or with
    Zipf(s) weights over a seeded permutation of the collection (Gumbel
    top-k, i.e. sequential weighted sampling without replacement).

Every tensor has its own counter-derived sub-stream (seed, name, index), so
any tensor can be regenerated alone.
"""
from __future__ import annotations

import os
import zlib
from dataclasses import dataclass, field, replace

import numpy as np
import torch

__all__ = [
    "ModelShape", "Workload", "MODELS", "WORKLOADS", "sub_seed", "make_weights",
    "make_prefix", "make_prefix_batch", "make_workload_pairs", "make_fulldoc_tokens",
]


@dataclass(frozen=True)
class ModelShape:
    name: str
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rope_theta: float = 1e6
    rms_eps: float = 1e-6

    @property
    def score_token_id(self) -> int:
        return self.vocab - 1

    def with_layers(self, n_layers: int) -> "ModelShape":
        return replace(self, n_layers=n_layers, name=f"{self.name}-{n_layers}l")


QWEN3_VOCAB = 151936

MODELS = {
    "qwen3-0.6b": ModelShape("qwen3-0.6b", 28, 1024, 16, 8, 128, 3072, QWEN3_VOCAB),
    "qwen3-4b": ModelShape("qwen3-4b", 36, 2560, 32, 8, 128, 9728, QWEN3_VOCAB),
    "qwen3-8b": ModelShape("qwen3-8b", 36, 4096, 32, 8, 128, 12288, QWEN3_VOCAB),
}


@dataclass(frozen=True)
class Workload:
    """A scoring workload: model shape, document store and pair list."""
    name: str
    model: ModelShape
    n_docs: int
    m_choices: tuple            # prefix length per doc drawn uniformly from these
    n_queries: int
    docs_per_query: int
    qlen_min: int
    qlen_max: int
    zipf_s: float = 0.0         # 0 -> uniform candidate draw
    fulldoc_tokens: int = 0     # >0: the uncompressed comparison run
    pair_set: str = ""          # workloads naming the same pair set score the same pairs (default: own name)

    @property
    def n_pairs(self) -> int:
        return self.n_queries * self.docs_per_query


WORKLOADS = {
    # 2-layer Qwen3-0.6B-width model, 64 docs with m=64, 32 queries x 8 docs, 24-token queries.
    "qwen3-0.6b-2l": Workload("qwen3-0.6b-2l", MODELS["qwen3-0.6b"].with_layers(2), 64, (64,), 32, 8, 24, 24),
    # Full Qwen3-0.6B, 1000 docs m=64, 100 x 100 pairs, queries 8..64 tokens.
    "qwen3-0.6b": Workload("qwen3-0.6b", MODELS["qwen3-0.6b"], 1000, (64,), 100, 100, 8, 64),
    # Qwen3-4B, 2000 docs m=128, 50 x 200 pairs, queries 32..256 tokens.
    "qwen3-4b": Workload("qwen3-4b", MODELS["qwen3-4b"], 2000, (128,), 50, 200, 32, 256),
    # Qwen3-8B, 1000 docs m in {32,64,128,256}, 200 x 100 Zipf(1.1) pairs, queries 8..64.
    "qwen3-8b-zipf": Workload("qwen3-8b-zipf", MODELS["qwen3-8b"], 1000, (32, 64, 128, 256), 200, 100, 8, 64, 1.1,
                              pair_set="qwen3-8b-m64"),
    # The same pairs with every prefix m=64 (the headline workload).
    "qwen3-8b-m64": Workload("qwen3-8b-m64", MODELS["qwen3-8b"], 1000, (64,), 200, 100, 8, 64, 1.1),
    # The same pairs scored uncompressed: [512 doc tokens ; query ; score token], no prefix.
    "qwen3-8b-fulldoc": Workload("qwen3-8b-fulldoc", MODELS["qwen3-8b"], 1000, (0,), 200, 100, 8, 64, 1.1, 512,
                                 pair_set="qwen3-8b-m64"),
}


def sub_seed(seed: int, *tags) -> int:
    """Counter-style sub-stream seed: splitmix64 over (seed, crc32 of each tag)."""
    x = (int(seed) * 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF
    for t in tags:
        x ^= zlib.crc32(str(t).encode()) & 0xFFFFFFFF
        x = (x + 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF
        z = x
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & 0xFFFFFFFFFFFFFFFF
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & 0xFFFFFFFFFFFFFFFF
        x = z ^ (z >> 31)
    return x & 0x7FFFFFFFFFFFFFFF


def _generator(device, seed: int, *tags) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(sub_seed(seed, *tags))
    return g


def _normal_bf16(shape, std, device, seed, *tags, portable=False) -> torch.Tensor:
    if portable:
        # float64 draws of torch's CPU generator: its double normal path is scalar
        # Box-Muller on the Mersenne-Twister stream on every host CPU (the float32
        # path is vectorised differently on x86 and Arm), so after rounding to bf16
        # the same seed gives the same bytes on either machine
        g = _generator("cpu", seed, *tags)
        x = torch.randn(shape, generator=g, dtype=torch.float64)
        if std != 1.0:
            x.mul_(std)
        return x.to(torch.bfloat16).to(device)
    g = _generator(device, seed, *tags)
    x = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(torch.bfloat16)


def _gain_bf16(n, norms, device, seed, *tags, portable=False) -> torch.Tensor:
    if norms == "ones":
        return torch.ones(n, device=device, dtype=torch.bfloat16)
    if portable:
        g = _generator("cpu", seed, *tags)
        x = 1.0 + 0.1 * torch.randn(n, generator=g, dtype=torch.float64)
        return x.to(torch.bfloat16).to(device)
    g = _generator(device, seed, *tags)
    x = 1.0 + 0.1 * torch.randn(n, generator=g, device=device, dtype=torch.float32)
    return x.to(torch.bfloat16)


def make_weights(shape: ModelShape, seed: int = 0, device="cpu", norms: str = "ones",
                 std: float = 0.02, zero: tuple = (), portable: bool = False) -> dict:
    """Random-init bf16 decoder weights.  ``zero`` names tensors to set to 0
    (used by closed-form checks).  Layout: matrices are [out, in].

    ``portable`` draws every tensor from the host generator in float64 (see
    _normal_bf16), so the bytes are the same on any host and do not depend on
    the GPU: stored expected values computed on one machine then hold on
    another.  The tensors are drawn in parallel threads (one sub-stream each)."""
    s = shape
    D, Hq, Hkv, H, F = s.head_dim, s.n_q_heads, s.n_kv_heads, s.hidden, s.ffn

    def mat(name, l, rows, cols):
        if name in zero:
            return lambda: torch.zeros(rows, cols, device=device, dtype=torch.bfloat16)
        return lambda: _normal_bf16((rows, cols), std, device, seed, name, l, portable=portable)

    def gain(n, name, *tags):
        return lambda: _gain_bf16(n, norms, device, seed, name, *tags, portable=portable)

    jobs = {
        ("embed",): lambda: _normal_bf16((s.vocab, H), std, device, seed, "embed", portable=portable),
        ("final_norm",): gain(H, "final_norm"),
        ("score_head",): mat("score_head", 0, 2, H),
    }
    for l in range(s.n_layers):
        jobs[("attn_norm", l)] = gain(H, "attn_norm", l)
        jobs[("wq", l)] = mat("wq", l, Hq * D, H)
        jobs[("wk", l)] = mat("wk", l, Hkv * D, H)
        jobs[("wv", l)] = mat("wv", l, Hkv * D, H)
        jobs[("q_norm", l)] = gain(D, "q_norm", l)
        jobs[("k_norm", l)] = gain(D, "k_norm", l)
        jobs[("wo", l)] = mat("wo", l, H, Hq * D)
        jobs[("mlp_norm", l)] = gain(H, "mlp_norm", l)
        jobs[("w_gate", l)] = mat("w_gate", l, F, H)
        jobs[("w_up", l)] = mat("w_up", l, F, H)
        jobs[("w_down", l)] = mat("w_down", l, H, F)
    if portable:
        from concurrent.futures import ThreadPoolExecutor

        keys = sorted(jobs, key=lambda k: k != ("embed",))  # the largest draw first
        with ThreadPoolExecutor(max_workers=max(1, min(32, os.cpu_count() or 1))) as ex:
            done = dict(zip(keys, ex.map(lambda k: jobs[k](), keys)))
    else:
        done = {k: f() for k, f in jobs.items()}
    w = {"embed": done[("embed",)], "final_norm": done[("final_norm",)], "score_head": done[("score_head",)]}
    for name in ("attn_norm", "wq", "wk", "wv", "q_norm", "k_norm", "wo", "mlp_norm", "w_gate", "w_up", "w_down"):
        w[name] = [done[(name, l)] for l in range(s.n_layers)]
    return w


def make_prefix(shape: ModelShape, m: int, doc: int, seed: int = 0, device="cpu", portable: bool = False):
    """Stored prefix states of one document: K, V bf16 [L, m, Hkv, D], N(0,1)
    (``portable`` as in make_weights)."""
    s = shape
    k = _normal_bf16((s.n_layers, m, s.n_kv_heads, s.head_dim), 1.0, device, seed, "prefix_k", doc, portable=portable)
    v = _normal_bf16((s.n_layers, m, s.n_kv_heads, s.head_dim), 1.0, device, seed, "prefix_v", doc, portable=portable)
    return k, v


def make_doc_representations(shape: ModelShape, doc_m: dict, seed: int = 0, device="cpu"):
    """Selected document representations c_1..c_m per document (the prefix
    inputs of offline prefix construction): bf16 rows ~ N(0,1) of width hidden,
    documents in sorted doc-id order.  Returns (doc_ids int64, x_offsets int32
    [n+1], x bf16 [sum m, hidden])."""
    docs = sorted(doc_m)
    offs = np.concatenate([[0], np.cumsum([doc_m[d] for d in docs])]).astype(np.int32)
    parts = [_normal_bf16((doc_m[d], shape.hidden), 1.0, device, seed, "doc_repr", d) for d in docs]
    x = torch.cat(parts) if parts else torch.zeros((0, shape.hidden), dtype=torch.bfloat16, device=device)
    return np.asarray(docs, dtype=np.int64), offs, x


def make_prefix_batch(shape: ModelShape, m: int, docs, seed: int = 0, device="cpu"):
    """Prefix states for many documents of the same m in one draw per doc
    group: K, V bf16 [n_docs, L, m, Hkv, D].  The sub-stream is keyed by
    (m, first doc id, count), so it is reproducible for the same doc list."""
    docs = list(docs)
    s = shape
    shp = (len(docs), s.n_layers, m, s.n_kv_heads, s.head_dim)
    tag = (m, docs[0] if docs else -1, len(docs))
    k = _normal_bf16(shp, 1.0, device, seed, "prefix_k_batch", *tag)
    v = _normal_bf16(shp, 1.0, device, seed, "prefix_v_batch", *tag)
    return k, v


def doc_prefix_lengths(wl: Workload, seed: int = 0) -> np.ndarray:
    rng = np.random.default_rng(sub_seed(seed, "doc_m", wl.name))
    choices = np.asarray(wl.m_choices, dtype=np.int32)
    return choices[rng.integers(0, len(choices), size=wl.n_docs)]


def make_workload_pairs(wl: Workload, seed: int = 0):
    """Pair list of a workload.  Returns dict with q_offsets [n+1] int32,
    q_tokens int32, doc_ids [n] int64, query_of_pair [n] int32 (pairs are
    listed query by query, each query's candidates in draw order)."""
    rng = np.random.default_rng(sub_seed(seed, "pairs", wl.pair_set or wl.name))
    n_docs, k = wl.n_docs, wl.docs_per_query
    if wl.zipf_s > 0:
        order = rng.permutation(n_docs)            # rank -> doc id
        ranks = np.arange(1, n_docs + 1, dtype=np.float64)
        logw = -wl.zipf_s * np.log(ranks)
    doc_ids, qlens, qid = [], [], []
    for q in range(wl.n_queries):
        if wl.zipf_s > 0:
            gumbel = -np.log(-np.log(rng.random(n_docs)))
            top = np.argsort(-(logw + gumbel), kind="stable")[:k]
            cands = order[top]
        else:
            cands = rng.choice(n_docs, size=k, replace=False)
        L = int(rng.integers(wl.qlen_min, wl.qlen_max + 1))
        for d in cands:
            doc_ids.append(int(d))
            qlens.append(L)
            qid.append(q)
    # one token sequence per query, shared by its candidate pairs
    q_tok = [rng.integers(0, wl.model.vocab, size=qlens[i * k], dtype=np.int64) for i in range(wl.n_queries)]
    offs = np.zeros(len(doc_ids) + 1, dtype=np.int64)
    np.cumsum(qlens, out=offs[1:])
    toks = np.concatenate([q_tok[q] for q in qid]) if qid else np.zeros(0, np.int64)
    return {
        "q_offsets": offs.astype(np.int32),
        "q_tokens": toks.astype(np.int32),
        "doc_ids": np.asarray(doc_ids, dtype=np.int64),
        "query_of_pair": np.asarray(qid, dtype=np.int32),
    }


def make_fulldoc_tokens(wl: Workload, doc: int, seed: int = 0) -> np.ndarray:
    """The fixed random document text of one doc for the uncompressed run."""
    rng = np.random.default_rng(sub_seed(seed, "fulldoc", doc))
    return rng.integers(0, wl.model.vocab, size=wl.fulldoc_tokens, dtype=np.int64).astype(np.int32)


def random_pairs(n_pairs: int, n_docs: int, qlen_min: int, qlen_max: int, vocab: int, seed: int = 0,
                 doc_id_base: int = 0):
    """Small ad-hoc pair lists for tests: independent queries, docs drawn
    with replacement."""
    rng = np.random.default_rng(sub_seed(seed, "random_pairs", n_pairs, n_docs))
    lens = rng.integers(qlen_min, qlen_max + 1, size=n_pairs)
    offs = np.zeros(n_pairs + 1, dtype=np.int64)
    np.cumsum(lens, out=offs[1:])
    toks = rng.integers(0, vocab, size=int(offs[-1]))
    docs = doc_id_base + rng.integers(0, n_docs, size=n_pairs)
    return {"q_offsets": offs.astype(np.int32), "q_tokens": toks.astype(np.int32),
            "doc_ids": docs.astype(np.int64)}
