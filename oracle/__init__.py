"""fp64 CPU oracle for the DoPR online scoring pass (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product library never loads it and
shares no code with it.  The arithmetic lives in ``dopr_oracle.c`` (plain
loops, fp64); this module compiles it with gcc and marshals numpy arrays.

Method summary (DoPR, Sec. 3.1 and Sec. 3.4): a pair (q, d) is scored by running
the decoder over [q ; t_score] only, every layer attending to the document's
stored prefix key/value states before the causal online keys, and taking the
yes-minus-no logit at the score token.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dopr_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libdopr_oracle.so")
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB_PATH) -> str:
    """Compile the oracle with gcc (portable flags: the same source builds on
    x86_64 and aarch64).  Returns the path of the shared object."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", src, "-o", out + ".tmp", "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(out + ".tmp", out)
    return out


class _Model(ctypes.Structure):
    _fields_ = [
        ("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32),
        ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32), ("vocab", ctypes.c_int32),
        ("score_token_id", ctypes.c_int32),
        ("rope_theta", ctypes.c_double), ("rms_eps", ctypes.c_double),
        ("embed", ctypes.c_void_p),
        ("attn_norm", ctypes.c_void_p), ("wq", ctypes.c_void_p), ("wk", ctypes.c_void_p),
        ("wv", ctypes.c_void_p), ("q_norm", ctypes.c_void_p), ("k_norm", ctypes.c_void_p),
        ("wo", ctypes.c_void_p), ("mlp_norm", ctypes.c_void_p), ("w_gate", ctypes.c_void_p),
        ("w_up", ctypes.c_void_p), ("w_down", ctypes.c_void_p),
        ("final_norm", ctypes.c_void_p), ("score_head", ctypes.c_void_p),
    ]


def load(lib_path: str | None = None):
    """Load (building first if needed) the oracle shared object."""
    global _lib
    if lib_path is None and _lib is not None:
        return _lib
    # DOPR_ORACLE_LIB lets the mutation test point the pins at a modified build.
    path = lib_path or os.environ.get("DOPR_ORACLE_LIB") or build()
    lib = ctypes.CDLL(path)
    P = ctypes.c_void_p
    i32, f64 = ctypes.c_int32, ctypes.c_double
    lib.oracle_bf16_to_f64.argtypes = [ctypes.c_uint16]
    lib.oracle_bf16_to_f64.restype = f64
    lib.oracle_num_threads.restype = ctypes.c_int
    lib.oracle_rmsnorm.argtypes = [P, P, ctypes.c_int, f64, P]
    lib.oracle_rope.argtypes = [P, ctypes.c_int, f64, f64]
    lib.oracle_attend.argtypes = [P, P, P, ctypes.c_int, ctypes.c_int, f64, P]
    lib.oracle_silu.argtypes = [f64]
    lib.oracle_silu.restype = f64
    lib.oracle_forward.argtypes = [P, ctypes.c_int, P, ctypes.c_int, ctypes.c_int, P, P, P, P, P, P, P]
    lib.oracle_attn_probs.argtypes = [P, P, ctypes.c_int, ctypes.c_int, f64, P]
    lib.oracle_salience.argtypes = [ctypes.c_int, P, ctypes.c_int, P]
    lib.oracle_select_topk.argtypes = [ctypes.c_int, P, ctypes.c_int, P]
    lib.oracle_mlp_head.argtypes = [P, P, ctypes.c_int, P, P, P, f64, ctypes.c_int]
    lib.oracle_mlp_head.restype = f64
    lib.oracle_score_head.argtypes = [P, P]
    lib.oracle_score_head.restype = f64
    lib.oracle_embed.argtypes = [P, ctypes.c_int, P, P]
    lib.oracle_score_pairs.argtypes = [P, ctypes.c_int, P, P, P, P, P, P, P]
    lib.oracle_pack_plan.argtypes = [ctypes.c_int, P, P, P, P, i32, P, P, P, P, P]
    if lib_path is None:
        _lib = lib
    return lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _u16(a) -> np.ndarray:
    """bf16 payload as uint16 bit patterns (torch bf16 tensors or uint16 arrays)."""
    try:
        import torch

        if isinstance(a, torch.Tensor):
            assert a.dtype == torch.bfloat16, a.dtype
            return np.ascontiguousarray(a.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
    except ImportError:  # pragma: no cover
        pass
    a = np.asarray(a)
    assert a.dtype == np.uint16, a.dtype
    return np.ascontiguousarray(a)


def bf16_to_f64(a) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    u = _u16(a).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


@dataclass
class Shape:
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rope_theta: float = 1e6
    rms_eps: float = 1e-6
    score_token_id: int = 0


class OracleModel:
    """Decoder weights held as bf16 bit patterns, viewed by the C oracle.

    ``weights`` maps names to arrays (torch bf16 tensors or uint16):
    embed [V,H]; per layer lists attn_norm [H], wq [Hq*D,H], wk/wv [Hkv*D,H],
    q_norm/k_norm [D], wo [H,Hq*D], mlp_norm [H], w_gate/w_up [F,H],
    w_down [H,F]; final_norm [H]; score_head [2,H] (row 0 yes, row 1 no).
    """

    _PER_LAYER = ("attn_norm", "wq", "wk", "wv", "q_norm", "k_norm", "wo",
                  "mlp_norm", "w_gate", "w_up", "w_down")

    def __init__(self, shape: Shape, weights: dict, lib_path: str | None = None):
        self.shape = shape
        self.lib = load(lib_path)
        self._keep = []
        s = shape
        m = _Model()
        m.n_layers, m.hidden, m.n_q_heads, m.n_kv_heads = s.n_layers, s.hidden, s.n_q_heads, s.n_kv_heads
        m.head_dim, m.ffn, m.vocab, m.score_token_id = s.head_dim, s.ffn, s.vocab, s.score_token_id
        m.rope_theta, m.rms_eps = float(s.rope_theta), float(s.rms_eps)

        def hold(a):
            u = _u16(a)
            self._keep.append(u)
            return u.ctypes.data

        m.embed = hold(weights["embed"])
        self._final_norm = bf16_to_f64(weights["final_norm"])
        m.final_norm = hold(weights["final_norm"])
        m.score_head = hold(weights["score_head"])
        for name in self._PER_LAYER:
            arr = (ctypes.c_void_p * s.n_layers)(*[hold(w) for w in weights[name]])
            self._keep.append(arr)
            setattr(m, name, ctypes.cast(arr, ctypes.c_void_p).value)
        self._m = m

    @property
    def ref(self):
        return ctypes.byref(self._m)

    # -- whole-model entry points -------------------------------------
    def embed(self, ids) -> np.ndarray:
        ids = np.ascontiguousarray(np.asarray(ids, dtype=np.int32))
        x = np.zeros((len(ids), self.shape.hidden), dtype=np.float64)
        rc = self.lib.oracle_embed(self.ref, len(ids), _ptr(ids), _ptr(x))
        if rc != 0:
            raise ValueError(f"oracle_embed rc={rc}")
        return x

    def forward(self, x0, pos0: int, prefix_k=None, prefix_v=None, want_kv=False, want_attn=False,
                want_probs=False):
        """Causal pass over online vectors x0 [T,H] at positions pos0..;
        prefix_k/v: [L,m,Hkv,D] fp64 or None.  Returns dict with 'h' and
        optionally 'k', 'v' ([L,T,Hkv,D]), 'attn' ([L,T,Hq*D]) and 'probs'
        ([T, m+T], the last layer's head-averaged attention weights)."""
        s = self.shape
        x0 = _f64(x0)
        T = x0.shape[0]
        m = 0 if prefix_k is None else int(np.asarray(prefix_k).shape[1])
        pk = None if m == 0 else _f64(prefix_k)
        pv = None if m == 0 else _f64(prefix_v)
        h = np.zeros((T, s.hidden))
        k = np.zeros((s.n_layers, T, s.n_kv_heads, s.head_dim)) if want_kv else None
        v = np.zeros_like(k) if want_kv else None
        a = np.zeros((s.n_layers, T, s.n_q_heads * s.head_dim)) if want_attn else None
        pr = np.zeros((T, m + T)) if want_probs else None
        rc = self.lib.oracle_forward(self.ref, T, _ptr(x0), int(pos0), m, _ptr(pk), _ptr(pv),
                                     _ptr(h), _ptr(k), _ptr(v), _ptr(a), _ptr(pr))
        if rc != 0:
            raise ValueError(f"oracle_forward rc={rc}")
        out = {"h": h}
        if want_kv:
            out["k"], out["v"] = k, v
        if want_attn:
            out["attn"] = a
        if want_probs:
            out["probs"] = pr
        return out

    def select(self, ids, top_k: int, top_p: int):
        """Attention-based key token selection (Sec. 3.2.1) for one document of
        token ids: encode it alone at positions 0..n-1, salience u from the last
        layer's head-averaged attention, the top_k positions (ascending), and
        their final-layer states (after the final RMSNorm).
        Returns (u [n], positions [k], states [k, H])."""
        x = self.embed(ids)
        out = self.forward(x, 0, want_probs=True)
        n = len(ids)
        u = salience(out["probs"], top_p)
        pos = select_topk(u, top_k)
        g = self._final_norm
        states = np.stack([rmsnorm(out["h"][i], g, self.shape.rms_eps) for i in pos]) if len(pos) else \
            np.zeros((0, self.shape.hidden))
        return u, pos, states

    def score_head(self, h) -> float:
        h = _f64(h)
        return float(self.lib.oracle_score_head(self.ref, _ptr(h)))

    def mlp_head(self, h, head: dict) -> float:
        """The MLP scoring head on a final state h [H]; head: w1 bf16 [d, H],
        b1 bf16 [d], w2 bf16 [d], b2 float, act int."""
        h = _f64(h)
        w1, b1, w2 = _u16(head["w1"]), _u16(head["b1"]), _u16(head["w2"])
        return float(self.lib.oracle_mlp_head(self.ref, _ptr(h), int(w1.shape[0]), _ptr(w1), _ptr(b1), _ptr(w2),
                                              float(head["b2"]), int(head["act"])))

    def score_pairs(self, q_offsets, q_tokens, pair_doc, docs) -> np.ndarray:
        """docs: list of (K, V) per document index, each [L,m,Hkv,D] (fp64
        arrays, or bf16 payloads widened exactly here); pair_doc indexes docs."""
        n = len(q_offsets) - 1
        qo = np.ascontiguousarray(np.asarray(q_offsets, dtype=np.int32))
        qt = np.ascontiguousarray(np.asarray(q_tokens, dtype=np.int32))
        if qt.size == 0:
            qt = np.zeros(1, dtype=np.int32)
        pd = np.ascontiguousarray(np.asarray(pair_doc, dtype=np.int32))
        dk, dv, dm = [], [], []
        for K, V in docs:
            K = K if (isinstance(K, np.ndarray) and K.dtype == np.float64) else bf16_to_f64(K)
            V = V if (isinstance(V, np.ndarray) and V.dtype == np.float64) else bf16_to_f64(V)
            dk.append(_f64(K))
            dv.append(_f64(V))
            dm.append(int(K.shape[1]))
        dm = np.ascontiguousarray(np.asarray(dm if dm else [0], dtype=np.int32))
        kp = (ctypes.c_void_p * max(1, len(dk)))(*[a.ctypes.data for a in dk])
        vp = (ctypes.c_void_p * max(1, len(dv)))(*[a.ctypes.data for a in dv])
        out = np.zeros(max(n, 1), dtype=np.float64)
        rc = self.lib.oracle_score_pairs(self.ref, n, _ptr(qo), _ptr(qt), _ptr(pd), _ptr(dm),
                                         ctypes.cast(kp, ctypes.c_void_p), ctypes.cast(vp, ctypes.c_void_p),
                                         _ptr(out))
        if rc != 0:
            raise ValueError(f"oracle_score_pairs rc={rc}")
        return out[:n]


# -- single-op entry points (used by the pins) ---------------------------

def rmsnorm(x, g, eps) -> np.ndarray:
    lib = load()
    x, g = _f64(x), _f64(g)
    y = np.zeros_like(x)
    lib.oracle_rmsnorm(_ptr(x), _ptr(g), x.size, float(eps), _ptr(y))
    return y


def rope(x, pos, theta) -> np.ndarray:
    lib = load()
    y = _f64(x).copy()
    lib.oracle_rope(_ptr(y), y.size, float(pos), float(theta))
    return y


def attend(q, K, V, scale) -> np.ndarray:
    lib = load()
    q, K, V = _f64(q), _f64(K), _f64(V)
    out = np.zeros(q.size)
    lib.oracle_attend(_ptr(q), _ptr(K), _ptr(V), K.shape[0], q.size, float(scale), _ptr(out))
    return out


def attn_probs(q, K, scale) -> np.ndarray:
    q, K = _f64(q), _f64(K)
    n, D = K.shape
    p = np.zeros(n)
    load().oracle_attn_probs(_ptr(q), _ptr(K), n, D, float(scale), _ptr(p))
    return p


def salience(A, top_p: int) -> np.ndarray:
    """Column top-p means of a causal [n, n] attention matrix (Sec. 3.2.1)."""
    A = _f64(A)
    n = A.shape[0]
    u = np.zeros(n)
    rc = load().oracle_salience(n, _ptr(A), int(top_p), _ptr(u))
    if rc != 0:
        raise ValueError(f"oracle_salience rc={rc}")
    return u


def select_topk(u, K: int) -> np.ndarray:
    """Ascending positions of the K largest u (ties to the lower position)."""
    u = _f64(u)
    idx = np.zeros(max(len(u), 1), dtype=np.int32)
    k = load().oracle_select_topk(len(u), _ptr(u), int(K), _ptr(idx))
    if k < 0:
        raise ValueError("oracle_select_topk failed")
    return idx[:k]


def silu(x: float) -> float:
    return float(load().oracle_silu(float(x)))


def num_threads() -> int:
    return int(load().oracle_num_threads())


def pack_plan(q_offsets, q_tokens, doc_ids, pair_m, score_token_id):
    """Reference batch plan (see oracle_pack_plan).  Returns dict of int32 arrays."""
    lib = load()
    qo = np.ascontiguousarray(np.asarray(q_offsets, dtype=np.int32))
    n = len(qo) - 1
    qt = np.ascontiguousarray(np.asarray(q_tokens, dtype=np.int32))
    if qt.size == 0:
        qt = np.zeros(1, dtype=np.int32)
    di = np.ascontiguousarray(np.asarray(doc_ids, dtype=np.int64))
    pm = np.ascontiguousarray(np.asarray(pair_m, dtype=np.int32))
    T = int(qo[-1] - qo[0]) + n if n > 0 else 0
    perm = np.zeros(max(n, 1), np.int32)
    tok_off = np.zeros(n + 1, np.int32)
    tok_pos = np.zeros(max(T, 1), np.int32)
    tok_id = np.zeros(max(T, 1), np.int32)
    tok_pair = np.zeros(max(T, 1), np.int32)
    rc = lib.oracle_pack_plan(n, _ptr(qo), _ptr(qt), _ptr(di), _ptr(pm), int(score_token_id),
                              _ptr(perm), _ptr(tok_off), _ptr(tok_pos), _ptr(tok_id), _ptr(tok_pair))
    if rc != 0:
        raise ValueError(f"oracle_pack_plan rc={rc}")
    return {"perm": perm[:n], "tok_off": tok_off, "tok_pos": tok_pos[:T], "tok_id": tok_id[:T],
            "tok_pair": tok_pair[:T]}
