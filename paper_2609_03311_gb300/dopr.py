"""Thin ctypes binding of libdopr.so (the C ABI in include/dopr.h).

Only argument marshalling lives here: every step of the scoring pass runs in
the library's CUDA kernels.  Importing this module loads the library and
raises if it has not been built (``python -m paper_2609_03311_gb300.build``);
there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

from . import build as _build

_LIB = None

(OK, ERR_INVALID_ARG, ERR_UNKNOWN_DOC, ERR_INCOMPLETE, ERR_OUT_OF_MEMORY, ERR_CUDA, ERR_TIMEOUT, ERR_UNSUPPORTED,
 ERR_INTERNAL, ERR_RANGE) = range(10)
STATUS_NAMES = ["OK", "INVALID_ARG", "UNKNOWN_DOC", "INCOMPLETE", "OUT_OF_MEMORY", "CUDA", "TIMEOUT", "UNSUPPORTED",
                "INTERNAL", "RANGE"]

(W_EMBED, W_ATTN_NORM, W_Q, W_K, W_V, W_Q_NORM, W_K_NORM, W_O, W_MLP_NORM, W_GATE, W_UP, W_DOWN, W_FINAL_NORM,
 W_SCORE_HEAD) = range(14)

EPI_STORE, EPI_RESID_ADD, EPI_SWIGLU = 0, 1, 2


class DoprError(RuntimeError):
    def __init__(self, status: int, msg: str):
        self.status = status
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__(f"DOPR_ERR_{name}: {msg}")


class KernelStat(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 24), ("launches", ctypes.c_int64), ("time_ms", ctypes.c_double),
                ("flops", ctypes.c_double), ("bytes", ctypes.c_double)]


class ModelConfig(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("n_layers", "hidden", "n_q_heads", "n_kv_heads", "head_dim", "ffn",
                                              "vocab", "score_token_id", "max_position")] + \
               [("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float)]


def lib_path() -> str:
    """The library this process loads: the checked build when DOPR_CHECKED=1."""
    return _build.LIB_CHECKED if os.environ.get("DOPR_CHECKED") == "1" else _build.LIB


def load():
    """Load libdopr.so; raises OSError if it is missing."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = lib_path()
    if not os.path.exists(path):
        raise OSError(f"libdopr.so not built at {path}; run paper_2609_03311_gb300.build.build()")
    L = ctypes.CDLL(path)
    P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    sig = {
        "dopr_model_create": ([P, P], i32),
        "dopr_model_put_weight": ([P, i32, i32, P, i64, i32], i32),
        "dopr_model_destroy": ([P], i32),
        "dopr_store_create": ([P, i64, i64, P], i32),
        "dopr_store_put": ([P, i64, i32, i32, P, P, i32], i32),
        "dopr_store_destroy": ([P], i32),
        "dopr_prefix_bytes": ([P, i32], i64),
        "dopr_score": ([P, P, i32, P, P, P, P, P, i32], i32),
        "dopr_debug_pack_plan": ([P, P, i32, P, P, P, P, P, P, P, P], i32),
        "dopr_debug_gemm": ([i32, i32, i32, P, P, P, i32, P], i32),
        "dopr_debug_wait_timeout": ([i32], i32),
        "dopr_pack_order_noalloc": ([P, i32, P, P, P, P, P], i32),
        "dopr_profile_enable": ([P, i32], i32),
        "dopr_profile_read": ([P, P, i32], i32),
        "dopr_build_prefixes": ([P, P, i32, P, P, P, i32, P], i32),
        "dopr_debug_store_read": ([P, i64, i32, P, P], i32),
        "dopr_debug_attention_plan": ([i32, i32, i32, P, i32, P], i32),
        "dopr_select_prefix_inputs": ([P, i32, P, P, i32, i32, P, P, P, P], i32),
        "dopr_model_set_mlp_head": ([P, i32, i32, P, P, P, ctypes.c_float, i32], i32),
        "dopr_last_error": ([], ctypes.c_char_p),
        "dopr_version": ([], ctypes.c_char_p),
    }
    for name, (args, res) in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = res
    _LIB = L
    return L


def _check(status: int):
    if status != OK:
        raise DoprError(status, load().dopr_last_error().decode())


def _ptr(x):
    """Pointer of a torch tensor or numpy array (None passes NULL)."""
    if x is None:
        return None
    if isinstance(x, torch.Tensor):
        return ctypes.c_void_p(x.data_ptr())
    return x.ctypes.data_as(ctypes.c_void_p)


def _host(a, dtype):
    if isinstance(a, torch.Tensor):
        a = a.cpu().numpy()
    return np.ascontiguousarray(np.asarray(a, dtype=dtype))


def make_config(shape, max_position: int = 8192) -> ModelConfig:
    """ModelConfig from any object with the synth.ModelShape fields."""
    c = ModelConfig()
    c.n_layers, c.hidden, c.n_q_heads, c.n_kv_heads = shape.n_layers, shape.hidden, shape.n_q_heads, shape.n_kv_heads
    c.head_dim, c.ffn, c.vocab = shape.head_dim, shape.ffn, shape.vocab
    c.score_token_id = shape.score_token_id
    c.max_position = max_position
    c.rope_theta, c.rms_eps = shape.rope_theta, shape.rms_eps
    return c


def prefix_bytes(cfg: ModelConfig, m: int) -> int:
    return int(load().dopr_prefix_bytes(ctypes.byref(cfg), int(m)))


def version() -> str:
    return load().dopr_version().decode()


_PER_LAYER = [("attn_norm", W_ATTN_NORM), ("wq", W_Q), ("wk", W_K), ("wv", W_V), ("q_norm", W_Q_NORM),
              ("k_norm", W_K_NORM), ("wo", W_O), ("mlp_norm", W_MLP_NORM), ("w_gate", W_GATE), ("w_up", W_UP),
              ("w_down", W_DOWN)]


class Model:
    """A decoder on the GPU.  ``weights`` follows synth.make_weights (bf16
    torch tensors on the host or the current CUDA device)."""

    def __init__(self, cfg: ModelConfig, weights: dict | None = None):
        self.cfg = cfg
        self._h = ctypes.c_void_p()
        _check(load().dopr_model_create(ctypes.byref(cfg), ctypes.byref(self._h)))
        if weights is not None:
            self.put_weights(weights)

    def put(self, kind: int, layer: int, t: torch.Tensor):
        assert t.dtype == torch.bfloat16
        t = t.contiguous()
        _check(load().dopr_model_put_weight(self._h, kind, layer, _ptr(t), t.numel(), int(t.is_cuda)))

    def put_weights(self, w: dict):
        self.put(W_EMBED, 0, w["embed"])
        self.put(W_FINAL_NORM, 0, w["final_norm"])
        self.put(W_SCORE_HEAD, 0, w["score_head"])
        for name, kind in _PER_LAYER:
            for l, t in enumerate(w[name]):
                self.put(kind, l, t)

    def close(self):
        if self._h:
            load().dopr_model_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Store:
    """Device prefix store for doc ids 0..max_doc_id in a pool of pool_bytes."""

    def __init__(self, cfg: ModelConfig, max_doc_id: int, pool_bytes: int):
        self.cfg = cfg
        self._h = ctypes.c_void_p()
        # the library places the store on the calling thread's current device
        self.device = torch.cuda.current_device() if torch.cuda.is_available() else 0
        _check(load().dopr_store_create(ctypes.byref(cfg), int(max_doc_id), int(pool_bytes), ctypes.byref(self._h)))

    def put_layer(self, doc_id: int, layer: int, k: torch.Tensor, v: torch.Tensor):
        """k, v: bf16 [m, n_kv_heads, 128] for one layer."""
        assert k.dtype == torch.bfloat16 and v.dtype == torch.bfloat16 and k.shape == v.shape
        k, v = k.contiguous(), v.contiguous()
        _check(load().dopr_store_put(self._h, int(doc_id), int(k.shape[0]), int(layer), _ptr(k), _ptr(v),
                                     int(k.is_cuda)))

    def put(self, doc_id: int, k: torch.Tensor, v: torch.Tensor):
        """k, v: bf16 [n_layers, m, n_kv_heads, 128]."""
        for l in range(k.shape[0]):
            self.put_layer(doc_id, l, k[l], v[l])

    def read_layer(self, doc_id: int, layer: int, m: int):
        """The stored (fp16) K and V of one layer as float16 [m, n_kv_heads, 128] numpy arrays."""
        shape = (m, self.cfg.n_kv_heads, self.cfg.head_dim)
        k, v = np.zeros(shape, np.float16), np.zeros(shape, np.float16)
        _check(load().dopr_debug_store_read(self._h, int(doc_id), int(layer), k.ctypes.data, v.ctypes.data))
        return k, v

    def close(self):
        if self._h:
            load().dopr_store_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def set_mlp_head(model: Model, head: dict | None):
    """Use the MLP scoring head {w1 bf16 [d, H], b1 bf16 [d], w2 bf16 [d], b2 float,
    act 0..3} instead of the yes/no rows; None restores the rows."""
    if head is None:
        _check(load().dopr_model_set_mlp_head(model._h, 0, 0, None, None, None, 0.0, 0))
        return
    w1, b1, w2 = (head[k].contiguous() for k in ("w1", "b1", "w2"))
    assert w1.dtype == b1.dtype == w2.dtype == torch.bfloat16
    _check(load().dopr_model_set_mlp_head(model._h, int(w1.shape[0]), int(head["act"]), _ptr(w1), _ptr(b1), _ptr(w2),
                                          float(head["b2"]), int(w1.is_cuda)))


def build_prefixes(model: Model, store: Store, doc_ids, x_offsets, x: torch.Tensor, stream=None):
    """Offline prefix construction: forward each document's representations
    x[x_offsets[d]:x_offsets[d+1]] (bf16 [rows, hidden], on the GPU or the host)
    and store every layer's keys and values for doc_ids[d]."""
    di, xo = _host(doc_ids, np.int64), _host(x_offsets, np.int32)
    assert x.dtype == torch.bfloat16 and x.dim() == 2
    x = x.contiguous()
    st = ctypes.c_void_p(stream.cuda_stream if stream is not None else
                         (torch.cuda.current_stream().cuda_stream if x.is_cuda else 0))
    _check(load().dopr_build_prefixes(model._h, store._h, len(di), di.ctypes.data, xo.ctypes.data, _ptr(x),
                                      int(x.is_cuda), st))


def select_prefix_inputs(model: Model, doc_offsets, doc_tokens, top_k: int, top_p: int, stream=None):
    """Attention-based key token selection: (positions int32 [n_docs, top_k]
    ascending with -1 padding, states bf16 [n_docs, top_k, hidden], salience
    float32 [tokens])."""
    off, tok = _host(doc_offsets, np.int32), _host(doc_tokens, np.int32)
    n = len(off) - 1
    H = model.cfg.hidden
    pos = np.full((max(n, 1), top_k), -1, np.int32)
    x = torch.zeros((max(n, 1), top_k, H), dtype=torch.bfloat16)
    u = np.zeros(max(int(off[-1]) if n > 0 else 0, 1), np.float32)
    st = ctypes.c_void_p(stream.cuda_stream if stream is not None else torch.cuda.current_stream().cuda_stream)
    _check(load().dopr_select_prefix_inputs(model._h, n, off.ctypes.data, tok.ctypes.data, int(top_k), int(top_p),
                                            pos.ctypes.data, _ptr(x), u.ctypes.data, st))
    return pos[:n], x[:n], u[:int(off[-1]) if n > 0 else 0]


def score(model: Model, store: Store, q_offsets, q_tokens, doc_ids, out=None, stream=None) -> torch.Tensor:
    """Score pairs.  CUDA tensors in -> scored in place on the device
    (io_on_device=1); anything else -> host arrays copied by the library."""
    n = len(q_offsets) - 1
    st = ctypes.c_void_p(stream.cuda_stream if stream is not None else torch.cuda.current_stream().cuda_stream)
    if isinstance(q_offsets, torch.Tensor) and q_offsets.is_cuda:
        assert q_offsets.dtype == torch.int32 and q_tokens.dtype == torch.int32 and doc_ids.dtype == torch.int64
        if out is None:
            out = torch.empty(n, dtype=torch.float32, device=q_offsets.device)
        _check(load().dopr_score(model._h, store._h, n, _ptr(q_offsets), _ptr(q_tokens), _ptr(doc_ids), _ptr(out),
                                 st, 1))
        return out
    qo, qt, di = _host(q_offsets, np.int32), _host(q_tokens, np.int32), _host(doc_ids, np.int64)
    if out is None:
        out = torch.empty(n, dtype=torch.float32)
    assert out.device.type == "cpu" and out.dtype == torch.float32
    _check(load().dopr_score(model._h, store._h, n, _ptr(qo), _ptr(qt) if qt.size else None, _ptr(di), _ptr(out),
                             st, 0))
    return out


def pack_plan(model: Model, store: Store, q_offsets, q_tokens, doc_ids) -> dict:
    qo, qt, di = _host(q_offsets, np.int32), _host(q_tokens, np.int32), _host(doc_ids, np.int64)
    n = len(qo) - 1
    T = int(qo[-1] - qo[0]) + n if n > 0 else 0
    perm = np.zeros(max(n, 1), np.int32)
    tok_off = np.zeros(n + 1, np.int32)
    tok_pos = np.zeros(max(T, 1), np.int32)
    tok_id = np.zeros(max(T, 1), np.int32)
    tok_pair = np.zeros(max(T, 1), np.int32)
    _check(load().dopr_debug_pack_plan(model._h, store._h, n, _ptr(qo), _ptr(qt) if qt.size else None, _ptr(di),
                                       _ptr(perm), _ptr(tok_off), _ptr(tok_pos), _ptr(tok_id), _ptr(tok_pair)))
    return {"perm": perm[:n], "tok_off": tok_off, "tok_pos": tok_pos[:T], "tok_id": tok_id[:T],
            "tok_pair": tok_pair[:T]}


def attention_plan(m: int, rows_per_tile: int, tok_len) -> np.ndarray:
    """The attention tiles of one document's run of pairs (host-only, no GPU):
    int32 [n_tiles, 24] rows {kind, tok_begin, n_tok, n_keys, n_seg, 0, 0, 0, seg[16]}."""
    tl = _host(tok_len, np.int32)
    cap = int(tl.sum()) + 1
    out = np.zeros((cap, 24), np.int32)
    n = load().dopr_debug_attention_plan(int(m), int(rows_per_tile), len(tl), _ptr(tl), cap, _ptr(out))
    if n < 0:
        _check(-n)
    return out[:n]


def gemm(A: torch.Tensor, B: torch.Tensor, epilogue: int = EPI_STORE, out: torch.Tensor | None = None):
    """The projection kernel alone: A [M,K] fp16, B [N,K] fp16 (CUDA)."""
    assert A.dtype == torch.float16 and B.dtype == torch.float16 and A.is_contiguous() and B.is_contiguous()
    M, K = A.shape
    N = B.shape[0]
    if out is None:
        if epilogue == EPI_RESID_ADD:
            out = torch.zeros(M, N, dtype=torch.float32, device=A.device)
        elif epilogue == EPI_SWIGLU:
            out = torch.empty(M, N // 2, dtype=torch.float16, device=A.device)
        else:
            out = torch.empty(M, N, dtype=torch.float16, device=A.device)
    st = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    _check(load().dopr_debug_gemm(M, N, K, _ptr(A), _ptr(B), _ptr(out), epilogue, st))
    return out


def pack_order_noalloc(store: Store, q_offsets: torch.Tensor, doc_ids: torch.Tensor, perm: torch.Tensor,
                       tok_off: torch.Tensor, stream=None):
    """The allocation-free packer ordering step (device tensors in and out)."""
    assert q_offsets.is_cuda and doc_ids.is_cuda and perm.is_cuda and tok_off.is_cuda
    assert q_offsets.dtype == torch.int32 and doc_ids.dtype == torch.int64
    assert perm.dtype == torch.int32 and tok_off.dtype == torch.int32
    n = q_offsets.numel() - 1
    # the C ABI takes no buffer sizes: every extent the packer kernels index is checked here
    if n < 0 or doc_ids.numel() < n or perm.numel() < n or tok_off.numel() < n + 1:
        raise ValueError(f"pack_order_noalloc: buffers too short for {n} pairs (doc_ids {doc_ids.numel()}, "
                         f"perm {perm.numel()}, tok_off {tok_off.numel()}; need {n}, {n}, {n + 1})")
    for name, t in (("q_offsets", q_offsets), ("doc_ids", doc_ids), ("perm", perm), ("tok_off", tok_off)):
        if not t.is_contiguous() or t.device.index != store.device:
            raise ValueError(f"pack_order_noalloc: {name} must be contiguous on cuda:{store.device}")
    st = ctypes.c_void_p(stream.cuda_stream if stream is not None else torch.cuda.current_stream().cuda_stream)
    _check(load().dopr_pack_order_noalloc(store._h, n, _ptr(q_offsets), _ptr(doc_ids), _ptr(perm), _ptr(tok_off),
                                          st))


def profile_enable(model: Model, on: bool = True):
    """Clear the per-kernel counters; time each launch with CUDA events while on."""
    _check(load().dopr_profile_enable(model._h, int(bool(on))))


def profile_read(model: Model) -> dict:
    """{family: {launches, time_ms, flops, bytes}} accumulated since profile_enable."""
    buf = (KernelStat * 32)()
    n = load().dopr_profile_read(model._h, buf, 32)
    return {buf[i].name.decode(): {"launches": int(buf[i].launches), "time_ms": float(buf[i].time_ms),
                                   "flops": float(buf[i].flops), "bytes": float(buf[i].bytes)} for i in range(n)}


def wait_timeout_probe(timeout_ms: int) -> int:
    """Returns the status of the bounded-wait probe (TIMEOUT expected)."""
    return int(load().dopr_debug_wait_timeout(int(timeout_ms)))
