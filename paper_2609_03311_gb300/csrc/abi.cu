// abi.cu -- C ABI of libdopr (include/dopr.h): the model and prefix-store
// objects, host-side validation, and the engine that runs the online scoring
// pass (DoPR Sec. 3.4) as a sequence of sm_103a kernels on the caller's stream.
//
// Engine of dopr_score:
//   1. validate (host inputs on the host; device inputs in the packer kernel);
//   2. device packer part 1: stable sort by doc id, packed token offsets;
//   3. one small device->host read (offsets, slots, error word) to size launches;
//   4. host splits the sorted pairs into chunks of whole pairs (<= chunk_cap
//      tokens) and each chunk into attention work items (runs of <= 8 pairs of
//      one document); packer part 2 writes token ids and positions;
//   5. per chunk: embed+norm, then per layer QKV GEMM, QK-norm+RoPE, attention
//      over prefix + causal keys, O GEMM (+residual), norm, gate/up GEMM
//      (+SwiGLU), down GEMM (+residual), next norm; finally the score head,
//      which scatters scores to input order.
#include <cudaTypedefs.h>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "device_common.cuh"
#include "internal.h"

struct dopr_model : dopr::Model {};
struct dopr_store : dopr::Store {};

namespace dopr {

// A named NVTX range for the lifetime of the object (per call, chunk and layer), so a
// profiler can attribute kernels; it costs a function call when no tool is attached.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  NvtxRange(const char* fmt, int v) {
    char b[48];
    snprintf(b, sizeof b, fmt, v);
    nvtxRangePushA(b);
  }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};
namespace {

thread_local std::string g_last_error;

dopr_status fail(dopr_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

#define CUDA_TRY(call)                                                                            \
  do {                                                                                            \
    cudaError_t e_ = (call);                                                                      \
    if (e_ != cudaSuccess)                                                                        \
      return fail(e_ == cudaErrorMemoryAllocation ? DOPR_ERR_OUT_OF_MEMORY : DOPR_ERR_CUDA,       \
                  "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, __LINE__);   \
  } while (0)

#define STATUS_TRY(call)            \
  do {                              \
    dopr_status s_ = (call);        \
    if (s_ != DOPR_OK) return s_;   \
  } while (0)

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

dopr_status check_cfg(const dopr_model_config* c) {
  if (!c) return fail(DOPR_ERR_INVALID_ARG, "config is NULL");
  if (c->n_layers <= 0 || c->hidden <= 0 || c->n_q_heads <= 0 || c->n_kv_heads <= 0 || c->ffn <= 0 ||
      c->vocab <= 0 || c->max_position <= 0)
    return fail(DOPR_ERR_INVALID_ARG, "config sizes must be positive");
  if (c->score_token_id < 0 || c->score_token_id >= c->vocab)
    return fail(DOPR_ERR_INVALID_ARG, "score_token_id %d outside [0, vocab)", c->score_token_id);
  if (!(c->rope_theta > 0.f) || !(c->rms_eps >= 0.f)) return fail(DOPR_ERR_INVALID_ARG, "bad rope_theta / rms_eps");
  if (c->head_dim != HEAD_DIM) return fail(DOPR_ERR_UNSUPPORTED, "head_dim must be 128 (got %d)", c->head_dim);
  if (c->n_q_heads % c->n_kv_heads) return fail(DOPR_ERR_UNSUPPORTED, "n_q_heads must be a multiple of n_kv_heads");
  const int G = c->n_q_heads / c->n_kv_heads;
  if (16 % G != 0 && G % 16 != 0) return fail(DOPR_ERR_UNSUPPORTED, "GQA group size %d not supported", G);
  if (c->hidden % GEMM_BN) return fail(DOPR_ERR_UNSUPPORTED, "hidden must be a multiple of 256");
  if (c->ffn % 128) return fail(DOPR_ERR_UNSUPPORTED, "ffn must be a multiple of 128");
  if (((c->n_q_heads + 2 * c->n_kv_heads) * HEAD_DIM) % GEMM_BN)
    return fail(DOPR_ERR_UNSUPPORTED, "(n_q_heads + 2 n_kv_heads) * 128 must be a multiple of 256");
  if ((c->n_q_heads * HEAD_DIM) % GEMM_BK) return fail(DOPR_ERR_UNSUPPORTED, "n_q_heads * 128 % 64");
  if (c->max_position > (1 << 20)) return fail(DOPR_ERR_UNSUPPORTED, "max_position above 2^20");
  return DOPR_OK;
}

template <typename T>
dopr_status dev_alloc(T** p, size_t count) {
  *p = nullptr;
  if (count == 0) return DOPR_OK;
  CUDA_TRY(cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T)));
  return DOPR_OK;
}
template <typename T>
void dev_free(T*& p) {
  if (p) cudaFree(p);
  p = nullptr;
}
template <typename T>
dopr_status host_alloc(T** p, size_t count) {
  *p = nullptr;
  if (count == 0) return DOPR_OK;
  CUDA_TRY(cudaMallocHost(reinterpret_cast<void**>(p), count * sizeof(T)));
  return DOPR_OK;
}
template <typename T>
void host_free(T*& p) {
  if (p) cudaFreeHost(p);
  p = nullptr;
}

int32_t kind_count() { return DOPR_W_SCORE_HEAD + 1; }
bool kind_is_global(int32_t k) {
  return k == DOPR_W_EMBED || k == DOPR_W_FINAL_NORM || k == DOPR_W_SCORE_HEAD;
}

void free_store(Store* s) {
  dev_free(s->pool); dev_free(s->d_slot_of); dev_free(s->d_slot_m); dev_free(s->d_slot_row); dev_free(s->d_slot_ok);
  dev_free(s->d_range);
}

void free_workspace(Workspace& w) {
  dev_free(w.r); dev_free(w.xn); dev_free(w.qkv); dev_free(w.o); dev_free(w.act);
  dev_free(w.ss_e); dev_free(w.ss_a); dev_free(w.ss_m); dev_free(w.r_s); dev_free(w.ss_s);
  dev_free(w.q_off); dev_free(w.q_tok); dev_free(w.doc_ids); dev_free(w.scores);
  dev_free(w.pair_slot); dev_free(w.perm); dev_free(w.sorted_slot); dev_free(w.tok_off);
  dev_free(w.tok_id); dev_free(w.tok_pos); dev_free(w.tok_pair); dev_free(w.doc_count);
  dev_free(w.items); dev_free(w.tiles); dev_free(w.err);
  host_free(w.h_tok_off); host_free(w.h_sorted_slot); host_free(w.h_err); host_free(w.h_items);
  host_free(w.h_tiles);
  dev_free(w.sel_A); dev_free(w.sel_a_off); dev_free(w.sel_u); dev_free(w.sel_pos); dev_free(w.sel_x);
  if (w.sel_empty) {
    free_store(w.sel_empty);
    delete static_cast<dopr_store*>(w.sel_empty);
  }
  w = Workspace{};
}

void free_model(Model* m) {
  dev_free(m->embed); dev_free(m->attn_norm); dev_free(m->w_qkv); dev_free(m->q_norm); dev_free(m->k_norm);
  dev_free(m->w_o); dev_free(m->mlp_norm); dev_free(m->w_gu); dev_free(m->w_down); dev_free(m->final_norm);
  dev_free(m->score_head); dev_free(m->rope);
  dev_free(m->mlp_w1); dev_free(m->mlp_b1); dev_free(m->mlp_w2);
  free_workspace(m->ws);
  for (cudaEvent_t e : m->prof.events) cudaEventDestroy(e);
  m->prof.events.clear();
}

dopr_status build_weight_maps(Model* m) {
  const auto& c = m->cfg;
  const int H = c.hidden, F = c.ffn, L = c.n_layers;
  m->tm_qkv.resize(L); m->tm_o.resize(L); m->tm_gu.resize(L); m->tm_down.resize(L);
  for (int l = 0; l < L; ++l) {
    bool ok = make_tmap_16b_2d(&m->tm_qkv[l], m->w_qkv + (size_t)l * m->qkv_dim * H, H, m->qkv_dim, (uint64_t)H * 2,
                               GEMM_BK, GEMM_B_BOX, true, true) &&
              make_tmap_16b_2d(&m->tm_o[l], m->w_o + (size_t)l * H * m->o_dim, m->o_dim, H, (uint64_t)m->o_dim * 2,
                               GEMM_BK, GEMM_B_BOX, true, true) &&
              make_tmap_16b_2d(&m->tm_gu[l], m->w_gu + (size_t)l * 2 * F * H, H, 2 * F, (uint64_t)H * 2, GEMM_BK,
                               GEMM_B_BOX, true, true) &&
              make_tmap_16b_2d(&m->tm_down[l], m->w_down + (size_t)l * H * F, F, H, (uint64_t)F * 2, GEMM_BK,
                               GEMM_B_BOX, true, true);
    if (!ok) return fail(DOPR_ERR_CUDA, "cuTensorMapEncodeTiled failed for layer %d weights", l);
  }
  m->maps_ok = true;
  return DOPR_OK;
}

dopr_status alloc_chunk_buffers(Model* m, int cap) {
  const auto& c = m->cfg;
  Workspace& w = m->ws;
  w.chunk_cap = cap;
  STATUS_TRY(dev_alloc(&w.r, (size_t)cap * c.hidden));
  STATUS_TRY(dev_alloc(&w.xn, (size_t)cap * c.hidden));
  STATUS_TRY(dev_alloc(&w.qkv, (size_t)cap * m->qkv_dim));
  STATUS_TRY(dev_alloc(&w.o, (size_t)cap * m->o_dim));
  STATUS_TRY(dev_alloc(&w.act, (size_t)cap * c.ffn));
  STATUS_TRY(dev_alloc(&w.ss_e, (size_t)cap));
  const size_t parts = (size_t)(c.hidden / GEMM_BN) * GEMM_SS_PER_TILE;
  STATUS_TRY(dev_alloc(&w.ss_a, (size_t)cap * parts));
  STATUS_TRY(dev_alloc(&w.ss_m, (size_t)cap * parts));
  STATUS_TRY(dev_alloc(&w.r_s, (size_t)cap * c.hidden));
  STATUS_TRY(dev_alloc(&w.ss_s, (size_t)cap * parts));
  STATUS_TRY(dev_alloc(&w.err, 1));
  STATUS_TRY(host_alloc(&w.h_err, 1));
  bool ok = make_tmap_16b_2d(&w.tm_xn, w.xn, c.hidden, cap, (uint64_t)c.hidden * 2, GEMM_BK, GEMM_BM, true, true) &&
            make_tmap_16b_2d(&w.tm_o, w.o, m->o_dim, cap, (uint64_t)m->o_dim * 2, GEMM_BK, GEMM_BM, true, true) &&
            make_tmap_16b_2d(&w.tm_act, w.act, c.ffn, cap, (uint64_t)c.ffn * 2, GEMM_BK, GEMM_BM, true, true);
  if (!ok) return fail(DOPR_ERR_CUDA, "cuTensorMapEncodeTiled failed for activation buffers");
  return DOPR_OK;
}

// Grow a device buffer to at least `need` elements (at least doubling); the
// capacity reads 0 while the buffer is not allocated, so a failed growth is
// retried by the next call instead of leaving a stale capacity.
template <typename T>
dopr_status grow_dev(T** p, int64_t& cap, int64_t need) {
  if (need <= cap) return DOPR_OK;
  const int64_t n = std::max<int64_t>(need, 2 * cap);
  dev_free(*p);
  cap = 0;
  STATUS_TRY(dev_alloc(p, (size_t)n));
  cap = n;
  return DOPR_OK;
}

// Grow the per-call buffers.
dopr_status ensure_call_buffers(Model* m, int64_t n_pairs, int64_t n_tokens, int64_t n_qtokens, int64_t n_docs) {
  Workspace& w = m->ws;
  if (n_pairs > w.pair_cap) {
    const int64_t cap = std::max<int64_t>(n_pairs, 2 * w.pair_cap);
    dev_free(w.q_off); dev_free(w.doc_ids); dev_free(w.scores); dev_free(w.pair_slot); dev_free(w.perm);
    dev_free(w.sorted_slot); dev_free(w.tok_off); dev_free(w.items);
    w.pair_cap = w.item_cap = 0;  // stays 0 if the growth fails, so no later call uses a freed buffer
    STATUS_TRY(dev_alloc(&w.q_off, cap + 1));
    STATUS_TRY(dev_alloc(&w.doc_ids, cap));
    STATUS_TRY(dev_alloc(&w.scores, cap));
    STATUS_TRY(dev_alloc(&w.pair_slot, cap));
    STATUS_TRY(dev_alloc(&w.perm, cap));
    STATUS_TRY(dev_alloc(&w.sorted_slot, cap));
    STATUS_TRY(dev_alloc(&w.tok_off, cap + 1));
    STATUS_TRY(dev_alloc(&w.items, 2 * (cap + 1024)));
    w.pair_cap = cap;
    w.item_cap = 2 * (cap + 1024);
  }
  if (n_pairs > w.h_pair_cap) {
    const int64_t cap = std::max<int64_t>(n_pairs, 2 * w.h_pair_cap);
    host_free(w.h_tok_off); host_free(w.h_sorted_slot); host_free(w.h_items);
    w.h_pair_cap = w.h_item_cap = 0;
    STATUS_TRY(host_alloc(&w.h_tok_off, cap + 1));
    STATUS_TRY(host_alloc(&w.h_sorted_slot, cap));
    STATUS_TRY(host_alloc(&w.h_items, 2 * (cap + 1024)));
    w.h_pair_cap = cap;
    w.h_item_cap = 2 * (cap + 1024);
  }
  if (n_tokens > w.tok_cap) {
    const int64_t cap = std::max<int64_t>(n_tokens, 2 * w.tok_cap);
    dev_free(w.tok_id); dev_free(w.tok_pos); dev_free(w.tok_pair);
    w.tok_cap = 0;
    STATUS_TRY(dev_alloc(&w.tok_id, cap));
    STATUS_TRY(dev_alloc(&w.tok_pos, cap));
    STATUS_TRY(dev_alloc(&w.tok_pair, cap));
    w.tok_cap = cap;
  }
  if (n_tokens > w.tile_cap) {  // a tile holds at least one token
    const int64_t cap = std::max<int64_t>(n_tokens, 2 * w.tile_cap);
    dev_free(w.tiles);
    host_free(w.h_tiles);
    w.tile_cap = 0;
    STATUS_TRY(dev_alloc(&w.tiles, cap));
    STATUS_TRY(host_alloc(&w.h_tiles, cap));
    w.tile_cap = cap;
  }
  if (n_qtokens > w.qtok_cap) {
    const int64_t cap = std::max<int64_t>(n_qtokens, 2 * w.qtok_cap);
    dev_free(w.q_tok);
    w.qtok_cap = 0;
    STATUS_TRY(dev_alloc(&w.q_tok, cap));
    w.qtok_cap = cap;
  }
  if (n_docs > w.doc_cap) {
    dev_free(w.doc_count);
    w.doc_cap = 0;
    STATUS_TRY(dev_alloc(&w.doc_count, n_docs));
    w.doc_cap = n_docs;
  }
  return DOPR_OK;
}

dopr_status map_device_error(int e) {
  if (e & DEV_ERR_TIMEOUT) return fail(DOPR_ERR_TIMEOUT, "a bounded device wait timed out");
  if (e & DEV_ERR_UNKNOWN_DOC) return fail(DOPR_ERR_UNKNOWN_DOC, "a doc_id has no stored prefix");
  if (e & DEV_ERR_INCOMPLETE) return fail(DOPR_ERR_INCOMPLETE, "a doc is missing stored layers");
  if (e & DEV_ERR_BAD_TOKEN) return fail(DOPR_ERR_INVALID_ARG, "a token id is outside [0, vocab)");
  if (e & DEV_ERR_BAD_OFFSETS) return fail(DOPR_ERR_INVALID_ARG, "q_offsets must start at 0 and not decrease");
  if (e & DEV_ERR_POSITION) return fail(DOPR_ERR_INVALID_ARG, "m + query length + 1 exceeds max_position");
  if (e & DEV_ERR_BOUNDS) return fail(DOPR_ERR_INTERNAL, "checked build: an index outside its buffer (access skipped)");
  if (e & DEV_ERR_RANGE)
    return fail(DOPR_ERR_RANGE,
                "an intermediate fp16 operand (normed activations, q/k/v, SwiGLU output, attention output) or a "
                "score was not finite or exceeded 65504 in magnitude; the call's scores are invalid");
  return DOPR_OK;
}

const char* kKindNames[K_COUNT] = {"pack", "embed", "gemm_qkv", "qknorm_rope", "attention",
                                   "gemm_o", "rmsnorm", "gemm_gate_up", "gemm_down", "score", "prefix_store"};

// Launch `fn` as one kernel of family `kind`, counting it and, when profiling
// is on, bracketing it with CUDA events on `st`.
template <typename F>
cudaError_t prof_launch(Model* m, int kind, int n_launches, double flops, double bytes, cudaStream_t st, F&& fn) {
  Profiler& p = m->prof;
  p.launches[kind] += n_launches;
  p.flops[kind] += flops;
  p.bytes[kind] += bytes;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (p.on) {
    const size_t need = 2 * (p.pending.size() + 1);
    while (p.events.size() < need) {
      cudaEvent_t e;
      cudaError_t r = cudaEventCreate(&e);
      if (r != cudaSuccess) return r;
      p.events.push_back(e);
    }
    e0 = p.events[need - 2];
    e1 = p.events[need - 1];
    cudaEventRecord(e0, st);
  }
  cudaError_t r = fn();
  if (p.on) {
    cudaEventRecord(e1, st);
    p.pending.push_back(kind);
  }
  return r;
}

// After the stream has been synchronised: fold the recorded event pairs in.
void prof_collect(Model* m) {
  Profiler& p = m->prof;
  for (size_t i = 0; i < p.pending.size(); ++i) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, p.events[2 * i], p.events[2 * i + 1]) == cudaSuccess) p.ms[p.pending[i]] += ms;
  }
  p.pending.clear();
}

// A store serves a model when its per-layer K/V blocks have the model's shape and both
// bound positions alike (the packer checks m + query length against max_position, and
// dopr_pack_order_noalloc, which sees only the store, must accept exactly what
// dopr_score accepts).
bool same_shape(const dopr_model_config& a, const dopr_model_config& b) {
  return a.n_layers == b.n_layers && a.n_kv_heads == b.n_kv_heads && a.head_dim == b.head_dim &&
         a.max_position == b.max_position;
}

// Host validation of host-resident inputs (before any launch).
dopr_status validate_host_inputs(const Model* m, const Store* s, int32_t n, const int32_t* qo, const int32_t* qt,
                                 const int64_t* doc) {
  if (qo[0] != 0) return fail(DOPR_ERR_INVALID_ARG, "q_offsets[0] must be 0");
  for (int32_t p = 0; p < n; ++p) {
    const int32_t L = qo[p + 1] - qo[p];
    if (L < 0) return fail(DOPR_ERR_INVALID_ARG, "q_offsets decreases at pair %d", p);
    const int64_t d = doc[p];
    if (d < 0 || d > s->max_doc_id || s->slot_of[d] < 0)
      return fail(DOPR_ERR_UNKNOWN_DOC, "pair %d: doc_id %lld has no stored prefix", p, (long long)d);
    const int32_t slot = s->slot_of[d];
    if (!s->slot_ok[slot]) return fail(DOPR_ERR_INCOMPLETE, "pair %d: doc_id %lld is missing layers", p, (long long)d);
    if ((int64_t)s->slot_m[slot] + L + 1 > m->cfg.max_position)
      return fail(DOPR_ERR_INVALID_ARG, "pair %d: m + query length + 1 exceeds max_position", p);
  }
  const int64_t nt = qo[n];
  for (int64_t i = 0; i < nt; ++i)
    if (qt[i] < 0 || qt[i] >= m->cfg.vocab)
      return fail(DOPR_ERR_INVALID_ARG, "q_tokens[%lld] = %d outside [0, vocab)", (long long)i, qt[i]);
  return DOPR_OK;
}

// The packer's device arguments for one call.
PackArgs pack_args(Model* m, Store* s, int32_t n, const int32_t* dqo, const int32_t* dqt, const int64_t* ddoc) {
  Workspace& w = m->ws;
  PackArgs a{};
  a.n_pairs = n;
  a.q_off = dqo;
  a.q_tok = dqt;
  a.doc_ids = ddoc;
  a.max_doc_id = s->max_doc_id;
  a.slot_of = s->d_slot_of;
  a.slot_m = s->d_slot_m;
  a.slot_ok = s->d_slot_ok;
  a.vocab = m->cfg.vocab;
  a.score_token = m->cfg.score_token_id;
  a.max_position = m->cfg.max_position;
  a.doc_count = w.doc_count;
  a.pair_slot = w.pair_slot;
  a.perm = w.perm;
  a.sorted_slot = w.sorted_slot;
  a.tok_off = w.tok_off;
  a.tok_id = w.tok_id;
  a.tok_pos = w.tok_pos;
  a.tok_pair = w.tok_pair;
  a.err = w.err;
  return a;
}

struct Plan {
  int64_t n_tokens = 0;
  std::vector<int32_t> chunk_pair;   // chunk c covers sorted pairs [chunk_pair[c], chunk_pair[c+1])
  std::vector<int32_t> chunk_item;   // and attention items [chunk_item[c], chunk_item[c+1]) (every pair)
  std::vector<int32_t> chunk_litem;  // mma.sync-kernel items [chunk_litem[c], chunk_litem[c+1])
  std::vector<int32_t> chunk_tile;   // tensor-core tiles [chunk_tile[c], chunk_tile[c+1])
  std::vector<int32_t> chunk_ltile;  // long tensor-core tiles, after all short ones
  int32_t n_items = 0, n_litems = 0, n_tiles = 0, n_ltiles = 0;
};

// Attention plan of a call: tensor-core tiles of at most TT tokens -- short ones
// within ATTN_TC_MAX_KEYS key columns, long ones (whose first token alone needs
// more) without a key limit -- and, when G gives no tile shape, runs of pairs for
// the mma.sync kernel.  Tiles keep at most ATTN_TC_MAX_SEGS pairs.
struct AttnPlanner {
  int TT = 0;
  std::vector<AttnTile> tiles, ltiles;
  std::vector<AttnItem> litems;

  // The sorted pairs [pb, pe) of one document (token offsets `to`, t0 the chunk's first token).
  // Each tile takes up to TT consecutive tokens (at most ATTN_TC_MAX_SEGS pairs).  It is a
  // tensor-core tile when its key columns fit ATTN_TC_MAX_KEYS -- the tile is cut where the
  // next token would overflow -- and a long tile, with no key limit, when not even its first
  // token fits.  Both kernels compute a row identically, so which one a row lands in does not
  // change its result.
  void add(const int32_t* to, int32_t t0, int32_t pb, int32_t pe, int32_t slot, int32_t m, int64_t pool_base) {
    auto c16 = [](int x) { return (x + 15) & ~15; };
    const int pre64 = ((m + 63) / 64) * 64;
    if (TT == 0) {
      for (int32_t p = pb; p < pe;) {
        const int32_t q = std::min(pe, p + ATTN_MAX_PAIRS);
        litems.push_back(AttnItem{p, q, slot, m});
        p = q;
      }
      return;
    }
    const int32_t end = to[pe] - t0;
    int32_t tok = to[pb] - t0, pf = pb;
    while (tok < end) {
      while (to[pf + 1] - t0 <= tok) ++pf;
      // the tokens [tok, tok + n) a tile takes, and its key columns
      auto grow = [&](bool limit_keys, int32_t& keys) {
        int32_t n = 0, closed = 0, pp = pf;
        keys = 0;
        while (n < TT && tok + n < end) {
          const int32_t t = tok + n;
          while (to[pp + 1] - t0 <= t) {  // pair pp lies wholly in the tile: its full segment
            closed += c16(to[pp + 1] - to[pp]);
            ++pp;
          }
          const int32_t k = pre64 + closed + c16(t - (to[pp] - t0) + 1);
          if ((limit_keys && k > ATTN_TC_MAX_KEYS) || pp - pf >= ATTN_TC_MAX_SEGS) break;
          keys = k;
          ++n;
        }
        return n;
      };
      int32_t keys = 0;
      int32_t n = grow(true, keys);
      const bool is_long = n == 0;
      if (is_long) n = grow(false, keys);
      AttnTile tl{};
      tl.pool_base = pool_base;
      tl.tok_begin = tok;
      tl.n_tok = n;
      tl.m = m;
      tl.n_keys = keys;
      for (int32_t sp = pf; to[sp] - t0 < tok + n; ++sp) {
        const int32_t ps = to[sp] - t0, nvis = std::min(to[sp + 1] - t0, tok + n) - ps;
        tl.seg[tl.n_seg++] = (int32_t)(((uint32_t)nvis << 16) | (uint16_t)(int16_t)(ps - tok));
      }
      (is_long ? ltiles : tiles).push_back(tl);
      tok += n;
    }
  }
  // The chunk's tiles go out most 64-key blocks first: CTAs take units round robin, so the
  // cheapest units come last and the CTAs finish together; within a block count the
  // tiles keep their order, so a document's tiles stay together and its prefix is read
  // from L2.  A row's result does not depend on the order (each tile is computed on its own).
  void close_chunk(Plan& plan) {
    auto by_keys = [](const AttnTile& x, const AttnTile& y) { return (x.n_keys + 63) / 64 > (y.n_keys + 63) / 64; };
    std::stable_sort(tiles.begin() + plan.chunk_tile.back(), tiles.end(), by_keys);
    std::stable_sort(ltiles.begin() + plan.chunk_ltile.back(), ltiles.end(), by_keys);
    plan.chunk_litem.push_back((int32_t)litems.size());
    plan.chunk_tile.push_back((int32_t)tiles.size());
    plan.chunk_ltile.push_back((int32_t)ltiles.size());
  }
  // Copy the plan to the workspace (host staging and device): the mma.sync items
  // after the first n_items entries, the short tiles, then the long tiles.
  dopr_status upload(Workspace& w, Plan& plan, int32_t n_items, cudaStream_t st) const {
    plan.n_items = n_items;
    plan.n_litems = (int32_t)litems.size();
    plan.n_tiles = (int32_t)tiles.size();
    plan.n_ltiles = (int32_t)ltiles.size();
    if (n_items + plan.n_litems > w.item_cap || n_items + plan.n_litems > w.h_item_cap ||
        plan.n_tiles + plan.n_ltiles > w.tile_cap)
      return fail(DOPR_ERR_UNSUPPORTED, "attention plan exceeds its buffers");
    std::copy(litems.begin(), litems.end(), w.h_items + n_items);
    std::copy(tiles.begin(), tiles.end(), w.h_tiles);
    std::copy(ltiles.begin(), ltiles.end(), w.h_tiles + tiles.size());
    if (n_items + plan.n_litems > 0)
      CUDA_TRY(cudaMemcpyAsync(w.items, w.h_items, sizeof(AttnItem) * (n_items + plan.n_litems),
                               cudaMemcpyHostToDevice, st));
    if (plan.n_tiles + plan.n_ltiles > 0)
      CUDA_TRY(cudaMemcpyAsync(w.tiles, w.h_tiles, sizeof(AttnTile) * (plan.n_tiles + plan.n_ltiles),
                               cudaMemcpyHostToDevice, st));
    return DOPR_OK;
  }
};

// Steps 1-4 of the engine.  Inputs are device pointers.  On return the packed
// plan is on the device and the chunking in `plan`.
dopr_status run_packer(Model* m, Store* s, int32_t n, const int32_t* dqo, const int32_t* dqt, const int64_t* ddoc,
                       cudaStream_t st, Plan& plan) {
  Workspace& w = m->ws;
  CUDA_TRY(cudaMemsetAsync(w.err, 0, sizeof(int), st));
  PackArgs a = pack_args(m, s, n, dqo, dqt, ddoc);
  CUDA_TRY(prof_launch(m, K_PACK, 4, 0.0, 24.0 * n, st, [&] { return launch_pack_order(a, st); }));
  CUDA_TRY(cudaMemcpyAsync(w.h_tok_off, w.tok_off, sizeof(int32_t) * (n + 1), cudaMemcpyDeviceToHost, st));
  CUDA_TRY(cudaMemcpyAsync(w.h_sorted_slot, w.sorted_slot, sizeof(int32_t) * n, cudaMemcpyDeviceToHost, st));
  CUDA_TRY(cudaMemcpyAsync(w.h_err, w.err, sizeof(int), cudaMemcpyDeviceToHost, st));
  CUDA_TRY(cudaStreamSynchronize(st));
  STATUS_TRY(map_device_error(*w.h_err));
  plan.n_tokens = w.h_tok_off[n];
  // token buffers sized from the packed total, then packer part 2
  STATUS_TRY(ensure_call_buffers(m, n, plan.n_tokens, 0, 0));
  a = pack_args(m, s, n, dqo, dqt, ddoc);
  CUDA_TRY(prof_launch(m, K_PACK, 1, 0.0, 16.0 * plan.n_tokens, st, [&] { return launch_pack_tokens(a, st); }));
  // chunks of whole pairs, then attention items (runs of one doc, <= ATTN_MAX_PAIRS),
  // and per chunk the tensor-core tiles and the mma.sync kernel's items
  const int cap = w.chunk_cap;
  AttnPlanner ap;
  ap.TT = attn_tc_rows_per_head(m->cfg.n_q_heads / m->cfg.n_kv_heads);
  plan.chunk_pair.assign(1, 0);
  plan.chunk_item.assign(1, 0);
  plan.chunk_litem.assign(1, 0);
  plan.chunk_tile.assign(1, 0);
  plan.chunk_ltile.assign(1, 0);
  int32_t items = 0;
  int32_t s0 = 0;
  while (s0 < n) {
    int32_t s1 = s0 + 1;
    if (w.h_tok_off[s1] - w.h_tok_off[s0] > cap)
      return fail(DOPR_ERR_UNSUPPORTED, "one pair has more tokens than a chunk (%d)", cap);
    while (s1 < n && w.h_tok_off[s1 + 1] - w.h_tok_off[s0] <= cap) ++s1;
    int32_t i = s0;
    while (i < s1) {
      int32_t j = i + 1;
      while (j < s1 && w.h_sorted_slot[j] == w.h_sorted_slot[i]) ++j;  // the document's run in this chunk
      const int32_t slot = w.h_sorted_slot[i], mm = s->slot_m[slot];
      for (int32_t a = i; a < j; a += ATTN_MAX_PAIRS)
        w.h_items[items++] = AttnItem{a, std::min(j, a + ATTN_MAX_PAIRS), slot, mm};
      ap.add(w.h_tok_off, w.h_tok_off[s0], i, j, slot, mm, s->slot_row[slot]);
      i = j;
    }
    plan.chunk_pair.push_back(s1);
    plan.chunk_item.push_back(items);
    ap.close_chunk(plan);
    s0 = s1;
  }
  return ap.upload(w, plan, items, st);
}

// Prefix build mode of run_layers: the packed "tokens" are the selected document
// representations (rows of x), each document one "pair" with no prefix and no score
// token; after every layer's QKV projection its keys and values go to the store, and
// the last layer stops there.
struct BuildArgs {
  const bf16* x;  // device, [total rows][hidden]
  int64_t rows;   // its rows
};

// Key token selection mode of run_layers: the packed tokens are documents'
// token ids, each document one "pair" with no prefix and no score token; the
// last layer runs in full, and after its QKV projection the selection kernels
// rank the chunk's tokens, after its MLP the selected rows' final states are
// gathered.
struct SelectState {
  int top_k, top_p;
  float* A;        // device, the largest chunk's sum of n^2
  int64_t a_elems;  // floats in A
  int64_t* a_off;  // device, per chunk document
  float* u;        // device, [all tokens]
  int32_t* positions;
  bf16* x;
};

dopr_status run_layers(Model* m, Store* s, const Plan& plan, float* d_scores, cudaStream_t st,
                       const BuildArgs* build = nullptr, SelectState* sel = nullptr) {
  Workspace& w = m->ws;
  const auto& c = m->cfg;
  const int H = c.hidden, F = c.ffn, L = c.n_layers, Hq = c.n_q_heads, Hkv = c.n_kv_heads;
  const int parts = H / GEMM_BN * GEMM_SS_PER_TILE;  // partial sums of squares per row from a residual epilogue
  const int mpad = ((s->max_m + 63) / 64) * 64;
  const int sms = m->num_sms;
  const bool scoring = !build && !sel;
  auto gemm_cost = [](double M, double N, double K, double out_bytes) {
    return std::make_pair(2.0 * M * N * K, (M * K + N * K) * 2.0 + out_bytes);
  };
  for (size_t ci = 0; ci + 1 < plan.chunk_pair.size(); ++ci) {
    NvtxRange chunk_range("dopr chunk %d", static_cast<int>(ci));
    const int32_t s0 = plan.chunk_pair[ci], s1 = plan.chunk_pair[ci + 1];
    const int32_t t0 = w.h_tok_off[s0], Tc = w.h_tok_off[s1] - t0;
    const double T = Tc;
    // attention work of this chunk: keys visible per (token, q head) and prefix bytes staged per item
    double attn_keys = 0.0, prefix_rows = 0.0;
    for (int32_t sp = s0; sp < s1; ++sp) {
      const double Tp = w.h_tok_off[sp + 1] - w.h_tok_off[sp];
      attn_keys += Tp * (scoring ? s->slot_m[w.h_sorted_slot[sp]] : 0) + Tp * (Tp + 1) / 2;
    }
    for (int32_t it = plan.chunk_item[ci]; it < plan.chunk_item[ci + 1]; ++it) prefix_rows += w.h_items[it].m;
    if (!scoring) prefix_rows = 0.0;
    const double attn_flops = 4.0 * HEAD_DIM * Hq * attn_keys;
    const double attn_bytes = T * (2.0 * Hq + 2.0 * Hkv) * HEAD_DIM * 2 + prefix_rows * Hkv * 2 * HEAD_DIM * 2;
    // algorithmic bytes: operands once, outputs once (residual: read + write fp32, plus the next norm's bf16 operand)
    const auto qkv = gemm_cost(T, m->qkv_dim, H, T * m->qkv_dim * 2.0);
    const auto op = gemm_cost(T, H, m->o_dim, T * H * 10.0);
    const auto gu = gemm_cost(T, 2.0 * F, H, T * F * 2.0);
    const auto dn = gemm_cost(T, H, F, T * H * 10.0);
    Extents ext;  // what the index tests of a checked build compare against
    ext.err = w.err;
    ext.rows = Tc;
    ext.table_rows = build ? build->rows : c.vocab;
    ext.pool_rows = s->pool_rows;
    ext.a_elems = sel ? sel->a_elems : 0;
    CUDA_TRY(prof_launch(m, K_EMBED_NORM, 1, 0.0, T * H * 8.0, st, [&] {
      return launch_embed(w.tok_id + t0, Tc, build ? build->x : m->embed, m->attn_norm, H, c.rms_eps, w.r, w.xn,
                          w.ss_e, ext, st);
    }));
    GemmParams base{};
    base.M = Tc;
    base.norm_dim = H;
    base.eps = c.rms_eps;
    base.err = w.err;
    const int32_t np = s1 - s0;
    double last_keys = 0.0;  // keys seen by the score-token rows alone
    for (int32_t sp = s0; sp < s1; ++sp)
      last_keys += (scoring ? s->slot_m[w.h_sorted_slot[sp]] : 0) + (w.h_tok_off[sp + 1] - w.h_tok_off[sp]);
    const double attn_flops_last = 4.0 * HEAD_DIM * Hq * last_keys;
    const double attn_bytes_last = np * 2.0 * Hq * HEAD_DIM * 2 + T * 2.0 * Hkv * HEAD_DIM * 2 +
                                   prefix_rows * Hkv * 2 * HEAD_DIM * 2;
    // this chunk's packed QKV buffer as TMA maps for the tensor-core attention:
    // Q boxes of 128 / G rows of the group's G heads, own-key boxes of 16, 32 and 64 rows
    const int TT = attn_tc_rows_per_head(Hq / Hkv);
    CUtensorMap tm_q{}, tm_kv{}, tm_kv32{}, tm_kv64{};
    const int n_tiles = plan.chunk_tile[ci + 1] - plan.chunk_tile[ci];
    const int n_ltiles = plan.chunk_ltile[ci + 1] - plan.chunk_ltile[ci];
    if (n_tiles + n_ltiles > 0 &&
        !(make_tmap_q_heads(&tm_q, w.qkv, m->qkv_dim, Tc, TT, Hq / Hkv) &&
          make_tmap_16b_2d(&tm_kv, w.qkv, m->qkv_dim, Tc, (uint64_t)m->qkv_dim * 2, 64, 16, true, true) &&
          make_tmap_16b_2d(&tm_kv32, w.qkv, m->qkv_dim, Tc, (uint64_t)m->qkv_dim * 2, 64, 32, true, true) &&
          make_tmap_16b_2d(&tm_kv64, w.qkv, m->qkv_dim, Tc, (uint64_t)m->qkv_dim * 2, 64, 64, true, true)))
      return fail(DOPR_ERR_CUDA, "cuTensorMapEncodeTiled failed for the QKV buffer");
    AttnTcArgs ta{};
    ta.tiles = w.tiles + plan.chunk_tile[ci];
    ta.n_units = n_tiles * Hkv;
    ta.out = w.o;
    ta.ld_out = m->o_dim;
    ta.Hq = Hq;
    ta.Hkv = Hkv;
    ta.err = w.err;
    ta.ext = ext;
    AttnTcArgs tl = ta;  // the long tiles, stored after every short tile
    tl.tiles = w.tiles + plan.n_tiles + plan.chunk_ltile[ci];
    tl.n_units = n_ltiles * Hkv;
    const int32_t li0 = plan.n_items + plan.chunk_litem[ci];
    const int32_t n_litems = plan.chunk_litem[ci + 1] - plan.chunk_litem[ci];
    const auto op_last = gemm_cost(np, H, m->o_dim, np * H * 10.0);
    const auto gu_last = gemm_cost(np, 2.0 * F, H, np * F * 2.0);
    const auto dn_last = gemm_cost(np, H, F, np * H * 8.0);
    for (int l = 0; l < L; ++l) {
      NvtxRange layer_range("dopr layer %d", l);
      // In the last layer only the score-token rows reach the score: after the full QKV
      // projection (every token's key and value is attended to), attention, O and the MLP
      // run on one compact row per pair.
      const bool final_layer = l + 1 == L;
      const bool last = scoring && final_layer;  // the scoring pass prunes its last layer to score rows
      GemmParams pq = base;  // QKV + attention-norm row scale + q/k norm + RoPE
      pq.N = m->qkv_dim;
      pq.K = H;
      pq.out = w.qkv;
      pq.ld_out = m->qkv_dim;
      if (l > 0) {  // layer 0's operand comes from the embedding, already normalised
        pq.ss_in = w.ss_a;
        pq.ss_parts = parts;
        pq.ss_pre = w.ss_m;
        pq.ss_pre_parts = parts;
      }
      pq.tok_pos = w.tok_pos + t0;
      pq.rope = m->rope;
      pq.q_norm = m->q_norm + (size_t)l * HEAD_DIM;
      pq.k_norm = m->k_norm + (size_t)l * HEAD_DIM;
      pq.q_cols = Hq * HEAD_DIM;
      pq.k_cols = Hkv * HEAD_DIM;
      CUDA_TRY(prof_launch(m, K_GEMM_QKV, 1, qkv.first, qkv.second, st,
                           [&] { return launch_gemm(EPI_QKV, w.tm_xn, m->tm_qkv[l], pq, sms, st); }));
      if (build) {  // this layer's keys and values are the document's stored prefix states
        CUDA_TRY(prof_launch(m, K_PREFIX_STORE, 1, 0.0, T * 2.0 * Hkv * HEAD_DIM * 2 * 2, st, [&] {
          return launch_prefix_store(w.qkv, m->qkv_dim, Tc, t0, Hq, Hkv, w.tok_pair, w.tok_pos, w.sorted_slot,
                                     s->d_slot_row, s->d_slot_m, l, reinterpret_cast<f16*>(s->pool), ext, st);
        }));
        if (final_layer) continue;
      }
      if (sel && final_layer) {  // rank the chunk's tokens on this layer's q and k
        SelectArgs sa{};
        sa.qkv = w.qkv;
        sa.ld_qkv = m->qkv_dim;
        sa.Hq = Hq;
        sa.Hkv = Hkv;
        sa.tok_pair = w.tok_pair;
        sa.tok_off = w.tok_off;
        sa.t0 = t0;
        sa.p0 = s0;
        sa.n_docs = s1 - s0;
        sa.n_rows = Tc;
        sa.a_off = sel->a_off;
        sa.A = sel->A;
        sa.top_p = sel->top_p;
        sa.top_k = sel->top_k;
        sa.u = sel->u + t0;
        sa.positions = sel->positions;
        sa.x = sel->x;
        sa.ext = ext;
        std::vector<int64_t> aoff(s1 - s0);
        int64_t acc = 0;
        for (int32_t d = s0; d < s1; ++d) {
          const int64_t nd = w.h_tok_off[d + 1] - w.h_tok_off[d];
          aoff[d - s0] = acc;
          acc += nd * nd;
        }
        CUDA_TRY(cudaMemcpyAsync(sel->a_off, aoff.data(), sizeof(int64_t) * aoff.size(), cudaMemcpyHostToDevice, st));
        CUDA_TRY(launch_select(sa, st));
      }
      AttnArgs aa{};
      aa.items = w.items + (last ? plan.chunk_item[ci] : li0);
      aa.n_items = last ? plan.chunk_item[ci + 1] - plan.chunk_item[ci] : n_litems;
      aa.tok_off = w.tok_off;
      aa.tok0 = t0;
      aa.qkv = w.qkv;
      aa.ld_qkv = m->qkv_dim;
      aa.out = w.o;
      aa.ld_out = m->o_dim;
      aa.slot_row = s->d_slot_row;
      aa.layer = l;
      aa.n_layers = L;
      aa.Hq = Hq;
      aa.Hkv = Hkv;
      aa.mpad_cap = mpad;
      aa.score_only = last ? 1 : 0;
      aa.pair_base = s0;
      aa.err = w.err;
      aa.ext = ext;
      const int attn_launches = (!last && ta.n_units > 0 ? 1 : 0) + (!last && tl.n_units > 0 ? 1 : 0) +
                                (aa.n_items > 0 ? 1 : 0);
      CUDA_TRY(prof_launch(m, K_ATTENTION, attn_launches, last ? attn_flops_last : attn_flops,
                           last ? attn_bytes_last : attn_bytes, st,
                           [&] {
                             // every layer but the last: tensor-core tiles, then the pairs beyond
                             // their key budget; the last layer: score-token rows of every pair
                             cudaError_t e = cudaSuccess;
                             if (!last && ta.n_units > 0) {
                               ta.layer = l;
                               e = launch_attention_tc(tm_q, tm_kv, tm_kv32, tm_kv64, s->tm_pool, ta, sms, st);
                             }
                             if (e == cudaSuccess && !last && tl.n_units > 0) {
                               tl.layer = l;
                               e = launch_attention_tc_long(tm_q, tm_kv, tm_kv32, tm_kv64, s->tm_pool, tl, sms, st);
                             }
                             if (e == cudaSuccess && aa.n_items > 0) e = launch_attention(s->tm_pool, aa, st);
                             return e;
                           }));
      const float* ss_pre = l == 0 ? w.ss_e : w.ss_a;  // the attention norm of this layer
      const int ss_pre_parts = l == 0 ? 1 : parts;
      float* resid = w.r;
      int rows = Tc;
      if (last) {
        CUDA_TRY(prof_launch(m, K_SCORE, 1, 0.0, np * (H * 8.0 + ss_pre_parts * 8.0), st, [&] {
          return launch_gather_score_rows(w.r, ss_pre, H, ss_pre_parts, w.tok_off, t0, s0, s1, w.r_s, w.ss_s, ext,
                                          st);
        }));
        ss_pre = w.ss_s;
        resid = w.r_s;
        rows = np;
      }
      GemmParams po = base;  // O projection + residual, emits the MLP norm's operand
      po.M = rows;
      po.N = H;
      po.K = m->o_dim;
      po.out = resid;
      po.ld_out = H;
      po.xn_out = w.xn;
      po.xn_gain = m->mlp_norm + (size_t)l * H;
      po.ss_out = w.ss_m;
      po.ss_out_parts = parts;
      po.ss_pre = ss_pre;
      po.ss_pre_parts = ss_pre_parts;
      CUDA_TRY(prof_launch(m, K_GEMM_O, 1, last ? op_last.first : op.first, last ? op_last.second : op.second, st,
                           [&] { return launch_gemm(EPI_RESID_ADD, w.tm_o, m->tm_o[l], po, sms, st); }));
      GemmParams pg = base;  // gate/up + MLP-norm row scale + SwiGLU
      pg.M = rows;
      pg.N = 2 * F;
      pg.K = H;
      pg.out = w.act;
      pg.ld_out = F;
      pg.ss_in = w.ss_m;
      pg.ss_parts = parts;
      pg.ss_pre = ss_pre;
      pg.ss_pre_parts = ss_pre_parts;
      CUDA_TRY(prof_launch(m, K_GEMM_GATE_UP, 1, last ? gu_last.first : gu.first, last ? gu_last.second : gu.second,
                           st, [&] { return launch_gemm(EPI_SWIGLU, w.tm_xn, m->tm_gu[l], pg, sms, st); }));
      GemmParams pd = base;  // down projection + residual, emits the next attention norm's operand
      pd.M = rows;
      pd.N = H;
      pd.K = F;
      pd.out = resid;
      pd.ld_out = H;
      if (!final_layer) {  // a next layer exists: emit its attention norm's operand
        pd.xn_out = w.xn;
        pd.xn_gain = m->attn_norm + (size_t)(l + 1) * H;
        pd.ss_out = w.ss_a;
        pd.ss_out_parts = parts;
        pd.ss_pre = w.ss_m;  // the MLP norm of this layer
        pd.ss_pre_parts = parts;
      }
      CUDA_TRY(prof_launch(m, K_GEMM_DOWN, 1, last ? dn_last.first : dn.first, last ? dn_last.second : dn.second, st,
                           [&] { return launch_gemm(EPI_RESID_ADD, w.tm_act, m->tm_down[l], pd, sms, st); }));
    }
    if (scoring) {
      if (m->mlp_width > 0) {
        const double wd = m->mlp_width;
        CUDA_TRY(prof_launch(m, K_SCORE, 1, 2.0 * H * wd * (s1 - s0), (s1 - s0) * (H * 4.0 + 4.0) + wd * H * 2.0, st,
                             [&] {
                               return launch_score_mlp(w.r_s, H, w.tok_off, t0, s0, s1, 1, w.perm, m->final_norm,
                                                       c.rms_eps, m->mlp_width, m->mlp_act, m->mlp_w1, m->mlp_b1,
                                                       m->mlp_w2, m->mlp_b2, d_scores, ext, st);
                             }));
      } else {
        CUDA_TRY(prof_launch(m, K_SCORE, 1, 4.0 * H * (s1 - s0), (s1 - s0) * (H * 4.0 + 4.0), st, [&] {
          return launch_score(w.r_s, H, w.tok_off, t0, s0, s1, 1, w.perm, m->final_norm, m->score_head, c.rms_eps,
                              d_scores, ext, st);
        }));
      }
    } else if (sel) {  // final states of the selected rows: the representations C_d
      SelectArgs sa{};
      sa.tok_off = w.tok_off;
      sa.t0 = t0;
      sa.p0 = s0;
      sa.n_docs = s1 - s0;
      sa.top_k = sel->top_k;
      sa.positions = sel->positions;
      sa.x = sel->x;
      sa.ext = ext;
      CUDA_TRY(launch_select_gather(sa, w.r, H, m->final_norm, c.rms_eps, st));
    }
  }
  return DOPR_OK;
}

// The slot of doc_id: reserved on its first use with prefix length m (a later use
// must give the same m).  Host mirrors and device tables are updated together.
dopr_status store_reserve(Store* s, int64_t doc_id, int32_t m, int32_t* slot_out) {
  const auto& c = s->cfg;
  int32_t slot = s->slot_of[doc_id];
  if (slot >= 0 && s->slot_m[slot] != m)
    return fail(DOPR_ERR_INVALID_ARG, "doc %lld was stored with m = %d, not %d", (long long)doc_id, s->slot_m[slot], m);
  if (slot < 0) {
    const int64_t need = 2 * (int64_t)c.n_kv_heads * m * c.n_layers;  // K and V rows of 128, every layer
    if (s->used_rows + need > s->pool_rows)
      return fail(DOPR_ERR_OUT_OF_MEMORY, "store pool full (%lld of %lld rows used, %lld needed)",
                  (long long)s->used_rows, (long long)s->pool_rows, (long long)need);
    slot = s->n_slots++;
    s->slot_m.push_back(m);
    s->slot_row.push_back(s->used_rows);
    s->slot_layers.emplace_back(c.n_layers, 0);
    s->slot_ok.push_back(0);
    s->used_rows += need;
    s->slot_of[doc_id] = slot;
    const int64_t row = s->slot_row[slot];
    CUDA_TRY(cudaMemcpy(s->d_slot_m + slot, &m, sizeof(int32_t), cudaMemcpyHostToDevice));
    CUDA_TRY(cudaMemcpy(s->d_slot_row + slot, &row, sizeof(int64_t), cudaMemcpyHostToDevice));
    CUDA_TRY(cudaMemcpy(s->d_slot_of + doc_id, &slot, sizeof(int32_t), cudaMemcpyHostToDevice));
    s->max_m = std::max(s->max_m, m);
  }
  *slot_out = slot;
  return DOPR_OK;
}

// Record that `layer` of `slot` holds valid states (present = 1) or not; the slot
// becomes scoreable once every layer is present.
dopr_status store_mark(Store* s, int32_t slot, int layer, bool present) {
  const int L = s->cfg.n_layers;
  s->slot_layers[slot][layer] = present ? 1 : 0;
  bool all = true;
  for (int l = 0; l < L; ++l) all = all && s->slot_layers[slot][l];
  const uint8_t ok = all ? 1 : 0;
  if (s->slot_ok[slot] != ok) {
    s->slot_ok[slot] = ok;
    CUDA_TRY(cudaMemcpy(s->d_slot_ok + slot, &ok, 1, cudaMemcpyHostToDevice));
  }
  return DOPR_OK;
}

dopr_status check_ready(Model* m, Store* s) {
  if (!m || !s) return fail(DOPR_ERR_INVALID_ARG, "model or store is NULL");
  if (!same_shape(m->cfg, s->cfg)) return fail(DOPR_ERR_INVALID_ARG, "store shape (layers, kv heads, head_dim, max_position) does not match the model");
  const int L = m->cfg.n_layers;
  for (int k = 0; k < kind_count(); ++k)
    for (int l = 0; l < (kind_is_global(k) ? 1 : L); ++l)
      if (!m->have[k * L + l]) return fail(DOPR_ERR_INCOMPLETE, "weight kind %d layer %d was never put", k, l);
  return DOPR_OK;
}

}  // namespace

void set_last_error_message(const std::string& msg) { g_last_error = msg; }

bool make_tmap_16b_2d(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint64_t row_stride_bytes,
                      uint32_t box_cols, uint32_t box_rows, bool swizzle128, bool half) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, half ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                  const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE,
                  swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// The Q columns of a packed QKV buffer [rows][cols] as a 3-D tensor: 128 elements of a head
// (innermost), rows, heads (256 bytes apart); the box takes 64 elements of box_heads heads over
// box_rows rows, stored head after head (fp16, 128-byte swizzle).
bool make_tmap_q_heads(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows,
                       uint32_t box_heads) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {128, rows, cols / 128};
  cuuint64_t strides[2] = {cols * 2, 256};
  cuuint32_t box[3] = {64, box_rows, box_heads};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace dopr

using namespace dopr;

extern "C" {

const char* dopr_version(void) { return "dopr-gb300 0.1 (sm_103a)"; }

const char* dopr_last_error(void) { return g_last_error.c_str(); }

int64_t dopr_prefix_bytes(const dopr_model_config* cfg, int32_t m) {
  if (!cfg || m < 0 || cfg->n_layers <= 0 || cfg->n_kv_heads <= 0 || cfg->head_dim <= 0) return -1;
  return (int64_t)m * cfg->n_layers * 2 * cfg->n_kv_heads * cfg->head_dim * 2;
}

dopr_status dopr_model_create(const dopr_model_config* cfg, dopr_model** out) {
  g_last_error.clear();
  if (!out) return fail(DOPR_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  STATUS_TRY(check_cfg(cfg));
  if (!encode_fn()) return fail(DOPR_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
  dopr_model* m = new dopr_model();
  m->cfg = *cfg;
  const auto& c = *cfg;
  const size_t H = c.hidden, F = c.ffn, L = c.n_layers;
  m->qkv_dim = (c.n_q_heads + 2 * c.n_kv_heads) * HEAD_DIM;
  m->o_dim = c.n_q_heads * HEAD_DIM;
  dopr_status st = DOPR_OK;
  auto guard = [&](dopr_status s) {
    if (s != DOPR_OK && st == DOPR_OK) st = s;
    return s == DOPR_OK;
  };
  cudaGetDevice(&m->device);
  cudaDeviceGetAttribute(&m->num_sms, cudaDevAttrMultiProcessorCount, m->device);
  guard(gemm_setup() == cudaSuccess && attn_setup() == cudaSuccess && attn_tc_setup() == cudaSuccess && select_setup() == cudaSuccess
            ? DOPR_OK
            : fail(DOPR_ERR_CUDA, "kernel attribute setup failed: %s", cudaGetErrorString(cudaGetLastError())));
  if (st == DOPR_OK &&
      guard(dev_alloc(&m->embed, (size_t)c.vocab * H)) && guard(dev_alloc(&m->attn_norm, L * H)) &&
      guard(dev_alloc(&m->w_qkv, L * m->qkv_dim * H)) && guard(dev_alloc(&m->q_norm, L * HEAD_DIM)) &&
      guard(dev_alloc(&m->k_norm, L * HEAD_DIM)) && guard(dev_alloc(&m->w_o, L * H * m->o_dim)) &&
      guard(dev_alloc(&m->mlp_norm, L * H)) && guard(dev_alloc(&m->w_gu, L * 2 * F * H)) &&
      guard(dev_alloc(&m->w_down, L * H * F)) && guard(dev_alloc(&m->final_norm, H)) &&
      guard(dev_alloc(&m->score_head, 2 * H)) && guard(dev_alloc(&m->rope, (size_t)c.max_position * (HEAD_DIM / 2)))) {
    // RoPE table: angle = pos * theta^(-2i/128), evaluated in double on the host.
    std::vector<float2> tab((size_t)c.max_position * (HEAD_DIM / 2));
    for (int p = 0; p < c.max_position; ++p)
      for (int i = 0; i < HEAD_DIM / 2; ++i) {
        const double a = (double)p * pow((double)c.rope_theta, -2.0 * i / (double)HEAD_DIM);
        tab[(size_t)p * (HEAD_DIM / 2) + i] = make_float2((float)cos(a), (float)sin(a));
      }
    if (cudaMemcpy(m->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice) != cudaSuccess)
      guard(fail(DOPR_ERR_CUDA, "rope table upload failed"));
  }
  if (st == DOPR_OK) guard(build_weight_maps(m));
  if (st == DOPR_OK) {
    // Chunk size: enough rows to fill the GEMM tiles, bounded to ~2.5 GB of activations.
    const int64_t per_tok = (int64_t)H * 6 + (int64_t)m->qkv_dim * 2 + (int64_t)m->o_dim * 2 + (int64_t)F * 2;
    int64_t cap = (int64_t)2500 * 1000 * 1000 / per_tok;
    cap = std::min<int64_t>(cap, 32768);
    cap = std::max<int64_t>(cap, (int64_t)c.max_position);
    cap = (cap + 127) / 128 * 128;
    guard(alloc_chunk_buffers(m, (int)cap));
  }
  if (st != DOPR_OK) {
    free_model(m);
    delete m;
    return st;
  }
  m->have.assign((size_t)kind_count() * L, 0);
  *out = m;
  return DOPR_OK;
}

dopr_status dopr_model_put_weight(dopr_model* m, int32_t kind, int32_t layer, const void* src, int64_t n_elems,
                                  int32_t src_on_device) {
  g_last_error.clear();
  if (!m || !src) return fail(DOPR_ERR_INVALID_ARG, "model or src is NULL");
  const auto& c = m->cfg;
  const int64_t H = c.hidden, F = c.ffn, D = HEAD_DIM, Hq = c.n_q_heads, Hkv = c.n_kv_heads;
  if (kind < 0 || kind >= kind_count()) return fail(DOPR_ERR_INVALID_ARG, "bad weight kind %d", kind);
  if (kind_is_global(kind)) layer = 0;
  else if (layer < 0 || layer >= c.n_layers) return fail(DOPR_ERR_INVALID_ARG, "bad layer %d", layer);
  const size_t l = (size_t)layer;
  const cudaMemcpyKind dir = src_on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
  int64_t expect = 0;
  void* dst = nullptr;
  bool matrix = false;  // projection matrices are held as fp16 for the tensor cores
  switch (kind) {
    case DOPR_W_EMBED: expect = (int64_t)c.vocab * H; dst = m->embed; break;
    case DOPR_W_ATTN_NORM: expect = H; dst = m->attn_norm + l * H; break;
    case DOPR_W_Q: expect = Hq * D * H; dst = m->w_qkv + l * m->qkv_dim * H; matrix = true; break;
    case DOPR_W_K: expect = Hkv * D * H; dst = m->w_qkv + (l * m->qkv_dim + Hq * D) * H; matrix = true; break;
    case DOPR_W_V: expect = Hkv * D * H; dst = m->w_qkv + (l * m->qkv_dim + (Hq + Hkv) * D) * H; matrix = true; break;
    case DOPR_W_Q_NORM: expect = D; dst = m->q_norm + l * D; break;
    case DOPR_W_K_NORM: expect = D; dst = m->k_norm + l * D; break;
    case DOPR_W_O: expect = H * Hq * D; dst = m->w_o + l * H * m->o_dim; matrix = true; break;
    case DOPR_W_MLP_NORM: expect = H; dst = m->mlp_norm + l * H; break;
    case DOPR_W_GATE:
    case DOPR_W_UP:
      expect = F * H;
      dst = m->w_gu + l * 2 * F * H + (kind == DOPR_W_UP ? 128 * H : 0);
      matrix = true;
      break;
    case DOPR_W_DOWN: expect = H * F; dst = m->w_down + l * H * F; matrix = true; break;
    case DOPR_W_FINAL_NORM: expect = H; dst = m->final_norm; break;
    case DOPR_W_SCORE_HEAD: expect = 2 * H; dst = m->score_head; break;
  }
  if (n_elems != expect)
    return fail(DOPR_ERR_INVALID_ARG, "weight kind %d: %lld elements given, %lld expected", kind, (long long)n_elems,
                (long long)expect);
  CUDA_TRY(cudaSetDevice(m->device));
  if (!matrix) {
    CUDA_TRY(cudaMemcpy(dst, src, (size_t)expect * 2, dir));
  } else {
    // stage, widen bf16 -> fp16 (exact in fp16's normal range), then place; a value
    // outside fp16's range (or not finite) fails the put and leaves the weight as it was
    void* stage = nullptr;
    const size_t bytes = ((size_t)expect * 2 + 15) & ~(size_t)15;
    CUDA_TRY(cudaMalloc(&stage, bytes + 16));
    int* d_range = reinterpret_cast<int*>(static_cast<uint8_t*>(stage) + bytes);
    int range = 0;
    cudaError_t e = cudaMemcpy(stage, src, (size_t)expect * 2, dir);
    if (e == cudaSuccess) e = cudaMemset(d_range, 0, sizeof(int));
    if (e == cudaSuccess) e = launch_bf16_to_f16(stage, expect, d_range, 0);
    if (e == cudaSuccess) e = cudaMemcpy(&range, d_range, sizeof(int), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && range) {
      cudaFree(stage);
      return fail(DOPR_ERR_INVALID_ARG,
                  "weight kind %d layer %d: a value is not finite or exceeds the fp16 range (|x| > 65504)", kind, layer);
    }
    if (e == cudaSuccess) {
      if (kind == DOPR_W_GATE || kind == DOPR_W_UP)  // rows 128b.. go to rows 256b (+128 for up)
        e = cudaMemcpy2D(dst, 256 * H * 2, stage, 128 * H * 2, 128 * H * 2, F / 128, cudaMemcpyDeviceToDevice);
      else
        e = cudaMemcpy(dst, stage, (size_t)expect * 2, cudaMemcpyDeviceToDevice);
    }
    cudaFree(stage);
    if (e != cudaSuccess) return fail(DOPR_ERR_CUDA, "weight upload failed: %s", cudaGetErrorString(e));
  }
  m->have[(size_t)kind * c.n_layers + l] = 1;
  return DOPR_OK;
}

dopr_status dopr_model_set_mlp_head(dopr_model* m, int32_t width, int32_t activation, const void* w1, const void* b1,
                                    const void* w2, float b2, int32_t src_on_device) {
  g_last_error.clear();
  if (!m) return fail(DOPR_ERR_INVALID_ARG, "model is NULL");
  if (width < 0 || width > 16384) return fail(DOPR_ERR_INVALID_ARG, "width %d outside [0, 16384]", width);
  if (activation < 0 || activation > 3) return fail(DOPR_ERR_INVALID_ARG, "activation %d outside [0, 3]", activation);
  CUDA_TRY(cudaSetDevice(m->device));
  dev_free(m->mlp_w1); dev_free(m->mlp_b1); dev_free(m->mlp_w2);
  m->mlp_w1 = m->mlp_b1 = m->mlp_w2 = nullptr;
  m->mlp_width = 0;
  if (width == 0) return DOPR_OK;  // back to the yes/no rows
  if (!w1 || !b1 || !w2) return fail(DOPR_ERR_INVALID_ARG, "NULL head weight");
  const int H = m->cfg.hidden;
  STATUS_TRY(dev_alloc(&m->mlp_w1, (size_t)width * H));
  STATUS_TRY(dev_alloc(&m->mlp_b1, (size_t)width));
  STATUS_TRY(dev_alloc(&m->mlp_w2, (size_t)width));
  const cudaMemcpyKind kind = src_on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
  CUDA_TRY(cudaMemcpy(m->mlp_w1, w1, sizeof(bf16) * (size_t)width * H, kind));
  CUDA_TRY(cudaMemcpy(m->mlp_b1, b1, sizeof(bf16) * (size_t)width, kind));
  CUDA_TRY(cudaMemcpy(m->mlp_w2, w2, sizeof(bf16) * (size_t)width, kind));
  m->mlp_width = width;
  m->mlp_act = activation;
  m->mlp_b2 = b2;
  return DOPR_OK;
}

dopr_status dopr_model_destroy(dopr_model* m) {
  g_last_error.clear();
  if (!m) return DOPR_OK;
  cudaSetDevice(m->device);
  free_model(m);
  delete m;
  return DOPR_OK;
}

dopr_status dopr_store_create(const dopr_model_config* cfg, int64_t max_doc_id, int64_t pool_bytes, dopr_store** out) {
  g_last_error.clear();
  if (!out) return fail(DOPR_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  STATUS_TRY(check_cfg(cfg));
  if (max_doc_id < 0 || max_doc_id >= (1ll << 31) - 1) return fail(DOPR_ERR_INVALID_ARG, "bad max_doc_id");
  if (pool_bytes < 0) return fail(DOPR_ERR_INVALID_ARG, "bad pool_bytes");
  if (pool_bytes / 256 >= (1ll << 31)) return fail(DOPR_ERR_UNSUPPORTED, "pool above 512 GiB");
  dopr_store* s = new dopr_store();
  s->cfg = *cfg;
  s->max_doc_id = max_doc_id;
  s->pool_rows = pool_bytes / 256;
  s->pool_bytes = s->pool_rows * 256;
  cudaGetDevice(&s->device);
  const size_t nd = (size_t)max_doc_id + 1;
  dopr_status st = DOPR_OK;
  auto guard = [&](dopr_status x) {
    if (x != DOPR_OK && st == DOPR_OK) st = x;
    return x == DOPR_OK;
  };
  if (guard(dev_alloc(&s->pool, (size_t)std::max<int64_t>(s->pool_bytes, 256))) &&
      guard(dev_alloc(&s->d_slot_of, nd)) && guard(dev_alloc(&s->d_slot_m, nd)) &&
      guard(dev_alloc(&s->d_slot_row, nd)) && guard(dev_alloc(&s->d_slot_ok, nd)) && guard(dev_alloc(&s->d_range, 1))) {
    if (cudaMemset(s->d_slot_of, 0xFF, nd * sizeof(int32_t)) != cudaSuccess ||
        cudaMemset(s->d_slot_ok, 0, nd) != cudaSuccess || cudaMemset(s->d_slot_m, 0, nd * sizeof(int32_t)) ||
        cudaMemset(s->pool, 0, (size_t)std::max<int64_t>(s->pool_bytes, 256)) != cudaSuccess)
      guard(fail(DOPR_ERR_CUDA, "store initialisation failed"));
  }
  if (st == DOPR_OK &&
      !make_tmap_16b_2d(&s->tm_pool, s->pool, HEAD_DIM, std::max<int64_t>(s->pool_rows, 1), HEAD_DIM * 2, 64, 64, true,
                        true))
    guard(fail(DOPR_ERR_CUDA, "cuTensorMapEncodeTiled failed for the store pool"));
  if (st != DOPR_OK) {
    free_store(s);
    delete s;
    return st;
  }
  s->tm_pool_ok = true;
  s->slot_of.assign(nd, -1);
  *out = s;
  return DOPR_OK;
}

dopr_status dopr_store_put(dopr_store* s, int64_t doc_id, int32_t m, int32_t layer, const void* k, const void* v,
                           int32_t src_on_device) {
  g_last_error.clear();
  if (!s) return fail(DOPR_ERR_INVALID_ARG, "store is NULL");
  const auto& c = s->cfg;
  if (doc_id < 0 || doc_id > s->max_doc_id) return fail(DOPR_ERR_INVALID_ARG, "doc_id %lld out of range", (long long)doc_id);
  if (m < 0 || m > MAX_PREFIX) return fail(DOPR_ERR_INVALID_ARG, "m = %d outside [0, %d]", m, MAX_PREFIX);
  if (layer < 0 || layer >= c.n_layers) return fail(DOPR_ERR_INVALID_ARG, "bad layer %d", layer);
  if (m > 0 && (!k || !v)) return fail(DOPR_ERR_INVALID_ARG, "k or v is NULL");
  const int64_t Hkv = c.n_kv_heads;
  const int64_t rows_per_layer = 2 * Hkv * m;  // K and V, [head][m] rows of 128
  CUDA_TRY(cudaSetDevice(s->device));
  int32_t slot = -1;
  STATUS_TRY(store_reserve(s, doc_id, m, &slot));
  if (m > 0) {
    const size_t bytes = (size_t)m * Hkv * HEAD_DIM * 2;
    f16* base = reinterpret_cast<f16*>(s->pool) + (size_t)(s->slot_row[slot] + layer * rows_per_layer) * HEAD_DIM;
    const bf16 *dk = static_cast<const bf16*>(k), *dv = static_cast<const bf16*>(v);
    bf16* stage = nullptr;
    if (!src_on_device) {
      CUDA_TRY(cudaMalloc(&stage, 2 * bytes));
      cudaError_t e1 = cudaMemcpy(stage, k, bytes, cudaMemcpyHostToDevice);
      cudaError_t e2 = cudaMemcpy(stage + bytes / 2, v, bytes, cudaMemcpyHostToDevice);
      if (e1 != cudaSuccess || e2 != cudaSuccess) {
        cudaFree(stage);
        return fail(DOPR_ERR_CUDA, "prefix upload failed");
      }
      dk = stage;
      dv = stage + bytes / 2;
    }
    int range = 0;
    cudaError_t e = cudaMemsetAsync(s->d_range, 0, sizeof(int), 0);
    if (e == cudaSuccess)
      e = launch_store_transpose(dk, dv, m, (int)Hkv, base, base + (size_t)Hkv * m * HEAD_DIM, s->d_range, 0);
    if (e == cudaSuccess) e = cudaMemcpy(&range, s->d_range, sizeof(int), cudaMemcpyDeviceToHost);
    if (stage) cudaFree(stage);
    if (e != cudaSuccess) return fail(DOPR_ERR_CUDA, "prefix store copy failed: %s", cudaGetErrorString(e));
    if (range) {
      // the layer now holds clamped data: mark it missing until a valid put replaces it
      STATUS_TRY(store_mark(s, slot, layer, false));
      return fail(DOPR_ERR_INVALID_ARG, "doc %lld layer %d: a prefix value is not finite or exceeds the fp16 range",
                  (long long)doc_id, layer);
    }
  }
  return store_mark(s, slot, layer, true);
}

dopr_status dopr_build_prefixes(dopr_model* m, dopr_store* s, int32_t n_docs, const int64_t* doc_ids,
                                const int32_t* x_offsets, const void* x, int32_t x_on_device, void* cuda_stream) {
  g_last_error.clear();
  NvtxRange call_range("dopr_build_prefixes");
  STATUS_TRY(check_ready(m, s));
  if (n_docs < 0) return fail(DOPR_ERR_INVALID_ARG, "n_docs < 0");
  if (n_docs == 0) return DOPR_OK;
  if (!doc_ids || !x_offsets) return fail(DOPR_ERR_INVALID_ARG, "NULL array");
  const auto& c = m->cfg;
  const int H = c.hidden, L = c.n_layers;
  if (x_offsets[0] != 0) return fail(DOPR_ERR_INVALID_ARG, "x_offsets[0] must be 0");
  std::vector<char> seen;
  for (int32_t d = 0; d < n_docs; ++d) {
    const int32_t md = x_offsets[d + 1] - x_offsets[d];
    if (md < 0 || md > MAX_PREFIX) return fail(DOPR_ERR_INVALID_ARG, "doc %d: m = %d outside [0, %d]", d, md, MAX_PREFIX);
    if (md > c.max_position) return fail(DOPR_ERR_INVALID_ARG, "doc %d: m = %d beyond max_position", d, md);
    if (doc_ids[d] < 0 || doc_ids[d] > s->max_doc_id)
      return fail(DOPR_ERR_INVALID_ARG, "doc_id %lld out of range", (long long)doc_ids[d]);
  }
  {
    std::vector<int64_t> ids(doc_ids, doc_ids + n_docs);
    std::sort(ids.begin(), ids.end());
    if (std::adjacent_find(ids.begin(), ids.end()) != ids.end())
      return fail(DOPR_ERR_INVALID_ARG, "a doc_id appears twice in one build");
  }
  const int64_t rows = x_offsets[n_docs];
  if (rows > 0 && !x) return fail(DOPR_ERR_INVALID_ARG, "x is NULL");
  CUDA_TRY(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  Workspace& w = m->ws;
  // slots first (validated above, so only a full pool can fail here)
  std::vector<int32_t> slot(n_docs);
  for (int32_t d = 0; d < n_docs; ++d) STATUS_TRY(store_reserve(s, doc_ids[d], x_offsets[d + 1] - x_offsets[d], &slot[d]));
  // the documents with a prefix are the "pairs" of the pass, their rows its tokens
  std::vector<int32_t> pd;
  for (int32_t d = 0; d < n_docs; ++d)
    if (x_offsets[d + 1] > x_offsets[d]) pd.push_back(d);
  const int32_t n = (int32_t)pd.size();
  if (n > 0) {
    STATUS_TRY(ensure_call_buffers(m, n, rows, 0, 0));
    std::vector<int32_t> tok_id(rows), tok_pos(rows), tok_pair(rows);
    w.h_tok_off[0] = 0;
    for (int32_t p = 0; p < n; ++p) {
      const int32_t d = pd[p], md = x_offsets[d + 1] - x_offsets[d];
      w.h_sorted_slot[p] = slot[d];
      for (int32_t j = 0; j < md; ++j) {
        const int32_t t = w.h_tok_off[p] + j;
        tok_id[t] = x_offsets[d] + j;  // row of x (the embedding kernel gathers it)
        tok_pos[t] = j;
        tok_pair[t] = p;
      }
      w.h_tok_off[p + 1] = w.h_tok_off[p] + md;
    }
    const int64_t T = w.h_tok_off[n];
    CUDA_TRY(cudaMemcpyAsync(w.tok_off, w.h_tok_off, sizeof(int32_t) * (n + 1), cudaMemcpyHostToDevice, st));
    CUDA_TRY(cudaMemcpyAsync(w.sorted_slot, w.h_sorted_slot, sizeof(int32_t) * n, cudaMemcpyHostToDevice, st));
    CUDA_TRY(cudaMemcpyAsync(w.tok_id, tok_id.data(), sizeof(int32_t) * T, cudaMemcpyHostToDevice, st));
    CUDA_TRY(cudaMemcpyAsync(w.tok_pos, tok_pos.data(), sizeof(int32_t) * T, cudaMemcpyHostToDevice, st));
    CUDA_TRY(cudaMemcpyAsync(w.tok_pair, tok_pair.data(), sizeof(int32_t) * T, cudaMemcpyHostToDevice, st));
    // chunks of whole documents; attention with no prefix, so a chunk's documents form one run
    AttnPlanner ap;
    ap.TT = attn_tc_rows_per_head(c.n_q_heads / c.n_kv_heads);
    Plan plan;
    plan.n_tokens = T;
    plan.chunk_pair.assign(1, 0);
    plan.chunk_item.assign(1, 0);
    plan.chunk_litem.assign(1, 0);
    plan.chunk_tile.assign(1, 0);
    plan.chunk_ltile.assign(1, 0);
    for (int32_t s0 = 0; s0 < n;) {
      int32_t s1 = s0 + 1;
      while (s1 < n && w.h_tok_off[s1 + 1] - w.h_tok_off[s0] <= w.chunk_cap) ++s1;
      ap.add(w.h_tok_off, w.h_tok_off[s0], s0, s1, 0, 0, 0);
      plan.chunk_pair.push_back(s1);
      plan.chunk_item.push_back(0);
      ap.close_chunk(plan);
      s0 = s1;
    }
    STATUS_TRY(ap.upload(w, plan, 0, st));
    // the representations on the device
    const bf16* dx = static_cast<const bf16*>(x);
    bf16* stage = nullptr;
    if (!x_on_device) {
      CUDA_TRY(cudaMalloc(&stage, sizeof(bf16) * (size_t)rows * H));
      cudaError_t e = cudaMemcpyAsync(stage, x, sizeof(bf16) * (size_t)rows * H, cudaMemcpyHostToDevice, st);
      if (e != cudaSuccess) {
        cudaFree(stage);
        return fail(DOPR_ERR_CUDA, "prefix input upload failed");
      }
      dx = stage;
    }
    CUDA_TRY(cudaMemsetAsync(w.err, 0, sizeof(int), st));
    BuildArgs b{dx, (int64_t)rows};
    const dopr_status rs = run_layers(m, s, plan, nullptr, st, &b);
    cudaError_t e = cudaMemcpyAsync(w.h_err, w.err, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (stage) cudaFree(stage);
    STATUS_TRY(rs);
    if (e != cudaSuccess) return fail(DOPR_ERR_CUDA, "prefix build failed: %s", cudaGetErrorString(e));
    STATUS_TRY(map_device_error(*w.h_err));
  }
  for (int32_t d = 0; d < n_docs; ++d)
    for (int l = 0; l < L; ++l) STATUS_TRY(store_mark(s, slot[d], l, true));
  return DOPR_OK;
}

dopr_status dopr_select_prefix_inputs(dopr_model* m, int32_t n_docs, const int32_t* doc_offsets,
                                      const int32_t* doc_tokens, int32_t top_k, int32_t top_p, int32_t* positions,
                                      void* x_out, float* salience, void* cuda_stream) {
  g_last_error.clear();
  NvtxRange call_range("dopr_select_prefix_inputs");
  if (!m) return fail(DOPR_ERR_INVALID_ARG, "model is NULL");
  const auto& c = m->cfg;
  const int H = c.hidden, L = c.n_layers;
  for (int k = 0; k < kind_count(); ++k)
    for (int l = 0; l < (kind_is_global(k) ? 1 : L); ++l)
      if (!m->have[k * L + l]) return fail(DOPR_ERR_INCOMPLETE, "weight kind %d layer %d was never put", k, l);
  if (n_docs < 0) return fail(DOPR_ERR_INVALID_ARG, "n_docs < 0");
  if (n_docs == 0) return DOPR_OK;
  if (!doc_offsets || !doc_tokens || !positions || !x_out) return fail(DOPR_ERR_INVALID_ARG, "NULL array");
  if (top_k < 1 || top_k > MAX_PREFIX) return fail(DOPR_ERR_INVALID_ARG, "top_k = %d outside [1, %d]", top_k, MAX_PREFIX);
  if (top_p < 1) return fail(DOPR_ERR_INVALID_ARG, "top_p < 1");
  if (doc_offsets[0] != 0) return fail(DOPR_ERR_INVALID_ARG, "doc_offsets[0] must be 0");
  for (int32_t d = 0; d < n_docs; ++d) {
    const int32_t nd = doc_offsets[d + 1] - doc_offsets[d];
    if (nd < 1 || nd > SEL_MAX_N) return fail(DOPR_ERR_INVALID_ARG, "document %d: %d tokens outside [1, %d]", d, nd, SEL_MAX_N);
    if (nd > c.max_position) return fail(DOPR_ERR_INVALID_ARG, "document %d: %d tokens beyond max_position", d, nd);
  }
  const int64_t T = doc_offsets[n_docs];
  for (int64_t t = 0; t < T; ++t)
    if (doc_tokens[t] < 0 || doc_tokens[t] >= c.vocab) return fail(DOPR_ERR_INVALID_ARG, "token %lld out of range", (long long)t);
  CUDA_TRY(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  Workspace& w = m->ws;
  // a store of one empty document gives the attention kernels a valid pool map
  // (made once per model and kept, like the selection buffers below)
  if (!w.sel_empty) {
    dopr_store* empty = nullptr;
    STATUS_TRY(dopr_store_create(&c, 0, 256, &empty));
    w.sel_empty = empty;
  }
  dopr_status rs = ensure_call_buffers(m, n_docs, T, 0, 0);
  if (rs != DOPR_OK) return rs;
  std::vector<int32_t> tok_pos(T), tok_pair(T);
  for (int32_t d = 0; d < n_docs; ++d) {
    w.h_tok_off[d] = doc_offsets[d];
    w.h_sorted_slot[d] = 0;
    for (int32_t j = doc_offsets[d]; j < doc_offsets[d + 1]; ++j) {
      tok_pos[j] = j - doc_offsets[d];
      tok_pair[j] = d;
    }
  }
  w.h_tok_off[n_docs] = (int32_t)T;
  CUDA_TRY(cudaMemcpyAsync(w.tok_off, w.h_tok_off, sizeof(int32_t) * (n_docs + 1), cudaMemcpyHostToDevice, st));
  CUDA_TRY(cudaMemcpyAsync(w.sorted_slot, w.h_sorted_slot, sizeof(int32_t) * n_docs, cudaMemcpyHostToDevice, st));
  CUDA_TRY(cudaMemcpyAsync(w.tok_id, doc_tokens, sizeof(int32_t) * T, cudaMemcpyHostToDevice, st));
  CUDA_TRY(cudaMemcpyAsync(w.tok_pos, tok_pos.data(), sizeof(int32_t) * T, cudaMemcpyHostToDevice, st));
  CUDA_TRY(cudaMemcpyAsync(w.tok_pair, tok_pair.data(), sizeof(int32_t) * T, cudaMemcpyHostToDevice, st));
  // chunks of whole documents; no prefix, so a chunk's documents form one attention run
  AttnPlanner ap;
  ap.TT = attn_tc_rows_per_head(c.n_q_heads / c.n_kv_heads);
  Plan plan;
  plan.n_tokens = T;
  plan.chunk_pair.assign(1, 0);
  plan.chunk_item.assign(1, 0);
  plan.chunk_litem.assign(1, 0);
  plan.chunk_tile.assign(1, 0);
  plan.chunk_ltile.assign(1, 0);
  int64_t a_max = 0;
  int32_t docs_max = 0;
  for (int32_t s0 = 0; s0 < n_docs;) {
    int32_t s1 = s0 + 1;
    while (s1 < n_docs && w.h_tok_off[s1 + 1] - w.h_tok_off[s0] <= w.chunk_cap) ++s1;
    ap.add(w.h_tok_off, w.h_tok_off[s0], s0, s1, 0, 0, 0);
    int64_t a = 0;
    for (int32_t d = s0; d < s1; ++d) a += (int64_t)(doc_offsets[d + 1] - doc_offsets[d]) * (doc_offsets[d + 1] - doc_offsets[d]);
    a_max = std::max(a_max, a);
    docs_max = std::max(docs_max, s1 - s0);
    plan.chunk_pair.push_back(s1);
    plan.chunk_item.push_back(0);
    ap.close_chunk(plan);
    s0 = s1;
  }
  STATUS_TRY(ap.upload(w, plan, 0, st));
  // selection buffers, grown on demand and kept for the next call
  STATUS_TRY(grow_dev(&w.sel_A, w.sel_a_cap, a_max));
  STATUS_TRY(grow_dev(&w.sel_a_off, w.sel_doc_cap, docs_max));
  STATUS_TRY(grow_dev(&w.sel_u, w.sel_tok_cap, T));
  STATUS_TRY(grow_dev(&w.sel_pos, w.sel_pos_cap, (int64_t)n_docs * top_k));
  STATUS_TRY(grow_dev(&w.sel_x, w.sel_x_cap, (int64_t)n_docs * top_k * H));
  SelectState sel{top_k, top_p, w.sel_A, a_max, w.sel_a_off, w.sel_u, w.sel_pos, w.sel_x};
  cudaError_t e = cudaMemsetAsync(w.err, 0, sizeof(int), st);
  rs = e == cudaSuccess ? run_layers(m, w.sel_empty, plan, nullptr, st, nullptr, &sel)
                         : fail(DOPR_ERR_CUDA, "memset failed");
  if (rs == DOPR_OK) {
    e = cudaMemcpyAsync(positions, sel.positions, sizeof(int32_t) * n_docs * top_k, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(x_out, sel.x, sizeof(bf16) * (size_t)n_docs * top_k * H, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess && salience) e = cudaMemcpyAsync(salience, sel.u, sizeof(float) * T, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(w.h_err, w.err, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) rs = fail(DOPR_ERR_CUDA, "selection failed: %s", cudaGetErrorString(e));
  } else {
    cudaStreamSynchronize(st);
  }
  STATUS_TRY(rs);
  return map_device_error(*w.h_err);
}

dopr_status dopr_debug_store_read(const dopr_store* s, int64_t doc_id, int32_t layer, void* k_out, void* v_out) {
  g_last_error.clear();
  if (!s) return fail(DOPR_ERR_INVALID_ARG, "store is NULL");
  if (doc_id < 0 || doc_id > s->max_doc_id || s->slot_of[doc_id] < 0)
    return fail(DOPR_ERR_UNKNOWN_DOC, "doc %lld is not stored", (long long)doc_id);
  if (layer < 0 || layer >= s->cfg.n_layers) return fail(DOPR_ERR_INVALID_ARG, "bad layer %d", layer);
  const int32_t slot = s->slot_of[doc_id], md = s->slot_m[slot];
  const int Hkv = s->cfg.n_kv_heads;
  if (md == 0) return DOPR_OK;
  if (!k_out || !v_out) return fail(DOPR_ERR_INVALID_ARG, "NULL output");
  CUDA_TRY(cudaSetDevice(s->device));
  const size_t n = (size_t)2 * Hkv * md * HEAD_DIM;
  std::vector<uint16_t> buf(n);
  const uint16_t* src =
      reinterpret_cast<const uint16_t*>(s->pool) + (size_t)(s->slot_row[slot] + (int64_t)layer * 2 * Hkv * md) * HEAD_DIM;
  CUDA_TRY(cudaMemcpy(buf.data(), src, n * sizeof(uint16_t), cudaMemcpyDeviceToHost));
  uint16_t* ko = static_cast<uint16_t*>(k_out);
  uint16_t* vo = static_cast<uint16_t*>(v_out);
  for (int g = 0; g < Hkv; ++g)  // pool [K|V][head][m][128] -> caller [m][head][128]
    for (int j = 0; j < md; ++j)
      for (int e = 0; e < HEAD_DIM; ++e) {
        ko[((size_t)j * Hkv + g) * HEAD_DIM + e] = buf[((size_t)g * md + j) * HEAD_DIM + e];
        vo[((size_t)j * Hkv + g) * HEAD_DIM + e] = buf[((size_t)(Hkv + g) * md + j) * HEAD_DIM + e];
      }
  return DOPR_OK;
}

dopr_status dopr_store_destroy(dopr_store* s) {
  g_last_error.clear();
  if (!s) return DOPR_OK;
  cudaSetDevice(s->device);
  free_store(s);
  delete s;
  return DOPR_OK;
}

dopr_status dopr_score(dopr_model* m, dopr_store* s, int32_t n, const int32_t* q_offsets, const int32_t* q_tokens,
                       const int64_t* doc_ids, float* scores, void* cuda_stream, int32_t io_on_device) {
  g_last_error.clear();
  NvtxRange call_range("dopr_score");
  STATUS_TRY(check_ready(m, s));
  if (n < 0) return fail(DOPR_ERR_INVALID_ARG, "n_pairs < 0");
  if (n == 0) return DOPR_OK;
  if (!q_offsets || !doc_ids || !scores) return fail(DOPR_ERR_INVALID_ARG, "NULL array");
  CUDA_TRY(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  Workspace& w = m->ws;
  const int32_t *dqo = q_offsets, *dqt = q_tokens;
  const int64_t* ddoc = doc_ids;
  if (!io_on_device) {
    if (n > 0 && q_offsets[n] > 0 && !q_tokens) return fail(DOPR_ERR_INVALID_ARG, "q_tokens is NULL");
    STATUS_TRY(validate_host_inputs(m, s, n, q_offsets, q_tokens, doc_ids));
    const int64_t nq = q_offsets[n];
    STATUS_TRY(ensure_call_buffers(m, n, 0, std::max<int64_t>(nq, 1), s->max_doc_id + 1));
    CUDA_TRY(cudaMemcpyAsync(w.q_off, q_offsets, sizeof(int32_t) * (n + 1), cudaMemcpyHostToDevice, st));
    if (nq > 0) CUDA_TRY(cudaMemcpyAsync(w.q_tok, q_tokens, sizeof(int32_t) * nq, cudaMemcpyHostToDevice, st));
    CUDA_TRY(cudaMemcpyAsync(w.doc_ids, doc_ids, sizeof(int64_t) * n, cudaMemcpyHostToDevice, st));
    dqo = w.q_off;
    dqt = w.q_tok;
    ddoc = w.doc_ids;
  } else {
    STATUS_TRY(ensure_call_buffers(m, n, 0, 0, s->max_doc_id + 1));
  }
  Plan plan;
  STATUS_TRY(run_packer(m, s, n, dqo, dqt, ddoc, st, plan));
  // scores land in the workspace and reach the caller only once the device error
  // word is known to be clear: a failed call writes nothing
  STATUS_TRY(run_layers(m, s, plan, w.scores, st));
  CUDA_TRY(cudaMemcpyAsync(w.h_err, w.err, sizeof(int), cudaMemcpyDeviceToHost, st));
  CUDA_TRY(cudaStreamSynchronize(st));
  prof_collect(m);
  STATUS_TRY(map_device_error(*w.h_err));
  CUDA_TRY(cudaMemcpyAsync(scores, w.scores, sizeof(float) * n,
                           io_on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, st));
  CUDA_TRY(cudaStreamSynchronize(st));
  return DOPR_OK;
}

dopr_status dopr_debug_pack_plan(dopr_model* m, dopr_store* s, int32_t n, const int32_t* q_offsets,
                                 const int32_t* q_tokens, const int64_t* doc_ids, int32_t* perm, int32_t* tok_off,
                                 int32_t* tok_pos, int32_t* tok_id, int32_t* tok_pair) {
  g_last_error.clear();
  if (!m || !s) return fail(DOPR_ERR_INVALID_ARG, "model or store is NULL");
  if (!same_shape(m->cfg, s->cfg)) return fail(DOPR_ERR_INVALID_ARG, "store shape (layers, kv heads, head_dim, max_position) does not match the model");
  if (n < 0 || !q_offsets || (n > 0 && (!doc_ids || !perm || !tok_off))) return fail(DOPR_ERR_INVALID_ARG, "bad args");
  if (n == 0) {
    tok_off[0] = 0;
    return DOPR_OK;
  }
  STATUS_TRY(validate_host_inputs(m, s, n, q_offsets, q_tokens, doc_ids));
  CUDA_TRY(cudaSetDevice(m->device));
  Workspace& w = m->ws;
  const int64_t nq = q_offsets[n];
  STATUS_TRY(ensure_call_buffers(m, n, 0, std::max<int64_t>(nq, 1), s->max_doc_id + 1));
  cudaStream_t st = 0;
  CUDA_TRY(cudaMemcpy(w.q_off, q_offsets, sizeof(int32_t) * (n + 1), cudaMemcpyHostToDevice));
  if (nq > 0) CUDA_TRY(cudaMemcpy(w.q_tok, q_tokens, sizeof(int32_t) * nq, cudaMemcpyHostToDevice));
  CUDA_TRY(cudaMemcpy(w.doc_ids, doc_ids, sizeof(int64_t) * n, cudaMemcpyHostToDevice));
  Plan plan;
  STATUS_TRY(run_packer(m, s, n, w.q_off, w.q_tok, w.doc_ids, st, plan));
  const int64_t T = plan.n_tokens;
  CUDA_TRY(cudaStreamSynchronize(st));
  CUDA_TRY(cudaMemcpy(perm, w.perm, sizeof(int32_t) * n, cudaMemcpyDeviceToHost));
  CUDA_TRY(cudaMemcpy(tok_off, w.tok_off, sizeof(int32_t) * (n + 1), cudaMemcpyDeviceToHost));
  if (tok_pos) CUDA_TRY(cudaMemcpy(tok_pos, w.tok_pos, sizeof(int32_t) * T, cudaMemcpyDeviceToHost));
  if (tok_id) CUDA_TRY(cudaMemcpy(tok_id, w.tok_id, sizeof(int32_t) * T, cudaMemcpyDeviceToHost));
  if (tok_pair) CUDA_TRY(cudaMemcpy(tok_pair, w.tok_pair, sizeof(int32_t) * T, cudaMemcpyDeviceToHost));
  CUDA_TRY(cudaMemcpy(w.h_err, w.err, sizeof(int), cudaMemcpyDeviceToHost));
  prof_collect(m);
  return map_device_error(*w.h_err);
}

int32_t dopr_debug_attention_plan(int32_t m, int32_t rows_per_tile, int32_t n_pairs, const int32_t* tok_len,
                                  int32_t max_tiles, int32_t* out) {
  g_last_error.clear();
  if (m < 0 || rows_per_tile < 1 || rows_per_tile > 128 || n_pairs < 1 || !tok_len || max_tiles < 0 || !out) {
    fail(DOPR_ERR_INVALID_ARG, "bad attention-plan arguments");
    return -DOPR_ERR_INVALID_ARG;
  }
  std::vector<int32_t> to(n_pairs + 1, 0);
  for (int32_t p = 0; p < n_pairs; ++p) {
    if (tok_len[p] < 1 || to[p] > INT32_MAX - tok_len[p]) {
      fail(DOPR_ERR_INVALID_ARG, "tok_len[%d] must be >= 1", p);
      return -DOPR_ERR_INVALID_ARG;
    }
    to[p + 1] = to[p] + tok_len[p];
  }
  AttnPlanner pl;
  pl.TT = rows_per_tile;
  pl.add(to.data(), 0, 0, n_pairs, 0, m, 0);
  std::vector<std::pair<int32_t, const AttnTile*>> all;  // (kind, tile) in token order
  for (const AttnTile& t : pl.tiles) all.push_back({0, &t});
  for (const AttnTile& t : pl.ltiles) all.push_back({1, &t});
  std::sort(all.begin(), all.end(), [](const auto& a, const auto& b) { return a.second->tok_begin < b.second->tok_begin; });
  if ((int64_t)all.size() > max_tiles) {
    fail(DOPR_ERR_INVALID_ARG, "the plan has %zu tiles, max_tiles is %d", all.size(), max_tiles);
    return -DOPR_ERR_INVALID_ARG;
  }
  for (size_t i = 0; i < all.size(); ++i) {
    const AttnTile& t = *all[i].second;
    int32_t* o = out + 24 * i;
    o[0] = all[i].first;
    o[1] = t.tok_begin;
    o[2] = t.n_tok;
    o[3] = t.n_keys;
    o[4] = t.n_seg;
    o[5] = o[6] = o[7] = 0;
    for (int j = 0; j < ATTN_TC_MAX_SEGS; ++j) o[8 + j] = j < t.n_seg ? t.seg[j] : 0;
  }
  return (int32_t)all.size();
}

dopr_status dopr_debug_gemm(int32_t M, int32_t N, int32_t K, const void* A, const void* B, void* out,
                            int32_t epilogue, void* cuda_stream) {
  g_last_error.clear();
  if (M < 0 || N <= 0 || K <= 0 || !A || !B || !out) return fail(DOPR_ERR_INVALID_ARG, "bad gemm args");
  if (K % GEMM_BK || N % GEMM_BN) return fail(DOPR_ERR_UNSUPPORTED, "K % 64 and N % 256 must be 0");
  if (epilogue < 0 || epilogue > 2) return fail(DOPR_ERR_INVALID_ARG, "bad epilogue %d", epilogue);
  if (M == 0) return DOPR_OK;
  if (gemm_setup() != cudaSuccess) return fail(DOPR_ERR_CUDA, "gemm setup failed");
  CUtensorMap ta, tb;
  if (!make_tmap_16b_2d(&ta, A, K, M, (uint64_t)K * 2, GEMM_BK, GEMM_BM, true, true) ||
      !make_tmap_16b_2d(&tb, B, K, N, (uint64_t)K * 2, GEMM_BK, GEMM_B_BOX, true, true))
    return fail(DOPR_ERR_CUDA, "cuTensorMapEncodeTiled failed (pointers must be 16-byte aligned)");
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  int* err = nullptr;
  CUDA_TRY(cudaMalloc(&err, sizeof(int)));
  cudaMemsetAsync(err, 0, sizeof(int), st);
  GemmParams gp{};
  gp.M = M;
  gp.N = N;
  gp.K = K;
  gp.out = out;
  gp.ld_out = epilogue == EPI_SWIGLU ? N / 2 : N;
  gp.err = err;
  cudaError_t e = launch_gemm(epilogue, ta, tb, gp, sms, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  int h = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&h, err, sizeof(int), cudaMemcpyDeviceToHost);
  cudaFree(err);
  if (e != cudaSuccess) return fail(DOPR_ERR_CUDA, "gemm failed: %s", cudaGetErrorString(e));
  return map_device_error(h);
}

dopr_status dopr_profile_enable(dopr_model* m, int32_t enable) {
  g_last_error.clear();
  if (!m) return fail(DOPR_ERR_INVALID_ARG, "model is NULL");
  m->prof.reset();
  m->prof.on = enable != 0;
  return DOPR_OK;
}

int32_t dopr_profile_read(const dopr_model* m, dopr_kernel_stat* out, int32_t max_entries) {
  if (!m) return -1;
  for (int k = 0; k < K_COUNT && k < max_entries && out; ++k) {
    memset(&out[k], 0, sizeof(out[k]));
    snprintf(out[k].name, sizeof(out[k].name), "%s", kKindNames[k]);
    out[k].launches = m->prof.launches[k];
    out[k].time_ms = m->prof.ms[k];
    out[k].flops = m->prof.flops[k];
    out[k].bytes = m->prof.bytes[k];
  }
  return K_COUNT;
}

dopr_status dopr_debug_wait_timeout(int32_t timeout_ms) {
  g_last_error.clear();
  if (timeout_ms <= 0 || timeout_ms > 10000) return fail(DOPR_ERR_INVALID_ARG, "timeout_ms in (0, 10000]");
  int* err = nullptr;
  CUDA_TRY(cudaMalloc(&err, sizeof(int)));
  cudaMemset(err, 0, sizeof(int));
  cudaError_t e = launch_wait_timeout_probe(err, (uint64_t)timeout_ms * 1000000ull, 0);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  int h = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&h, err, sizeof(int), cudaMemcpyDeviceToHost);
  cudaFree(err);
  if (e != cudaSuccess) return fail(DOPR_ERR_CUDA, "probe failed: %s", cudaGetErrorString(e));
  return map_device_error(h);
}

}  // extern "C"
