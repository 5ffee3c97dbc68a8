// internal.h -- host-side structures of libdopr and the launchers each kernel
// file exports to the engine (abi.cu).  Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/dopr.h"

namespace dopr {

typedef __nv_bfloat16 bf16;
typedef __half f16;  // tensor-core operand type of the scoring pass (fp32 accumulation)

constexpr int HEAD_DIM = 128;
constexpr int MAX_PREFIX = 256;       // largest m the store accepts
constexpr int ATTN_MAX_PAIRS = 8;     // pairs of one doc per attention work item
constexpr uint64_t WAIT_TIMEOUT_NS = 4000000000ull;  // bounded device waits: 4 s

// Buffer extents the index tests of a checked build compare against (see
// index_ok in device_common.cuh); plain builds carry them unused.
struct Extents {
  int* err = nullptr;      // the call's device error word
  int64_t rows = 0;        // rows of the chunk's activation buffers (packed tokens)
  int64_t table_rows = 0;  // rows of the table a gather reads (embedding, or a build's input vectors)
  int64_t pool_rows = 0;   // 256-byte rows of the store pool
  int64_t a_elems = 0;     // floats of the key token selection's attention matrices
};

// One attention work item: consecutive sorted pairs that share a document.
struct AttnItem {
  int32_t pair_begin, pair_end;  // sorted pair indices [begin, end)
  int32_t slot;                  // store slot of the document
  int32_t m;                     // its prefix length
};

// Tensor-core attention (k_attn_tc.cu).  A tile is up to 128 / G consecutive
// packed tokens of pairs of one document; its keys are the prefix (ceil64(m)
// columns) then one segment per pair it touches, from the pair's first token to
// the tile's last, each padded to a multiple of 16 columns.  A tile keeps within
// ATTN_TC_MAX_KEYS columns (k_attn_tc) unless its first token alone needs more
// (a long tile, k_attn_tc_long, no key limit).  The mma.sync kernel (k_attn.cu)
// takes the last layer's score-token rows, and every row when 128 / G gives no
// tile shape.
constexpr int ATTN_TC_MAX_KEYS = 256;
constexpr int ATTN_TC_MAX_SEGS = 16;  // own segments are >= 16 columns each
struct __align__(16) AttnTile {
  int64_t pool_base;   // first store-pool row of the document's slot
  int32_t tok_begin;   // first token, relative to the chunk
  int32_t n_tok;       // tokens in the tile (<= 128 / G)
  int32_t m;           // the document's prefix length
  int32_t n_keys;      // key columns (multiple of 16, <= ATTN_TC_MAX_KEYS)
  int32_t n_seg;       // own segments, one per pair the tile touches, in token order
  int32_t pad;
  // segment s: the pair starts at token tok_begin + (int16_t)(seg[s] & 0xffff) (<= 0 for
  // a pair begun before the tile) and has seg[s] >> 16 tokens up to the tile's end
  int32_t seg[ATTN_TC_MAX_SEGS];
};

struct Store {
  dopr_model_config cfg{};
  int device = 0;
  int64_t max_doc_id = 0;
  int64_t pool_bytes = 0, pool_rows = 0, used_rows = 0;  // rows of 128 fp16 (256 B)
  uint8_t* pool = nullptr;          // prefix K/V as fp16 (converted from the bf16 the caller passes)
  int* d_range = nullptr;           // set by the put conversion when a value leaves the fp16 range
  int32_t* d_slot_of = nullptr;     // [max_doc_id+1] doc -> slot, -1 absent
  int32_t* d_slot_m = nullptr;      // [max_doc_id+1] per slot prefix length
  int64_t* d_slot_row = nullptr;    // [max_doc_id+1] first pool row of the slot block
  uint8_t* d_slot_ok = nullptr;     // [max_doc_id+1] all layers present
  std::vector<int32_t> slot_of;     // host mirrors
  std::vector<int32_t> slot_m;
  std::vector<int64_t> slot_row;
  std::vector<std::vector<uint8_t>> slot_layers;
  std::vector<uint8_t> slot_ok;
  int32_t n_slots = 0;
  int32_t max_m = 0;
  CUtensorMap tm_pool{};
  bool tm_pool_ok = false;
};

struct Workspace {
  int chunk_cap = 0;  // tokens per chunk
  float* r = nullptr;          // [chunk][H] fp32 residual stream
  f16* xn = nullptr;           // [chunk][H] norm operand (see GemmParams)
  f16* qkv = nullptr;          // [chunk][(Hq+2Hkv)*128] q, k after norm+RoPE, v
  f16* o = nullptr;            // [chunk][Hq*128] attention output
  f16* act = nullptr;          // [chunk][F] SwiGLU output
  float* ss_e = nullptr;       // [chunk] sum of squares of the embedded rows
  float* ss_a = nullptr;       // [chunk][2H/256] partial sums of squares for the attention norm
  float* ss_m = nullptr;       // [chunk][2H/256] partial sums of squares for the MLP norm
  float* r_s = nullptr;        // [chunk][H] score-token rows of the last layer (compact)
  float* ss_s = nullptr;       // [chunk][2H/256] their attention-norm partial sums
  CUtensorMap tm_xn{}, tm_o{}, tm_act{};
  // per call, grown on demand
  int64_t pair_cap = 0, tok_cap = 0, qtok_cap = 0, doc_cap = 0, item_cap = 0;
  int32_t* q_off = nullptr;
  int32_t* q_tok = nullptr;
  int64_t* doc_ids = nullptr;
  float* scores = nullptr;
  int32_t* pair_slot = nullptr;
  int32_t* perm = nullptr;
  int32_t* sorted_slot = nullptr;
  int32_t* tok_off = nullptr;
  int32_t* tok_id = nullptr;
  int32_t* tok_pos = nullptr;
  int32_t* tok_pair = nullptr;
  int32_t* doc_count = nullptr;  // [max_doc_id+1] counting-sort buckets
  AttnItem* items = nullptr;     // all items of the call, then the mma.sync kernel's items
  AttnTile* tiles = nullptr;     // tensor-core attention tiles of the call
  int64_t tile_cap = 0;
  int* err = nullptr;
  // pinned host staging
  int32_t* h_tok_off = nullptr;
  int32_t* h_sorted_slot = nullptr;
  int* h_err = nullptr;
  AttnItem* h_items = nullptr;
  AttnTile* h_tiles = nullptr;
  int64_t h_pair_cap = 0, h_item_cap = 0;
  // key token selection (dopr_select_prefix_inputs), grown on demand and kept
  Store* sel_empty = nullptr;  // a store of one empty document: a valid pool map for the attention kernels
  float* sel_A = nullptr;      // per-document attention matrices of the largest chunk (sum of n^2)
  int64_t* sel_a_off = nullptr;
  float* sel_u = nullptr;      // salience of every token
  int32_t* sel_pos = nullptr;  // [docs][top_k]
  bf16* sel_x = nullptr;       // [docs][top_k][H]
  int64_t sel_a_cap = 0, sel_doc_cap = 0, sel_tok_cap = 0, sel_pos_cap = 0, sel_x_cap = 0;
};

// Per-kernel-family launch counters and (when enabled) CUDA-event timing.
enum KernelKind : int {
  K_PACK = 0, K_EMBED_NORM, K_GEMM_QKV, K_QKNORM_ROPE, K_ATTENTION, K_GEMM_O, K_RMSNORM, K_GEMM_GATE_UP,
  K_GEMM_DOWN, K_SCORE, K_PREFIX_STORE, K_COUNT
};
struct Profiler {
  bool on = false;
  int64_t launches[K_COUNT] = {};
  double ms[K_COUNT] = {}, flops[K_COUNT] = {}, bytes[K_COUNT] = {};
  std::vector<cudaEvent_t> events;  // pairs (start, end), reused across calls
  std::vector<int> pending;         // kind of each recorded pair
  void reset() {
    for (int k = 0; k < K_COUNT; ++k) launches[k] = 0, ms[k] = flops[k] = bytes[k] = 0;
    pending.clear();
  }
};

struct Model {
  dopr_model_config cfg{};
  Profiler prof;
  int device = 0;
  int num_sms = 0;
  int qkv_dim = 0;  // (Hq + 2 Hkv) * 128
  int o_dim = 0;    // Hq * 128
  bf16* embed = nullptr;       // [V][H]
  bf16* attn_norm = nullptr;   // [L][H]
  f16* w_qkv = nullptr;        // [L][qkv_dim][H]   (projection matrices held as fp16)
  bf16* q_norm = nullptr;      // [L][128]
  bf16* k_norm = nullptr;      // [L][128]
  f16* w_o = nullptr;          // [L][H][o_dim]
  bf16* mlp_norm = nullptr;    // [L][H]
  f16* w_gu = nullptr;         // [L][2F][H], gate/up interleaved in 128-row blocks
  f16* w_down = nullptr;       // [L][H][F]
  bf16* final_norm = nullptr;  // [H]
  bf16* score_head = nullptr;  // [2][H]
  // optional MLP scoring head (replaces the yes/no rows when mlp_width > 0)
  int mlp_width = 0, mlp_act = 0;
  bf16* mlp_w1 = nullptr;  // [width][H]
  bf16* mlp_b1 = nullptr;  // [width]
  bf16* mlp_w2 = nullptr;  // [width]
  float mlp_b2 = 0.f;
  float2* rope = nullptr;      // [max_position][64] (cos, sin)
  std::vector<uint8_t> have;   // [kind * L + layer]
  std::vector<CUtensorMap> tm_qkv, tm_o, tm_gu, tm_down;
  bool maps_ok = false;
  Workspace ws;
};

// ------------------------------------------------------------ launchers
// Tensor map helper (driver entry point resolved at run time).
// 2-D map over 16-bit elements (fp16 when `half` is set, else bf16).
bool make_tmap_16b_2d(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint64_t row_stride_bytes,
                      uint32_t box_cols, uint32_t box_rows, bool swizzle128, bool half);
bool make_tmap_q_heads(CUtensorMap* map, const void* base, uint64_t cols, uint64_t rows, uint32_t box_rows,
                       uint32_t box_heads);

// GEMM epilogues.
enum GemmEpi : int { EPI_STORE = 0, EPI_RESID_ADD = 1, EPI_SWIGLU = 2, EPI_QKV = 3 };
constexpr int GEMM_BM = 128, GEMM_BN = 256, GEMM_BK = 64;
// Rows of a B (weight) tensor-map box: each CTA of a pair stages 128 of a tile's 256 B rows.
constexpr int GEMM_B_BOX = 128;
constexpr int GEMM_SS_PER_TILE = 2;  // partial sums of squares a residual epilogue writes per row and n-tile
struct GemmParams {
  int M, N, K;
  void* out;          // fp16 [M][ld_out] (store, QKV, SwiGLU: ld_out = N/2) or fp32 residual [M][ld_out]
  int64_t ld_out;
  // Fused RMSNorm.  rs(ss, parts) = rsqrt(sum_i ss[row*parts + i] / norm_dim + eps); a null
  // array means 1.  Producer (residual epilogue): xn_out = f16(r' * xn_gain * rs(ss_pre)) and
  // ss_out[row*ss_out_parts + n-tile] = partial sum of r'^2.  Consumer: accumulator rows are
  // scaled by rs(ss_in) / rs(ss_pre), so the operand stays near unit scale in fp16.
  const float* ss_in;
  int ss_parts;
  const float* ss_pre;
  int ss_pre_parts;
  int norm_dim;
  float eps;
  f16* xn_out;
  const bf16* xn_gain;
  float* ss_out;
  int ss_out_parts;
  // QKV epilogue: per-head RMSNorm gains and RoPE at tok_pos[row]
  const int32_t* tok_pos;
  const float2* rope;
  const bf16* q_norm;
  const bf16* k_norm;
  int q_cols, k_cols;
  int* err;
  uint64_t timeout_ns;
};
cudaError_t gemm_setup();
// C[M][N] = A[M][K] * B[N][K]^T followed by the epilogue `epi`.
cudaError_t launch_gemm(int epi, const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmParams& p, int num_sms,
                        cudaStream_t st);

// Row kernels.
// r[t] = E[tok_id[t]] (fp32), ss[t] = sum(r[t]^2), xn[t] = f16(r[t] * rsqrt(ss[t]/H + eps) * gain):
// the embedding and the first RMSNorm.
cudaError_t launch_embed(const int32_t* tok_id, int T, const bf16* embed, const bf16* gain, int H, float eps, float* r,
                         f16* xn, float* ss, const Extents& ext, cudaStream_t st);
// In place: n bf16 values -> fp16; *range |= 1 (device int) when a value is not finite
// or above 65504 in magnitude.
cudaError_t launch_bf16_to_f16(void* buf, int64_t n, int* range, cudaStream_t st);
// Score head over sorted pairs [p_begin, p_end): the score-token row of pair s is
// r[tok_off[s+1]-1-tok0], or r[s - p_begin] when `compact` is set.
cudaError_t launch_score(const float* r, int H, const int32_t* tok_off, int tok0, int p_begin, int p_end, int compact,
                         const int32_t* perm, const bf16* gain, const bf16* head, float eps, float* scores,
                         const Extents& ext, cudaStream_t st);
// Compact the score-token rows of sorted pairs [p_begin, p_end): dst_r[i] = r[row(i)] (H floats) and
// dst_ss[i] = ss[row(i)] (parts floats), row(i) = tok_off[p_begin+i+1]-1-tok0.
cudaError_t launch_score_mlp(const float* r, int H, const int32_t* tok_off, int tok0, int p_begin, int p_end,
                             int compact, const int32_t* perm, const bf16* gain, float eps, int width, int act,
                             const bf16* w1, const bf16* b1, const bf16* w2, float b2, float* scores,
                             const Extents& ext, cudaStream_t st);
cudaError_t launch_gather_score_rows(const float* r, const float* ss, int H, int parts, const int32_t* tok_off,
                                     int tok0, int p_begin, int p_end, float* dst_r, float* dst_ss, const Extents& ext,
                                     cudaStream_t st);
// [m][Hkv][128] bf16 -> [Hkv][m][128] fp16 for K and V; *range |= 1 when a value
// is not finite or exceeds the fp16 range (|x| > 65504).
cudaError_t launch_store_transpose(const bf16* k, const bf16* v, int m, int Hkv, f16* dk, f16* dv, int* range,
                                   cudaStream_t st);

// Attention.
struct AttnArgs {
  const AttnItem* items;
  int n_items;
  const int32_t* tok_off;  // sorted pair -> first packed token
  int32_t tok0;            // first packed token of this chunk
  const f16* qkv;
  int ld_qkv;
  f16* out;
  int ld_out;
  const int64_t* slot_row;
  int layer, n_layers, Hq, Hkv;
  int mpad_cap;  // prefix rows reserved in shared memory (multiple of 64)
  int score_only;  // 1: only each pair's score-token rows, written to out row (pair - pair_base)
  int pair_base;
  int* err;
  Extents ext;
};
cudaError_t attn_setup();
cudaError_t launch_attention(const CUtensorMap& tm_pool, const AttnArgs& a, cudaStream_t st);

// Arguments of the tensor-core attention kernel.
struct AttnTcArgs {
  const AttnTile* tiles;
  int n_units;  // tiles x kv heads
  f16* out;
  int ld_out;
  int layer, Hq, Hkv;
  int* err;
  Extents ext;
};
// Q rows per head in a 128-row tile; 0 when the group size does not divide 128 into boxes of >= 8 rows.
inline int attn_tc_rows_per_head(int G) { return (G >= 1 && G <= 16 && 128 % G == 0) ? 128 / G : 0; }
cudaError_t attn_tc_setup();
// tm_q: the Q heads of the chunk's packed QKV buffer as a 3-D map (make_tmap_q_heads), box 64
// columns x (128 / G) rows x G heads; tm_kv, tm_kv32, tm_kv64: the same buffer, boxes 64 x 16,
// 64 x 32 and 64 x 64; tm_pool: the store pool, box 64 x 64 (all fp16, 128-byte swizzle).
cudaError_t launch_attention_tc(const CUtensorMap& tm_q, const CUtensorMap& tm_kv, const CUtensorMap& tm_kv32,
                                const CUtensorMap& tm_kv64, const CUtensorMap& tm_pool, const AttnTcArgs& a,
                                int num_sms, cudaStream_t st);
// Tiles with more than ATTN_TC_MAX_KEYS key columns (same maps and arguments).
cudaError_t launch_attention_tc_long(const CUtensorMap& tm_q, const CUtensorMap& tm_kv, const CUtensorMap& tm_kv32,
                                     const CUtensorMap& tm_kv64, const CUtensorMap& tm_pool, const AttnTcArgs& a,
                                     int num_sms, cudaStream_t st);

// Packer.
struct PackArgs {
  int n_pairs;
  const int32_t* q_off;
  const int32_t* q_tok;
  const int64_t* doc_ids;
  int64_t max_doc_id;
  const int32_t* slot_of;
  const int32_t* slot_m;
  const uint8_t* slot_ok;
  int vocab, score_token, max_position;
  int32_t* doc_count;  // [max_doc_id+1], zeroed by the launcher
  int32_t* pair_slot;
  int32_t* perm;
  int32_t* sorted_slot;
  int32_t* tok_off;
  int32_t* tok_id;
  int32_t* tok_pos;
  int32_t* tok_pair;
  int* err;
};
// Device packer, first part: validation, stable sort by doc id, packed token
// offsets (tok_off).  Zeroes doc_count itself.
cudaError_t launch_pack_order(const PackArgs& a, cudaStream_t st);
// Second part, once the token buffers are sized: token ids, positions, pair index.
cudaError_t launch_pack_tokens(const PackArgs& a, cudaStream_t st);

// Sets the message dopr_last_error() returns on this thread.
void set_last_error_message(const std::string& msg);

// Debug kernel: bounded wait on a barrier nothing completes.
// Key token selection (k_select.cu), per chunk of whole documents (pairs p0 ..
// p0 + n_docs - 1, chunk rows 0 .. n_rows - 1).
constexpr int SEL_MAX_N = 2048;  // longest document the selection takes
struct SelectArgs {
  const f16* qkv;  // the chunk's q | k | v rows after the last layer's projection
  int ld_qkv, Hq, Hkv;
  const int32_t* tok_pair;  // packed token -> document (pair) index
  const int32_t* tok_off;   // document -> first packed token
  int t0, p0, n_docs, n_rows;
  const int64_t* a_off;     // chunk document -> offset of its n x n A-bar in A
  float* A;
  int top_p, top_k;
  float* u;                 // salience of chunk row t at u[t]
  int32_t* positions;       // [all documents][top_k]
  bf16* x;                  // [all documents][top_k][hidden]
  Extents ext;
};
cudaError_t select_setup();
cudaError_t launch_select(const SelectArgs& a, cudaStream_t st);
cudaError_t launch_select_gather(const SelectArgs& a, const float* r, int H, const bf16* gain, float eps,
                                 cudaStream_t st);
// Prefix build: K/V rows of chunk tokens [0, T) (packed tokens t0 + t) into the store pool.
cudaError_t launch_prefix_store(const f16* qkv, int ld_qkv, int T, int t0, int Hq, int Hkv, const int32_t* tok_pair,
                                const int32_t* tok_pos, const int32_t* pair_slot, const int64_t* slot_row,
                                const int32_t* slot_m, int layer, f16* pool, const Extents& ext, cudaStream_t st);
cudaError_t launch_wait_timeout_probe(int* err, uint64_t timeout_ns, cudaStream_t st);

}  // namespace dopr
