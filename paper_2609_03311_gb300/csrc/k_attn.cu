// k_attn.cu -- prefix-plus-causal grouped-query attention of the online pass
// (DoPR Sec. 3.4: the online tokens [q ; t_score] attend to the document's
// stored prefix keys/values, then causally to their own keys).
//
// One CTA per (work item, kv head).  A work item is a run of consecutive
// sorted pairs that share one document, so the CTA stages that document's
// prefix K and V for its kv head (m x 128 each) into shared memory ONCE with
// TMA (128-byte swizzle) and reuses it for every query row of every pair in
// the run.  Rows are (token j, q head of the group) with the G q heads of one
// kv head interleaved, so a 16-row warp tile covers 16/G tokens x G heads.
//
// Pairs are packed contiguously, so the own keys/values of a batch of
// consecutive pairs are one block of rows: the CTA loads them once (cp.async)
// for as many pairs as fit OWN_CAP rows, then the batch's 16-row tiles are
// dealt round-robin to the warps with no further barriers.  A warp reads its
// Q tile straight from global memory into mma fragments, sweeps the prefix in
// 32-key blocks, then its own causal keys in 16-key blocks, with the online
// (running max / running sum) softmax.  Pairs longer
// than OWN_CAP stream their own keys in OWN_CAP chunks per 64-row group.
// Scores and P.V use warp-level fp16 mma with fp32 accumulation (the store
// keeps the prefix as fp16); row maxima and sums use quad shuffles.  This
// kernel takes the score-token rows of the last layer (one row per pair and
// q head), and every row when the GQA group size gives the tensor-core
// kernels no tile shape.
#include <math.h>

#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int WARPS = 4;
constexpr int THREADS = WARPS * 32;
constexpr int ROW_BYTES = HEAD_DIM * 2;
constexpr int BOX_BYTES = 64 * 128;          // TMA box: 64 rows x 64 elements
constexpr int OWN_CAP = 64;                  // own key rows resident at once
constexpr int OWN_ROWS = OWN_CAP + 16;       // + zeroed tail read by the last 16-key block
constexpr int OWN_BYTES = OWN_ROWS * ROW_BYTES;
constexpr int MAX_BATCH = 32;                // pairs per resident batch
#ifndef DOPR_ATTN_MIN_BLOCKS
#define DOPR_ATTN_MIN_BLOCKS 2                 // resident CTAs per SM the register budget targets
#endif

// Prefix tile: byte offset of (row r, 16-byte chunk c) in 64-row boxes, each
// split into two 64-element halves, 128-byte swizzled (what TMA writes).
__device__ __forceinline__ uint32_t off_pre(int r, int c) {
  return static_cast<uint32_t>((((r >> 6) * 2 + (c >> 3)) * 64 + (r & 63)) * 128 + (((c & 7) ^ (r & 7)) << 4));
}
// Own-key tile: 256-byte rows, 16-byte chunks XOR-swizzled by the row (conflict-free ldmatrix).
__device__ __forceinline__ uint32_t off_own(int r, int c) {
  return static_cast<uint32_t>(r * ROW_BYTES + ((c ^ (r & 7)) << 4));
}

struct TileState {
  float o[16][4];
  float mrow[2], lrow[2];
};

// One block of NT*8 keys for one warp's 16 rows.  Keys kk >= n_valid are
// masked; with CAUSAL key kk is visible to a row of token j only if key0 + kk <= j.
template <int NT, bool CAUSAL, bool PREFIX>
__device__ __forceinline__ void attend(uint32_t kt, uint32_t vt, int kbase, int lane, const uint32_t (&qf)[8][4],
                                       TileState& st, int n_valid, int key0, const int (&jr)[2], float scale_log2) {
  auto off = [](int r, int c) { return PREFIX ? off_pre(r, c) : off_own(r, c); };
  float s[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
    for (int np = 0; np < NT / 2; ++np) {
      const int key = kbase + np * 16 + (lane & 7) + ((lane >> 4) << 3);
      const int c = 2 * ks + ((lane >> 3) & 1);
      uint32_t b0, b1, b2, b3;
      ldmatrix_x4(kt + off(key, c), b0, b1, b2, b3);
      mma_f16_16816(s[2 * np], qf[ks], b0, b1);
      mma_f16_16816(s[2 * np + 1], qf[ks], b2, b3);
    }
  }
  float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int kk = nt * 8 + (lane & 3) * 2 + (e & 1);
      bool ok = kk < n_valid;
      if (CAUSAL) ok = ok && (key0 + kk <= jr[e >> 1]);
      const float v = ok ? s[nt][e] * scale_log2 : -INFINITY;
      s[nt][e] = v;
      mx[e >> 1] = fmaxf(mx[e >> 1], v);
    }
  float alpha[2], base[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 1));
    mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 2));
    const float mnew = fmaxf(st.mrow[i], mx[i]);
    base[i] = (mnew == -INFINITY) ? 0.f : mnew;
    alpha[i] = exp2f(st.mrow[i] - base[i]);
    st.mrow[i] = mnew;
  }
  float rs[2] = {0.f, 0.f};
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float p = exp2f(s[nt][e] - base[e >> 1]);
      s[nt][e] = p;
      rs[e >> 1] += p;
    }
  st.lrow[0] = st.lrow[0] * alpha[0] + rs[0];
  st.lrow[1] = st.lrow[1] * alpha[1] + rs[1];
#pragma unroll
  for (int dt = 0; dt < 16; ++dt) {
    st.o[dt][0] *= alpha[0];
    st.o[dt][1] *= alpha[0];
    st.o[dt][2] *= alpha[1];
    st.o[dt][3] *= alpha[1];
  }
#pragma unroll
  for (int kk = 0; kk < NT / 2; ++kk) {
    uint32_t pa[4];
    pa[0] = pack_f16x2(s[2 * kk][0], s[2 * kk][1]);
    pa[1] = pack_f16x2(s[2 * kk][2], s[2 * kk][3]);
    pa[2] = pack_f16x2(s[2 * kk + 1][0], s[2 * kk + 1][1]);
    pa[3] = pack_f16x2(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
    for (int dp = 0; dp < 8; ++dp) {
      const int key = kbase + kk * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
      const int c = 2 * dp + (lane >> 4);
      uint32_t b0, b1, b2, b3;
      ldmatrix_x4_trans(vt + off(key, c), b0, b1, b2, b3);
      mma_f16_16816(st.o[2 * dp], pa, b0, b1);
      mma_f16_16816(st.o[2 * dp + 1], pa, b2, b3);
    }
  }
}

struct PairGeom {
  int tb;  // first row of the pair in this chunk
  int T;   // tokens (query + score token)
  int R;   // rows = T * G
};

// Q fragments of rows row0..row0+15 straight from global memory (rows >= R read as 0).
__device__ __forceinline__ void load_q(const AttnArgs& a, const PairGeom& pg, int g, int G, int row0, int lane,
                                       uint32_t (&qf)[8][4]) {
  const int ra = row0 + (lane >> 2), rb = ra + 8;
  const uint32_t* qa = nullptr;
  const uint32_t* qb = nullptr;
  if (ra < pg.R && index_ok(a.ext.err, pg.tb + ra / G, a.ext.rows))
    qa = reinterpret_cast<const uint32_t*>(a.qkv + static_cast<int64_t>(pg.tb + ra / G) * a.ld_qkv +
                                           (g * G + ra % G) * HEAD_DIM);
  if (rb < pg.R && index_ok(a.ext.err, pg.tb + rb / G, a.ext.rows))
    qb = reinterpret_cast<const uint32_t*>(a.qkv + static_cast<int64_t>(pg.tb + rb / G) * a.ld_qkv +
                                           (g * G + rb % G) * HEAD_DIM);
  const int t = lane & 3;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int w = ks * 8 + t;  // 32-bit word index of columns 16ks + 2t
    qf[ks][0] = qa ? __ldg(qa + w) : 0u;
    qf[ks][1] = qb ? __ldg(qb + w) : 0u;
    qf[ks][2] = qa ? __ldg(qa + w + 4) : 0u;
    qf[ks][3] = qb ? __ldg(qb + w + 4) : 0u;
  }
}

__device__ __forceinline__ void init_state(TileState& st) {
#pragma unroll
  for (int dt = 0; dt < 16; ++dt) st.o[dt][0] = st.o[dt][1] = st.o[dt][2] = st.o[dt][3] = 0.f;
  st.mrow[0] = st.mrow[1] = -INFINITY;
  st.lrow[0] = st.lrow[1] = 0.f;
}

// Normalise and store the tile's rows < R (compact row per pair in score-only mode).
__device__ __forceinline__ void store_tile(const AttnArgs& a, const PairGeom& pg, int s, int g, int G, int row0,
                                           int lane, TileState& st) {
  float l0 = st.lrow[0], l1 = st.lrow[1];
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f, inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
  for (int hr = 0; hr < 2; ++hr) {
    const int row = row0 + (lane >> 2) + hr * 8;
    const int orow = a.score_only ? s - a.pair_base : pg.tb + row / G;
    if (row < pg.R && index_ok(a.ext.err, orow, a.ext.rows)) {
      const int hh = row % G;
      f16* dst = a.out + static_cast<int64_t>(orow) * a.ld_out + (g * G + hh) * HEAD_DIM + (lane & 3) * 2;
      const float inv = hr ? inv1 : inv0;
      bool bad = false;
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) {
        const float y0 = st.o[dt][2 * hr] * inv, y1 = st.o[dt][2 * hr + 1] * inv;
        bad |= !(fp16_ok(y0) && fp16_ok(y1));
        *reinterpret_cast<uint32_t*>(dst + dt * 8) = pack_f16x2(y0, y1);
      }
      if (bad && a.err) atomicOr(a.err, DEV_ERR_RANGE);
    }
  }
}

// Own keys/values of chunk rows [row_begin, row_begin + count) into own-buffer
// rows 0..count-1; rows count .. count+15 are zeroed.  All threads take part.
__device__ __forceinline__ void load_own(const AttnArgs& a, int g, uint32_t sOK, uint32_t sOV, int row_begin,
                                         int count, int tid) {
  const int kcol = (a.Hq + g) * HEAD_DIM;
  const int vcol = (a.Hq + a.Hkv + g) * HEAD_DIM;
  const int rows = min(OWN_ROWS, count + 16);
  for (int idx = tid; idx < rows * 32; idx += THREADS) {
    const int kv = idx & 1, rc = idx >> 1, r = rc >> 4, c = rc & 15;
    const bool ok = r < count && index_ok(a.ext.err, row_begin + r, a.ext.rows);
    const f16* src = a.qkv + static_cast<int64_t>(row_begin + (ok ? r : 0)) * a.ld_qkv + (kv ? vcol : kcol) + c * 8;
    cp_async16((kv ? sOV : sOK) + off_own(r, c), src, ok);
  }
  cp_async_commit();
  cp_async_wait_all();
}

__global__ void __launch_bounds__(THREADS, DOPR_ATTN_MIN_BLOCKS) k_attn(const __grid_constant__ CUtensorMap tm_pool, AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sPK = smem_u32(smem);
  const uint32_t sPV = sPK + a.mpad_cap * ROW_BYTES;
  const uint32_t sOK = sPV + a.mpad_cap * ROW_BYTES;
  const uint32_t sOV = sOK + OWN_BYTES;
  const uint32_t bar = sOV + OWN_BYTES;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const AttnItem item = a.items[blockIdx.x];
  const int g = blockIdx.y;
  const int G = a.Hq / a.Hkv;
  const int m = item.m;
  const int nbox = (m + 63) >> 6;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HEAD_DIM));

  // ---- stage the prefix K/V of (doc, layer, kv head g) once
  if (tid == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (m > 0) {
    if (tid == 0) {
      const int64_t base = a.slot_row[item.slot];
      const int rowK = static_cast<int>(base + (static_cast<int64_t>(a.layer) * 2 * a.Hkv + g) * m);
      const int rowV = static_cast<int>(base + ((static_cast<int64_t>(a.layer) * 2 + 1) * a.Hkv + g) * m);
      if (kCheckedBuild) {  // report only: the tensor map bounds the copies itself
        index_ok(a.ext.err, rowK + m - 1, a.ext.pool_rows);
        index_ok(a.ext.err, rowV + m - 1, a.ext.pool_rows);
      }
      mbar_arrive_expect_tx(bar, static_cast<uint32_t>(nbox) * 4u * BOX_BYTES);
      for (int b = 0; b < nbox; ++b)
        for (int h = 0; h < 2; ++h) {
          tma_load_2d(sPK + (b * 2 + h) * BOX_BYTES, &tm_pool, bar, h * 64, rowK + b * 64);
          tma_load_2d(sPV + (b * 2 + h) * BOX_BYTES, &tm_pool, bar, h * 64, rowV + b * 64);
        }
    }
    const bool landed = mbar_wait(bar, 0, a.err, WAIT_TIMEOUT_NS);
    if (!__syncthreads_and(landed)) {  // uniform decision: every thread leaves together
      if (tid == 0) mbar_wait(bar, 0, a.err, 100000000ull);  // let the copies land first
      return;
    }
    // Rows m .. nbox*64-1 of the boxes hold other data: zero them so masked keys
    // contribute exactly 0 to P.V.
    uint8_t* gk = smem;
    uint8_t* gv = smem + a.mpad_cap * ROW_BYTES;
    for (int i = m * 16 + tid; i < nbox * 64 * 16; i += THREADS) {
      const int r = i / 16, c = i % 16;
      *reinterpret_cast<uint4*>(gk + off_pre(r, c)) = make_uint4(0, 0, 0, 0);
      *reinterpret_cast<uint4*>(gv + off_pre(r, c)) = make_uint4(0, 0, 0, 0);
    }
    // (the barrier before the first own-key load orders these writes)
  }

  auto geom = [&](int s) {
    PairGeom pg;
    pg.tb = a.tok_off[s] - a.tok0;
    pg.T = a.tok_off[s + 1] - a.tok_off[s];
    pg.R = pg.T * G;
    return pg;
  };
  auto prefix_pass = [&](const uint32_t (&qf)[8][4], TileState& st, const int (&jr)[2]) {
    for (int k0 = 0; k0 < m; k0 += 32)
      attend<4, false, true>(sPK, sPV, k0, lane, qf, st, min(32, m - k0), 0, jr, scale_log2);
  };

  int s = item.pair_begin;
  while (s < item.pair_end) {
    const PairGeom p0 = geom(s);
    if (p0.T <= OWN_CAP) {
      // ---- resident batch: pairs [s, e) whose own rows fit OWN_CAP together
      int e = s + 1, rows = p0.T;
      while (e < item.pair_end && e - s < MAX_BATCH) {
        const int t = a.tok_off[e + 1] - a.tok_off[e];
        if (rows + t > OWN_CAP) break;
        rows += t;
        ++e;
      }
      __syncthreads();  // previous users of the own buffer are done
      load_own(a, g, sOK, sOV, p0.tb, rows, tid);
      __syncthreads();
      int tile = 0;
      for (int sp = s; sp < e; ++sp) {
        const PairGeom pg = geom(sp);
        const int rbeg = a.score_only ? (pg.T - 1) * G : 0;
        const int own_base = pg.tb - p0.tb;
        for (int row0 = rbeg; row0 < pg.R; row0 += 16, ++tile) {
          if ((tile % WARPS) != warp) continue;
          uint32_t qf[8][4];
          load_q(a, pg, g, G, row0, lane, qf);
          TileState st;
          init_state(st);
          const int jr[2] = {(row0 + (lane >> 2)) / G, (row0 + (lane >> 2) + 8) / G};
          prefix_pass(qf, st, jr);
          const int jmax = min(pg.T - 1, (row0 + 15) / G);
          for (int k0 = 0; k0 <= jmax; k0 += 16)
            attend<2, true, false>(sOK, sOV, own_base + k0, lane, qf, st, 16, k0, jr, scale_log2);
          store_tile(a, pg, sp, g, G, row0, lane, st);
        }
      }
      s = e;
    } else {
      // ---- long pair: 64-row groups, own keys streamed in OWN_CAP chunks
      const PairGeom pg = p0;
      const int rbeg = a.score_only ? (pg.T - 1) * G : 0;
      for (int rg = rbeg; rg < pg.R; rg += WARPS * 16) {
        const int row0 = rg + warp * 16;
        const bool active = row0 < pg.R;
        uint32_t qf[8][4];
        TileState st;
        init_state(st);
        const int jr[2] = {(row0 + (lane >> 2)) / G, (row0 + (lane >> 2) + 8) / G};
        if (active) {
          load_q(a, pg, g, G, row0, lane, qf);
          prefix_pass(qf, st, jr);
        }
        const int jmax_g = min(pg.T - 1, (rg + WARPS * 16 - 1) / G);
        const int jmax = min(pg.T - 1, (row0 + 15) / G);
        for (int c0 = 0; c0 <= jmax_g; c0 += OWN_CAP) {
          __syncthreads();
          load_own(a, g, sOK, sOV, pg.tb + c0, min(OWN_CAP, jmax_g + 1 - c0), tid);
          __syncthreads();
          if (active)
            for (int k0 = c0; k0 <= min(jmax, c0 + OWN_CAP - 1); k0 += 16)
              attend<2, true, false>(sOK, sOV, k0 - c0, lane, qf, st, 16, k0, jr, scale_log2);
        }
        if (active) store_tile(a, pg, s, g, G, row0, lane, st);
      }
      ++s;
    }
  }
}

inline size_t attn_smem_bytes(int mpad_cap) {
  return 1024 + 2 * static_cast<size_t>(mpad_cap) * ROW_BYTES + 2 * OWN_BYTES + 64;
}

}  // namespace

cudaError_t attn_setup() {
  return cudaFuncSetAttribute(k_attn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(attn_smem_bytes(MAX_PREFIX)));
}

cudaError_t launch_attention(const CUtensorMap& tm_pool, const AttnArgs& a, cudaStream_t st) {
  if (a.n_items <= 0) return cudaSuccess;
  dim3 grid(a.n_items, a.Hkv);
  k_attn<<<grid, THREADS, attn_smem_bytes(a.mpad_cap), st>>>(tm_pool, a);
  return cudaGetLastError();
}

}  // namespace dopr
