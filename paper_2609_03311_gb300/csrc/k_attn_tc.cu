// k_attn_tc.cu -- prefix-plus-causal grouped-query attention of the online pass
// on the 5th-generation tensor cores (DoPR Sec. 3.4: the online tokens
// [q ; t_score] attend to the document's stored prefix keys/values, then
// causally to their own keys).
//
// Work unit = (tile, kv head g).  A tile holds up to TT = 128 / G consecutive
// packed tokens of pairs that share one document; its 128 rows are the G q
// heads of group g of those tokens, head-major (row = hh * TT + token), so each
// q head's rows arrive as one TMA box of the packed QKV buffer.  Its key
// columns are the document's prefix (columns [0, ceil64(m))) followed, for each
// pair the tile touches, by that pair's own keys from its first token up to the
// tile's last token, each pair's segment starting on a 16-column boundary: a row
// then meets its keys at the same positions of the same 16-key MMA steps
// whatever other pairs share its tile.  The host keeps every tile within 256
// key columns.
//
// Persistent CTAs, one per SM, warp-specialised:
//   warp 0    TMA producer: the Q tile (two stages), then the tile's key blocks
//             of 64 columns into a K ring and a V ring (four stages each) --
//             prefix blocks from the store pool in 64-row boxes, own-key
//             segments from the packed QKV buffer in 16-row boxes;
//   warp 1    MMA issuer: S = Q K^T for every key block into TMEM (fp32, up to
//             256 columns), then O = P V block by block, V read as an MN-major
//             operand, into a separate 128-column TMEM accumulator;
//   warps 2-5 softmax and epilogue, one thread per tile row (its TMEM lane): an
//             exact two-pass softmax over the row's S (the maximum over the
//             visible keys, then exp2 and the sum in key order), P written as
//             fp16 into a two-stage ring in the UMMA K-major layout, and after
//             the last P V step O / sum as fp16.
// The exact maximum, the in-order sum and the aligned own segments make every
// row's result independent of how the batch was cut into tiles.
// Every wait is bounded; a CTA that gives up lets its copies and MMAs land and
// frees its TMEM before it exits.
#include <limits.h>
#include <math.h>

#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int TILE_M = 128;
constexpr int KBLK = 64;  // key columns per block
constexpr int GROUP_ROWS = 16;
constexpr int Q_STAGES = 2, KV_STAGES = 4, P_STAGES = 2;
constexpr int Q_HALF = TILE_M * 128;    // 128 rows x 64 16-bit elements
constexpr int Q_BYTES = 2 * Q_HALF;     // 32 KB
constexpr int KV_HALF = KBLK * 128;     // 64 rows x 64 elements
constexpr int KV_BYTES = 2 * KV_HALF;   // 16 KB
constexpr int P_BYTES = TILE_M * 128;   // 128 rows x 64 keys
constexpr int GROUP_BYTES = 2 * GROUP_ROWS * 128;
constexpr int THREADS = 192;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t S_COL = 0, O_COL = 256;

constexpr int OFF_Q = 0;
constexpr int OFF_K = OFF_Q + Q_STAGES * Q_BYTES;
constexpr int OFF_V = OFF_K + KV_STAGES * KV_BYTES;
constexpr int OFF_P = OFF_V + KV_STAGES * KV_BYTES;
constexpr int OFF_BAR = OFF_P + P_STAGES * P_BYTES;
// q_full/empty, k_full/empty, v_full/empty, p_full/empty, then s_full, s_free, o_full, o_free, drain
constexpr int BAR_Q_FULL = 0, BAR_Q_EMPTY = BAR_Q_FULL + Q_STAGES;
constexpr int BAR_K_FULL = BAR_Q_EMPTY + Q_STAGES, BAR_K_EMPTY = BAR_K_FULL + KV_STAGES;
constexpr int BAR_V_FULL = BAR_K_EMPTY + KV_STAGES, BAR_V_EMPTY = BAR_V_FULL + KV_STAGES;
constexpr int BAR_P_FULL = BAR_V_EMPTY + KV_STAGES, BAR_P_EMPTY = BAR_P_FULL + P_STAGES;
constexpr int BAR_S_FULL = BAR_P_EMPTY + P_STAGES, BAR_S_FREE = BAR_S_FULL + 1, BAR_O_FULL = BAR_S_FREE + 1,
              BAR_O_FREE = BAR_O_FULL + 1, BAR_DRAIN = BAR_O_FREE + 1, N_BARS = BAR_DRAIN + 1;
constexpr int SMEM_BYTES = 1024 + OFF_BAR + N_BARS * 8 + 16;
static_assert(SMEM_BYTES <= 227 * 1024, "shared memory budget");

constexpr uint32_t IDESC_S = umma_idesc_f16(TILE_M, KBLK);
constexpr uint32_t IDESC_O = umma_idesc_f16_bmn(TILE_M, HEAD_DIM);

struct Ring {
  int stage = 0;
  uint32_t phase = 0;
  __device__ __forceinline__ void next(int n) {
    if (++stage == n) {
      stage = 0;
      phase ^= 1u;
    }
  }
};

__device__ __forceinline__ int ceil16(int x) { return (x + 15) & ~15; }
__device__ __forceinline__ int ceil64(int x) { return (x + 63) & ~63; }

// Walks the own-key 16-row groups of a tile in key order: pair p's group k
// covers packed rows [ps + 16k, ps + 16k + 16) at key column key.
struct GroupCursor {
  const int32_t* tok_off;
  int tok0, tok_end;  // chunk-relative token range of the tile: [.., tok_end)
  int p, ps, nvis, k, key;
  __device__ __forceinline__ void start(const int32_t* to, int t0, int pair_first, int tend, int pre64) {
    tok_off = to;
    tok0 = t0;
    tok_end = tend;
    p = pair_first;
    key = pre64;
    k = 0;
    load_pair();
  }
  __device__ __forceinline__ void load_pair() {
    ps = tok_off[p] - tok0;
    nvis = min(tok_off[p + 1] - tok0, tok_end) - ps;
  }
  __device__ __forceinline__ void advance() {
    key += GROUP_ROWS;
    k += GROUP_ROWS;
    if (k >= nvis) {
      k = 0;
      ++p;
      if (tok_off[p] - tok0 < tok_end) load_pair();
    }
  }
};

// Bits [lo, hi) of a 32-bit word, the range clipped to [0, 32).
__device__ __forceinline__ uint32_t bits_in(int lo, int hi) {
  lo = max(lo, 0);
  hi = min(hi, 32);
  if (hi <= lo) return 0u;
  const uint32_t upto = hi >= 32 ? 0xffffffffu : ((1u << hi) - 1u);
  return upto & ~((1u << lo) - 1u);
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Maximum of the 32 values whose mask bit is set (-inf when none).
__device__ __forceinline__ float masked_max32(const uint32_t (&v)[32], uint32_t mask) {
  float t[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const float a = (mask >> (2 * i)) & 1u ? __uint_as_float(v[2 * i]) : -INFINITY;
    const float b = (mask >> (2 * i + 1)) & 1u ? __uint_as_float(v[2 * i + 1]) : -INFINITY;
    t[i] = fmaxf(a, b);
  }
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
    for (int i = 0; i < w; ++i) t[i] = fmaxf(t[2 * i], t[2 * i + 1]);
  return t[0];
}

// P for 32 columns: 2^(s * scale - mxs) where the mask bit is set, else 0, stored
// as fp16 into 16-byte chunks 4*half .. 4*half+3 of the row's 128-byte P line
// (128-byte swizzle).  Returns sum + the two 16-column partial sums, each a
// fixed pairwise tree, added in column order.
__device__ __forceinline__ float exp_chunk(const uint32_t (&v)[32], uint32_t mask, float scale_log2, float mxs,
                                           float sum, uint8_t* prow, int half, int r) {
  float p[32];
#pragma unroll
  for (int e = 0; e < 32; ++e) {
    const float x = ex2_approx(fmaf(__uint_as_float(v[e]), scale_log2, -mxs));
    p[e] = (mask >> e) & 1u ? x : 0.f;
  }
  uint32_t w[16];
#pragma unroll
  for (int e = 0; e < 16; ++e) w[e] = pack_f16x2(p[2 * e], p[2 * e + 1]);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int chunk = half * 4 + q;
    *reinterpret_cast<uint4*>(prow + ((chunk ^ (r & 7)) << 4)) =
        make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
  }
#pragma unroll
  for (int gidx = 0; gidx < 2; ++gidx) {
    float t[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) t[i] = p[16 * gidx + 2 * i] + p[16 * gidx + 2 * i + 1];
#pragma unroll
    for (int w2 = 4; w2 >= 1; w2 >>= 1)
#pragma unroll
      for (int i = 0; i < w2; ++i) t[i] = t[2 * i] + t[2 * i + 1];
    sum += t[0];
  }
  return sum;
}

__device__ __forceinline__ void zero_chunk(uint8_t* prow, int half, int r) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int chunk = half * 4 + q;
    *reinterpret_cast<uint4*>(prow + ((chunk ^ (r & 7)) << 4)) = make_uint4(0, 0, 0, 0);
  }
}

__global__ void __launch_bounds__(THREADS, 1)
    k_attn_tc(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kv,
              const __grid_constant__ CUtensorMap tm_pool, AttnTcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t s0 = smem_u32(smem);
  const uint32_t sQ = s0 + OFF_Q, sK = s0 + OFF_K, sV = s0 + OFF_V, sP = s0 + OFF_P;
  auto bar = [&](int i) { return s0 + OFF_BAR + 8u * static_cast<uint32_t>(i); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_BAR + N_BARS * 8);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.Hq / a.Hkv;
  const int TT = TILE_M / G;

  if (threadIdx.x == 0) {
    for (int i = 0; i < Q_STAGES; ++i) {
      mbar_init(bar(BAR_Q_FULL + i), 1);
      mbar_init(bar(BAR_Q_EMPTY + i), 1);
    }
    for (int i = 0; i < KV_STAGES; ++i) {
      mbar_init(bar(BAR_K_FULL + i), 1);
      mbar_init(bar(BAR_K_EMPTY + i), 1);
      mbar_init(bar(BAR_V_FULL + i), 1);
      mbar_init(bar(BAR_V_EMPTY + i), 1);
    }
    for (int i = 0; i < P_STAGES; ++i) {
      mbar_init(bar(BAR_P_FULL + i), 4);
      mbar_init(bar(BAR_P_EMPTY + i), 1);
    }
    mbar_init(bar(BAR_S_FULL), 1);
    mbar_init(bar(BAR_S_FREE), 4);
    mbar_init(bar(BAR_O_FULL), 1);
    mbar_init(bar(BAR_O_FREE), 4);
    mbar_init(bar(BAR_DRAIN), 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_kv);
    tma_prefetch_desc(&tm_pool);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ======================= TMA producer
      Ring rq, rk, rv;
      uint32_t armed = 0, armed_par = 0;  // bit per barrier index (< 32): ever armed / parity of the last arm
      auto arm = [&](int b, uint32_t par, uint32_t bytes) {
        mbar_arrive_expect_tx(bar(b), bytes);
        armed |= 1u << b;
        armed_par = (armed_par & ~(1u << b)) | (par << b);
      };
      bool ok = true;
      for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x) {
        const AttnTile t = a.tiles[u / a.Hkv];
        const int g = u % a.Hkv;
        const int pre64 = ceil64(t.m);
        const int nb = (t.n_keys + KBLK - 1) / KBLK;
        // ---- Q: one box of TT rows per (q head of the group, 64-column half)
        if (!mbar_wait(bar(BAR_Q_EMPTY + rq.stage), rq.phase ^ 1u, a.err, WAIT_TIMEOUT_NS)) {
          ok = false;
          break;
        }
        arm(BAR_Q_FULL + rq.stage, rq.phase, Q_BYTES);
        for (int hh = 0; hh < G; ++hh)
          for (int h = 0; h < 2; ++h)
            tma_load_2d(sQ + rq.stage * Q_BYTES + h * Q_HALF + hh * TT * 128, &tm_q, bar(BAR_Q_FULL + rq.stage),
                        (g * G + hh) * HEAD_DIM + h * 64, t.tok_begin);
        rq.next(Q_STAGES);
        // ---- key blocks: K ring, then V ring
        const int64_t base = a.slot_row[t.slot];
        for (int kv = 0; kv < 2 && ok; ++kv) {
          Ring& r = kv ? rv : rk;
          const int full0 = kv ? BAR_V_FULL : BAR_K_FULL, empty0 = kv ? BAR_V_EMPTY : BAR_K_EMPTY;
          const uint32_t ring = kv ? sV : sK;
          const int pool_row = static_cast<int>(base + ((static_cast<int64_t>(a.layer) * 2 + kv) * a.Hkv + g) * t.m);
          const int col0 = (a.Hq + kv * a.Hkv + g) * HEAD_DIM;
          GroupCursor cur;
          cur.start(a.tok_off, a.tok0, t.pair_first, t.tok_begin + t.n_tok, pre64);
          for (int j = 0; j < nb; ++j) {
            if (!mbar_wait(bar(empty0 + r.stage), r.phase ^ 1u, a.err, WAIT_TIMEOUT_NS)) {
              ok = false;
              break;
            }
            const uint32_t dst = ring + r.stage * KV_BYTES;
            const uint32_t fb = bar(full0 + r.stage);
            if (j * KBLK < pre64) {
              arm(full0 + r.stage, r.phase, KV_BYTES);
              for (int h = 0; h < 2; ++h) tma_load_2d(dst + h * KV_HALF, &tm_pool, fb, h * 64, pool_row + j * KBLK);
            } else {
              const int groups = min(KBLK, t.n_keys - j * KBLK) / GROUP_ROWS;
              arm(full0 + r.stage, r.phase, groups * GROUP_BYTES);
              for (int q = 0; q < groups; ++q) {
                const int off = cur.key - j * KBLK;  // 0, 16, 32, 48 when the plan is consistent
                if (off >= 0 && off < KBLK)  // otherwise the copy is skipped and the wait below times out
                  for (int h = 0; h < 2; ++h)
                    tma_load_2d(dst + off * 128 + h * KV_HALF, &tm_kv, fb, col0 + h * 64, cur.ps + cur.k);
                cur.advance();
              }
            }
            r.next(KV_STAGES);
          }
        }
      }
      if (!ok) {  // every copy this thread started lands before the CTA can exit
        for (int b = 0; b < 32; ++b)
          if (armed & (1u << b)) mbar_wait(bar(b), (armed_par >> b) & 1u, a.err, 100000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ======================= MMA issuer
      Ring rq, rk, rv, rp;
      bool ok = true;
      int local = 0;
      for (int u = blockIdx.x; u < a.n_units && ok; u += gridDim.x, ++local) {
        const AttnTile t = a.tiles[u / a.Hkv];
        const int nb = (t.n_keys + KBLK - 1) / KBLK;
        const uint32_t tpar = static_cast<uint32_t>(local & 1);
        if (!mbar_wait(bar(BAR_Q_FULL + rq.stage), rq.phase, a.err, WAIT_TIMEOUT_NS) ||
            !mbar_wait(bar(BAR_S_FREE), tpar ^ 1u, a.err, WAIT_TIMEOUT_NS)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // S = Q K^T, one 64-column block per K stage
        const uint64_t qd = umma_desc_sw128(sQ + rq.stage * Q_BYTES);
        for (int j = 0; j < nb && ok; ++j) {
          if (!mbar_wait(bar(BAR_K_FULL + rk.stage), rk.phase, a.err, WAIT_TIMEOUT_NS)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t kd = umma_desc_sw128(sK + rk.stage * KV_BYTES);
#pragma unroll
          for (int ks = 0; ks < HEAD_DIM / 16; ++ks)  // 16 elements = 32 bytes of K per step, halves 16 KB / 8 KB apart
            umma_f16(tmem + S_COL + j * KBLK, qd + ((ks >> 2) * Q_HALF + (ks & 3) * 32) / 16,
                     kd + ((ks >> 2) * KV_HALF + (ks & 3) * 32) / 16, IDESC_S, ks > 0);
          umma_commit(bar(BAR_K_EMPTY + rk.stage));
          rk.next(KV_STAGES);
        }
        if (!ok) break;
        umma_commit(bar(BAR_S_FULL));
        umma_commit(bar(BAR_Q_EMPTY + rq.stage));
        rq.next(Q_STAGES);
        // O = P V, block by block as the softmax hands over P
        if (!mbar_wait(bar(BAR_O_FREE), tpar ^ 1u, a.err, WAIT_TIMEOUT_NS)) {
          ok = false;
          break;
        }
        for (int j = 0; j < nb && ok; ++j) {
          if (!mbar_wait(bar(BAR_P_FULL + rp.stage), rp.phase, a.err, WAIT_TIMEOUT_NS) ||
              !mbar_wait(bar(BAR_V_FULL + rv.stage), rv.phase, a.err, WAIT_TIMEOUT_NS)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int steps = min(KBLK, t.n_keys - j * KBLK) / 16;  // only rows the producer loaded
          const uint64_t pd = umma_desc_sw128(sP + rp.stage * P_BYTES);
          for (int kk = 0; kk < steps; ++kk)
            umma_f16(tmem + O_COL, pd + (kk * 32) / 16,
                     umma_desc_sw128_mn(sV + rv.stage * KV_BYTES + kk * 2048, KV_HALF, 1024), IDESC_O,
                     (j | kk) != 0);
          umma_commit(bar(BAR_P_EMPTY + rp.stage));
          umma_commit(bar(BAR_V_EMPTY + rv.stage));
          rp.next(P_STAGES);
          rv.next(KV_STAGES);
        }
        if (ok) umma_commit(bar(BAR_O_FULL));
      }
      // every MMA this thread issued is complete once the drain barrier flips
      umma_commit(bar(BAR_DRAIN));
      mbar_wait(bar(BAR_DRAIN), 0, a.err, ok ? WAIT_TIMEOUT_NS : 100000000ull);
    }
  } else {
    // ======================= softmax + epilogue: warps 2..5 -> TMEM lane quarters 2, 3, 0, 1
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;  // tile row
    const int hh = r / TT, jj = r % TT;
    const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HEAD_DIM));
    uint8_t* prow0 = smem + OFF_P + r * 128;
    Ring rp;
    int local = 0;
    for (int u = blockIdx.x; u < a.n_units; u += gridDim.x, ++local) {
      const AttnTile t = a.tiles[u / a.Hkv];
      const int g = u % a.Hkv;
      const int pre64 = ceil64(t.m);
      const int ncol = ((t.n_keys + KBLK - 1) / KBLK) * KBLK;
      const bool valid = jj < t.n_tok;
      const int tk = t.tok_begin + jj;  // this row's token (chunk-relative)
      // Visible keys: prefix columns [0, m) and own columns [olo, ohi].  Rows past
      // the tile's tokens see the prefix only; nothing of theirs is stored.
      int olo = INT_MAX, ohi = -1;
      if (valid) {
        int p = t.pair_first, seg = pre64;
        for (;;) {
          const int ps = a.tok_off[p] - a.tok0, pe = a.tok_off[p + 1] - a.tok0;
          if (tk < pe) {
            olo = seg;
            ohi = seg + (tk - ps);
            break;
          }
          seg += ceil16(min(pe, t.tok_begin + t.n_tok) - ps);
          ++p;
        }
      }
      const int wlo = __reduce_min_sync(0xffffffffu, olo);
      const int whi = __reduce_max_sync(0xffffffffu, ohi);
      auto chunk_live = [&](int c0) { return c0 < t.m || (c0 <= whi && c0 + 31 >= wlo); };
      auto vis_mask = [&](int c0) { return bits_in(-c0, t.m - c0) | bits_in(olo - c0, ohi + 1 - c0); };

      if (!mbar_wait(bar(BAR_S_FULL), static_cast<uint32_t>(local & 1), a.err, WAIT_TIMEOUT_NS)) break;
      tc_fence_after();
      // ---- pass 1: the row maximum over the visible keys (two 32-column loads per wait)
      float mx = -INFINITY;
      for (int c0 = 0; c0 < ncol; c0 += KBLK) {
        const bool l0 = chunk_live(c0), l1 = chunk_live(c0 + 32);
        if (!l0 && !l1) continue;
        uint32_t v0[32], v1[32];
        if (l0) tmem_ld32(trow + S_COL + c0, v0);
        if (l1) tmem_ld32(trow + S_COL + c0 + 32, v1);
        tmem_ld_wait();
        if (l0) mx = fmaxf(mx, masked_max32(v0, vis_mask(c0)));
        if (l1) mx = fmaxf(mx, masked_max32(v1, vis_mask(c0 + 32)));
      }
      const float mxs = (mx == -INFINITY) ? 0.f : mx * scale_log2;
      // ---- pass 2: P = 2^((s - max) * scale) per 64-key block; the sum adds
      // fixed-shape 16-key partial sums in key order
      float sum = 0.f;
      bool ok = true;
      for (int c0 = 0; c0 < ncol; c0 += KBLK) {
        if (!mbar_wait(bar(BAR_P_EMPTY + rp.stage), rp.phase ^ 1u, a.err, WAIT_TIMEOUT_NS)) {
          ok = false;
          break;
        }
        const bool l0 = chunk_live(c0), l1 = chunk_live(c0 + 32);
        uint32_t v0[32], v1[32];
        if (l0) tmem_ld32(trow + S_COL + c0, v0);
        if (l1) tmem_ld32(trow + S_COL + c0 + 32, v1);
        if (l0 || l1) tmem_ld_wait();
        uint8_t* prow = prow0 + rp.stage * P_BYTES;
        if (l0)
          sum = exp_chunk(v0, vis_mask(c0), scale_log2, mxs, sum, prow, 0, r);
        else
          zero_chunk(prow, 0, r);
        if (l1)
          sum = exp_chunk(v1, vis_mask(c0 + 32), scale_log2, mxs, sum, prow, 1, r);
        else
          zero_chunk(prow, 1, r);
        fence_proxy_async_smem();  // generic-proxy P writes -> visible to the tensor core
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(BAR_P_FULL + rp.stage));
        rp.next(P_STAGES);
      }
      if (!ok) break;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(BAR_S_FREE));
      // ---- epilogue: O / sum -> fp16 at (token, q head g * G + hh)
      if (!mbar_wait(bar(BAR_O_FULL), static_cast<uint32_t>(local & 1), a.err, WAIT_TIMEOUT_NS)) break;
      tc_fence_after();
      const float inv = sum > 0.f ? 1.f / sum : 0.f;
      f16* dst = a.out + static_cast<int64_t>(tk) * a.ld_out + (g * G + hh) * HEAD_DIM;
#pragma unroll 1
      for (int c0 = 0; c0 < HEAD_DIM; c0 += 64) {
        uint32_t v[2][32];
        tmem_ld32(trow + O_COL + c0, v[0]);
        tmem_ld32(trow + O_COL + c0 + 32, v[1]);
        tmem_ld_wait();
        if (valid) {
#pragma unroll
          for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const uint32_t* x = v[c] + 8 * q;
              uint4 o;
              o.x = pack_f16x2(__uint_as_float(x[0]) * inv, __uint_as_float(x[1]) * inv);
              o.y = pack_f16x2(__uint_as_float(x[2]) * inv, __uint_as_float(x[3]) * inv);
              o.z = pack_f16x2(__uint_as_float(x[4]) * inv, __uint_as_float(x[5]) * inv);
              o.w = pack_f16x2(__uint_as_float(x[6]) * inv, __uint_as_float(x[7]) * inv);
              *reinterpret_cast<uint4*>(dst + c0 + c * 32 + 8 * q) = o;
            }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(BAR_O_FREE));
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

}  // namespace

cudaError_t attn_tc_setup() {
  return cudaFuncSetAttribute(k_attn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
}

cudaError_t launch_attention_tc(const CUtensorMap& tm_q, const CUtensorMap& tm_kv, const CUtensorMap& tm_pool,
                                const AttnTcArgs& a, int num_sms, cudaStream_t st) {
  if (a.n_units <= 0) return cudaSuccess;
  const int grid = a.n_units < num_sms ? a.n_units : num_sms;
  k_attn_tc<<<grid, THREADS, SMEM_BYTES, st>>>(tm_q, tm_kv, tm_pool, a);
  return cudaGetLastError();
}

}  // namespace dopr
