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
//   warp 0    TMA producer: the Q tile (two stages), the tile's key blocks of
//             64 columns into a K ring (five stages) and a V ring (three) --
//             prefix blocks from the store pool in 64-row boxes, own-key
//             segments from the packed QKV buffer in the largest of 64-, 32-
//             or 16-row boxes that stays inside one pair's visible tokens;
//   warp 1    MMA issuer: S = Q K^T into the unit's TMEM region (fp32, up to
//             256 columns; one MMA per 16-element step spans every key block
//             held in consecutive ring stages), then O = P V block by block
//             with P read from TMEM and V from shared memory as an MN-major
//             operand, into the region's upper 128 columns (over S blocks 2
//             and 3, when the unit has them, once the softmax has read them);
//             S of the next unit goes in before P V of this one;
//   warps 2-9 two softmax/epilogue warpgroups taking alternate units, one
//             thread per tile row (its TMEM lane): an exact two-pass softmax
//             over the row's S (the maximum over the visible keys, then exp2
//             and fixed-shape 16-key sums added in key order), P written as
//             fp16 into TMEM over S columns already read, and after the last
//             P V step O / sum as fp16, staged per warp for whole-line stores.
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
constexpr int NSLOT = 2;  // tiles in flight: one softmax warpgroup and one TMEM region each
constexpr int Q_STAGES = 2, K_STAGES = 5, V_STAGES = 3;
constexpr int Q_HALF = TILE_M * 128;    // 128 rows x 64 16-bit elements
constexpr int Q_BYTES = 2 * Q_HALF;     // 32 KB
constexpr int KV_HALF = KBLK * 128;     // 64 rows x 64 elements
constexpr int KV_BYTES = 2 * KV_HALF;   // 16 KB
constexpr int GROUP_BYTES = 2 * GROUP_ROWS * 128;
constexpr int EP_WARP_BYTES = 32 * 128;  // one warp's 32 rows x 64 fp16 columns of O on the way out
constexpr int THREADS = 64 + NSLOT * 128;
constexpr int MAX_BLOCKS = ATTN_TC_MAX_KEYS / KBLK;  // 4
// TMEM region of a slot (256 columns): S at [0, 64 nb); P of block j, fp16, at
// [32 j, 32 j + 32) over S columns the softmax has read; O at [128, 256), over
// S blocks 2 and 3 when the unit has them.
constexpr uint32_t TMEM_COLS = 512, SLOT_COLS = 256, O_COL = 128;

// Shared memory.  The K ring is half-major ([half][stage][64 rows][128 B]): the
// rows of consecutive stages follow one another, so the blocks of a unit that
// sit in consecutive stages are one K-major operand for a single wide S MMA.
// Q and V stages keep their two 64-column halves together.
constexpr int OFF_Q = 0;
constexpr int OFF_K = OFF_Q + Q_STAGES * Q_BYTES;
constexpr int OFF_V = OFF_K + K_STAGES * KV_BYTES;
constexpr int OFF_EP = OFF_V + V_STAGES * KV_BYTES;
constexpr int OFF_BAR = OFF_EP + NSLOT * 4 * EP_WARP_BYTES;
constexpr int BAR_Q_FULL = 0, BAR_Q_EMPTY = BAR_Q_FULL + Q_STAGES;
constexpr int BAR_K_FULL = BAR_Q_EMPTY + Q_STAGES, BAR_K_EMPTY = BAR_K_FULL + K_STAGES;
constexpr int BAR_V_FULL = BAR_K_EMPTY + K_STAGES, BAR_V_EMPTY = BAR_V_FULL + V_STAGES;
constexpr int BAR_P_FULL = BAR_V_EMPTY + V_STAGES;             // [slot][block]: P of the block is in TMEM
constexpr int BAR_S_FULL = BAR_P_FULL + NSLOT * MAX_BLOCKS;    // [slot]: S complete
constexpr int BAR_R_FREE = BAR_S_FULL + NSLOT;                 // [slot]: the region's O read out
constexpr int BAR_O_FULL = BAR_R_FREE + NSLOT;                 // [slot]: O complete
constexpr int BAR_DRAIN = BAR_O_FULL + NSLOT, N_BARS = BAR_DRAIN + 1;
static_assert(BAR_V_FULL + V_STAGES <= 32, "the producer tracks the barriers it arms in one 32-bit mask");
constexpr int SMEM_BYTES = 1024 + OFF_BAR + N_BARS * 8 + 16;
static_assert(SMEM_BYTES <= 227 * 1024, "shared memory budget");

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

// Own segment s of a tile: first token (relative to tok_begin) and token count.
__device__ __forceinline__ int seg_start(int32_t v) { return static_cast<int>(static_cast<int16_t>(v & 0xffff)); }
__device__ __forceinline__ int seg_len(int32_t v) { return static_cast<int>(static_cast<uint32_t>(v) >> 16); }

// Pull a tile record (two 128-byte lines at most) into L1 ahead of its use.
__device__ __forceinline__ void prefetch_tile(const AttnTile* t) {
  const char* c = reinterpret_cast<const char*>(t);
  asm volatile("prefetch.global.L1 [%0];" ::"l"(c));
  asm volatile("prefetch.global.L1 [%0];" ::"l"(c + sizeof(AttnTile) - 1));
}

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

// P for 32 columns: 2^(s * scale - mxs) where the mask bit is set, else 0, packed
// as fp16 pairs (key 2i in the low half of pk[i]) for a TMEM store.  Returns
// sum + the two 16-column partial sums, each a fixed pairwise tree, added in
// column order.
__device__ __forceinline__ float exp_pack(uint32_t (&v)[32], uint32_t mask, float scale_log2, float mxs, float sum,
                                          uint32_t (&pk)[16]) {
#pragma unroll
  for (int e = 0; e < 32; ++e) {
    const float x = ex2_approx(fmaf(__uint_as_float(v[e]), scale_log2, -mxs));
    v[e] = __float_as_uint((mask >> e) & 1u ? x : 0.f);
  }
#pragma unroll
  for (int i = 0; i < 16; ++i) pk[i] = pack_f16x2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
#pragma unroll
  for (int gidx = 0; gidx < 2; ++gidx) {
    float t[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) t[i] = __uint_as_float(v[16 * gidx + 2 * i]) + __uint_as_float(v[16 * gidx + 2 * i + 1]);
#pragma unroll
    for (int w2 = 4; w2 >= 1; w2 >>= 1)
#pragma unroll
      for (int i = 0; i < w2; ++i) t[i] = t[2 * i] + t[2 * i + 1];
    sum += t[0];
  }
  return sum;
}

__global__ void __launch_bounds__(THREADS, 1)
    k_attn_tc(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kv,
              const __grid_constant__ CUtensorMap tm_kv32, const __grid_constant__ CUtensorMap tm_kv64,
              const __grid_constant__ CUtensorMap tm_pool, AttnTcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t s0 = smem_u32(smem);
  const uint32_t sQ = s0 + OFF_Q, sK = s0 + OFF_K, sV = s0 + OFF_V;
  auto bar = [&](int i) { return s0 + OFF_BAR + 8u * static_cast<uint32_t>(i); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_BAR + N_BARS * 8);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.Hq / a.Hkv;
  const int TT = TILE_M / G;
  // this CTA's units: blockIdx.x + i * gridDim.x, i < n_local; unit i goes to slot i % 2
  const int n_local = blockIdx.x < a.n_units ? (a.n_units - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
  auto unit_of = [&](int i) { return blockIdx.x + i * gridDim.x; };

  if (threadIdx.x == 0) {
    for (int i = 0; i < Q_STAGES; ++i) {
      mbar_init(bar(BAR_Q_FULL + i), 1);
      mbar_init(bar(BAR_Q_EMPTY + i), 1);
    }
    for (int i = 0; i < K_STAGES; ++i) {
      mbar_init(bar(BAR_K_FULL + i), 1);
      mbar_init(bar(BAR_K_EMPTY + i), 1);
    }
    for (int i = 0; i < V_STAGES; ++i) {
      mbar_init(bar(BAR_V_FULL + i), 1);
      mbar_init(bar(BAR_V_EMPTY + i), 1);
    }
    for (int i = 0; i < NSLOT * MAX_BLOCKS; ++i) mbar_init(bar(BAR_P_FULL + i), 4);
    for (int i = 0; i < NSLOT; ++i) {
      mbar_init(bar(BAR_S_FULL + i), 1);
      mbar_init(bar(BAR_R_FREE + i), 4);
      mbar_init(bar(BAR_O_FULL + i), 1);
    }
    mbar_init(bar(BAR_DRAIN), 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_kv);
    tma_prefetch_desc(&tm_kv32);
    tma_prefetch_desc(&tm_kv64);
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
      // ======================= TMA producer: Q, then K blocks, then V blocks, unit after unit
      Ring rq, rk, rv;
      uint32_t armed = 0, armed_par = 0;  // bit per barrier index: ever armed / parity of the last arm
      auto arm = [&](int b, uint32_t par, uint32_t bytes) {
        mbar_arrive_expect_tx(bar(b), bytes);
        armed |= 1u << b;
        armed_par = (armed_par & ~(1u << b)) | (par << b);
      };
      // Q and K of unit i + 1 go out before V of unit i: the MMA issuer runs
      // S(i + 1) ahead of P V(i), so V(i) may wait for ring space behind P V(i).
      auto issue_q = [&](int tok_begin, int g) -> bool {
        if (!mbar_wait(bar(BAR_Q_EMPTY + rq.stage), rq.phase ^ 1u, a.err, WAIT_TIMEOUT_NS)) return false;
        arm(BAR_Q_FULL + rq.stage, rq.phase, Q_BYTES);
        for (int h = 0; h < 2; ++h)  // one box per 64-column half: TT rows of each of the group's G heads
          tma_load_3d(sQ + rq.stage * Q_BYTES + h * Q_HALF, &tm_q, bar(BAR_Q_FULL + rq.stage), h * 64, tok_begin,
                      g * G);
        rq.next(Q_STAGES);
        return true;
      };
      auto issue_keys = [&](const AttnTile* tp, int g, int kv) -> bool {
        Ring& r = kv ? rv : rk;
        const int full0 = kv ? BAR_V_FULL : BAR_K_FULL, empty0 = kv ? BAR_V_EMPTY : BAR_K_EMPTY;
        const uint32_t ring = kv ? sV : sK;
        const int m = tp->m, n_keys = tp->n_keys, tok_begin = tp->tok_begin;
        const int pre64 = ceil64(m);
        const int nb = (n_keys + KBLK - 1) / KBLK;
        const int pool_row = static_cast<int>(tp->pool_base + ((static_cast<int64_t>(a.layer) * 2 + kv) * a.Hkv + g) * m);
        const int col0 = (a.Hq + kv * a.Hkv + g) * HEAD_DIM;
        if (kCheckedBuild) {  // report only: the tensor maps bound every copy themselves
          index_ok(a.ext.err, tok_begin + seg_start(tp->seg[0]), a.ext.rows);
          index_ok(a.ext.err, tok_begin + tp->n_tok - 1, a.ext.rows);
          if (m > 0) index_ok(a.ext.err, pool_row + m - 1, a.ext.pool_rows);
        }
        int si = 0, k = 0, key = pre64;  // own-key cursor: segment, row within it, key column
        int sv = tp->seg[0];
        for (int j = 0; j < nb; ++j) {
          if (!mbar_wait(bar(empty0 + r.stage), r.phase ^ 1u, a.err, WAIT_TIMEOUT_NS)) return false;
          // half h of the stage: K halves lie K_STAGES * 8 KB apart (see OFF_K), V halves 8 KB apart
          const uint32_t dst = kv ? ring + r.stage * KV_BYTES : ring + r.stage * KV_HALF;
          const uint32_t hstride = kv ? KV_HALF : K_STAGES * KV_HALF;
          const uint32_t fb = bar(full0 + r.stage);
          if (j * KBLK < pre64) {
            arm(full0 + r.stage, r.phase, KV_BYTES);
            for (int h = 0; h < 2; ++h) tma_load_2d(dst + h * hstride, &tm_pool, fb, h * 64, pool_row + j * KBLK);
          } else {
            const int groups = min(KBLK, n_keys - j * KBLK) / GROUP_ROWS;
            arm(full0 + r.stage, r.phase, groups * GROUP_BYTES);
            if (groups * GROUP_ROWS == KBLK && key == j * KBLK && k + KBLK <= seg_len(sv)) {
              // the whole block is 64 consecutive tokens of one pair: one 64-row box per half
              for (int h = 0; h < 2; ++h)
                tma_load_2d(dst + h * hstride, &tm_kv64, fb, col0 + h * 64, tok_begin + seg_start(sv) + k);
              key += KBLK;
              k += KBLK;
              if (k >= seg_len(sv) && si + 1 < ATTN_TC_MAX_SEGS) {
                k = 0;
                sv = tp->seg[++si];
              }
            } else {
              for (int q = 0; q < groups;) {
                const int off = key - j * KBLK;  // 0, 16, 32, 48 when the plan is consistent
                // two groups at once when both are 16 consecutive visible tokens of this pair
                const int n = (q + 2 <= groups && k + 2 * GROUP_ROWS <= seg_len(sv)) ? 2 : 1;
                if (off >= 0 && off + n * GROUP_ROWS <= KBLK)  // otherwise skipped and the wait times out
                  for (int h = 0; h < 2; ++h)
                    tma_load_2d(dst + off * 128 + h * hstride, n == 2 ? &tm_kv32 : &tm_kv, fb, col0 + h * 64,
                                tok_begin + seg_start(sv) + k);
                key += n * GROUP_ROWS;
                k += n * GROUP_ROWS;
                q += n;
                if (k >= seg_len(sv) && si + 1 < ATTN_TC_MAX_SEGS) {
                  k = 0;
                  sv = tp->seg[++si];
                }
              }
            }
          }
          r.next(kv ? V_STAGES : K_STAGES);
        }
        return true;
      };
      bool ok = true;
      for (int i = 0; i <= n_local && ok; ++i) {
        if (i + 1 < n_local) prefetch_tile(a.tiles + unit_of(i + 1) / a.Hkv);
        if (i < n_local) {
          const int u = unit_of(i);
          const AttnTile* tp = a.tiles + u / a.Hkv;
          ok = issue_q(tp->tok_begin, u % a.Hkv) && issue_keys(tp, u % a.Hkv, 0);
        }
        if (ok && i > 0) {
          const int u = unit_of(i - 1);
          ok = issue_keys(a.tiles + u / a.Hkv, u % a.Hkv, 1);
        }
      }
      if (!ok) {  // every copy this thread started lands before the CTA can exit
        for (int b = 0; b < 32; ++b)
          if (armed & (1u << b)) mbar_wait(bar(b), (armed_par >> b) & 1u, a.err, 100000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ======================= MMA issuer: an event loop over non-blocking barrier tests.
      // P V blocks of unit ip go in as soon as their P and V are there; S blocks of
      // unit is (at most one unit ahead) as soon as Q, the slot's region and K are.
      Ring rq, rk, rv;
      uint32_t ppar = 0;            // bit slot * MAX_BLOCKS + j: parity of the next P_FULL completion
      int is = 0, js = 0, nbs = 0;  // S: unit, next block, blocks
      bool s_open = false;          // unit is's Q and region are in hand
      int ip = 0, jp = 0;           // P V: unit, next block
      int nk_p = -1;                // key columns of unit ip (read once it is needed)
      // Idle polls are cheap barrier tests; the error word (a global load) and the clock
      // are read only every IDLE_CHECK idle polls, so a hand-off is seen within one poll.
      constexpr uint32_t IDLE_CHECK = 2048;
      uint32_t idle = 0;
      uint64_t idle_since = 0;
      bool ok = true;
      while (ip < n_local) {
        bool prog = false;
        // ---- O = P V of unit ip, whose S is complete; P is read from TMEM
        if (ip < is) {
          const int slot = ip & 1;
          if (nk_p < 0) nk_p = a.tiles[unit_of(ip) / a.Hkv].n_keys;  // once per unit, not per poll
          const int n_keys = nk_p;
          const int nbp = (n_keys + KBLK - 1) / KBLK;
          auto p_ready = [&](int j) {
            return mbar_test(bar(BAR_P_FULL + slot * MAX_BLOCKS + j), (ppar >> (slot * MAX_BLOCKS + j)) & 1u);
          };
          while (jp < nbp) {
            bool ready = p_ready(jp);
            // O (columns 128..255) covers S blocks 2 and 3: with more than two blocks the
            // softmax must be past its last S read, i.e. the last block's P is in
            if (ready && jp == 0 && nbp > 2) ready = p_ready(nbp - 1);
            if (!ready || !mbar_test(bar(BAR_V_FULL + rv.stage), rv.phase)) break;
            tc_fence_after();
            const int steps = min(KBLK, n_keys - jp * KBLK) / 16;  // only rows the producer loaded
            const uint32_t pcol = tmem + slot * SLOT_COLS + 32 * jp;  // 16 keys = 8 columns per step
            for (int kk = 0; kk < steps; ++kk)
              umma_f16_ts(tmem + slot * SLOT_COLS + O_COL, pcol + 8 * kk,
                          umma_desc_sw128_mn(sV + rv.stage * KV_BYTES + kk * 2048, KV_HALF, 1024), IDESC_O,
                          (jp | kk) != 0);
            umma_commit(bar(BAR_V_EMPTY + rv.stage));
            rv.next(V_STAGES);
            ++jp;
            prog = true;
          }
          if (jp == nbp) {
            umma_commit(bar(BAR_O_FULL + slot));
            for (int j = 0; j < nbp; ++j) ppar ^= 1u << (slot * MAX_BLOCKS + j);  // each block's barrier completed once
            ++ip;
            jp = 0;
            nk_p = -1;
            prog = true;
          }
        }
        // ---- S = Q K^T of unit is
        if (is < n_local && is <= ip + 1) {
          const int slot = is & 1;
          if (!s_open && mbar_test(bar(BAR_Q_FULL + rq.stage), rq.phase) &&
              mbar_test(bar(BAR_R_FREE + slot), ((is >> 1) & 1) ^ 1u)) {
            s_open = true;
            js = 0;
            nbs = (a.tiles[unit_of(is) / a.Hkv].n_keys + KBLK - 1) / KBLK;
            if (is + 1 < n_local) prefetch_tile(a.tiles + unit_of(is + 1) / a.Hkv);
            tc_fence_after();
            prog = true;
          }
          while (s_open && js < nbs) {
            // the unit's next blocks that sit in consecutive ring stages form one B operand of
            // 64 * run rows: one N = 64 * run MMA per 16-element step once all of them are in
            const int run = min(nbs - js, K_STAGES - rk.stage);
            bool landed = true;
            for (int t = 0; t < run && landed; ++t) landed = mbar_test(bar(BAR_K_FULL + rk.stage + t), rk.phase);
            if (!landed) break;
            tc_fence_after();
            const uint64_t qd = umma_desc_sw128(sQ + rq.stage * Q_BYTES);
            const uint64_t kd = umma_desc_sw128(sK + rk.stage * KV_HALF);
            const uint32_t idesc = umma_idesc_f16(TILE_M, run * KBLK);
#pragma unroll
            for (int ks = 0; ks < HEAD_DIM / 16; ++ks)  // 16 elements = 32 bytes per step; Q halves 16 KB apart
              umma_f16(tmem + slot * SLOT_COLS + js * KBLK, qd + ((ks >> 2) * Q_HALF + (ks & 3) * 32) / 16,
                       kd + ((ks >> 2) * K_STAGES * KV_HALF + (ks & 3) * 32) / 16, idesc, ks > 0);
            for (int t = 0; t < run; ++t) {
              umma_commit(bar(BAR_K_EMPTY + rk.stage));
              rk.next(K_STAGES);
            }
            js += run;
            prog = true;
          }
          if (s_open && js == nbs) {
            umma_commit(bar(BAR_S_FULL + slot));
            umma_commit(bar(BAR_Q_EMPTY + rq.stage));
            rq.next(Q_STAGES);
            ++is;
            s_open = false;
          }
        }
        if (prog) {
          idle = 0;
        } else if (++idle % IDLE_CHECK == 0) {
          const uint64_t now = globaltimer_ns();
          if (idle == IDLE_CHECK) idle_since = now;  // the first check of this idle stretch
          if ((ld_volatile(a.err) & DEV_ERR_TIMEOUT) || now - idle_since > WAIT_TIMEOUT_NS) {
            atomicOr(a.err, DEV_ERR_TIMEOUT);
            ok = false;
            break;
          }
        }
      }
      // every MMA this thread issued is complete once the drain barrier flips
      umma_commit(bar(BAR_DRAIN));
      mbar_wait(bar(BAR_DRAIN), 0, a.err, ok ? WAIT_TIMEOUT_NS : 100000000ull);
    }
  } else {
    // ======================= softmax + epilogue: warpgroup `slot` = warps 2 + 4 slot .. 5 + 4 slot,
    // TMEM lane quarter warp % 4
    const int slot = (warp - 2) >> 2;
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;  // tile row
    const int jj = r % TT;  // this row's token within the tile (its q head is r / TT)
    const uint32_t trow = tmem + slot * SLOT_COLS + (static_cast<uint32_t>(quarter * 32) << 16);
    const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HEAD_DIM));
    uint8_t* stg = smem + OFF_EP + (slot * 4 + quarter) * EP_WARP_BYTES;  // this warp's staging lines
    for (int i = slot, k = 0; i < n_local; i += NSLOT, ++k) {
      const uint32_t par = static_cast<uint32_t>(k & 1);
      const int u = unit_of(i);
      if (i + NSLOT < n_local) prefetch_tile(a.tiles + unit_of(i + NSLOT) / a.Hkv);
      const AttnTile* tp = a.tiles + u / a.Hkv;
      const int g = u % a.Hkv;
      const int m = tp->m, n_tok = tp->n_tok, n_seg = tp->n_seg;
      const int pre64 = ceil64(m);
      const int ncol = ((tp->n_keys + KBLK - 1) / KBLK) * KBLK;
      const bool valid = jj < n_tok;
      // Visible keys: prefix columns [0, m) and own columns [olo, ohi].  Rows past
      // the tile's tokens see the prefix only; nothing of theirs is stored.
      int olo = INT_MAX, ohi = -1;
      if (valid) {
        int seg = pre64;
        for (int si = 0; si < n_seg; ++si) {
          const int sv = tp->seg[si];
          const int st = seg_start(sv), len = seg_len(sv);
          if (jj < st + len) {
            olo = seg;
            ohi = seg + (jj - st);
            break;
          }
          seg += ceil16(len);
        }
      }
      const int wlo = __reduce_min_sync(0xffffffffu, olo);
      const int whi = __reduce_max_sync(0xffffffffu, ohi);
      auto chunk_live = [&](int c0) { return c0 < m || (c0 <= whi && c0 + 31 >= wlo); };
      auto vis_mask = [&](int c0) { return bits_in(-c0, m - c0) | bits_in(olo - c0, ohi + 1 - c0); };

      if (!mbar_wait(bar(BAR_S_FULL + slot), par, a.err, WAIT_TIMEOUT_NS)) break;
      tc_fence_after();
      // ---- pass 1: the row maximum over the visible keys
      float mx = -INFINITY;
      for (int c0 = 0; c0 < ncol; c0 += 32) {
        if (!chunk_live(c0)) continue;
        uint32_t v[32];
        tmem_ld32(trow + c0, v);
        tmem_ld_wait();
        mx = fmaxf(mx, masked_max32(v, vis_mask(c0)));
      }
      const float mxs = (mx == -INFINITY) ? 0.f : mx * scale_log2;
      // ---- pass 2: P = 2^((s - max) * scale) per 64-key block, as fp16 into TMEM
      // columns [32 j, 32 j + 32) (S columns this pass has read); the sum adds
      // fixed-shape 16-key partial sums in key order
      float sum = 0.f;
      for (int c0 = 0, j = 0; c0 < ncol; c0 += KBLK, ++j) {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int cb = c0 + 32 * half;
          uint32_t pk[16];
          if (chunk_live(cb)) {
            uint32_t v[32];
            tmem_ld32(trow + cb, v);
            tmem_ld_wait();
            sum = exp_pack(v, vis_mask(cb), scale_log2, mxs, sum, pk);
          } else {
#pragma unroll
            for (int q = 0; q < 16; ++q) pk[q] = 0u;
          }
          tmem_st16(trow + 32 * j + 16 * half, pk);
        }
        tmem_st_wait();
        tc_fence_before();  // this block's S reads and P writes precede the MMAs that follow
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(BAR_P_FULL + slot * MAX_BLOCKS + j));
      }
      // ---- epilogue: O / sum -> fp16 at (token, q head g * G + hh), 64 columns at a
      // time through this warp's staging lines (128 bytes per row, 16-byte chunks
      // swizzled by the row), each store instruction writing four 128-byte row pieces
      if (!mbar_wait(bar(BAR_O_FULL + slot), par, a.err, WAIT_TIMEOUT_NS)) break;
      tc_fence_after();
      const float inv = sum > 0.f ? 1.f / sum : 0.f;
      bool bad = false;  // a stored output value not finite or beyond fp16's range
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
#pragma unroll
        for (int c2 = 0; c2 < 2; ++c2) {
          uint32_t v[32];
          tmem_ld32(trow + O_COL + 64 * h + 32 * c2, v);
          tmem_ld_wait();
          if (h == 1 && c2 == 1) {  // O is out of TMEM: the region is free
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(BAR_R_FREE + slot));
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t* x = v + 8 * q;
            float y[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              y[e] = __uint_as_float(x[e]) * inv;
              bad |= valid && !fp16_ok(y[e]);  // rows past the tile's tokens are not stored
            }
            uint4 o;
            o.x = pack_f16x2(y[0], y[1]);
            o.y = pack_f16x2(y[2], y[3]);
            o.z = pack_f16x2(y[4], y[5]);
            o.w = pack_f16x2(y[6], y[7]);
            const int chunk = c2 * 4 + q;
            *reinterpret_cast<uint4*>(stg + lane * 128 + ((chunk ^ (lane & 7)) << 4)) = o;
          }
        }
        __syncwarp();
#pragma unroll
        for (int it = 0; it < 8; ++it) {
          const int rr = it * 4 + (lane >> 3), ch = lane & 7;
          const int row = quarter * 32 + rr;  // tile row
          const int j2 = row % TT;
          if (j2 < n_tok && index_ok(a.ext.err, tp->tok_begin + j2, a.ext.rows)) {
            const uint4 x = *reinterpret_cast<const uint4*>(stg + rr * 128 + ((ch ^ (rr & 7)) << 4));
            *reinterpret_cast<uint4*>(a.out + static_cast<int64_t>(tp->tok_begin + j2) * a.ld_out +
                                      (g * G + row / TT) * HEAD_DIM + 64 * h + ch * 8) = x;
          }
        }
        __syncwarp();  // staging reads finish before the next half's writes
      }
      if (bad) atomicOr(a.err, DEV_ERR_RANGE);
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

// ============================================================================
// Long tiles: more key columns than one TMEM region holds (long queries, the
// longest prefixes with long queries, uncompressed documents).  One unit at a
// time per CTA, one softmax warpgroup, the keys in 128-column chunks through
// two S buffers: pass A computes S chunk by chunk for the exact row maximum,
// pass B computes each chunk again, writes P as fp16 into a four-stage TMEM
// ring and accumulates O = P V (P from TMEM, as in the short kernel) in its own
// 128 TMEM columns.  The row results are the short kernel's: the same maximum,
// the same 16-key sums in key order, the same MMA steps.
namespace lt {
constexpr int Q_STAGES = 2, K_STAGES = 5, V_STAGES = 4, P_STAGES = 4;
constexpr int CH = 128;  // key columns per S chunk
constexpr int THREADS = 64 + 128;
// TMEM: O at [0, 128), S buffer b at S_COL + CH b, P stage s (64 keys as fp16) at P_COL + 32 s
constexpr uint32_t O_COL = 0, S_COL = 128, P_COL = 384;
constexpr int OFF_Q = 0;
constexpr int OFF_K = OFF_Q + Q_STAGES * Q_BYTES;  // half-major, as in the short kernel
constexpr int OFF_V = OFF_K + K_STAGES * KV_BYTES;
constexpr int OFF_EP = OFF_V + V_STAGES * KV_BYTES;
constexpr int OFF_BAR = OFF_EP + 4 * EP_WARP_BYTES;
constexpr int B_Q_FULL = 0, B_Q_EMPTY = B_Q_FULL + Q_STAGES;
constexpr int B_K_FULL = B_Q_EMPTY + Q_STAGES, B_K_EMPTY = B_K_FULL + K_STAGES;
constexpr int B_V_FULL = B_K_EMPTY + K_STAGES, B_V_EMPTY = B_V_FULL + V_STAGES;
constexpr int B_P_FULL = B_V_EMPTY + V_STAGES, B_P_EMPTY = B_P_FULL + P_STAGES;
constexpr int B_S_FULL = B_P_EMPTY + P_STAGES, B_S_FREE = B_S_FULL + 2;
constexpr int B_O_FULL = B_S_FREE + 2, B_O_FREE = B_O_FULL + 1, B_DRAIN = B_O_FREE + 1, N_BARS = B_DRAIN + 1;
constexpr int SMEM_BYTES = 1024 + OFF_BAR + N_BARS * 8 + 16;
static_assert(SMEM_BYTES <= 227 * 1024, "shared memory budget");
static_assert(B_V_FULL + V_STAGES <= 32, "producer arm mask");
static_assert(P_COL + 32 * P_STAGES <= TMEM_COLS, "P ring inside the allocation");
}  // namespace lt

__global__ void __launch_bounds__(lt::THREADS, 1)
    k_attn_tc_long(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kv,
                   const __grid_constant__ CUtensorMap tm_kv32, const __grid_constant__ CUtensorMap tm_kv64,
                   const __grid_constant__ CUtensorMap tm_pool, AttnTcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t s0 = smem_u32(smem);
  const uint32_t sQ = s0 + lt::OFF_Q, sK = s0 + lt::OFF_K, sV = s0 + lt::OFF_V;
  auto bar = [&](int i) { return s0 + lt::OFF_BAR + 8u * static_cast<uint32_t>(i); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + lt::OFF_BAR + lt::N_BARS * 8);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = a.Hq / a.Hkv;
  const int TT = TILE_M / G;
  const int n_local = blockIdx.x < a.n_units ? (a.n_units - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
  auto unit_of = [&](int i) { return blockIdx.x + i * gridDim.x; };
  auto blocks_of = [](int n_keys) { return (n_keys + KBLK - 1) / KBLK; };

  if (threadIdx.x == 0) {
    for (int i = 0; i < lt::Q_STAGES; ++i) {
      mbar_init(bar(lt::B_Q_FULL + i), 1);
      mbar_init(bar(lt::B_Q_EMPTY + i), 1);
    }
    for (int i = 0; i < lt::K_STAGES; ++i) {
      mbar_init(bar(lt::B_K_FULL + i), 1);
      mbar_init(bar(lt::B_K_EMPTY + i), 1);
    }
    for (int i = 0; i < lt::V_STAGES; ++i) {
      mbar_init(bar(lt::B_V_FULL + i), 1);
      mbar_init(bar(lt::B_V_EMPTY + i), 1);
    }
    for (int i = 0; i < lt::P_STAGES; ++i) {
      mbar_init(bar(lt::B_P_FULL + i), 4);
      mbar_init(bar(lt::B_P_EMPTY + i), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(lt::B_S_FULL + i), 1);
      mbar_init(bar(lt::B_S_FREE + i), 4);
    }
    mbar_init(bar(lt::B_O_FULL), 1);
    mbar_init(bar(lt::B_O_FREE), 4);
    mbar_init(bar(lt::B_DRAIN), 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_kv);
    tma_prefetch_desc(&tm_kv32);
    tma_prefetch_desc(&tm_kv64);
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
      // ======================= TMA producer: Q; pass A's K blocks; pass B's K and V blocks chunk by chunk
      Ring rq, rk, rv;
      uint32_t armed = 0, armed_par = 0;
      auto arm = [&](int b, uint32_t par, uint32_t bytes) {
        mbar_arrive_expect_tx(bar(b), bytes);
        armed |= 1u << b;
        armed_par = (armed_par & ~(1u << b)) | (par << b);
      };
      // a block stream of one tile's K or V rows: blocks must be issued in order 0, 1, ...
      struct Stream {
        int kv, si, k, sv, pool_row, col0;
      };
      auto start = [&](const AttnTile* tp, int g, int kv) {
        Stream st;
        st.kv = kv;
        st.si = 0;
        st.k = 0;
        st.sv = tp->seg[0];
        st.pool_row = static_cast<int>(tp->pool_base + ((static_cast<int64_t>(a.layer) * 2 + kv) * a.Hkv + g) * tp->m);
        st.col0 = (a.Hq + kv * a.Hkv + g) * HEAD_DIM;
        if (kCheckedBuild) {  // report only: the tensor maps bound every copy themselves
          index_ok(a.ext.err, tp->tok_begin + seg_start(tp->seg[0]), a.ext.rows);
          index_ok(a.ext.err, tp->tok_begin + tp->n_tok - 1, a.ext.rows);
          if (tp->m > 0) index_ok(a.ext.err, st.pool_row + tp->m - 1, a.ext.pool_rows);
        }
        return st;
      };
      auto issue_block = [&](const AttnTile* tp, Stream& st, int j) -> bool {
        Ring& r = st.kv ? rv : rk;
        const int stages = st.kv ? lt::V_STAGES : lt::K_STAGES;
        const int full0 = st.kv ? lt::B_V_FULL : lt::B_K_FULL, empty0 = st.kv ? lt::B_V_EMPTY : lt::B_K_EMPTY;
        if (!mbar_wait(bar(empty0 + r.stage), r.phase ^ 1u, a.err, WAIT_TIMEOUT_NS)) return false;
        // half h of the stage: K halves lie K_STAGES * 8 KB apart (half-major K ring), V halves 8 KB apart
        const uint32_t dst = st.kv ? sV + r.stage * KV_BYTES : sK + r.stage * KV_HALF;
        const uint32_t hstride = st.kv ? KV_HALF : lt::K_STAGES * KV_HALF;
        const uint32_t fb = bar(full0 + r.stage);
        if (j * KBLK < ceil64(tp->m)) {
          arm(full0 + r.stage, r.phase, KV_BYTES);
          for (int h = 0; h < 2; ++h) tma_load_2d(dst + h * hstride, &tm_pool, fb, h * 64, st.pool_row + j * KBLK);
        } else {
          const int groups = min(KBLK, tp->n_keys - j * KBLK) / GROUP_ROWS;
          arm(full0 + r.stage, r.phase, groups * GROUP_BYTES);
          if (groups * GROUP_ROWS == KBLK && st.k + KBLK <= seg_len(st.sv)) {
            // the whole block is 64 consecutive tokens of one pair: one 64-row box per half
            for (int h = 0; h < 2; ++h)
              tma_load_2d(dst + h * hstride, &tm_kv64, fb, st.col0 + h * 64, tp->tok_begin + seg_start(st.sv) + st.k);
            st.k += KBLK;
            if (st.k >= seg_len(st.sv) && st.si + 1 < ATTN_TC_MAX_SEGS) {
              st.k = 0;
              st.sv = tp->seg[++st.si];
            }
          } else {
            for (int q = 0; q < groups;) {
              // two groups at once when both are 16 consecutive visible tokens of this pair
              const int n = (q + 2 <= groups && st.k + 2 * GROUP_ROWS <= seg_len(st.sv)) ? 2 : 1;
              for (int h = 0; h < 2; ++h)
                tma_load_2d(dst + q * GROUP_ROWS * 128 + h * hstride, n == 2 ? &tm_kv32 : &tm_kv, fb,
                            st.col0 + h * 64, tp->tok_begin + seg_start(st.sv) + st.k);
              st.k += n * GROUP_ROWS;
              q += n;
              if (st.k >= seg_len(st.sv) && st.si + 1 < ATTN_TC_MAX_SEGS) {
                st.k = 0;
                st.sv = tp->seg[++st.si];
              }
            }
          }
        }
        r.next(stages);
        return true;
      };
      bool ok = true;
      for (int i = 0; i < n_local && ok; ++i) {
        const int u = unit_of(i);
        const AttnTile* tp = a.tiles + u / a.Hkv;
        const int g = u % a.Hkv;
        const int nb = blocks_of(tp->n_keys);
        if (i + 1 < n_local) prefetch_tile(a.tiles + unit_of(i + 1) / a.Hkv);
        if (!mbar_wait(bar(lt::B_Q_EMPTY + rq.stage), rq.phase ^ 1u, a.err, WAIT_TIMEOUT_NS)) {
          ok = false;
          break;
        }
        arm(lt::B_Q_FULL + rq.stage, rq.phase, Q_BYTES);
        for (int h = 0; h < 2; ++h)
          tma_load_3d(sQ + rq.stage * Q_BYTES + h * Q_HALF, &tm_q, bar(lt::B_Q_FULL + rq.stage), h * 64,
                      tp->tok_begin, g * G);
        rq.next(lt::Q_STAGES);
        Stream ka = start(tp, g, 0);
        for (int j = 0; j < nb && ok; ++j) ok = issue_block(tp, ka, j);
        Stream kb = start(tp, g, 0), vb = start(tp, g, 1);
        for (int c = 0; c * 2 < nb && ok; ++c) {
          for (int j = 2 * c; j < min(nb, 2 * c + 2) && ok; ++j) ok = issue_block(tp, kb, j);
          for (int j = 2 * c; j < min(nb, 2 * c + 2) && ok; ++j) ok = issue_block(tp, vb, j);
        }
      }
      if (!ok) {
        for (int b = 0; b < 32; ++b)
          if (armed & (1u << b)) mbar_wait(bar(b), (armed_par >> b) & 1u, a.err, 100000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ======================= MMA issuer
      Ring rq, rk, rv, rp;
      uint32_t cc = 0;  // S chunks issued (both passes, all units): buffer cc & 1
      bool ok = true;
      auto wait = [&](int b, uint32_t par) { return ok = ok && mbar_wait(bar(b), par, a.err, WAIT_TIMEOUT_NS); };
      // S of key chunk c (its one or two 64-key blocks from the K ring) into buffer cc & 1
      auto issue_s = [&](int c, int nb) -> bool {
        const uint32_t buf = cc & 1u;
        if (!wait(lt::B_S_FREE + buf, ((cc >> 1) & 1u) ^ 1u)) return false;
        tc_fence_after();
        const uint64_t qd = umma_desc_sw128(sQ + rq.stage * Q_BYTES);
        const int je = min(nb, 2 * c + 2);
        for (int j = 2 * c; j < je;) {
          // the chunk's blocks in consecutive ring stages: one N = 64 * run MMA per step
          const int run = min(je - j, lt::K_STAGES - rk.stage);
          for (int t = 0; t < run; ++t)
            if (!wait(lt::B_K_FULL + rk.stage + t, rk.phase)) return false;
          tc_fence_after();
          const uint64_t kd = umma_desc_sw128(sK + rk.stage * KV_HALF);
          const uint32_t idesc = umma_idesc_f16(TILE_M, run * KBLK);
#pragma unroll
          for (int ks = 0; ks < HEAD_DIM / 16; ++ks)
            umma_f16(tmem + lt::S_COL + lt::CH * buf + (j - 2 * c) * KBLK, qd + ((ks >> 2) * Q_HALF + (ks & 3) * 32) / 16,
                     kd + ((ks >> 2) * lt::K_STAGES * KV_HALF + (ks & 3) * 32) / 16, idesc, ks > 0);
          for (int t = 0; t < run; ++t) {
            umma_commit(bar(lt::B_K_EMPTY + rk.stage));
            rk.next(lt::K_STAGES);
          }
          j += run;
        }
        umma_commit(bar(lt::B_S_FULL + buf));
        ++cc;
        return true;
      };
      for (int i = 0; i < n_local && ok; ++i) {
        const int n_keys = a.tiles[unit_of(i) / a.Hkv].n_keys;
        const int nb = blocks_of(n_keys), nc = (nb + 1) / 2;
        if (!wait(lt::B_Q_FULL + rq.stage, rq.phase)) break;
        tc_fence_after();
        for (int c = 0; c < nc && ok; ++c) issue_s(c, nb);  // pass A
        if (ok) issue_s(0, nb);                              // pass B
        for (int c = 0; c < nc && ok; ++c) {
          if (c + 1 < nc && !issue_s(c + 1, nb)) break;
          if (c == 0 && !wait(lt::B_O_FREE, (static_cast<uint32_t>(i) & 1u) ^ 1u)) break;
          for (int j = 2 * c; j < min(nb, 2 * c + 2) && ok; ++j) {
            if (!wait(lt::B_P_FULL + rp.stage, rp.phase) || !wait(lt::B_V_FULL + rv.stage, rv.phase)) break;
            tc_fence_after();
            const int steps = min(KBLK, n_keys - j * KBLK) / 16;
            const uint32_t pcol = tmem + lt::P_COL + 32 * rp.stage;  // 16 keys = 8 columns per step
            const uint64_t vd = umma_desc_sw128_mn(sV + rv.stage * KV_BYTES, KV_HALF, 1024);
            for (int kk = 0; kk < steps; ++kk)
              umma_f16_ts(tmem + lt::O_COL, pcol + 8 * kk, vd + (kk * 2048) / 16, IDESC_O, (j | kk) != 0);
            umma_commit(bar(lt::B_P_EMPTY + rp.stage));
            umma_commit(bar(lt::B_V_EMPTY + rv.stage));
            rp.next(lt::P_STAGES);
            rv.next(lt::V_STAGES);
          }
        }
        if (!ok) break;
        umma_commit(bar(lt::B_O_FULL));
        umma_commit(bar(lt::B_Q_EMPTY + rq.stage));
        rq.next(lt::Q_STAGES);
      }
      umma_commit(bar(lt::B_DRAIN));
      mbar_wait(bar(lt::B_DRAIN), 0, a.err, ok ? WAIT_TIMEOUT_NS : 100000000ull);
    }
  } else {
    // ======================= softmax + epilogue: warps 2..5 -> TMEM lane quarters 2, 3, 0, 1
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const int jj = r % TT;  // this row's token within the tile (its q head is r / TT)
    const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HEAD_DIM));
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    uint8_t* stg = smem + lt::OFF_EP + quarter * EP_WARP_BYTES;  // this warp's staging lines
    Ring rp;
    uint32_t cc = 0;
    bool ok = true;
    for (int i = 0; i < n_local && ok; ++i) {
      const int u = unit_of(i);
      if (i + 1 < n_local) prefetch_tile(a.tiles + unit_of(i + 1) / a.Hkv);
      const AttnTile* tp = a.tiles + u / a.Hkv;
      const int g = u % a.Hkv;
      const int m = tp->m, n_tok = tp->n_tok, n_seg = tp->n_seg;
      const int pre64 = ceil64(m);
      const int nb = blocks_of(tp->n_keys), nc = (nb + 1) / 2, ncol = nb * KBLK;
      const bool valid = jj < n_tok;
      int olo = INT_MAX, ohi = -1;
      if (valid) {
        int seg = pre64;
        for (int si = 0; si < n_seg; ++si) {
          const int sv = tp->seg[si];
          const int st = seg_start(sv), len = seg_len(sv);
          if (jj < st + len) {
            olo = seg;
            ohi = seg + (jj - st);
            break;
          }
          seg += ceil16(len);
        }
      }
      // every 32-column chunk of S is read and put through the mask: a chunk no
      // row of the warp sees contributes -inf to the maximum and exact zeros to P
      // and to the sum, so skipping it would not change a bit
      auto vis_mask = [&](int c0) { return bits_in(-c0, m - c0) | bits_in(olo - c0, ohi + 1 - c0); };
      // ---- pass A: the row maximum, chunk by chunk
      float mx = -INFINITY;
      for (int c = 0; c < nc && ok; ++c) {
        const uint32_t buf = cc & 1u;
        if (!mbar_wait(bar(lt::B_S_FULL + buf), (cc >> 1) & 1u, a.err, WAIT_TIMEOUT_NS)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int c0 = c * lt::CH; c0 < min(ncol, c * lt::CH + lt::CH); c0 += KBLK) {
          const uint32_t sb = lane_base + lt::S_COL + lt::CH * buf + (c0 - c * lt::CH);
          uint32_t v0[32], v1[32];
          tmem_ld32(sb, v0);
          tmem_ld32(sb + 32, v1);
          tmem_ld_wait();
          mx = fmaxf(mx, masked_max32(v0, vis_mask(c0)));
          mx = fmaxf(mx, masked_max32(v1, vis_mask(c0 + 32)));
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(lt::B_S_FREE + buf));
        ++cc;
      }
      if (!ok) break;
      const float mxs = (mx == -INFINITY) ? 0.f : mx * scale_log2;
      // ---- pass B: P per 64-key block, 16-key sums in key order
      float sum = 0.f;
      for (int c = 0; c < nc && ok; ++c) {
        const uint32_t buf = cc & 1u;
        if (!mbar_wait(bar(lt::B_S_FULL + buf), (cc >> 1) & 1u, a.err, WAIT_TIMEOUT_NS)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int j = 2 * c; j < min(nb, 2 * c + 2); ++j) {
          if (!mbar_wait(bar(lt::B_P_EMPTY + rp.stage), rp.phase ^ 1u, a.err, WAIT_TIMEOUT_NS)) {
            ok = false;
            break;
          }
          const int cb = j * KBLK;
          const uint32_t sb = lane_base + lt::S_COL + lt::CH * buf + (cb - c * lt::CH);
          uint32_t v0[32], v1[32], pk[16];
          tmem_ld32(sb, v0);
          tmem_ld32(sb + 32, v1);
          tmem_ld_wait();
          sum = exp_pack(v0, vis_mask(cb), scale_log2, mxs, sum, pk);
          tmem_st16(lane_base + lt::P_COL + 32 * rp.stage, pk);
          sum = exp_pack(v1, vis_mask(cb + 32), scale_log2, mxs, sum, pk);
          tmem_st16(lane_base + lt::P_COL + 32 * rp.stage + 16, pk);
          tmem_st_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar(lt::B_P_FULL + rp.stage));
          rp.next(lt::P_STAGES);
        }
        if (!ok) break;
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(lt::B_S_FREE + buf));
        ++cc;
      }
      if (!ok) break;
      // ---- epilogue: O / sum -> fp16, 64 columns at a time through this warp's staging lines
      if (!mbar_wait(bar(lt::B_O_FULL), static_cast<uint32_t>(i) & 1u, a.err, WAIT_TIMEOUT_NS)) break;
      tc_fence_after();
      const float inv = sum > 0.f ? 1.f / sum : 0.f;
      bool bad = false;  // a stored output value not finite or beyond fp16's range
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        uint32_t v2[2][32];
        tmem_ld32(lane_base + lt::O_COL + 64 * h, v2[0]);
        tmem_ld32(lane_base + lt::O_COL + 64 * h + 32, v2[1]);
        tmem_ld_wait();
        if (h == 1) {  // O is out of TMEM
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar(lt::B_O_FREE));
        }
#pragma unroll
        for (int c2 = 0; c2 < 2; ++c2) {
          const uint32_t* v = v2[c2];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t* x = v + 8 * q;
            float y[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              y[e] = __uint_as_float(x[e]) * inv;
              bad |= valid && !fp16_ok(y[e]);  // rows past the tile's tokens are not stored
            }
            uint4 o;
            o.x = pack_f16x2(y[0], y[1]);
            o.y = pack_f16x2(y[2], y[3]);
            o.z = pack_f16x2(y[4], y[5]);
            o.w = pack_f16x2(y[6], y[7]);
            const int chunk = c2 * 4 + q;
            *reinterpret_cast<uint4*>(stg + lane * 128 + ((chunk ^ (lane & 7)) << 4)) = o;
          }
        }
        __syncwarp();
#pragma unroll
        for (int it = 0; it < 8; ++it) {
          const int rr = it * 4 + (lane >> 3), ch = lane & 7;
          const int row = quarter * 32 + rr;  // tile row
          const int j2 = row % TT;
          if (j2 < n_tok && index_ok(a.ext.err, tp->tok_begin + j2, a.ext.rows)) {
            const uint4 x = *reinterpret_cast<const uint4*>(stg + rr * 128 + ((ch ^ (rr & 7)) << 4));
            *reinterpret_cast<uint4*>(a.out + static_cast<int64_t>(tp->tok_begin + j2) * a.ld_out +
                                      (g * G + row / TT) * HEAD_DIM + 64 * h + ch * 8) = x;
          }
        }
        __syncwarp();  // staging reads finish before the next half's writes
      }
      if (bad) atomicOr(a.err, DEV_ERR_RANGE);
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
  const cudaError_t e = cudaFuncSetAttribute(k_attn_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_attn_tc_long, cudaFuncAttributeMaxDynamicSharedMemorySize, lt::SMEM_BYTES);
}

cudaError_t launch_attention_tc(const CUtensorMap& tm_q, const CUtensorMap& tm_kv, const CUtensorMap& tm_kv32,
                                const CUtensorMap& tm_kv64, const CUtensorMap& tm_pool, const AttnTcArgs& a,
                                int num_sms, cudaStream_t st) {
  if (a.n_units <= 0) return cudaSuccess;
  const int grid = a.n_units < num_sms ? a.n_units : num_sms;
  k_attn_tc<<<grid, THREADS, SMEM_BYTES, st>>>(tm_q, tm_kv, tm_kv32, tm_kv64, tm_pool, a);
  return cudaGetLastError();
}

cudaError_t launch_attention_tc_long(const CUtensorMap& tm_q, const CUtensorMap& tm_kv, const CUtensorMap& tm_kv32,
                                     const CUtensorMap& tm_kv64, const CUtensorMap& tm_pool, const AttnTcArgs& a,
                                     int num_sms, cudaStream_t st) {
  if (a.n_units <= 0) return cudaSuccess;
  const int grid = a.n_units < num_sms ? a.n_units : num_sms;
  k_attn_tc_long<<<grid, lt::THREADS, lt::SMEM_BYTES, st>>>(tm_q, tm_kv, tm_kv32, tm_kv64, tm_pool, a);
  return cudaGetLastError();
}

}  // namespace dopr
