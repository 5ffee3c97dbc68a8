// k_attn.cu -- prefix-plus-causal grouped-query attention of the online pass
// (DoPR Sec. 3.4: the online tokens [q ; t_score] attend to the document's
// stored prefix keys/values, then causally to their own keys).
//
// One CTA per (work item, kv head).  A work item is a run of consecutive
// sorted pairs that share one document, so the CTA stages that document's
// prefix K and V for its kv head (m x 128 bf16 each) into shared memory ONCE
// with TMA (128-byte swizzle) and reuses it for every query row of every pair
// in the run.  Rows are (token j, q head of the group) with the G q heads of
// one kv head interleaved, so a 16-row warp tile covers 16/G tokens x G heads.
// Per 64-row block the warps sweep the prefix blocks, then stream the pair's
// own keys 0..j in 64-key chunks (cp.async, zero-filled past the end).
// Scores and P.V use warp-level fp16 mma with fp32 accumulation (the stored
// bf16 prefix is widened to fp16 in shared memory after it lands); the softmax
// is the online (running max / running sum) form with quad shuffles.
#include <math.h>

#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int WARPS = 4;
constexpr int THREADS = WARPS * 32;
constexpr int ROWS = WARPS * 16;   // rows per row block
constexpr int KEYS = 64;           // keys per block
constexpr int ROW_BYTES = HEAD_DIM * 2;
constexpr int BOX_BYTES = 64 * 128;      // TMA box: 64 rows x 64 elements
constexpr int OWN_BYTES = KEYS * ROW_BYTES;  // own K (or V) chunk
constexpr int Q_BYTES = 16 * ROW_BYTES;      // per-warp Q tile

// Byte offset of (row r, 16-byte chunk c) in a tile of 64-row boxes, each box
// split into two 64-element halves, 128-byte swizzled (what TMA writes).
__device__ __forceinline__ uint32_t off64(int r, int c) {
  return static_cast<uint32_t>((((r >> 6) * 2 + (c >> 3)) * 64 + (r & 63)) * 128 + (((c & 7) ^ (r & 7)) << 4));
}
// Same layout for a 16-row tile.
__device__ __forceinline__ uint32_t off16(int r, int c) {
  return static_cast<uint32_t>(((c >> 3) * 16 + r) * 128 + (((c & 7) ^ (r & 7)) << 4));
}

// One 64-key block for one warp's 16 rows.  kbase/vbase point at a 64-row box
// pair of the K and V tiles.  Keys kk >= n_valid are masked; with CAUSAL a key
// kk is visible to a row of token j only if key0 + kk <= j.
template <bool CAUSAL>
__device__ __forceinline__ void attend_block(uint32_t kbase, uint32_t vbase, int lane, const uint32_t (&qf)[8][4],
                                             float (&o)[16][4], float (&mrow)[2], float (&lrow)[2], int n_valid,
                                             int key0, const int (&jr)[2], float scale_log2) {
  float s[8][4];
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
    for (int np = 0; np < 4; ++np) {
      const int key = np * 16 + (lane & 7) + ((lane >> 4) << 3);
      const int c = 2 * ks + ((lane >> 3) & 1);
      uint32_t b0, b1, b2, b3;
      ldmatrix_x4(kbase + off64(key, c), b0, b1, b2, b3);
      mma_f16_16816(s[2 * np], qf[ks], b0, b1);
      mma_f16_16816(s[2 * np + 1], qf[ks], b2, b3);
    }
  }
  float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
  for (int nt = 0; nt < 8; ++nt)
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
    const float mnew = fmaxf(mrow[i], mx[i]);
    base[i] = (mnew == -INFINITY) ? 0.f : mnew;
    alpha[i] = exp2f(mrow[i] - base[i]);
    mrow[i] = mnew;
  }
  float rs[2] = {0.f, 0.f};
#pragma unroll
  for (int nt = 0; nt < 8; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float p = exp2f(s[nt][e] - base[e >> 1]);
      s[nt][e] = p;
      rs[e >> 1] += p;
    }
  lrow[0] = lrow[0] * alpha[0] + rs[0];
  lrow[1] = lrow[1] * alpha[1] + rs[1];
#pragma unroll
  for (int dt = 0; dt < 16; ++dt) {
    o[dt][0] *= alpha[0];
    o[dt][1] *= alpha[0];
    o[dt][2] *= alpha[1];
    o[dt][3] *= alpha[1];
  }
#pragma unroll
  for (int kk = 0; kk < 4; ++kk) {
    uint32_t a[4];
    a[0] = pack_f16x2(s[2 * kk][0], s[2 * kk][1]);
    a[1] = pack_f16x2(s[2 * kk][2], s[2 * kk][3]);
    a[2] = pack_f16x2(s[2 * kk + 1][0], s[2 * kk + 1][1]);
    a[3] = pack_f16x2(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
    for (int dp = 0; dp < 8; ++dp) {
      const int key = kk * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
      const int c = 2 * dp + (lane >> 4);
      uint32_t b0, b1, b2, b3;
      ldmatrix_x4_trans(vbase + off64(key, c), b0, b1, b2, b3);
      mma_f16_16816(o[2 * dp], a, b0, b1);
      mma_f16_16816(o[2 * dp + 1], a, b2, b3);
    }
  }
}

__global__ void __launch_bounds__(THREADS) k_attn(const __grid_constant__ CUtensorMap tm_pool, AttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sPK = smem_u32(smem);
  const uint32_t sPV = sPK + a.mpad_cap * ROW_BYTES;
  const uint32_t sOK = sPV + a.mpad_cap * ROW_BYTES;
  const uint32_t sOV = sOK + OWN_BYTES;
  const uint32_t sQ0 = sOV + OWN_BYTES;
  const uint32_t bar = sQ0 + WARPS * Q_BYTES;

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
    // The stored prefix is bf16: widen it to fp16 in place (element-wise, so the
    // swizzled layout is unchanged).  Rows m .. nbox*64-1 of the boxes hold other
    // data: zero them so masked keys contribute exactly 0 to P.V.
    uint8_t* gk = smem;
    uint8_t* gv = smem + a.mpad_cap * ROW_BYTES;
    for (int i = tid; i < nbox * 64 * 16; i += THREADS) {
      const int r = i / 16, c = i % 16;
      uint4* pk = reinterpret_cast<uint4*>(gk + off64(r, c));
      uint4* pv = reinterpret_cast<uint4*>(gv + off64(r, c));
      if (r >= m) {
        *pk = make_uint4(0, 0, 0, 0);
        *pv = make_uint4(0, 0, 0, 0);
      } else {
        uint4 x = *pk, y = *pv;
        x = make_uint4(bf16x2_to_f16x2(x.x), bf16x2_to_f16x2(x.y), bf16x2_to_f16x2(x.z), bf16x2_to_f16x2(x.w));
        y = make_uint4(bf16x2_to_f16x2(y.x), bf16x2_to_f16x2(y.y), bf16x2_to_f16x2(y.z), bf16x2_to_f16x2(y.w));
        *pk = x;
        *pv = y;
      }
    }
    __syncthreads();
  }

  const f16* qkv = a.qkv;
  const int ld = a.ld_qkv;
  const int kcol = (a.Hq + g) * HEAD_DIM;
  const int vcol = (a.Hq + a.Hkv + g) * HEAD_DIM;
  const uint32_t sQ = sQ0 + warp * Q_BYTES;

  for (int s = item.pair_begin; s < item.pair_end; ++s) {
    const int tb = a.tok_off[s] - a.tok0;          // first row of the pair in this chunk
    const int T = a.tok_off[s + 1] - a.tok_off[s];  // query tokens + score token
    const int R = T * G;
    const int rbeg = a.score_only ? (T - 1) * G : 0;  // score-only: just the score token's G rows
    for (int rb = 0; rbeg + rb * ROWS < R; ++rb) {
      const int row0 = rbeg + rb * ROWS + warp * 16;
      const bool active = row0 < R;
      const int jmax = min(T - 1, (rbeg + rb * ROWS + ROWS - 1) / G);
      // ---- Q tile of this warp (16 rows; rows >= R zero-filled)
      if (active) {
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int idx = lane + i * 32, r = idx >> 4, c = idx & 15;
          const int row = row0 + r;
          const bool ok = row < R;
          const int j = ok ? row / G : 0, hh = ok ? row % G : 0;
          const f16* src = qkv + static_cast<int64_t>(tb + j) * ld + (g * G + hh) * HEAD_DIM + c * 8;
          cp_async16(sQ + off16(r, c), src, ok);
        }
      }
      cp_async_commit();
      cp_async_wait_all();
      __syncwarp();
      uint32_t qf[8][4];
      float o[16][4];
      float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
      int jr[2];
      {
        const int r0 = row0 + (lane >> 2);
        jr[0] = r0 / G;
        jr[1] = (r0 + 8) / G;
      }
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) o[dt][0] = o[dt][1] = o[dt][2] = o[dt][3] = 0.f;
      if (active) {
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const int r = (lane & 7) + (((lane >> 3) & 1) << 3);
          const int c = 2 * ks + (lane >> 4);
          ldmatrix_x4(sQ + off16(r, c), qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3]);
        }
        // ---- prefix keys: visible to every online token
        for (int kb = 0; kb < nbox; ++kb)
          attend_block<false>(sPK + kb * 2 * BOX_BYTES, sPV + kb * 2 * BOX_BYTES, lane, qf, o, mrow, lrow,
                              min(KEYS, m - kb * KEYS), 0, jr, scale_log2);
      }
      // ---- own keys 0..jmax in chunks of 64, causal
      for (int c0 = 0; c0 <= jmax; c0 += KEYS) {
        __syncthreads();  // previous chunk fully consumed
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int idx = tid + i * THREADS;  // 0 .. 2047
          const int kv = idx >> 10, rem = idx & 1023, key = rem >> 4, c = rem & 15;
          const bool ok = c0 + key <= jmax;
          const int row = tb + (ok ? c0 + key : 0);
          const f16* src = qkv + static_cast<int64_t>(row) * ld + (kv ? vcol : kcol) + c * 8;
          cp_async16((kv ? sOV : sOK) + off64(key, c), src, ok);
        }
        cp_async_commit();
        cp_async_wait_all();
        __syncthreads();
        if (active)
          attend_block<true>(sOK, sOV, lane, qf, o, mrow, lrow, min(KEYS, jmax + 1 - c0), c0, jr, scale_log2);
      }
      // ---- normalise and store rows < R
      if (active) {
        float l0 = lrow[0], l1 = lrow[1];
        l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
        l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
        const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f, inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
        for (int hr = 0; hr < 2; ++hr) {
          const int row = row0 + (lane >> 2) + hr * 8;
          if (row < R) {
            const int j = row / G, hh = row % G;
            const int orow = a.score_only ? s - a.pair_base : tb + j;  // compact rows in score-only mode
            f16* dst = a.out + static_cast<int64_t>(orow) * a.ld_out + (g * G + hh) * HEAD_DIM + (lane & 3) * 2;
            const float inv = hr ? inv1 : inv0;
#pragma unroll
            for (int dt = 0; dt < 16; ++dt)
              *reinterpret_cast<uint32_t*>(dst + dt * 8) = pack_f16x2(o[dt][2 * hr] * inv, o[dt][2 * hr + 1] * inv);
          }
        }
      }
    }
  }
}

inline size_t attn_smem_bytes(int mpad_cap) {
  return 1024 + 2 * static_cast<size_t>(mpad_cap) * ROW_BYTES + 2 * OWN_BYTES + WARPS * Q_BYTES + 64;
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
