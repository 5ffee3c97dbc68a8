// k_gemm.cu -- dense projections of the decoder (QKV, O, gate/up, down) on
// the 5th-generation tensor cores: C[M][N] = A[M][K] * B[N][K]^T, fp16
// operands, fp32 accumulate in tensor memory, fused epilogues.
//
// Design (sm_103a, CTA pairs, persistent): a cluster of two CTAs on two SMs
// computes one 256 x 256 output tile with tcgen05 cta_group::2 MMAs (M = 256,
// N = 256, K = 16).  Each CTA stages its own 128 rows of A and its own 128 of
// the tile's 256 B rows per 64-wide k-block (32 KiB a stage, 6-stage ring,
// 128-byte swizzle); the MMAs read both CTAs' shared memory, so per SM a
// third less operand data moves into shared memory and out of it into the
// tensor core per FLOP than with a 128 x 256 tile on one SM.  Roles:
//   warp 0      (both CTAs) TMA producer; the copies of both CTAs complete on
//               the leader's full barrier of the stage;
//   warp 1      allocates 512 TMEM columns in both CTAs (two accumulators of
//               256 columns); in the leader one thread issues the MMAs and
//               commits stage releases and accumulator-ready barriers to both
//               CTAs (multicast);
//   warps 2..9  (both CTAs) epilogue on the CTA's 128 rows of the tile:
//               tcgen05.ld the finished accumulator (one TMEM lane quarter =
//               32 rows per warp, one row per thread; two warps per quarter,
//               each taking half of the tile's 256 columns), apply the
//               epilogue in that row-per-thread layout, then transpose 32x32-
//               word chunks through padded shared memory so every global
//               access is a 128-byte row segment written by 8 consecutive
//               lanes; finally tell the leader the accumulator is free, so the
//               next tile's MMAs overlap the epilogue.
// Tiles are visited in L2 groups (pair_tile_order): blocks of activation rows (up to
// 48 MiB: 4,096 rows at K = 4,096) that stay in L2 while the weight tiles stream past
// them, or, for the residual-epilogue launches, blocks of weight columns while the
// activations stream.  Groups of 2,048 activation rows at every K streamed the weights
// twice as often from HBM (gate/up: 3.5 GB read per 26,800-row launch instead of 1.9),
// and under the power cap that traffic cost about 1 % of SM clock and throughput.
//
// Fused epilogues (the decoder's RMSNorms live here, not in separate kernels):
//   RMSNorm(r) * g = rs * (r (.) g) with rs = rsqrt(mean(r^2) + eps).  The
//   residual-add epilogue writes r' = r + C, the next GEMM's operand
//   f16(r' (.) g_next * rs_pre) -- rs_pre is the row's previous norm factor,
//   which keeps the operand near unit scale -- and, per row and 256-column
//   tile, the partial sum of r'^2.  The consuming GEMM sums those partials
//   (in a fixed order) and scales its accumulator rows by rs / rs_pre.
//   QKV epilogue: row scale, then per 128-column q/k head RMSNorm with the
//   q/k gain and rotate-half RoPE at the token's position (pairs i, i+64),
//   the rotation applied in the transposed layout so RoPE-table reads coalesce.
//   SwiGLU epilogue: silu(rs * gate) * (rs * up).
//   Every value written as fp16 is checked against fp16's range (DEV_ERR_RANGE).
// Every barrier wait is bounded (DEV_ERR_TIMEOUT) and the kernel always drains
// its own MMAs and frees TMEM before returning.
#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int BM = GEMM_BM, BN = GEMM_BN, BK = GEMM_BK;  // BM: one CTA's rows of a pair tile
static_assert(GEMM_B_BOX == BM, "each CTA of a pair stages 128 of a tile's 256 B rows");
constexpr int A_BYTES = BM * BK * 2;  // 16 KiB
constexpr int THREADS = 320;
constexpr int EPI_WARPS = 8;
constexpr int XPOSE_WORDS = 32 * 33;  // per epilogue warp: 32 rows x 32 words, padded row stride 33
constexpr int XPOSE_BYTES = EPI_WARPS * XPOSE_WORDS * 4;
constexpr int BAR_BYTES = 256;

// silu(x) = x / (1 + e^-x) with the fast division (within 2 ulp of fp32, far below the fp16
// rounding of the output; tends to 0 as x -> -inf): the exact division's instruction
// sequence made the SwiGLU epilogue outlast short main loops (K = 1,024).
__device__ __forceinline__ float silu_f(float x) { return __fdividef(x, 1.0f + __expf(-x)); }

// RMSNorm factor of a row from its partial sums of squares, added in index
// order.  When the count allows, the partials arrive as independent 16-byte
// loads (up to 32 in flight) instead of one dependent load per partial.
__device__ __forceinline__ float norm_factor(const float* ss, int parts, const GemmParams& p, int row) {
  if (!ss) return 1.f;
  const float* s = ss + static_cast<int64_t>(min(row, p.M - 1)) * parts;
  float t = 0.f;
  if ((parts & 3) == 0) {
    for (int i = 0; i < parts; i += 32) {
      float4 v[8];
#pragma unroll
      for (int q = 0; q < 8; ++q)
        v[q] = i + 4 * q < parts ? __ldg(reinterpret_cast<const float4*>(s + i) + q) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int q = 0; q < 8; ++q)
        if (i + 4 * q < parts) {
          t += v[q].x;
          t += v[q].y;
          t += v[q].z;
          t += v[q].w;
        }
    }
  } else {
    for (int i = 0; i < parts; ++i) t += s[i];
  }
  return rsqrtf(t / static_cast<float>(p.norm_dim) + p.eps);
}
// Consumer-side row scale: the operand was written as r * g * rs(ss_pre).
__device__ __forceinline__ float row_scale(const GemmParams& p, int row) {
  return norm_factor(p.ss_in, p.ss_parts, p, row) / norm_factor(p.ss_pre, p.ss_pre_parts, p, row);
}

// The warp's 32 rows x 32 words sit in `xs` (row-per-lane layout, stride 33).
// Write them out transposed: lane L covers rows i*4 + L/8 (i = 0..7) and words
// (L%8)*4 .. +3, i.e. 8 lanes per 128-byte row segment.  Word w of row r goes to
// dst_lo(r) + w for w < 16 and to dst_hi(r) + (w - 16) for w >= 16 (two 64-byte
// segments; for one contiguous 128-byte segment pass dst_hi = dst_lo + 16).
template <typename RowPtr>
__device__ __forceinline__ void store_words_transposed(const uint32_t* xs, int lane, int row0, int M, RowPtr dst) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = i * 4 + (lane >> 3);
    const int w = (lane & 7) * 4;
    if (row0 + r < M) {
      uint4 v;
      v.x = xs[r * 33 + w + 0];
      v.y = xs[r * 33 + w + 1];
      v.z = xs[r * 33 + w + 2];
      v.w = xs[r * 33 + w + 3];
      *reinterpret_cast<uint4*>(dst(r, w)) = v;
    }
  }
}

// What an epilogue reads that does not depend on the accumulator: fetched while
// the tile's main loop still runs, so its load latency is off the epilogue's path.
struct EpiPre {
  float scale;  // this thread's row: the consumer row scale (QKV, SwiGLU) or the previous norm factor
  int pos[8];   // QKV: positions of the 8 rows a lane rotates in the transposed layout
};

template <int EPI>
__device__ __forceinline__ void epilogue_prefetch(const GemmParams& p, int mb, int nb, int quarter, int part,
                                                  int lane, EpiPre& pre) {
  const int row0 = mb * BM + quarter * 32;
  if constexpr (EPI == EPI_RESID_ADD) {
    pre.scale = p.xn_out ? norm_factor(p.ss_pre, p.ss_pre_parts, p, row0 + lane) : 1.f;
  } else if constexpr (EPI == EPI_STORE) {
    pre.scale = 1.f;
  } else {
    pre.scale = row_scale(p, row0 + lane);
  }
  if constexpr (EPI == EPI_QKV) {
    if (nb * BN + part * 128 < p.q_cols + p.k_cols)
#pragma unroll
      for (int i = 0; i < 8; ++i) pre.pos[i] = p.tok_pos[min(row0 + i * 4 + (lane >> 3), p.M - 1)];
  }
}

template <int EPI>
__device__ __forceinline__ void epilogue_tile(const GemmParams& p, uint32_t taddr, int mb, int nb, int quarter,
                                              int part, int lane, uint32_t* xs, const EpiPre& pre) {
  const int row0 = mb * BM + quarter * 32;  // first row of this warp; lane = row - row0 = TMEM lane
  bool bad = false;  // a value written as fp16 is not finite or beyond 65504 (reported once per tile)
  // this lane's row exists (rows past M hold whatever the operand buffers held there; never stored)
  const bool live = row0 + lane < p.M;
  if constexpr (EPI == EPI_STORE || EPI == EPI_QKV) {
    f16* out = reinterpret_cast<f16*>(p.out);
    const float rs = pre.scale;
    {
      const int hh = part;                 // this warp's 128-column head of the tile
      const int hc = nb * BN + hh * 128;  // first output column of this head
      const bool rope = (EPI == EPI_QKV) && hc < p.q_cols + p.k_cols;
      if (rope) {
        // per-head RMSNorm of the row-scaled values: sum of squares in the row layout
        float ss = 0.f;
#pragma unroll 1
        for (int c = 0; c < 128; c += 32) {
          uint32_t v[32];
          tmem_ld32(taddr + hh * 128 + c, v);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; ++j) ss += __uint_as_float(v[j]) * __uint_as_float(v[j]);
        }
        const float inv_row = rs * rsqrtf(ss * rs * rs * (1.f / 128.f) + p.eps);
        const bf16* wgt = hc < p.q_cols ? p.q_norm : p.k_norm;
        // the rotation runs in the transposed layout: lane L owns rows i*4 + L/8 and
        // columns w4 .. w4+3 of each 32-column chunk, so RoPE-table reads and the
        // stores are contiguous 8-lane row segments
        const int w4 = (lane & 7) * 4;
        float inv_i[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) inv_i[i] = __shfl_sync(0xffffffffu, inv_row, i * 4 + (lane >> 3));
#pragma unroll 1
        for (int c = 0; c < 64; c += 32) {
          // the rows' (cos, sin) for frequencies c+w4 .. +3 (rows past M read position
          // 0's entries and are not stored), ahead of the accumulator reads below
          float4 c01[8], c23[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float4* cs = reinterpret_cast<const float4*>(p.rope + static_cast<int64_t>(pre.pos[i]) * 64 + c + w4);
            c01[i] = cs[0];
            c23[i] = cs[1];
          }
          float g1[4], g2[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            g1[k] = __bfloat162float(wgt[c + w4 + k]);
            g2[k] = __bfloat162float(wgt[64 + c + w4 + k]);
          }
          float4 x1[8], x2[8];
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            uint32_t v[32];
            tmem_ld32(taddr + hh * 128 + half * 64 + c, v);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 32; ++j) xs[lane * 33 + j] = v[j];
            __syncwarp();
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const int r = i * 4 + (lane >> 3);
              const float4 t = make_float4(__uint_as_float(xs[r * 33 + w4]), __uint_as_float(xs[r * 33 + w4 + 1]),
                                           __uint_as_float(xs[r * 33 + w4 + 2]), __uint_as_float(xs[r * 33 + w4 + 3]));
              if (half == 0)
                x1[i] = t;
              else
                x2[i] = t;
            }
            __syncwarp();
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int r = i * 4 + (lane >> 3);
            if (row0 + r < p.M) {
              const float cosv[4] = {c01[i].x, c01[i].z, c23[i].x, c23[i].z};
              const float sinv[4] = {c01[i].y, c01[i].w, c23[i].y, c23[i].w};
              const float a[4] = {x1[i].x, x1[i].y, x1[i].z, x1[i].w}, b[4] = {x2[i].x, x2[i].y, x2[i].z, x2[i].w};
              float y1[4], y2[4];
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const float u = a[k] * inv_i[i] * g1[k], w = b[k] * inv_i[i] * g2[k];
                y1[k] = u * cosv[k] - w * sinv[k];
                y2[k] = w * cosv[k] + u * sinv[k];
                bad |= !(fp16_ok(y1[k]) && fp16_ok(y2[k]));
              }
              f16* orow = out + static_cast<int64_t>(row0 + r) * p.ld_out + hc + c + w4;
              *reinterpret_cast<uint2*>(orow) = make_uint2(pack_f16x2(y1[0], y1[1]), pack_f16x2(y1[2], y1[3]));
              *reinterpret_cast<uint2*>(orow + 64) = make_uint2(pack_f16x2(y2[0], y2[1]), pack_f16x2(y2[2], y2[3]));
            }
          }
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < 128; c += 64) {
          uint32_t a[32], b[32];
          tmem_ld32(taddr + hh * 128 + c, a);
          tmem_ld32(taddr + hh * 128 + c + 32, b);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            const float a0 = __uint_as_float(a[j]) * rs, a1 = __uint_as_float(a[j + 1]) * rs;
            const float b0 = __uint_as_float(b[j]) * rs, b1 = __uint_as_float(b[j + 1]) * rs;
            bad |= live && !(fp16_ok(a0) && fp16_ok(a1) && fp16_ok(b0) && fp16_ok(b1));
            xs[lane * 33 + j / 2] = pack_f16x2(a0, a1);
            xs[lane * 33 + 16 + j / 2] = pack_f16x2(b0, b1);
          }
          __syncwarp();
          store_words_transposed(xs, lane, row0, p.M, [&](int r, int wd) {
            return out + static_cast<int64_t>(row0 + r) * p.ld_out + hc + c + 2 * wd;
          });
          __syncwarp();
        }
      }
    }
  } else if constexpr (EPI == EPI_RESID_ADD) {
    // r += C, then (optionally) the next RMSNorm's operand f16(r * g * rs_pre) and partial sums of r^2.
    // Lane L owns rows i*4 + L/8 (i = 0..7) and columns (L%8)*4..+3 of each 32-column chunk; the
    // residual values of chunk c+1 are loaded while chunk c is processed.
    float* res = reinterpret_cast<float*>(p.out);
    const int w4 = (lane & 7) * 4;
    float ss[8], prev[8];
    // each lane fetched its own row's previous norm factor; the row layout below takes them by shuffle
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      ss[i] = 0.f;
      prev[i] = __shfl_sync(0xffffffffu, pre.scale, i * 4 + (lane >> 3));
    }
    auto rrow = [&](int i, int c) {
      return reinterpret_cast<float4*>(res + static_cast<int64_t>(row0 + i * 4 + (lane >> 3)) * p.ld_out + nb * BN +
                                       c + w4);
    };
    const int cbeg = part * (BN / 2), cend = cbeg + BN / 2;  // this warp's half of the columns
    float4 cur[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
      cur[i] = (row0 + i * 4 + (lane >> 3) < p.M) ? *rrow(i, cbeg) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
    for (int c = cbeg; c < cend; c += 32) {
      float4 nxt[8];
#pragma unroll
      for (int i = 0; i < 8; ++i)
        nxt[i] = (c + 32 < cend && row0 + i * 4 + (lane >> 3) < p.M) ? *rrow(i, c + 32)
                                                                      : make_float4(0.f, 0.f, 0.f, 0.f);
      uint32_t v[32];
      tmem_ld32(taddr + c, v);
      tmem_ld_wait();
#pragma unroll
      for (int j = 0; j < 32; ++j) xs[lane * 33 + j] = v[j];
      __syncwarp();
      const int col = nb * BN + c + w4;
      float4 g4 = make_float4(0.f, 0.f, 0.f, 0.f);
      if (p.xn_out) {
        const uint2 gw = *reinterpret_cast<const uint2*>(p.xn_gain + col);
        const float2 g01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&gw.x));
        const float2 g23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&gw.y));
        g4 = make_float4(g01.x, g01.y, g23.x, g23.y);
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int r = i * 4 + (lane >> 3);
        if (row0 + r < p.M) {
          float4 x = cur[i];
          x.x += __uint_as_float(xs[r * 33 + w4 + 0]);
          x.y += __uint_as_float(xs[r * 33 + w4 + 1]);
          x.z += __uint_as_float(xs[r * 33 + w4 + 2]);
          x.w += __uint_as_float(xs[r * 33 + w4 + 3]);
          *rrow(i, c) = x;
          if (p.xn_out) {
            ss[i] += x.x * x.x + x.y * x.y + x.z * x.z + x.w * x.w;
            const float sc = prev[i];
            const float n0 = x.x * g4.x * sc, n1 = x.y * g4.y * sc, n2 = x.z * g4.z * sc, n3 = x.w * g4.w * sc;
            bad |= !(fp16_ok(n0) && fp16_ok(n1) && fp16_ok(n2) && fp16_ok(n3));
            uint2 o;
            o.x = pack_f16x2(n0, n1);
            o.y = pack_f16x2(n2, n3);
            *reinterpret_cast<uint2*>(p.xn_out + static_cast<int64_t>(row0 + r) * p.ld_out + col) = o;
          }
        }
        cur[i] = nxt[i];
      }
      __syncwarp();
    }
    if (p.ss_out) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float t = ss[i];
        t += __shfl_xor_sync(0xffffffffu, t, 1);
        t += __shfl_xor_sync(0xffffffffu, t, 2);
        t += __shfl_xor_sync(0xffffffffu, t, 4);
        const int r = i * 4 + (lane >> 3);
        if ((lane & 7) == 0 && row0 + r < p.M)
          p.ss_out[static_cast<int64_t>(row0 + r) * p.ss_out_parts + nb * GEMM_SS_PER_TILE + part] = t;
      }
    }
  } else {  // EPI_SWIGLU: columns 0..127 gate, 128..255 up of the same 128 outputs
    f16* out = reinterpret_cast<f16*>(p.out);
    const float rs = pre.scale;
    {
      const int c = part * 64;  // this warp's 64 of the tile's 128 outputs
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        uint32_t g[32], u[32];
        tmem_ld32(taddr + c + 32 * half, g);
        tmem_ld32(taddr + BN / 2 + c + 32 * half, u);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
          const float a0 = silu_f(__uint_as_float(g[j]) * rs) * (__uint_as_float(u[j]) * rs);
          const float a1 = silu_f(__uint_as_float(g[j + 1]) * rs) * (__uint_as_float(u[j + 1]) * rs);
          bad |= live && !(fp16_ok(a0) && fp16_ok(a1));
          xs[lane * 33 + 16 * half + j / 2] = pack_f16x2(a0, a1);
        }
      }
      __syncwarp();
      store_words_transposed(xs, lane, row0, p.M, [&](int r, int wd) {
        return out + static_cast<int64_t>(row0 + r) * p.ld_out + nb * (BN / 2) + c + 2 * wd;
      });
      __syncwarp();
    }
  }
  report_range(p.err, bad);
}

// ============================================================================
// The pair kernel.  Barriers:
//   full[s]   leader's: armed by the leader for both CTAs' bytes; both CTAs' copies
//             complete on it (the peer addresses it through the cluster window);
//   empty[s]  each CTA's: the leader's commit arrives on both (multicast);
//   tfull[a]  each CTA's: the leader's commit at the end of a tile, multicast;
//   tempty[a] leader's: all 16 epilogue warps of the pair arrive when TMEM is read.
constexpr int PAIR_BM = 2 * BM;                 // rows of a pair tile
constexpr int PAIR_STAGES = 6;
constexpr int PAIR_B_BYTES = BM * BK * 2;       // this CTA's 128 of the tile's 256 B rows: 16 KiB
constexpr int PAIR_STAGE_BYTES = A_BYTES + PAIR_B_BYTES;
constexpr int PAIR_SMEM_BYTES = 1024 + PAIR_STAGES * PAIR_STAGE_BYTES + XPOSE_BYTES + BAR_BYTES;
// L2 tile groups.  A 256-row block of A and a 256-row block of B hold the same bytes
// (256 K 2); a group holds as many blocks as fit GROUP_BYTES (row groups at most 16).
// Row groups keep blocks of A in L2 while B streams past (once per group); column
// groups keep blocks of B while A streams.  Measured DRAM reads per 26,800-row launch
// (row / column groups): QKV 0.76 / 0.78 GB, O 1.31 / 1.07, gate/up 1.95 / 2.74, down
// 3.93 / 3.12: the launches whose epilogue streams the fp32 residual (O, down) keep
// their weight columns better, the others their activation rows.
constexpr int64_t GROUP_BYTES = 48ll << 20;
struct TileOrder {
  int group;   // blocks per group
  bool by_n;   // column groups
};
__device__ __forceinline__ TileOrder pair_tile_order(int n_tiles, int K, bool by_n) {
  const int64_t g = GROUP_BYTES / (static_cast<int64_t>(K) * 2 * 2 * BM);
  const int64_t cap = by_n ? n_tiles : 16;
  return TileOrder{g < 1 ? 1 : g > cap ? static_cast<int>(cap) : static_cast<int>(g), by_n};
}
constexpr uint32_t PAIR_IDESC = umma_idesc_f16(PAIR_BM, BN);
// TMEM columns a pair CTA allocates, and accumulators (256 columns each) it cycles through
constexpr int PAIR_ACCS = 2;
constexpr uint32_t PAIR_TMEM_COLS = PAIR_ACCS * BN;
static_assert(PAIR_SMEM_BYTES <= 227 * 1024, "shared memory budget");

// Tile t of the launch: within a group the grouped operand's blocks vary fastest, so the
// tiles of one wave share the streamed operand's blocks too.
__device__ __forceinline__ void pair_tile_coords(int t, int m_tiles, int n_tiles, TileOrder o, int& mb, int& nb) {
  if (o.by_n) {
    const int group = o.group * m_tiles;
    const int g = t / group;
    const int first_n = g * o.group;
    const int gn = min(o.group, n_tiles - first_n);
    const int r = t - g * group;
    nb = first_n + r % gn;
    mb = r / gn;
  } else {
    const int group = o.group * n_tiles;
    const int g = t / group;
    const int first_m = g * o.group;
    const int gm = min(o.group, m_tiles - first_m);
    const int r = t - g * group;
    mb = first_m + r % gm;
    nb = r / gm;
  }
}

template <int EPI>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
    k_gemm_pair(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + PAIR_STAGES * A_BYTES;
  uint32_t* xpose = reinterpret_cast<uint32_t*>(smem + PAIR_STAGES * PAIR_STAGE_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + PAIR_STAGES * PAIR_STAGE_BYTES + XPOSE_BYTES);
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (PAIR_STAGES + s); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * PAIR_STAGES + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * PAIR_STAGES + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * PAIR_STAGES + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * PAIR_STAGES + 5);
  static_assert((2 * PAIR_STAGES + 5) * 8 + 4 <= BAR_BYTES, "barrier area");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  const int m_tiles = (p.M + PAIR_BM - 1) / PAIR_BM, n_tiles = p.N / BN, k_blocks = p.K / BK;
  const TileOrder order = pair_tile_order(n_tiles, p.K, EPI == EPI_RESID_ADD);
  int total = m_tiles * n_tiles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < PAIR_STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar(a), 1);
      mbar_init(tempty_bar(a), 2 * EPI_WARPS);
    }
    mbar_init(drain_bar, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_slot), PAIR_TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers exist before either addresses the other's
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  {
    // the MMAs write both CTAs' TMEM at the leader's address: both allocations must agree
    uint32_t other;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(other) : "r"(mapa_shared(smem_u32(tmem_slot), rank ^ 1u)));
    if (other != tmem_base) {
      if (threadIdx.x == 0) atomicOr(p.err, DEV_ERR_BOUNDS);
      total = 0;  // no tile runs
    }
  }

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs): own A rows and own half of B's rows
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int t = pair; t < total && ok; t += n_pairs) {
        int mb, nb;
        pair_tile_coords(t, m_tiles, n_tiles, order, mb, nb);
        for (int kb = 0; kb < k_blocks; ++kb) {
          if (!mbar_wait_cluster(empty_bar(stage), phase ^ 1u, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          if (leader) mbar_arrive_expect_tx(full_bar(stage), 2 * PAIR_STAGE_BYTES);
          const uint32_t fb = mapa_shared(full_bar(stage), 0);
          tma_load_2d_pair(sA + stage * A_BYTES, &tmA, fb, kb * BK, mb * PAIR_BM + static_cast<int>(rank) * BM);
          tma_load_2d_pair(sB + stage * PAIR_B_BYTES, &tmB, fb, kb * BK, nb * BN + static_cast<int>(rank) * BM);
          if (++stage == PAIR_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // copies in flight land within microseconds; give them that long before the
        // CTA can reach its exit (no barrier to wait on: they count on the leader's)
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 20000ull) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ---------------- MMA issuer (leader only)
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool ok = true;
      for (int t = pair; t < total && ok; t += n_pairs, ++local) {
        const int acc = local % PAIR_ACCS;
        const uint32_t acc_phase = (local / PAIR_ACCS) & 1;
        if (!mbar_wait_cluster(tempty_bar(acc), acc_phase ^ 1u, p.err, p.timeout_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < k_blocks; ++kb) {
          if (!mbar_wait_cluster(full_bar(stage), phase, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = umma_desc_sw128(sA + stage * A_BYTES);
          const uint64_t bd = umma_desc_sw128(sB + stage * PAIR_B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)  // +32 bytes along K per step, in 16-byte units
            umma_f16_pair(d_tmem, ad + 2 * k, bd + 2 * k, PAIR_IDESC, (kb | k) != 0);
          umma_commit_pair_mc(empty_bar(stage), 3);  // both CTAs' stage is free once these MMAs end
          if (++stage == PAIR_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (ok) umma_commit_pair_mc(tfull_bar(acc), 3);
      }
      // All MMAs this thread issued are complete once drain_bar flips.
      umma_commit_pair_mc(drain_bar, 1);
      mbar_wait(drain_bar, 0, p.err, ok ? p.timeout_ns : 100000000ull);
    }
  } else {
    // ---------------- epilogue warps 2..9 (both CTAs) on this CTA's 128 rows of the tile
    const int quarter = warp & 3;
    const int part = (warp - 2) >> 2;
    uint32_t* xs = xpose + (warp - 2) * XPOSE_WORDS;
    int local = 0;
    for (int t = pair; t < total; t += n_pairs, ++local) {
      int mb2, nb;
      pair_tile_coords(t, m_tiles, n_tiles, order, mb2, nb);
      const int mb = 2 * mb2 + static_cast<int>(rank);  // this CTA's 128-row block
      const int acc = local % PAIR_ACCS;
      const uint32_t acc_phase = (local / PAIR_ACCS) & 1;
      EpiPre pre;
      epilogue_prefetch<EPI>(p, mb, nb, quarter, part, lane, pre);
      if (!mbar_wait_cluster(tfull_bar(acc), acc_phase, p.err, p.timeout_ns)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
      epilogue_tile<EPI>(p, taddr, mb, nb, quarter, part, lane, xs, pre);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(mapa_shared(tempty_bar(acc), 0));
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // neither CTA leaves while the other may still address its barriers or TMEM
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc_pair(tmem_base, PAIR_TMEM_COLS);
  }
}

template <int EPI>
cudaError_t set_smem() {
  return cudaFuncSetAttribute(k_gemm_pair<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, PAIR_SMEM_BYTES);
}

}  // namespace

cudaError_t gemm_setup() {
  cudaError_t e;
  if ((e = set_smem<EPI_STORE>())) return e;
  if ((e = set_smem<EPI_RESID_ADD>())) return e;
  if ((e = set_smem<EPI_SWIGLU>())) return e;
  return set_smem<EPI_QKV>();
}

cudaError_t launch_gemm(int epi, const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmParams& params,
                        int num_sms, cudaStream_t st) {
  if (params.M <= 0) return cudaSuccess;
  GemmParams p = params;
  p.timeout_ns = WAIT_TIMEOUT_NS;
  // one CTA pair per two SMs (persistent), never more pairs than 256-row tiles
  const int tiles = ((p.M + PAIR_BM - 1) / PAIR_BM) * (p.N / BN);
  const int pairs = tiles < num_sms / 2 ? tiles : num_sms / 2;
  const int grid = 2 * (pairs > 0 ? pairs : 1);
  switch (epi) {
    case EPI_STORE:
      k_gemm_pair<EPI_STORE><<<grid, THREADS, PAIR_SMEM_BYTES, st>>>(tmA, tmB, p);
      break;
    case EPI_RESID_ADD:
      k_gemm_pair<EPI_RESID_ADD><<<grid, THREADS, PAIR_SMEM_BYTES, st>>>(tmA, tmB, p);
      break;
    case EPI_SWIGLU:
      k_gemm_pair<EPI_SWIGLU><<<grid, THREADS, PAIR_SMEM_BYTES, st>>>(tmA, tmB, p);
      break;
    default:
      k_gemm_pair<EPI_QKV><<<grid, THREADS, PAIR_SMEM_BYTES, st>>>(tmA, tmB, p);
      break;
  }
  return cudaGetLastError();
}

}  // namespace dopr
