// k_gemm.cu -- dense projections of the decoder (QKV, O, gate/up, down) on
// the 5th-generation tensor cores: C[M][N] = A[M][K] * B[N][K]^T, bf16 in,
// fp32 accumulate in tensor memory, fused epilogues.
//
// Design (sm_103a, one CTA per SM, persistent):
//   warp 0      TMA producer: 128x64 A tile + 256x64 B tile per stage, 128-byte
//               swizzle, 4-stage shared-memory ring guarded by full/empty mbarriers;
//   warp 1      allocates 512 TMEM columns (two 128x256 fp32 accumulators) and one
//               elected thread issues tcgen05.mma (M=128, N=256, K=16) per k-step,
//               committing stage releases and accumulator-ready barriers;
//   warps 2..5  epilogue: tcgen05.ld rows of the finished accumulator (one TMEM lane
//               quarter per warp, one output row per thread), apply the epilogue and
//               store, then release the accumulator so the next tile's MMAs overlap.
// Tiles are visited in groups of 16 M-blocks so the weight tiles a wave reads
// stay in L2 while the activation rows of the group are reused across N.
// Every barrier wait is bounded (DEV_ERR_TIMEOUT) and the kernel always drains
// its own copies and MMAs and frees TMEM before returning.
#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int BM = GEMM_BM, BN = GEMM_BN, BK = GEMM_BK;
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;  // 16 KiB
constexpr int B_BYTES = BN * BK * 2;  // 32 KiB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 2 * BN;     // two accumulators
constexpr int THREADS = 192;
constexpr int GROUP_M = 16;
constexpr int BAR_BYTES = 256;
constexpr int SMEM_BYTES = 1024 /*alignment slack*/ + STAGES * STAGE_BYTES + BAR_BYTES;
constexpr uint32_t IDESC = umma_idesc_bf16(BM, BN);

struct GemmParams {
  int M, N, K;
  void* out;
  int64_t ld_out;
  int* err;
  uint64_t timeout_ns;
};

__device__ __forceinline__ void tile_coords(int t, int m_tiles, int n_tiles, int& mb, int& nb) {
  const int group = GROUP_M * n_tiles;
  const int g = t / group;
  const int first_m = g * GROUP_M;
  const int gm = min(GROUP_M, m_tiles - first_m);
  const int r = t - g * group;
  mb = first_m + r % gm;
  nb = r / gm;
}

__device__ __forceinline__ float silu_f(float x) { return x / (1.0f + __expf(-x)); }

template <int EPI>
__device__ __forceinline__ void epilogue_tile(const GemmParams& p, uint32_t taddr, int row, int nb) {
  const bool in = row < p.M;
  if constexpr (EPI == EPI_STORE_BF16) {
    bf16* dst = reinterpret_cast<bf16*>(p.out) + static_cast<int64_t>(row) * p.ld_out + static_cast<int64_t>(nb) * BN;
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      uint32_t v[32];
      tmem_ld32(taddr + c, v);
      tmem_ld_wait();
      if (in) {
        uint4* d4 = reinterpret_cast<uint4*>(dst + c);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint4 w;
          w.x = pack_bf16x2(__uint_as_float(v[8 * q + 0]), __uint_as_float(v[8 * q + 1]));
          w.y = pack_bf16x2(__uint_as_float(v[8 * q + 2]), __uint_as_float(v[8 * q + 3]));
          w.z = pack_bf16x2(__uint_as_float(v[8 * q + 4]), __uint_as_float(v[8 * q + 5]));
          w.w = pack_bf16x2(__uint_as_float(v[8 * q + 6]), __uint_as_float(v[8 * q + 7]));
          d4[q] = w;
        }
      }
    }
  } else if constexpr (EPI == EPI_RESID_ADD_F32) {
    float* dst = reinterpret_cast<float*>(p.out) + static_cast<int64_t>(row) * p.ld_out + static_cast<int64_t>(nb) * BN;
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      uint32_t v[32];
      tmem_ld32(taddr + c, v);
      tmem_ld_wait();
      if (in) {
        float4* d4 = reinterpret_cast<float4*>(dst + c);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          float4 r = d4[q];
          r.x += __uint_as_float(v[4 * q + 0]);
          r.y += __uint_as_float(v[4 * q + 1]);
          r.z += __uint_as_float(v[4 * q + 2]);
          r.w += __uint_as_float(v[4 * q + 3]);
          d4[q] = r;
        }
      }
    }
  } else {  // EPI_SWIGLU_BF16: columns 0..127 gate, 128..255 up of the same 128 outputs
    bf16* dst = reinterpret_cast<bf16*>(p.out) + static_cast<int64_t>(row) * p.ld_out +
                static_cast<int64_t>(nb) * (BN / 2);
#pragma unroll 1
    for (int c = 0; c < BN / 2; c += 32) {
      uint32_t g[32], u[32];
      tmem_ld32(taddr + c, g);
      tmem_ld32(taddr + BN / 2 + c, u);
      tmem_ld_wait();
      if (in) {
        uint4* d4 = reinterpret_cast<uint4*>(dst + c);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float a[8];
#pragma unroll
          for (int e = 0; e < 8; ++e)
            a[e] = silu_f(__uint_as_float(g[8 * q + e])) * __uint_as_float(u[8 * q + e]);
          uint4 w;
          w.x = pack_bf16x2(a[0], a[1]);
          w.y = pack_bf16x2(a[2], a[3]);
          w.z = pack_bf16x2(a[4], a[5]);
          w.w = pack_bf16x2(a[6], a[7]);
          d4[q] = w;
        }
      }
    }
  }
}

template <int EPI>
__global__ void __launch_bounds__(THREADS, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + STAGES * A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 5);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m_tiles = (p.M + BM - 1) / BM, n_tiles = p.N / BN, k_blocks = p.K / BK;
  const int total = m_tiles * n_tiles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar(a), 1);
      mbar_init(tempty_bar(a), 4);
    }
    mbar_init(drain_bar, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, issued_par = 0;  // per stage: ever armed / parity of last arm
      bool ok = true;
      for (int t = blockIdx.x; t < total && ok; t += gridDim.x) {
        int mb, nb;
        tile_coords(t, m_tiles, n_tiles, mb, nb);
        for (int kb = 0; kb < k_blocks; ++kb) {
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full_bar(stage), STAGE_BYTES);
          tma_load_2d(sA + stage * A_BYTES, &tmA, full_bar(stage), kb * BK, mb * BM);
          tma_load_2d(sB + stage * B_BYTES, &tmB, full_bar(stage), kb * BK, nb * BN);
          issued |= 1u << stage;
          issued_par = (issued_par & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // Let every copy this thread started land before the CTA can exit.
        for (int s = 0; s < STAGES; ++s)
          if (issued & (1u << s)) mbar_wait(full_bar(s), (issued_par >> s) & 1u, p.err, 100000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      int stage = 0;
      uint32_t phase = 0;
      int local = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < total && ok; t += gridDim.x, ++local) {
        const int acc = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, p.err, p.timeout_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < k_blocks; ++kb) {
          if (!mbar_wait(full_bar(stage), phase, p.err, p.timeout_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = umma_desc_sw128(sA + stage * A_BYTES);
          const uint64_t bd = umma_desc_sw128(sB + stage * B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)  // +32 bytes along K per step, in 16-byte units
            umma_bf16(d_tmem, ad + 2 * k, bd + 2 * k, IDESC, (kb | k) != 0);
          umma_commit(empty_bar(stage));
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (ok) umma_commit(tfull_bar(acc));
      }
      // All MMAs this thread issued are complete once drain_bar flips.
      umma_commit(drain_bar);
      mbar_wait(drain_bar, 0, p.err, ok ? p.timeout_ns : 100000000ull);
    }
  } else {
    // ---------------- epilogue warps 2..5 -> TMEM lane quarters 2,3,0,1
    const int quarter = warp & 3;
    int local = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x, ++local) {
      int mb, nb;
      tile_coords(t, m_tiles, n_tiles, mb, nb);
      const int acc = local & 1;
      const uint32_t acc_phase = (local >> 1) & 1;
      if (!mbar_wait(tfull_bar(acc), acc_phase, p.err, p.timeout_ns)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
      const int row = mb * BM + quarter * 32 + lane;
      epilogue_tile<EPI>(p, taddr, row, nb);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty_bar(acc));
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

}  // namespace

cudaError_t gemm_setup() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(k_gemm_tc<EPI_STORE_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES)))
    return e;
  if ((e = cudaFuncSetAttribute(k_gemm_tc<EPI_RESID_ADD_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SMEM_BYTES)))
    return e;
  return cudaFuncSetAttribute(k_gemm_tc<EPI_SWIGLU_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
}

cudaError_t launch_gemm(int epi, const CUtensorMap& tmA, const CUtensorMap& tmB, int M, int N, int K, void* out,
                        int64_t ld_out, int* err, int num_sms, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  GemmParams p{M, N, K, out, ld_out, err, WAIT_TIMEOUT_NS};
  const int tiles = ((M + BM - 1) / BM) * (N / BN);
  const int grid = tiles < num_sms ? tiles : num_sms;
  switch (epi) {
    case EPI_STORE_BF16:
      k_gemm_tc<EPI_STORE_BF16><<<grid, THREADS, SMEM_BYTES, st>>>(tmA, tmB, p);
      break;
    case EPI_RESID_ADD_F32:
      k_gemm_tc<EPI_RESID_ADD_F32><<<grid, THREADS, SMEM_BYTES, st>>>(tmA, tmB, p);
      break;
    default:
      k_gemm_tc<EPI_SWIGLU_BF16><<<grid, THREADS, SMEM_BYTES, st>>>(tmA, tmB, p);
      break;
  }
  return cudaGetLastError();
}

}  // namespace dopr
