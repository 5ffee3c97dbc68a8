// k_rows.cu -- the memory-bound per-row kernels of the decoder pass:
//   embedding gather + input RMSNorm (first layer), RMSNorm of the fp32
//   residual stream, per-head RMSNorm + RoPE of q and k (positions m + j),
//   the two-row score head, and the prefix-store layout transpose.
// One warp per row (or per head vector); 16-byte vector accesses.
#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int ROW_WARPS = 8;  // warps per block for row kernels

// x = r * rsqrt(mean(r^2) + eps) * g for one row held in global memory; the
// row is read twice (second read hits L1/L2).
__device__ __forceinline__ void norm_row_store(const float* r, int H, const bf16* g, float eps, bf16* out, int lane) {
  float ss = 0.f;
  for (int c = lane * 4; c < H; c += 128) {
    const float4 v = *reinterpret_cast<const float4*>(r + c);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / static_cast<float>(H) + eps);
  for (int c = lane * 8; c < H; c += 256) {
    const float4 a = *reinterpret_cast<const float4*>(r + c);
    const float4 b = *reinterpret_cast<const float4*>(r + c + 4);
    const uint4 gw = *reinterpret_cast<const uint4*>(g + c);
    const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&gw);
    const float2 g0 = __bfloat1622float2(g2[0]), g1 = __bfloat1622float2(g2[1]);
    const float2 g2f = __bfloat1622float2(g2[2]), g3 = __bfloat1622float2(g2[3]);
    uint4 o;
    o.x = pack_bf16x2(a.x * inv * g0.x, a.y * inv * g0.y);
    o.y = pack_bf16x2(a.z * inv * g1.x, a.w * inv * g1.y);
    o.z = pack_bf16x2(b.x * inv * g2f.x, b.y * inv * g2f.y);
    o.w = pack_bf16x2(b.z * inv * g3.x, b.w * inv * g3.y);
    *reinterpret_cast<uint4*>(out + c) = o;
  }
}

__global__ void __launch_bounds__(ROW_WARPS * 32)
    k_embed_norm(const int32_t* __restrict__ tok_id, int T, const bf16* __restrict__ embed,
                 const bf16* __restrict__ gain, int H, float eps, float* __restrict__ r, bf16* __restrict__ xn) {
  const int row = blockIdx.x * ROW_WARPS + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= T) return;
  const bf16* e = embed + static_cast<int64_t>(tok_id[row]) * H;
  float* rr = r + static_cast<int64_t>(row) * H;
  for (int c = lane * 8; c < H; c += 256) {
    const uint4 w = *reinterpret_cast<const uint4*>(e + c);
    const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&w);
    const float2 a = __bfloat1622float2(w2[0]), b = __bfloat1622float2(w2[1]);
    const float2 cc = __bfloat1622float2(w2[2]), d = __bfloat1622float2(w2[3]);
    *reinterpret_cast<float4*>(rr + c) = make_float4(a.x, a.y, b.x, b.y);
    *reinterpret_cast<float4*>(rr + c + 4) = make_float4(cc.x, cc.y, d.x, d.y);
  }
  __syncwarp();
  norm_row_store(rr, H, gain, eps, xn + static_cast<int64_t>(row) * H, lane);
}

__global__ void __launch_bounds__(ROW_WARPS * 32)
    k_rmsnorm(const float* __restrict__ r, int T, int H, const bf16* __restrict__ gain, float eps,
              bf16* __restrict__ xn) {
  const int row = blockIdx.x * ROW_WARPS + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= T) return;
  norm_row_store(r + static_cast<int64_t>(row) * H, H, gain, eps, xn + static_cast<int64_t>(row) * H, lane);
}

// One warp per (token, head) vector of 128: lane holds elements 2l, 2l+1 and
// their rotate-half partners 64+2l, 65+2l.
__global__ void __launch_bounds__(ROW_WARPS * 32)
    k_qknorm_rope(bf16* __restrict__ qkv, int T, int ld, int Hq, int Hkv, const bf16* __restrict__ qn,
                  const bf16* __restrict__ kn, const int32_t* __restrict__ tok_pos, const float2* __restrict__ rope,
                  float eps) {
  const int heads = Hq + Hkv;
  const int64_t idx = static_cast<int64_t>(blockIdx.x) * ROW_WARPS + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (idx >= static_cast<int64_t>(T) * heads) return;
  const int t = static_cast<int>(idx / heads), h = static_cast<int>(idx % heads);
  bf16* v = qkv + static_cast<int64_t>(t) * ld + h * HEAD_DIM;  // k heads follow the q heads
  const bf16* w = h < Hq ? qn : kn;
  const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(v + 2 * lane));
  const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(v + 64 + 2 * lane));
  const float ss = warp_sum(x.x * x.x + x.y * x.y + y.x * y.x + y.y * y.y);
  const float inv = rsqrtf(ss * (1.0f / HEAD_DIM) + eps);
  const float2 wx = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(w + 2 * lane));
  const float2 wy = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(w + 64 + 2 * lane));
  const float x0 = x.x * inv * wx.x, x1 = x.y * inv * wx.y;
  const float y0 = y.x * inv * wy.x, y1 = y.y * inv * wy.y;
  const float2* cs = rope + static_cast<int64_t>(tok_pos[t]) * (HEAD_DIM / 2) + 2 * lane;
  const float2 c0 = cs[0], c1 = cs[1];  // (cos, sin) for frequencies 2l and 2l+1
  *reinterpret_cast<uint32_t*>(v + 2 * lane) = pack_bf16x2(x0 * c0.x - y0 * c0.y, x1 * c1.x - y1 * c1.y);
  *reinterpret_cast<uint32_t*>(v + 64 + 2 * lane) = pack_bf16x2(y0 * c0.x + x0 * c0.y, y1 * c1.x + x1 * c1.y);
}

// Score head at the score-token row of each sorted pair in [p_begin, p_end):
// s = <W[0] - W[1], RMSNorm(r_row) * g>, written to scores[perm[pair]].
__global__ void __launch_bounds__(ROW_WARPS * 32)
    k_score(const float* __restrict__ r, int H, const int32_t* __restrict__ tok_off, int tok0, int p_begin, int p_end,
            const int32_t* __restrict__ perm, const bf16* __restrict__ gain, const bf16* __restrict__ head,
            float eps, float* __restrict__ scores) {
  const int s = p_begin + blockIdx.x * ROW_WARPS + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (s >= p_end) return;
  const float* x = r + static_cast<int64_t>(tok_off[s + 1] - 1 - tok0) * H;
  float ss = 0.f;
  for (int c = lane * 4; c < H; c += 128) {
    const float4 v = *reinterpret_cast<const float4*>(x + c);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  const float inv = rsqrtf(warp_sum(ss) / static_cast<float>(H) + eps);
  float yes = 0.f, no = 0.f;
  for (int c = lane * 2; c < H; c += 64) {
    const float2 v = *reinterpret_cast<const float2*>(x + c);
    const float2 g = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(gain + c));
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(head + c));
    const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(head + H + c));
    const float h0 = v.x * inv * g.x, h1 = v.y * inv * g.y;
    yes += h0 * a.x + h1 * a.y;
    no += h0 * b.x + h1 * b.y;
  }
  yes = warp_sum(yes);
  no = warp_sum(no);
  if (lane == 0) scores[perm[s]] = yes - no;
}

// [m][Hkv][128] -> [Hkv][m][128] for K and V (16-byte granules).
__global__ void k_store_transpose(const uint4* __restrict__ k, const uint4* __restrict__ v, int m, int Hkv,
                                  uint4* __restrict__ dk, uint4* __restrict__ dv) {
  const int64_t n = static_cast<int64_t>(m) * Hkv * (HEAD_DIM / 8);
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(i % (HEAD_DIM / 8));
    const int64_t rest = i / (HEAD_DIM / 8);
    const int h = static_cast<int>(rest % Hkv);
    const int64_t j = rest / Hkv;
    const int64_t o = (static_cast<int64_t>(h) * m + j) * (HEAD_DIM / 8) + c;
    dk[o] = k[i];
    dv[o] = v[i];
  }
}

// Test kernel: one bounded wait on an mbarrier that is never completed.
__global__ void k_wait_timeout_probe(int* err, uint64_t timeout_ns) {
  __shared__ uint64_t bar;
  const uint32_t b = smem_u32(&bar);
  if (threadIdx.x == 0) {
    mbar_init(b, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(b, 0, err, timeout_ns);  // nothing arrives: gives up
  __syncthreads();
}

inline int blocks_for(int64_t rows) { return static_cast<int>((rows + ROW_WARPS - 1) / ROW_WARPS); }

}  // namespace

cudaError_t launch_embed_norm(const int32_t* tok_id, int T, const bf16* embed, const bf16* gain, int H, float eps,
                              float* r, bf16* xn, cudaStream_t st) {
  if (T <= 0) return cudaSuccess;
  k_embed_norm<<<blocks_for(T), ROW_WARPS * 32, 0, st>>>(tok_id, T, embed, gain, H, eps, r, xn);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm(const float* r, int T, int H, const bf16* gain, float eps, bf16* xn, cudaStream_t st) {
  if (T <= 0) return cudaSuccess;
  k_rmsnorm<<<blocks_for(T), ROW_WARPS * 32, 0, st>>>(r, T, H, gain, eps, xn);
  return cudaGetLastError();
}

cudaError_t launch_qknorm_rope(bf16* qkv, int T, int ld, int Hq, int Hkv, const bf16* qn, const bf16* kn,
                               const int32_t* tok_pos, const float2* rope, float eps, cudaStream_t st) {
  if (T <= 0) return cudaSuccess;
  k_qknorm_rope<<<blocks_for(static_cast<int64_t>(T) * (Hq + Hkv)), ROW_WARPS * 32, 0, st>>>(
      qkv, T, ld, Hq, Hkv, qn, kn, tok_pos, rope, eps);
  return cudaGetLastError();
}

cudaError_t launch_score(const float* r, int H, const int32_t* tok_off, int tok0, int p_begin, int p_end,
                         const int32_t* perm, const bf16* gain, const bf16* head, float eps, float* scores,
                         cudaStream_t st) {
  if (p_end <= p_begin) return cudaSuccess;
  k_score<<<blocks_for(p_end - p_begin), ROW_WARPS * 32, 0, st>>>(r, H, tok_off, tok0, p_begin, p_end, perm, gain,
                                                                  head, eps, scores);
  return cudaGetLastError();
}

cudaError_t launch_store_transpose(const bf16* k, const bf16* v, int m, int Hkv, bf16* dk, bf16* dv,
                                   cudaStream_t st) {
  if (m <= 0) return cudaSuccess;
  const int64_t n = static_cast<int64_t>(m) * Hkv * (HEAD_DIM / 8);
  const int blocks = static_cast<int>((n + 255) / 256);
  k_store_transpose<<<blocks, 256, 0, st>>>(reinterpret_cast<const uint4*>(k), reinterpret_cast<const uint4*>(v), m,
                                            Hkv, reinterpret_cast<uint4*>(dk), reinterpret_cast<uint4*>(dv));
  return cudaGetLastError();
}

cudaError_t launch_wait_timeout_probe(int* err, uint64_t timeout_ns, cudaStream_t st) {
  k_wait_timeout_probe<<<1, 32, 0, st>>>(err, timeout_ns);
  return cudaGetLastError();
}

}  // namespace dopr
