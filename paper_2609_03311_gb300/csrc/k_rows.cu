// k_rows.cu -- the memory-bound per-row kernels of the decoder pass: the
//   embedding gather (with the first RMSNorm's operand and sum of squares),
//   the two-row score head, and the prefix-store layout transpose.  The other
//   RMSNorms and the q/k norm + RoPE are fused into the GEMM epilogues.
// One warp per row (or per head vector); 16-byte vector accesses.
#include <algorithm>

#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int ROW_WARPS = 8;  // warps per block for row kernels

// One warp per row: r = E[id] widened to fp32, ss = sum(r^2),
// xn = f16(r * rsqrt(ss/H + eps) * g).  The row is read twice (the second read hits L1).
__global__ void __launch_bounds__(ROW_WARPS * 32)
    k_embed(const int32_t* __restrict__ tok_id, int T, const bf16* __restrict__ embed, const bf16* __restrict__ gain,
            int H, float eps, float* __restrict__ r, f16* __restrict__ xn, float* __restrict__ ss_out, Extents ext) {
  const int row = blockIdx.x * ROW_WARPS + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= T) return;
  const int64_t id = tok_id[row];
  if (!index_ok(ext.err, id, ext.table_rows) || !index_ok(ext.err, row, ext.rows)) return;
  const bf16* e = embed + id * H;
  float* rr = r + static_cast<int64_t>(row) * H;
  f16* xr = xn + static_cast<int64_t>(row) * H;
  float ss = 0.f;
  for (int c = lane * 8; c < H; c += 256) {
    const uint4 w = *reinterpret_cast<const uint4*>(e + c);
    const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&w);
    float v[8];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 a = __bfloat1622float2(w2[k]);
      v[2 * k] = a.x;
      v[2 * k + 1] = a.y;
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) ss += v[k] * v[k];
    *reinterpret_cast<float4*>(rr + c) = make_float4(v[0], v[1], v[2], v[3]);
    *reinterpret_cast<float4*>(rr + c + 4) = make_float4(v[4], v[5], v[6], v[7]);
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / static_cast<float>(H) + eps);
  bool bad = false;
  for (int c = lane * 8; c < H; c += 256) {
    const uint4 w = *reinterpret_cast<const uint4*>(e + c);
    const uint4 gw = *reinterpret_cast<const uint4*>(gain + c);
    const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&w);
    const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&gw);
    uint32_t o[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 a = __bfloat1622float2(w2[k]), b = __bfloat1622float2(g2[k]);
      const float x0 = a.x * inv * b.x, x1 = a.y * inv * b.y;
      bad |= !(fp16_ok(x0) && fp16_ok(x1));
      o[k] = pack_f16x2(x0, x1);
    }
    *reinterpret_cast<uint4*>(xr + c) = make_uint4(o[0], o[1], o[2], o[3]);
  }
  report_range(ext.err, bad);
  if (lane == 0) ss_out[row] = ss;
}

// In place bf16 -> fp16 over n values (n even), one 32-bit word per thread and
// step; *range |= 1 when a value is not finite or outside fp16's range.
__global__ void k_bf16_to_f16(uint32_t* __restrict__ buf, int64_t n_words, int* range) {
  bool bad = false;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n_words;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    buf[i] = bf16x2_to_f16x2(buf[i], bad);
  if (bad) atomicOr(range, 1);
}

// Score head at the score-token row of each sorted pair in [p_begin, p_end):
// s = <W[0] - W[1], RMSNorm(r_row) * g>, written to scores[perm[pair]].
__global__ void __launch_bounds__(ROW_WARPS * 32)
    k_score(const float* __restrict__ r, int H, const int32_t* __restrict__ tok_off, int tok0, int p_begin, int p_end,
            int compact, const int32_t* __restrict__ perm, const bf16* __restrict__ gain,
            const bf16* __restrict__ head, float eps, float* __restrict__ scores, Extents ext) {
  const int s = p_begin + blockIdx.x * ROW_WARPS + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (s >= p_end) return;
  const int64_t row = compact ? s - p_begin : tok_off[s + 1] - 1 - tok0;
  if (!index_ok(ext.err, row, ext.rows)) return;
  const float* x = r + row * H;
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
  const float sc = yes - no;
  report_range(ext.err, !isfinite(sc));
  if (lane == 0) scores[perm[s]] = sc;
}

// MLP scoring head (Sec. 3.2.3): one CTA per pair.  hn = RMSNorm(row) * g in
// shared memory; each warp takes hidden units j = warp, warp + 8, ...: z = W1[j] . hn
// + b1[j], act(z) * w2[j] summed; the block sum + b2 is the score.
constexpr int MLP_THREADS = 256;
__device__ __forceinline__ float head_act(float z, int act) {
  switch (act) {
    case 0: return fmaxf(z, 0.f);
    case 1: return 0.5f * z * (1.f + erff(z * 0.70710678118654752f));
    case 2: return z / (1.f + expf(-z));
    default: return tanhf(z);
  }
}
__global__ void __launch_bounds__(MLP_THREADS)
    k_score_mlp(const float* __restrict__ r, int H, const int32_t* __restrict__ tok_off, int tok0, int p_begin,
                int compact, const int32_t* __restrict__ perm, const bf16* __restrict__ gain, float eps, int width,
                int act, const bf16* __restrict__ w1, const bf16* __restrict__ b1, const bf16* __restrict__ w2,
                float b2, float* __restrict__ scores, Extents ext) {
  extern __shared__ float hn[];  // [H], then 32 partial sums
  float* red = hn + H;
  const int s = p_begin + blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t row = compact ? s - p_begin : tok_off[s + 1] - 1 - tok0;
  if (!index_ok(ext.err, row, ext.rows)) return;  // uniform across the block
  const float* x = r + row * H;
  float ss = 0.f;
  for (int c = threadIdx.x; c < H; c += blockDim.x) ss += x[c] * x[c];
  ss = warp_sum(ss);
  if (lane == 0) red[warp] = ss;
  __syncthreads();
  float tot = 0.f;
  for (int w = 0; w < MLP_THREADS / 32; ++w) tot += red[w];
  const float inv = rsqrtf(tot / static_cast<float>(H) + eps);
  for (int c = threadIdx.x; c < H; c += blockDim.x) hn[c] = x[c] * inv * __bfloat162float(gain[c]);
  __syncthreads();
  float part = 0.f;
  for (int j = warp; j < width; j += MLP_THREADS / 32) {
    const bf16* wr = w1 + static_cast<int64_t>(j) * H;
    float z = 0.f;
    for (int c = lane * 2; c < H; c += 64) {
      const float2 wv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(wr + c));
      z += wv.x * hn[c] + wv.y * hn[c + 1];
    }
    z = warp_sum(z) + __bfloat162float(b1[j]);
    part += head_act(z, act) * __bfloat162float(w2[j]);
  }
  __syncthreads();
  if (lane == 0) red[warp] = part;
  __syncthreads();
  if (threadIdx.x == 0) {
    float sc = b2;
    for (int w = 0; w < MLP_THREADS / 32; ++w) sc += red[w];
    if (!isfinite(sc) && ext.err) atomicOr(ext.err, DEV_ERR_RANGE);
    scores[perm[s]] = sc;
  }
}

// One warp per pair: copy its score-token row of r (and of the partial sums) to row i.
__global__ void __launch_bounds__(ROW_WARPS * 32)
    k_gather_score_rows(const float* __restrict__ r, const float* __restrict__ ss, int H, int parts,
                        const int32_t* __restrict__ tok_off, int tok0, int p_begin, int p_end,
                        float* __restrict__ dst_r, float* __restrict__ dst_ss, Extents ext) {
  const int i = blockIdx.x * ROW_WARPS + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (p_begin + i >= p_end) return;
  const int64_t row = tok_off[p_begin + i + 1] - 1 - tok0;
  if (!index_ok(ext.err, row, ext.rows) || !index_ok(ext.err, i, ext.rows)) return;
  const float4* src = reinterpret_cast<const float4*>(r + row * H);
  float4* dst = reinterpret_cast<float4*>(dst_r + static_cast<int64_t>(i) * H);
  for (int c = lane; c < H / 4; c += 32) dst[c] = src[c];
  for (int c = lane; c < parts; c += 32) dst_ss[static_cast<int64_t>(i) * parts + c] = ss[row * parts + c];
}

// [m][Hkv][128] bf16 -> [Hkv][m][128] fp16 for K and V (8 elements per thread).
// bf16 -> fp16 is exact for every value of fp16's normal range; values beyond it
// (or not finite) are flagged in *range.
__device__ __forceinline__ uint4 bf16x8_to_f16x8(uint4 x, int& bad) {
  uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[i]));
    bad |= !(fabsf(f.x) <= 65504.f) || !(fabsf(f.y) <= 65504.f);
    w[i] = pack_f16x2(f.x, f.y);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}
__global__ void k_store_transpose(const uint4* __restrict__ k, const uint4* __restrict__ v, int m, int Hkv,
                                  uint4* __restrict__ dk, uint4* __restrict__ dv, int* range) {
  const int64_t n = static_cast<int64_t>(m) * Hkv * (HEAD_DIM / 8);
  int bad = 0;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(i % (HEAD_DIM / 8));
    const int64_t rest = i / (HEAD_DIM / 8);
    const int h = static_cast<int>(rest % Hkv);
    const int64_t j = rest / Hkv;
    const int64_t o = (static_cast<int64_t>(h) * m + j) * (HEAD_DIM / 8) + c;
    dk[o] = bf16x8_to_f16x8(k[i], bad);
    dv[o] = bf16x8_to_f16x8(v[i], bad);
  }
  if (bad) atomicOr(range, 1);
}

// Prefix build (Sec. 3.3): copy each token's key (after the q/k norm and RoPE) and
// raw value of every kv head from the packed QKV buffer into its document's block of
// the store pool, in the layout dopr_store_put writes: per layer, K then V, per kv
// head, m rows of 128.  One warp per (token, kv head, K|V), 8 bytes a lane.
__global__ void k_prefix_store(const f16* __restrict__ qkv, int ld_qkv, int T, int t0, int Hq, int Hkv,
                               const int32_t* __restrict__ tok_pair, const int32_t* __restrict__ tok_pos,
                               const int32_t* __restrict__ pair_slot, const int64_t* __restrict__ slot_row,
                               const int32_t* __restrict__ slot_m, int layer, f16* __restrict__ pool, Extents ext) {
  const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= static_cast<int64_t>(T) * Hkv * 2) return;
  const int kv = static_cast<int>(w & 1);
  const int g = static_cast<int>((w >> 1) % Hkv);
  const int t = static_cast<int>((w >> 1) / Hkv);
  const int p = tok_pair[t0 + t], j = tok_pos[t0 + t];
  const int slot = pair_slot[p];
  const int64_t row = slot_row[slot] + (static_cast<int64_t>(layer * 2 + kv) * Hkv + g) * slot_m[slot] + j;
  if (!index_ok(ext.err, j, slot_m[slot]) || !index_ok(ext.err, row, ext.pool_rows)) return;
  const uint2* src = reinterpret_cast<const uint2*>(qkv + static_cast<int64_t>(t) * ld_qkv + (Hq + kv * Hkv + g) * HEAD_DIM);
  reinterpret_cast<uint2*>(pool + row * HEAD_DIM)[lane] = src[lane];
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

cudaError_t launch_embed(const int32_t* tok_id, int T, const bf16* embed, const bf16* gain, int H, float eps, float* r,
                         f16* xn, float* ss, const Extents& ext, cudaStream_t st) {
  if (T <= 0) return cudaSuccess;
  k_embed<<<blocks_for(T), ROW_WARPS * 32, 0, st>>>(tok_id, T, embed, gain, H, eps, r, xn, ss, ext);
  return cudaGetLastError();
}

cudaError_t launch_bf16_to_f16(void* buf, int64_t n, int* range, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  const int64_t words = n / 2;
  int blocks = static_cast<int>(std::min<int64_t>((words + 255) / 256, 4096));
  k_bf16_to_f16<<<blocks, 256, 0, st>>>(static_cast<uint32_t*>(buf), words, range);
  return cudaGetLastError();
}

cudaError_t launch_score(const float* r, int H, const int32_t* tok_off, int tok0, int p_begin, int p_end, int compact,
                         const int32_t* perm, const bf16* gain, const bf16* head, float eps, float* scores,
                         const Extents& ext, cudaStream_t st) {
  if (p_end <= p_begin) return cudaSuccess;
  k_score<<<blocks_for(p_end - p_begin), ROW_WARPS * 32, 0, st>>>(r, H, tok_off, tok0, p_begin, p_end, compact, perm,
                                                                  gain, head, eps, scores, ext);
  return cudaGetLastError();
}

cudaError_t launch_score_mlp(const float* r, int H, const int32_t* tok_off, int tok0, int p_begin, int p_end,
                             int compact, const int32_t* perm, const bf16* gain, float eps, int width, int act,
                             const bf16* w1, const bf16* b1, const bf16* w2, float b2, float* scores,
                             const Extents& ext, cudaStream_t st) {
  if (p_end <= p_begin) return cudaSuccess;
  k_score_mlp<<<p_end - p_begin, MLP_THREADS, (H + 32) * sizeof(float), st>>>(
      r, H, tok_off, tok0, p_begin, compact, perm, gain, eps, width, act, w1, b1, w2, b2, scores, ext);
  return cudaGetLastError();
}

cudaError_t launch_gather_score_rows(const float* r, const float* ss, int H, int parts, const int32_t* tok_off,
                                     int tok0, int p_begin, int p_end, float* dst_r, float* dst_ss,
                                     const Extents& ext, cudaStream_t st) {
  if (p_end <= p_begin) return cudaSuccess;
  k_gather_score_rows<<<blocks_for(p_end - p_begin), ROW_WARPS * 32, 0, st>>>(r, ss, H, parts, tok_off, tok0, p_begin,
                                                                              p_end, dst_r, dst_ss, ext);
  return cudaGetLastError();
}

cudaError_t launch_store_transpose(const bf16* k, const bf16* v, int m, int Hkv, f16* dk, f16* dv, int* range,
                                   cudaStream_t st) {
  if (m <= 0) return cudaSuccess;
  const int64_t n = static_cast<int64_t>(m) * Hkv * (HEAD_DIM / 8);
  const int blocks = static_cast<int>((n + 255) / 256);
  k_store_transpose<<<blocks, 256, 0, st>>>(reinterpret_cast<const uint4*>(k), reinterpret_cast<const uint4*>(v), m,
                                            Hkv, reinterpret_cast<uint4*>(dk), reinterpret_cast<uint4*>(dv), range);
  return cudaGetLastError();
}

cudaError_t launch_prefix_store(const f16* qkv, int ld_qkv, int T, int t0, int Hq, int Hkv, const int32_t* tok_pair,
                                const int32_t* tok_pos, const int32_t* pair_slot, const int64_t* slot_row,
                                const int32_t* slot_m, int layer, f16* pool, const Extents& ext, cudaStream_t st) {
  const int64_t threads = static_cast<int64_t>(T) * Hkv * 2 * 32;
  if (threads <= 0) return cudaSuccess;
  k_prefix_store<<<static_cast<unsigned>((threads + 255) / 256), 256, 0, st>>>(
      qkv, ld_qkv, T, t0, Hq, Hkv, tok_pair, tok_pos, pair_slot, slot_row, slot_m, layer, pool, ext);
  return cudaGetLastError();
}

cudaError_t launch_wait_timeout_probe(int* err, uint64_t timeout_ns, cudaStream_t st) {
  k_wait_timeout_probe<<<1, 32, 0, st>>>(err, timeout_ns);
  return cudaGetLastError();
}

}  // namespace dopr
