// k_select.cu -- attention-based key token selection (DoPR Sec. 3.2.1, applied
// offline as in Sec. 3.3): from a document-only pass, the last layer's
// attention weights averaged over the q heads (A-bar, n x n, causal), each
// token's salience u_i = the mean of the top-p entries of column i, the
// top-K positions, and their final-layer states after the final RMSNorm.
//
// These kernels run once per document in the offline path; they are plain
// CUDA-core code sized for documents of up to SEL_MAX_N tokens.
#include <float.h>
#include <math.h>

#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int PROB_THREADS = 256;
constexpr int SORT_THREADS = 1024;

__device__ __forceinline__ float block_reduce(float v, float* red, bool is_max) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float x = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, x) : v + x;
  }
  __syncthreads();  // red is reused across calls
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < nw ? red[lane] : (is_max ? -FLT_MAX : 0.f);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float x = __shfl_xor_sync(0xffffffffu, v, o);
      v = is_max ? fmaxf(v, x) : v + x;
    }
    if (lane == 0) red[0] = v;
  }
  __syncthreads();
  return red[0];
}

// One CTA per token row t of the chunk: row t of its document's A-bar.
// A is [n][n] per document at a_off[doc] (fp32); entries above the diagonal are 0.
__global__ void __launch_bounds__(PROB_THREADS) k_sal_probs(const f16* __restrict__ qkv, int ld_qkv, int Hq, int Hkv,
                                                            const int32_t* __restrict__ tok_pair,
                                                            const int32_t* __restrict__ tok_off, int t0, int p0,
                                                            const int64_t* __restrict__ a_off, float* __restrict__ A,
                                                            Extents ext) {
  extern __shared__ float sm[];
  float* q = sm;                  // [128]
  float* red = q + HEAD_DIM;      // [32]
  float* s = red + 32;            // [n]
  float* acc = s + SEL_MAX_N;     // [n]
  const int t = blockIdx.x;       // chunk row
  const int p = tok_pair[t0 + t];
  const int ts = tok_off[p] - t0, n = tok_off[p + 1] - tok_off[p];
  const int jt = t - ts;          // row within the document
  const int G = Hq / Hkv;
  // block-uniform: the document's rows in the chunk and its row of A-bar
  if (!index_ok(ext.err, ts, ext.rows) || !index_ok(ext.err, ts + n - 1, ext.rows) ||
      !index_ok(ext.err, a_off[p - p0] + static_cast<int64_t>(jt + 1) * n - 1, ext.a_elems))
    return;
  const float scale = rsqrtf(static_cast<float>(HEAD_DIM));
  for (int i = threadIdx.x; i <= jt; i += blockDim.x) acc[i] = 0.f;
  for (int h = 0; h < Hq; ++h) {
    const int g = h / G;
    __syncthreads();
    if (threadIdx.x < HEAD_DIM) q[threadIdx.x] = __half2float(qkv[static_cast<int64_t>(t) * ld_qkv + h * HEAD_DIM + threadIdx.x]);
    __syncthreads();
    float mx = -FLT_MAX;
    for (int i = threadIdx.x; i <= jt; i += blockDim.x) {
      const uint4* kr = reinterpret_cast<const uint4*>(qkv + static_cast<int64_t>(ts + i) * ld_qkv + (Hq + g) * HEAD_DIM);
      float d = 0.f;
#pragma unroll 4
      for (int c = 0; c < HEAD_DIM / 8; ++c) {
        const uint4 w = kr[c];
        const __half2* h2 = reinterpret_cast<const __half2*>(&w);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __half22float2(h2[e]);
          d = fmaf(q[c * 8 + 2 * e], f.x, d);
          d = fmaf(q[c * 8 + 2 * e + 1], f.y, d);
        }
      }
      s[i] = d * scale;
      mx = fmaxf(mx, s[i]);
    }
    mx = block_reduce(mx, red, true);
    float z = 0.f;
    for (int i = threadIdx.x; i <= jt; i += blockDim.x) {
      s[i] = expf(s[i] - mx);
      z += s[i];
    }
    z = block_reduce(z, red, false);
    const float w = 1.f / (z * static_cast<float>(Hq));
    for (int i = threadIdx.x; i <= jt; i += blockDim.x) acc[i] += s[i] * w;
  }
  __syncthreads();
  float* row = A + a_off[p - p0] + static_cast<int64_t>(jt) * n;
  for (int i = threadIdx.x; i < n; i += blockDim.x) row[i] = i <= jt ? acc[i] : 0.f;
}

// Bitonic sort of SEL_MAX_N keys in shared memory, descending by `val` with
// ties to the smaller `idx` (idx may be null: values only).
__device__ void bitonic_desc(float* val, int* idx) {
  for (int k = 2; k <= SEL_MAX_N; k <<= 1)
    for (int j = k >> 1; j > 0; j >>= 1) {
      __syncthreads();
      for (int i = threadIdx.x; i < SEL_MAX_N; i += blockDim.x) {
        const int l = i ^ j;
        if (l > i) {
          const bool up = (i & k) == 0;  // this run sorts descending when up
          const float a = val[i], b = val[l];
          const int ia = idx ? idx[i] : 0, ib = idx ? idx[l] : 0;
          const bool a_first = a > b || (a == b && ia < ib);  // a precedes b in the final order
          if (up != a_first) {
            val[i] = b;
            val[l] = a;
            if (idx) {
              idx[i] = ib;
              idx[l] = ia;
            }
          }
        }
      }
    }
  __syncthreads();
}

// One CTA per token (column i of its document): u_i = mean of the top-p of A[i..n-1][i].
__global__ void __launch_bounds__(SORT_THREADS) k_sal_colstat(const int32_t* __restrict__ tok_pair,
                                                              const int32_t* __restrict__ tok_off, int t0, int p0,
                                                              const int64_t* __restrict__ a_off,
                                                              const float* __restrict__ A, int top_p,
                                                              float* __restrict__ u, Extents ext) {
  __shared__ float v[SEL_MAX_N];
  __shared__ float red[32];
  const int t = blockIdx.x;
  const int p = tok_pair[t0 + t];
  const int ts = tok_off[p] - t0, n = tok_off[p + 1] - tok_off[p];
  const int i = t - ts;
  const int cnt = n - i, k = min(top_p, cnt);
  if (!index_ok(ext.err, a_off[p - p0] + static_cast<int64_t>(n) * n - 1, ext.a_elems)) return;  // block-uniform
  const float* col = A + a_off[p - p0] + i;
  float sum = 0.f;
  if (k == cnt) {
    for (int r = threadIdx.x; r < cnt; r += blockDim.x) sum += col[static_cast<int64_t>(i + r) * n];
  } else {
    for (int r = threadIdx.x; r < SEL_MAX_N; r += blockDim.x)
      v[r] = r < cnt ? col[static_cast<int64_t>(i + r) * n] : -FLT_MAX;
    bitonic_desc(v, nullptr);
    for (int r = threadIdx.x; r < k; r += blockDim.x) sum += v[r];
  }
  sum = block_reduce(sum, red, false);
  if (threadIdx.x == 0) u[t] = sum / static_cast<float>(k);
}

// One CTA per document of the chunk: the min(K, n) most salient positions,
// ties to the lower position, in ascending order; -1 after them.
__global__ void __launch_bounds__(SORT_THREADS) k_sal_topk(const int32_t* __restrict__ tok_off, int t0, int p0,
                                                           const float* __restrict__ u, int K,
                                                           int32_t* __restrict__ positions) {
  __shared__ float v[SEL_MAX_N];
  __shared__ int ix[SEL_MAX_N];
  __shared__ int flag[SEL_MAX_N];
  const int p = p0 + blockIdx.x;
  const int ts = tok_off[p] - t0, n = tok_off[p + 1] - tok_off[p];
  const int k = min(K, n);
  for (int r = threadIdx.x; r < SEL_MAX_N; r += blockDim.x) {
    v[r] = r < n ? u[ts + r] : -FLT_MAX;
    ix[r] = r < n ? r : 0x7fffffff;
    flag[r] = 0;
  }
  bitonic_desc(v, ix);
  for (int r = threadIdx.x; r < k; r += blockDim.x) flag[ix[r]] = 1;
  __syncthreads();
  if (threadIdx.x == 0) {  // compact the flags in position order (n <= SEL_MAX_N: one pass)
    int j = 0;
    int32_t* out = positions + static_cast<int64_t>(p) * K;
    for (int r = 0; r < n && j < k; ++r)
      if (flag[r]) out[j++] = r;
    for (; j < K; ++j) out[j] = -1;
  }
}

// One warp per (document, selected slot): x = bf16(RMSNorm(r_row) * g_final), zeros for -1.
__global__ void k_sal_gather(const float* __restrict__ r, int H, const int32_t* __restrict__ tok_off, int t0,
                             int p0, int n_docs, const int32_t* __restrict__ positions, int K,
                             const bf16* __restrict__ gain, float eps, bf16* __restrict__ x, Extents ext) {
  const int w = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (w >= n_docs * K) return;
  const int p = p0 + w / K, j = w % K;
  const int pos = positions[static_cast<int64_t>(p) * K + j];
  bf16* dst = x + (static_cast<int64_t>(p) * K + j) * H;
  if (pos < 0) {
    for (int c = lane; c < H; c += 32) dst[c] = __float2bfloat16(0.f);
    return;
  }
  const int64_t rr = static_cast<int64_t>(tok_off[p] - t0) + pos;
  if (!index_ok(ext.err, rr, ext.rows)) return;
  const float* row = r + rr * H;
  float ss = 0.f;
  for (int c = lane; c < H; c += 32) ss += row[c] * row[c];
  ss = warp_sum(ss);
  const float rs = rsqrtf(ss / static_cast<float>(H) + eps);
  for (int c = lane; c < H; c += 32) dst[c] = __float2bfloat16(row[c] * rs * __bfloat162float(gain[c]));
}

}  // namespace

cudaError_t select_setup() {
  return cudaFuncSetAttribute(k_sal_probs, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>((HEAD_DIM + 32 + 2 * SEL_MAX_N) * sizeof(float)));
}

cudaError_t launch_select(const SelectArgs& a, cudaStream_t st) {
  if (a.n_rows <= 0) return cudaSuccess;
  const size_t smem = (HEAD_DIM + 32 + 2 * SEL_MAX_N) * sizeof(float);
  k_sal_probs<<<a.n_rows, PROB_THREADS, smem, st>>>(a.qkv, a.ld_qkv, a.Hq, a.Hkv, a.tok_pair, a.tok_off, a.t0, a.p0,
                                                    a.a_off, a.A, a.ext);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_sal_colstat<<<a.n_rows, SORT_THREADS, 0, st>>>(a.tok_pair, a.tok_off, a.t0, a.p0, a.a_off, a.A, a.top_p, a.u,
                                                   a.ext);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  k_sal_topk<<<a.n_docs, SORT_THREADS, 0, st>>>(a.tok_off, a.t0, a.p0, a.u, a.top_k, a.positions);
  return cudaGetLastError();
}

cudaError_t launch_select_gather(const SelectArgs& a, const float* r, int H, const bf16* gain, float eps,
                                 cudaStream_t st) {
  const int64_t threads = static_cast<int64_t>(a.n_docs) * a.top_k * 32;
  if (threads <= 0) return cudaSuccess;
  k_sal_gather<<<static_cast<unsigned>((threads + 255) / 256), 256, 0, st>>>(r, H, a.tok_off, a.t0, a.p0, a.n_docs,
                                                                             a.positions, a.top_k, gain, eps, a.x,
                                                                             a.ext);
  return cudaGetLastError();
}

}  // namespace dopr
