// k_pack.cu -- device batch packer of the online pass.
//
// DoPR's online efficiency comes from reusing a document's stored prefix
// across all queries that retrieved it (Sec. 3.4, "cross-query prefix state
// reuse").  The packer orders the batch so that all pairs of one document are
// adjacent: a stable counting sort on doc_id (ties keep input order), then
// lays every pair's [query tokens ; score token] end to end in that order
// with RoPE positions m_doc + j.  Steps:
//   1. validate pairs, look up store slots, histogram doc ids;
//   2. exclusive scan of the histogram (bucket start offsets);
//   3. stable placement (one warp, match_any groups equal doc ids per 32 pairs);
//   4. exclusive scan of per-pair token counts (packed token offsets);
//   5. (after the host has sized the token buffers) token ids / positions.
#include "device_common.cuh"
#include "internal.h"

namespace dopr {
namespace {

constexpr int INPUT_ERRORS = DEV_ERR_UNKNOWN_DOC | DEV_ERR_INCOMPLETE | DEV_ERR_BAD_TOKEN | DEV_ERR_BAD_OFFSETS |
                             DEV_ERR_POSITION;

__global__ void k_pack_validate(PackArgs a) {
  for (int p = blockIdx.x * blockDim.x + threadIdx.x; p < a.n_pairs; p += gridDim.x * blockDim.x) {
    const int64_t doc = a.doc_ids[p];
    int flag = 0, slot = -1;
    if (doc < 0 || doc > a.max_doc_id) {
      flag |= DEV_ERR_UNKNOWN_DOC;
    } else {
      slot = a.slot_of[doc];
      if (slot < 0)
        flag |= DEV_ERR_UNKNOWN_DOC;
      else if (!a.slot_ok[slot])
        flag |= DEV_ERR_INCOMPLETE;
    }
    const int L = a.q_off[p + 1] - a.q_off[p];
    if (L < 0 || (p == 0 && a.q_off[0] != 0)) flag |= DEV_ERR_BAD_OFFSETS;
    if (!flag && a.slot_m[slot] + L + 1 > a.max_position) flag |= DEV_ERR_POSITION;
    if (flag) {
      atomicOr(a.err, flag);
      a.pair_slot[p] = -1;
    } else {
      a.pair_slot[p] = slot;
      atomicAdd(&a.doc_count[doc], 1);
    }
  }
}

// Block-wide exclusive scan of n ints in place (1024 threads, each owning a
// contiguous segment).  Returns the total to thread 0 via *total if non-null.
__device__ void block_scan_inplace(int32_t* data, int64_t n, int32_t* total) {
  __shared__ int32_t warp_sums[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t seg = (n + blockDim.x - 1) / blockDim.x;
  const int64_t b = min(n, tid * seg), e = min(n, b + seg);
  int32_t local = 0;
  for (int64_t i = b; i < e; ++i) local += data[i];
  // inclusive warp scan of the per-thread totals
  int32_t x = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int32_t w = lane < (blockDim.x >> 5) ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    warp_sums[lane] = w;  // inclusive over warps
  }
  __syncthreads();
  int32_t run = x - local + (warp > 0 ? warp_sums[warp - 1] : 0);
  for (int64_t i = b; i < e; ++i) {
    const int32_t v = data[i];
    data[i] = run;
    run += v;
  }
  if (total && tid == blockDim.x - 1) *total = run;
}

__global__ void __launch_bounds__(1024) k_pack_scan_docs(PackArgs a) {
  if (ld_volatile(a.err) & INPUT_ERRORS) return;
  block_scan_inplace(a.doc_count, a.max_doc_id + 1, nullptr);
}

// One warp walks the pairs in input order, 32 at a time; lanes with equal
// doc ids form a group whose leader reserves consecutive bucket slots, so the
// order inside each bucket is the input order.
__global__ void k_pack_place(PackArgs a) {
  if (ld_volatile(a.err) & INPUT_ERRORS) return;
  const int lane = threadIdx.x;
  for (int base = 0; base < a.n_pairs; base += 32) {
    const int p = base + lane;
    const bool valid = p < a.n_pairs;
    const long long doc = valid ? a.doc_ids[p] : -1;
    const unsigned mask = __match_any_sync(0xffffffffu, static_cast<unsigned long long>(doc));
    const int leader = __ffs(mask) - 1;
    const int rank = __popc(mask & ((1u << lane) - 1u));
    int pos = 0;
    if (valid && lane == leader) {
      pos = a.doc_count[doc];
      a.doc_count[doc] = pos + __popc(mask);
    }
    pos = __shfl_sync(0xffffffffu, pos, leader);
    if (valid) {
      a.perm[pos + rank] = p;
      a.sorted_slot[pos + rank] = a.pair_slot[p];
    }
    __syncwarp();
  }
}

__global__ void __launch_bounds__(1024) k_pack_offsets(PackArgs a) {
  if (ld_volatile(a.err) & INPUT_ERRORS) return;
  const int n = a.n_pairs;
  for (int s = threadIdx.x; s < n; s += blockDim.x) {
    const int p = a.perm[s];
    a.tok_off[s] = a.q_off[p + 1] - a.q_off[p] + 1;
  }
  __syncthreads();
  block_scan_inplace(a.tok_off, n, a.tok_off + n);
}

// One warp per sorted pair.
__global__ void k_pack_tokens(PackArgs a) {
  if (ld_volatile(a.err) & INPUT_ERRORS) return;
  const int s = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (s >= a.n_pairs) return;
  const int p = a.perm[s];
  const int q0 = a.q_off[p], L = a.q_off[p + 1] - q0;
  const int off = a.tok_off[s];
  const int m = a.slot_m[a.sorted_slot[s]];
  for (int j = lane; j <= L; j += 32) {
    int tok = j < L ? a.q_tok[q0 + j] : a.score_token;
    if (tok < 0 || tok >= a.vocab) {
      atomicOr(a.err, DEV_ERR_BAD_TOKEN);
      tok = 0;
    }
    a.tok_id[off + j] = tok;
    a.tok_pos[off + j] = m + j;
    a.tok_pair[off + j] = s;
  }
}

}  // namespace

cudaError_t launch_pack_order(const PackArgs& a, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(a.doc_count, 0, sizeof(int32_t) * (a.max_doc_id + 1), st);
  if (e) return e;
  if (a.n_pairs <= 0) return cudaSuccess;
  const int blocks = (a.n_pairs + 255) / 256;
  k_pack_validate<<<blocks < 1024 ? blocks : 1024, 256, 0, st>>>(a);
  k_pack_scan_docs<<<1, 1024, 0, st>>>(a);
  k_pack_place<<<1, 32, 0, st>>>(a);
  k_pack_offsets<<<1, 1024, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_pack_tokens(const PackArgs& a, cudaStream_t st) {
  if (a.n_pairs <= 0) return cudaSuccess;
  k_pack_tokens<<<(a.n_pairs + 7) / 8, 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace dopr
