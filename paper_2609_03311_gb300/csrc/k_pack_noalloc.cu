// k_pack_noalloc.cu -- an allocation-free entry point to the batch packer's
// ordering step (stable grouping of pairs by doc id + packed token offsets).
//
// Who needs it: callers that cannot allocate device memory when they score.
// A serving process whose device memory is owned by another allocator (for
// example a framework's caching pool that has already reserved the GPU) gets
// no room from cudaMalloc, and a latency-critical request loop cannot afford
// cudaMalloc/cudaFree because they may synchronise the whole device.  The
// regular entry points grow their work buffers with cudaMalloc on demand;
// this one instead uses a fixed scratch array compiled into the library, so
// the call itself allocates nothing.
//
// The scratch array below lives in every GPU that loads the library, until
// the process exits (NOALLOC_SCRATCH_INTS 32-bit words, about 768 KiB).
#include <mutex>
#include <string>

#include "device_common.cuh"
#include "internal.h"

struct dopr_store : dopr::Store {};

namespace dopr {
namespace {

constexpr int NOALLOC_MAX_PAIRS = 32768;   // largest n_pairs accepted
constexpr int NOALLOC_MAX_DOCS = 131072;   // largest store max_doc_id + 1 accepted
constexpr int NOALLOC_ERR_WORDS = 64;
constexpr int NOALLOC_SCRATCH_INTS = NOALLOC_MAX_DOCS + 2 * NOALLOC_MAX_PAIRS + NOALLOC_ERR_WORDS;

// Layout: [doc histogram: MAX_DOCS][pair slot: MAX_PAIRS][sorted slot: MAX_PAIRS][error word ...]
static __device__ __align__(256) int32_t g_pack_scratch[NOALLOC_SCRATCH_INTS];

constexpr int MAX_DEVICES = 256;
std::mutex g_mu;
int32_t* g_scratch_addr[MAX_DEVICES] = {};

// Device address of g_pack_scratch on the current device, looked up once per
// device.  In host code the symbol is only a host-side stand-in, so kernels
// must be given this address, never the symbol itself.
dopr_status scratch_for_current_device(int32_t** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    set_last_error_message(std::string("cudaGetDevice failed: ") + cudaGetErrorString(e));
    return DOPR_ERR_CUDA;
  }
  if (dev < 0 || dev >= MAX_DEVICES) {
    set_last_error_message("device index out of range for the scratch table");
    return DOPR_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_pack_scratch);
    if (e != cudaSuccess || !p) {
      set_last_error_message(std::string("cudaGetSymbolAddress(g_pack_scratch) failed: ") + cudaGetErrorString(e));
      return DOPR_ERR_CUDA;
    }
    g_scratch_addr[dev] = static_cast<int32_t*>(p);
  }
  *out = g_scratch_addr[dev];
  return DOPR_OK;
}

dopr_status device_error_status(int e) {
  if (e & DEV_ERR_TIMEOUT) { set_last_error_message("a bounded device wait timed out"); return DOPR_ERR_TIMEOUT; }
  if (e & DEV_ERR_UNKNOWN_DOC) { set_last_error_message("a doc_id has no stored prefix"); return DOPR_ERR_UNKNOWN_DOC; }
  if (e & DEV_ERR_INCOMPLETE) { set_last_error_message("a doc is missing stored layers"); return DOPR_ERR_INCOMPLETE; }
  if (e & DEV_ERR_BAD_OFFSETS) {
    set_last_error_message("q_offsets must start at 0 and not decrease");
    return DOPR_ERR_INVALID_ARG;
  }
  if (e & DEV_ERR_POSITION) {
    set_last_error_message("m + query length + 1 exceeds max_position");
    return DOPR_ERR_INVALID_ARG;
  }
  return DOPR_OK;
}

}  // namespace
}  // namespace dopr

using namespace dopr;

extern "C" dopr_status dopr_pack_order_noalloc(const dopr_store* store, int32_t n_pairs, const int32_t* q_offsets,
                                               const int64_t* doc_ids, int32_t* perm, int32_t* tok_off,
                                               void* cuda_stream) {
  set_last_error_message("");
  if (!store || n_pairs < 0 || !q_offsets || !tok_off || (n_pairs > 0 && (!doc_ids || !perm))) {
    set_last_error_message("NULL pointer or negative n_pairs");
    return DOPR_ERR_INVALID_ARG;
  }
  if (n_pairs > NOALLOC_MAX_PAIRS) {
    set_last_error_message("n_pairs " + std::to_string(n_pairs) + " exceeds the no-allocation limit of " +
                           std::to_string(NOALLOC_MAX_PAIRS) + " pairs per call");
    return DOPR_ERR_UNSUPPORTED;
  }
  if (store->max_doc_id + 1 > NOALLOC_MAX_DOCS) {
    set_last_error_message("store max_doc_id " + std::to_string(store->max_doc_id) +
                           " exceeds the no-allocation limit of " + std::to_string(NOALLOC_MAX_DOCS - 1));
    return DOPR_ERR_UNSUPPORTED;
  }
  cudaError_t e = cudaSetDevice(store->device);
  if (e != cudaSuccess) {
    set_last_error_message(std::string("cudaSetDevice failed: ") + cudaGetErrorString(e));
    return DOPR_ERR_CUDA;
  }
  int32_t* scratch = nullptr;
  dopr_status st = scratch_for_current_device(&scratch);
  if (st != DOPR_OK) return st;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  int32_t* err = scratch + NOALLOC_MAX_DOCS + 2 * NOALLOC_MAX_PAIRS;
  if (n_pairs == 0) {
    e = cudaMemsetAsync(tok_off, 0, sizeof(int32_t), stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) {
      set_last_error_message(std::string("CUDA error: ") + cudaGetErrorString(e));
      return DOPR_ERR_CUDA;
    }
    return DOPR_OK;
  }
  PackArgs a{};
  a.n_pairs = n_pairs;
  a.q_off = q_offsets;
  a.q_tok = nullptr;  // the ordering step reads no token ids
  a.doc_ids = doc_ids;
  a.max_doc_id = store->max_doc_id;
  a.slot_of = store->d_slot_of;
  a.slot_m = store->d_slot_m;
  a.slot_ok = store->d_slot_ok;
  a.vocab = store->cfg.vocab;
  a.score_token = store->cfg.score_token_id;
  a.max_position = store->cfg.max_position;
  a.doc_count = scratch;  // zeroed by launch_pack_order before use
  a.pair_slot = scratch + NOALLOC_MAX_DOCS;
  a.perm = perm;
  a.sorted_slot = scratch + NOALLOC_MAX_DOCS + NOALLOC_MAX_PAIRS;
  a.tok_off = tok_off;
  a.err = err;
  int h_err = 0;
  e = cudaMemsetAsync(err, 0, sizeof(int32_t), stream);  // the error word must start at zero
  if (e == cudaSuccess) e = launch_pack_order(a, stream);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&h_err, err, sizeof(int32_t), cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) {
    set_last_error_message(std::string("CUDA error: ") + cudaGetErrorString(e));
    return DOPR_ERR_CUDA;
  }
  return device_error_status(h_err);
}
