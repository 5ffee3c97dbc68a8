/*
 * dopr.h -- C ABI of the GB300-native DoPR online scoring library (libdopr.so).
 *
 * DoPR (Sec. 3.1 "Problem Formulation", Sec. 3.3 "Offline Compression",
 * Sec. 3.4 "Online Reranking") stores, for every document d, the multi-layer
 * key/value states C~_d of K_infer = m compressed prefix positions.  Online,
 * a pair (q, d) is scored by running the decoder over [q ; t_score] only,
 * each layer attending to d's stored prefix keys/values before the causal
 * online keys, and reading the score at t_score.  This library implements
 * that online pass on one GPU: a device-resident prefix store, a batch
 * packer that groups pairs by document, and the decoder kernels.
 *
 * Conventions for every entry point:
 *   - Plain C types only.  bf16 tensors are passed as `const void*` to
 *     16-bit bit patterns (IEEE bfloat16).  Matrices are row-major.
 *   - Inputs are borrowed for the duration of the call; the library copies
 *     what it keeps.  Outputs go to caller-owned buffers.  Library objects
 *     are opaque and released by the matching *_destroy.
 *   - Every argument is validated before any device work is launched; on an
 *     error nothing is written to caller buffers and the object is left as
 *     it was.  The status says what went wrong; dopr_last_error() returns a
 *     thread-local message for the last failing call on this thread.
 *   - Device work runs on the device that is current when the object is
 *     created; use the same device for all calls on that object.
 *   - Objects are not thread-safe: serialise calls on one object.
 */
#ifndef DOPR_H
#define DOPR_H

#include <stdint.h>

#if defined(__GNUC__)
#define DOPR_API __attribute__((visibility("default")))
#else
#define DOPR_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DOPR_OK = 0,
    DOPR_ERR_INVALID_ARG = 1,   /* bad pointer, size, index or shape          */
    DOPR_ERR_UNKNOWN_DOC = 2,   /* a doc_id has no stored prefix              */
    DOPR_ERR_INCOMPLETE = 3,    /* a weight or a doc layer was never supplied */
    DOPR_ERR_OUT_OF_MEMORY = 4, /* device allocation or the store pool full   */
    DOPR_ERR_CUDA = 5,          /* a CUDA runtime/driver call failed          */
    DOPR_ERR_TIMEOUT = 6,       /* a bounded device wait ran out; the result
                                   of that call is invalid, the context is not */
    DOPR_ERR_UNSUPPORTED = 7,   /* a shape this build does not handle         */
    DOPR_ERR_INTERNAL = 8,      /* a checked build (DOPR_CHECKED) met an index
                                   outside its buffer and skipped the access:
                                   a library defect; the call's outputs are
                                   invalid, the context is not               */
    DOPR_ERR_RANGE = 9          /* a value the tensor cores take as an fp16
                                   operand (normed activations, q/k/v, the
                                   SwiGLU output, the attention output) or a
                                   score was not finite or exceeded 65504 in
                                   magnitude: the inputs leave the range the
                                   fp16 path computes on; the call's outputs
                                   are invalid, the context is not           */
} dopr_status;

/*
 * Decoder shape (Qwen3 family, the paper's backbone, Sec. 4.1).
 * Supported: head_dim == 128; n_q_heads % n_kv_heads == 0;
 * hidden % 256 == 0; ffn % 128 == 0; (n_q_heads + 2 n_kv_heads) * 128 % 256 == 0.
 * score_token_id is t_score (Sec. 3.1), appended by the library to every
 * query.  Positions m + j of online tokens must be < max_position.
 */
typedef struct {
    int32_t n_layers;
    int32_t hidden;
    int32_t n_q_heads;
    int32_t n_kv_heads;
    int32_t head_dim;
    int32_t ffn;
    int32_t vocab;
    int32_t score_token_id;
    int32_t max_position;
    float rope_theta;   /* RoPE base, rotate-half pairs (i, i + head_dim/2) */
    float rms_eps;      /* RMSNorm epsilon                                  */
} dopr_model_config;

typedef struct dopr_model dopr_model;
typedef struct dopr_store dopr_store;

/* Weight kinds for dopr_model_put_weight; shapes are [rows][cols] bf16. */
typedef enum {
    DOPR_W_EMBED = 0,      /* [vocab][hidden]             (layer ignored) */
    DOPR_W_ATTN_NORM = 1,  /* [hidden]      input RMSNorm gain            */
    DOPR_W_Q = 2,          /* [n_q_heads*128][hidden]                     */
    DOPR_W_K = 3,          /* [n_kv_heads*128][hidden]                    */
    DOPR_W_V = 4,          /* [n_kv_heads*128][hidden]                    */
    DOPR_W_Q_NORM = 5,     /* [128]         per-head RMSNorm gain on q    */
    DOPR_W_K_NORM = 6,     /* [128]         per-head RMSNorm gain on k    */
    DOPR_W_O = 7,          /* [hidden][n_q_heads*128]                     */
    DOPR_W_MLP_NORM = 8,   /* [hidden]      post-attention RMSNorm gain   */
    DOPR_W_GATE = 9,       /* [ffn][hidden]                               */
    DOPR_W_UP = 10,        /* [ffn][hidden]                               */
    DOPR_W_DOWN = 11,      /* [hidden][ffn]                               */
    DOPR_W_FINAL_NORM = 12,/* [hidden]                    (layer ignored) */
    DOPR_W_SCORE_HEAD = 13 /* [2][hidden]: row 0 "yes", row 1 "no"
                              (layer ignored)                             */
} dopr_weight_kind;

/* Create a model: allocates device memory for all weights of `cfg` (left
 * unset until put).  *out receives the handle.  Errors: INVALID_ARG,
 * UNSUPPORTED, OUT_OF_MEMORY, CUDA. */
DOPR_API dopr_status dopr_model_create(const dopr_model_config *cfg, dopr_model **out);

/* Copy one weight tensor into the model (converted to the library's own
 * device layout).  `src` holds n_elems bf16 values in the layout listed
 * under dopr_weight_kind; src_on_device != 0 means `src` is a device
 * pointer.  Re-putting a weight replaces it.  Synchronous.  The
 * projection matrices (Q, K, V, O, gate, up, down) are held as fp16 for
 * the tensor cores: a value that is not finite or exceeds 65504 in
 * magnitude fails the put (the weight is then left as it was).
 * Errors: INVALID_ARG (kind, layer or n_elems wrong; a projection value
 * outside fp16's range), CUDA. */
DOPR_API dopr_status dopr_model_put_weight(dopr_model *model, int32_t kind, int32_t layer, const void *src,
                                  int64_t n_elems, int32_t src_on_device);

/*
 * Replace the yes/no score rows by the paper's lightweight MLP head on the
 * score token's state (Sec. 3.2.3, s = MLP(h_score); its shape is not given):
 * one hidden layer of `width` units over hn = RMSNorm(h) * final_norm,
 *   s = sum_j w2[j] * act(W1[j] . hn + b1[j]) + b2,
 * W1 bf16 [width][hidden], b1 and w2 bf16 [width]; activation 0 ReLU,
 * 1 GELU (erf form), 2 SiLU, 3 tanh.  src_on_device != 0: device pointers.
 * width == 0 restores the yes/no rows.  Synchronous.
 * Errors: INVALID_ARG, OUT_OF_MEMORY, CUDA.
 */
DOPR_API dopr_status dopr_model_set_mlp_head(dopr_model *model, int32_t width, int32_t activation, const void *w1,
                                            const void *b1, const void *w2, float b2, int32_t src_on_device);

/* Release a model and its device memory.  NULL is accepted. */
DOPR_API dopr_status dopr_model_destroy(dopr_model *model);

/*
 * Prefix store (Sec. 3.3: the offline store of C~_d; Sec. 3.4: fetched per
 * candidate).  Holds doc ids 0..max_doc_id in a device pool of pool_bytes
 * bytes; each document takes dopr_prefix_bytes(cfg, m) bytes of it.
 * Errors: INVALID_ARG, UNSUPPORTED, OUT_OF_MEMORY, CUDA.
 */
DOPR_API dopr_status dopr_store_create(const dopr_model_config *cfg, int64_t max_doc_id, int64_t pool_bytes,
                              dopr_store **out);

/*
 * Store one layer of a document's compressed prefix states (Sec. 3.4 and
 * its footnote: the multi-layer K/V obtained by forwarding the selected
 * representations as prefix inputs).
 *   k, v: bf16 [m][n_kv_heads][head_dim].  k is the key after the per-head
 *         RMSNorm and after RoPE at positions 0..m-1; v is the raw value.
 *   0 <= m <= 256 (the largest K_infer of the paper's settings, Tab. 8);
 *   m == 0 stores an empty prefix (the pass then equals a query-only forward).
 * The first put of a doc reserves its block; later puts must give the same
 * m (a different m is INVALID_ARG) and replace that layer.  A doc can be
 * scored once all n_layers layers were put.  The store keeps the values as
 * fp16 (exact for bf16 values in fp16's normal range); a value that is not
 * finite or exceeds 65504 in magnitude fails the put with INVALID_ARG and
 * leaves that layer marked missing.  Synchronous.
 * Errors: INVALID_ARG, OUT_OF_MEMORY (pool full), CUDA.
 */
DOPR_API dopr_status dopr_store_put(dopr_store *store, int64_t doc_id, int32_t m, int32_t layer, const void *k,
                           const void *v, int32_t src_on_device);

/* Release a store.  NULL is accepted. */
DOPR_API dopr_status dopr_store_destroy(dopr_store *store);

/*
 * Offline prefix construction (Sec. 3.3; Sec. 3.4's footnote): for each
 * document d, forward its selected representations c_1..c_m (the compressed
 * document inputs C~_d is built from) causally through the model as prefix
 * inputs at positions 0..m-1, and store every layer's key (after the q/k
 * norm and RoPE) and value as the document's prefix states -- the states
 * dopr_store_put would be given.  The last layer stops after its key/value
 * projection.
 *   doc_ids   [n_docs] int64, host; distinct, each in [0, max_doc_id].
 *   x_offsets [n_docs+1] int32, host: document d's representations are rows
 *             x_offsets[d] .. x_offsets[d+1]-1 of x; x_offsets[0] == 0,
 *             0 <= m_d <= 256 and m_d <= max_position.
 *   x         bf16 [x_offsets[n_docs]][hidden]; a device pointer when
 *             x_on_device != 0, else host memory (copied in by the call).
 *   cuda_stream: a cudaStream_t, or NULL for the default stream.
 * Documents are reserved (or must match an earlier reservation's m) before
 * any kernel runs; on success every layer of every document is present.
 * Synchronous.  Errors: INVALID_ARG, INCOMPLETE (model weights missing),
 * OUT_OF_MEMORY (pool full), CUDA, TIMEOUT.
 */
DOPR_API dopr_status dopr_build_prefixes(dopr_model *model, dopr_store *store, int32_t n_docs, const int64_t *doc_ids,
                                         const int32_t *x_offsets, const void *x, int32_t x_on_device,
                                         void *cuda_stream);

/*
 * Attention-based key token selection (Sec. 3.2.1), as the offline
 * construction of Sec. 3.3 applies it: encode each document alone (its
 * token ids at positions 0..n-1; no prefix, no score token), average the
 * last layer's attention weights over the q heads into A[n][n] (row =
 * attending token, causal), score token i by the mean of the top_p largest
 * entries of column i (of its min(top_p, n - i) causal entries), keep the
 * top_k most salient positions (equal salience to the lower position) and
 * return them in ascending order with their final-layer states after the
 * final RMSNorm -- the representations dopr_build_prefixes takes.  The paper
 * leaves p open; top_p >= n gives the column mean.
 *   doc_offsets [n_docs+1] int32, host: document d is doc_tokens[off[d] .. off[d+1]);
 *               off[0] == 0, 1 <= n_d <= 2048 and n_d <= max_position.
 *   doc_tokens  int32 token ids in [0, vocab), host.
 *   1 <= top_k <= 256, top_p >= 1.
 *   positions   [n_docs][top_k] int32, host: ascending, -1 past min(top_k, n_d).
 *   x_out       [n_docs][top_k][hidden] bf16, host: the states at `positions`
 *               (zero rows for -1).
 *   salience    [off[n_docs]] float, host, or NULL: u of every token.
 * Device memory of n^2 floats per document of a chunk is allocated for the
 * call.  Synchronous.  Errors: INVALID_ARG, INCOMPLETE (model weights
 * missing), OUT_OF_MEMORY, CUDA, TIMEOUT.
 */
DOPR_API dopr_status dopr_select_prefix_inputs(dopr_model *model, int32_t n_docs, const int32_t *doc_offsets,
                                               const int32_t *doc_tokens, int32_t top_k, int32_t top_p,
                                               int32_t *positions, void *x_out, float *salience, void *cuda_stream);

/*
 * A stored layer of one document, read back for testing: k_out and v_out
 * (host, fp16 bits [m][n_kv_heads][head_dim], the dopr_store_put layout).
 * A document with m == 0 writes nothing.  Synchronous.
 * Errors: INVALID_ARG, UNKNOWN_DOC (never stored), CUDA.
 */
DOPR_API dopr_status dopr_debug_store_read(const dopr_store *store, int64_t doc_id, int32_t layer, void *k_out,
                                           void *v_out);

/* Bytes of stored prefix state for one document of m prefix positions:
 * m * n_layers * 2 (K,V) * n_kv_heads * head_dim * 2 bytes.  This is the
 * document-side memory figure of Tab. 3 / Tab. 9.  Returns -1 on a bad cfg. */
DOPR_API int64_t dopr_prefix_bytes(const dopr_model_config *cfg, int32_t m);

/*
 * Score a batch of (query, document) pairs (Sec. 3.4).
 *   q_offsets [n_pairs+1] int32: query p is q_tokens[q_offsets[p] .. q_offsets[p+1]);
 *             q_offsets[0] == 0, non-decreasing; empty queries are allowed
 *             (the pair is then scored on the score token alone).
 *   q_tokens  int32 token ids in [0, vocab).
 *   doc_ids   [n_pairs] int64, each with a complete prefix in `store`.
 *   scores    [n_pairs] float, written in input order: the "yes" minus
 *             "no" logit at the score token.
 *   cuda_stream: a cudaStream_t, or NULL for the default stream.
 *   io_on_device: 0 = the four arrays are host memory (copied in and out by
 *             the call); 1 = device memory (read and written in place).
 * Arithmetic: the tensor-core operands (activations, projection weights,
 * q/k/v, attention probabilities) are fp16 -- the bf16 inputs widen to fp16
 * exactly in its normal range -- with fp32 accumulation, an fp32 residual
 * stream and fp32 norms, softmax and score head.
 * The call is synchronous in both modes: it synchronises `cuda_stream`
 * once after packing (to size the launches) and once after the last
 * kernel, reads the device error word, and only when it is clear copies
 * the scores into `scores` (a third synchronisation): a call that fails,
 * on the host or on the device, writes nothing.  Pairs of one doc_id are
 * grouped so that their prefix is staged once per group; scores do not
 * depend on batch order.  With io_on_device = 1 the inputs are validated
 * on the device and an invalid batch returns its error before any decoder
 * kernel runs.
 * Valid range: every fp16 operand must stay within +-65504 (the bf16
 * inputs are checked at put time; intermediates are checked as they are
 * written, see DOPR_ERR_RANGE).
 * Errors: INVALID_ARG, UNKNOWN_DOC, INCOMPLETE, OUT_OF_MEMORY, CUDA, TIMEOUT,
 * RANGE, INTERNAL (checked builds).
 */
DOPR_API dopr_status dopr_score(dopr_model *model, dopr_store *store, int32_t n_pairs, const int32_t *q_offsets,
                       const int32_t *q_tokens, const int64_t *doc_ids, float *scores, void *cuda_stream,
                       int32_t io_on_device);

/*
 * The packing plan dopr_score uses (its device packer), copied to host
 * arrays, for testing.  Inputs as in dopr_score (host memory).  Outputs,
 * all host int32:
 *   perm     [n_pairs]    input index of the pair in sorted position s;
 *                         pairs are ordered by (doc_id, input index)
 *   tok_off  [n_pairs+1]  first packed token of sorted pair s
 *   tok_pos  [T]          RoPE position of packed token t (m_doc + j)
 *   tok_id   [T]          token id of packed token t (score token last)
 *   tok_pair [T]          sorted pair index of packed token t
 * with T = q_offsets[n_pairs] - q_offsets[0] + n_pairs.
 * Errors: as dopr_score.
 */
DOPR_API dopr_status dopr_debug_pack_plan(dopr_model *model, dopr_store *store, int32_t n_pairs, const int32_t *q_offsets,
                                 const int32_t *q_tokens, const int64_t *doc_ids, int32_t *perm, int32_t *tok_off,
                                 int32_t *tok_pos, int32_t *tok_id, int32_t *tok_pair);

/*
 * The attention tile plan of one document's run of pairs, computed on the
 * host exactly as dopr_score plans it (no device work: usable without a GPU),
 * for testing the tiling rule of the prefix-plus-causal attention (Sec. 3.4).
 *   m              the document's prefix length (keys), >= 0;
 *   rows_per_tile  tokens per tile (128 / G for G q heads per kv head), 1..128;
 *   n_pairs        pairs of the run, >= 1; tok_len [n_pairs] int32 >= 1: the
 *                  packed tokens (query + score token) of each pair, laid out
 *                  consecutively in this order;
 *   out            [max_tiles][24] int32, caller-owned; tile t, in token order:
 *                  {kind (0 = tensor-core tile of at most 256 key columns, 1 =
 *                  long tile), tok_begin, n_tok, n_keys, n_seg, 0, 0, 0,
 *                  seg[0..15]}, seg[s] = (visible tokens << 16) | (uint16_t)
 *                  (first token of the pair - tok_begin), one per pair the tile
 *                  touches, in pair order.
 * Returns the number of tiles (>= 1), or -DOPR_ERR_INVALID_ARG for bad
 * arguments or when max_tiles is too small (nothing is written then).
 */
DOPR_API int32_t dopr_debug_attention_plan(int32_t m, int32_t rows_per_tile, int32_t n_pairs, const int32_t *tok_len,
                                           int32_t max_tiles, int32_t *out);

/*
 * The dense projection kernel alone, for testing: C = A * B^T with A fp16
 * [M][K], B fp16 [N][K] (IEEE half, device pointers), fp32 accumulation.
 *   epilogue 0: out fp16 [M][N] = C
 *   epilogue 1: out fp32 [M][N] += C            (residual add)
 *   epilogue 2: out fp16 [M][N/2] = silu(G) * U, where B's rows come in
 *               blocks of 256: rows 256b..256b+127 are gate rows 128b.., rows
 *               256b+128..256b+255 the matching up rows (SwiGLU, Sec. 4.1 backbone)
 * Requires K % 64 == 0 and N % 256 == 0.  Runs on cuda_stream (NULL = default)
 * and returns after completion.  Errors: INVALID_ARG, UNSUPPORTED, CUDA, TIMEOUT.
 */
DOPR_API dopr_status dopr_debug_gemm(int32_t M, int32_t N, int32_t K, const void *A, const void *B, void *out,
                            int32_t epilogue, void *cuda_stream);

/*
 * Runs one test kernel whose bounded wait on a barrier that nothing
 * completes must give up after about timeout_ms milliseconds.  Returns
 * DOPR_ERR_TIMEOUT when the kernel reported the expired wait (the expected
 * result), DOPR_OK if it did not.  Used to check the timeout path of the
 * device waits without hanging the GPU.
 */
DOPR_API dopr_status dopr_debug_wait_timeout(int32_t timeout_ms);

/*
 * Allocation-free packing (the paper has no counterpart; this is a service
 * entry point of this library).  For callers that cannot allocate device
 * memory while they score -- their GPU memory is owned by another allocator
 * (e.g. a framework's caching pool), or cudaMalloc/cudaFree would stall a
 * latency-critical loop by synchronising the device -- this runs the same
 * device packer ordering step as dopr_score (pairs ordered by (doc_id, input
 * index), packed token offsets) using only caller buffers and a fixed scratch
 * array compiled into the library.  It calls no cudaMalloc/cudaFree.
 *   q_offsets [n_pairs+1] int32, doc_ids [n_pairs] int64: DEVICE memory,
 *             same meaning as in dopr_score.
 *   perm      [n_pairs] int32 DEVICE output: input index of sorted pair s.
 *   tok_off   [n_pairs+1] int32 DEVICE output: first packed token of sorted
 *             pair s (query tokens + the score token per pair).
 * Validation is dopr_score's: unknown or incomplete documents, decreasing
 * offsets and m + query length + 1 > max_position (the store's, which
 * dopr_score requires to equal the model's) fail the call.  The C ABI carries
 * no buffer sizes: the caller guarantees the extents above.
 * Limits: n_pairs <= 32768 and store max_doc_id < 131072; larger requests
 * return DOPR_ERR_UNSUPPORTED with a message and launch nothing.  The scratch
 * array (about 768 KiB) is held by every GPU that loads the library until the
 * process exits.  The first call on a device looks the array's device address
 * up (cudaGetSymbolAddress) with that device current; make that first call
 * before any stream capture.  Every call shares the one array: calls that
 * overlap on the GPU (other streams, other host threads) race and must be
 * serialised by the caller.  The call runs on cuda_stream (NULL = default)
 * and returns after its results are written (it synchronises the stream).
 * Errors: INVALID_ARG, UNKNOWN_DOC, INCOMPLETE, UNSUPPORTED, CUDA.
 */
DOPR_API dopr_status dopr_pack_order_noalloc(const dopr_store *store, int32_t n_pairs, const int32_t *q_offsets,
                                             const int64_t *doc_ids, int32_t *perm, int32_t *tok_off,
                                             void *cuda_stream);

/*
 * Per-kernel accounting, for measurement.  Every dopr_score call counts its
 * kernel launches per kernel family (pack, embed, gemm_qkv, qknorm_rope,
 * attention, gemm_o, rmsnorm, gemm_gate_up, gemm_down, score, prefix_store;
 * dopr_build_prefixes counts into the same families) together with
 * the algorithmic floating-point operations and device-memory bytes of those
 * launches (the minimum the operation needs: each input read once, each output
 * written once).  While enabled, each launch is also bracketed with CUDA
 * events on the call's stream and the elapsed device time summed per family.
 * dopr_profile_enable clears all counters.  dopr_profile_read copies up to
 * max_entries families into `out` and returns the number of families
 * (or -1 on a NULL model).
 */
typedef struct {
    char name[24];
    int64_t launches;
    double time_ms;   /* summed event time while enabled, else 0 */
    double flops;     /* algorithmic FLOPs                        */
    double bytes;     /* algorithmic device-memory bytes           */
} dopr_kernel_stat;

DOPR_API dopr_status dopr_profile_enable(dopr_model *model, int32_t enable);
DOPR_API int32_t dopr_profile_read(const dopr_model *model, dopr_kernel_stat *out, int32_t max_entries);

/* Thread-local message describing the last failed call on this thread
 * ("" if none).  The pointer stays valid until the next call on the thread. */
DOPR_API const char *dopr_last_error(void);

/* Library version string. */
DOPR_API const char *dopr_version(void);

#ifdef __cplusplus
}
#endif

#endif /* DOPR_H */
