/*
 * fe.h -- C-ABI of the GB300 joint evaluator (FlashEvaluator, arXiv 2603.02565).
 *
 * The library scores all K candidate sequences of each request in one pass
 * (the joint mapping E_theta(z) in R^K of Section 3) and selects
 * argmax_k s_k (Eq. 1).  It follows the QKV-Cache structure of Section 4:
 *   1. the request context is encoded once into per-layer keys/values
 *      (Section 4.2, "context-side key and value representations ... computed
 *      only once");
 *   2. every DISTINCT element of U(z) = union of the K sequences
 *      (Section 4.1) gets its request-conditioned representation once
 *      (cross-attention to the context + FFN; the Q-Cache of Section 4.2);
 *   3. sequences are assembled by integer index plus position embeddings added
 *      after indexing, prefixed with [CLS] and pooled by SeqEnc (Section 4.3);
 *   4. self-attention across the K sequence vectors, then a shared score head
 *      (Section 4.4), then the argmax of Eq. 1 (ties -> smallest k).
 *
 * Model definition (the paper leaves block internals open; these are the
 * readings this library implements):
 *   LN(x)   = (x - mean) / sqrt(var + ln_eps), biased var, no affine params.
 *   MHA     = per head softmax(q_h k_h^T / sqrt(d_h)) v_h, heads are
 *             contiguous column blocks of width d_h = d / n_heads.
 *   context : X = LN(context); K_l = X WK_l, V_l = X WV_l       (l < n_layers)
 *   element : h = pool row; per layer: h += MHA(LN(h) WQ_l, K_l, V_l) WO_l;
 *             h += ReLU(LN(h) W1_l + b1_l) W2_l + b2_l;  H = LN(h)
 *   SeqEnc  : x_0 = cls, x_j = H[i_{k,j}] + P[j-1];  o = MHA(x_0 WQs, x WKs, x WVs)
 *             c = cls + o WOs;  c += ReLU(LN(c) W1s + b1s) W2s + b2s
 *   cross   : C' = C + MHA(Z WQx, Z WKx, Z WVx) WOx,  Z = LN(C)  (over the K rows)
 *   head    : s_k = ReLU(LN(C'_k) W1h + b1h) . w2h + b2h
 *
 * Arithmetic: bf16 tensor-core products with fp32 accumulation.  Activations
 * feeding a product are carried as an unevaluated pair of bf16 values
 * (hi + lo), so each product is hi*W + lo*W (plus hi*W_lo when the weights
 * are not exactly bf16); softmax, LayerNorm and residual streams are fp32.
 *
 * Threading: a context is not thread-safe; calls on one context must be
 * serialised (one in flight at a time per context).  Different contexts are
 * independent.
 */
#ifndef FE_H_
#define FE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Return codes.  No exception ever crosses this boundary. */
enum {
  FE_OK = 0,
  FE_ERR_INVALID_ARG = 1,   /* null pointer, negative or zero size where >0 is required  */
  FE_ERR_UNSUPPORTED = 2,   /* shape outside the limits listed below                     */
  FE_ERR_INDEX = 3,         /* some cand_idx outside [0, M): those requests get NaN / -1 */
  FE_ERR_WORKSPACE = 4,     /* workspace could not be sized for the call                 */
  FE_ERR_OOM = 5,           /* device allocation failed                                  */
  FE_ERR_CUDA = 6,          /* a CUDA call failed (message in fe_last_error_message)     */
  FE_ERR_NUMERIC = 7,       /* a request produced a NaN score: its best index is -1      */
  FE_ERR_TIMEOUT = 8        /* a bounded device-side wait gave up; results are invalid   */
};

/* Element type of the context / pool inputs. */
enum { FE_IO_BF16 = 0, FE_IO_F32 = 1 };

typedef struct fe_config {
  int32_t d;          /* model width; multiple of 32, 32 <= d <= 512                  */
  int32_t n_heads;    /* heads; d / n_heads must be 32 or 64                          */
  int32_t n_layers;   /* depth of the element cross-attention stack, 1..8            */
  int32_t ffn_mult;   /* FFN width F = ffn_mult * d, 1..8 (the readings use 4)        */
  int32_t max_L;      /* rows of the position table P; sequences have L <= max_L     */
  int32_t io_dtype;   /* FE_IO_BF16 or FE_IO_F32 for context and pool                 */
  float   ln_eps;     /* LayerNorm epsilon (1e-5)                                     */
  int32_t n_tasks;    /* task-specific prediction heads T (end of Section 4.4): 0 or 1
                         is the single shared head; 2..4 add a fusion module
                         s_k = sum_t fuse_w[t] s_{k,t} + fuse_b (T * d <= 512)      */
  int32_t no_cross_seq; /* 1: the variant without cross-sequence interaction
                         (Appendix B.4, "- CrossSeq"): C' = C; 0: the full model    */
  int32_t elem_self_attn; /* 1: self-attention over the request's element set before
                         the cross-attention stack, H^(1) of Section 4.2:
                         h += MHA(LN(h) WQe, LN(h) WKe, LN(h) WVe) WOe over the set  */
  int32_t encode_pool;  /* 1: the element set is the whole pool (U(z) = C(x), U = M,
                         Section 4.1) instead of the distinct sequence elements    */
  int32_t linear_context_attn; /* 1: the element -> context attention is linear
                         (kernelized) attention with phi(x) = elu(x) + 1, as the
                         online deployment uses for long contexts (Appendix B.3):
                         per request, layer and head the context is a d_h x d_h
                         state S = phi(K)^T V with z = sum phi(K); an element
                         reads phi(q) S / (phi(q) . z)                           */
} fe_config;

typedef struct fe_ctx fe_ctx;

/*
 * Number of floats fe_init expects in `weights`, for this configuration.
 * Returns 0 for an invalid configuration.
 *
 * Weight order (all fp32, row-major, y = x W with W stored [in, out]):
 *   for l in 0..n_layers-1:
 *     WQ_l[d,d] WK_l[d,d] WV_l[d,d] WO_l[d,d] W1_l[d,F] b1_l[F] W2_l[F,d] b2_l[d]
 *   P[max_L,d] cls[d] WQs[d,d] WKs[d,d] WVs[d,d] WOs[d,d] W1s[d,F] b1s[F] W2s[F,d] b2s[d]
 *   WQx[d,d] WKx[d,d] WVx[d,d] WOx[d,d]          (absent when no_cross_seq = 1)
 *   for t in 0..T-1 (T = max(n_tasks, 1)):
 *     W1h_t[d,d] b1h_t[d] w2h_t[d] b2h_t[1]      (task t's head)
 *   fuse_w[T] fuse_b[1]                          (only when T >= 2)
 *   WQe[d,d] WKe[d,d] WVe[d,d] WOe[d,d]          (only when elem_self_attn = 1)
 */
size_t fe_weight_count(const fe_config* cfg);

/*
 * Create a context on the current CUDA device: validates `cfg`, copies the
 * weights (host memory, fe_weight_count(cfg) floats, caller keeps ownership)
 * to the device and precomputes the weight-only products of SeqEnc
 * ([CLS] WQs, [CLS] WKs, [CLS] WVs, P WKs, P WVs).  Weights whose values are
 * all bf16-representable are stored as one bf16 plane, others as a hi/lo pair.
 * On success *out owns device memory until fe_destroy.
 * Errors: FE_ERR_INVALID_ARG, FE_ERR_UNSUPPORTED, FE_ERR_OOM, FE_ERR_CUDA.
 */
int fe_init(const fe_config* cfg, const float* weights, size_t n_floats, fe_ctx** out);

/*
 * Weight blob: the parameters theta of the evaluator E_theta (Section 3)
 * together with their configuration, as one self-describing buffer (a file
 * on disk, for example).  The paper defines no storage format; this one is
 * the library's.  Layout, every field little-endian:
 *   bytes  0..3    magic "FEW1"
 *   bytes  4..7    uint32 version, 1
 *   bytes  8..55   the twelve fe_config fields in declaration order, 4 bytes
 *                  each (int32, except ln_eps: IEEE-754 float32)
 *   bytes 56..63   uint64 n = fe_weight_count(config)
 *   bytes 64..     n float32 weights in the order fe_weight_count documents
 * fe_blob_parse checks a blob on the host (no CUDA call): magic, version,
 * configuration, n and the total size, which must be exactly 64 + 4 n bytes.
 * On success it writes the configuration to *cfg_out and n to *n_floats_out
 * (when not NULL).  Errors: FE_ERR_INVALID_ARG (null pointer, wrong magic,
 * n or size), FE_ERR_UNSUPPORTED (a version other than 1, or a configuration
 * that fe_init refuses).
 * fe_init_blob is fe_blob_parse followed by fe_init with the blob's weights;
 * the blob stays caller-owned and may be freed when the call returns.  Same
 * errors as both.
 */
int fe_blob_parse(const void* blob, size_t bytes, fe_config* cfg_out, size_t* n_floats_out);
int fe_init_blob(const void* blob, size_t bytes, fe_ctx** out);

/*
 * Size the device workspace for batches up to (B, C, M, K, L) and build the
 * TMA descriptors for it.  Optional: fe_evaluate grows the workspace itself
 * when a call exceeds the reserved shape (that call then allocates).
 * Limits: 1 <= C <= 65536, M <= 262144, K <= 4096, L <= max_L, B <= 65535.
 * Errors: FE_ERR_INVALID_ARG, FE_ERR_UNSUPPORTED, FE_ERR_OOM, FE_ERR_CUDA.
 */
int fe_reserve(fe_ctx* ctx, int B, int C, int M, int K, int L);

/*
 * Score a batch of B requests (device pointers, contiguous row-major):
 *   context  [B, C, d]  io_dtype     request contexts (x of Section 3)
 *   pool     [B, M, d]  io_dtype     candidate pools C(x), one row per element
 *   cand_idx [B, K, L]  int32        sequence k of request b is the pool rows
 *                                    cand_idx[b,k,0..L-1] (L_k of Section 3)
 *   scores_out [B, K]   float32      s_k of Section 4.4 (the fused score with
 *                                    several task heads)
 *   best_out   [B]      int32        argmax_k s_k, smallest k on ties (Eq. 1)
 * The work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 * stream) and the call waits for it, then returns the batch status:
 *   FE_ERR_INDEX   some request had an index outside [0, M): that request's
 *                  scores are NaN and its best index -1; others are valid.
 *   FE_ERR_NUMERIC some request produced a NaN score (best index -1).
 * Inputs must be 16-byte aligned.  The caller owns every buffer.  Repeated
 * calls with the same shape and pointers replay one captured CUDA graph.
 */
int fe_evaluate(fe_ctx* ctx, int B, int C, int M, int K, int L,
                const void* context, const void* pool, const int32_t* cand_idx,
                float* scores_out, int32_t* best_out, void* stream);

/*
 * As fe_evaluate, but returns right after enqueueing (argument errors are
 * still reported immediately).  The batch status of the most recent call is
 * returned by fe_last_status, which waits for that call to finish.
 */
int fe_evaluate_async(fe_ctx* ctx, int B, int C, int M, int K, int L,
                      const void* context, const void* pool, const int32_t* cand_idx,
                      float* scores_out, int32_t* best_out, void* stream);
int fe_last_status(fe_ctx* ctx);

/*
 * As fe_evaluate, for callers whose buffers live in HOST memory (same shapes
 * and types).  Copies the inputs to library-owned device buffers on `stream`,
 * evaluates, copies scores and best indices back and waits.  Page-locked host
 * buffers give the fastest copies; pageable ones work.
 */
int fe_evaluate_host(fe_ctx* ctx, int B, int C, int M, int K, int L,
                     const void* context, const void* pool, const int32_t* cand_idx,
                     float* scores_out, int32_t* best_out, void* stream);

/*
 * The candidate-factorized evaluation E^ind of the same model and weights
 * (Appendix A.3: every candidate scored as if on its own).  Same arguments
 * and outputs as fe_evaluate_async (it returns after enqueueing; the batch
 * status comes from fe_last_status), and the same scores: only the cost
 * structure changes.  The context K/V are recomputed for every candidate
 * sequence (B*K*C context rows instead of B*C) and every occurrence of an
 * element is encoded on its own (B*K*L element rows instead of the B*|U(z)|
 * distinct ones); the SeqEnc, cross-sequence and head steps are unchanged.
 * Timing it against fe_evaluate on the same batch measures T_joint / T_ind
 * (Section 5.2 relates it to 1/rho, rho = K*L / |U(z)|).  Requires d <= 128,
 * bf16 inputs and weights and C a multiple of 128 (else FE_ERR_UNSUPPORTED);
 * the workspace it reserves (K-fold context K/V) stays allocated.  The layout
 * hook (fe_debug_layout) then reports U_b = K*L and the identity slots
 * (-1 for rejected requests).
 */
int fe_evaluate_factorized(fe_ctx* ctx, int B, int C, int M, int K, int L,
                           const void* context, const void* pool, const int32_t* cand_idx,
                           float* scores_out, int32_t* best_out, void* stream);

/*
 * Pipelined form of fe_evaluate_host for serving loops whose inputs arrive in
 * host memory.  fe_submit_host enqueues one batch and returns at once: the
 * inputs are copied to one of three library-owned device staging slots on
 * the library's own copy stream, the batch runs on the library's own compute
 * stream once its copy is complete, and scores/best are copied back into the
 * caller's host buffers.  The copy of one batch therefore overlaps the
 * evaluation of the previous ones; every batch still moves its own inputs and
 * results across the host link.  fe_wait_host waits for the oldest
 * outstanding submission and returns its batch status (as fe_evaluate).
 * At most three submissions may be outstanding (a fourth returns
 * FE_ERR_INVALID_ARG); with three, a slot's next copy may start as soon as
 * the batch two submissions back has completed, so the host's wake-up and
 * submission latency stays off the device's critical path.  The host
 * buffers of a submission must stay valid and
 * unchanged until its fe_wait_host returns (page-locked buffers for overlap).
 * While submissions are outstanding, fe_evaluate, fe_evaluate_async and
 * fe_evaluate_host return FE_ERR_INVALID_ARG (they share the workspace), and a
 * batch larger than the reserved workspace is refused until every submission
 * has been waited for.  Same shapes, types and status codes as fe_evaluate.
 * The paper evaluates one request batch at a time; this overlap of transfer
 * and compute across batches is the library's own.
 */
int fe_submit_host(fe_ctx* ctx, int B, int C, int M, int K, int L,
                   const void* context, const void* pool, const int32_t* cand_idx,
                   float* scores_out, int32_t* best_out);
int fe_wait_host(fe_ctx* ctx);

/*
 * Test hook: the distinct-element layout of the last evaluated batch, copied
 * to host memory.  U_out[B] = |U(z_b)| (Section 4.1); slot_out[B,K,L] = rank of
 * cand_idx[b,k,j] among the distinct indices of request b in ascending order
 * (-1 for requests rejected with FE_ERR_INDEX).  Waits for the last call.
 */
int fe_debug_layout(fe_ctx* ctx, int32_t* slot_out, int32_t* U_out);

/*
 * Test hook: copy an intermediate of the last batch to host memory as fp32,
 * row-major.  `name` is one of:
 *   "ctx_ln"  [B*C, d]      LN(context); only where it is materialised: with
 *                           d <= 128, bf16 inputs and bf16-exact weights the
 *                           context LayerNorm and K/V projection run as one
 *                           kernel and this name returns FE_ERR_UNSUPPORTED
 *   "ctx_kv"  [B*C, 2*n_layers*d]  K_0 | V_0 | K_1 | V_1 ... (held as f16, the
 *                           attention operand precision)
 *   "elem"    [sum U, d]    H, the final element representations, requests in
 *                           order, each request's elements in ascending pool index
 *   "seq"     [B*K, d]      c_k, the SeqEnc output
 *   "cross"   [B*K, d]      C', the cross-sequence output (FE_ERR_UNSUPPORTED
 *                           when no_cross_seq = 1: C' = C is "seq")
 *                           (both FE_ERR_UNSUPPORTED when the sequence-stage
 *                           kernel kept them on chip: see
 *                           fe_debug_keep_intermediates)
 *   "task_scores" [B*K, T]  every task head's score s_{k,t} before the fusion
 *                           (T = 1: the score itself)
 * `max_floats` is the capacity of `dst`; *n_floats receives the element count
 * (also when dst is NULL).  Waits for the last call.
 */
int fe_debug_fetch(fe_ctx* ctx, const char* name, float* dst, size_t max_floats,
                   size_t* n_floats);

/*
 * Test hook: with on = 1, later batches also store the SeqEnc output c and the
 * cross-sequence output C' ("seq" and "cross" of fe_debug_fetch) where the
 * sequence-stage kernel otherwise keeps them on chip (d = 128, K <= 128,
 * L <= 31, one score head, bf16-exact weights); on = 0 stops it.  The extra
 * stores cost time.  Errors: FE_ERR_INVALID_ARG, FE_ERR_CUDA.
 */
int fe_debug_keep_intermediates(fe_ctx* ctx, int on);

/*
 * Tracing.  fe_profile(ctx, 1) makes later evaluations launch kernel by kernel
 * (no graph) with a pair of CUDA events on the caller's stream around every
 * launch; fe_profile(ctx, 0) returns to graph replay.  fe_profile_read waits
 * for the recorded work and reports, per launch site (in launch order):
 *   names     site names, max_sites x 32 chars, NUL-terminated
 *   launches  launches recorded at the site
 *   total_ms  summed event time of those launches
 * and clears the counters.  *n_sites receives the number of sites.
 * fe_kernels_per_batch returns how many kernels the last batch launched.
 */
int fe_profile(fe_ctx* ctx, int enable);
int fe_profile_read(fe_ctx* ctx, int max_sites, char* names, int* launches, double* total_ms, int* n_sites);
int fe_kernels_per_batch(fe_ctx* ctx);

/*
 * Distinct-element layout without any device allocation.  The paper has no
 * counterpart: this entry point exists for callers that are not allowed to
 * allocate GPU memory -- for example a serving runtime whose memory pool owns
 * the device and forbids cudaMalloc after start-up, or code that must not
 * trigger the implicit synchronisation an allocation can cause.
 *
 * It computes what the first stage of fe_evaluate computes, with no fe_ctx:
 *   U_out    [B]        int32, device: number of distinct pool rows of request b
 *                       (0 for a request with an index outside [0, M))
 *   slot_out [B, K, L]  int32, device: rank of cand_idx[b,k,j] among request b's
 *                       distinct rows in ascending order (-1 for such a request)
 * from cand_idx [B, K, L] int32 on the device.  The work is enqueued on
 * `stream` and the call returns without waiting.
 *
 * Scratch (offsets, flags, distinct lists, a status word and a counter) lives
 * in a fixed file-scope device array of 4.5 MiB that every GPU loading
 * the library holds until the process exits.  Limits: B <= 65536,
 * M <= 262144 and B * min(M, K*L) <= 1048576; larger batches are rejected with
 * FE_ERR_UNSUPPORTED before anything is enqueued.  The call allocates nothing:
 * no cudaMalloc, no cudaFree, no allocating library routine.
 *
 * The first call on a device looks up the array's device address and sets a
 * kernel attribute on that device; make that first call before any stream
 * capture.  All calls on a device share the one array and each call clears
 * the part that must start at zero, so calls whose work overlaps on the GPU
 * (different streams, no ordering between them) race and corrupt each other.
 * Returns FE_OK, FE_ERR_INVALID_ARG, FE_ERR_UNSUPPORTED or FE_ERR_CUDA.
 */
int fe_distinct_layout_noalloc(const int32_t* cand_idx, int B, int M, int K, int L,
                               int32_t* U_out, int32_t* slot_out, void* stream);

/*
 * Test hook for the allocation-failure path (no counterpart in the paper).
 * fail_at > 0 makes the fail_at-th device or page-locked allocation that the
 * library makes from now on fail as if the device were out of memory: the
 * entry point making it returns FE_ERR_OOM after releasing what it had
 * allocated (fe_init leaves no context; a failed workspace grow leaves the
 * context with no workspace, and its next call reserves again).  0 disarms
 * the hook; a negative value leaves it as it is.  *live_out, when not NULL,
 * receives the number of the library's allocations that are live, over all
 * contexts.  The setting is process-wide; host only; returns FE_OK.
 */
int fe_debug_alloc_hook(int fail_at, int64_t* live_out);

/*
 * Test hook for the bounded device-side waits (no counterpart in the paper).
 * Enqueues on `stream` one thread that waits, through the batch kernels' own
 * bounded mbarrier wait, on a barrier that nothing arrives on, with a limit of
 * limit_us microseconds (1..1000000) instead of the batch kernels' one
 * second; no copy or tensor-core work is in flight.  The status word then
 * reaches the host as a batch's does (copied to the page-locked word and
 * cleared), so the call waits and returns FE_ERR_TIMEOUT; the context stays
 * usable for the next batch.  Reserves a minimal workspace when the context
 * has none.  Errors: FE_ERR_INVALID_ARG (null context, limit out of range,
 * host submissions outstanding), FE_ERR_CUDA.
 */
int fe_debug_wait_probe(fe_ctx* ctx, uint32_t limit_us, void* stream);

/* Release every device resource owned by ctx (waits for its work first). */
int fe_destroy(fe_ctx* ctx);

/* Static description of a return code. */
const char* fe_strerror(int code);

/* Thread-local detail of the last FE_ERR_CUDA / FE_ERR_UNSUPPORTED on this thread. */
const char* fe_last_error_message(void);

#ifdef __cplusplus
}
#endif

#endif /* FE_H_ */
