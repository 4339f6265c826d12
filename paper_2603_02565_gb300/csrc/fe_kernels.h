// Internal interface between the host orchestration (fe_api.cu) and the
// kernels (fe_gemm.cu, fe_attn.cu, fe_misc.cu).  Not part of the C-ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace fe {

typedef __nv_bfloat16 bf16;

// Device status bits, OR-ed into the per-batch status word.
enum : int {
  ST_INDEX = 1,    // a request had an out-of-range candidate index
  ST_NUMERIC = 2,  // a request produced a NaN score
  ST_TIMEOUT = 4,  // a bounded wait gave up
};

// Whether batch kernels are launched with programmatic stream serialisation
// (overlapping each kernel's launch and prologue with its predecessor's tail).
// On unless the environment sets FE_NO_PDL=1.
bool pdl_enabled();

template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                            Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl_enabled() ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// The same launch with thread-block clusters of cs CTAs along x (cs > 1).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_kc(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, int cs,
                             Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl_enabled() ? 1 : 0;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)cs;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cs > 1 ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// ---------------------------------------------------------------------------
// tcgen05 GEMM:  D[r, n] = sum over planes  A_p[r, :] . B_q[n, :]
// A: activation as two bf16 planes (hi, lo), row-major [rows, K_pad]
// B: weights transposed, [N, K_pad], one or two bf16 planes (hi[, lo])
// Persistent CTAs walk 128 x BN tiles; BN <= 512 (two N=256 MMAs above 256).
// ---------------------------------------------------------------------------
// Eq. 1's argmax fused into the kernel that computes the scores (fe_select.cuh).
struct SelArgs {
  unsigned long long* keys;  // [B], zero at launch
  int* nan;                  // [B], zero at launch
  unsigned* ticket;          // zero at launch
  const int* bad;            // [B]
  int32_t* best;             // [B]
  int B, K;
  int* status;               // the batch status word
  int* host_status;          // page-locked host word (device-accessible)
};

enum GemmEpilogue : int {
  EPI_STORE = 0,    // out = [ReLU](acc + bias) as split planes
  EPI_RESID_LN = 1, // x = resid + acc + bias -> x_out (fp32) and LN(x) as split planes; BN == N
                   // (or N = cs BN over a cluster)
  EPI_HEAD = 2,     // task heads s_t = ReLU(acc_t + bias_t) . w2_t + b2_t over column blocks of
                   // head_d, fused s = sum_t fuse_w[t] s_t + fuse_b (one task: s = s_0); BN == N
  EPI_LN_FOLD = 3,  // LN(x) W from the raw rows x: out = rstd (acc - mu colsum(W)) as one f16 plane;
                   // A is ONE exact bf16 plane (a_l unused), (mu, rstd) per row in row_stats
};

struct GemmParams {
  int rows;             // row extent of the A descriptors
  const int* rows_dev;  // when set: number of valid rows, read on the device
  int N;                // output columns
  int BN;               // columns per CTA (multiple of 32, <= 512)
  int K_pad;            // reduction length, multiple of 64
  int nb;               // weight planes: 1 (exact bf16) or 2 (hi + lo)
  int stages;           // shared-memory pipeline depth (chosen by gemm_launch)
  int nacc;             // TMEM accumulators, 1 or 2 (chosen by gemm_launch)
  int cs;               // EPI_RESID_LN: CTAs per cluster sharing one row tile (N = cs * BN, BN <= 128), 0/1: none
  const float* bias;    // [N] or null
  int relu;
  int out_f16;          // EPI_STORE: one f16 plane through o_h (attention operands) instead of bf16 hi/lo
  // EPI_STORE: output columns below lq_n are not stored; each 32-column chunk c of such a row r leaves
  // as the partial dot product logits[r * ld_logit + c / 32] = sum_i out[r, c + i] lq[c + i]
  const float* lq;
  int lq_n;
  float* logits;
  int ld_logit;
  // EPI_RESID_LN (outputs through the o_x / o_h / o_l tensor maps)
  const float* resid;   // residual rows (ldr == 0: one row broadcast to every row)
  int ldr;
  float eps;
  // EPI_LN_FOLD
  const float2* row_stats;  // [rows] (mean, rstd) of the raw rows
  const float* colsum;      // [N] column sums of W
  // EPI_HEAD
  int n_tasks;          // 1..4 heads of head_d columns each (columns past n_tasks * head_d are padding)
  int head_d;
  const float* w2;      // [N]
  const float* b2;      // [n_tasks]
  const float* fuse_w;  // [n_tasks] (n_tasks > 1)
  const float* fuse_b;  // [1] (n_tasks > 1)
  float* scores;        // [rows]
  float* task_scores;   // [rows, n_tasks] or null
  // EPI_HEAD with sel.keys: the argmax of Eq. 1 fused into the epilogue (fe_select.cuh)
  SelArgs sel;
  int* status;
};

// Raises the dynamic shared-memory limit of the GEMM kernels (call once per device, outside capture).
cudaError_t gemm_prepare();
size_t gemm_smem_bytes(int BN, int nb, int stages, int cs = 1, int na = 2);
int gemm_max_stages(int BN, int nb, int K_pad, int cs = 1, int na = 2);
// Clusters of cs CTAs (2, 4 or 8) that can be resident at once for the EPI_RESID_LN kernels (0 when
// such clusters cannot be scheduled, or when FE_GEMM_CLUSTERS=0); valid after gemm_prepare.
int gemm_cluster_capacity(int cs);
// o_h / o_l: output bf16 planes (EPI_STORE: the product, EPI_RESID_LN: LN(x)), tensor maps with
// 32 x 32 boxes and the 64-byte swizzle; o_x: the fp32 x_out rows of EPI_RESID_LN, 32 x 32 boxes,
// 128-byte swizzle.  Unused maps may be null.
cudaError_t gemm_launch(int epi, const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* b_h,
                        const CUtensorMap* b_l, const CUtensorMap* o_h, const CUtensorMap* o_l,
                        const CUtensorMap* o_x, const GemmParams& p, cudaStream_t s);

// ---------------------------------------------------------------------------
// Attention output projection + FFN block for rows of width d <= 128 (fe_ffn.cu):
//   x = x0 + A W_O,   x_out = x + ReLU(LN(x) W1 + b1) W2 + b2, and LN(x_out),
// optionally followed by a tail product LN(x_out) W_t (N = tail_n <= 256).
// A: attention output planes (64 x 128 boxes, 128-byte swizzle); W_O^T [d, d_pad]
// and W2^T [d, F_pad] planes with 64 x d boxes; W1^T [F, d_pad] planes with
// 64 x 128 boxes; W_t^T [tail_n, d_pad] planes with 64 x tail_n boxes.  o_x:
// x_out (fp32, 32 x 32 boxes); o_h / o_l: LN(x_out) planes with 64 x 128
// boxes and the 128-byte swizzle (stored when store_ln); to_h / to_l: the tail
// output, one f16 plane (tail_f16) or a split pair, 32 x 32 boxes with the
// 64-byte swizzle.  x0 rows are fp32 [rows, ldx0] (o_x may write the same
// rows), or one row x0_row added to every row.
// ---------------------------------------------------------------------------
struct FfnParams {
  int rows;             // row extent of the A descriptors
  const int* rows_dev;  // when set: number of valid rows, read on the device
  int d, d_pad, F, nb;
  const float* b1;      // [F]
  const float* b2;      // [d]
  const float* x0;      // block input rows, unless x0_row is set
  int ldx0;             // multiple of 4
  const float* x0_row;  // [d], when set: the same input row for every row
  int tail_n;           // 0: no tail product
  int tail_f16;         // tail output as one f16 plane (else a split pair)
  int store_ln;         // store LN(x_out)
  float eps;
  int* status;
  // With tail_q0 set (a split-pair tail of 2d columns, keys | values of SeqEnc):
  // the key columns are not stored; each 32-column group g of them is reduced
  // with q0 (the [CLS] query cls WQs, fp32 [d]) and written to
  // tail_logits[row * (d / 32) + g] (fp32); the value columns are stored as usual.
  const float* tail_q0;
  float* tail_logits;
  int tail_col0;        // tail output column c is stored at column c - tail_col0 of the output map
};
// The same block for rows of width d = 256 (fe_ffn256.cu): x0 + A W_O, the
// FFN, x_out (fp32, in place over x when x0_row is null), LN(x_out) (split
// pair, by TMA through o_h / o_l, when store_ln), and with tail the next
// layer's Q = LN(x_out) W_Q as f16 rows.  Weights are bf16-exact transposed
// planes read through 64 x 128 boxes: W_O^T and W_Q^T [256, 256], W1^T
// [F, 256], W2^T [256, F].
struct Ffn256Params {
  int rows;             // row extent of the A descriptors
  const int* rows_dev;  // when set: number of valid rows, read on the device
  int F;
  const float* b1;      // [F]
  const float* b2;      // [256]
  float* x;             // [rows, ldx]: x0 in (unless x0_row), x_out out
  int ldx;              // multiple of 4
  const float* x0_row;  // [256], when set: the same input row for every row
  int store_ln;
  int tail;
  float eps;
  int* status;
};
bool ffn256_supported(int d, int F, int nb);
cudaError_t ffn256_prepare();
// x_st: fp32 x rows, 32 x 32 boxes (128-byte swizzle); q_st: Q rows, 64 x 128 boxes (128-byte swizzle)
cudaError_t ffn256_launch(const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* wo, const CUtensorMap* w1,
                          const CUtensorMap* w2, const CUtensorMap* wt, const CUtensorMap* o_h, const CUtensorMap* o_l,
                          const CUtensorMap* x_st, const CUtensorMap* q_st, const Ffn256Params& p, cudaStream_t s);
bool ffn_supported(int d, int d_pad, int F, int nb);
bool ffn_tail_supported(int d, int d_pad, int F, int nb, int tail_n, int tail_f16);
cudaError_t ffn_prepare();
cudaError_t ffn_launch(const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* wo_h,
                       const CUtensorMap* wo_l, const CUtensorMap* w1_h, const CUtensorMap* w1_l,
                       const CUtensorMap* w2_h, const CUtensorMap* w2_l, const CUtensorMap* o_h,
                       const CUtensorMap* o_l, const CUtensorMap* o_x, const CUtensorMap* t_h,
                       const CUtensorMap* t_l, const CUtensorMap* to_h, const CUtensorMap* to_l,
                       const FfnParams& p, cudaStream_t s);

// ---------------------------------------------------------------------------
// Distinct-element gather + LayerNorm + the first layer's Q projection in one
// kernel (fe_embed.cu), for d <= 128, bf16 pool rows and bf16-exact WQ:
//   h[r] = pool[b M + list[b cap + r - off[b]]] (fp32), Q[r] = LN(h[r]) WQ (f16)
// w: WQ^T [d, d_pad] bf16, 64 x d boxes, 128-byte swizzle; q_out: Q's f16
// store map (32 x 32 boxes, 64-byte swizzle).  Rows past off[B] are not written.
// ---------------------------------------------------------------------------
struct EmbedParams {
  const bf16* pool;     // [B * M, d]
  int B, M, cap;
  const int* off;       // [B + 1] row offsets of the requests' distinct elements
  const int* list;      // [B, cap] the distinct elements' pool rows within their request
  int rows;             // row extent of h and Q
  int d, d_pad;
  float eps;
  float* h;             // [rows, ldh] fp32
  int ldh;
  int* status;
};
bool embed_q_supported(int d, int d_pad, int nb, int io_f32);
cudaError_t embed_q_prepare();
cudaError_t embed_q_launch(const CUtensorMap* w, const CUtensorMap* q_out, const EmbedParams& p, cudaStream_t s);

// ---------------------------------------------------------------------------
// Context LayerNorm + K/V projection in one kernel (d <= 128, bf16 inputs,
// bf16-exact weights, N = 2 * n_layers * d in {256, 512}).
// x: raw context rows [rows, d] bf16, 64 x 128 boxes, 128-byte swizzle;
// w: W^T [N, d_pad] bf16, 64 x 128 boxes, 128-byte swizzle;
// o: the f16 K/V, head-major: [N / dh blocks][rows][dh] (block = one head of
// K_l or V_l), 3D map with 32 x 32 x 1 boxes, 64-byte swizzle.
// ---------------------------------------------------------------------------
struct CtxKvParams {
  int rows, d, N, dh;
  float eps;
  int* status;
  // output row r reads context row ((r / C) / rep) * C + r % C: rep = 1 for one
  // K/V per request, rep = K for one per candidate sequence (C % 128 == 0)
  int C, rep;
  // linear-attention state mode (non-null): no K/V is written; the states
  // [segment = row / C][layer][head][dh*dh + dh] receive phi(K)^T V and
  // sum phi(K) (feature map elu + 1) over the segment's rows
  float* states;
};
bool ctxkv_supported(int d, int d_pad, int N, int nb, int io_f32);
// whether the state mode applies: two layers (N = 4d), d in {64, 128}, dh in {32, 64}, C % 128 == 0
bool ctxkv_state_supported(int d, int d_pad, int N, int dh, int C);
cudaError_t ctxkv_prepare();
cudaError_t ctxkv_launch(const CUtensorMap* x, const CUtensorMap* w, const CUtensorMap* o, int d_pad,
                         const CtxKvParams& p, cudaStream_t s);

// ---------------------------------------------------------------------------
// Flash-style multi-head attention over request segments (tcgen05, f16
// operands, fp32 accumulation and softmax).  Segment b: query rows
// [q_off(b), q_off(b) + q_cnt(b)), key and value rows
// [b * kv_stride, b * kv_stride + kv_cnt), or, with kv_self, the segment's
// own rows [q_off(b), q_off(b) + q_cnt(b)) (self-attention within segments).  Head h reads columns q_col + h*dh
// of Q, k_col + h*dh of K, v_col + h*dh of V (each one f16 plane) and writes
// columns o_col + h*dh of the bf16 hi/lo output planes.  The Q map has boxes
// of dh x 128, the K/V maps dh x (64 for dh = 32, else 128), with the 64-byte
// (dh = 32) or 128-byte (dh = 64) swizzle.
// ---------------------------------------------------------------------------
struct AttnParams {
  int n_segments, n_heads;
  int max_q;             // largest q_cnt of any segment (grid sizing)
  int max_q_tiles;       // set by attn_launch
  const int* q_off_dev;  // null: q_off = b * q_stride
  const int* q_cnt_dev;  // null: q_cnt = q_cnt_fixed
  int q_stride;
  int q_cnt_fixed;
  int kv_stride;
  int kv_cnt;
  int q_col, k_col, v_col, o_col;
  int kv3d;              // K/V head-major (3D maps: x within the head, row, block = column / dh)
  int kv_self;           // keys / values are the segment's query rows (kv_stride, kv_cnt unused)
  int kv_seg;            // V through a 3D map [segment][kv_cnt][col]: rows past kv_cnt read as zeros
  bf16 *o_h, *o_l;
  int ldo;
  float scale_log2;      // log2(e) / sqrt(d_h)
  int* status;
};
cudaError_t attn_prepare();
// Keys per chunk of the attention kernel for head size dh: the row count of the
// key/value tensor-map boxes (tK, tV) that attn_launch expects.
int attn_chunk_keys(int dh);
cudaError_t attn_launch(int dh, const CUtensorMap* q, const CUtensorMap* k, const CUtensorMap* v, const AttnParams& p,
                        cudaStream_t s);

// ---------------------------------------------------------------------------
// Linear-attention context module (fe_linattn.cu): feature map elu(x) + 1.
// lin_state: for segment s (context rows [s*C, s*C + C)), layer l, head h:
//   states[((s * Ly + l) * H + h) * SB ...] = S [dh][dh] (row-major) | z [dh],
//   SB = dh*dh + dh, S = sum_c phi(K_l[c,h]) V_l[c,h]^T, z = sum_c phi(K_l[c,h]);
//   kv holds K_l | V_l column blocks (f16), head-major (hm: [col/dh][rows_alloc][dh])
//   or row-major [rows][ld].
// lin_attn: element rows [off(s), off(s) + cnt(s)) of segment s read layer l:
//   out[row, h*dh + j] = (phi(q_h) S)_j / (phi(q_h) . z), written as a bf16 hi/lo pair.
// ---------------------------------------------------------------------------
cudaError_t linattn_prepare();
cudaError_t lin_state_launch(const bf16* kv, int hm, int rows_alloc, int ld, int n_seg, int C, int d, int dh, int Ly,
                             int H, float* states, cudaStream_t s);
cudaError_t lin_attn_launch(const bf16* q, int ldq, const float* states, int n_seg, int Ly, int l, int H, int dh,
                            const int* off_dev, const int* cnt_dev, int stride, int cnt_fixed, bf16* o_h, bf16* o_l,
                            int ldo, cudaStream_t s);

// ---------------------------------------------------------------------------
// element-wise / gather / selection kernels (fe_misc.cu)
// ---------------------------------------------------------------------------
// Raises the dynamic shared-memory limit of the compaction kernel (once per device).
cudaError_t misc_prepare();
// A bounded wait that nothing completes (test hook): sets ST_TIMEOUT in *status after limit_ns.
cudaError_t wait_probe_launch(int* status, uint64_t limit_ns, cudaStream_t s);
// Distinct-element compaction of every request: bitmap over the pool, ranks,
// distinct list, |U(z_b)|, bad-request flags; the last CTA scans U into offsets.
// Candidate-factorized layout (every occurrence its own element): per request b
// U[b] = K*L, off[b] = b*K*L (off[B] = B*K*L), list[b*K*L + i] = cand[b, i],
// slot[b, i] = i; a request with an index outside [0, M) gets bad[b] = 1,
// slot -1, list entries 0 (in range for the gather; its scores become NaN).
// Whole-pool layout: U[b] = M, off[b] = b*M, list[b*M + i] = i, slot[b, i] =
// cand[b, i]; a request with an index outside [0, M) gets bad[b] = 1, slots -1.
cudaError_t pool_layout_launch(const int32_t* cand, int B, int M, int KL, int* U, int* off, int* bad, int* slot,
                               int* list, int* status, cudaStream_t s);
cudaError_t identity_layout_launch(const int32_t* cand, int B, int M, int KL, int* U, int* off, int* bad,
                                   int* slot, int* list, int* status, cudaStream_t s);
cudaError_t compact_launch(const int32_t* cand, int B, int M, int K, int L, int cap, int* U, int* off,
                           int* bad, int* slot_local, int* list, int* status, unsigned* ticket,
                           cudaStream_t s);
// Per-row LN of the context -> split planes [rows, ldo]
// (mean, rstd) of each bf16 row of d columns (LayerNorm without affine parameters, biased variance)
cudaError_t row_stats_launch(const bf16* x, int rows, int d, float eps, float2* out, cudaStream_t s);
// out[n] = sum_k (W_h[n, k] + W_l[n, k]) over k < K of the transposed weight planes (W_l may be null)
cudaError_t colsum_launch(const bf16* w_h, const bf16* w_l, int ld, int N, int K, float* out, cudaStream_t s);
cudaError_t ctx_ln_launch(const void* x, int io_f32, int rows, int d, float eps, bf16* out_h, bf16* out_l,
                          int ldo, cudaStream_t s);
// Gather distinct pool rows of every request -> residual stream h (fp32) and LN(h) planes
cudaError_t gather_ln_launch(const void* pool, int io_f32, int B, int M, int d, int cap, const int* off,
                             const int* list, int max_rows, float eps, float* h, int ldh, bf16* ln_h,
                             bf16* ln_l, int ldln, cudaStream_t s);
// [CLS]-query attention of SeqEnc over [CLS; elements + P]; one warp per sequence
struct ClsParams {
  int B, K, L, d, H;
  const int* off;
  const int* bad;
  const int* slot_local;  // [B, K, L]
  const float* elog;      // [rows, d / 32] element [CLS] logit partials q0 . (H WKs) per 32-column chunk
  const bf16 *kv_h, *kv_l;  // element projections [rows, 2d]: values in columns d .. 2d - 1
  int ldkv;
  const float* qkP;       // [max_L, H] q0 . (P WKs) per head
  const float* qk0;       // [H] q0 . ([CLS] WKs) per head
  const float* v0;        // [CLS] WVs
  const float* vP;        // P WVs  [max_L, d]
  bf16 *o_h, *o_l;
  int ldo;
  float scale;            // 1 / sqrt(d_h)
};
// qk[j * H + h] = q0 . kP[j] over head h's columns for j < max_L, and qk[max_L * H + h] = q0 . k0
cudaError_t cls_consts_launch(const float* q0, const float* k0, const float* kP, int max_L, int d, int H, float* qk,
                              cudaStream_t s);
cudaError_t cls_attn_launch(const ClsParams& p, cudaStream_t s);

// ---------------------------------------------------------------------------
// The sequence stage in one kernel (fe_seq.cu), for d = 128, d_h in {32, 64},
// K <= 128, L <= 31, one score head and bf16-exact weights: index-based
// assembly and the [CLS] attention of SeqEnc (Section 4.3), SeqEnc's output
// projection and FFN, the cross-sequence block (Section 4.4), the score head
// and the argmax of Eq. 1.  A tile holds G whole requests (G K <= 128 rows,
// row = request-local sequence), so the cross-sequence attention and the
// argmax never leave the CTA.
// Weight maps: W^T planes with 64 x 128 boxes and the 128-byte swizzle:
// WOs [d, d], W1s [F, d], W2s [d, F], [WQx | WKx | WVx] [3d, d], WOx [d, d],
// W1h [d, d].
// ---------------------------------------------------------------------------
struct SeqParams {
  int B, K, L, H, dh, F;
  int G;                     // requests per tile
  const int* off;            // [B + 1] element row offsets
  const int* bad;            // [B]
  const int* slot;           // [B, K, L] request-local slots
  const float* elog;         // [rows, d / 32] per-32-column [CLS] logit partials q0 . (H WKs)
  const bf16* v_h;           // element values H WVs, one f16 plane (bits), [rows, d] row-major
  const float *v0, *vP;      // [CLS] WVs, P WVs [max_L, d]
  const float *qkP, *qk0;    // q0 . (P WKs)_j per head [j][4] and q0 . ([CLS] WKs) per head [4], q0 = [CLS] WQs
  const float *cls, *b1s, *b2s, *b1h, *w2h, *b2h;
  int cross;                 // 0: no cross-sequence block (C' = C)
  float eps;
  float scale_log2;          // log2(e) / sqrt(d_h)
  float* scores;             // [B, K]
  float* task_scores;        // [B, K] the single head's score again (the per-task scores of one task), or null
  float* c_out;              // [B K, d] c (SeqEnc output), or null
  float* cp_out;             // [B K, d] C', or null
  SelArgs sel;               // best, status, host status, ticket (keys / nan unused)
};
bool seq_supported(int d, int dh, int F, int nb, int n_tasks, int K, int L);
// the weight-only [CLS] logits of the kernel: out[j * 4 + h] = q0 . kP[j] over head h
// (j < max_L), out[max_L * 4 + h] = q0 . k0 over head h
cudaError_t seq_consts_launch(const float* q0, const float* k0, const float* kP, int max_L, int d, int dh, float* out,
                              cudaStream_t s);
cudaError_t seq_prepare();
cudaError_t seq_launch(const CUtensorMap* wos, const CUtensorMap* w1s, const CUtensorMap* w2s,
                       const CUtensorMap* qkvx, const CUtensorMap* wox, const CUtensorMap* w1h, const SeqParams& p,
                       cudaStream_t s);
// weight preparation: out[(row0 + n) * ldo + k] = split(W[k * N + n]) for k < Kin, n < N
cudaError_t transpose_split_launch(const float* W, int Kin, int N, bf16* out_h, bf16* out_l, int ldo,
                                   int row0, cudaStream_t s);
// out[r, n] = sum_k X[r, k] W[k, n]  (fp32; init-time weight-only products)
cudaError_t small_matmul_launch(const float* X, int R, int Kd, const float* W, int N, float* out,
                                cudaStream_t s);

}  // namespace fe
