// C-ABI of the joint evaluator: weights, workspace, TMA descriptors, the
// launch sequence of one evaluation and its CUDA-graph cache.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <limits>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "fe.h"
#include "fe_kernels.h"

using fe::bf16;

namespace {

thread_local std::string g_msg;

int set_cuda_err(cudaError_t e, const char* what) {
  g_msg = std::string(what) + ": " + cudaGetErrorString(e);
  return FE_ERR_CUDA;
}

// Every device and page-locked allocation of the library goes through
// dev_alloc / host_alloc: they count the live allocations and, for tests
// (fe_debug_alloc_hook), can make a chosen allocation fail as if the device
// were out of memory.
std::atomic<long long> g_live_allocs{0};
std::atomic<int> g_fail_countdown{0};  // > 0: the allocation that takes it to 0 fails

bool injected_failure() {
  int n = g_fail_countdown.load();
  while (n > 0)
    if (g_fail_countdown.compare_exchange_weak(n, n - 1)) return n == 1;
  return false;
}

cudaError_t dev_alloc(void** p, size_t bytes) {
  *p = nullptr;
  if (injected_failure()) return cudaErrorMemoryAllocation;
  const cudaError_t e = cudaMalloc(p, bytes);
  if (e == cudaSuccess) {
    ++g_live_allocs;
  } else {
    *p = nullptr;
    cudaGetLastError();  // an allocation failure must not surface as a later call's CUDA error
  }
  return e;
}

void dev_free(void* p) {
  if (p && cudaFree(p) == cudaSuccess) --g_live_allocs;
}

cudaError_t host_alloc(void** p, size_t bytes) {
  *p = nullptr;
  if (injected_failure()) return cudaErrorMemoryAllocation;
  const cudaError_t e = cudaMallocHost(p, bytes);
  if (e == cudaSuccess) {
    ++g_live_allocs;
  } else {
    *p = nullptr;
    cudaGetLastError();
  }
  return e;
}

void host_free(void* p) {
  if (p && cudaFreeHost(p) == cudaSuccess) --g_live_allocs;
}

#define FE_CK(call)                                                     \
  do {                                                                  \
    cudaError_t e_ = (call);                                            \
    if (e_ != cudaSuccess) return set_cuda_err(e_, #call);              \
  } while (0)

inline int round_up(int x, int m) { return (x + m - 1) / m * m; }

// ---------------------------------------------------------------------------
// TMA descriptor encoding (driver entry point, no link-time libcuda dependency)
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// A bf16 matrix stored as one or two planes (hi, lo), row-major [rows, ld].
// A bf16 hi/lo pair of row-major planes, or (attention operands: context K/V,
// element queries, cross-sequence Q/K/V) a single f16 plane in h.
struct Planes {
  bf16* h = nullptr;  // f16 bits for the single-plane attention operands
  bf16* l = nullptr;
  int ld = 0;
  int rows = 0;
  CUtensorMap th{}, tl{};  // operand loads: 64 x 128 boxes, 128-byte swizzle
  CUtensorMap sh{}, sl{};  // epilogue stores: 32 x 32 boxes, 64-byte swizzle
  CUtensorMap ah{}, al{};  // attention queries: d_h x 128 boxes
  CUtensorMap kh{}, kl{};  // attention keys / values: d_h x (64 for d_h = 32, else 128) boxes
};

// fp32 rows (the residual streams), with the epilogue's store descriptor.
struct F32Rows {
  float* p = nullptr;
  int ld = 0;
  int rows = 0;
  CUtensorMap sx{};  // 32 x 32 boxes, 128-byte swizzle
};

int alloc_planes(Planes& p, int rows, int ld, bool two, std::vector<void*>& owned) {
  p.rows = rows < 128 ? 128 : rows;  // TMA boxes of 128 rows stay inside every allocation
  p.ld = ld;
  const size_t bytes = (size_t)p.rows * ld * sizeof(bf16);
  if (dev_alloc((void**)&p.h, bytes) != cudaSuccess) return FE_ERR_OOM;
  owned.push_back(p.h);
  FE_CK(cudaMemset(p.h, 0, bytes));
  if (two) {
    if (dev_alloc((void**)&p.l, bytes) != cudaSuccess) return FE_ERR_OOM;
    owned.push_back(p.l);
    FE_CK(cudaMemset(p.l, 0, bytes));
  }
  return FE_OK;
}

int encode_map_t(CUtensorMap* m, CUtensorMapDataType dt, size_t esz, const void* base, int cols, int rows,
                 int box_cols, int box_rows, CUtensorMapSwizzle sw) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) {
    g_msg = "cuTensorMapEncodeTiled is unavailable";
    return FE_ERR_CUDA;
  }
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * esz};
  cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1u, 1u};
  CUresult r = fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    g_msg = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
    return FE_ERR_CUDA;
  }
  return FE_OK;
}

// Head-major f16 blocks [blocks][rows][dh]: 3D map with box box_x x box_rows x 1.
int encode_map_hm(CUtensorMap* m, const void* base, int dh, int rows, int blocks, int box_x, int box_rows,
                  CUtensorMapSwizzle sw) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) {
    g_msg = "cuTensorMapEncodeTiled is unavailable";
    return FE_ERR_CUDA;
  }
  cuuint64_t dims[3] = {(cuuint64_t)dh, (cuuint64_t)rows, (cuuint64_t)blocks};
  cuuint64_t strides[2] = {(cuuint64_t)dh * 2, (cuuint64_t)rows * dh * 2};
  cuuint32_t box[3] = {(cuuint32_t)box_x, (cuuint32_t)box_rows, 1u};
  cuuint32_t es[3] = {1u, 1u, 1u};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    g_msg = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
    return FE_ERR_CUDA;
  }
  return FE_OK;
}

// f16 rows grouped in segments of seg_rows, [segments][seg_rows][cols]: 3D map
// with box box_x x box_rows x 1, so that a box reaching past its segment's end
// reads zeros there (the cross-sequence attention's V).
int encode_map_seg(CUtensorMap* m, const void* base, int cols, int seg_rows, int segments, int box_x, int box_rows,
                   CUtensorMapSwizzle sw) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) {
    g_msg = "cuTensorMapEncodeTiled is unavailable";
    return FE_ERR_CUDA;
  }
  cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)seg_rows, (cuuint64_t)segments};
  cuuint64_t strides[2] = {(cuuint64_t)cols * 2, (cuuint64_t)seg_rows * cols * 2};
  cuuint32_t box[3] = {(cuuint32_t)box_x, (cuuint32_t)box_rows, 1u};
  cuuint32_t es[3] = {1u, 1u, 1u};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    g_msg = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
    return FE_ERR_CUDA;
  }
  return FE_OK;
}

// Operand tiles: 64 bf16 (128 B) x box_rows, 128-byte swizzle.
int encode_map(CUtensorMap* m, const bf16* base, int cols, int rows, int box_rows) {
  return encode_map_t(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, cols, rows, 64, box_rows,
                      CU_TENSOR_MAP_SWIZZLE_128B);
}

// Descriptors of an activation (A operand): 128-row boxes on both planes.
int map_act(Planes& p) {
  int rc = encode_map(&p.th, p.h, p.ld, p.rows, 128);
  if (rc == FE_OK) rc = encode_map(&p.tl, p.l, p.ld, p.rows, 128);
  return rc;
}

// Descriptors of a GEMM output written by the epilogue.
int map_out(Planes& p) {
  int rc = encode_map_t(&p.sh, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, p.h, p.ld, p.rows, 32, 32,
                        CU_TENSOR_MAP_SWIZZLE_64B);
  if (rc == FE_OK)
    rc = encode_map_t(&p.sl, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, p.l, p.ld, p.rows, 32, 32,
                      CU_TENSOR_MAP_SWIZZLE_64B);
  return rc;
}

// Descriptors of a single-plane f16 attention operand: the GEMM epilogue's
// store map and the attention kernel's Q and K/V head-slice maps.
int map_attn(Planes& p, int dh) {
  const CUtensorMapSwizzle sw = dh == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B;
  const int kv_rows = fe::attn_chunk_keys(dh);
  int rc = encode_map_t(&p.sh, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, p.h, p.ld, p.rows, 32, 32,
                        CU_TENSOR_MAP_SWIZZLE_64B);
  if (rc == FE_OK) rc = encode_map_t(&p.ah, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, p.h, p.ld, p.rows, dh, 128, sw);
  if (rc == FE_OK) rc = encode_map_t(&p.kh, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, p.h, p.ld, p.rows, dh, kv_rows, sw);
  return rc;
}

// The fused context kernel's K/V, head-major [ld / dh blocks][rows][dh]: its
// store map (32 x 32 boxes) and the attention kernel's key/value map, so that
// every key chunk of one head is one contiguous block.
int map_attn_hm(Planes& p, int dh) {
  const CUtensorMapSwizzle sw = dh == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B;
  const int kv_rows = fe::attn_chunk_keys(dh);
  int rc = encode_map_hm(&p.sh, p.h, dh, p.rows, p.ld / dh, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
  if (rc == FE_OK) rc = encode_map_hm(&p.kh, p.h, dh, p.rows, p.ld / dh, dh, kv_rows, sw);
  return rc;
}

int alloc_f32(F32Rows& f, int rows, int ld, std::vector<void*>& owned) {
  f.rows = rows < 128 ? 128 : rows;
  f.ld = ld;
  const size_t bytes = (size_t)f.rows * ld * sizeof(float);
  if (dev_alloc((void**)&f.p, bytes) != cudaSuccess) return FE_ERR_OOM;
  owned.push_back(f.p);
  FE_CK(cudaMemset(f.p, 0, bytes));
  return encode_map_t(&f.sx, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, f.p, ld, f.rows, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B);
}

// A weight matrix W[K, N] stored transposed as B operand [N, K_pad] plus its GEMM tiling.
struct Weight {
  Planes p;
  int N = 0, K_pad = 0, BN = 0, stages = 0;
  CUtensorMap fh{}, fl{};  // W1 of the fused FFN: 64 x 128 boxes; a fused FFN's tail weight: 64 x N
  CUtensorMap b128{};      // the d = 256 FFN kernel's boxes: 64 x 128 of the (single) plane
  // RESID_LN with clusters, N = cs x 128 or cs x 64: boxes of 64 x 128 / 64 x 64 on both planes
  CUtensorMap c128h{}, c128l{}, c64h{}, c64l{};
  bool cmaps = false;
  // products with many row tiles, N % 256 == 0: 256-column tiles (boxes of 64 x 256 on both planes)
  CUtensorMap c256h{}, c256l{};
  bool wide = false;
};

int largest_bn(int N, int cap) {
  for (int bn = cap; bn >= 32; bn -= 32)
    if (N % bn == 0) return bn;
  return 0;
}

struct Shape {
  int B = 0, C = 0, M = 0, K = 0, L = 0;
  bool fact = false;  // candidate-factorized evaluation (fe_evaluate_factorized)
  bool operator==(const Shape& o) const {
    return B == o.B && C == o.C && M == o.M && K == o.K && L == o.L && fact == o.fact;
  }
};

struct IoPtrs {
  const void* ctx;
  const void* pool;
  const int32_t* idx;
  float* scores;
  int32_t* best;
  int* hstatus;  // page-locked word that receives the batch status
  bool operator==(const IoPtrs& o) const {
    return ctx == o.ctx && pool == o.pool && idx == o.idx && scores == o.scores && best == o.best &&
           hstatus == o.hstatus;
  }
};

// One staging slot of the pipelined host entry (fe_submit_host): device copies
// of a batch's inputs and outputs, its status word and its events.
struct HostSlot {
  void* ctx = nullptr;
  void* pool = nullptr;
  int32_t* idx = nullptr;
  float* scores = nullptr;
  int32_t* best = nullptr;
  int* hstatus = nullptr;      // page-locked
  cudaEvent_t in_ev = nullptr;   // inputs copied in
  cudaEvent_t run_ev = nullptr;  // batch evaluated (its results may be copied out)
  cudaEvent_t done_ev = nullptr; // batch and copy-out complete (the slot is free again)
};

struct GraphEntry {
  Shape s;
  IoPtrs io;
  int launches = 0;
  cudaGraphExec_t exec = nullptr;
  unsigned long long last_use = 0;
};

}  // namespace

struct fe_ctx {
  fe_config cfg{};
  int device = 0;
  int d = 0, H = 0, dh = 0, Ly = 0, F = 0, dpad = 0, Fpad = 0, nb = 1;
  bool fused_ffn = false;  // FFN1 + FFN2 in one kernel (d <= 128)
  // the argmax fused into the score head: [keys: B_cap x 8 B][NaN flags: B_cap x 4 B][ticket]
  unsigned long long* sel_keys = nullptr;
  int* sel_nan = nullptr;
  unsigned* sel_ticket = nullptr;
  size_t sel_bytes = 0;
  bool sel_dirty = false;  // a batch stopped before its score head: clear the words before the next one
  bool fused_embed = false;  // gather + LN + the first layer's Q projection in one kernel
  bool tail_q = false;     // the fused FFN of layer l also projects the next layer's Q
  bool ffn_w = false;      // d = 256: the output projection and FFN in one kernel (fe_ffn256.cu), with the Q tail
  bool tail_kv = false;    // the fused FFN of the last layer also projects [WKs | WVs]
  bool fused_ctxkv = false;  // context LN + K/V projection in one kernel (d <= 128, bf16 inputs)
  bool ctx_fold = false;     // otherwise with bf16 inputs: the GEMM multiplies the raw rows and folds the LN in
  float2* ctx_stats = nullptr;  // [B C] (mean, rstd) of the context rows (ctx_fold)
  float* kv_colsum = nullptr;   // [2 Ly d] column sums of the K/V weight (ctx_fold)
  bool seq_ok = false;       // the sequence stage can run as one kernel (fe_seq.cu) for suitable K, L
  bool keep_inter = false;   // store c and C' even where the sequence-stage kernel keeps them on chip
  int n_sms = 148;
  float* elog = nullptr;     // [rows, d / 32] the elements' [CLS] logit partials (sequence-stage kernel)
  Planes vI16;               // [rows, d] the elements' SeqEnc value rows H WVs, one f16 plane (sequence-stage kernel)
  CUtensorMap ctxkv_w{};     // W^T of the K/V projection, 64 x 128 boxes, for the fused kernel
  std::vector<void*> owned_w;  // weight allocations
  std::vector<void*> owned_ws; // workspace allocations
  float* w32 = nullptr;        // every weight in fp32, fe_weight_count order
  std::vector<size_t> woff;    // offsets into w32, by tensor index
  // transposed bf16 weights
  Weight ctx_kv;
  std::vector<Weight> wq, wo, w1, w2;
  Weight kvs, os, w1s, w2s, qkvx, ox, w1h;
  Weight qkve, oe;                  // element self-attention H^(1): [WQe | WKe | WVe], WOe
  int n_tasks = 1;                  // task heads T
  float* head_vec = nullptr;        // b1 [head cols] | w2 [head cols] | b2 [T] | fuse_w [T] | fuse_b [1]
  float* task_scores = nullptr;     // [S, T], every head's score of the last batch
  float* lin_states = nullptr;      // linear-attention context states [segments][Ly][H][d_h^2 + d_h]
  float *q0 = nullptr, *k0 = nullptr, *v0 = nullptr, *kP = nullptr, *vP = nullptr;
  float* qk = nullptr;  // [max_L + 1][4]: q0 . kP[j] and q0 . k0 per head (the sequence-stage kernel)
  float* qkH = nullptr;  // [max_L + 1][H]: the same per head for any H (the [CLS] attention kernel)
  // workspace
  Shape cap_shape;  // reserved maxima
  int cap_rows = 0; // element rows of the reservation: B * min(M, K*L), or B * K * L once factorized
  bool cap_fact = false;      // the reservation covers candidate-factorized batches
  long long kv_rows = 0;      // context K/V rows of the reservation: B * C, or B * K * C
  int *status = nullptr, *U = nullptr, *off = nullptr, *bad = nullptr, *slot = nullptr, *list = nullptr;
  unsigned* ticket = nullptr;
  Planes X, KV, xln, q, a, mid, kvI, o, cln, mids, z, qkv, ax, lncp, eqkv;  // eqkv: H^(1) Q | K | V
  F32Rows h, c, cp;
  void* in_ctx = nullptr;
  void* in_pool = nullptr;
  int32_t* in_idx = nullptr;
  float* out_scores = nullptr;
  int32_t* out_best = nullptr;
  int* host_status = nullptr;  // page-locked
  cudaEvent_t done_ev = nullptr;
  cudaStream_t cap_stream = nullptr;
  // pipelined host entry: kHostSlots slots, a copy-in stream and a compute stream
  static constexpr int kHostSlots = 3;
  HostSlot slots[kHostSlots];
  cudaStream_t copy_stream = nullptr, sub_stream = nullptr, out_stream = nullptr;  // host entry: copy-in, batches, copy-out
  cudaStream_t ctx_stream = nullptr;  // a batch's context K/V, beside its compaction and element gather
  cudaEvent_t fork_ev = nullptr, kv_ev = nullptr;
  bool fork_ctx = false;  // the GEMM context path, unless FE_NO_FORK=1
  int next_slot = 0;       // slot of the next submission; slots are used in turn
  int n_outstanding = 0;   // submissions not yet waited for (the oldest is next_slot - n_outstanding)
  std::vector<GraphEntry> graphs;
  unsigned long long use_clock = 0;
  bool use_graph = true;
  Shape last_shape;
  bool have_last = false;
  // tracing
  struct Site {
    std::string name;
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pending, spare;
    double total_ms = 0.0;
    int launches = 0;
  };
  bool profiling = false;
  std::vector<Site> sites;
  int launches_batch = 0;  // kernels launched by the batch being enqueued
  int launches_last = 0;
};

namespace {

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

// Counts a kernel launch of the batch and, while tracing, brackets it with events.
struct Prof {
  fe_ctx* c;
  cudaStream_t s;
  std::pair<cudaEvent_t, cudaEvent_t> ev{nullptr, nullptr};
  fe_ctx::Site* site = nullptr;
  Prof(fe_ctx* c_, const char* name, cudaStream_t s_) : c(c_), s(s_) {
    ++c->launches_batch;
    if (!c->profiling) return;
    for (auto& x : c->sites)
      if (x.name == name) site = &x;
    if (!site) {
      c->sites.emplace_back();
      site = &c->sites.back();
      site->name = name;
    }
    if (!site->spare.empty()) {
      ev = site->spare.back();
      site->spare.pop_back();
    } else {
      cudaEventCreate(&ev.first);
      cudaEventCreate(&ev.second);
    }
    cudaEventRecord(ev.first, s);
  }
  ~Prof() {
    if (site) {
      cudaEventRecord(ev.second, s);
      site->pending.push_back(ev);
    }
  }
};

bool config_ok(const fe_config* c) {
  if (!c) return false;
  const int d = c->d;
  if (d != 32 && d != 64 && d != 128 && d != 256 && d != 512) return false;
  if (c->n_heads <= 0 || d % c->n_heads) return false;
  const int dh = d / c->n_heads;
  if (dh != 32 && dh != 64) return false;
  if (c->n_layers < 1 || c->n_layers > 8) return false;
  if (c->ffn_mult < 1 || c->ffn_mult > 8) return false;
  if (c->max_L < 1 || c->max_L > 4096) return false;
  if (c->io_dtype != FE_IO_BF16 && c->io_dtype != FE_IO_F32) return false;
  if (!(c->ln_eps >= 0.f)) return false;
  if (c->n_tasks < 0 || c->n_tasks > 4 || (c->n_tasks > 1 && c->n_tasks * d > 512)) return false;
  if (c->no_cross_seq != 0 && c->no_cross_seq != 1) return false;
  if (c->elem_self_attn != 0 && c->elem_self_attn != 1) return false;
  if (c->encode_pool != 0 && c->encode_pool != 1) return false;
  if (c->linear_context_attn != 0 && c->linear_context_attn != 1) return false;
  return true;
}

// task heads T and the head product's width: T * d columns, padded to a
// column tile the GEMM supports (at most 256, or 512)
int n_tasks_of(const fe_config* c) { return c->n_tasks > 1 ? c->n_tasks : 1; }
int head_cols(const fe_config* c) {
  const int n = n_tasks_of(c) * c->d;
  return n <= 256 ? n : 512;
}

// sizes of the weight tensors in fe_weight_count order
std::vector<size_t> weight_sizes(const fe_config* c) {
  const size_t d = c->d, F = (size_t)c->ffn_mult * c->d;
  std::vector<size_t> s;
  for (int l = 0; l < c->n_layers; ++l) {
    s.push_back(d * d);  // WQ
    s.push_back(d * d);  // WK
    s.push_back(d * d);  // WV
    s.push_back(d * d);  // WO
    s.push_back(d * F);  // W1
    s.push_back(F);      // b1
    s.push_back(F * d);  // W2
    s.push_back(d);      // b2
  }
  s.push_back((size_t)c->max_L * d);  // P
  s.push_back(d);                     // cls
  for (int i = 0; i < 4; ++i) s.push_back(d * d);  // WQs WKs WVs WOs
  s.push_back(d * F);                 // W1s
  s.push_back(F);                     // b1s
  s.push_back(F * d);                 // W2s
  s.push_back(d);                     // b2s
  for (int i = 0; i < 4; ++i) s.push_back(c->no_cross_seq ? 0 : d * d);  // WQx WKx WVx WOx
  const int T = n_tasks_of(c);
  for (int t = 0; t < T; ++t) {
    s.push_back(d * d);               // W1h_t
    s.push_back(d);                   // b1h_t
    s.push_back(d);                   // w2h_t
    s.push_back(1);                   // b2h_t
  }
  if (T > 1) {
    s.push_back((size_t)T);           // fuse_w
    s.push_back(1);                   // fuse_b
  }
  if (c->elem_self_attn)
    for (int i = 0; i < 4; ++i) s.push_back(d * d);  // WQe WKe WVe WOe
  return s;
}

// element self-attention weight i (0 WQe, 1 WKe, 2 WVe, 3 WOe): the last four tensors
const float* ew(const fe_ctx* c, int i);

// tensor indices into weight_sizes()
enum { T_WQ = 0, T_WK, T_WV, T_WO, T_W1, T_B1, T_W2, T_B2, T_PER_LAYER };
int t_tail(const fe_ctx* c, int i) { return T_PER_LAYER * c->Ly + i; }
enum { T_P = 0, T_CLS, T_WQS, T_WKS, T_WVS, T_WOS, T_W1S, T_B1S, T_W2S, T_B2S, T_WQX, T_WKX, T_WVX, T_WOX, T_W1H,
       T_B1H, T_W2H, T_B2H };

const float* wptr(const fe_ctx* c, int tensor) { return c->w32 + c->woff[tensor]; }
const float* lw(const fe_ctx* c, int l, int i) { return wptr(c, T_PER_LAYER * l + i); }
const float* tw(const fe_ctx* c, int i) { return wptr(c, t_tail(c, i)); }
// task t's head tensor j (0 W1h, 1 b1h, 2 w2h, 3 b2h); the fusion weights follow the last head
const float* hw(const fe_ctx* c, int t, int j) { return tw(c, T_W1H + 4 * t + j); }
const float* ew(const fe_ctx* c, int i) { return wptr(c, (int)c->woff.size() - 4 + i); }

// Allocate the transposed weight [N, K_pad] and pick its tiling.
int make_weight(fe_ctx* c, Weight& w, int N, int Kin, int bn_cap) {
  w.N = N;
  w.K_pad = round_up(Kin, 64);
  w.BN = largest_bn(N, bn_cap);
  if (w.BN == 0) {
    g_msg = "no column tile divides N";
    return FE_ERR_UNSUPPORTED;
  }
  w.stages = fe::gemm_max_stages(w.BN, c->nb, w.K_pad);
  int rc = alloc_planes(w.p, N, w.K_pad, c->nb > 1, c->owned_w);
  if (rc != FE_OK) return rc;
  const int box = w.BN > 256 ? 256 : w.BN;
  rc = encode_map(&w.p.th, w.p.h, w.p.ld, w.p.rows, box);
  if (rc == FE_OK) rc = encode_map(&w.p.tl, c->nb > 1 ? w.p.l : w.p.h, w.p.ld, w.p.rows, box);
  if (rc == FE_OK && N >= 256 && N % 128 == 0) {
    const bf16* lo = c->nb > 1 ? w.p.l : w.p.h;
    rc = encode_map(&w.c128h, w.p.h, w.p.ld, w.p.rows, 128);
    if (rc == FE_OK) rc = encode_map(&w.c128l, lo, w.p.ld, w.p.rows, 128);
    if (rc == FE_OK) rc = encode_map(&w.c64h, w.p.h, w.p.ld, w.p.rows, 64);
    if (rc == FE_OK) rc = encode_map(&w.c64l, lo, w.p.ld, w.p.rows, 64);
    w.cmaps = rc == FE_OK;
  }
  if (rc == FE_OK && N % 256 == 0) {
    rc = encode_map(&w.c256h, w.p.h, w.p.ld, w.p.rows, 256);
    if (rc == FE_OK) rc = encode_map(&w.c256l, c->nb > 1 ? w.p.l : w.p.h, w.p.ld, w.p.rows, 256);
    w.wide = rc == FE_OK;
  }
  return rc;
}

// The weight of a fused FFN's tail product: 64 x N boxes (N <= 256).
int map_tail(Weight& w, bool two) {
  int rc = encode_map(&w.fh, w.p.h, w.p.ld, w.p.rows, w.N);
  if (rc == FE_OK) rc = encode_map(&w.fl, two ? w.p.l : w.p.h, w.p.ld, w.p.rows, w.N);
  return rc;
}

int map_fused_w1(Weight& w, bool two) {
  int rc = encode_map(&w.fh, w.p.h, w.p.ld, w.p.rows, 128);
  if (rc == FE_OK) rc = encode_map(&w.fl, two ? w.p.l : w.p.h, w.p.ld, w.p.rows, 128);
  return rc;
}

int fill_weight(Weight& w, const float* W, int Kin, int N, int row0) {
  FE_CK(fe::transpose_split_launch(W, Kin, N, w.p.h, w.p.l, w.p.ld, row0, 0));
  return FE_OK;
}

void free_list(std::vector<void*>& v) {
  for (void* p : v) dev_free(p);
  v.clear();
}

void clear_graphs(fe_ctx* c) {
  for (auto& g : c->graphs)
    if (g.exec) cudaGraphExecDestroy(g.exec);
  c->graphs.clear();
}

int gemm(fe_ctx* c, const char* site, int epi, const Planes& A, const Weight& W, int rows, const int* rows_dev,
         fe::GemmParams p, const Planes* out, const F32Rows* xout, cudaStream_t s) {
  if (rows <= 0) return FE_OK;
  Prof pf(c, site, s);
  p.rows = rows;
  p.rows_dev = rows_dev;
  p.N = W.N;
  p.BN = (epi == fe::EPI_STORE || epi == fe::EPI_LN_FOLD) ? W.BN : W.N;
  p.K_pad = W.K_pad;
  p.nb = c->nb;
  p.stages = 0;  // chosen by gemm_launch
  p.nacc = 0;
  p.cs = 1;
  p.status = c->status;
  p.eps = c->cfg.ln_eps;
  const CUtensorMap *bh = &W.p.th, *bl = &W.p.tl;
  // stored products with fewer 128-column tiles than half the SMs (the sequence
  // side of wide shapes): 64-column tiles, twice the CTAs
  if (epi == fe::EPI_STORE && W.cmaps && p.BN == 128 &&
      2LL * ((rows + 127) / 128) * (W.N / 128) < c->n_sms) {
    p.BN = 64;
    bh = &W.c64h;
    bl = &W.c64l;
  }
  // 256-column tiles when they still fill every SM: each stage then feeds MMAs of
  // N = 256, twice the work per wait of the issuing thread
  if ((epi == fe::EPI_STORE || epi == fe::EPI_LN_FOLD) && W.wide && p.BN < 256 &&
      (long long)((rows + 127) / 128) * (W.N / 256) >= c->n_sms) {
    p.BN = 256;
    bh = &W.c256h;
    bl = &W.c256l;
  }
  // LayerNorm (or score-head) rows wider than 128 columns with fewer row tiles
  // than SMs: a cluster of cs CTAs shares each row tile, 128 (or, with very few
  // tiles, 64) columns per CTA, and exchanges the row statistics (the head's
  // partial dot products) through distributed shared memory, so that more SMs
  // multiply and the epilogue is split cs ways
  if ((epi == fe::EPI_RESID_LN || (epi == fe::EPI_HEAD && p.n_tasks <= 2)) && W.cmaps) {
    const int mtiles = (rows + 127) / 128;
    int cs = W.N / 128, bn = 128;
    if (mtiles * cs * 4 <= c->n_sms && cs * 2 <= 8) {
      cs *= 2;
      bn = 64;
    }
    if (mtiles < c->n_sms && cs <= 8 && fe::gemm_cluster_capacity(cs) > 0) {
      p.cs = cs;
      p.BN = bn;
      bh = bn == 128 ? &W.c128h : &W.c64h;
      bl = bn == 128 ? &W.c128l : &W.c64l;
    }
  }
  FE_CK(fe::gemm_launch(epi, &A.th, &A.tl, bh, bl, out ? &out->sh : nullptr, out ? &out->sl : nullptr,
                        xout ? &xout->sx : nullptr, p, s));
  return FE_OK;
}

// x = x0 + A W_O, then the FFN: x written to x (in place over x0 when x0_row is null), LN(x_out) to
// ln_out when store_ln, and with a tail weight WT the product LN(x_out) WT to tail_out (f16 when tail_f16)
int ffn(fe_ctx* c, const char* site, const Planes& A, const Weight& WO, const Weight& W1, const Weight& W2,
        const float* b1, const float* b2, const float* x0_row, const F32Rows& x, const Planes& ln_out, int rows,
        const int* rows_dev, cudaStream_t s, int store_ln = 1, const Weight* WT = nullptr,
        const Planes* tail_out = nullptr, int tail_f16 = 0, float* tail_logits = nullptr) {
  if (rows <= 0) return FE_OK;
  Prof pf(c, site, s);
  fe::FfnParams p{};
  p.rows = rows;
  p.rows_dev = rows_dev;
  p.d = c->d;
  p.d_pad = c->dpad;
  p.F = c->F;
  p.nb = c->nb;
  p.b1 = b1;
  p.b2 = b2;
  p.x0 = x0_row ? nullptr : x.p;
  p.ldx0 = x.ld;
  p.x0_row = x0_row;
  p.tail_n = WT ? WT->N : 0;
  p.tail_f16 = tail_f16;
  p.store_ln = store_ln;
  p.eps = c->cfg.ln_eps;
  p.status = c->status;
  p.tail_q0 = tail_logits ? c->q0 : nullptr;
  p.tail_logits = tail_logits;
  // with logits the key columns are not stored: the value columns go to column 0 of a
  // [rows, d] buffer, or stay at column d of a [rows, 2d] one
  p.tail_col0 = (tail_logits && tail_out && tail_out->ld < 2 * c->d) ? c->d : 0;
  FE_CK(fe::ffn_launch(&A.th, &A.tl, &WO.p.th, &WO.p.tl, &W1.fh, &W1.fl, &W2.p.th, &W2.p.tl, &ln_out.th, &ln_out.tl,
                       &x.sx, WT ? &WT->fh : nullptr, WT ? &WT->fl : nullptr, tail_out ? &tail_out->sh : nullptr,
                       tail_out ? &tail_out->sl : nullptr, p, s));
  return FE_OK;
}

// The d = 256 output projection + FFN block (fe_ffn256.cu): x0 rows are x
// itself unless x0_row is given; x_out goes to x; LN(x_out) to ln_out when
// store_ln; with WQ the next layer's Q (f16) to q_out.
int ffn256(fe_ctx* c, const char* site, const Planes& A, const Weight& WO, const Weight& W1, const Weight& W2,
           const float* b1, const float* b2, const float* x0_row, const F32Rows& x, const Planes& ln_out, int rows,
           const int* rows_dev, cudaStream_t s, int store_ln, const Weight* WQ = nullptr, Planes* q_out = nullptr) {
  if (rows <= 0) return FE_OK;
  Prof pf(c, site, s);
  fe::Ffn256Params p{};
  p.rows = rows;
  p.rows_dev = rows_dev;
  p.F = c->F;
  p.b1 = b1;
  p.b2 = b2;
  p.x = x.p;
  p.ldx = x.ld;
  p.x0_row = x0_row;
  p.store_ln = store_ln;
  p.tail = WQ ? 1 : 0;
  p.eps = c->cfg.ln_eps;
  p.status = c->status;
  FE_CK(fe::ffn256_launch(&A.th, &A.tl, &WO.b128, &W1.b128, &W2.b128, WQ ? &WQ->b128 : nullptr, &ln_out.th,
                          &ln_out.tl, &x.sx, q_out ? &q_out->th : nullptr, p, s));
  return FE_OK;
}

#define FE_RC(call)              \
  do {                           \
    int rc_ = (call);            \
    if (rc_ != FE_OK) return rc_; \
  } while (0)

// The fused argmax of Eq. 1 for a batch (fe_select.cuh).
fe::SelArgs sel_args(fe_ctx* c, int B, int K, const IoPtrs& io) {
  fe::SelArgs a{};
  a.keys = c->sel_keys;
  a.nan = c->sel_nan;
  a.ticket = c->sel_ticket;
  a.bad = c->bad;
  a.best = io.best;
  a.B = B;
  a.K = K;
  a.status = c->status;
  a.host_status = io.hstatus;
  return a;
}

// Whether a batch of K sequences of length L runs its sequence stage (assembly
// to argmax) as one kernel.
bool seq_fused(const fe_ctx* c, int K, int L) {
  return c->seq_ok && fe::seq_supported(c->d, c->dh, c->F, c->nb, c->n_tasks, K, L);
}

// The whole evaluation of one batch, enqueued on s (captured into a graph by the caller).
int enqueue_batch(fe_ctx* c, const Shape& sh, const IoPtrs& io, cudaStream_t s) {
  const int B = sh.B, C = sh.C, M = sh.M, K = sh.K, L = sh.L;
  const int d = c->d, Ly = c->Ly;
  const int io_f32 = c->cfg.io_dtype == FE_IO_F32;
  const bool fact = sh.fact;  // every occurrence its own element, one context K/V per sequence
  const int cap = fact ? K * L : (c->cfg.encode_pool ? M : ((M < K * L) ? M : K * L));
  const int R = B * cap;
  const int S = B * K;
  const bool use_seq = seq_fused(c, K, L);
  c->launches_batch = 0;
  // The status word and the fused argmax's words are zero here: the score
  // head's last CTA clears them after copying the status to io.hstatus.
  if (K == 0) {
    FE_CK(cudaMemsetAsync(c->status, 0, sizeof(int), s));
    FE_CK(cudaMemsetAsync(io.best, 0xFF, (size_t)B * sizeof(int32_t), s));
    FE_CK(cudaMemcpyAsync(io.hstatus, c->status, sizeof(int), cudaMemcpyDeviceToHost, s));
    return FE_OK;
  }
  const int* sumU = c->off + B;  // device: number of distinct elements of the batch

  // (a0) the distinct-element layout of every request: the identity layout
  // (factorized) and the whole pool here; the compaction after the context
  // kernel, beside which it runs
  if (fact) {
    Prof pf(c, "layout", s);
    FE_CK(fe::identity_layout_launch(io.idx, B, M, K * L, c->U, c->off, c->bad, c->slot, c->list, c->status, s));
  } else if (c->cfg.encode_pool) {
    Prof pf(c, "pool_layout", s);
    FE_CK(fe::pool_layout_launch(io.idx, B, M, K * L, c->U, c->off, c->bad, c->slot, c->list, c->status, s));
  }
  // (a1) context keys/values, once per request, on a side stream (joined before
  // the first element layer), so that they run beside the compaction and the
  // element gather, which do not read them
  cudaStream_t sc = s;
  // (small batches keep one stream: the fork's event edges cost more than it overlaps)
  const bool fork = c->fork_ctx && (long long)B * C >= 8192;
  if (fork) {
    FE_CK(cudaEventRecord(c->fork_ev, s));
    FE_CK(cudaStreamWaitEvent(c->ctx_stream, c->fork_ev, 0));
    sc = c->ctx_stream;
  }
  const bool lin_fused = c->cfg.linear_context_attn && c->fused_ctxkv &&
                         fe::ctxkv_state_supported(d, c->dpad, 2 * Ly * d, c->dh, C);
  if (c->fused_ctxkv) {
    CUtensorMap tx{};
    FE_RC(encode_map(&tx, static_cast<const bf16*>(io.ctx), d, B * C, 128));
    fe::CtxKvParams p{};
    p.rows = B * C * (fact ? K : 1);  // factorized: the context of every sequence
    p.d = d;
    p.N = 2 * Ly * d;
    p.dh = c->dh;
    p.eps = c->cfg.ln_eps;
    p.status = c->status;
    p.C = C;
    p.rep = fact ? K : 1;
    if (lin_fused) p.states = c->lin_states;  // the context goes straight to its linear-attention states
    Prof pf(c, lin_fused ? "ctx_ln_state" : "ctx_ln_kv", sc);
    FE_CK(fe::ctxkv_launch(&tx, &c->ctxkv_w, &c->KV.sh, c->dpad, p, sc));
  } else if (c->ctx_fold) {
    // LN(x) W = rstd (x W) - mu rstd colsum(W): the GEMM multiplies the raw bf16
    // context rows (one exact plane) and applies the row statistics in its epilogue
    {
      Prof pf(c, "ctx_stats", sc);
      FE_CK(fe::row_stats_launch(static_cast<const bf16*>(io.ctx), B * C, d, c->cfg.ln_eps, c->ctx_stats, sc));
    }
    Planes raw;
    raw.h = static_cast<bf16*>(const_cast<void*>(io.ctx));
    raw.ld = d;
    raw.rows = B * C;
    FE_RC(encode_map(&raw.th, raw.h, d, B * C, 128));
    raw.tl = raw.th;
    fe::GemmParams p{};
    p.row_stats = c->ctx_stats;
    p.colsum = c->kv_colsum;
    FE_RC(gemm(c, "gemm_ctx_kv", fe::EPI_LN_FOLD, raw, c->ctx_kv, B * C, nullptr, p, &c->KV, nullptr, sc));
  } else {
    {
      Prof pf(c, "ctx_ln", sc);
      FE_CK(fe::ctx_ln_launch(io.ctx, io_f32, B * C, d, c->cfg.ln_eps, c->X.h, c->X.l, c->X.ld, sc));
    }
    fe::GemmParams p{};
    p.out_f16 = 1;
    FE_RC(gemm(c, "gemm_ctx_kv", fe::EPI_STORE, c->X, c->ctx_kv, B * C, nullptr, p, &c->KV, nullptr, sc));
  }
  if (!fact && !c->cfg.encode_pool) {
    Prof pf(c, "compact", s);
    FE_CK(fe::compact_launch(io.idx, B, M, K, L, cap, c->U, c->off, c->bad, c->slot, c->list, c->status, c->ticket,
                           s));
  }
  // (a1') linear attention: the context of every request (sequence, once
  // factorized) reduced to its per-layer, per-head states (unless the
  // context kernel already did)
  if (c->cfg.linear_context_attn && !lin_fused) {
    Prof pf(c, "lin_state", sc);
    FE_CK(fe::lin_state_launch(c->KV.h, c->fused_ctxkv ? 1 : 0, c->KV.rows, c->KV.ld, fact ? B * K : B, C, d, c->dh,
                               Ly, c->H, c->lin_states, sc));
  }
  if (fork) FE_CK(cudaEventRecord(c->kv_ev, sc));
  // (a2) distinct elements: gather + LN (+ the first layer's Q), then the cross-attention stack
  if (c->fused_embed) {
    fe::EmbedParams ep{};
    ep.pool = static_cast<const bf16*>(io.pool);
    ep.B = B;
    ep.M = M;
    ep.cap = cap;
    ep.off = c->off;
    ep.list = c->list;
    ep.rows = R;
    ep.d = d;
    ep.d_pad = c->dpad;
    ep.eps = c->cfg.ln_eps;
    ep.h = c->h.p;
    ep.ldh = c->h.ld;
    ep.status = c->status;
    Prof pf(c, "embed_q", s);
    FE_CK(fe::embed_q_launch(&c->wq[0].p.th, &c->q.sh, ep, s));
  } else {
    Prof pf(c, "gather_ln", s);
    FE_CK(fe::gather_ln_launch(io.pool, io_f32, B, M, d, cap, c->off, c->list, R, c->cfg.ln_eps, c->h.p, d, c->xln.h,
                             c->xln.l, c->xln.ld, s));
  }
  // (a2') element self-attention H^(1) over each request's element set
  // (Section 4.2): h += MHA(LN(h) WQe, LN(h) WKe, LN(h) WVe) WOe, the keys and
  // values of a request being its own element rows
  if (c->cfg.elem_self_attn && !fact) {
    fe::GemmParams p{};
    p.out_f16 = 1;
    FE_RC(gemm(c, "gemm_elem_qkv", fe::EPI_STORE, c->xln, c->qkve, R, sumU, p, &c->eqkv, nullptr, s));
    fe::AttnParams ap{};
    ap.n_segments = B;
    ap.max_q = cap;
    ap.q_off_dev = c->off;
    ap.q_cnt_dev = c->U;
    ap.kv_self = 1;
    ap.n_heads = c->H;
    ap.q_col = 0;
    ap.k_col = d;
    ap.v_col = 2 * d;
    ap.o_col = 0;
    ap.o_h = c->a.h;
    ap.o_l = c->a.l;
    ap.ldo = c->a.ld;
    ap.scale_log2 = 1.4426950408889634f / sqrtf((float)c->dh);
    ap.status = c->status;
    {
      Prof pf(c, "attn_elem_self", s);
      FE_CK(fe::attn_launch(c->dh, &c->eqkv.ah, &c->eqkv.kh, &c->eqkv.kh, ap, s));
    }
    fe::GemmParams po{};
    po.resid = c->h.p;
    po.ldr = d;
    FE_RC(gemm(c, "gemm_elem_o_ln", fe::EPI_RESID_LN, c->a, c->oe, R, sumU, po, &c->xln, &c->h, s));
  }
  if (fork) FE_CK(cudaStreamWaitEvent(s, c->kv_ev, 0));  // the context K/V (or states) are complete
  for (int l = 0; l < Ly; ++l) {
    // (otherwise the embedding kernel or the previous layer's fused FFN wrote Q)
    if ((l == 0 && !c->fused_embed) || (l > 0 && !c->tail_q && !c->ffn_w)) {
      fe::GemmParams p{};
      p.out_f16 = 1;
      FE_RC(gemm(c, "gemm_item_q", fe::EPI_STORE, c->xln, c->wq[l], R, sumU, p, &c->q, nullptr, s));
    }

    fe::AttnParams ap{};
    if (fact) {  // segment = one sequence: its L occurrences over its own context K/V
      ap.n_segments = B * K;
      ap.max_q = L;
      ap.q_stride = L;
      ap.q_cnt_fixed = L;
    } else {
      ap.n_segments = B;
      ap.max_q = cap;
      ap.q_off_dev = c->off;
      ap.q_cnt_dev = c->U;
    }
    ap.n_heads = c->H;
    ap.kv_stride = C;
    ap.kv_cnt = C;
    ap.q_col = 0;
    ap.k_col = 2 * l * d;
    ap.v_col = (2 * l + 1) * d;
    ap.kv3d = c->fused_ctxkv ? 1 : 0;
    ap.o_col = 0;
    ap.o_h = c->a.h;
    ap.o_l = c->a.l;
    ap.ldo = c->a.ld;
    ap.scale_log2 = 1.4426950408889634f / sqrtf((float)c->dh);
    ap.status = c->status;
    if (c->cfg.linear_context_attn) {
      Prof pf(c, "lin_attn_item_ctx", s);
      FE_CK(fe::lin_attn_launch(c->q.h, c->q.ld, c->lin_states, fact ? B * K : B, Ly, l, c->H, c->dh,
                                fact ? nullptr : c->off, fact ? nullptr : c->U, L, L, c->a.h, c->a.l, c->a.ld, s));
    } else {
      Prof pf(c, "attn_item_ctx", s);
      FE_CK(fe::attn_launch(c->dh, &c->q.ah, &c->KV.kh, &c->KV.kh, ap, s));
    }

    if (c->fused_ffn) {
      // the tail: the next layer's Q (f16), or after the last layer SeqEnc's element K/V (split);
      // LN(x_out) itself is stored when something else reads it (the last layer's: the element encodings)
      const bool last = l == Ly - 1;
      const Weight* WT = !last ? (c->tail_q ? &c->wq[l + 1] : nullptr) : (c->tail_kv ? &c->kvs : nullptr);
      const Planes* TO = !last ? &c->q : (use_seq ? &c->vI16 : &c->kvI);
      FE_RC(ffn(c, "ffn_item", c->a, c->wo[l], c->w1[l], c->w2[l], lw(c, l, T_B1), lw(c, l, T_B2), nullptr, c->h,
                c->xln, R, sumU, s, (last || !c->tail_q) ? 1 : 0, WT, WT ? TO : nullptr,
                (!last || (use_seq && WT)) ? 1 : 0, (last && WT) ? c->elog : nullptr));
    } else if (c->ffn_w) {
      // d = 256: the next layer's Q as the tail; LN(x_out) stored after the last
      // layer (the element encodings, which SeqEnc's projection reads)
      const bool last = l == Ly - 1;
      FE_RC(ffn256(c, "ffn_item", c->a, c->wo[l], c->w1[l], c->w2[l], lw(c, l, T_B1), lw(c, l, T_B2), nullptr, c->h,
                   c->xln, R, sumU, s, last ? 1 : 0, last ? nullptr : &c->wq[l + 1], last ? nullptr : &c->q));
    } else {
      fe::GemmParams po{};
      po.resid = c->h.p;
      po.ldr = d;
      FE_RC(gemm(c, "gemm_item_o_ln", fe::EPI_RESID_LN, c->a, c->wo[l], R, sumU, po, &c->xln, &c->h, s));

      fe::GemmParams p1{};
      p1.bias = lw(c, l, T_B1);
      p1.relu = 1;
      FE_RC(gemm(c, "gemm_item_ffn1", fe::EPI_STORE, c->xln, c->w1[l], R, sumU, p1, &c->mid, nullptr, s));

      fe::GemmParams p2{};
      p2.bias = lw(c, l, T_B2);
      p2.resid = c->h.p;
      p2.ldr = d;
      FE_RC(gemm(c, "gemm_item_ffn2_ln", fe::EPI_RESID_LN, c->mid, c->w2[l], R, sumU, p2, &c->xln, &c->h, s));
    }
  }
  // element projections of SeqEnc: H WKs | H WVs (unless the last fused FFN did them)
  if (!(c->fused_ffn && c->tail_kv)) {
    // the key half leaves as the [CLS] logit partials only
    fe::GemmParams p{};
    p.lq = c->q0;
    p.lq_n = d;
    p.logits = c->elog;
    p.ld_logit = d / 32;
    FE_RC(gemm(c, "gemm_item_seq_kv", fe::EPI_STORE, c->xln, c->kvs, R, sumU, p, &c->kvI, nullptr, s));
  }
  if (use_seq) {
    // (a3 - a6) in one kernel: assembly + [CLS] attention, SeqEnc, the
    // cross-sequence block, the head and the argmax, G whole requests per tile
    const int HN = c->w1h.N;
    fe::SeqParams sp{};
    sp.B = B;
    sp.K = K;
    sp.L = L;
    sp.H = c->H;
    sp.dh = c->dh;
    sp.F = c->F;
    const int per_sm = (B + c->n_sms - 1) / c->n_sms;
    sp.G = std::max(1, std::min(128 / K, per_sm));
    sp.off = c->off;
    sp.bad = c->bad;
    sp.slot = c->slot;
    sp.elog = c->elog;
    sp.v_h = c->vI16.h;
    sp.v0 = c->v0;
    sp.vP = c->vP;
    sp.qkP = c->qk;
    sp.qk0 = c->qk + (size_t)c->cfg.max_L * 4;
    sp.cls = tw(c, T_CLS);
    sp.b1s = tw(c, T_B1S);
    sp.b2s = tw(c, T_B2S);
    sp.b1h = c->head_vec;
    sp.w2h = c->head_vec + HN;
    sp.b2h = c->head_vec + 2 * HN;
    sp.cross = c->cfg.no_cross_seq ? 0 : 1;
    sp.eps = c->cfg.ln_eps;
    sp.scale_log2 = 1.4426950408889634f / sqrtf((float)c->dh);
    sp.scores = io.scores;
    sp.task_scores = c->task_scores;
    sp.c_out = c->keep_inter ? c->c.p : nullptr;
    sp.cp_out = c->keep_inter && !c->cfg.no_cross_seq ? c->cp.p : nullptr;
    sp.sel = sel_args(c, B, K, io);
    Prof pf(c, "seq_stage", s);
    FE_CK(fe::seq_launch(&c->os.p.th, &c->w1s.fh, &c->w2s.p.th, &c->qkvx.p.th, &c->ox.p.th, &c->w1h.p.th, sp, s));
    c->launches_last = c->launches_batch;
    return FE_OK;
  }
  // (a3, a4) index-based assembly + [CLS] attention, then c = cls + o WOs, FFN
  {
    fe::ClsParams cp{};
    cp.B = B;
    cp.K = K;
    cp.L = L;
    cp.d = d;
    cp.H = c->H;
    cp.off = c->off;
    cp.bad = c->bad;
    cp.slot_local = c->slot;
    cp.kv_h = c->kvI.h;
    cp.kv_l = c->kvI.l;
    cp.ldkv = c->kvI.ld;
    cp.elog = c->elog;
    cp.qkP = c->qkH;
    cp.qk0 = c->qkH + (size_t)c->cfg.max_L * c->H;
    cp.v0 = c->v0;
    cp.vP = c->vP;
    cp.o_h = c->o.h;
    cp.o_l = c->o.l;
    cp.ldo = c->o.ld;
    cp.scale = 1.0f / sqrtf((float)c->dh);
    Prof pf(c, "seq_cls_attn", s);
    FE_CK(fe::cls_attn_launch(cp, s));
  }
  if (c->fused_ffn) {
    FE_RC(ffn(c, "ffn_seq", c->o, c->os, c->w1s, c->w2s, tw(c, T_B1S), tw(c, T_B2S), tw(c, T_CLS), c->c, c->z, S,
              nullptr, s));
  } else if (c->ffn_w) {
    FE_RC(ffn256(c, "ffn_seq", c->o, c->os, c->w1s, c->w2s, tw(c, T_B1S), tw(c, T_B2S), tw(c, T_CLS), c->c, c->z, S,
                 nullptr, s, 1));
  } else {
    {
      fe::GemmParams p{};
      p.resid = tw(c, T_CLS);
      p.ldr = 0;
      FE_RC(gemm(c, "gemm_seq_o_ln", fe::EPI_RESID_LN, c->o, c->os, S, nullptr, p, &c->cln, &c->c, s));
    }
    {
      fe::GemmParams p{};
      p.bias = tw(c, T_B1S);
      p.relu = 1;
      FE_RC(gemm(c, "gemm_seq_ffn1", fe::EPI_STORE, c->cln, c->w1s, S, nullptr, p, &c->mids, nullptr, s));
    }
    {
      fe::GemmParams p{};
      p.bias = tw(c, T_B2S);
      p.resid = c->c.p;
      p.ldr = d;
      FE_RC(gemm(c, "gemm_seq_ffn2_ln", fe::EPI_RESID_LN, c->mids, c->w2s, S, nullptr, p, &c->z, &c->c, s));
    }
  }
  // (a5) cross-sequence attention over the K sequence vectors of each request
  // (absent in the variant without cross-sequence interaction: C' = C)
  if (!c->cfg.no_cross_seq) {
    fe::GemmParams p{};
    p.out_f16 = 1;
    FE_RC(gemm(c, "gemm_cross_qkv", fe::EPI_STORE, c->z, c->qkvx, S, nullptr, p, &c->qkv, nullptr, s));
    fe::AttnParams ap{};
    ap.n_segments = B;
    ap.n_heads = c->H;
    ap.max_q = K;
    ap.q_stride = K;
    ap.q_cnt_fixed = K;
    ap.kv_stride = K;
    ap.kv_cnt = K;
    ap.q_col = 0;
    ap.k_col = d;
    ap.v_col = 2 * d;
    ap.o_col = 0;
    ap.o_h = c->ax.h;
    ap.o_l = c->ax.l;
    ap.ldo = c->ax.ld;
    ap.scale_log2 = 1.4426950408889634f / sqrtf((float)c->dh);
    ap.status = c->status;
    // V as [request][K][3d], so that a key chunk reaching past K reads zeros, not the next request's rows
    CUtensorMap vseg;
    FE_RC(encode_map_seg(&vseg, c->qkv.h, c->qkv.ld, K, B, c->dh, fe::attn_chunk_keys(c->dh),
                         c->dh == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B));
    ap.kv_seg = 1;
    {
      Prof pf(c, "attn_cross_seq", s);
      FE_CK(fe::attn_launch(c->dh, &c->qkv.ah, &c->qkv.kh, &vseg, ap, s));
    }
    fe::GemmParams po{};
    po.resid = c->c.p;
    po.ldr = d;
    FE_RC(gemm(c, "gemm_cross_o_ln", fe::EPI_RESID_LN, c->ax, c->ox, S, nullptr, po, &c->lncp, &c->cp, s));
  }
  // (a6) score heads (task heads and their fusion) and selection
  {
    const int HN = c->w1h.N;
    fe::GemmParams p{};
    p.n_tasks = c->n_tasks;
    p.head_d = d;
    p.bias = c->head_vec;
    p.w2 = c->head_vec + HN;
    p.b2 = c->head_vec + 2 * HN;
    p.fuse_w = c->head_vec + 2 * HN + c->n_tasks;
    p.fuse_b = c->head_vec + 2 * HN + 2 * c->n_tasks;
    p.scores = io.scores;
    p.task_scores = c->task_scores;
    // (a6) Eq. 1's argmax over each request's K scores, in the same launch
    p.sel = sel_args(c, B, K, io);
    // LN(C') from the cross-sequence block, or LN(C) = Z without it
    const Planes& hin = c->cfg.no_cross_seq ? c->z : c->lncp;
    FE_RC(gemm(c, "gemm_head", fe::EPI_HEAD, hin, c->w1h, S, nullptr, p, nullptr, nullptr, s));
  }
  c->launches_last = c->launches_batch;
  return FE_OK;
}

int status_to_rc(int st) {
  if (st & fe::ST_TIMEOUT) return FE_ERR_TIMEOUT;
  if (st & fe::ST_INDEX) return FE_ERR_INDEX;
  if (st & fe::ST_NUMERIC) return FE_ERR_NUMERIC;
  return FE_OK;
}

int check_shape(const fe_ctx* c, int B, int C, int M, int K, int L) {
  if (B < 0 || C < 1 || M < 0 || K < 0 || L < 0) {
    g_msg = "negative size or C < 1";
    return FE_ERR_INVALID_ARG;
  }
  if (C > 65536 || M > 262144 || K > 4096 || L > c->cfg.max_L || B > 65535) {
    g_msg = "shape outside the supported limits";
    return FE_ERR_UNSUPPORTED;
  }
  const long long cap = (M < (long long)K * L) ? M : (long long)K * L;
  if ((long long)B * cap > (1ll << 30) || (long long)B * C > (1ll << 30) || (long long)B * K > (1ll << 30)) {
    g_msg = "batch too large";
    return FE_ERR_UNSUPPORTED;
  }
  return FE_OK;
}

int reserve_body(fe_ctx* c, const Shape& s, bool fact);

// Sizes the workspace for shape s (growing monotonically).  Shapes outside
// the limits are refused before anything changes.  Otherwise the old
// workspace is released first; when an allocation of the new one fails,
// whatever was allocated is released too and the reservation is left empty,
// so the context holds no stale buffer and the next call reserves again.
int reserve_impl(fe_ctx* c, Shape s) {
  FE_RC(check_shape(c, s.B, s.C, s.M, s.K, s.L));
  // grow monotonically
  s.B = std::max(s.B, c->cap_shape.B);
  s.C = std::max(s.C, c->cap_shape.C);
  s.M = std::max(s.M, c->cap_shape.M);
  s.K = std::max(s.K, c->cap_shape.K);
  s.L = std::max(s.L, c->cap_shape.L);
  const bool fact = s.fact || c->cap_fact;
  if (fact && ((long long)s.B * s.K * s.L > (1ll << 30) || (long long)s.B * s.K * s.C > (1ll << 30))) {
    g_msg = "batch too large for the factorized evaluation";
    return FE_ERR_UNSUPPORTED;
  }
  const int rc = reserve_body(c, s, fact);
  if (rc != FE_OK) {
    cudaDeviceSynchronize();
    free_list(c->owned_ws);
    c->cap_shape = Shape{};
    c->cap_rows = 0;
    c->cap_fact = false;
    c->kv_rows = 0;
    c->have_last = false;
    c->status = nullptr;  // the next reservation allocates these zeroed
    c->sel_keys = nullptr;
    c->sel_dirty = false;
  }
  return rc;
}

int reserve_body(fe_ctx* c, const Shape& s, const bool fact) {
  FE_CK(cudaDeviceSynchronize());
  clear_graphs(c);
  free_list(c->owned_ws);
  c->have_last = false;
  const int d = c->d, Ly = c->Ly;
  const long long capL = (long long)s.K * s.L;
  // element rows per request: the distinct elements (at most min(M, K*L)),
  // the whole pool (M), and K*L once the factorized evaluation is used
  const long long cap_joint = c->cfg.encode_pool ? s.M : ((s.M < capL) ? s.M : capL);
  const int cap = (int)std::max(cap_joint, fact ? capL : 0ll);
  const int B = s.B > 0 ? s.B : 1;
  const int R = B * (cap > 0 ? cap : 1);
  const int S = B * (s.K > 0 ? s.K : 1);
  const int BC = B * s.C;
  const long long kv_rows = (long long)BC * (fact && s.K > 0 ? s.K : 1);
  auto dalloc = [&](void** p, size_t bytes) -> int {
    if (bytes == 0) bytes = 16;
    if (dev_alloc(p, bytes) != cudaSuccess) {
      g_msg = "cudaMalloc of " + std::to_string(bytes) + " bytes failed";
      return FE_ERR_OOM;
    }
    c->owned_ws.push_back(*p);
    if (cudaMemset(*p, 0, bytes) != cudaSuccess) return set_cuda_err(cudaGetLastError(), "cudaMemset");
    return FE_OK;
  };
  FE_RC(dalloc((void**)&c->status, sizeof(int)));
  FE_RC(dalloc((void**)&c->ticket, sizeof(unsigned)));
  FE_RC(dalloc((void**)&c->U, (size_t)B * sizeof(int)));
  FE_RC(dalloc((void**)&c->off, (size_t)(B + 1) * sizeof(int)));
  FE_RC(dalloc((void**)&c->bad, (size_t)B * sizeof(int)));
  c->sel_bytes = (size_t)B * (sizeof(unsigned long long) + sizeof(int)) + sizeof(unsigned);
  FE_RC(dalloc((void**)&c->sel_keys, c->sel_bytes));
  c->sel_nan = reinterpret_cast<int*>(c->sel_keys + B);
  c->sel_ticket = reinterpret_cast<unsigned*>(c->sel_nan + B);
  FE_RC(dalloc((void**)&c->slot, (size_t)B * (size_t)(capL > 0 ? capL : 1) * sizeof(int)));
  FE_RC(dalloc((void**)&c->list, (size_t)R * sizeof(int)));
  FE_RC(dalloc((void**)&c->elog, (size_t)R * (size_t)(d / 32) * sizeof(float)));
  if (c->seq_ok) {
    FE_RC(alloc_planes(c->vI16, R, d, false, c->owned_ws));
    FE_RC(encode_map_t(&c->vI16.sh, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c->vI16.h, d, c->vI16.rows, 32, 32,
                       CU_TENSOR_MAP_SWIZZLE_64B));
  }
  FE_RC(alloc_f32(c->h, R, d, c->owned_ws));
  FE_RC(alloc_f32(c->c, S, d, c->owned_ws));
  FE_RC(alloc_f32(c->cp, S, d, c->owned_ws));
  const size_t esz = c->cfg.io_dtype == FE_IO_F32 ? 4 : 2;
  FE_RC(dalloc(&c->in_ctx, (size_t)BC * d * esz));
  FE_RC(dalloc(&c->in_pool, (size_t)B * (s.M > 0 ? s.M : 1) * d * esz));
  FE_RC(dalloc((void**)&c->in_idx, (size_t)B * (size_t)(capL > 0 ? capL : 1) * sizeof(int32_t)));
  FE_RC(dalloc((void**)&c->out_scores, (size_t)S * sizeof(float)));
  FE_RC(dalloc((void**)&c->out_best, (size_t)B * sizeof(int32_t)));
  FE_RC(dalloc((void**)&c->task_scores, (size_t)S * c->n_tasks * sizeof(float)));
  if (c->cfg.linear_context_attn) {
    const long long segs = s.C > 0 ? kv_rows / s.C : 1;  // requests, or sequences once factorized
    FE_RC(dalloc((void**)&c->lin_states, (size_t)segs * Ly * c->H * (c->dh * c->dh + c->dh) * sizeof(float)));
  }
  // pipelined host entry: slot 0 uses the staging above, the others their own copies
  c->slots[0].ctx = c->in_ctx;
  c->slots[0].pool = c->in_pool;
  c->slots[0].idx = c->in_idx;
  c->slots[0].scores = c->out_scores;
  c->slots[0].best = c->out_best;
  for (int k = 1; k < fe_ctx::kHostSlots; ++k) {
    FE_RC(dalloc(&c->slots[k].ctx, (size_t)BC * d * esz));
    FE_RC(dalloc(&c->slots[k].pool, (size_t)B * (s.M > 0 ? s.M : 1) * d * esz));
    FE_RC(dalloc((void**)&c->slots[k].idx, (size_t)B * (size_t)(capL > 0 ? capL : 1) * sizeof(int32_t)));
    FE_RC(dalloc((void**)&c->slots[k].scores, (size_t)S * sizeof(float)));
    FE_RC(dalloc((void**)&c->slots[k].best, (size_t)B * sizeof(int32_t)));
  }
  if (!c->fused_ctxkv && !c->ctx_fold) FE_RC(alloc_planes(c->X, BC, c->dpad, true, c->owned_ws));
  if (c->ctx_fold) FE_RC(dalloc((void**)&c->ctx_stats, (size_t)BC * sizeof(float2)));
  FE_RC(alloc_planes(c->KV, (int)kv_rows, 2 * Ly * d, false, c->owned_ws));
  FE_RC(alloc_planes(c->xln, R, c->dpad, true, c->owned_ws));
  FE_RC(alloc_planes(c->q, R, d, false, c->owned_ws));
  FE_RC(alloc_planes(c->a, R, c->dpad, true, c->owned_ws));
  FE_RC(alloc_planes(c->mid, R, c->Fpad, true, c->owned_ws));
  FE_RC(alloc_planes(c->kvI, R, 2 * d, true, c->owned_ws));
  FE_RC(alloc_planes(c->o, S, c->dpad, true, c->owned_ws));
  FE_RC(alloc_planes(c->cln, S, c->dpad, true, c->owned_ws));
  FE_RC(alloc_planes(c->mids, S, c->Fpad, true, c->owned_ws));
  FE_RC(alloc_planes(c->z, S, c->dpad, true, c->owned_ws));
  FE_RC(alloc_planes(c->qkv, S, 3 * d, false, c->owned_ws));
  if (c->cfg.elem_self_attn) FE_RC(alloc_planes(c->eqkv, R, 3 * d, false, c->owned_ws));
  FE_RC(alloc_planes(c->ax, S, c->dpad, true, c->owned_ws));
  FE_RC(alloc_planes(c->lncp, S, c->dpad, true, c->owned_ws));
  if (!c->fused_ctxkv && !c->ctx_fold) FE_RC(map_act(c->X));
  for (Planes* p : {&c->xln, &c->a, &c->mid, &c->o, &c->cln, &c->mids, &c->z, &c->ax, &c->lncp}) FE_RC(map_act(*p));
  for (Planes* p : {&c->xln, &c->mid, &c->kvI, &c->cln, &c->mids, &c->z, &c->lncp}) FE_RC(map_out(*p));
  for (Planes* p : {&c->q, &c->qkv}) FE_RC(map_attn(*p, c->dh));
  if (c->ffn_w) FE_RC(encode_map(&c->q.th, c->q.h, c->q.ld, c->q.rows, 128));  // the d = 256 FFN's Q stores
  if (c->cfg.elem_self_attn) FE_RC(map_attn(c->eqkv, c->dh));
  FE_RC(c->fused_ctxkv ? map_attn_hm(c->KV, c->dh) : map_attn(c->KV, c->dh));
  c->cap_shape = s;
  c->cap_shape.fact = false;
  c->cap_rows = R;
  c->cap_fact = fact;
  c->kv_rows = kv_rows;
  return FE_OK;
}

bool fits(const fe_ctx* c, const Shape& s) {
  const Shape& r = c->cap_shape;
  return r.B > 0 && s.B <= r.B && s.C <= r.C && s.M <= r.M && s.K <= r.K && s.L <= r.L && (!s.fact || c->cap_fact);
}

int launch_batch_impl(fe_ctx* c, const Shape& s, const IoPtrs& io, cudaStream_t stream);

// A batch normally ends with its score head clearing the status word and the
// fused argmax's words; after a launch that stopped early they are cleared here.
int launch_batch(fe_ctx* c, const Shape& s, const IoPtrs& io, cudaStream_t stream) {
  if (c->sel_dirty && c->sel_keys) {
    FE_CK(cudaMemsetAsync(c->status, 0, sizeof(int), stream));
    FE_CK(cudaMemsetAsync(c->sel_keys, 0, c->sel_bytes, stream));
    c->sel_dirty = false;
  }
  const int rc = launch_batch_impl(c, s, io, stream);
  if (rc != FE_OK) c->sel_dirty = true;
  return rc;
}

int launch_batch_impl(fe_ctx* c, const Shape& s, const IoPtrs& io, cudaStream_t stream) {
  if (!fits(c, s)) FE_RC(reserve_impl(c, s));
  c->last_shape = s;
  c->have_last = true;
  if (!c->use_graph || c->profiling) {
    FE_RC(enqueue_batch(c, s, io, stream));
    FE_CK(cudaEventRecord(c->done_ev, stream));
    return FE_OK;
  }
  GraphEntry* hit = nullptr;
  for (auto& g : c->graphs)
    if (g.s == s && g.io == io) hit = &g;
  if (!hit) {
    if (c->graphs.size() >= 16) {
      size_t oldest = 0;
      for (size_t i = 1; i < c->graphs.size(); ++i)
        if (c->graphs[i].last_use < c->graphs[oldest].last_use) oldest = i;
      cudaGraphExecDestroy(c->graphs[oldest].exec);
      c->graphs.erase(c->graphs.begin() + oldest);
    }
    cudaGraph_t graph = nullptr;
    FE_CK(cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal));
    int rc = enqueue_batch(c, s, io, c->cap_stream);
    cudaError_t e = cudaStreamEndCapture(c->cap_stream, &graph);
    if (rc != FE_OK) {
      if (graph) cudaGraphDestroy(graph);
      return rc;
    }
    if (e != cudaSuccess) return set_cuda_err(e, "cudaStreamEndCapture");
    GraphEntry g;
    g.s = s;
    g.io = io;
    g.launches = c->launches_last;
    e = cudaGraphInstantiate(&g.exec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) return set_cuda_err(e, "cudaGraphInstantiate");
    c->graphs.push_back(g);
    hit = &c->graphs.back();
  }
  hit->last_use = ++c->use_clock;
  c->launches_last = hit->launches;
  FE_CK(cudaGraphLaunch(hit->exec, stream));
  FE_CK(cudaEventRecord(c->done_ev, stream));
  return FE_OK;
}

int wait_status(fe_ctx* c) {
  FE_CK(cudaEventSynchronize(c->done_ev));
  FE_CK(cudaGetLastError());
  return status_to_rc(*c->host_status);
}

int check_io(const void* ctx, const void* pool, const int32_t* idx, const float* scores, const int32_t* best, int B,
             int M, int K, int L) {
  if (B == 0) return FE_OK;
  if (!ctx || !best || (K > 0 && !scores) || (K * L > 0 && !idx) || (K * L > 0 && M > 0 && !pool)) {
    g_msg = "null pointer";
    return FE_ERR_INVALID_ARG;
  }
  auto mis = [](const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15u); };
  if (mis(ctx) || mis(pool) || mis(idx) || mis(scores) || mis(best)) {
    g_msg = "buffers must be 16-byte aligned";
    return FE_ERR_INVALID_ARG;
  }
  return FE_OK;
}

// The workspace is shared by every call: while pipelined host submissions are
// in flight, no other evaluation may be enqueued.
int no_outstanding(fe_ctx* c) {
  if (c->n_outstanding > 0) {
    g_msg = "host submissions are outstanding: call fe_wait_host first";
    return FE_ERR_INVALID_ARG;
  }
  return FE_OK;
}

}  // namespace

extern "C" {

size_t fe_weight_count(const fe_config* cfg) {
  if (!config_ok(cfg)) return 0;
  size_t n = 0;
  for (size_t s : weight_sizes(cfg)) n += s;
  return n;
}

int fe_init(const fe_config* cfg, const float* weights, size_t n_floats, fe_ctx** out) {
  if (!out || !cfg || !weights) {
    g_msg = "null argument";
    return FE_ERR_INVALID_ARG;
  }
  *out = nullptr;
  if (!config_ok(cfg)) {
    g_msg = "unsupported configuration (d in {32,64,128,256,512}, d/n_heads in {32,64})";
    return FE_ERR_UNSUPPORTED;
  }
  const size_t need = fe_weight_count(cfg);
  if (n_floats != need) {
    g_msg = "weight count " + std::to_string(n_floats) + " != " + std::to_string(need);
    return FE_ERR_INVALID_ARG;
  }
  fe_ctx* c = new fe_ctx();
  c->cfg = *cfg;
  if (cudaGetDevice(&c->device) != cudaSuccess) {
    delete c;
    g_msg = "no CUDA device";
    return FE_ERR_CUDA;
  }
  c->d = cfg->d;
  c->H = cfg->n_heads;
  c->dh = cfg->d / cfg->n_heads;
  c->Ly = cfg->n_layers;
  c->F = cfg->ffn_mult * cfg->d;
  c->dpad = round_up(c->d, 64);
  c->Fpad = round_up(c->F, 64);
  const char* ng = std::getenv("FE_NO_GRAPH");
  c->use_graph = !(ng && ng[0] == '1');
  // one bf16 plane when every weight is bf16-representable, else hi + lo
  c->nb = 1;
  for (size_t i = 0; i < n_floats; ++i) {
    uint32_t u;
    std::memcpy(&u, weights + i, 4);
    if (u & 0xFFFFu) {
      c->nb = 2;
      break;
    }
  }
  auto fail = [&](int rc) {
    fe_destroy(c);
    return rc;
  };
  int rc = FE_OK;
  if (fe::gemm_prepare() != cudaSuccess || fe::attn_prepare() != cudaSuccess || fe::misc_prepare() != cudaSuccess ||
      fe::ffn_prepare() != cudaSuccess || fe::ctxkv_prepare() != cudaSuccess || fe::linattn_prepare() != cudaSuccess ||
      fe::embed_q_prepare() != cudaSuccess || fe::seq_prepare() != cudaSuccess || fe::ffn256_prepare() != cudaSuccess)
    return fail(set_cuda_err(cudaGetLastError(), "kernel attributes"));
  {
    size_t o = 0;
    for (size_t s : weight_sizes(cfg)) {
      c->woff.push_back(o);
      o += s;
    }
  }
  if (dev_alloc((void**)&c->w32, n_floats * sizeof(float)) != cudaSuccess) return fail(FE_ERR_OOM);
  c->owned_w.push_back(c->w32);
  if (cudaMemcpy(c->w32, weights, n_floats * sizeof(float), cudaMemcpyHostToDevice) != cudaSuccess)
    return fail(set_cuda_err(cudaGetLastError(), "weight copy"));
  const int d = c->d, F = c->F, Ly = c->Ly;
  if ((rc = make_weight(c, c->ctx_kv, 2 * Ly * d, d, 128)) != FE_OK) return fail(rc);
  for (int l = 0; l < Ly; ++l) {
    if ((rc = fill_weight(c->ctx_kv, lw(c, l, T_WK), d, d, 2 * l * d)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->ctx_kv, lw(c, l, T_WV), d, d, (2 * l + 1) * d)) != FE_OK) return fail(rc);
  }
  c->fused_ctxkv = fe::ctxkv_supported(d, c->dpad, 2 * Ly * d, c->nb, c->cfg.io_dtype == FE_IO_F32);
  if (c->fused_ctxkv && (rc = encode_map(&c->ctxkv_w, c->ctx_kv.p.h, c->ctx_kv.p.ld, c->ctx_kv.p.rows, 128)) != FE_OK)
    return fail(rc);
  c->ctx_fold = !c->fused_ctxkv && c->cfg.io_dtype != FE_IO_F32 && d % 64 == 0;
  if (c->ctx_fold) {
    if (dev_alloc((void**)&c->kv_colsum, (size_t)c->ctx_kv.N * sizeof(float)) != cudaSuccess) return fail(FE_ERR_OOM);
    c->owned_w.push_back(c->kv_colsum);
    if (fe::colsum_launch(c->ctx_kv.p.h, c->nb > 1 ? c->ctx_kv.p.l : nullptr, c->ctx_kv.p.ld, c->ctx_kv.N, d,
                          c->kv_colsum, 0) != cudaSuccess)
      return fail(set_cuda_err(cudaGetLastError(), "K/V weight column sums"));
  }
  c->wq.resize(Ly);
  c->wo.resize(Ly);
  c->w1.resize(Ly);
  c->w2.resize(Ly);
  for (int l = 0; l < Ly; ++l) {
    if ((rc = make_weight(c, c->wq[l], d, d, 128)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->wq[l], lw(c, l, T_WQ), d, d, 0)) != FE_OK) return fail(rc);
    if ((rc = make_weight(c, c->wo[l], d, d, 512)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->wo[l], lw(c, l, T_WO), d, d, 0)) != FE_OK) return fail(rc);
    if ((rc = make_weight(c, c->w1[l], F, d, 128)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->w1[l], lw(c, l, T_W1), d, F, 0)) != FE_OK) return fail(rc);
    if ((rc = make_weight(c, c->w2[l], d, F, 512)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->w2[l], lw(c, l, T_W2), F, d, 0)) != FE_OK) return fail(rc);
  }
  c->fused_ffn = fe::ffn_supported(d, c->dpad, F, c->nb);
  if (c->fused_ffn) {
    for (int l = 0; l < Ly; ++l)
      if ((rc = map_fused_w1(c->w1[l], c->nb > 1)) != FE_OK) return fail(rc);
  }
  c->ffn_w = !c->fused_ffn && fe::ffn256_supported(d, F, c->nb);
  if (c->ffn_w) {
    for (int l = 0; l < Ly; ++l)
      for (Weight* w : {&c->wq[l], &c->wo[l], &c->w1[l], &c->w2[l]})
        if ((rc = encode_map(&w->b128, w->p.h, w->p.ld, w->p.rows, 128)) != FE_OK) return fail(rc);
  }
  if ((rc = make_weight(c, c->kvs, 2 * d, d, 128)) != FE_OK) return fail(rc);
  if ((rc = fill_weight(c->kvs, tw(c, T_WKS), d, d, 0)) != FE_OK) return fail(rc);
  if ((rc = fill_weight(c->kvs, tw(c, T_WVS), d, d, d)) != FE_OK) return fail(rc);
  if ((rc = make_weight(c, c->os, d, d, 512)) != FE_OK) return fail(rc);
  if ((rc = fill_weight(c->os, tw(c, T_WOS), d, d, 0)) != FE_OK) return fail(rc);
  if ((rc = make_weight(c, c->w1s, F, d, 128)) != FE_OK) return fail(rc);
  if ((rc = fill_weight(c->w1s, tw(c, T_W1S), d, F, 0)) != FE_OK) return fail(rc);
  if (c->fused_ffn && (rc = map_fused_w1(c->w1s, c->nb > 1)) != FE_OK) return fail(rc);
  c->tail_q = c->fused_ffn && Ly > 1 && fe::ffn_tail_supported(d, c->dpad, F, c->nb, d, 1);
  c->fused_embed = fe::embed_q_supported(d, c->dpad, c->nb, cfg->io_dtype == FE_IO_F32 ? 1 : 0) &&
                   !cfg->elem_self_attn && c->wq[0].N == d && c->wq[0].BN == d;
  c->tail_kv = c->fused_ffn && fe::ffn_tail_supported(d, c->dpad, F, c->nb, 2 * d, 0);
  if (c->tail_q)
    for (int l = 1; l < Ly; ++l)
      if ((rc = map_tail(c->wq[l], c->nb > 1)) != FE_OK) return fail(rc);
  if (c->tail_kv && (rc = map_tail(c->kvs, c->nb > 1)) != FE_OK) return fail(rc);
  c->seq_ok = c->fused_ffn && c->tail_kv && fe::seq_supported(d, c->dh, F, c->nb, n_tasks_of(cfg), 1, 1);
  if (cudaDeviceGetAttribute(&c->n_sms, cudaDevAttrMultiProcessorCount, c->device) != cudaSuccess)
    return fail(set_cuda_err(cudaGetLastError(), "device attribute"));
  if ((rc = make_weight(c, c->w2s, d, F, 512)) != FE_OK) return fail(rc);
  if ((rc = fill_weight(c->w2s, tw(c, T_W2S), F, d, 0)) != FE_OK) return fail(rc);
  if (c->ffn_w)
    for (Weight* w : {&c->os, &c->w1s, &c->w2s})
      if ((rc = encode_map(&w->b128, w->p.h, w->p.ld, w->p.rows, 128)) != FE_OK) return fail(rc);
  if (!cfg->no_cross_seq) {
    if ((rc = make_weight(c, c->qkvx, 3 * d, d, 128)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->qkvx, tw(c, T_WQX), d, d, 0)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->qkvx, tw(c, T_WKX), d, d, d)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->qkvx, tw(c, T_WVX), d, d, 2 * d)) != FE_OK) return fail(rc);
    if ((rc = make_weight(c, c->ox, d, d, 512)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->ox, tw(c, T_WOX), d, d, 0)) != FE_OK) return fail(rc);
  }
  if (cfg->elem_self_attn) {
    if ((rc = make_weight(c, c->qkve, 3 * d, d, 128)) != FE_OK) return fail(rc);
    for (int i = 0; i < 3; ++i)
      if ((rc = fill_weight(c->qkve, ew(c, i), d, d, i * d)) != FE_OK) return fail(rc);
    if ((rc = make_weight(c, c->oe, d, d, 512)) != FE_OK) return fail(rc);
    if ((rc = fill_weight(c->oe, ew(c, 3), d, d, 0)) != FE_OK) return fail(rc);
  }
  // the task heads' first layers as one product of head_cols(cfg) columns
  // (task t in columns [t d, t d + d), padding columns zero), and their
  // vectors gathered into one buffer
  const int T = n_tasks_of(cfg), HN = head_cols(cfg);
  c->n_tasks = T;
  if ((rc = make_weight(c, c->w1h, HN, d, 512)) != FE_OK) return fail(rc);
  for (int t = 0; t < T; ++t)
    if ((rc = fill_weight(c->w1h, hw(c, t, 0), d, d, t * d)) != FE_OK) return fail(rc);
  {
    const size_t nv = 2 * (size_t)HN + 2 * T + 1;
    if (dev_alloc((void**)&c->head_vec, nv * sizeof(float)) != cudaSuccess) return fail(FE_ERR_OOM);
    c->owned_w.push_back(c->head_vec);
    FE_CK(cudaMemset(c->head_vec, 0, nv * sizeof(float)));
    for (int t = 0; t < T; ++t) {
      FE_CK(cudaMemcpy(c->head_vec + t * d, hw(c, t, 1), d * sizeof(float), cudaMemcpyDeviceToDevice));
      FE_CK(cudaMemcpy(c->head_vec + HN + t * d, hw(c, t, 2), d * sizeof(float), cudaMemcpyDeviceToDevice));
      FE_CK(cudaMemcpy(c->head_vec + 2 * HN + t, hw(c, t, 3), sizeof(float), cudaMemcpyDeviceToDevice));
    }
    if (T > 1) {
      FE_CK(cudaMemcpy(c->head_vec + 2 * HN + T, hw(c, T, 0), (T + 1) * sizeof(float), cudaMemcpyDeviceToDevice));
    } else {
      const float one = 1.f;  // a single head: its score is the score
      FE_CK(cudaMemcpy(c->head_vec + 2 * HN + 1, &one, sizeof(float), cudaMemcpyHostToDevice));
    }
  }
  // weight-only products of SeqEnc: [CLS] W and P W
  const int mL = cfg->max_L;
  float* consts = nullptr;
  if (dev_alloc((void**)&consts, ((size_t)(3 + 2 * mL) * d + (size_t)(mL + 1) * (4 + c->H)) * sizeof(float)) !=
      cudaSuccess)
    return fail(FE_ERR_OOM);
  c->owned_w.push_back(consts);
  c->q0 = consts;
  c->k0 = consts + d;
  c->v0 = consts + 2 * d;
  c->kP = consts + 3 * d;
  c->vP = consts + (size_t)(3 + mL) * d;
  c->qk = consts + (size_t)(3 + 2 * mL) * d;
  c->qkH = c->qk + (size_t)(mL + 1) * 4;
  if (fe::small_matmul_launch(tw(c, T_CLS), 1, d, tw(c, T_WQS), d, c->q0, 0) != cudaSuccess ||
      fe::small_matmul_launch(tw(c, T_CLS), 1, d, tw(c, T_WKS), d, c->k0, 0) != cudaSuccess ||
      fe::small_matmul_launch(tw(c, T_CLS), 1, d, tw(c, T_WVS), d, c->v0, 0) != cudaSuccess ||
      fe::small_matmul_launch(tw(c, T_P), mL, d, tw(c, T_WKS), d, c->kP, 0) != cudaSuccess ||
      fe::small_matmul_launch(tw(c, T_P), mL, d, tw(c, T_WVS), d, c->vP, 0) != cudaSuccess ||
      fe::seq_consts_launch(c->q0, c->k0, c->kP, mL, d, c->dh, c->qk, 0) != cudaSuccess ||
      fe::cls_consts_launch(c->q0, c->k0, c->kP, mL, d, c->H, c->qkH, 0) != cudaSuccess)
    return fail(set_cuda_err(cudaGetLastError(), "SeqEnc constants"));
  if (host_alloc((void**)&c->host_status, sizeof(int)) != cudaSuccess) return fail(FE_ERR_OOM);
  *c->host_status = 0;
  if (cudaEventCreateWithFlags(&c->done_ev, cudaEventDisableTiming) != cudaSuccess ||
      cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&c->sub_stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&c->out_stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&c->ctx_stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&c->fork_ev, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&c->kv_ev, cudaEventDisableTiming) != cudaSuccess)
    return fail(set_cuda_err(cudaGetLastError(), "stream/event"));
  {
    // only for the GEMM context path: the fused context kernel holds every SM
    // (its resident weight half), so the gather waits for it either way, and the
    // fork measured slower there (0.1681 -> 0.1721 ms per serving batch)
    const char* nf = std::getenv("FE_NO_FORK");
    c->fork_ctx = !c->fused_ctxkv && !(nf && nf[0] == '1');
  }
  for (HostSlot& hs : c->slots) {
    if (host_alloc((void**)&hs.hstatus, sizeof(int)) != cudaSuccess) return fail(FE_ERR_OOM);
    *hs.hstatus = 0;
    if (cudaEventCreateWithFlags(&hs.in_ev, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&hs.run_ev, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&hs.done_ev, cudaEventDisableTiming) != cudaSuccess)
      return fail(set_cuda_err(cudaGetLastError(), "stream/event"));
  }
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return fail(set_cuda_err(e, "fe_init"));
  *out = c;
  return FE_OK;
}

namespace {

constexpr size_t kBlobHeader = 64;

uint32_t rd_u32(const unsigned char* p) {
  return (uint32_t)p[0] | ((uint32_t)p[1] << 8) | ((uint32_t)p[2] << 16) | ((uint32_t)p[3] << 24);
}

int32_t rd_i32(const unsigned char* p) {
  const uint32_t u = rd_u32(p);
  int32_t v;
  std::memcpy(&v, &u, 4);
  return v;
}

}  // namespace

int fe_blob_parse(const void* blob, size_t bytes, fe_config* cfg_out, size_t* n_floats_out) {
  if (!blob || !cfg_out) {
    g_msg = "null argument";
    return FE_ERR_INVALID_ARG;
  }
  const unsigned char* b = static_cast<const unsigned char*>(blob);
  if (bytes < kBlobHeader) {
    g_msg = "blob shorter than its 64-byte header";
    return FE_ERR_INVALID_ARG;
  }
  if (std::memcmp(b, "FEW1", 4) != 0) {
    g_msg = "not a weight blob (magic is not FEW1)";
    return FE_ERR_INVALID_ARG;
  }
  const uint32_t version = rd_u32(b + 4);
  if (version != 1) {
    g_msg = "weight blob version " + std::to_string(version) + " (this library reads version 1)";
    return FE_ERR_UNSUPPORTED;
  }
  fe_config c{};
  c.d = rd_i32(b + 8);
  c.n_heads = rd_i32(b + 12);
  c.n_layers = rd_i32(b + 16);
  c.ffn_mult = rd_i32(b + 20);
  c.max_L = rd_i32(b + 24);
  c.io_dtype = rd_i32(b + 28);
  const uint32_t eps_bits = rd_u32(b + 32);
  std::memcpy(&c.ln_eps, &eps_bits, 4);
  c.n_tasks = rd_i32(b + 36);
  c.no_cross_seq = rd_i32(b + 40);
  c.elem_self_attn = rd_i32(b + 44);
  c.encode_pool = rd_i32(b + 48);
  c.linear_context_attn = rd_i32(b + 52);
  const uint64_t n = (uint64_t)rd_u32(b + 56) | ((uint64_t)rd_u32(b + 60) << 32);
  if (!config_ok(&c)) {
    g_msg = "the blob's configuration is not supported";
    return FE_ERR_UNSUPPORTED;
  }
  const size_t need = fe_weight_count(&c);
  if (n != need) {
    g_msg = "the blob holds " + std::to_string(n) + " weights, its configuration needs " + std::to_string(need);
    return FE_ERR_INVALID_ARG;
  }
  if (bytes != kBlobHeader + 4 * need) {
    g_msg = "blob size " + std::to_string(bytes) + " != 64 + 4 * " + std::to_string(need);
    return FE_ERR_INVALID_ARG;
  }
  *cfg_out = c;
  if (n_floats_out) *n_floats_out = need;
  return FE_OK;
}

int fe_init_blob(const void* blob, size_t bytes, fe_ctx** out) {
  if (!out) {
    g_msg = "null argument";
    return FE_ERR_INVALID_ARG;
  }
  *out = nullptr;
  fe_config cfg{};
  size_t n = 0;
  FE_RC(fe_blob_parse(blob, bytes, &cfg, &n));
  const unsigned char* w = static_cast<const unsigned char*>(blob) + kBlobHeader;
  if (reinterpret_cast<uintptr_t>(w) % alignof(float) == 0)
    return fe_init(&cfg, reinterpret_cast<const float*>(w), n, out);
  std::vector<float> aligned(n);
  std::memcpy(aligned.data(), w, n * sizeof(float));
  return fe_init(&cfg, aligned.data(), n, out);
}

int fe_debug_alloc_hook(int fail_at, int64_t* live_out) {
  if (fail_at >= 0) g_fail_countdown.store(fail_at);
  if (live_out) *live_out = g_live_allocs.load();
  return FE_OK;
}

int fe_debug_wait_probe(fe_ctx* c, uint32_t limit_us, void* stream) {
  if (!c || limit_us == 0 || limit_us > 1000000u) {
    g_msg = "null context or limit outside 1..1000000 us";
    return FE_ERR_INVALID_ARG;
  }
  DeviceGuard g(c->device);
  FE_RC(no_outstanding(c));
  if (!c->status) FE_RC(reserve_impl(c, Shape{1, 1, 1, 1, 1}));
  cudaStream_t s = (cudaStream_t)stream;
  // the status word's way to the host is the batch's: copied to the
  // page-locked word, then cleared for the next batch
  FE_CK(fe::wait_probe_launch(c->status, (uint64_t)limit_us * 1000ull, s));
  FE_CK(cudaMemcpyAsync(c->host_status, c->status, sizeof(int), cudaMemcpyDeviceToHost, s));
  FE_CK(cudaMemsetAsync(c->status, 0, sizeof(int), s));
  FE_CK(cudaEventRecord(c->done_ev, s));
  return wait_status(c);
}

int fe_reserve(fe_ctx* c, int B, int C, int M, int K, int L) {
  if (!c) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  Shape s{B, C, M, K, L};
  return reserve_impl(c, s);
}

int fe_evaluate_async(fe_ctx* c, int B, int C, int M, int K, int L, const void* context, const void* pool,
                      const int32_t* cand_idx, float* scores_out, int32_t* best_out, void* stream) {
  if (!c) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  FE_RC(no_outstanding(c));
  FE_RC(check_shape(c, B, C, M, K, L));
  FE_RC(check_io(context, pool, cand_idx, scores_out, best_out, B, M, K, L));
  if (B == 0) {
    *c->host_status = 0;
    FE_CK(cudaEventRecord(c->done_ev, (cudaStream_t)stream));
    return FE_OK;
  }
  Shape s{B, C, M, K, L};
  IoPtrs io{context, pool, cand_idx, scores_out, best_out, c->host_status};
  return launch_batch(c, s, io, (cudaStream_t)stream);
}

int fe_last_status(fe_ctx* c) {
  if (!c) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  return wait_status(c);
}

int fe_evaluate(fe_ctx* c, int B, int C, int M, int K, int L, const void* context, const void* pool,
                const int32_t* cand_idx, float* scores_out, int32_t* best_out, void* stream) {
  FE_RC(fe_evaluate_async(c, B, C, M, K, L, context, pool, cand_idx, scores_out, best_out, stream));
  return fe_last_status(c);
}

int fe_evaluate_factorized(fe_ctx* c, int B, int C, int M, int K, int L, const void* context, const void* pool,
                           const int32_t* cand_idx, float* scores_out, int32_t* best_out, void* stream) {
  if (!c) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  FE_RC(no_outstanding(c));
  FE_RC(check_shape(c, B, C, M, K, L));
  FE_RC(check_io(context, pool, cand_idx, scores_out, best_out, B, M, K, L));
  if (!c->fused_ctxkv || C % 128 != 0) {
    g_msg = "the factorized evaluation needs d <= 128, bf16 inputs and weights, and C a multiple of 128";
    return FE_ERR_UNSUPPORTED;
  }
  if (c->cfg.encode_pool || c->cfg.elem_self_attn) {
    g_msg = "the factorized evaluation encodes every occurrence on its own; encode_pool and the element "
            "self-attention over a set do not apply";
    return FE_ERR_UNSUPPORTED;
  }
  // with no pool row every index is out of range: the joint evaluation gives the same outputs
  Shape s{B, C, M, K, L, M > 0 && K * L > 0};
  if (B == 0) {
    *c->host_status = 0;
    FE_CK(cudaEventRecord(c->done_ev, (cudaStream_t)stream));
    return FE_OK;
  }
  IoPtrs io{context, pool, cand_idx, scores_out, best_out, c->host_status};
  return launch_batch(c, s, io, (cudaStream_t)stream);
}

int fe_evaluate_host(fe_ctx* c, int B, int C, int M, int K, int L, const void* context, const void* pool,
                     const int32_t* cand_idx, float* scores_out, int32_t* best_out, void* stream) {
  if (!c) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  FE_RC(no_outstanding(c));
  FE_RC(check_shape(c, B, C, M, K, L));
  if (B == 0) return FE_OK;
  if (!context || !best_out || (K > 0 && !scores_out) || (K * L > 0 && !cand_idx) || (K * L > 0 && M > 0 && !pool)) {
    g_msg = "null pointer";
    return FE_ERR_INVALID_ARG;
  }
  Shape s{B, C, M, K, L};
  if (!fits(c, s)) FE_RC(reserve_impl(c, s));
  cudaStream_t st = (cudaStream_t)stream;
  const size_t esz = c->cfg.io_dtype == FE_IO_F32 ? 4 : 2;
  FE_CK(cudaMemcpyAsync(c->in_ctx, context, (size_t)B * C * c->d * esz, cudaMemcpyHostToDevice, st));
  if (M > 0 && pool)
    FE_CK(cudaMemcpyAsync(c->in_pool, pool, (size_t)B * M * c->d * esz, cudaMemcpyHostToDevice, st));
  if (K * L > 0)
    FE_CK(cudaMemcpyAsync(c->in_idx, cand_idx, (size_t)B * K * L * sizeof(int32_t), cudaMemcpyHostToDevice, st));
  IoPtrs io{c->in_ctx, c->in_pool, c->in_idx, c->out_scores, c->out_best, c->host_status};
  FE_RC(launch_batch(c, s, io, st));
  if (K > 0) FE_CK(cudaMemcpyAsync(scores_out, c->out_scores, (size_t)B * K * sizeof(float), cudaMemcpyDeviceToHost, st));
  FE_CK(cudaMemcpyAsync(best_out, c->out_best, (size_t)B * sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  FE_CK(cudaEventRecord(c->done_ev, st));
  return wait_status(c);
}

int fe_submit_host(fe_ctx* c, int B, int C, int M, int K, int L, const void* context, const void* pool,
                   const int32_t* cand_idx, float* scores_out, int32_t* best_out) {
  if (!c) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  FE_RC(check_shape(c, B, C, M, K, L));
  if (!context || !best_out || (K > 0 && !scores_out) || (K * L > 0 && !cand_idx) || (K * L > 0 && M > 0 && !pool)) {
    g_msg = "null pointer";
    return FE_ERR_INVALID_ARG;
  }
  if (c->n_outstanding >= fe_ctx::kHostSlots) {
    g_msg = "three host submissions are outstanding: call fe_wait_host first";
    return FE_ERR_INVALID_ARG;
  }
  Shape s{B, C, M, K, L};
  if (!fits(c, s)) {
    if (c->n_outstanding > 0) {
      g_msg = "a larger batch needs more workspace: wait for the outstanding submissions first";
      return FE_ERR_INVALID_ARG;
    }
    FE_RC(reserve_impl(c, s));
  }
  const int k = c->next_slot;
  HostSlot& hs = c->slots[k];
  if (B == 0) {
    *hs.hstatus = 0;
    FE_CK(cudaEventRecord(hs.done_ev, c->sub_stream));
  } else {
    // copy-in on its own stream, once this slot's previous batch is complete
    const size_t esz = c->cfg.io_dtype == FE_IO_F32 ? 4 : 2;
    FE_CK(cudaStreamWaitEvent(c->copy_stream, hs.done_ev, 0));
    FE_CK(cudaMemcpyAsync(hs.ctx, context, (size_t)B * C * c->d * esz, cudaMemcpyHostToDevice, c->copy_stream));
    if (M > 0 && pool)
      FE_CK(cudaMemcpyAsync(hs.pool, pool, (size_t)B * M * c->d * esz, cudaMemcpyHostToDevice, c->copy_stream));
    if (K * L > 0)
      FE_CK(cudaMemcpyAsync(hs.idx, cand_idx, (size_t)B * K * L * sizeof(int32_t), cudaMemcpyHostToDevice,
                            c->copy_stream));
    FE_CK(cudaEventRecord(hs.in_ev, c->copy_stream));
    // the batch on the compute stream; its copy-out on a stream of its own, so
    // that the next batch follows this one on the compute stream at once
    FE_CK(cudaStreamWaitEvent(c->sub_stream, hs.in_ev, 0));
    IoPtrs io{hs.ctx, hs.pool, hs.idx, hs.scores, hs.best, hs.hstatus};
    FE_RC(launch_batch(c, s, io, c->sub_stream));
    FE_CK(cudaEventRecord(hs.run_ev, c->sub_stream));
    FE_CK(cudaStreamWaitEvent(c->out_stream, hs.run_ev, 0));
    if (K > 0)
      FE_CK(cudaMemcpyAsync(scores_out, hs.scores, (size_t)B * K * sizeof(float), cudaMemcpyDeviceToHost,
                            c->out_stream));
    FE_CK(cudaMemcpyAsync(best_out, hs.best, (size_t)B * sizeof(int32_t), cudaMemcpyDeviceToHost, c->out_stream));
    FE_CK(cudaEventRecord(hs.done_ev, c->out_stream));
  }
  c->n_outstanding += 1;
  c->next_slot = (c->next_slot + 1) % fe_ctx::kHostSlots;
  return FE_OK;
}

int fe_wait_host(fe_ctx* c) {
  if (!c) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  if (c->n_outstanding == 0) {
    g_msg = "no host submission outstanding";
    return FE_ERR_INVALID_ARG;
  }
  // the oldest outstanding submission: slots are used in turn
  const int k = (c->next_slot + fe_ctx::kHostSlots - c->n_outstanding) % fe_ctx::kHostSlots;
  HostSlot& hs = c->slots[k];
  c->n_outstanding -= 1;
  FE_CK(cudaEventSynchronize(hs.done_ev));
  FE_CK(cudaGetLastError());
  return status_to_rc(*hs.hstatus);
}

int fe_debug_layout(fe_ctx* c, int32_t* slot_out, int32_t* U_out) {
  if (!c || !slot_out || !U_out) return FE_ERR_INVALID_ARG;
  if (!c->have_last) {
    g_msg = "no evaluated batch";
    return FE_ERR_INVALID_ARG;
  }
  DeviceGuard g(c->device);
  FE_CK(cudaEventSynchronize(c->done_ev));
  const Shape& s = c->last_shape;
  FE_CK(cudaMemcpy(U_out, c->U, (size_t)s.B * sizeof(int), cudaMemcpyDeviceToHost));
  FE_CK(cudaMemcpy(slot_out, c->slot, (size_t)s.B * s.K * s.L * sizeof(int), cudaMemcpyDeviceToHost));
  return FE_OK;
}

// IEEE binary16 bits -> float (normal, subnormal, zero, infinity, NaN)
static float f16_to_float(uint16_t h) {
  const uint32_t sign = (uint32_t)(h & 0x8000u) << 16;
  const uint32_t ex = (h >> 10) & 0x1Fu, man = h & 0x3FFu;
  float mag;
  if (ex == 0) {
    mag = std::ldexp((float)man, -24);
  } else if (ex == 31) {
    mag = man ? std::numeric_limits<float>::quiet_NaN() : std::numeric_limits<float>::infinity();
  } else {
    mag = std::ldexp((float)(man | 0x400u), (int)ex - 25);
  }
  uint32_t u;
  std::memcpy(&u, &mag, 4);
  u |= sign;
  std::memcpy(&mag, &u, 4);
  return mag;
}

int fe_debug_fetch(fe_ctx* c, const char* name, float* dst, size_t max_floats, size_t* n_floats) {
  if (!c || !name || !n_floats) return FE_ERR_INVALID_ARG;
  if (!c->have_last) {
    g_msg = "no evaluated batch";
    return FE_ERR_INVALID_ARG;
  }
  DeviceGuard g(c->device);
  FE_CK(cudaEventSynchronize(c->done_ev));
  const Shape& s = c->last_shape;
  const int d = c->d;
  const Planes* pl = nullptr;
  const float* f32 = nullptr;
  size_t rows = 0, cols = 0;
  const std::string n(name);
  if (n == "ctx_ln") {
    if (c->fused_ctxkv || c->ctx_fold) {
      g_msg = "ctx_ln is not materialised: the context K/V product folds the LayerNorm into its epilogue";
      return FE_ERR_UNSUPPORTED;
    }
    pl = &c->X;
    rows = (size_t)s.B * s.C;
    cols = d;
  } else if (n == "ctx_kv") {
    if (c->cfg.linear_context_attn && c->fused_ctxkv &&
        fe::ctxkv_state_supported(d, c->dpad, 2 * c->Ly * d, c->dh, s.C)) {
      g_msg = "ctx_kv is not materialised: the context kernel reduces it to linear-attention states on chip";
      return FE_ERR_UNSUPPORTED;
    }
    pl = &c->KV;
    rows = (size_t)s.B * s.C;
    cols = 2 * c->Ly * d;
  } else if (n == "elem") {
    int sum = 0;
    FE_CK(cudaMemcpy(&sum, c->off + s.B, sizeof(int), cudaMemcpyDeviceToHost));
    pl = &c->xln;
    rows = (size_t)sum;
    cols = d;
  } else if (n == "seq") {
    if (seq_fused(c, s.K, s.L) && !c->keep_inter) {
      g_msg = "seq is kept on chip by the sequence-stage kernel (fe_debug_keep_intermediates stores it)";
      return FE_ERR_UNSUPPORTED;
    }
    f32 = c->c.p;
    rows = (size_t)s.B * s.K;
    cols = d;
  } else if (n == "cross") {
    if (c->cfg.no_cross_seq) {
      g_msg = "no cross-sequence block in this configuration (C' = C: fetch \"seq\")";
      return FE_ERR_UNSUPPORTED;
    }
    if (seq_fused(c, s.K, s.L) && !c->keep_inter) {
      g_msg = "cross is kept on chip by the sequence-stage kernel (fe_debug_keep_intermediates stores it)";
      return FE_ERR_UNSUPPORTED;
    }
    f32 = c->cp.p;
    rows = (size_t)s.B * s.K;
    cols = d;
  } else if (n == "task_scores") {
    f32 = c->task_scores;
    rows = (size_t)s.B * s.K;
    cols = (size_t)c->n_tasks;
  } else {
    g_msg = "unknown buffer name";
    return FE_ERR_INVALID_ARG;
  }
  *n_floats = rows * cols;
  if (!dst) return FE_OK;
  if (max_floats < rows * cols) {
    g_msg = "destination too small";
    return FE_ERR_INVALID_ARG;
  }
  if (f32) {
    FE_CK(cudaMemcpy(dst, f32, rows * cols * sizeof(float), cudaMemcpyDeviceToHost));
    return FE_OK;
  }
  if (pl == &c->KV && c->fused_ctxkv) {  // head-major [cols / dh][pl->rows][dh]
    std::vector<uint16_t> hh((size_t)pl->rows * pl->ld);
    FE_CK(cudaMemcpy(hh.data(), pl->h, hh.size() * 2, cudaMemcpyDeviceToHost));
    const size_t dh = (size_t)c->dh;
    for (size_t r = 0; r < rows; ++r)
      for (size_t j = 0; j < cols; ++j)
        dst[r * cols + j] = f16_to_float(hh[((j / dh) * pl->rows + r) * dh + j % dh]);
    return FE_OK;
  }
  std::vector<uint16_t> hh((size_t)rows * pl->ld), ll((size_t)rows * pl->ld);
  if (rows) FE_CK(cudaMemcpy(hh.data(), pl->h, hh.size() * 2, cudaMemcpyDeviceToHost));
  if (!pl->l) {  // single f16 plane
    for (size_t r = 0; r < rows; ++r)
      for (size_t j = 0; j < cols; ++j) dst[r * cols + j] = f16_to_float(hh[r * pl->ld + j]);
    return FE_OK;
  }
  if (rows) FE_CK(cudaMemcpy(ll.data(), pl->l, ll.size() * 2, cudaMemcpyDeviceToHost));
  for (size_t r = 0; r < rows; ++r)
    for (size_t j = 0; j < cols; ++j) {
      const uint32_t a = (uint32_t)hh[r * pl->ld + j] << 16, b = (uint32_t)ll[r * pl->ld + j] << 16;
      float fa, fb;
      std::memcpy(&fa, &a, 4);
      std::memcpy(&fb, &b, 4);
      dst[r * cols + j] = fa + fb;
    }
  return FE_OK;
}

int fe_debug_keep_intermediates(fe_ctx* c, int on) {
  if (!c || (on != 0 && on != 1)) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  if (c->keep_inter != (on == 1)) {
    FE_CK(cudaDeviceSynchronize());
    clear_graphs(c);
    c->keep_inter = on == 1;
  }
  return FE_OK;
}

int fe_profile(fe_ctx* c, int enable) {
  if (!c) return FE_ERR_INVALID_ARG;
  c->profiling = enable != 0;
  return FE_OK;
}

int fe_profile_read(fe_ctx* c, int max_sites, char* names, int* launches, double* total_ms, int* n_sites) {
  if (!c || !n_sites || max_sites < 0) return FE_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  FE_CK(cudaDeviceSynchronize());
  for (auto& site : c->sites) {
    for (auto& ev : site.pending) {
      float ms = 0.f;
      FE_CK(cudaEventElapsedTime(&ms, ev.first, ev.second));
      site.total_ms += ms;
      site.launches += 1;
      site.spare.push_back(ev);
    }
    site.pending.clear();
  }
  *n_sites = (int)c->sites.size();
  for (int i = 0; i < (int)c->sites.size() && i < max_sites; ++i) {
    auto& site = c->sites[i];
    if (names) {
      std::strncpy(names + 32 * i, site.name.c_str(), 31);
      names[32 * i + 31] = 0;
    }
    if (launches) launches[i] = site.launches;
    if (total_ms) total_ms[i] = site.total_ms;
    site.launches = 0;
    site.total_ms = 0.0;
  }
  return FE_OK;
}

int fe_kernels_per_batch(fe_ctx* c) { return c ? c->launches_last : 0; }

int fe_destroy(fe_ctx* c) {
  if (!c) return FE_OK;
  {
    DeviceGuard g(c->device);
    cudaDeviceSynchronize();
    clear_graphs(c);
    for (auto& site : c->sites) {
      for (auto& ev : site.pending) {
        cudaEventDestroy(ev.first);
        cudaEventDestroy(ev.second);
      }
      for (auto& ev : site.spare) {
        cudaEventDestroy(ev.first);
        cudaEventDestroy(ev.second);
      }
    }
    free_list(c->owned_ws);
    free_list(c->owned_w);
    host_free(c->host_status);
    if (c->done_ev) cudaEventDestroy(c->done_ev);
    if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
    for (HostSlot& hs : c->slots) {
      if (hs.done_ev) cudaEventSynchronize(hs.done_ev);
      if (hs.in_ev) cudaEventDestroy(hs.in_ev);
      if (hs.run_ev) cudaEventDestroy(hs.run_ev);
      if (hs.done_ev) cudaEventDestroy(hs.done_ev);
      host_free(hs.hstatus);
    }
    if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
    if (c->sub_stream) cudaStreamDestroy(c->sub_stream);
    if (c->out_stream) cudaStreamDestroy(c->out_stream);
    if (c->ctx_stream) cudaStreamDestroy(c->ctx_stream);
    if (c->fork_ev) cudaEventDestroy(c->fork_ev);
    if (c->kv_ev) cudaEventDestroy(c->kv_ev);
  }
  delete c;
  return FE_OK;
}

const char* fe_strerror(int code) {
  switch (code) {
    case FE_OK: return "ok";
    case FE_ERR_INVALID_ARG: return "invalid argument";
    case FE_ERR_UNSUPPORTED: return "unsupported shape or configuration";
    case FE_ERR_INDEX: return "candidate index outside [0, M)";
    case FE_ERR_WORKSPACE: return "workspace could not be sized";
    case FE_ERR_OOM: return "device allocation failed";
    case FE_ERR_CUDA: return "CUDA error";
    case FE_ERR_NUMERIC: return "NaN score";
    case FE_ERR_TIMEOUT: return "device-side wait timed out";
    default: return "unknown error";
  }
}

const char* fe_last_error_message(void) { return g_msg.c_str(); }

}  // extern "C"
