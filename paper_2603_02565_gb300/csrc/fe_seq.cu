// The sequence stage of the evaluator in one kernel, for rows of width
// d = 128: index-based assembly with position embeddings and the [CLS]
// attention of SeqEnc (Section 4.3), SeqEnc's output projection, residual on
// [CLS] and FFN, the cross-sequence self-attention block (Section 4.4), the
// shared score head and the argmax of Eq. 1.
//
// A tile is 128 rows holding G whole requests (row = lr K + k: sequence k of
// the tile's request lr), so everything a request needs -- its K sequence
// vectors for the cross-sequence attention and its K scores for the argmax --
// stays in one CTA; nothing of the stage goes to memory but the scores and
// best indices.  Per tile:
//   A  (epilogue warps) for every sequence: the [CLS] logits of its L element
//      rows come precomputed per element (q0 . (H WKs), q0 = cls WQs, from the
//      last element layer's tail), plus q0 . (P WKs) per position; softmax
//      over [CLS; L tokens] per head; o = p_cls v0 + sum_j p_j (H_j WVs +
//      P_j WVs) with the value rows gathered by 8-byte loads; o -> shared
//      memory as the split operand tile
//   B  c = cls + o WOs; c += W2s ReLU(W1s LN(c) + b1s) + b2s  (the FFN in
//      128-column chunks, the hidden activation in TMEM, as fe_ffn.cu)
//   C  Z = LN(c); Q | K | V = Z [WQx | WKx | WVx] (f16 tiles in shared
//      memory); per head S = Q K^T over the tile's 128 rows with the
//      block-diagonal request mask, softmax, P (f16, in TMEM) V
//   D  C' = c + A WOx; LN(C')
//   E  s = ReLU(LN(C') W1h + b1h) . w2h + b2h; per request the smallest k
//      attaining the maximum
// Roles: warp 0 lane 0 streams the weights (16 KB boxes, two per 128 x 128
// chunk, in consumption order through a ring of seven slots, by TMA), warp 1 lane 0 issues tcgen05.mma,
// warps 2-17 run the gathers, softmaxes and epilogues (four warps per TMEM lane
// quadrant, each owning a quarter of a row's columns).  Products take split
// bf16 activations (hi + lo) times exact bf16 weights with fp32 accumulation;
// the attention operands Q, K, V, P are single f16 planes; LayerNorm,
// softmax and residuals are fp32.
#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {

constexpr int BM = 128;
constexpr int D = 128;
constexpr int BK = 64;
constexpr int FC = 128;  // FFN columns per chunk
constexpr int NA1 = 3;   // TMEM buffers for FFN1 chunks
constexpr int LA = 2;    // FFN1 chunks issued ahead of the FFN2 that consumes them
constexpr int kEpiWarps = 16;
constexpr int kThreads = 64 + 32 * kEpiWarps;  // 576
constexpr int kMaxL = 31;
constexpr int kMaxF = 1024;
constexpr uint32_t kAPlane = BM * BK * 2;  // 16 KB: 128 rows x 64 bf16
constexpr uint32_t kBox = kAPlane;         // a weight box: 128 rows x 64 columns (a chunk is two)
constexpr int kRing = 7;                   // weight box slots
constexpr int kStageSlot = 2;              // slots 2..6 also stage the tile's element rows during the gathers
constexpr int NST = 240;                   // element rows staged: f16 values (256 B) + logit partials (16 B),
                                           // then the L rows of P WVs (fp32, 512 B each)
constexpr uint32_t kOffV = 4 * kAPlane;               // 64 KB: the split A tile [kb][plane]
constexpr uint32_t kOffRing = kOffV + 32768;          // the V tiles, one per head
constexpr uint32_t kOffMisc = kOffRing + kRing * kBox;
// misc: b1s [kMaxF], b2s, cls, b1h, w2h [D], q0.kP [32][4], q0.k0 [4], row-statistic
// exchange [2][4][128], scores [128], request flags [128], barriers, TMEM slot
constexpr uint32_t kMiscB1 = 0;
constexpr uint32_t kMiscB2 = kMiscB1 + kMaxF * 4;
constexpr uint32_t kMiscCls = kMiscB2 + D * 4;
constexpr uint32_t kMiscB1h = kMiscCls + D * 4;
constexpr uint32_t kMiscW2h = kMiscB1h + D * 4;
constexpr uint32_t kMiscQkP = kMiscW2h + D * 4;
constexpr uint32_t kMiscQk0 = kMiscQkP + 32 * 4 * 4;
constexpr uint32_t kMiscRed = kMiscQk0 + 64;
constexpr uint32_t kMiscV0 = kMiscRed + 4 * 2 * 128 * 4;   // [CLS] WVs [D], then b2h
constexpr uint32_t kMiscSc = kMiscV0 + D * 4 + 16;
constexpr uint32_t kMiscFlag = kMiscSc + 128 * 4;
constexpr uint32_t kMiscBars = kMiscFlag + 128 * 4;
constexpr uint32_t kMiscBytes = kMiscBars + 64 * 8 + 64;
constexpr size_t kSmem = 1024 + kOffMisc + kMiscBytes;

__device__ __forceinline__ float relu_keep_nan(float x) {
  float r;
  asm("max.NaN.f32 %0, %1, 0f00000000;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ void arrive1(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// One arrival per warp, on a barrier whose count is the number of arriving
// warps: the lanes synchronise first, which orders every lane's earlier
// (fenced) writes before the single arrival.  Lanes that left the tile loop
// on a timed-out wait take no part.
__device__ __forceinline__ void warp_arrive(uint64_t* bar) {
  const unsigned m = __activemask();
  __syncwarp(m);
  if ((int)(threadIdx.x & 31) == __ffs(m) - 1) arrive1(bar);
}

__device__ __forceinline__ uint64_t desc_swz(uint32_t saddr, uint32_t sbo, uint32_t swz) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(sbo >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)swz << 61;
  return d;
}

// The weight chunk the tile consumes i-th: its map and box origin.  Order: WOs,
// then FFN1 chunk s and FFN2 chunk s - LA interleaved as the MMA issuer takes
// them, then WQx, WKx, WVx, WOx (with the cross-sequence block), then W1h.
struct ChunkSrc {
  int kind;  // 0 WOs, 1 W1s, 2 W2s, 3 QKVx, 4 WOx, 5 W1h
  int idx;
};

__device__ __forceinline__ ChunkSrc chunk_of(int i, int nf, int cross) {
  if (i == 0) return {0, 0};
  int r = i - 1;
  for (int s = 0; s < nf + LA; ++s) {
    if (s < nf) {
      if (r == 0) return {1, s};
      --r;
    }
    if (s >= LA) {
      if (r == 0) return {2, s - LA};
      --r;
    }
  }
  if (cross) {
    if (r < 3) return {3, r};
    if (r == 3) return {4, 0};
    r -= 4;
  }
  return {5, 0};
}

// Contiguous bytes global -> shared by the copy engine, completion on an mbarrier
// (16-byte aligned addresses, a multiple of 16 bytes).
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// 32 lanes x 32 columns from registers, no wait (tmem_st_wait completes it)
__device__ __forceinline__ void tmem_st32_nw(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
}

// This thread's 32 columns of row r (32 qt .. 32 qt + 31) as a split bf16
// pair into the A tile (128-byte swizzle, [kb][plane]).
__device__ __forceinline__ void store_split32(uint8_t* sA, int r, int qt, const float* v) {
  uint32_t hi[16], lo[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) split2(v[2 * j], v[2 * j + 1], hi[j], lo[j]);
  uint8_t* rowp = sA + (size_t)((qt >> 1) * 2) * kAPlane + (size_t)r * 128u;
#pragma unroll
  for (int jj = 0; jj < 4; ++jj) {
    const uint32_t o = (uint32_t)((4 * (qt & 1) + jj) ^ (r & 7)) << 4;
    *reinterpret_cast<uint4*>(rowp + o) = make_uint4(hi[4 * jj], hi[4 * jj + 1], hi[4 * jj + 2], hi[4 * jj + 3]);
    *reinterpret_cast<uint4*>(rowp + kAPlane + o) = make_uint4(lo[4 * jj], lo[4 * jj + 1], lo[4 * jj + 2], lo[4 * jj + 3]);
  }
}

// The residual step shared by SeqEnc and the cross-sequence block (one copy
// of the code for its three uses): x = acc [+ add] [+ bias] (this thread's 32
// columns 32 qt .. 32 qt + 31 of row r; written back to the accumulator when
// anything was added, and to out_row when given), then LN(x) as the split A
// tile.  acc_t and add_t are TMEM addresses of the thread's lane quadrant (add:
// whether add_t is added); the row statistics are exchanged with the other three
// warps of the quadrant.
__device__ __noinline__ void epi_resid_ln(uint8_t* sA, float* red, uint32_t acc_t, bool add, uint32_t add_t,
                                          const float* bias, float* out_row, int r, int q, int qt, float eps) {
  const uint32_t c = (uint32_t)(32 * qt);
  float v[32];
  tmem_ld32(acc_t + c, v);
  if (add) {
    float w[32];
    tmem_ld32(add_t + c, w);
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] += w[j];
  }
  if (bias) {
#pragma unroll
    for (int j = 0; j < 32; j += 4) {
      const float4 b = *reinterpret_cast<const float4*>(bias + c + j);
      v[j] += b.x;
      v[j + 1] += b.y;
      v[j + 2] += b.z;
      v[j + 3] += b.w;
    }
  }
  if (add || bias) tmem_st32_nw(acc_t + c, v);
  if (out_row) {
#pragma unroll
    for (int j = 0; j < 32; j += 4)
      *reinterpret_cast<float4*>(out_row + c + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
  }
  // four independent partial sums per statistic (short dependency chains)
  float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int j = 0; j < 32; ++j) s4[j & 3] += v[j];
  red[qt * 128 + r] = (s4[0] + s4[1]) + (s4[2] + s4[3]);
  asm volatile("bar.sync %0, 128;" ::"r"(1 + q) : "memory");
  const float mean = ((red[r] + red[128 + r]) + (red[256 + r] + red[384 + r])) * (1.f / (float)D);
#pragma unroll
  for (int i = 0; i < 4; ++i) s4[i] = 0.f;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float dv = v[j] - mean;
    s4[j & 3] = fmaf(dv, dv, s4[j & 3]);
  }
  red[512 + qt * 128 + r] = (s4[0] + s4[1]) + (s4[2] + s4[3]);
  asm volatile("bar.sync %0, 128;" ::"r"(1 + q) : "memory");
  const float rstd =
      1.0f / sqrtf(((red[512 + r] + red[640 + r]) + (red[768 + r] + red[896 + r])) * (1.f / (float)D) + eps);
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = (v[j] - mean) * rstd;
  store_split32(sA, r, qt, v);
  if (add || bias) tmem_st_wait();
}

// D (+)= (64-column block of the split A tile: hi plane at sa, lo plane at
// sa + 16 KB) . (weight box at w)^T, N = 128: eight products, one copy of the
// issue code for every weight chunk but FFN2's.
__device__ __noinline__ void mma_half(uint32_t dst, uint32_t sa, uint32_t w, uint32_t idesc, bool acc) {
  const uint64_t a0 = umma_desc_sw128(sa);
  const uint64_t w0 = umma_desc_sw128(w);
#pragma unroll
  for (int kk = 0; kk < BK / 16; ++kk) {
    const uint64_t ah = desc_adv(a0, kk * 32);
    const uint64_t wh = desc_adv(w0, kk * 32);
    umma_bf16(dst, ah, wh, idesc, (acc || kk != 0) ? 1u : 0u);
    umma_bf16(dst, desc_adv(ah, kAPlane), wh, idesc, 1u);
  }
}

}  // namespace

// Phase A for one lane of the epilogue warps: rows rr_k = ew + kEpiWarps (4 k + g),
// k < NR = 128 / (4 kEpiWarps) (g = lane / 8), of which the lane owns value columns 16 li .. 16 li + 15
// (li = lane % 8; head hc).  Per row, for head hc: the [CLS] query's logits
// against [CLS] and the L assembled tokens (the element's partial plus the
// position part), their softmax, and o = p_cls v0 + sum_j p_j (v_j + vP_j)
// over the lane's columns, written into the split A tile.  Both lanes that own
// columns of head hc compute its softmax (no exchange between lanes); the NR
// rows go through the token loop together so that their loads overlap.
// kStaged: every element row of the tile is in the staging area, so every
// load is a shared-memory load; otherwise rows past the staged ones are read
// from memory.
template <int DH, bool kStaged>
__device__ __forceinline__ void cls_rows(uint8_t* sA, const int* sErow, const uint8_t* sStage, const float* sVP,
                                         const float* sQkP, const float* sQk0, const float* sV0, const bf16* v_h,
                                         const float* elog, int e0, int nst, int rows_v, int L, float sl2, int ew,
                                         int lane) {
  constexpr int NR = BM / (4 * kEpiWarps);
  const int g = lane >> 3, li = lane & 7;
  const int hc = (16 * li) / DH;
  // lanes 4-7 of a group hold their two 8-column halves in the other order
  // (register i <-> column 16 li + ((i + 8 rot) mod 16)), so that each 16-byte
  // load of a staged row and of a position row touches distinct banks
  const int rot = (li >> 2) & 1;
  int rrow[NR];
  bool live[NR];
#pragma unroll
  for (int k = 0; k < NR; ++k) {
    rrow[k] = ew + kEpiWarps * (4 * k + g);
    live[k] = rrow[k] < rows_v && sErow[rrow[k] * 32] >= 0;  // not padding, not a rejected request
  }
  // the element part of the logit of element row e for head hc (unscaled)
  auto part = [&](int e) -> float {
    const int er = e - e0;
    const float* src = (kStaged || (unsigned)er < (unsigned)nst)
                           ? reinterpret_cast<const float*>(sStage + NST * 256 + er * 16)
                           : elog + (size_t)e * 4;
    return DH == 32 ? src[hc] : src[2 * hc] + src[2 * hc + 1];
  };
  const float s0 = sQk0[hc] * sl2;
  float m[NR];
#pragma unroll
  for (int k = 0; k < NR; ++k) m[k] = s0;
#pragma unroll 1
  for (int j = 0; j < L; ++j) {
    const float qp = sQkP[j * 4 + hc];
#pragma unroll
    for (int k = 0; k < NR; ++k)
      if (live[k]) m[k] = fmaxf(m[k], (part(sErow[rrow[k] * 32 + j]) + qp) * sl2);
  }
  float sum[NR], o[NR][16];
#pragma unroll
  for (int k = 0; k < NR; ++k) {
    sum[k] = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) o[k][i] = 0.f;
  }
#pragma unroll 1
  for (int j = 0; j < L; ++j) {
    const float qp = sQkP[j * 4 + hc];
    const float4* vp = reinterpret_cast<const float4*>(sVP + (size_t)j * D + 16 * li);
    const float4 pp[4] = {vp[(2 * rot) & 3], vp[(1 + 2 * rot) & 3], vp[(2 + 2 * rot) & 3], vp[(3 + 2 * rot) & 3]};
#pragma unroll
    for (int k = 0; k < NR; ++k) {
      if (!live[k]) continue;
      const int e = sErow[rrow[k] * 32 + j];
      const int er = e - e0;
      const uint4* src = (kStaged || (unsigned)er < (unsigned)nst)
                             ? reinterpret_cast<const uint4*>(sStage + (size_t)er * 256 + 32 * li)
                             : reinterpret_cast<const uint4*>(v_h + (size_t)e * D + 16 * li);
      const uint4 a4 = src[rot], b4 = src[rot ^ 1];
      const float w = ex2_approx((part(e) + qp) * sl2 - m[k]);
      sum[k] += w;
      const uint32_t wv[8] = {a4.x, a4.y, a4.z, a4.w, b4.x, b4.y, b4.z, b4.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&wv[2 * i]));
        const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&wv[2 * i + 1]));
        o[k][4 * i] = fmaf(w, a.x + pp[i].x, o[k][4 * i]);
        o[k][4 * i + 1] = fmaf(w, a.y + pp[i].y, o[k][4 * i + 1]);
        o[k][4 * i + 2] = fmaf(w, b.x + pp[i].z, o[k][4 * i + 2]);
        o[k][4 * i + 3] = fmaf(w, b.y + pp[i].w, o[k][4 * i + 3]);
      }
    }
  }
#pragma unroll
  for (int k = 0; k < NR; ++k) {
    const int rr = rrow[k];
    if (live[k]) {
      const float pc = ex2_approx(s0 - m[k]);
      const float inv = 1.f / (sum[k] + pc);
#pragma unroll
      for (int i = 0; i < 16; ++i) o[k][i] = fmaf(pc, sV0[16 * li + ((i + 8 * rot) & 15)], o[k][i]) * inv;
    } else if (rr < rows_v) {
      // a rejected request's scores become NaN; o = v0 keeps its rows finite
#pragma unroll
      for (int i = 0; i < 16; ++i) o[k][i] = sV0[16 * li + ((i + 8 * rot) & 15)];
    }
    // o -> row rr of the split tile: registers 0-7 (columns 16 li + 8 rot ..) are
    // 16-byte piece 2 (li % 4) + rot of plane li / 4, registers 8-15 the other piece
    uint32_t hi[8], lo[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) split2(o[k][2 * i], o[k][2 * i + 1], hi[i], lo[i]);
    uint8_t* rowp = sA + (size_t)((li >> 2) * 2) * kAPlane + (size_t)rr * 128u;
    const uint32_t o0 = (uint32_t)((2 * (li & 3) + rot) ^ (rr & 7)) << 4;
    const uint32_t o1 = (uint32_t)((2 * (li & 3) + (rot ^ 1)) ^ (rr & 7)) << 4;
    *reinterpret_cast<uint4*>(rowp + o0) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
    *reinterpret_cast<uint4*>(rowp + o1) = make_uint4(hi[4], hi[5], hi[6], hi[7]);
    *reinterpret_cast<uint4*>(rowp + kAPlane + o0) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    *reinterpret_cast<uint4*>(rowp + kAPlane + o1) = make_uint4(lo[4], lo[5], lo[6], lo[7]);
  }
}

template <int DH>
__global__ void __launch_bounds__(kThreads, 1)
    seq_kernel(const __grid_constant__ CUtensorMap tWOs, const __grid_constant__ CUtensorMap tW1s,
               const __grid_constant__ CUtensorMap tW2s, const __grid_constant__ CUtensorMap tQKV,
               const __grid_constant__ CUtensorMap tWOx, const __grid_constant__ CUtensorMap tW1h,
               const SeqParams p) {
  constexpr int H = D / DH;
  constexpr uint32_t kVRow = DH * 2;                 // bytes per row of a V tile
  constexpr uint32_t kVTile = BM * kVRow;            // one head's V tile: 128 keys x DH
  constexpr uint32_t kVSbo = 8 * kVRow;
  constexpr uint32_t kVSwz = DH == 32 ? 4u : 2u;     // 64-byte / 128-byte swizzle
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  uint8_t* sA = smem;
  uint8_t* sV = smem + kOffV;
  uint8_t* sR = smem + kOffRing;
  uint8_t* misc = smem + kOffMisc;
  float* sB1 = reinterpret_cast<float*>(misc + kMiscB1);
  float* sB2 = reinterpret_cast<float*>(misc + kMiscB2);
  float* sCls = reinterpret_cast<float*>(misc + kMiscCls);
  float* sB1h = reinterpret_cast<float*>(misc + kMiscB1h);
  float* sW2h = reinterpret_cast<float*>(misc + kMiscW2h);
  float* sQkP = reinterpret_cast<float*>(misc + kMiscQkP);  // [j][4]: q0 . kP[j] per head
  float* sQk0 = reinterpret_cast<float*>(misc + kMiscQk0);  // [4]: q0 . k0 per head
  float* red = reinterpret_cast<float*>(misc + kMiscRed);   // [statistic][quarter][row]
  float* sSc = reinterpret_cast<float*>(misc + kMiscSc);
  float* sV0 = reinterpret_cast<float*>(misc + kMiscV0);
  int* sFlag = reinterpret_cast<int*>(misc + kMiscFlag);    // request of the tile has a non-finite value row
  int* sErow = reinterpret_cast<int*>(sV);                  // during the gathers: [row][32] element rows,
                                                            // then the token weights at sV + 16 KB
  uint64_t* bars = reinterpret_cast<uint64_t*>(misc + kMiscBars);
  uint64_t* w_full = bars;            // [kRing]
  uint64_t* w_empty = bars + 8;       // [kRing]
  uint64_t* a_full = bars + 16;       // o written in sA
  uint64_t* o_done = bars + 17;       // o WOs complete
  uint64_t* ln_full = bars + 18;      // x in the accumulator, LN(x) in sA
  uint64_t* acc1_full = bars + 19;    // [NA1]
  uint64_t* acc1_empty = bars + 22;   // [NA1]
  uint64_t* mid_full = bars + 25;     // [NA1]
  uint64_t* acc2_full = bars + 28;    // the FFN complete
  uint64_t* z_full = bars + 29;       // c in the accumulator, LN(c) in sA
  uint64_t* qkv_full = bars + 30;     // the Q | K | V product complete
  uint64_t* qkv_ready = bars + 31;    // Q, K in sA and V in sV
  uint64_t* s_full = bars + 32;       // [2]
  uint64_t* p_full = bars + 34;       // [2]
  uint64_t* s_free = bars + 36;       // [2] PV has read the S/P buffer
  uint64_t* o_full = bars + 38;       // every head's PV complete
  uint64_t* a2_full = bars + 39;      // attention output in sA
  uint64_t* ox_full = bars + 40;      // A WOx complete
  uint64_t* lnc_full = bars + 41;     // LN(C') in sA
  uint64_t* head_full = bars + 42;    // the head product complete
  uint64_t* st_full = bars + 43;      // the tile's element rows staged
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 48);
  volatile uint32_t* last_flag = reinterpret_cast<volatile uint32_t*>(bars + 49);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int K = p.K, L = p.L, G = p.G, F = p.F;
  const int nf = F / FC;
  const int tiles = (p.B + G - 1) / G;
  const int nch = 1 + 2 * nf + (p.cross ? 4 : 0) + 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kRing; ++i) {
      mbar_init(w_full + i, 1);
      mbar_init(w_empty + i, 1);
    }
    for (int i = 0; i < NA1; ++i) {
      mbar_init(acc1_full + i, 1);
      mbar_init(acc1_empty + i, 1);
      mbar_init(mid_full + i, kEpiWarps);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full + i, 1);
      mbar_init(p_full + i, kEpiWarps);
      mbar_init(s_free + i, 1);
    }
    mbar_init(a_full, kEpiWarps);
    mbar_init(o_done, 1);
    mbar_init(ln_full, kEpiWarps);
    mbar_init(acc2_full, 1);
    mbar_init(z_full, kEpiWarps);
    mbar_init(qkv_full, 1);
    mbar_init(qkv_ready, kEpiWarps);
    mbar_init(o_full, 1);
    mbar_init(a2_full, kEpiWarps);
    mbar_init(ox_full, 1);
    mbar_init(lnc_full, kEpiWarps);
    mbar_init(head_full, 1);
    mbar_init(st_full, 1);
    fence_mbar_init();
    prefetch_tmap(&tWOs);
    prefetch_tmap(&tW1s);
    prefetch_tmap(&tW2s);
    prefetch_tmap(&tQKV);
    prefetch_tmap(&tWOx);
    prefetch_tmap(&tW1h);
  }
  // parameters (not outputs of an earlier kernel): read before the dependency wait
  for (int i = threadIdx.x; i < F; i += kThreads) sB1[i] = p.b1s[i];
  for (int i = threadIdx.x; i < D; i += kThreads) {
    sB2[i] = p.b2s[i];
    sCls[i] = p.cls[i];
    sB1h[i] = p.b1h[i];
    sW2h[i] = p.w2h[i];
    sV0[i] = p.v0[i];
  }
  if (threadIdx.x == 0) sV0[D] = p.b2h[0];
  // the [CLS] query's logits against each position embedding's key part and
  // against [CLS] itself, per head (unscaled; weight-only constants)
  for (int i = threadIdx.x; i < L * 4; i += kThreads) sQkP[i] = p.qkP[i];
  if (threadIdx.x < 4) sQk0[threadIdx.x] = p.qk0[threadIdx.x];
  // TMEM: FFN1 chunk buffers [128 i, 128 i + 128), i < 3 (later Q | K | V, then the
  // S/P buffers [0, 256) with the attention output at [256, 384), then A WOx at
  // [0, 128) and the head product at [128, 256)); the d-column accumulator of
  // x, c and C' at [384, 512)
  if (warp == 0) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t acc2 = tmem + (uint32_t)(NA1 * FC);
  pdl_trigger();
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer: the weight chunks of every tile ----------------
      int ws = 0, tl = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        bool gathered = false;  // the tile's gathers are done: the staging slots are weight slots again
        for (int ib = 0; ib < 2 * nch; ++ib, ++ws) {
          const int i = ib >> 1, box = ib & 1;
          const int slot = ws % kRing;
          if (slot >= kStageSlot && !gathered) {
            if (!mbar_wait_compact(a_full, tl & 1, p.sel.status)) {
              ok = false;
              break;
            }
            gathered = true;
          }
          if (ws >= kRing && !mbar_wait_compact(w_empty + slot, ((ws / kRing) - 1) & 1, p.sel.status)) {
            ok = false;
            break;
          }
          const ChunkSrc cs = chunk_of(i, nf, p.cross);
          const CUtensorMap* m = &tWOs;
          int x0 = 0, x1 = BK, y = 0;
          if (cs.kind == 1) {
            m = &tW1s;
            y = cs.idx * FC;
          } else if (cs.kind == 2) {
            m = &tW2s;
            x0 = cs.idx * FC;
            x1 = x0 + BK;
          } else if (cs.kind == 3) {
            m = &tQKV;
            y = cs.idx * D;
          } else if (cs.kind == 4) {
            m = &tWOx;
          } else if (cs.kind == 5) {
            m = &tW1h;
          }
          mbar_arrive_expect_tx(w_full + slot, kBox);
          tma_load_2d(sR + (size_t)slot * kBox, m, box ? x1 : x0, y, w_full + slot);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc = umma_idesc_bf16(BM, FC);
      const uint32_t idesc_s = umma_idesc_f16(BM, BM);
      const uint32_t idesc_pv = umma_idesc_f16(BM, DH) | (1u << 16);  // V is MN-major
      int ws = 0, gf = 0, tl = 0;
      bool ok = true;
      auto wait = [&](uint64_t* bar, uint32_t par) -> bool {
        if (!mbar_wait_compact(bar, par, p.sel.status)) ok = false;
        return ok;
      };
      // the next weight box landed: its shared-memory address (0 on a timeout)
      auto next_box = [&]() -> uint32_t {
        const int slot = ws % kRing;
        if (!wait(w_full + slot, (ws / kRing) & 1)) return 0u;
        tc_fence_after();
        return smem_u32(sR + (size_t)slot * kBox);
      };
      // the box's slot is free once the products issued so far complete
      auto release_box = [&]() {
        umma_commit(w_empty + ws % kRing);
        ++ws;
      };
      // dst = (split A tile in sA) . (the next weight chunk)^T, N = 128, K = 128,
      // box by box: each box's slot is released after its eight products
      auto mma_sa = [&](uint32_t dst) -> bool {
        for (int kb = 0; kb < 2; ++kb) {
          const uint32_t w = next_box();
          if (!w) return false;
          mma_half(dst, smem_u32(sA) + (uint32_t)(kb * 2) * kAPlane, w, idesc, kb != 0);
          release_box();
        }
        return true;
      };
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        // ---- B: o WOs into the FFN1 buffer that chunk 0 of this tile uses next
        if (!wait(a_full, tl & 1)) break;
        {
          const int bo = gf % NA1;
          if (gf >= NA1 && !wait(acc1_empty + bo, ((gf / NA1) - 1) & 1)) break;
          tc_fence_after();
          if (!mma_sa(tmem + (uint32_t)(bo * FC))) break;
          umma_commit(o_done);
        }
        // ---- B: FFN1 / FFN2 once x is in the accumulator and LN(x) in sA
        if (!wait(ln_full, tl & 1)) break;
        tc_fence_after();
        const int gf0 = gf;
        for (int s = 0; s < nf + LA && ok; ++s) {
          if (s < nf) {
            const int g = gf0 + s, b = g % NA1;
            if (s > 0 && g >= NA1 && !wait(acc1_empty + b, ((g / NA1) - 1) & 1)) break;
            if (!mma_sa(tmem + (uint32_t)(b * FC))) break;
            umma_commit(acc1_full + b);
          }
          if (s >= LA) {
            const int c = s - LA, g = gf0 + c, b = g % NA1;
            if (!wait(mid_full + b, (g / NA1) & 1)) break;
            // each 32-column piece of the buffer: 32 hidden units as the hi plane
            // (16 columns of bf16 pairs) then the lo plane; the W2s chunk's two boxes
            // are 64-column halves of the chunk's hidden units, 128 output rows each
            const uint32_t mt = tmem + (uint32_t)(b * FC);
            bool got = true;
            for (int hh = 0; hh < 2; ++hh) {
              const uint32_t w = next_box();
              if (!w) {
                got = false;
                break;
              }
              const uint64_t w0 = umma_desc_sw128(w);
#pragma unroll
              for (int k4 = 0; k4 < 4; ++k4) {
                const int kk = 4 * hh + k4;
                const uint32_t mh = mt + (uint32_t)(32 * (kk >> 1) + 8 * (kk & 1)), ml = mh + 16;
                const uint64_t wh = desc_adv(w0, (uint32_t)k4 * 32);
                umma_bf16_tmem_a(acc2, mh, wh, idesc, 1u);
                umma_bf16_tmem_a(acc2, ml, wh, idesc, 1u);
              }
              release_box();
            }
            if (!got) break;
            umma_commit(acc1_empty + b);
            if (c == nf - 1) umma_commit(acc2_full);
          }
        }
        if (!ok) break;
        gf = gf0 + nf;
        if (!wait(z_full, tl & 1)) break;
        tc_fence_after();
        if (p.cross) {
          // ---- C: Q | K | V = Z [WQx | WKx | WVx] into TMEM [0, 384)
          for (int i = 0; i < 3 && ok; ++i)
            if (!mma_sa(tmem + (uint32_t)(i * 128))) break;
          if (!ok) break;
          umma_commit(qkv_full);
          if (!wait(qkv_ready, tl & 1)) break;
          tc_fence_after();
          // S_h = Q_h K_h^T over the tile's 128 rows into S/P buffer (tl H + h) % 2
          auto issue_s = [&](int h) -> bool {
            const int g = tl * H + h, buf = g & 1;
            if (g >= 2 && !wait(s_free + buf, ((g - 2) >> 1) & 1)) return false;
            tc_fence_after();
            const int c0 = h * DH;
            const uint64_t qd = umma_desc_sw128(smem_u32(sA + (uint32_t)(c0 / BK) * kAPlane));
            const uint64_t kd = umma_desc_sw128(smem_u32(sA + (uint32_t)(2 + c0 / BK) * kAPlane));
#pragma unroll
            for (int kk = 0; kk < DH / 16; ++kk) {
              const uint32_t o = (uint32_t)(c0 % BK) * 2u + (uint32_t)kk * 32u;
              umma_bf16(tmem + (uint32_t)(buf * 128), desc_adv(qd, o), desc_adv(kd, o), idesc_s, kk != 0 ? 1u : 0u);
            }
            umma_commit(s_full + buf);
            return true;
          };
          if (!issue_s(0)) break;
          if (H > 1 && !issue_s(1)) break;
          for (int h = 0; h < H && ok; ++h) {
            const int g = tl * H + h, buf = g & 1;
            if (!wait(p_full + buf, (g >> 1) & 1)) break;
            tc_fence_after();
            // PV_h: A = P_h from the S/P buffer (each half-row warp's 64 keys as 32
            // columns of f16 pairs at the start of its 64 S columns), B = V_h
            const uint32_t pt = tmem + (uint32_t)(buf * 128);
            const uint64_t vd = desc_swz(smem_u32(sV + (uint32_t)h * kVTile), kVSbo, kVSwz);
#pragma unroll
            for (int kk = 0; kk < BM / 16; ++kk)
              umma_bf16_tmem_a(tmem + 256u + (uint32_t)(h * DH), pt + (uint32_t)((kk >> 2) * 64 + (kk & 3) * 8),
                               desc_adv(vd, (uint32_t)kk * 16u * kVRow), idesc_pv, kk != 0 ? 1u : 0u);
            umma_commit(s_free + buf);
            if (h + 2 < H && !issue_s(h + 2)) break;
          }
          if (!ok) break;
          umma_commit(o_full);
          // ---- D: A WOx into [0, 128)
          if (!wait(a2_full, tl & 1)) break;
          if (!mma_sa(tmem)) break;
          umma_commit(ox_full);
          if (!wait(lnc_full, tl & 1)) break;
          tc_fence_after();
        }
        // ---- E: the head's first layer into [128, 256)
        if (!mma_sa(tmem + 128u)) break;
        umma_commit(head_full);
      }
    }
  } else {
    // ---------------- gathers, softmax and epilogues (warps 2..9) ----------------
    const int ew = warp - 2, q = warp & 3, qt = ew >> 2;  // lane quadrant, column quarter
    const int et = threadIdx.x - 64;
    const int r = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const float sl2 = p.scale_log2;
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 128;" ::"r"(1 + q) : "memory"); };  // the quadrant's 4 warps
    auto epi_sync = [&]() { asm volatile("bar.sync 5, %0;" ::"n"(32 * kEpiWarps) : "memory"); };
    bool ok = true;
    auto wait = [&](uint64_t* bar, uint32_t par) -> bool {
      if (!mbar_wait_compact(bar, par, p.sel.status)) ok = false;
      return ok;
    };
    int tl = 0, gf = 0;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
      const int b0 = t * G;
      const int Gv = min(G, p.B - b0);
      const int rows_v = Gv * K;
      const bool rvalid = r < rows_v;
      const int lr = r / K;
      // ================= A: assembly and the [CLS] attention =================
      // the tile's element rows [e0, e0 + nst) to shared memory by two bulk copies
      // (values, logit partials), over weight slots 2..6, which the producer
      // leaves alone until the gathers are done; rows past NST are read from memory
      uint8_t* sStage = sR + (size_t)kStageSlot * kBox;
      const int e0 = p.off[b0];
      const int nst = min(p.off[b0 + Gv] - e0, NST);
      const float* sVP = reinterpret_cast<const float*>(sStage + NST * 272);
      if (et == 0) {
        mbar_arrive_expect_tx(st_full, (uint32_t)nst * 272u + (uint32_t)L * (D * 4));
        if (nst > 0) {
          bulk_g2s(sStage, p.v_h + (size_t)e0 * D, (uint32_t)nst * 256u, st_full);
          bulk_g2s(sStage + NST * 256, p.elog + (size_t)e0 * 4, (uint32_t)nst * 16u, st_full);
        }
        bulk_g2s(sStage + NST * 272, p.vP, (uint32_t)L * (D * 4), st_full);
      }
      // element row of every occurrence of the tile (-1 for a rejected request)
      for (int i = et; i < rows_v * L; i += 32 * kEpiWarps) {
        const int rr = i / L, j = i - rr * L;
        const int b = b0 + rr / K;
        int e = -1;
        if (!p.bad[b]) e = p.off[b] + p.slot[(size_t)(b0 * K + rr) * L + j];
        sErow[rr * 32 + j] = e;
      }
      if (et < G) sFlag[et] = (et < Gv && p.bad[b0 + et]) ? 2 : 0;  // bit 1: a rejected request
      epi_sync();
      if (!wait(st_full, tl & 1)) break;
      if (nst == p.off[b0 + Gv] - e0)
        cls_rows<DH, true>(sA, sErow, sStage, sVP, sQkP, sQk0, sV0, p.v_h, p.elog, e0, nst, rows_v, L, sl2, ew, lane);
      else
        cls_rows<DH, false>(sA, sErow, sStage, sVP, sQkP, sQk0, sV0, p.v_h, p.elog, e0, nst, rows_v, L, sl2, ew, lane);
      // x0 = [CLS] into the accumulator (read by this thread in the previous tile's last phase)
      tmem_st32_nw(acc2 + lane_off + (uint32_t)(32 * qt), sCls + 32 * qt);
      tmem_st_wait();
      fence_async_shared();
      tc_fence_before();
      warp_arrive(a_full);
      // ================= B: c = cls + o WOs, FFN =================
      {
        const uint32_t proj = tmem + (uint32_t)((gf % NA1) * FC);
        if (!wait(o_done, tl & 1)) break;
        tc_fence_after();
        epi_resid_ln(sA, red, acc2 + lane_off, true, proj + lane_off, nullptr, nullptr, r, q, qt, p.eps);
        fence_async_shared();
        tc_fence_before();
        warp_arrive(ln_full);
      }
      for (int f = 0; f < nf; ++f, ++gf) {
        const int ba = gf % NA1;
        if (!wait(acc1_full + ba, (gf / NA1) & 1)) break;
        tc_fence_after();
        {
          // this thread's 32 hidden units: the hi plane (16 columns of bf16
          // pairs) then the lo plane over the same 32 TMEM columns
          const uint32_t col = tmem + lane_off + (uint32_t)(ba * FC + 32 * qt);
          const float* bias = sB1 + f * FC + 32 * qt;
          float v[32];
          tmem_ld32(col, v);
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int j = 0; j < 16; ++j)
            split2_trunc(relu_keep_nan(v[2 * j] + bias[2 * j]), relu_keep_nan(v[2 * j + 1] + bias[2 * j + 1]), hi[j],
                         lo[j]);
          tmem_st16_nowait(col, hi);
          tmem_st16_nowait(col + 16u, lo);
        }
        tmem_st_wait();
        tc_fence_before();
        warp_arrive(mid_full + ba);
      }
      if (!ok) break;
      // c = acc2 + b2s; Z = LN(c) (the cross-sequence block's input, or the head's)
      if (!wait(acc2_full, tl & 1)) break;
      tc_fence_after();
      epi_resid_ln(sA, red, acc2 + lane_off, false, 0u, sB2, (p.c_out && rvalid) ? p.c_out + (size_t)(b0 * K + r) * D : nullptr,
                   r, q, qt, p.eps);
      fence_async_shared();
      tc_fence_before();
      warp_arrive(z_full);
      if (p.cross) {
        // ================= C: cross-sequence attention =================
        if (!wait(qkv_full, tl & 1)) break;
        tc_fence_after();
        // Q and K as f16 K-major tiles [kb][128 rows x 128 B] at sA and sA + 32 KB;
        // V per head as an MN-major tile [128 keys x DH] in sV; a V row with a
        // non-finite value is written as zeros (P = 0 for other requests' rows
        // must not meet 0 x NaN) and marks its request
        bool bad_v = false;
#pragma unroll 1
        for (int part = 0; part < 3; ++part) {
          {
            const int c = 32 * qt;
            float v[32];
            tmem_ld32(tmem + lane_off + (uint32_t)(part * 128 + c), v);
            uint32_t w[16];
            bool fin = true;
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              if (part == 2) fin = fin && isfinite(v[2 * j]) && isfinite(v[2 * j + 1]);
              w[j] = pack_f16x2(v[2 * j], v[2 * j + 1]);
            }
            if (part < 2) {
              uint8_t* rowp = sA + (size_t)(part * 2 + c / BK) * kAPlane + (size_t)r * 128u;
#pragma unroll
              for (int jj = 0; jj < 4; ++jj) {
                const uint32_t o = (uint32_t)(((c % BK) / 8 + jj) ^ (r & 7)) << 4;
                *reinterpret_cast<uint4*>(rowp + o) = make_uint4(w[4 * jj], w[4 * jj + 1], w[4 * jj + 2], w[4 * jj + 3]);
              }
            } else {
              if (!fin) {
                bad_v = true;
#pragma unroll
                for (int j = 0; j < 16; ++j) w[j] = 0u;
              }
              const int h = c / DH, cc = c % DH;
              uint8_t* rowp = sV + (size_t)h * kVTile + (size_t)r * kVRow;
#pragma unroll
              for (int jj = 0; jj < 4; ++jj) {
                const int j16 = cc / 8 + jj;
                const int sw = DH == 32 ? (j16 ^ ((r >> 1) & 3)) : (j16 ^ (r & 7));
                *reinterpret_cast<uint4*>(rowp + ((uint32_t)sw << 4)) =
                    make_uint4(w[4 * jj], w[4 * jj + 1], w[4 * jj + 2], w[4 * jj + 3]);
              }
            }
          }
        }
        if (bad_v && rvalid) atomicOr(sFlag + lr, 1);  // bit 0: a non-finite value row
        fence_async_shared();
        tc_fence_before();
        warp_arrive(qkv_ready);
        // per head: softmax over the row's own request's K keys (keys of other
        // requests and padding rows take no part: -inf)
        const int klo = rvalid ? lr * K : 0, khi = rvalid ? lr * K + K : 0;
        float lh[4] = {1.f, 1.f, 1.f, 1.f};
        float* rmax = red;  // [quarter][row] (the LayerNorm statistics are consumed by now)
        float* rsum = red + 512;
#pragma unroll 1
        for (int h = 0; h < H; ++h) {
          const int g = tl * H + h, buf = g & 1;
          if (!wait(s_full + buf, (g >> 1) & 1)) break;
          tc_fence_after();
          const uint32_t tile = tmem + lane_off + (uint32_t)(buf * 128);
          float v[32];
          tmem_ld32(tile + (uint32_t)(32 * qt), v);  // keys 32 qt .. 32 qt + 31
          float mx = -INFINITY;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int key = 32 * qt + i;
            if (key < klo || key >= khi) v[i] = -INFINITY;
            mx = fmaxf(mx, v[i]);
          }
          rmax[qt * 128 + r] = mx;
          pair_sync();  // also: every warp of the quadrant has read its S columns before P overwrites them
          float m = fmaxf(fmaxf(rmax[r], rmax[128 + r]), fmaxf(rmax[256 + r], rmax[384 + r])) * sl2;
          if (m == -INFINITY) m = 0.f;  // a padding row: every P is 0
          float s4[4] = {0.f, 0.f, 0.f, 0.f};
          uint32_t pk[16];
#pragma unroll
          for (int i = 0; i < 32; i += 2) {
            const float p0 = ex2_approx(fmaf(v[i], sl2, -m));
            const float p1 = ex2_approx(fmaf(v[i + 1], sl2, -m));
            s4[(i >> 1) & 3] += p0 + p1;
            pk[i / 2] = pack_f16x2(p0, p1);
          }
          // P of keys 64 k + 32 j + [0, 32) in f16 pairs at columns 64 k + 16 j + [0, 16)
          tmem_st16_nowait(tile + (uint32_t)(64 * (qt >> 1) + 16 * (qt & 1)), pk);
          rsum[qt * 128 + r] = (s4[0] + s4[1]) + (s4[2] + s4[3]);
          tmem_st_wait();
          tc_fence_before();
          warp_arrive(p_full + buf);
          pair_sync();
          const float lt = (rsum[r] + rsum[128 + r]) + (rsum[256 + r] + rsum[384 + r]);
          const float lv = lt == 0.f ? 1.f : lt;  // 0 only for a padding row (a NaN stays NaN)
          lh[0] = h == 0 ? lv : lh[0];
          lh[1] = h == 1 ? lv : lh[1];
          lh[2] = h == 2 ? lv : lh[2];
          lh[3] = h == 3 ? lv : lh[3];
        }
        if (!ok) break;
        // the attention output O_h / l_h as the split A tile of the output projection
        if (!wait(o_full, tl & 1)) break;
        tc_fence_after();
        {
          float v[32];
          tmem_ld32(tmem + lane_off + 256u + (uint32_t)(32 * qt), v);
          const int hh = (32 * qt) / DH;
          const float inv = 1.f / (hh == 0 ? lh[0] : hh == 1 ? lh[1] : hh == 2 ? lh[2] : lh[3]);
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] *= inv;
          store_split32(sA, r, qt, v);
        }
        fence_async_shared();
        tc_fence_before();
        warp_arrive(a2_full);
        // ================= D: C' = c + A WOx, LN(C') =================
        if (!wait(ox_full, tl & 1)) break;
        tc_fence_after();
        epi_resid_ln(sA, red, acc2 + lane_off, true, tmem + lane_off, nullptr,
                     (p.cp_out && rvalid) ? p.cp_out + (size_t)(b0 * K + r) * D : nullptr, r, q, qt, p.eps);
        fence_async_shared();
        tc_fence_before();
        warp_arrive(lnc_full);
      }
      // ================= E: score head and the argmax of Eq. 1 =================
      if (!wait(head_full, tl & 1)) break;
      tc_fence_after();
      {
        float part = 0.f;
        {
          float v[32];
          tmem_ld32(tmem + 128u + lane_off + (uint32_t)(32 * qt), v);
          const int c = 32 * qt;
#pragma unroll
          for (int j = 0; j < 32; ++j) part = fmaf(relu_keep_nan(v[j] + sB1h[c + j]), sW2h[c + j], part);
        }
        tc_fence_before();
        red[qt * 128 + r] = part;
        pair_sync();
        float s = (red[r] + red[128 + r]) + (red[256 + r] + red[384 + r]) + sV0[D];
        if (rvalid) {
          if (sFlag[lr]) s = __int_as_float(0x7fc00000);
          p.scores[(size_t)(b0 * K + r)] = s;
          if (p.task_scores) p.task_scores[(size_t)(b0 * K + r)] = s;
          sSc[r] = s;
        }
      }
      epi_sync();
      // request lr2 of the tile, one warp each: the smallest k attaining the
      // maximum; -1 for a rejected request or a NaN score (the latter also flags
      // the batch)
      for (int lr2 = ew; lr2 < Gv; lr2 += kEpiWarps) {
        float mx = -INFINITY;
        int bk = 0x7FFFFFFF;
        bool nan = false;
        for (int k = lane; k < K; k += 32) {
          const float v = sSc[lr2 * K + k];
          if (v != v)
            nan = true;
          else if (v > mx || bk == 0x7FFFFFFF) {
            mx = v;
            bk = k;
          }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const float om = __shfl_xor_sync(0xffffffffu, mx, o);
          const int ok2 = __shfl_xor_sync(0xffffffffu, bk, o);
          if (ok2 != 0x7FFFFFFF && (bk == 0x7FFFFFFF || om > mx || (om == mx && ok2 < bk))) {
            mx = om;
            bk = ok2;
          }
        }
        nan = __any_sync(0xffffffffu, nan);
        if (lane == 0) {
          const bool rejected = (sFlag[lr2] & 2) != 0;
          const int best = (nan || rejected) ? -1 : bk;
          if (nan && !rejected) atomicOr(p.sel.status, ST_NUMERIC);
          p.sel.best[b0 + lr2] = best;
        }
      }
      epi_sync();
    }
  }

  __syncwarp();  // each warp arrives whole: single lanes ran the producer and MMA loops
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
  // the last CTA to finish hands the batch status to the host word and clears
  // the status and the ticket for the next batch
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) *last_flag = atomicAdd(p.sel.ticket, 1u) == gridDim.x - 1 ? 1u : 0u;
  __syncthreads();
  if (*last_flag && threadIdx.x == 0) {
    __threadfence();
    const int st = atomicExch(p.sel.status, 0);
    *p.sel.ticket = 0u;
    *reinterpret_cast<volatile int*>(p.sel.host_status) = st;
    __threadfence_system();
  }
}

// q0 . kP[j] per head (out[j * 4 + h], j < max_L) and q0 . k0 per head
// (out[max_L * 4 + h]); heads past H are 0.  Init time.
__global__ void seq_consts_kernel(const float* q0, const float* k0, const float* kP, int max_L, int d, int dh,
                                  float* out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (max_L + 1) * 4) return;
  const int j = i / 4, h = i % 4;
  float acc = 0.f;
  if (h * dh < d) {
    const float* kv = j < max_L ? kP + (size_t)j * d : k0;
    for (int c = h * dh; c < h * dh + dh; ++c) acc = fmaf(q0[c], kv[c], acc);
  }
  out[i] = acc;
}

cudaError_t seq_consts_launch(const float* q0, const float* k0, const float* kP, int max_L, int d, int dh, float* out,
                              cudaStream_t s) {
  const int n = (max_L + 1) * 4;
  seq_consts_kernel<<<(n + 127) / 128, 128, 0, s>>>(q0, k0, kP, max_L, d, dh, out);
  return cudaGetLastError();
}

namespace {
int g_seq_sms = 0;
}

bool seq_supported(int d, int dh, int F, int nb, int n_tasks, int K, int L) {
  return d == D && (dh == 32 || dh == 64) && F % FC == 0 && F >= FC && F <= kMaxF && nb == 1 && n_tasks <= 1 &&
         K >= 1 && K <= BM && L >= 1 && L <= kMaxL;
}

cudaError_t seq_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_seq_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(seq_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(seq_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
  return e;
}

cudaError_t seq_launch(const CUtensorMap* wos, const CUtensorMap* w1s, const CUtensorMap* w2s,
                       const CUtensorMap* qkvx, const CUtensorMap* wox, const CUtensorMap* w1h, const SeqParams& p0,
                       cudaStream_t s) {
  if (p0.B <= 0 || p0.K <= 0) return cudaSuccess;
  if (!seq_supported(D, p0.dh, p0.F, 1, 1, p0.K, p0.L) || p0.H * p0.dh != D || p0.G < 1 || p0.G * p0.K > BM)
    return cudaErrorInvalidValue;
  const long long tiles = (p0.B + p0.G - 1) / p0.G;
  long long grid = g_seq_sms > 0 ? g_seq_sms : 148;
  if (grid > tiles) grid = tiles;
  // without the cross-sequence block its maps are never read
  const CUtensorMap* qk = p0.cross ? qkvx : wos;
  const CUtensorMap* wx = p0.cross ? wox : wos;
  if (p0.dh == 32)
    return launch_k(seq_kernel<32>, dim3((unsigned)grid), dim3(kThreads), kSmem, s, *wos, *w1s, *w2s, *qk, *wx, *w1h,
                    p0);
  return launch_k(seq_kernel<64>, dim3((unsigned)grid), dim3(kThreads), kSmem, s, *wos, *w1s, *w2s, *qk, *wx, *w1h,
                  p0);
}

}  // namespace fe
