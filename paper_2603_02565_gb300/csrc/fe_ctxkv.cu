// Query Context Module of Section 4.2 in one kernel: X = LN(context rows),
// [K_0 | V_0 | K_1 | V_1 ...] = X [WK_0 | WV_0 | ...], for rows of width
// d <= 128 with bf16 inputs and bf16-exact weights.  LN(context) never
// reaches memory; K/V leave as one f16 plane (the attention operand).
//
// The N = 2 * n_layers * d output columns are split in two halves; CTA c
// owns half c % 2 (its slice of W^T stays resident in shared memory) and
// walks 128-row blocks of context rows:
//   warp 0 lane 0 : TMA -- the resident weight half once, then the raw
//                   context block of every tile into one of two staging
//                   buffers
//   warp 1 lane 0 : tcgen05.mma -- X W_half (N/2 <= 256 columns) into one of
//                   two TMEM accumulators, so the epilogue drains one tile
//                   while the next is multiplied
//   warps 2-9     : LayerNorm, two threads per context row (one 64-column
//                   half each, partial sums exchanged by shuffle), from the
//                   staged raw block into the split (hi/lo bf16) A operand tile
//   warps 10-17   : epilogue -- TMEM -> f16 -> 32 x 32 staging blocks -> TMA
//                   tensor stores; warps w and w+4 on TMEM lane quadrant w % 4,
//                   alternating 32-column chunks
// Each context row is normalised once per column half; the raw rows are
// bf16, so the second reading costs d * 2 bytes per row.
#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {
constexpr int BM = 128;
constexpr int BK = 64;
constexpr int kLnWarps = 8;
constexpr int kEpiWarps = 8;
constexpr int kThreads = 32 * (2 + kLnWarps + kEpiWarps);  // 576
constexpr uint32_t kPlane = BM * BK * 2;                     // 16 KB: 128 rows x 64 bf16
constexpr uint32_t kStage = 2048;                            // store staging: 32 rows x 32 f16, 64-byte swizzle
constexpr size_t kSmemMaxBlock = 232448;

struct CtxKvLayout {
  uint32_t w_bytes, a_bytes, raw_bytes;
  size_t smem;
};

__host__ __device__ inline CtxKvLayout ctxkv_layout(int d_pad, int N) {
  CtxKvLayout L;
  L.w_bytes = (uint32_t)(d_pad / BK) * (uint32_t)(N / 2) * (BK * 2);  // [kb][N/2 rows x 128 B]
  L.a_bytes = (uint32_t)(d_pad / BK) * 2u * kPlane;                   // [kb][hi, lo]
  L.raw_bytes = (uint32_t)(d_pad / BK) * kPlane;                      // one raw block [kb]
  L.smem = 1024 + (size_t)L.w_bytes + L.a_bytes + 2 * (size_t)L.raw_bytes + kEpiWarps * 2 * kStage + 256;
  return L;
}

__device__ __forceinline__ void arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }
}  // namespace

template <int NKB>
__global__ void __launch_bounds__(kThreads, 1)
    ctxkv_kernel(const __grid_constant__ CUtensorMap tX, const __grid_constant__ CUtensorMap tW,
                 const __grid_constant__ CUtensorMap tO, const CtxKvParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  const int Nh = p.N / 2, d = p.d;
  const CtxKvLayout LY = ctxkv_layout(NKB * BK, p.N);
  uint8_t* sW = smem;                                 // [kb][Nh rows x 128 B]
  uint8_t* sA = sW + LY.w_bytes;                      // [kb][hi, lo]
  uint8_t* sRaw = sA + LY.a_bytes;                    // [2 buffers][kb]
  uint8_t* sStg = sRaw + 2 * (size_t)LY.raw_bytes;    // [epilogue warp][2][2 KB]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sStg + kEpiWarps * 2 * kStage);
  uint64_t* w_full = bars;         // resident weight half loaded
  uint64_t* raw_full = bars + 1;   // [2] raw context block staged
  uint64_t* raw_empty = bars + 3;  // [2] the LayerNorm threads are done with it
  uint64_t* a_full = bars + 5;     // A tile written
  uint64_t* a_empty = bars + 6;    // the MMAs of the tile have read the A tile
  uint64_t* acc_full = bars + 7;   // [2] accumulator complete in TMEM
  uint64_t* acc_empty = bars + 9;  // [2] accumulator drained
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 11);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(raw_full + i, 1);
      mbar_init(raw_empty + i, 32 * kLnWarps);
      mbar_init(acc_full + i, 1);
      mbar_init(acc_empty + i, kEpiWarps);
    }
    mbar_init(a_full, 32 * kLnWarps);
    mbar_init(a_empty, 1);
    fence_mbar_init();
    prefetch_tmap(&tX);
    prefetch_tmap(&tW);
    prefetch_tmap(&tO);
  }
  // TMEM: accumulator i at columns [256 i, 256 i + Nh)
  if (warp == 0) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // CTA c: column half c % 2, row blocks c / 2, c / 2 + G, ... with G = gridDim.x / 2
  const int half = blockIdx.x & 1, G = gridDim.x >> 1;
  const int nblk = (p.rows + BM - 1) / BM;
  const int first = blockIdx.x >> 1;
  const int n_off = half * Nh;  // this CTA's output columns
  // the weight is a parameter: its load may start before the dependency wait
  if (warp == 0 && lane == 0 && first < nblk) {
    mbar_arrive_expect_tx(w_full, LY.w_bytes);
    for (int kb = 0; kb < NKB; ++kb)
      for (int n0 = 0; n0 < Nh; n0 += BM)
        tma_load_2d(sW + (size_t)kb * Nh * (BK * 2) + (size_t)n0 * (BK * 2), &tW, kb * BK, n_off + n0, w_full);
  }
  pdl_trigger();
  pdl_wait();
  if (first >= nblk) {
    if (warp == 0) tmem_dealloc(tmem, 512);
    return;
  }

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA: raw context blocks ----------------
      int it = 0;
      for (int t = first; t < nblk; t += G, ++it) {
        const int rb = it & 1;
        if (it >= 2 && !mbar_wait_bounded(raw_empty + rb, ((it >> 1) - 1) & 1, p.status)) break;
        mbar_arrive_expect_tx(raw_full + rb, LY.raw_bytes);
        // context row of this block (one K/V per candidate sequence: rep > 1)
        const int r0 = t * BM;
        const int in_row = p.rep > 1 ? ((r0 / p.C) / p.rep) * p.C + r0 % p.C : r0;
        for (int kb = 0; kb < NKB; ++kb)
          tma_load_2d(sRaw + (size_t)rb * LY.raw_bytes + (size_t)kb * kPlane, &tX, kb * BK, in_row, raw_full + rb);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc = umma_idesc_bf16(BM, Nh);
      bool ok = mbar_wait_bounded(w_full, 0, p.status);
      int it = 0;
      for (int t = first; t < nblk && ok; t += G, ++it) {
        const int ab = it & 1;
        if (it >= 2 && !mbar_wait_bounded(acc_empty + ab, ((it >> 1) - 1) & 1, p.status)) break;
        if (!mbar_wait_bounded(a_full, it & 1, p.status)) break;
        tc_fence_after();
        const uint32_t dst = tmem + (uint32_t)(256 * ab);
        const uint64_t a0 = umma_desc_sw128(smem_u32(sA));
        const uint64_t w0 = umma_desc_sw128(smem_u32(sW));
#pragma unroll
        for (int kb = 0; kb < NKB; ++kb) {
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint64_t ah = desc_adv(a0, (uint32_t)(kb * 2) * kPlane + kk * 32);
            const uint64_t wh = desc_adv(w0, (uint32_t)kb * (uint32_t)Nh * (BK * 2) + kk * 32);
            umma_bf16(dst, ah, wh, idesc, (kb | kk) != 0 ? 1u : 0u);
            umma_bf16(dst, desc_adv(ah, kPlane), wh, idesc, 1u);
          }
        }
        umma_commit(a_empty);  // the A tile frees once these MMAs complete
        umma_commit(acc_full + ab);
      }
    }
  } else if (warp < 2 + kLnWarps) {
    // ---------------- LayerNorm: two threads per row ----------------
    // lanes l and l ^ 16 share row r; part 0 takes pieces [0, 8 NKB / 2), part 1 the rest
    const int r = (warp - 2) * 16 + (lane & 15), part = lane >> 4;
    constexpr int kPieces = 4 * NKB;  // 16-byte pieces (8 columns) per thread
    int it = 0;
    for (int t = first; t < nblk; t += G, ++it) {
      const int rb = it & 1;
      if (!mbar_wait_bounded(raw_full + rb, (it >> 1) & 1, p.status)) break;
      const uint8_t* raw = sRaw + (size_t)rb * LY.raw_bytes;
      // piece j of this thread: global piece g = part * kPieces + j, column 8 g,
      // 128-byte-swizzled within its 64-column block
      auto gpiece = [&](int j) { return part * kPieces + j; };
      auto piece_off = [&](int g) {
        return (size_t)(g >> 3) * kPlane + (uint32_t)r * 128u + ((uint32_t)((g & 7) ^ (r & 7)) << 4);
      };
      float s = 0.f;  // padding columns past d read as zeros
#pragma unroll
      for (int j = 0; j < kPieces; ++j) {
        const uint4 q = *reinterpret_cast<const uint4*>(raw + piece_off(gpiece(j)));
        s += (bf16_lo(q.x) + bf16_hi(q.x)) + (bf16_lo(q.y) + bf16_hi(q.y)) + (bf16_lo(q.z) + bf16_hi(q.z)) +
             (bf16_lo(q.w) + bf16_hi(q.w));
      }
      s += __shfl_xor_sync(0xffffffffu, s, 16);
      const float mean = s / (float)d;
      float q2 = 0.f;
#pragma unroll
      for (int j = 0; j < kPieces; ++j) {
        const int g = gpiece(j);
        if (8 * g < d) {  // d is a multiple of 32: pieces are wholly inside or outside
          const uint4 q = *reinterpret_cast<const uint4*>(raw + piece_off(g));
          const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float a = bf16_lo(w[e]) - mean, b = bf16_hi(w[e]) - mean;
            q2 = fmaf(a, a, q2);
            q2 = fmaf(b, b, q2);
          }
        }
      }
      q2 += __shfl_xor_sync(0xffffffffu, q2, 16);
      const float rstd = 1.0f / sqrtf(q2 / (float)d + p.eps);
      // the previous tile's MMAs must be done with the A tile
      if (it > 0 && !mbar_wait_bounded(a_empty, (it - 1) & 1, p.status)) break;
#pragma unroll
      for (int j = 0; j < kPieces; ++j) {
        const int g = gpiece(j);
        uint32_t hi[4] = {0u, 0u, 0u, 0u}, lo[4] = {0u, 0u, 0u, 0u};
        if (8 * g < d) {
          const uint4 q = *reinterpret_cast<const uint4*>(raw + piece_off(g));
          const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
          for (int e = 0; e < 4; ++e)
            split2((bf16_lo(w[e]) - mean) * rstd, (bf16_hi(w[e]) - mean) * rstd, hi[e], lo[e]);
        }
        // A planes: hi of k block g / 8 at (2 (g / 8)) * kPlane, lo one plane after
        const size_t o = piece_off(g) + (size_t)(g >> 3) * kPlane;
        *reinterpret_cast<uint4*>(sA + o) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        *reinterpret_cast<uint4*>(sA + o + kPlane) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
      }
      arrive(raw_empty + rb);
      fence_async_shared();
      arrive(a_full);
    }
  } else {
    // ---------------- epilogue: TMEM -> f16 -> TMA stores ----------------
    const int ew = warp - 2 - kLnWarps;  // 0..7
    const int q = warp & 3;              // TMEM lane quadrant this warp may access
    const int sub = ew >> 2;             // alternate 32-column chunks
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    uint8_t* stg0 = sStg + (size_t)ew * 2 * kStage;
    int nstore = 0;
    int it = 0;
    for (int t = first; t < nblk; t += G, ++it) {
      const int ab = it & 1;
      if (!mbar_wait_bounded(acc_full + ab, (it >> 1) & 1, p.status)) break;
      tc_fence_after();
      const int srow = t * BM + q * 32;
      for (int c = 32 * sub; c < Nh; c += 64) {
        float v[32];
        tmem_ld32(tmem + lane_off + (uint32_t)(256 * ab + c), v);
        // alternate staging buffers; the one written two stores ago must be read
        uint8_t* b = stg0 + (size_t)(nstore & 1) * kStage;
        if (lane == 0 && nstore >= 2) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
        __syncwarp();
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t o = (uint32_t)lane * 64u + ((uint32_t)(j ^ ((lane >> 1) & 3)) << 4);
          *reinterpret_cast<uint4*>(b + o) =
              make_uint4(pack_f16x2(v[8 * j], v[8 * j + 1]), pack_f16x2(v[8 * j + 2], v[8 * j + 3]),
                         pack_f16x2(v[8 * j + 4], v[8 * j + 5]), pack_f16x2(v[8 * j + 6], v[8 * j + 7]));
        }
        fence_async_shared();
        __syncwarp();
        if (lane == 0) {
          // head-major K/V: column n_off + c is block (n_off + c) / dh, offset (n_off + c) % dh
          tma_store_3d(&tO, b, (n_off + c) % p.dh, srow, (n_off + c) / p.dh);  // rows past the extent are clipped
          bulk_commit();
        }
        ++nstore;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) arrive(acc_empty + ab);
    }
    if (lane == 0) bulk_wait0();  // output stores complete before the CTA retires
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

namespace {
int g_ctxkv_sms = 0;
}

bool ctxkv_supported(int d, int d_pad, int N, int nb, int io_f32) {
  if (io_f32 || nb != 1 || d > 128 || d % 32 || (d_pad != 64 && d_pad != 128)) return false;
  if (N % 256 || N > 512) return false;  // halves of 128 or 256 columns
  return ctxkv_layout(d_pad, N).smem <= kSmemMaxBlock;
}

cudaError_t ctxkv_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_ctxkv_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(ctxkv_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMaxBlock);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(ctxkv_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMaxBlock);
  return e;
}

cudaError_t ctxkv_launch(const CUtensorMap* x, const CUtensorMap* w, const CUtensorMap* o, int d_pad,
                         const CtxKvParams& p, cudaStream_t s) {
  if (p.rows <= 0) return cudaSuccess;
  const CtxKvLayout LY = ctxkv_layout(d_pad, p.N);
  const long long nblk = (p.rows + BM - 1) / BM;
  // an even grid: CTA pairs (2i, 2i+1) take the two column halves of the same row blocks
  long long grid = g_ctxkv_sms > 0 ? g_ctxkv_sms : 148;
  if (grid > 2 * nblk) grid = 2 * nblk;
  grid &= ~1LL;
  if (d_pad > BK)
    return launch_k(ctxkv_kernel<2>, dim3((unsigned)grid), dim3(kThreads), LY.smem, s, *x, *w, *o, p);
  return launch_k(ctxkv_kernel<1>, dim3((unsigned)grid), dim3(kThreads), LY.smem, s, *x, *w, *o, p);
}

}  // namespace fe
