// Distinct-element embedding, LayerNorm and the first layer's query
// projection in one kernel (Section 4.2: the element encoder's input h is the
// element's pool row, and its first cross-attention layer queries with
// LN(h) WQ_0), for d <= 128 with bf16 inputs and bf16-exact weights.
//
// Compact row r of the batch (distinct element r - off[b] of request b, b the
// largest request with off[b] <= r) is pool row b M + list[b cap + r - off[b]].
// The LayerNorm has no affine parameters, so with mu and rstd the row's mean
// and 1 / sqrt(var + eps),
//     LN(h) WQ = rstd (h WQ) - rstd mu (1^T WQ):
// the MMA multiplies the raw bf16 rows and the epilogue applies the row
// statistics with the column sums of WQ (as the context kernel does).  A
// persistent CTA walks 128-row tiles:
//   warp 0 lane 0 : TMA -- WQ^T [d rows x d_pad] once, resident
//   warp 1 lane 0 : tcgen05.mma -- raw tile . WQ into a d-column TMEM accumulator
//   warps 2-9     : two threads per row gather it (16-byte loads) into the
//                   128-byte-swizzled operand tile, write h (fp32) and the
//                   row's statistics; once the product is complete, the
//                   epilogue: rstd acc - rstd mu colsum -> f16 -> 32 x 32
//                   staging blocks -> TMA tensor stores of Q
// LN(h) itself never reaches memory: nothing else reads it when the next
// kernels are the fused FFN blocks.
#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {
constexpr int BM = 128;
constexpr int BK = 64;
constexpr int kGWarps = 8;                     // gather / epilogue warps
constexpr int kThreads = 64 + 32 * kGWarps;    // 320
constexpr uint32_t kPlane = BM * BK * 2;       // 16 KB: 128 rows x 64 bf16
constexpr uint32_t kWBytes = 2 * 128 * BK * 2; // WQ^T: up to 2 k blocks of 128 rows x 128 B
constexpr uint32_t kABytes = 2 * kPlane;       // operand tile: up to 2 k blocks
constexpr uint32_t kStage = 2048;              // store staging: 32 rows x 32 f16, 64-byte swizzle
constexpr uint32_t kStgBytes = kGWarps * 2 * kStage;
constexpr int kMaxOff = 4096;                  // request offsets staged in shared memory (B < kMaxOff)
constexpr size_t kSmem = 1024 + kWBytes + kABytes + kStgBytes + 128 * 4 + 128 * 8 + 256 + 4 * kMaxOff;

__device__ __forceinline__ void arrive1(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
// The eight gather / epilogue warps: a barrier, and one that also returns the
// AND of their flags (so that they leave the tile loop together)
__device__ __forceinline__ void gather_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }
__device__ __forceinline__ bool gather_sync_and(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, 1, 256, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ float lo16(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float hi16(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }
__device__ __forceinline__ float sum8(const uint4& q) {
  return ((lo16(q.x) + hi16(q.x)) + (lo16(q.y) + hi16(q.y))) + ((lo16(q.z) + hi16(q.z)) + (lo16(q.w) + hi16(q.w)));
}
}  // namespace

template <int NKB>
__global__ void __launch_bounds__(kThreads, 1)
    embed_q_kernel(const __grid_constant__ CUtensorMap tW, const __grid_constant__ CUtensorMap tQ,
                   const EmbedParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  const int d = p.d;
  uint8_t* sW = smem;                 // WQ^T [kb][d rows x 128 B]
  uint8_t* sA = sW + kWBytes;         // raw rows [kb][128 rows x 128 B], 128-byte swizzle
  uint8_t* sStg = sA + kABytes;       // [gather warp][2][2 KB]
  float* colsum = reinterpret_cast<float*>(sStg + kStgBytes);  // [d] column sums of WQ
  float2* stats = reinterpret_cast<float2*>(colsum + 128);      // [128] (rstd, -rstd mu) per tile row
  uint64_t* bars = reinterpret_cast<uint64_t*>(stats + 128);
  uint64_t* w_full = bars;        // WQ^T loaded
  uint64_t* a_full = bars + 1;    // operand tile written
  uint64_t* acc_full = bars + 2;  // product complete in TMEM
  uint64_t* acc_empty = bars + 3; // product read by the epilogue
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 4);
  int* sOff = reinterpret_cast<int*>(bars + 32);  // [B + 1] request offsets (when B < kMaxOff)

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    mbar_init(a_full, 32 * kGWarps);
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, kGWarps);
    fence_mbar_init();
    prefetch_tmap(&tW);
    prefetch_tmap(&tQ);
  }
  if (warp == 0) tmem_alloc(tmem_slot, 128);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // the weight is a parameter: its load may start before the dependency wait
  if (threadIdx.x == 0) {
    mbar_arrive_expect_tx(w_full, (uint32_t)NKB * (uint32_t)d * (BK * 2));
    for (int kb = 0; kb < NKB; ++kb) tma_load_2d(sW + (size_t)kb * d * (BK * 2), &tW, kb * BK, 0, w_full);
  }
  pdl_trigger();
  pdl_wait();
  const int rows_valid = min(p.off[p.B], p.rows);  // off[B]: distinct elements of the batch
  const int tiles = (rows_valid + BM - 1) / BM;
  if ((int)blockIdx.x >= tiles) {
    if (threadIdx.x == 0) mbar_wait_bounded(w_full, 0, p.status);  // no TMA write may land after the CTA
    __syncwarp();
    if (warp == 0) tmem_dealloc(tmem, 128);
    return;
  }

  if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc = umma_idesc_bf16(BM, d);
      bool ok = mbar_wait_bounded(w_full, 0, p.status);
      int tl = 0;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        if (tl > 0 && !mbar_wait_bounded(acc_empty, (tl - 1) & 1, p.status)) break;
        if (!mbar_wait_bounded(a_full, tl & 1, p.status)) break;
        tc_fence_after();
        const uint64_t a0 = umma_desc_sw128(smem_u32(sA));
        const uint64_t w0 = umma_desc_sw128(smem_u32(sW));
#pragma unroll
        for (int kb = 0; kb < NKB; ++kb) {
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            umma_bf16(tmem, desc_adv(a0, (uint32_t)kb * kPlane + kk * 32),
                      desc_adv(w0, (uint32_t)kb * (uint32_t)d * (BK * 2) + kk * 32), idesc, (kb | kk) != 0 ? 1u : 0u);
        }
        umma_commit(acc_full);
      }
    }
  } else if (warp >= 2) {
    // ---------------- gather + statistics, then epilogue (warps 2..9) ----------------
    const int gw = warp - 2;
    // gather: row gr of the tile, lanes l and l ^ 16 share it; of each 64-column
    // k block part 0 takes the first four 16-byte pieces, part 1 the last four
    const int gr = gw * 16 + (lane & 15), part = lane >> 4;
    constexpr int kPieces = 4 * NKB;
    // epilogue: TMEM lane quadrant q (tile rows 32 q ..), alternate 32-column chunks
    const int q = warp & 3, half = gw >> 2;
    const int er = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    uint8_t* stg = sStg + (size_t)gw * 2 * kStage;
    // column sums of WQ: row i of the resident WQ^T (the swizzle only permutes a row's pieces)
    // the request offsets to shared memory: each row's request is found by a
    // binary search over them, which would otherwise be a chain of dependent
    // global loads
    const bool off_staged = p.B < kMaxOff;
    if (off_staged)
      for (int i = gw * 32 + lane; i <= p.B; i += 32 * kGWarps) sOff[i] = p.off[i];
    bool ok = mbar_wait_bounded(w_full, 0, p.status);
    {
      const int i = gw * 32 + lane;
      if (ok && i < d) {
        float cs = 0.f;
        for (int kb = 0; kb < NKB; ++kb) {
          const uint8_t* wr = sW + ((size_t)kb * d + i) * (BK * 2);
#pragma unroll
          for (int j = 0; j < 8; ++j) cs += sum8(*reinterpret_cast<const uint4*>(wr + 16 * j));
        }
        colsum[i] = cs;
      }
    }
    bool go = gather_sync_and(ok);  // uniform over the eight warps
    int nstore = 0, tl = 0;
    for (int t = blockIdx.x; t < tiles && go; t += gridDim.x, ++tl) {
      const int m0 = t * BM;
      // ---- gather (the previous tile's product, which read the operand tile,
      // is complete: every warp has waited for it; its statistics are read)
      if (tl > 0) {
        go = gather_sync_and(ok);
        if (!go) break;
      }
      const int row = m0 + gr;
      const bool valid = row < rows_valid;
      uint4 pc[kPieces];
#pragma unroll
      for (int j = 0; j < kPieces; ++j) pc[j] = make_uint4(0u, 0u, 0u, 0u);
      if (valid) {
        int lo = 0, hi = p.B - 1;  // largest b with off[b] <= row
        if (off_staged) {
          while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (sOff[mid] <= row)
              lo = mid;
            else
              hi = mid - 1;
          }
        } else {
          while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (p.off[mid] <= row)
              lo = mid;
            else
              hi = mid - 1;
          }
        }
        const int m = p.list[(size_t)lo * p.cap + (row - p.off[lo])];
        const bf16* src = p.pool + ((size_t)lo * p.M + m) * d;
#pragma unroll
        for (int j = 0; j < kPieces; ++j) {
          const int g = (j >> 2) * 8 + part * 4 + (j & 3);  // 16-byte piece: columns 8 g .. 8 g + 7
          if (8 * g < d) pc[j] = *reinterpret_cast<const uint4*>(src + 8 * g);
        }
      }
      // statistics of the row (padding columns are zeros and take no part in the variance)
      float s = 0.f;
#pragma unroll
      for (int j = 0; j < kPieces; ++j) s += sum8(pc[j]);
      s += __shfl_xor_sync(0xffffffffu, s, 16);
      const float mean = s / (float)d;
      float q2 = 0.f;
#pragma unroll
      for (int j = 0; j < kPieces; ++j) {
        const int g = (j >> 2) * 8 + part * 4 + (j & 3);
        if (8 * g < d) {
          const uint32_t w4[4] = {pc[j].x, pc[j].y, pc[j].z, pc[j].w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float a = lo16(w4[e]) - mean, b = hi16(w4[e]) - mean;
            q2 = fmaf(a, a, q2);
            q2 = fmaf(b, b, q2);
          }
        }
      }
      q2 += __shfl_xor_sync(0xffffffffu, q2, 16);
      const float rstd = 1.0f / sqrtf(q2 / (float)d + p.eps);
      // the operand tile's row gr, and h
#pragma unroll
      for (int j = 0; j < kPieces; ++j) {
        const int g = (j >> 2) * 8 + part * 4 + (j & 3);
        *reinterpret_cast<uint4*>(sA + (size_t)(g >> 3) * kPlane + (uint32_t)gr * 128u +
                                  ((uint32_t)((g & 7) ^ (gr & 7)) << 4)) = pc[j];
        if (valid && 8 * g < d) {
          float* hr = p.h + (size_t)row * p.ldh + 8 * g;
          *reinterpret_cast<float4*>(hr) = make_float4(lo16(pc[j].x), hi16(pc[j].x), lo16(pc[j].y), hi16(pc[j].y));
          *reinterpret_cast<float4*>(hr + 4) =
              make_float4(lo16(pc[j].z), hi16(pc[j].z), lo16(pc[j].w), hi16(pc[j].w));
        }
      }
      if (part == 0) stats[gr] = valid ? make_float2(rstd, -mean * rstd) : make_float2(0.f, 0.f);
      fence_async_shared();
      arrive1(a_full);
      gather_sync();  // every row's statistics written
      // ---- epilogue: Q = rstd acc - rstd mu colsum, f16, through the staging blocks
      // (a wait that gives up skips it; the warps leave the loop together at the top)
      ok = mbar_wait_bounded(acc_full, tl & 1, p.status);
      tc_fence_after();
      const float2 st = stats[er];
      const int srow = m0 + q * 32;
      for (int c = 32 * half; c < d && ok; c += 64) {
        float v[32];
        tmem_ld32(tmem + lane_off + (uint32_t)c, v);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = fmaf(st.x, v[i], st.y * colsum[c + i]);
        uint8_t* b = stg + (size_t)(nstore & 1) * kStage;
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
          tma_store_2d(&tQ, b, c, srow);  // rows past the extent are clipped
          bulk_commit();
        }
        ++nstore;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) arrive1(acc_empty);
    }
    if (lane == 0) bulk_wait0();  // Q stores complete before the CTA retires
  }

  __syncwarp();  // each warp arrives whole: single lanes ran the MMA loop
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 128);
}

namespace {
int g_embed_sms = 0;
}

bool embed_q_supported(int d, int d_pad, int nb, int io_f32) {
  if (io_f32 || nb != 1 || d > 128 || d < 32 || d % 32) return false;
  return d_pad == (d > BK ? 2 * BK : BK);
}

cudaError_t embed_q_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_embed_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(embed_q_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(embed_q_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
  return e;
}

cudaError_t embed_q_launch(const CUtensorMap* w, const CUtensorMap* q_out, const EmbedParams& p, cudaStream_t s) {
  if (p.rows <= 0 || p.B <= 0) return cudaSuccess;
  if (!embed_q_supported(p.d, p.d_pad, 1, 0) || !p.pool || !p.off || !p.list || !p.h || p.ldh < p.d || p.ldh % 4)
    return cudaErrorInvalidValue;
  const long long tiles = (p.rows + BM - 1) / BM;  // (the valid rows, read on the device, are fewer)
  long long grid = g_embed_sms > 0 ? g_embed_sms : 148;
  if (grid > tiles) grid = tiles;
  const dim3 g((unsigned)grid), b(kThreads);
  return p.d_pad > BK ? launch_k(embed_q_kernel<2>, g, b, kSmem, s, *w, *q_out, p)
                      : launch_k(embed_q_kernel<1>, g, b, kSmem, s, *w, *q_out, p);
}

}  // namespace fe
