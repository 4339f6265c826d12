// Attention output projection and position-wise FFN of one block of the
// evaluator (element layers of Section 4.2, the SeqEnc block of Section 4.3),
// in one kernel:
//     x = x0 + A W_O,   x_out = x + ReLU(LN(x) W1 + b1) W2 + b2,   also LN(x_out)
// (A the attention output, x0 the block's input rows, or one row broadcast
// to every row) for rows of width d <= 128, without writing x, LN(x) or the
// F-wide intermediate to memory.  A persistent CTA walks 128-row tiles, F in
// chunks of 128 columns:
//   warp 0 lane 0 : TMA producer -- the A tile (hi/lo) and a ring of weight
//                   slots in consumption order W_O, W1_0, W1_1, W1_2, W2_0,
//                   W1_3, W2_1, ...
//   warp 1 lane 0 : tcgen05.mma -- A W_O into the TMEM buffer of FFN1 chunk
//                   0; after the epilogue has written x into the d-column
//                   accumulator and LN(x) in shared memory, FFN1 chunk f
//                   (N = 128) into one of three TMEM buffers, two chunks ahead
//                   of FFN2 of chunk f-2, which reads its A operand from that
//                   TMEM buffer and accumulates on top of x
//   warps 2-9     : per tile: x0 rows written into the accumulator while the
//                   projection runs, then x = x0 + A W_O written there and
//                   LN(x) written over the A tile as FFN1's operand; per chunk:
//                   bias + ReLU, split into hi/lo bf16 and written back over
//                   the chunk's fp32 columns in TMEM; per tile: x_out =
//                   accumulator + b2, LayerNorm, stored with TMA tensor stores
//                   staged in the tile's own 4 KB blocks
// The MMA groups are 16 instructions of N >= 128 so that the tensor pipe has
// queued work while the issuing thread polls its barriers; x0 is read by the
// epilogue warps while the A tile is in flight, when they have nothing else to
// do; the biases sit in shared memory.
#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

// ReLU that keeps a NaN (max.NaN): a NaN activation reaches the score, and so
// the argmax's NaN flag, instead of becoming 0 as with fmaxf.
__device__ __forceinline__ float relu_nan(float x) {
  float r;
  asm("max.NaN.f32 %0, %1, 0f00000000;" : "=f"(r) : "f"(x));
  return r;
}

namespace {
constexpr int BM = 128;
constexpr int BK = 64;
constexpr int FC = 128;                        // FFN columns per chunk
constexpr int NA1 = 3;                         // TMEM buffers for FFN1 chunks
constexpr int LA = 2;                          // FFN1 chunks issued ahead of the FFN2 that consumes them
constexpr int kEpiWarps = 8;
constexpr int kThreads = 64 + 32 * kEpiWarps;  // 320
constexpr uint32_t kAPlane = BM * BK * 2;      // 16 KB: 128 rows x 64 bf16
constexpr uint32_t kResBlock = 4096;           // residual block: 32 rows x 32 fp32, 128-byte swizzle
constexpr size_t kSmemMaxBlock = 232448;
constexpr int kMaxRing = 8;                    // weight slots
constexpr uint32_t kBarBytes = 512;  // 64 barriers
constexpr uint32_t kRedBytes = 2 * 2 * 128 * 4;  // [sum|var][half][row]

struct FfnLayout {
  uint32_t a_bytes, slot_bytes, w1_chunk, w2_chunk, wo_bytes, bias_bytes;
  int ring;
  size_t smem;
};

__host__ __device__ inline FfnLayout ffn_layout(int d, int d_pad, int F, int nb) {
  FfnLayout L;
  L.a_bytes = (uint32_t)(d_pad / BK) * 2u * kAPlane;
  L.w1_chunk = (uint32_t)nb * (uint32_t)(d_pad / BK) * (FC * BK * 2);  // [kb][plane][128 rows x 64]
  L.w2_chunk = (uint32_t)nb * 2u * (uint32_t)d * (BK * 2);             // [plane][half][d rows x 64]
  L.wo_bytes = (uint32_t)nb * (uint32_t)(d_pad / BK) * (uint32_t)d * (BK * 2);  // [kb][plane][d rows x 64]
  L.slot_bytes = L.w1_chunk > L.w2_chunk ? L.w1_chunk : L.w2_chunk;
  L.slot_bytes = (L.slot_bytes + 1023u) & ~1023u;
  L.bias_bytes = ((uint32_t)(F + 2 * d) * 4u + 127u) & ~127u;  // b1, b2, the broadcast x0 row
  const size_t fixed = 1024 + L.a_bytes + L.bias_bytes + kBarBytes + kRedBytes;
  L.ring = fixed < kSmemMaxBlock ? (int)((kSmemMaxBlock - fixed) / L.slot_bytes) : 0;
  if (L.ring > kMaxRing) L.ring = kMaxRing;
  L.smem = fixed + (size_t)L.ring * L.slot_bytes;
  return L;
}

__device__ __forceinline__ void mbar_arrive_one(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
}  // namespace

// NKB: 64-wide k blocks of d (1 or 2); NB: weight planes (1 or 2).  Both are
// compile-time constants so that the MMA issue sequences have no branches.
template <int NKB, int NB>
__global__ void __launch_bounds__(kThreads, 1)
    ffn_kernel(const __grid_constant__ CUtensorMap tA_h, const __grid_constant__ CUtensorMap tA_l,
               const __grid_constant__ CUtensorMap tWo_h, const __grid_constant__ CUtensorMap tWo_l,
               const __grid_constant__ CUtensorMap tW1_h, const __grid_constant__ CUtensorMap tW1_l,
               const __grid_constant__ CUtensorMap tW2_h, const __grid_constant__ CUtensorMap tW2_l,
               const __grid_constant__ CUtensorMap tO_h, const __grid_constant__ CUtensorMap tO_l,
               const __grid_constant__ CUtensorMap tO_x, const __grid_constant__ CUtensorMap tT_h,
               const __grid_constant__ CUtensorMap tT_l, const __grid_constant__ CUtensorMap tTo_h,
               const __grid_constant__ CUtensorMap tTo_l, const FfnParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  constexpr int nb = NB, nkb = NKB;
  const int d = p.d, F = p.F;
  const FfnLayout LY = ffn_layout(d, NKB * BK, F, nb);
  const int nf = F / FC;
  // sA: the A tile [kb][plane], then LN(x) [kb][plane] in the same layout,
  // then LN(x_out) the same way (stored from there, and the tail's A operand).
  // sW: the weight ring; at the end of a tile the x_out staging blocks
  // [32-column chunk][row quadrant][4 KB] at its start, then the tail weight
  // [kb][plane][tail_n rows x 128 B], later the tail's output staging.
  uint8_t* sA = smem;
  uint8_t* sW = sA + LY.a_bytes;
  const int tail_n = p.tail_n;
  uint8_t* sT = sW + (size_t)d * 512u;
  float* sB1 = reinterpret_cast<float*>(sW + (size_t)LY.ring * LY.slot_bytes);
  float* sB2 = sB1 + F;
  float* sX0 = sB2 + d;  // the broadcast row x0, when there is one
  uint64_t* bars = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(sB1) + LY.bias_bytes);
  uint64_t* a_full = bars;           // A tile loaded
  uint64_t* o_done = bars + 1;       // A W_O complete in the accumulator (the A tile is read)
  uint64_t* w_full = bars + 2;       // [kMaxRing]
  uint64_t* w_empty = bars + 10;     // [kMaxRing]
  uint64_t* acc1_full = bars + 18;   // [NA1] FFN1 chunk complete in TMEM buffer
  uint64_t* acc1_empty = bars + 21;  // [NA1] FFN2 has read the buffer's hidden activation
  uint64_t* mid_full = bars + 24;    // [NA1] hidden activation written over the buffer
  uint64_t* acc2_full = bars + 27;
  uint64_t* ln_full = bars + 29;     // x back in the accumulator, LN(x) in sA
  uint64_t* r_empty = bars + 30;     // staging blocks free again (their last store has read them)
  uint64_t* tail_a = bars + 31;      // LN(x_out) written in sA
  uint64_t* wt_full = bars + 32;     // tail weight loaded
  uint64_t* tail_full = bars + 33;   // tail product complete in TMEM
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 40);
  float* red = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + kBarBytes);  // [sum|var][half][128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(a_full, 1);
    mbar_init(o_done, 1);
    for (int i = 0; i < kMaxRing; ++i) {
      mbar_init(w_full + i, 1);
      mbar_init(w_empty + i, 1);
    }
    for (int i = 0; i < NA1; ++i) {
      mbar_init(acc1_full + i, 1);
      mbar_init(acc1_empty + i, 1);
      mbar_init(mid_full + i, kEpiWarps);
    }
    mbar_init(acc2_full, 1);
    mbar_init(ln_full, kEpiWarps);
    mbar_init(r_empty, kEpiWarps);
    mbar_init(tail_a, kEpiWarps);
    mbar_init(wt_full, 1);
    mbar_init(tail_full, 1);
    fence_mbar_init();
    prefetch_tmap(&tA_h);
    prefetch_tmap(&tWo_h);
    prefetch_tmap(&tW1_h);
    prefetch_tmap(&tW2_h);
  }
  // biases and the broadcast row are parameters, not outputs of an earlier
  // kernel: read before the dependency wait
  for (int i = threadIdx.x; i < F; i += kThreads) sB1[i] = p.b1[i];
  for (int i = threadIdx.x; i < d; i += kThreads) {
    sB2[i] = p.b2[i];
    sX0[i] = p.x0_row ? p.x0_row[i] : 0.f;
  }
  // TMEM: FFN1 chunk buffers at columns [128 i, 128 i + 128), i < 3; the
  // d-column accumulator of A W_O, x and FFN2 at [384, 384 + d)
  if (warp == 0) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t acc2 = tmem + (uint32_t)(NA1 * FC);
  pdl_trigger();
  pdl_wait();
  int rows_valid = p.rows;
  if (p.rows_dev) rows_valid = min(*p.rows_dev, p.rows);
  const int tiles = (rows_valid + BM - 1) / BM;
  if ((int)blockIdx.x >= tiles) {
    if (warp == 0) tmem_dealloc(tmem, 512);
    return;
  }

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int tl = 0, ws = 0;
      bool ok = true;
      // kind 0: W_O; 1: W1 rows [f*128, f*128+128); 2: W2 columns [f*128, f*128+128)
      auto load_slot = [&](int kind, int f) -> bool {
        const int slot = ws % LY.ring;
        if (ws >= LY.ring && !mbar_wait_bounded(w_empty + slot, ((ws / LY.ring) - 1) & 1, p.status)) return false;
        uint8_t* dst = sW + (size_t)slot * LY.slot_bytes;
        if (kind == 0) {  // every d row, every k block: [kb][plane][d rows x 64]
          mbar_arrive_expect_tx(w_full + slot, LY.wo_bytes);
          for (int kb = 0; kb < nkb; ++kb)
            for (int q = 0; q < nb; ++q)
              tma_load_2d(dst + (size_t)(kb * nb + q) * d * (BK * 2), q ? &tWo_l : &tWo_h, kb * BK, 0, w_full + slot);
        } else if (kind == 1) {  // every k block: [kb][plane][128 rows x 64]
          mbar_arrive_expect_tx(w_full + slot, LY.w1_chunk);
          for (int kb = 0; kb < nkb; ++kb)
            for (int q = 0; q < nb; ++q)
              tma_load_2d(dst + (size_t)(kb * nb + q) * (FC * BK * 2), q ? &tW1_l : &tW1_h, kb * BK, f * FC,
                          w_full + slot);
        } else {  // two 64-column halves, every d row: [plane][half][d rows x 64]
          mbar_arrive_expect_tx(w_full + slot, LY.w2_chunk);
          for (int q = 0; q < nb; ++q)
            for (int hh = 0; hh < 2; ++hh)
              tma_load_2d(dst + (size_t)(q * 2 + hh) * d * (BK * 2), q ? &tW2_l : &tW2_h, f * FC + BK * hh, 0,
                          w_full + slot);
        }
        ++ws;
        return true;
      };
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        // sA holds the previous tile's output staging until its stores have read it
        if (tl > 0 && !mbar_wait_bounded(r_empty, (tl - 1) & 1, p.status)) break;
        mbar_arrive_expect_tx(a_full, LY.a_bytes);
        for (int kb = 0; kb < nkb; ++kb) {
          tma_load_2d(sA + (size_t)(kb * 2) * kAPlane, &tA_h, kb * BK, t * BM, a_full);
          tma_load_2d(sA + (size_t)(kb * 2 + 1) * kAPlane, &tA_l, kb * BK, t * BM, a_full);
        }
        if (!load_slot(0, 0)) break;
        for (int s = 0; s < nf + LA && ok; ++s) {
          if (s < nf && !load_slot(1, s)) ok = false;
          if (ok && s >= LA && !load_slot(2, s - LA)) ok = false;
        }
        if (ok && tail_n > 0) {
          // the tail weight, past the x_out staging, once every FFN MMA of the
          // tile (the last readers of the ring) has completed
          if (!mbar_wait_bounded(acc2_full, tl & 1, p.status)) break;
          mbar_arrive_expect_tx(wt_full, (uint32_t)nkb * nb * (uint32_t)tail_n * (BK * 2));
          for (int kb = 0; kb < nkb; ++kb)
            for (int q = 0; q < nb; ++q)
              tma_load_2d(sT + (size_t)(kb * nb + q) * tail_n * (BK * 2), q ? &tT_l : &tT_h, kb * BK, 0, wt_full);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc1 = umma_idesc_bf16(BM, FC);
      const uint32_t idesc2 = umma_idesc_bf16(BM, d);
      int tl = 0, ws = 0, gf = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        // ---- A W_O into the FFN1 buffer that chunk 0 of this tile uses next
        if (!mbar_wait_bounded(a_full, tl & 1, p.status)) break;
        {
          const int slot = ws % LY.ring, bo = gf % NA1;
          if (!mbar_wait_bounded(w_full + slot, (ws / LY.ring) & 1, p.status)) break;
          if (gf >= NA1 && !mbar_wait_bounded(acc1_empty + bo, ((gf / NA1) - 1) & 1, p.status)) break;
          tc_fence_after();
          const uint32_t dst = tmem + (uint32_t)(bo * FC);
          const uint64_t a0 = umma_desc_sw128(smem_u32(sA));
          const uint64_t w0 = umma_desc_sw128(smem_u32(sW + (size_t)slot * LY.slot_bytes));
#pragma unroll
          for (int kb = 0; kb < nkb; ++kb) {
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
              const uint64_t ah = desc_adv(a0, (uint32_t)(kb * 2) * kAPlane + kk * 32);
              const uint64_t wh = desc_adv(w0, (uint32_t)(kb * nb) * (uint32_t)d * (BK * 2) + kk * 32);
              umma_bf16(dst, ah, wh, idesc2, (kb | kk) != 0 ? 1u : 0u);
              umma_bf16(dst, desc_adv(ah, kAPlane), wh, idesc2, 1u);
              if (nb > 1) umma_bf16(dst, ah, desc_adv(wh, (uint32_t)d * (BK * 2)), idesc2, 1u);
            }
          }
          umma_commit(w_empty + slot);
          umma_commit(o_done);
          ++ws;
        }
        // ---- FFN1 / FFN2 once the epilogue has put x in the accumulator and LN(x) in sA
        if (!mbar_wait_bounded(ln_full, tl & 1, p.status)) break;
        tc_fence_after();
        const int gf0 = gf;
        for (int s = 0; s < nf + LA && ok; ++s) {
          if (s < nf) {
            // FFN1 chunk s -> acc1 buffer (gf0 + s) % NA1
            const int g = gf0 + s, b = g % NA1;
            // (chunk 0's buffer: waited for before the projection, read by the epilogue before ln_full)
            if (s > 0 && g >= NA1 && !mbar_wait_bounded(acc1_empty + b, ((g / NA1) - 1) & 1, p.status)) {
              ok = false;
              break;
            }
            const int slot = ws % LY.ring;
            if (!mbar_wait_bounded(w_full + slot, (ws / LY.ring) & 1, p.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t dst = tmem + (uint32_t)(b * FC);
            const uint64_t a0 = umma_desc_sw128(smem_u32(sA));
            const uint64_t w0 = umma_desc_sw128(smem_u32(sW + (size_t)slot * LY.slot_bytes));
#pragma unroll
            for (int kb = 0; kb < nkb; ++kb) {
#pragma unroll
              for (int kk = 0; kk < BK / 16; ++kk) {
                const uint64_t ah = desc_adv(a0, (uint32_t)(kb * 2) * kAPlane + kk * 32);
                const uint64_t wh = desc_adv(w0, (uint32_t)(kb * nb) * (FC * BK * 2) + kk * 32);
                umma_bf16(dst, ah, wh, idesc1, (kb | kk) != 0 ? 1u : 0u);
                umma_bf16(dst, desc_adv(ah, kAPlane), wh, idesc1, 1u);
                if (nb > 1) umma_bf16(dst, ah, desc_adv(wh, FC * BK * 2), idesc1, 1u);
              }
            }
            umma_commit(w_empty + slot);
            umma_commit(acc1_full + b);
            ++ws;
          }
          if (s >= LA) {
            // FFN2 chunk c = s - LA: acc2 += mid(c) . W2 chunk c, mid(c) from TMEM buffer g % NA1
            const int c = s - LA, g = gf0 + c, b = g % NA1;
            if (!mbar_wait_bounded(mid_full + b, (g / NA1) & 1, p.status)) {
              ok = false;
              break;
            }
            const int slot = ws % LY.ring;
            if (!mbar_wait_bounded(w_full + slot, (ws / LY.ring) & 1, p.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            // each 32-column piece of the buffer holds 32 hidden units: hi plane in
            // its first 16 columns, lo plane in the next 16 (two bf16 per column);
            // the W2 slot holds 64-column halves of the chunk, d rows each
            const uint32_t mt = tmem + (uint32_t)(b * FC);
            const uint64_t w0 = umma_desc_sw128(smem_u32(sW + (size_t)slot * LY.slot_bytes));
#pragma unroll
            for (int kk = 0; kk < FC / 16; ++kk) {
              const int hh = kk >> 2, k4 = kk & 3;
              const uint32_t mh = mt + (uint32_t)(32 * (kk >> 1) + 8 * (kk & 1)), ml = mh + 16;
              const uint64_t wh = desc_adv(w0, (uint32_t)hh * (uint32_t)d * (BK * 2) + k4 * 32);
              umma_bf16_tmem_a(acc2, mh, wh, idesc2, 1u);
              umma_bf16_tmem_a(acc2, ml, wh, idesc2, 1u);
              if (nb > 1) umma_bf16_tmem_a(acc2, mh, desc_adv(wh, 2u * (uint32_t)d * (BK * 2)), idesc2, 1u);
            }
            umma_commit(w_empty + slot);
            umma_commit(acc1_empty + b);
            ++ws;
            if (c == nf - 1) umma_commit(acc2_full);
          }
        }
        gf = gf0 + nf;
        if (ok && tail_n > 0) {
          // tail: LN(x_out) . W_t into TMEM columns [0, tail_n) (every FFN1
          // buffer is free once the FFN2 of the tile has completed)
          if (!mbar_wait_bounded(tail_a, tl & 1, p.status)) break;
          if (!mbar_wait_bounded(wt_full, tl & 1, p.status)) break;
          tc_fence_after();
          const uint32_t idesc3 = umma_idesc_bf16(BM, tail_n);
          const uint64_t a0 = umma_desc_sw128(smem_u32(sA));
          const uint64_t w0 = umma_desc_sw128(smem_u32(sT));
#pragma unroll
          for (int kb = 0; kb < nkb; ++kb) {
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
              const uint64_t ah = desc_adv(a0, (uint32_t)(kb * 2) * kAPlane + kk * 32);
              const uint64_t wh = desc_adv(w0, (uint32_t)(kb * nb) * (uint32_t)tail_n * (BK * 2) + kk * 32);
              umma_bf16(tmem, ah, wh, idesc3, (kb | kk) != 0 ? 1u : 0u);
              umma_bf16(tmem, desc_adv(ah, kAPlane), wh, idesc3, 1u);
              if (nb > 1) umma_bf16(tmem, ah, desc_adv(wh, (uint32_t)tail_n * (BK * 2)), idesc3, 1u);
            }
          }
          umma_commit(tail_full);
        }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..9) ----------------
    const int ew = warp - 2, q = warp & 3, half = ew >> 2;
    const int r = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    float* red_sum = red;
    float* red_var = red + 256;
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + q) : "memory"); };
    // tensor stores of this warp's staged blocks; the reads are awaited separately
    auto issue = [&](const CUtensorMap* m0p, const void* s0, const CUtensorMap* m1p, const void* s1, int col,
                     int row) {
      fence_async_shared();
      __syncwarp();
      if (lane == 0) {
        tma_store_2d(m0p, s0, col, row);
        if (m1p) tma_store_2d(m1p, s1, col, row);
        bulk_commit();
      }
      __syncwarp();
    };
    auto stores_read = [&]() {
      if (lane == 0) bulk_wait_read0();
      __syncwarp();
    };
    // one arrival per warp on barriers counted in warps (the lanes synchronise first)
    auto warp_arrive = [&](uint64_t* bar) {
      __syncwarp();
      if (lane == 0) mbar_arrive_one(bar);
    };
    int tl = 0, gf = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
      const int m0 = t * BM;
      const int srow = m0 + q * 32;
      const bool valid = m0 + r < rows_valid;
      // ---- x = x0 + A W_O for this thread's row, columns 32 half + 64 ci + [0, 32)
      // (x0 of rows past the valid count is 0): x0 goes into the accumulator
      // while the projection runs into the FFN1 buffer of chunk 0, x goes
      // back into the accumulator for FFN2 to add to, and LN(x) into sA (which
      // the projection has read) as FFN1's A tile.
      auto load_x0 = [&](int c, float* x) {
        const float* src = p.x0_row ? nullptr : p.x0 + (size_t)(m0 + r) * p.ldx0 + c;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
          if (p.x0_row)
            v = *reinterpret_cast<const float4*>(sX0 + c + 4 * j);
          else if (valid)
            v = *reinterpret_cast<const float4*>(src + 4 * j);
          x[4 * j] = v.x;
          x[4 * j + 1] = v.y;
          x[4 * j + 2] = v.z;
          x[4 * j + 3] = v.w;
        }
      };
      // x0 into the accumulator (this warp's lanes and columns, read by this
      // warp in the previous tile's final phase) while the projection runs
#pragma unroll
      for (int ci = 0; ci < 2; ++ci) {
        const int c = 32 * half + 64 * ci;
        if (c < d) {
          float xr[32];
          load_x0(c, xr);
          tmem_st32(acc2 + lane_off + (uint32_t)c, xr);
        }
      }
      const uint32_t proj = tmem + (uint32_t)((gf % NA1) * FC);  // A W_O
      if (!mbar_wait_bounded(o_done, tl & 1, p.status)) break;
      tc_fence_after();
      float s4[4] = {0.f, 0.f, 0.f, 0.f};  // four independent partial sums per statistic
#pragma unroll
      for (int ci = 0; ci < 2; ++ci) {
        const int c = 32 * half + 64 * ci;
        if (c < d) {
          float v[32], w[32];
          tmem_ld32(proj + lane_off + (uint32_t)c, v);
          tmem_ld32(acc2 + lane_off + (uint32_t)c, w);
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            v[j] += w[j];
            s4[j & 3] += v[j];
          }
          tmem_st32(acc2 + lane_off + (uint32_t)c, v);
        }
      }
      red_sum[half * 128 + r] = (s4[0] + s4[1]) + (s4[2] + s4[3]);
      pair_sync();
      const float mean0 = (red_sum[r] + red_sum[128 + r]) / (float)d;
      // x is read back from the accumulator rather than kept in registers
#pragma unroll
      for (int i = 0; i < 4; ++i) s4[i] = 0.f;
#pragma unroll
      for (int ci = 0; ci < 2; ++ci) {
        const int c = 32 * half + 64 * ci;
        if (c < d) {
          float v[32];
          tmem_ld32(acc2 + lane_off + (uint32_t)c, v);
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float dv = v[j] - mean0;
            s4[j & 3] = fmaf(dv, dv, s4[j & 3]);
          }
        }
      }
      red_var[half * 128 + r] = (s4[0] + s4[1]) + (s4[2] + s4[3]);
      pair_sync();
      const float rstd0 = 1.0f / sqrtf((red_var[r] + red_var[128 + r]) / (float)d + p.eps);
      // row r of planes (kb, hi) and (kb, lo), 128-byte swizzle: this warp's
      // four 16-byte pieces 4 half + jj; columns past d are zeros
#pragma unroll
      for (int ci = 0; ci < nkb; ++ci) {
        const int c = 32 * half + 64 * ci;
        uint32_t hi[16], lo[16];
        if (c < d) {
          float v[32];
          tmem_ld32(acc2 + lane_off + (uint32_t)c, v);
#pragma unroll
          for (int j = 0; j < 16; ++j) split2((v[2 * j] - mean0) * rstd0, (v[2 * j + 1] - mean0) * rstd0, hi[j], lo[j]);
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            hi[j] = 0u;
            lo[j] = 0u;
          }
        }
        uint8_t* rowp = sA + (size_t)(ci * 2) * kAPlane + (size_t)r * 128u;
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
          const uint32_t o = (uint32_t)((4 * half + jj) ^ (r & 7)) << 4;
          *reinterpret_cast<uint4*>(rowp + o) = make_uint4(hi[4 * jj], hi[4 * jj + 1], hi[4 * jj + 2], hi[4 * jj + 3]);
          *reinterpret_cast<uint4*>(rowp + kAPlane + o) =
              make_uint4(lo[4 * jj], lo[4 * jj + 1], lo[4 * jj + 2], lo[4 * jj + 3]);
        }
      }
      fence_async_shared();
      tc_fence_before();
      warp_arrive(ln_full);
      // ---- per chunk: mid = split(ReLU(acc1 + b1)) written back over this
      // warp's 64 columns of the chunk's TMEM buffer as FFN2's A operand
      for (int f = 0; f < nf; ++f, ++gf) {
        const int ba = gf % NA1;
        if (!mbar_wait_bounded(acc1_full + ba, (gf / NA1) & 1, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // this warp's 64 columns as two 32-column pieces, each read whole and
        // then overwritten by its own hi (16 columns) and lo (16 columns) planes
#pragma unroll
        for (int hp = 0; hp < 2; ++hp) {
          const uint32_t col = tmem + lane_off + (uint32_t)(ba * FC + 64 * half + 32 * hp);
          const float* bias = sB1 + f * FC + 64 * half + 32 * hp;
          float v[32];
          tmem_ld32(col, v);
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float2 bb = *reinterpret_cast<const float2*>(bias + 2 * j);
            split2_trunc(relu_nan(v[2 * j] + bb.x), relu_nan(v[2 * j + 1] + bb.y), hi[j], lo[j]);
          }
          tmem_st16_nowait(col, hi);
          tmem_st16_nowait(col + 16, lo);
        }
        tmem_st_wait();
        tc_fence_before();
        warp_arrive(mid_full + ba);
      }
      if (!ok) break;
      // ---- final: x_out = acc2 + b2 (acc2 = x + FFN2), LayerNorm, stores
      if (!mbar_wait_bounded(acc2_full, tl & 1, p.status)) break;
      tc_fence_after();
      // this warp's x_out staging blocks at the start of the weight ring (every
      // MMA of the tile has completed, and before r_empty the producer loads
      // only the tail weight, past them): column chunks half and half + 2 of
      // row quadrant q
      auto blk = [&](int ci) { return sW + (size_t)((half + 2 * ci) * 4 + q) * kResBlock; };
      // row chunk of 32 fp32 in a block: 16-byte piece j of row `lane`, 128-byte swizzle
      auto xoff = [&](int j) { return (uint32_t)lane * 128u + ((uint32_t)(j ^ (lane & 7)) << 4); };
      float sum2 = 0.f;
#pragma unroll
      for (int ci = 0; ci < 2; ++ci) {
        const int c = 32 * half + 64 * ci;
        if (c < d) {
          float v[32];
          tmem_ld32(acc2 + lane_off + (uint32_t)c, v);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 bb = *reinterpret_cast<const float4*>(sB2 + c + 4 * j);
            float4 x;
            x.x = v[4 * j] + bb.x;
            x.y = v[4 * j + 1] + bb.y;
            x.z = v[4 * j + 2] + bb.z;
            x.w = v[4 * j + 3] + bb.w;
            sum2 += (x.x + x.y) + (x.z + x.w);
            *reinterpret_cast<float4*>(blk(ci) + xoff(j)) = x;
          }
        }
      }
#pragma unroll
      for (int ci = 0; ci < 2; ++ci) {
        const int c = 32 * half + 64 * ci;
        if (c < d) issue(&tO_x, blk(ci), nullptr, nullptr, c, srow);
      }
      red_sum[half * 128 + r] = sum2;
      pair_sync();
      const float mean = (red_sum[r] + red_sum[128 + r]) / (float)d;
      float v4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int ci = 0; ci < 2; ++ci) {
        if (32 * half + 64 * ci < d) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 x = *reinterpret_cast<const float4*>(blk(ci) + xoff(j));
            const float d0 = x.x - mean, d1 = x.y - mean, d2 = x.z - mean, d3 = x.w - mean;
            v4[0] = fmaf(d0, d0, v4[0]);
            v4[1] = fmaf(d1, d1, v4[1]);
            v4[2] = fmaf(d2, d2, v4[2]);
            v4[3] = fmaf(d3, d3, v4[3]);
          }
        }
      }
      red_var[half * 128 + r] = (v4[0] + v4[1]) + (v4[2] + v4[3]);
      pair_sync();
      const float rstd = 1.0f / sqrtf((red_var[r] + red_var[128 + r]) / (float)d + p.eps);
      // LN(x_out) as the split tile [kb][plane] in sA, 128-byte swizzle (every
      // FFN1 has read the LN(x) tile there): row r, this warp's four 16-byte
      // pieces 4 half + jj of each plane; columns past d are zeros
#pragma unroll
      for (int ci = 0; ci < nkb; ++ci) {
        const int c = 32 * half + 64 * ci;
        uint32_t hi[16], lo[16];
        if (c < d) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 x = *reinterpret_cast<const float4*>(blk(ci) + xoff(j));
            split2((x.x - mean) * rstd, (x.y - mean) * rstd, hi[2 * j], lo[2 * j]);
            split2((x.z - mean) * rstd, (x.w - mean) * rstd, hi[2 * j + 1], lo[2 * j + 1]);
          }
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            hi[j] = 0u;
            lo[j] = 0u;
          }
        }
        uint8_t* rowp = sA + (size_t)(ci * 2) * kAPlane + (size_t)r * 128u;
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
          const uint32_t o = (uint32_t)((4 * half + jj) ^ (r & 7)) << 4;
          *reinterpret_cast<uint4*>(rowp + o) = make_uint4(hi[4 * jj], hi[4 * jj + 1], hi[4 * jj + 2], hi[4 * jj + 3]);
          *reinterpret_cast<uint4*>(rowp + kAPlane + o) =
              make_uint4(lo[4 * jj], lo[4 * jj + 1], lo[4 * jj + 2], lo[4 * jj + 3]);
        }
      }
      fence_async_shared();
      if (tail_n > 0) warp_arrive(tail_a);
      if (p.store_ln) {
        asm volatile("bar.sync 5, 256;" ::: "memory");  // every row of the tile written
        if (ew == 0 && lane == 0) {
          for (int kb = 0; kb < nkb; ++kb) {
            tma_store_2d(&tO_h, sA + (size_t)(kb * 2) * kAPlane, kb * BK, m0);
            tma_store_2d(&tO_l, sA + (size_t)(kb * 2 + 1) * kAPlane, kb * BK, m0);
          }
          bulk_commit();
        }
        __syncwarp();
      }
      if (tail_n > 0) {
        // tail output: 32-column chunks half, half + 2, ... of this warp's row
        // quadrant, f16 (one 2 KB block) or a split pair (two), through two
        // rotating staging buffers of this warp where the tail weight was
        if (!mbar_wait_bounded(tail_full, tl & 1, p.status)) break;
        tc_fence_after();
        const uint32_t tb = p.tail_f16 ? 2048u : 4096u;
        uint8_t* stg = sT + (size_t)ew * 2u * tb;
        int k = 0;
        for (int c = 32 * half; c < tail_n; c += 64) {
          float v[32];
          tmem_ld32(tmem + lane_off + (uint32_t)c, v);
          if (p.tail_q0 && c < d) {
            // a key group of SeqEnc: only its [CLS] logit partial q0 . k leaves the SM
            float acc = 0.f;
            const float4* q = reinterpret_cast<const float4*>(p.tail_q0 + c);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 qq = __ldg(q + j);
              acc = fmaf(v[4 * j], qq.x, acc);
              acc = fmaf(v[4 * j + 1], qq.y, acc);
              acc = fmaf(v[4 * j + 2], qq.z, acc);
              acc = fmaf(v[4 * j + 3], qq.w, acc);
            }
            if (valid) p.tail_logits[(size_t)(m0 + r) * (size_t)(d / 32) + (size_t)(c / 32)] = acc;
            continue;
          }
          uint8_t* b = stg + (size_t)(k & 1) * tb;
          if (lane == 0 && k >= 2) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
          __syncwarp();
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint32_t o = (uint32_t)lane * 64u + ((uint32_t)(j ^ ((lane >> 1) & 3)) << 4);
            if (p.tail_f16) {
              *reinterpret_cast<uint4*>(b + o) =
                  make_uint4(pack_f16x2(v[8 * j], v[8 * j + 1]), pack_f16x2(v[8 * j + 2], v[8 * j + 3]),
                             pack_f16x2(v[8 * j + 4], v[8 * j + 5]), pack_f16x2(v[8 * j + 6], v[8 * j + 7]));
            } else {
              uint32_t hi[4], lo[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) split2(v[8 * j + 2 * e], v[8 * j + 2 * e + 1], hi[e], lo[e]);
              *reinterpret_cast<uint4*>(b + o) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
              *reinterpret_cast<uint4*>(b + 2048 + o) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
          }
          issue(&tTo_h, b, p.tail_f16 ? nullptr : &tTo_l, b + 2048, c - p.tail_col0, srow);
          ++k;
        }
        tc_fence_before();  // TMEM read before r_empty lets the next tile's projection in
      }
      stores_read();
      if (lane == 0) mbar_arrive_one(r_empty);  // sA and the ring may take the next tile's loads
    }
    if (lane == 0) bulk_wait0();  // output tensor stores complete before the CTA retires
  }

  __syncwarp();  // each warp arrives whole: lane 0 of warps 0 and 1 ran the producer and MMA loops
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

namespace {
int g_ffn_sms = 0;
}

bool ffn_supported(int d, int d_pad, int F, int nb) {
  if (d > 128 || d % 32 || F % FC || F < FC || NA1 * FC + d > 512) return false;
  if (d_pad != (d > BK ? 2 * BK : BK)) return false;
  const FfnLayout L = ffn_layout(d, d_pad, F, nb);
  // the ring also stages x_out: d / 32 column chunks x 4 row quadrants x 4 KB
  return L.ring >= 2 && L.smem <= kSmemMaxBlock && (size_t)L.ring * L.slot_bytes >= (size_t)d * 512u;
}

bool ffn_tail_supported(int d, int d_pad, int F, int nb, int tail_n, int tail_f16) {
  if (!ffn_supported(d, d_pad, F, nb)) return false;
  if (tail_n < 32 || tail_n > 256 || tail_n % 32) return false;
  const FfnLayout L = ffn_layout(d, d_pad, F, nb);
  // past the x_out staging: the tail weight, then the tail staging (8 warps x 2 buffers)
  const size_t wt = (size_t)(d_pad / BK) * nb * tail_n * (BK * 2);
  const size_t stg = (size_t)kEpiWarps * 2u * (tail_f16 ? 2048u : 4096u);
  return (size_t)d * 512u + (wt > stg ? wt : stg) <= (size_t)L.ring * L.slot_bytes;
}

cudaError_t ffn_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_ffn_sms, cudaDevAttrMultiProcessorCount, dev);
  auto attr = [&](const void* f) {
    if (e == cudaSuccess) e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMaxBlock);
  };
  attr((const void*)ffn_kernel<1, 1>);
  attr((const void*)ffn_kernel<1, 2>);
  attr((const void*)ffn_kernel<2, 1>);
  attr((const void*)ffn_kernel<2, 2>);
  return e;
}

cudaError_t ffn_launch(const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* wo_h,
                       const CUtensorMap* wo_l, const CUtensorMap* w1_h, const CUtensorMap* w1_l,
                       const CUtensorMap* w2_h, const CUtensorMap* w2_l, const CUtensorMap* o_h,
                       const CUtensorMap* o_l, const CUtensorMap* o_x, const CUtensorMap* t_h,
                       const CUtensorMap* t_l, const CUtensorMap* to_h, const CUtensorMap* to_l,
                       const FfnParams& p, cudaStream_t s) {
  if (p.rows <= 0) return cudaSuccess;
  if (!p.x0_row && (!p.x0 || p.ldx0 < p.d || p.ldx0 % 4)) return cudaErrorInvalidValue;
  if (p.tail_n > 0 && (!t_h || !to_h || (!p.tail_f16 && !to_l) ||
                       !ffn_tail_supported(p.d, p.d_pad, p.F, p.nb, p.tail_n, p.tail_f16)))
    return cudaErrorInvalidValue;
  const FfnLayout LY = ffn_layout(p.d, p.d_pad, p.F, p.nb);
  const long long tiles = (p.rows + BM - 1) / BM;
  long long grid = g_ffn_sms > 0 ? g_ffn_sms : 148;
  if (grid > tiles) grid = tiles;
  auto kern = p.d_pad > BK ? (p.nb > 1 ? ffn_kernel<2, 2> : ffn_kernel<2, 1>)
                           : (p.nb > 1 ? ffn_kernel<1, 2> : ffn_kernel<1, 1>);
  // without a tail its maps are never read: any valid descriptor stands in
  const CUtensorMap* th = p.tail_n > 0 ? t_h : o_h;
  const CUtensorMap* tl = p.tail_n > 0 && p.nb > 1 ? t_l : th;
  const CUtensorMap* toh = p.tail_n > 0 ? to_h : o_h;
  const CUtensorMap* tol = p.tail_n > 0 && !p.tail_f16 ? to_l : toh;
  return launch_k(kern, dim3((unsigned)grid), dim3(kThreads), LY.smem, s, *a_h, *a_l, *wo_h,
                  p.nb > 1 ? *wo_l : *wo_h, *w1_h, p.nb > 1 ? *w1_l : *w1_h, *w2_h, p.nb > 1 ? *w2_l : *w2_h, *o_h,
                  *o_l, *o_x, *th, *tl, *toh, *tol, p);
}

}  // namespace fe
