// Attention output projection and position-wise FFN of one block (the element
// layers of Section 4.2, the SeqEnc block of Section 4.3) for rows of width
// d = 256, in one kernel:
//     x = x0 + A W_O,   x_out = x + ReLU(LN(x) W1 + b1) W2 + b2,   LN(x_out),
// and optionally the next layer's query projection LN(x_out) W_Q (f16 out).
// x, LN(x) and the F-wide hidden activation never reach memory.
//
// At d = 256 the split LN(x) operand of a 128-row tile alone is 128 KB of
// shared memory, so every weight streams through a ring of five 16 KB boxes
// (128 rows x 64 columns, 128-byte swizzle) in the order the MMAs consume
// them, and every product is a sequence of N = 128 MMAs of one box each:
//   W_O  : k block kb, output half nh                       (8 boxes)
//   FFN1 : chunk f of 128 hidden units, k block kb          (4 boxes)
//   FFN2 : chunk f, output half nh, 64-unit half of the chunk (4 boxes)
//   W_Q  : as W_O (the tail)                                  (8 boxes)
// TMEM: columns [0, 256) take A W_O, then the two FFN1 chunk buffers
// (128 columns each), then the tail product; the d-column accumulator of x
// and FFN2 sits at [256, 512).  FFN1 of chunk f runs one chunk ahead of FFN2
// of chunk f - 1, which reads its A operand (the split ReLU output) from TMEM.
// Roles: warp 0 lane 0 loads (TMA), warp 1 lane 0 issues tcgen05.mma, warps
// 2-9 (two per TMEM lane quadrant, each owning 128 of a row's 256 columns)
// run the epilogues: x0 + projection, LayerNorm statistics exchanged with the
// partner warp, LN(x) as the split operand tile over the A tile, bias + ReLU
// + split per chunk, x_out + b2 (staged over the A tile and stored by TMA),
// LN(x_out) over the A tile (stored by TMA), and the tail's f16 output (over
// the A tile, stored by TMA).  Products take split bf16 activations
// (hi + lo) times exact bf16 weights with fp32 accumulation; LayerNorm and
// residuals are fp32.
#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {
// TMA 2D load with an L2 cache policy (createpolicy): evict_last for the weight
// boxes that every SM re-reads, evict_first for the activation tiles that
// stream past them once.
__device__ __forceinline__ void tma_load_2d_hint(void* smem_dst, const CUtensorMap* map, int x, int y,
                                                 uint64_t* bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "l"(policy)
      : "memory");
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int D = 256;
constexpr int NKB = D / BK;   // 4
constexpr int FC = 128;       // hidden units per chunk
constexpr int kEpiWarps = 8;
constexpr int kThreads = 64 + 32 * kEpiWarps;  // 320
constexpr uint32_t kBox = BM * BK * 2;         // 16 KB
constexpr uint32_t kABytes = NKB * 2 * kBox;   // 128 KB: the split tile [kb][plane]
constexpr int kMaxF = 2048;
constexpr int kRing = 5;
constexpr uint32_t kOffMisc = kABytes + kRing * kBox;
// misc: b1 [kMaxF], b2 [D], the broadcast x0 row [D], row statistics
// [sum|var][half][row], barriers, TMEM slot
constexpr uint32_t kMiscB1 = 0;
constexpr uint32_t kMiscB2 = kMiscB1 + kMaxF * 4;
constexpr uint32_t kMiscX0 = kMiscB2 + D * 4;
constexpr uint32_t kMiscRed = kMiscX0 + D * 4;
constexpr uint32_t kMiscBars = kMiscRed + 2 * 2 * 128 * 4;
constexpr uint32_t kMiscBytes = kMiscBars + 32 * 8 + 16;
constexpr size_t kSmem = 1024 + kOffMisc + kMiscBytes;
static_assert(kSmem <= 232448, "shared memory budget");

__device__ __forceinline__ float relu_nan256(float x) {
  float r;
  asm("max.NaN.f32 %0, %1, 0f00000000;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ void arrive_one(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// dst (+)= (k block of the split A tile: hi plane at sa, lo plane at sa + 16 KB)
// . (weight box at w)^T, M = N = 128, K = 64: eight products.
__device__ __noinline__ void mma_box(uint32_t dst, uint32_t sa, uint32_t w, uint32_t idesc, bool acc) {
  const uint64_t a0 = umma_desc_sw128(sa);
  const uint64_t w0 = umma_desc_sw128(w);
#pragma unroll
  for (int kk = 0; kk < BK / 16; ++kk) {
    const uint64_t ah = desc_adv(a0, kk * 32);
    const uint64_t wh = desc_adv(w0, kk * 32);
    umma_bf16(dst, ah, wh, idesc, (acc || kk != 0) ? 1u : 0u);
    umma_bf16(dst, desc_adv(ah, kBox), wh, idesc, 1u);
  }
}

// Row r, columns c .. c + 31 (c a multiple of 32) as a split bf16 pair into
// the A tile [kb][plane] (128-byte swizzle).
__device__ __forceinline__ void store_split_cols(uint8_t* sA, int r, int c, const float* v) {
  uint32_t hi[16], lo[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) split2(v[2 * j], v[2 * j + 1], hi[j], lo[j]);
  uint8_t* rowp = sA + (size_t)((c >> 6) * 2) * kBox + (size_t)r * 128u;
  const int u0 = (c & 63) >> 3;
#pragma unroll
  for (int jj = 0; jj < 4; ++jj) {
    const uint32_t o = (uint32_t)((u0 + jj) ^ (r & 7)) << 4;
    *reinterpret_cast<uint4*>(rowp + o) = make_uint4(hi[4 * jj], hi[4 * jj + 1], hi[4 * jj + 2], hi[4 * jj + 3]);
    *reinterpret_cast<uint4*>(rowp + kBox + o) = make_uint4(lo[4 * jj], lo[4 * jj + 1], lo[4 * jj + 2], lo[4 * jj + 3]);
  }
}
}  // namespace

__global__ void __launch_bounds__(kThreads, 1)
    ffn256_kernel(const __grid_constant__ CUtensorMap tA_h, const __grid_constant__ CUtensorMap tA_l,
                  const __grid_constant__ CUtensorMap tWO, const __grid_constant__ CUtensorMap tW1,
                  const __grid_constant__ CUtensorMap tW2, const __grid_constant__ CUtensorMap tT,
                  const __grid_constant__ CUtensorMap tO_h, const __grid_constant__ CUtensorMap tO_l,
                  const __grid_constant__ CUtensorMap tX, const __grid_constant__ CUtensorMap tQ,
                  const Ffn256Params p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  uint8_t* sA = smem;              // the A tile, then LN(x), then LN(x_out) [kb][plane]
  uint8_t* sR = smem + kABytes;    // weight ring [kRing][16 KB]
  uint8_t* misc = smem + kOffMisc;
  float* sB1 = reinterpret_cast<float*>(misc + kMiscB1);
  float* sB2 = reinterpret_cast<float*>(misc + kMiscB2);
  float* sX0 = reinterpret_cast<float*>(misc + kMiscX0);
  float* red = reinterpret_cast<float*>(misc + kMiscRed);
  uint64_t* bars = reinterpret_cast<uint64_t*>(misc + kMiscBars);
  uint64_t* w_full = bars;           // [kRing]
  uint64_t* w_empty = bars + 5;      // [kRing]
  uint64_t* a_full = bars + 10;      // A tile loaded
  uint64_t* a_free = bars + 11;      // sA free for the next tile (LN(x_out) stored and read by the tail)
  uint64_t* o_done = bars + 12;      // A W_O complete
  uint64_t* ln_full = bars + 13;     // x in the accumulator, LN(x) in sA
  uint64_t* acc1_full = bars + 14;   // [2]
  uint64_t* acc1_empty = bars + 16;  // [2]
  uint64_t* mid_full = bars + 18;    // [2]
  uint64_t* acc2_full = bars + 20;   // FFN2 of the tile complete
  uint64_t* tail_a = bars + 21;      // LN(x_out) in sA
  uint64_t* tail_full = bars + 22;   // the tail product complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 24);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int F = p.F, nf = F / FC;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kRing; ++i) {
      mbar_init(w_full + i, 1);
      mbar_init(w_empty + i, 1);
    }
    mbar_init(a_full, 1);
    mbar_init(a_free, kEpiWarps);
    mbar_init(o_done, 1);
    mbar_init(ln_full, kEpiWarps);
    for (int i = 0; i < 2; ++i) {
      mbar_init(acc1_full + i, 1);
      mbar_init(acc1_empty + i, 1);
      mbar_init(mid_full + i, kEpiWarps);
    }
    mbar_init(acc2_full, 1);
    mbar_init(tail_a, kEpiWarps);
    mbar_init(tail_full, 1);
    fence_mbar_init();
    prefetch_tmap(&tA_h);
    prefetch_tmap(&tWO);
    prefetch_tmap(&tW1);
    prefetch_tmap(&tW2);
  }
  // biases and the broadcast row are parameters: read before the dependency wait
  for (int i = threadIdx.x; i < F; i += kThreads) sB1[i] = p.b1[i];
  for (int i = threadIdx.x; i < D; i += kThreads) {
    sB2[i] = p.b2[i];
    sX0[i] = p.x0_row ? p.x0_row[i] : 0.f;
  }
  if (warp == 0) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t acc2 = tmem + 256u;
  pdl_trigger();
  pdl_wait();
  int rows_valid = p.rows;
  if (p.rows_dev) rows_valid = min(*p.rows_dev, p.rows);
  const int tiles = (rows_valid + BM - 1) / BM;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int ws = 0, tl = 0;
      bool ok = true;
      // every CTA re-reads the same weight boxes while the activation tiles
      // stream past once: keep the weights in L2, let the activations go first
      const uint64_t keep = l2_policy_evict_last(), pass = l2_policy_evict_first();
      auto load = [&](const CUtensorMap* m, int x, int y) -> bool {
        const int slot = ws % kRing;
        if (ws >= kRing && !mbar_wait_compact(w_empty + slot, ((ws / kRing) - 1) & 1, p.status)) return false;
        mbar_arrive_expect_tx(w_full + slot, kBox);
        tma_load_2d_hint(sR + (size_t)slot * kBox, m, x, y, w_full + slot, keep);
        ++ws;
        return true;
      };
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        // W_O boxes (kb, nh) in the MMA's order; the first four may load while
        // the previous tile still uses sA
        for (int i = 0; i < 2 * NKB && ok; ++i) {
          if (i == kRing - 1) {
            if (tl > 0 && !mbar_wait_compact(a_free, (tl - 1) & 1, p.status)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(a_full, kABytes);
            for (int kb = 0; kb < NKB; ++kb) {
              tma_load_2d_hint(sA + (size_t)(kb * 2) * kBox, &tA_h, kb * BK, t * BM, a_full, pass);
              tma_load_2d_hint(sA + (size_t)(kb * 2 + 1) * kBox, &tA_l, kb * BK, t * BM, a_full, pass);
            }
          }
          if (!load(&tWO, (i >> 1) * BK, (i & 1) * 128)) ok = false;
        }
        for (int s = 0; s <= nf && ok; ++s) {
          if (s < nf)
            for (int kb = 0; kb < NKB && ok; ++kb)
              if (!load(&tW1, kb * BK, s * FC)) ok = false;
          if (s >= 1)
            for (int i = 0; i < 4 && ok; ++i)  // (nh, sub): sub fastest
              if (!load(&tW2, (s - 1) * FC + (i & 1) * BK, (i >> 1) * 128)) ok = false;
        }
        if (p.tail)
          for (int i = 0; i < 2 * NKB && ok; ++i)
            if (!load(&tT, (i >> 1) * BK, (i & 1) * 128)) ok = false;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc = umma_idesc_bf16(BM, 128);
      int ws = 0, tl = 0, gf = 0;
      bool ok = true;
      auto wait = [&](uint64_t* bar, uint32_t par) -> bool {
        if (!mbar_wait_compact(bar, par, p.status)) ok = false;
        return ok;
      };
      // the next weight box landed: its shared-memory address (0 on a timeout)
      auto next_box = [&]() -> uint32_t {
        const int slot = ws % kRing;
        if (!wait(w_full + slot, (ws / kRing) & 1)) return 0u;
        tc_fence_after();
        return smem_u32(sR + (size_t)slot * kBox);
      };
      // the box's slot frees once the products issued so far complete
      auto release = [&]() {
        umma_commit(w_empty + ws % kRing);
        ++ws;
      };
      // [0, 256) = LN-free product of the A tile in sA with a 256 x 256 weight
      // (W_O or W_Q), box by box: k block kb, output half nh
      auto mma_256 = [&]() -> bool {
        for (int i = 0; i < 2 * NKB; ++i) {
          const uint32_t w = next_box();
          if (!w) return false;
          const int kb = i >> 1, nh = i & 1;
          mma_box(tmem + (uint32_t)(nh * 128), smem_u32(sA) + (uint32_t)(kb * 2) * kBox, w, idesc, kb != 0);
          release();
        }
        return true;
      };
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        // ---- A W_O into [0, 256)
        if (!wait(a_full, tl & 1)) break;
        tc_fence_after();
        if (!mma_256()) break;
        umma_commit(o_done);
        // ---- FFN1 chunk s one chunk ahead of FFN2 chunk s - 1
        if (!wait(ln_full, tl & 1)) break;
        tc_fence_after();
        const int gf0 = gf;
        for (int s = 0; s <= nf && ok; ++s) {
          if (s < nf) {
            const int g = gf0 + s, b = g & 1;
            if (g >= 2 && !wait(acc1_empty + b, ((g >> 1) - 1) & 1)) break;
            tc_fence_after();
            for (int kb = 0; kb < NKB; ++kb) {
              const uint32_t w = next_box();
              if (!w) break;
              mma_box(tmem + (uint32_t)(b * FC), smem_u32(sA) + (uint32_t)(kb * 2) * kBox, w, idesc, kb != 0);
              release();
            }
            if (!ok) break;
            umma_commit(acc1_full + b);
          }
          if (s >= 1) {
            const int c = s - 1, g = gf0 + c, b = g & 1;
            if (!wait(mid_full + b, (g >> 1) & 1)) break;
            tc_fence_after();
            // each 32-column piece of the buffer: 32 hidden units as the hi plane
            // (16 columns of bf16 pairs) then the lo plane
            const uint32_t mt = tmem + (uint32_t)(b * FC);
            for (int i = 0; i < 4; ++i) {
              const int nh = i >> 1, sub = i & 1;
              const uint32_t w = next_box();
              if (!w) break;
              const uint64_t w0 = umma_desc_sw128(w);
#pragma unroll
              for (int k4 = 0; k4 < 4; ++k4) {
                const int kk = 4 * sub + k4;
                const uint32_t mh = mt + (uint32_t)(32 * (kk >> 1) + 8 * (kk & 1)), ml = mh + 16;
                const uint64_t wh = desc_adv(w0, (uint32_t)k4 * 32);
                umma_bf16_tmem_a(acc2 + (uint32_t)(nh * 128), mh, wh, idesc, 1u);
                umma_bf16_tmem_a(acc2 + (uint32_t)(nh * 128), ml, wh, idesc, 1u);
              }
              release();
            }
            if (!ok) break;
            umma_commit(acc1_empty + b);
            if (c == nf - 1) umma_commit(acc2_full);
          }
        }
        if (!ok) break;
        gf = gf0 + nf;
        // ---- the tail LN(x_out) W_Q into [0, 256)
        if (p.tail) {
          if (!wait(tail_a, tl & 1)) break;
          tc_fence_after();
          if (!mma_256()) break;
          umma_commit(tail_full);
        }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..9) ----------------
    // two warps per TMEM lane quadrant q; warp half hf owns columns
    // [128 hf, 128 hf + 128) of the row, as four 32-column pieces
    const int ew = warp - 2, q = warp & 3, hf = ew >> 2;
    const int et = threadIdx.x - 64;
    const int r = q * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const int c0 = 128 * hf;
    float* red_sum = red;        // [half][row]
    float* red_var = red + 256;  // [half][row]
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + q) : "memory"); };
    auto epi_sync = [&]() { asm volatile("bar.sync 5, %0;" ::"n"(32 * kEpiWarps) : "memory"); };
    auto warp_arrive = [&](uint64_t* bar) {
      __syncwarp();
      if (lane == 0) arrive_one(bar);
    };
    bool ok = true;
    auto wait = [&](uint64_t* bar, uint32_t par) -> bool {
      if (!mbar_wait_compact(bar, par, p.status)) ok = false;
      return ok;
    };
    // the row statistics over both halves: sum -> mean, then sum of squares -> rstd
    auto pair_mean = [&](float s) {
      red_sum[hf * 128 + r] = s;
      pair_sync();
      return (red_sum[r] + red_sum[128 + r]) * (1.f / (float)D);
    };
    auto pair_rstd = [&](float s) {
      red_var[hf * 128 + r] = s;
      pair_sync();
      return 1.0f / sqrtf((red_var[r] + red_var[128 + r]) * (1.f / (float)D) + p.eps);
    };
    int tl = 0, gf = 0;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
      const int m0 = t * BM;
      const bool valid = m0 + r < rows_valid;
      float* xrow = p.x + (size_t)(m0 + r) * p.ldx;
      // ---- x0 into the accumulator while the projection runs (x0 of rows past
      // the valid count is 0)
      for (int i = 0; i < 4; ++i) {
        const int c = c0 + 32 * i;
        float v[32];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
          if (p.x0_row)
            x = *reinterpret_cast<const float4*>(sX0 + c + 4 * j);
          else if (valid)
            x = *reinterpret_cast<const float4*>(xrow + c + 4 * j);
          v[4 * j] = x.x;
          v[4 * j + 1] = x.y;
          v[4 * j + 2] = x.z;
          v[4 * j + 3] = x.w;
        }
        tmem_st32(acc2 + lane_off + (uint32_t)c, v);
      }
      // ---- x = x0 + A W_O back into the accumulator, LN(x) over the A tile
      // (the projection, the tile's only reader, is complete)
      if (!wait(o_done, tl & 1)) break;
      tc_fence_after();
      float s4[4] = {0.f, 0.f, 0.f, 0.f};
      for (int i = 0; i < 4; ++i) {
        const int c = c0 + 32 * i;
        float v[32], w[32];
        tmem_ld32(tmem + lane_off + (uint32_t)c, v);
        tmem_ld32(acc2 + lane_off + (uint32_t)c, w);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          v[j] += w[j];
          s4[j & 3] += v[j];
        }
        tmem_st32(acc2 + lane_off + (uint32_t)c, v);
      }
      const float mean0 = pair_mean((s4[0] + s4[1]) + (s4[2] + s4[3]));
#pragma unroll
      for (int k = 0; k < 4; ++k) s4[k] = 0.f;
      for (int i = 0; i < 4; ++i) {
        float v[32];
        tmem_ld32(acc2 + lane_off + (uint32_t)(c0 + 32 * i), v);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float dv = v[j] - mean0;
          s4[j & 3] = fmaf(dv, dv, s4[j & 3]);
        }
      }
      const float rstd0 = pair_rstd((s4[0] + s4[1]) + (s4[2] + s4[3]));
      for (int i = 0; i < 4; ++i) {
        const int c = c0 + 32 * i;
        float v[32];
        tmem_ld32(acc2 + lane_off + (uint32_t)c, v);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = (v[j] - mean0) * rstd0;
        store_split_cols(sA, r, c, v);
      }
      fence_async_shared();
      tc_fence_before();
      warp_arrive(ln_full);
      // ---- per chunk: split(ReLU(acc1 + b1)) over this thread's 64 columns of
      // the chunk's TMEM buffer, FFN2's A operand
      for (int f = 0; f < nf; ++f, ++gf) {
        const int ba = gf & 1;
        if (!wait(acc1_full + ba, (gf >> 1) & 1)) break;
        tc_fence_after();
        for (int jp = 0; jp < 2; ++jp) {
          const uint32_t col = tmem + lane_off + (uint32_t)(ba * FC + 64 * hf + 32 * jp);
          const float* bias = sB1 + f * FC + 64 * hf + 32 * jp;
          float v[32];
          tmem_ld32(col, v);
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float2 bb = *reinterpret_cast<const float2*>(bias + 2 * j);
            split2_trunc(relu_nan256(v[2 * j] + bb.x), relu_nan256(v[2 * j + 1] + bb.y), hi[j], lo[j]);
          }
          tmem_st16_nowait(col, hi);
          tmem_st16_nowait(col + 16u, lo);
        }
        tmem_st_wait();
        tc_fence_before();
        warp_arrive(mid_full + ba);
      }
      if (!ok) break;
      // ---- x_out = acc2 + b2 to memory, staged in this warp's 16 KB of sA (every
      // FFN1 has read LN(x) there) as four 32 x 32 blocks (128-byte swizzle)
      // and stored by TMA; then LN(x_out) over the A tile
      if (!wait(acc2_full, tl & 1)) break;
      tc_fence_after();
      uint8_t* xst = sA + (size_t)ew * 16384u;
#pragma unroll
      for (int k = 0; k < 4; ++k) s4[k] = 0.f;
      for (int i = 0; i < 4; ++i) {
        const int c = c0 + 32 * i;
        float v[32];
        tmem_ld32(acc2 + lane_off + (uint32_t)c, v);
        uint8_t* blk = xst + (size_t)i * 4096u + (uint32_t)lane * 128u;
#pragma unroll
        for (int j = 0; j < 32; j += 4) {
          const float4 bb = *reinterpret_cast<const float4*>(sB2 + c + j);
          v[j] += bb.x;
          v[j + 1] += bb.y;
          v[j + 2] += bb.z;
          v[j + 3] += bb.w;
          s4[0] += v[j];
          s4[1] += v[j + 1];
          s4[2] += v[j + 2];
          s4[3] += v[j + 3];
          *reinterpret_cast<float4*>(blk + ((uint32_t)((j >> 2) ^ (lane & 7)) << 4)) =
              make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
        }
      }
      fence_async_shared();
      __syncwarp();
      if (lane == 0) {
        for (int i = 0; i < 4; ++i) tma_store_2d(&tX, xst + (size_t)i * 4096u, c0 + 32 * i, m0 + 32 * q);
        bulk_commit();
      }
      const float mean = pair_mean((s4[0] + s4[1]) + (s4[2] + s4[3]));
#pragma unroll
      for (int k = 0; k < 4; ++k) s4[k] = 0.f;
      for (int i = 0; i < 4; ++i) {
        const int c = c0 + 32 * i;
        float v[32];
        tmem_ld32(acc2 + lane_off + (uint32_t)c, v);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float dv = v[j] + sB2[c + j] - mean;
          s4[j & 3] = fmaf(dv, dv, s4[j & 3]);
        }
      }
      const float rstd = pair_rstd((s4[0] + s4[1]) + (s4[2] + s4[3]));
      if (lane == 0) bulk_wait_read0();
      epi_sync();  // every warp's x_out staging read: sA takes LN(x_out)
      for (int i = 0; i < 4; ++i) {
        const int c = c0 + 32 * i;
        float v[32];
        tmem_ld32(acc2 + lane_off + (uint32_t)c, v);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = (v[j] + sB2[c + j] - mean) * rstd;
        store_split_cols(sA, r, c, v);
      }
      fence_async_shared();
      tc_fence_before();
      if (p.tail) warp_arrive(tail_a);
      if (p.store_ln) {
        epi_sync();  // every row of the tile written
        if (et == 0) {
          for (int kb = 0; kb < NKB; ++kb) {
            tma_store_2d(&tO_h, sA + (size_t)(kb * 2) * kBox, kb * BK, m0);
            tma_store_2d(&tO_l, sA + (size_t)(kb * 2 + 1) * kBox, kb * BK, m0);
          }
          bulk_commit();
        }
      }
      // ---- the tail: Q = LN(x_out) W_Q as f16 over sA (the tail product has read
      // LN(x_out)): this thread's 128 columns of row r as 128-byte-swizzled
      // [kb][128 rows x 64] tiles, stored by TMA
      if (p.tail) {
        if (!wait(tail_full, tl & 1)) break;
        tc_fence_after();
        for (int i = 0; i < 4; ++i) {
          const int c = c0 + 32 * i;
          float v[32];
          tmem_ld32(tmem + lane_off + (uint32_t)c, v);
          uint8_t* rowp = sA + (size_t)(c >> 6) * kBox + (size_t)r * 128u;
          const int u0 = (c & 63) >> 3;
#pragma unroll
          for (int j = 0; j < 4; ++j)
            *reinterpret_cast<uint4*>(rowp + ((uint32_t)((u0 + j) ^ (r & 7)) << 4)) =
                make_uint4(pack_f16x2(v[8 * j], v[8 * j + 1]), pack_f16x2(v[8 * j + 2], v[8 * j + 3]),
                           pack_f16x2(v[8 * j + 4], v[8 * j + 5]), pack_f16x2(v[8 * j + 6], v[8 * j + 7]));
        }
        tc_fence_before();
        fence_async_shared();
        epi_sync();  // every row of Q written
        if (et == 0) {
          for (int kb = 0; kb < NKB; ++kb) tma_store_2d(&tQ, sA + (size_t)kb * kBox, kb * BK, m0);
          bulk_commit();
        }
      }
      // ---- sA and the TMEM columns [0, 256) may take the next tile once the
      // stores have read sA
      if (et == 0) bulk_wait_read0();
      epi_sync();
      warp_arrive(a_free);
    }
    if (et == 0) bulk_wait0();  // output tensor stores complete before the CTA retires
  }

  __syncwarp();  // each warp arrives whole: lane 0 of warps 0 and 1 ran the producer and MMA loops
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

namespace {
int g_ffn256_sms = 0;
}

bool ffn256_supported(int d, int F, int nb) { return d == D && nb == 1 && F % FC == 0 && F >= FC && F <= kMaxF; }

cudaError_t ffn256_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_ffn256_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(ffn256_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
  return e;
}

cudaError_t ffn256_launch(const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* wo, const CUtensorMap* w1,
                          const CUtensorMap* w2, const CUtensorMap* wt, const CUtensorMap* o_h, const CUtensorMap* o_l,
                          const CUtensorMap* x_st, const CUtensorMap* q_st, const Ffn256Params& p, cudaStream_t s) {
  if (p.rows <= 0) return cudaSuccess;
  if (!ffn256_supported(D, p.F, 1) || !x_st || (p.tail && !wt) || (p.tail && !q_st)) return cudaErrorInvalidValue;
  const long long tiles = (p.rows + BM - 1) / BM;
  long long grid = g_ffn256_sms > 0 ? g_ffn256_sms : 148;
  if (grid > tiles) grid = tiles;
  return launch_k(ffn256_kernel, dim3((unsigned)grid), dim3(kThreads), kSmem, s, *a_h, *a_l, *wo, *w1, *w2,
                  p.tail ? *wt : *wo, *o_h, *o_l, *x_st, p.tail ? *q_st : *o_h, p);
}

}  // namespace fe
