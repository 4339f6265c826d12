// tcgen05 GEMM of the joint evaluator with fused epilogues.
//
// Every dense product of the model (context K/V projection and element
// WQ / WO / FFN of Section 4.2, SeqEnc and cross-sequence projections of
// Sections 4.3-4.4, the score head) is  act[rows, K] x W[K, N]  with a small
// K (d or F).  The kernel is persistent and warp-specialised; each CTA walks
// 128-row x BN-column tiles (column tile fastest, so concurrently running CTAs
// share activation rows in L2):
//   warp 0 lane 0  : TMA producer, a ring of shared-memory stages that runs
//                    ahead across tile boundaries
//   warp 1 lane 0  : tcgen05.mma issuer into one of two TMEM accumulators
//   warps 2-9      : epilogue of the previous tile while the next one is
//                    multiplied; warps w and w+4 share TMEM lane quadrant
//                    w % 4 (tile rows (w % 4) * 32 + lane) and take
//                    alternate 32-column chunks
// The activation is a split pair (hi + lo bf16); the product is
// A_hi W_hi + A_lo W_hi (+ A_hi W_lo when the weights carry a lo plane).
#include <cstdlib>

#include "fe_common.cuh"
#include "fe_kernels.h"
#include "fe_select.cuh"

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
constexpr int BK = 64;                               // one 128-byte swizzle row of bf16
constexpr uint32_t kATile = BM * BK * 2;             // 16 KB per activation plane
constexpr size_t kSmemPerSM = 233472;                // 228 KB
constexpr size_t kSmemMaxBlock = 232448;             // 227 KB opt-in per block
constexpr int kEpiWarps = 8;                         // two per TMEM lane quadrant, alternating 32-column chunks
constexpr uint32_t kStageOut = 4096;                 // one staging buffer: 32 rows x 128 B
constexpr uint32_t kRedBytes = 4 * 2 * 128 * 4;      // row-reduction exchange: [parity][sum|var][half][128]
// alignment slack, barriers, staging; then the row-reduction area (red_bytes)
constexpr size_t kSmemFixed = 1024 + 256 + 1024 + kEpiWarps * 2 * kStageOut;
constexpr int kThreads = 64 + 32 * kEpiWarps;
constexpr int kMaxStages = 8;

int g_num_sms = 0;

__host__ __device__ inline uint32_t pow2_cols(int n) {
  return n <= 32 ? 32u : n <= 64 ? 64u : n <= 128 ? 128u : n <= 256 ? 256u : 512u;
}

// Row-reduction area: the pair exchange within a CTA, or with clusters of cs > 1
// the partial row sums of every CTA of the cluster, [sum|var][cs][half][128].
__host__ __device__ inline uint32_t red_bytes(int cs) { return cs > 1 ? (uint32_t)cs * 2048u : kRedBytes; }
constexpr int kMaxCluster = 8;
int g_cluster_cap[2][kMaxCluster + 1] = {};  // resident clusters of size cs with one / two CTAs per SM
int g_cluster_limit = -1;                 // FE_GEMM_CLUSTERS: 0 disables clusters, n > 0 caps clusters per launch
bool g_two_per_sm[4][2] = {};             // [EPI][NB - 1]: two CTAs fit on an SM (registers) at half the shared memory
}  // namespace

size_t gemm_smem_bytes(int BN, int nb, int stages, int cs, int na) {
  const size_t stage = (size_t)na * kATile + (size_t)nb * BN * BK * 2;
  return (size_t)stages * stage + kSmemFixed + red_bytes(cs);
}

int gemm_max_stages(int BN, int nb, int K_pad, int cs, int na) {
  (void)K_pad;  // stages run ahead across tiles, so the ring is not capped by one tile's k blocks
  const size_t stage = (size_t)na * kATile + (size_t)nb * BN * BK * 2;
  int s = (int)((kSmemMaxBlock - kSmemFixed - red_bytes(cs)) / stage);
  if (s > kMaxStages) s = kMaxStages;
  return s < 1 ? 1 : s;
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// ---- thread-block cluster helpers (the RESID_LN row exchange) ----
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// every thread of every CTA of the cluster; orders the barrier initialisation
// before any remote access, and keeps each CTA's shared memory alive until the
// cluster's last remote store to it
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t map_peer(uint32_t local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}
// 4-byte store into a peer CTA's shared memory, counted on the peer's mbarrier
__device__ __forceinline__ void st_async_peer(uint32_t addr, float v, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(addr),
               "r"(__float_as_uint(v)), "r"(bar)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded like mbar_wait_bounded, acquiring at cluster scope (the peers' stores)
__device__ __noinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, int* status) {
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((it & 255u) == 255u && (*reinterpret_cast<volatile int*>(status) & ST_TIMEOUT)) return false;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      atomicOr(status, ST_TIMEOUT);
      return false;
    }
  }
}

// NB: weight planes (1 when the weights are exact in bf16, else 2); a
// compile-time constant so that the MMA issue sequence has no branches
template <int EPI, int NB>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tA_h, const __grid_constant__ CUtensorMap tA_l,
                const __grid_constant__ CUtensorMap tB_h, const __grid_constant__ CUtensorMap tB_l,
                const __grid_constant__ CUtensorMap tO_h, const __grid_constant__ CUtensorMap tO_l,
                const __grid_constant__ CUtensorMap tO_x, const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);

  constexpr int nb = NB;
  const int BN = p.BN, S = p.stages;
  const int nacc = p.nacc;
  const int cs = p.cs > 1 ? p.cs : 1;  // (uniform) CTAs of a cluster sharing each row tile
  const uint32_t b_bytes = (uint32_t)BN * BK * 2;
  // activation planes: the split pair, or one exact bf16 plane (raw rows of EPI_LN_FOLD)
  constexpr int NA = EPI == EPI_LN_FOLD ? 1 : 2;
  const uint32_t stage_bytes = NA * kATile + (uint32_t)nb * b_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)S * stage_bytes);
  uint64_t* empty = full + S;
  uint64_t* tfull = empty + S;  // [2] accumulator ready for the epilogue
  uint64_t* tempty = tfull + 2; // [2] accumulator drained by the epilogue
  uint64_t* xbar = tempty + 2;  // [2] cluster row exchange: partial sums / partial variances received
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(xbar + 2);
  // output staging: two 4 KB buffers per epilogue warp, 1024-byte aligned; then
  // the row-reduction exchange of the two warps sharing a lane quadrant
  uint8_t* stg_base = smem + (((size_t)S * stage_bytes + 256 + 1023) & ~(size_t)1023);
  float* red = reinterpret_cast<float*>(stg_base + (size_t)kEpiWarps * 2 * kStageOut);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // set-up needs nothing from earlier kernels, so it runs before the
  // programmatic wait and overlaps the tail of the previous kernel
  const uint32_t ncols = pow2_cols(nacc * BN);
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull + a, 1);
      mbar_init(tempty + a, kEpiWarps);  // one arrival per epilogue warp
    }
    if (cs > 1) {
      mbar_init(xbar, 1);  // the local expect_tx; the peers' stores complete the bytes
      mbar_init(xbar + 1, 1);
    }
    fence_mbar_init();
    prefetch_tmap(&tA_h);
    prefetch_tmap(&tA_l);
    prefetch_tmap(&tB_h);
    if (nb > 1) prefetch_tmap(&tB_l);
  }
  if (warp == 0) tmem_alloc(tmem_slot, ncols);
  tc_fence_before();
  __syncthreads();
  if (cs > 1) cluster_sync_all();  // the peers' barriers exist before any store to them
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int nk = p.K_pad / BK;
  pdl_trigger();
  pdl_wait();
  int rows_valid = p.rows;
  if (p.rows_dev) rows_valid = min(*p.rows_dev, p.rows);
  // With clusters nt == cs and the grid is a multiple of cs: CTA rank k of a
  // cluster always takes column tile k, and the cluster's CTAs walk the same
  // row tiles in the same order (and leave together below).
  const int nt = p.N / BN;
  const int tiles = ((rows_valid + BM - 1) / BM) * nt;
  if ((int)blockIdx.x >= tiles) {  // nothing for this CTA (uniform)
    if (warp == 0) tmem_dealloc(tmem, ncols);
    if (EPI == EPI_HEAD && p.sel.keys) sel_ticket(p.sel, tmem_slot);  // (the slot is free once deallocated)
    return;
  }

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        const int m0 = (t / nt) * BM, n0 = (t % nt) * BN;
        for (int kb = 0; kb < nk; ++kb, ++it) {
          const int s = it % S;
          if (it >= S && !mbar_wait_bounded(empty + s, ((it / S) & 1) ^ 1, p.status)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + (size_t)s * stage_bytes;
          mbar_arrive_expect_tx(full + s, stage_bytes);
          tma_load_2d(st, &tA_h, kb * BK, m0, full + s);
          if (NA > 1) tma_load_2d(st + kATile, &tA_l, kb * BK, m0, full + s);
          for (int q = 0; q < nb; ++q) {
            const CUtensorMap* tb = q ? &tB_l : &tB_h;
            for (int h = 0; h < BN; h += 256)
              tma_load_2d(st + NA * kATile + q * b_bytes + (uint32_t)h * BK * 2, tb, kb * BK, n0 + h, full + s);
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const int nmma = BN > 256 ? 256 : BN;
      const uint32_t idesc = umma_idesc_bf16(BM, nmma);
      int it = 0, tl = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tl) {
        const int acc = tl % nacc, use = tl / nacc;
        if (use > 0 && !mbar_wait_bounded(tempty + acc, (use - 1) & 1, p.status)) break;
        tc_fence_after();
        const uint32_t dst = tmem + (uint32_t)(acc * BN);
        for (int kb = 0; kb < nk; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait_bounded(full + s, (it / S) & 1, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_u32(smem + (size_t)s * stage_bytes);
          // descriptors built once per stage; the k steps only add 32-byte offsets
          const uint64_t ah0 = umma_desc_sw128(st), al0 = umma_desc_sw128(st + kATile);
          const uint64_t bh0 = umma_desc_sw128(st + NA * kATile), bl0 = umma_desc_sw128(st + NA * kATile + b_bytes);
          for (int h = 0; h < BN; h += 256) {
            const uint32_t hb = (uint32_t)h * BK * 2;
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
              // (A_hi, W_hi), (A_lo, W_hi), (A_hi, W_lo)
              const uint64_t ah = desc_adv(ah0, kk * 32), al = desc_adv(al0, kk * 32);
              const uint64_t bh = desc_adv(bh0, hb + kk * 32);
              umma_bf16(dst + (uint32_t)h, ah, bh, idesc, (kb | kk) != 0 ? 1u : 0u);
              if (NA > 1) umma_bf16(dst + (uint32_t)h, al, bh, idesc, 1u);
              if (nb > 1) umma_bf16(dst + (uint32_t)h, ah, desc_adv(bl0, hb + kk * 32), idesc, 1u);
            }
          }
          umma_commit(empty + s);  // frees this stage once its MMAs complete
        }
        umma_commit(tfull + acc);  // accumulator complete (or abandoned after a timeout)
      }
    }
  } else {
    // ---------------- epilogue (warps 2..9) ----------------
    const int ew = warp - 2;     // 0..7
    const int q = warp & 3;      // TMEM lane quadrant this warp may access
    const int half = ew >> 2;    // which alternate 32-column chunks
    const int r = q * 32 + lane;
    uint8_t* stg0 = stg_base + (size_t)ew * 2 * kStageOut;
    int nstore = 0;              // bulk-store groups issued by this warp (selects the staging buffer)
    // the two warps of a lane quadrant meet at named barrier 1 + q (64 threads)
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + q) : "memory"); };
    // 32 rows x 32 columns of this warp leave through a staging buffer as TMA
    // tensor stores: bf16 planes with the 64-byte swizzle (2 KB each), fp32
    // rows with the 128-byte swizzle (4 KB); the TMA unit clips rows past the
    // tensor extent.  Two buffers alternate so one store drains while the
    // next chunk is written.
    auto next_stage = [&]() -> uint8_t* {
      uint8_t* b = stg0 + (size_t)(nstore & 1) * kStageOut;
      if (lane == 0 && nstore >= 2) asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
      __syncwarp();
      return b;
    };
    auto issue = [&](const CUtensorMap* m0p, const void* s0, const CUtensorMap* m1p, const void* s1, int col,
                     int row) {
      fence_async_shared();
      __syncwarp();
      if (lane == 0) {
        tma_store_2d(m0p, s0, col, row);
        if (m1p) tma_store_2d(m1p, s1, col, row);
        bulk_commit();
      }
      ++nstore;
    };
    auto stage_split = [&](const uint32_t* hi, const uint32_t* lo, int col, int row) {
      uint8_t* b = next_stage();
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t o = (uint32_t)lane * 64u + ((uint32_t)(j ^ ((lane >> 1) & 3)) << 4);
        *reinterpret_cast<uint4*>(b + o) = make_uint4(hi[4 * j], hi[4 * j + 1], hi[4 * j + 2], hi[4 * j + 3]);
        *reinterpret_cast<uint4*>(b + 2048 + o) = make_uint4(lo[4 * j], lo[4 * j + 1], lo[4 * j + 2], lo[4 * j + 3]);
      }
      issue(&tO_h, b, &tO_l, b + 2048, col, row);
    };

    // Clusters (EPI_RESID_LN, cs > 1): each CTA holds BN columns of the rows; the
    // row sums and then the sums of squared deviations of every warp are stored
    // into all cs CTAs' exchange areas ([cs][half][128] per kind) with st.async,
    // which counts the bytes on the receiver's xbar[kind]; one local thread
    // posts the expected cs * 1 KB.  Each CTA adds the 2 * cs partials of a row
    // in the same order, so the cluster's CTAs use identical statistics.  A
    // peer stores the next tile's partials of one kind only after it received
    // this CTA's partials of the other kind, which each warp sends after it read
    // the current ones, so one area per kind suffices.
    int tl = 0;
    const uint32_t my_rank = cs > 1 ? cluster_rank() : 0u;
    auto row_xchg = [&](int kind, float v, float& tot) -> bool {
      float* xs = red + (size_t)kind * cs * 256;
      const uint32_t slot = smem_u32(xs + (my_rank * 2 + half) * 128 + r);
      const uint32_t bar = smem_u32(xbar + kind);
      for (int k = 0; k < cs; ++k) st_async_peer(map_peer(slot, (uint32_t)k), v, map_peer(bar, (uint32_t)k));
      if (ew == 0 && lane == 0) mbar_arrive_expect_tx(xbar + kind, (uint32_t)cs * 1024u);
      if (!mbar_wait_cluster(xbar + kind, (uint32_t)tl & 1u, p.status)) return false;
      float a = 0.f;
      for (int k = 0; k < cs; ++k) a += xs[(2 * k) * 128 + r] + xs[(2 * k + 1) * 128 + r];
      tot = a;
      return true;
    };

    float xr[64];  // EPI_RESID_LN with BN <= 128: this warp's chunks of the row
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++tl) {
      const int acc = tl % nacc, use = tl / nacc;
      const int m0 = (t / nt) * BM, n0 = (t % nt) * BN;
      const int grow = m0 + r;
      const bool valid = grow < rows_valid;
      if (EPI == EPI_RESID_LN && BN <= 128) {
        // residual rows, loaded while the MMAs of this tile run
        const float* rrow = p.resid + (p.ldr ? (size_t)grow * p.ldr : (size_t)0);
#pragma unroll
        for (int ci = 0; ci < 2; ++ci) {
          const int c = 32 * half + 64 * ci;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            float4 qv = make_float4(0.f, 0.f, 0.f, 0.f);
            if (valid && c < BN) qv = reinterpret_cast<const float4*>(rrow + n0 + c)[j];
            xr[32 * ci + 4 * j] = qv.x;
            xr[32 * ci + 4 * j + 1] = qv.y;
            xr[32 * ci + 4 * j + 2] = qv.z;
            xr[32 * ci + 4 * j + 3] = qv.w;
          }
        }
      }
      if (!mbar_wait_bounded(tfull + acc, use & 1, p.status)) break;
      tc_fence_after();
      const int srow = m0 + q * 32;
      const uint32_t trow = tmem + (uint32_t)(acc * BN) + ((uint32_t)(q * 32) << 16);
      float* red_sum = red + (size_t)(tl & 1) * 512;  // [half][128]
      float* red_var = red_sum + 256;

      if (EPI == EPI_STORE) {
        for (int c = 32 * half; c < BN; c += 64) {
          float v[32];
          tmem_ld32(trow + (uint32_t)c, v);
          const int col = n0 + c;
          if (p.bias) {
            const float4* b4 = reinterpret_cast<const float4*>(p.bias + col);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 bb = __ldg(b4 + j);
              v[4 * j] += bb.x;
              v[4 * j + 1] += bb.y;
              v[4 * j + 2] += bb.z;
              v[4 * j + 3] += bb.w;
            }
          }
          if (p.relu) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = relu_nan(v[i]);
          }
          if (col < p.lq_n) {
            // a key chunk of SeqEnc: only its [CLS] logit partial leaves the SM
            const float4* q4 = reinterpret_cast<const float4*>(p.lq + col);
            float a = 0.f;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 qq = __ldg(q4 + j);
              a = fmaf(v[4 * j], qq.x, a);
              a = fmaf(v[4 * j + 1], qq.y, a);
              a = fmaf(v[4 * j + 2], qq.z, a);
              a = fmaf(v[4 * j + 3], qq.w, a);
            }
            if (valid) p.logits[(size_t)grow * p.ld_logit + (size_t)(col / 32)] = a;
            continue;
          }
          if (p.out_f16) {
            // one f16 plane (an attention operand)
            uint8_t* b = next_stage();
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint32_t o = (uint32_t)lane * 64u + ((uint32_t)(j ^ ((lane >> 1) & 3)) << 4);
              *reinterpret_cast<uint4*>(b + o) =
                  make_uint4(pack_f16x2(v[8 * j], v[8 * j + 1]), pack_f16x2(v[8 * j + 2], v[8 * j + 3]),
                             pack_f16x2(v[8 * j + 4], v[8 * j + 5]), pack_f16x2(v[8 * j + 6], v[8 * j + 7]));
            }
            issue(&tO_h, b, nullptr, nullptr, col, srow);
          } else {
            uint32_t hi[16], lo[16];
#pragma unroll
            for (int i = 0; i < 32; i += 2) split2(v[i], v[i + 1], hi[i / 2], lo[i / 2]);
            stage_split(hi, lo, col, srow);
          }
        }
      } else if (EPI == EPI_RESID_LN && BN <= 128) {
        // rows of at most 128 columns: each warp holds its (at most two) chunks of
        // x = resid + acc + bias in registers; the residual was loaded before the
        // accumulator was ready, TMEM is read once
        float sum = 0.f;
#pragma unroll
        for (int ci = 0; ci < 2; ++ci) {
          const int c = 32 * half + 64 * ci;
          if (c < BN) {
            float v[32];
            tmem_ld32(trow + (uint32_t)c, v);
#pragma unroll
            for (int i = 0; i < 32; ++i) xr[32 * ci + i] += v[i];
            if (p.bias) {
              const float4* b4 = reinterpret_cast<const float4*>(p.bias + n0 + c);
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                const float4 bb = __ldg(b4 + j);
                xr[32 * ci + 4 * j] += bb.x;
                xr[32 * ci + 4 * j + 1] += bb.y;
                xr[32 * ci + 4 * j + 2] += bb.z;
                xr[32 * ci + 4 * j + 3] += bb.w;
              }
            }
#pragma unroll
            for (int i = 0; i < 32; i += 4)
              sum += (xr[32 * ci + i] + xr[32 * ci + i + 1]) + (xr[32 * ci + i + 2] + xr[32 * ci + i + 3]);
            uint8_t* b = next_stage();
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const uint32_t o = (uint32_t)lane * 128u + ((uint32_t)(j ^ (lane & 7)) << 4);
              *reinterpret_cast<float4*>(b + o) =
                  make_float4(xr[32 * ci + 4 * j], xr[32 * ci + 4 * j + 1], xr[32 * ci + 4 * j + 2],
                              xr[32 * ci + 4 * j + 3]);
            }
            issue(&tO_x, b, nullptr, nullptr, n0 + c, srow);
          }
        }
        float mean, rstd, tot = 0.f;
        if (cs > 1) {
          if (!row_xchg(0, sum, tot)) break;
          mean = tot / (float)p.N;
        } else {
          red_sum[half * 128 + r] = sum;
          pair_sync();
          mean = (red_sum[r] + red_sum[128 + r]) / (float)BN;
        }
        float var = 0.f;
#pragma unroll
        for (int ci = 0; ci < 2; ++ci) {
          if (32 * half + 64 * ci < BN) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float dv = xr[32 * ci + i] - mean;
              var = fmaf(dv, dv, var);
            }
          }
        }
        if (cs > 1) {
          if (!row_xchg(1, var, tot)) break;
          rstd = 1.0f / sqrtf(tot / (float)p.N + p.eps);
        } else {
          red_var[half * 128 + r] = var;
          pair_sync();
          rstd = 1.0f / sqrtf((red_var[r] + red_var[128 + r]) / (float)BN + p.eps);
        }
#pragma unroll
        for (int ci = 0; ci < 2; ++ci) {
          const int c = 32 * half + 64 * ci;
          if (c < BN) {
            uint32_t hi[16], lo[16];
#pragma unroll
            for (int i = 0; i < 32; i += 2)
              split2((xr[32 * ci + i] - mean) * rstd, (xr[32 * ci + i + 1] - mean) * rstd, hi[i / 2], lo[i / 2]);
            stage_split(hi, lo, n0 + c, srow);
          }
        }
      } else if (EPI == EPI_RESID_LN) {
        // wider rows: x kept in TMEM between the passes
        float sum = 0.f;
        const float* rrow = p.resid + (p.ldr ? (size_t)grow * p.ldr : (size_t)0);
        for (int c = 32 * half; c < BN; c += 64) {
          float v[32];
          tmem_ld32(trow + (uint32_t)c, v);
          if (valid) {
            const float4* rr = reinterpret_cast<const float4*>(rrow + c);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 qv = rr[j];
              v[4 * j + 0] += qv.x;
              v[4 * j + 1] += qv.y;
              v[4 * j + 2] += qv.z;
              v[4 * j + 3] += qv.w;
            }
          }
          if (p.bias) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] += p.bias[c + i];
          }
#pragma unroll
          for (int i = 0; i < 32; i += 4) sum += (v[i] + v[i + 1]) + (v[i + 2] + v[i + 3]);
          tmem_st32(trow + (uint32_t)c, v);
          uint8_t* b = next_stage();
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const uint32_t o = (uint32_t)lane * 128u + ((uint32_t)(j ^ (lane & 7)) << 4);
            *reinterpret_cast<float4*>(b + o) = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
          }
          issue(&tO_x, b, nullptr, nullptr, c, srow);
        }
        red_sum[half * 128 + r] = sum;
        pair_sync();
        const float mean = (red_sum[r] + red_sum[128 + r]) / (float)BN;
        float var = 0.f;
        for (int c = 32 * half; c < BN; c += 64) {
          float v[32];
          tmem_ld32(trow + (uint32_t)c, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float dv = v[i] - mean;
            var = fmaf(dv, dv, var);
          }
        }
        red_var[half * 128 + r] = var;
        pair_sync();
        const float rstd = 1.0f / sqrtf((red_var[r] + red_var[128 + r]) / (float)BN + p.eps);
        for (int c = 32 * half; c < BN; c += 64) {
          float v[32];
          tmem_ld32(trow + (uint32_t)c, v);
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int i = 0; i < 32; i += 2)
            split2((v[i] - mean) * rstd, (v[i + 1] - mean) * rstd, hi[i / 2], lo[i / 2]);
          stage_split(hi, lo, c, srow);
        }
      } else if (EPI == EPI_LN_FOLD) {
        // LN(x) W = rstd (x W) - mu rstd colsum(W) from the raw rows' product,
        // rounded to one f16 plane (an attention operand)
        float2 ms = make_float2(0.f, 0.f);
        if (valid) ms = __ldg(p.row_stats + grow);
        const float nmr = -ms.x * ms.y;
        for (int c = 32 * half; c < BN; c += 64) {
          float v[32];
          tmem_ld32(trow + (uint32_t)c, v);
          const int col = n0 + c;
          const float4* cw = reinterpret_cast<const float4*>(p.colsum + col);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 cc = __ldg(cw + j);
            v[4 * j] = fmaf(v[4 * j], ms.y, nmr * cc.x);
            v[4 * j + 1] = fmaf(v[4 * j + 1], ms.y, nmr * cc.y);
            v[4 * j + 2] = fmaf(v[4 * j + 2], ms.y, nmr * cc.z);
            v[4 * j + 3] = fmaf(v[4 * j + 3], ms.y, nmr * cc.w);
          }
          uint8_t* b = next_stage();
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint32_t o = (uint32_t)lane * 64u + ((uint32_t)(j ^ ((lane >> 1) & 3)) << 4);
            *reinterpret_cast<uint4*>(b + o) =
                make_uint4(pack_f16x2(v[8 * j], v[8 * j + 1]), pack_f16x2(v[8 * j + 2], v[8 * j + 3]),
                           pack_f16x2(v[8 * j + 4], v[8 * j + 5]), pack_f16x2(v[8 * j + 6], v[8 * j + 7]));
          }
          issue(&tO_h, b, nullptr, nullptr, col, srow);
        }
      } else {  // EPI_HEAD
        // per task t: the dot product of ReLU(acc + b1) with w2 over its
        // head_d columns (a 32-column block lies in one task, head_d % 32 == 0)
        // (with a cluster, this CTA's BN columns from n0 on; at most two tasks)
        const int nt = p.n_tasks, ncol = nt * p.head_d;
        float acc4[4] = {0.f, 0.f, 0.f, 0.f};
        for (int c = 32 * half; c < BN && n0 + c < ncol; c += 64) {
          const int gc = n0 + c;
          float v[32];
          tmem_ld32(trow + (uint32_t)c, v);
          float a = 0.f;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float x = relu_nan(v[i] + p.bias[gc + i]);
            a = fmaf(x, p.w2[gc + i], a);
          }
          const int t = gc / p.head_d;
#pragma unroll
          for (int tt = 0; tt < 4; ++tt)
            if (tt == t) acc4[tt] += a;
        }
        float tot[4] = {0.f, 0.f, 0.f, 0.f};
        if (cs > 1) {
          // every warp's partial dot of task 0 (and 1) into every CTA of the cluster
          if (!row_xchg(0, acc4[0], tot[0])) break;
          if (nt > 1 && !row_xchg(1, acc4[1], tot[1])) break;
        } else {
          // both halves' partial sums, two tasks per exchange
#pragma unroll
          for (int t0 = 0; t0 < 4; t0 += 2) {
            if (t0 < nt) {
              if (t0 > 0) pair_sync();  // the previous round's reads are done
              red_sum[half * 128 + r] = acc4[t0];
              red_var[half * 128 + r] = acc4[t0 + 1];
              pair_sync();
              tot[t0] = red_sum[r] + red_sum[128 + r];
              tot[t0 + 1] = red_var[r] + red_var[128 + r];
            }
          }
        }
        // (uniform per warp: the warps of the first column half of the cluster's
        // first CTA write the scores)
        if (half == 0 && my_rank == 0) {
          float f = 0.f;
          if (valid) {
            if (nt == 1) {
              f = tot[0] + p.b2[0];
              if (p.task_scores) p.task_scores[grow] = f;
            } else {
              f = p.fuse_b[0];
#pragma unroll
              for (int t = 0; t < 4; ++t) {
                if (t < nt) {
                  const float st = tot[t] + p.b2[t];
                  if (p.task_scores) p.task_scores[(size_t)grow * nt + t] = st;
                  f = fmaf(p.fuse_w[t], st, f);
                }
              }
            }
          }
          if (p.sel.keys) sel_fold_warp(p.sel, grow, f, valid);  // the argmax over the request's K sequences
          if (valid) p.scores[grow] = f;
        }
      }
      // every TMEM read of this accumulator has completed (tcgen05.wait::ld)
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty + acc);
    }
    if (lane == 0) bulk_wait0();  // output tensor stores complete before the CTA retires
  }

  __syncwarp();  // each warp arrives whole: single lanes ran the producer and MMA loops
  tc_fence_before();
  __syncthreads();
  if (cs > 1) cluster_sync_all();  // no peer still stores into this CTA's exchange area
  if (warp == 0) tmem_dealloc(tmem, ncols);
  if (EPI == EPI_HEAD && p.sel.keys) sel_ticket(p.sel, tmem_slot);
}

template <int EPI, int NB>
static cudaError_t launch_t(const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* b_h,
                            const CUtensorMap* b_l, const CUtensorMap* o_h, const CUtensorMap* o_l,
                            const CUtensorMap* o_x, const GemmParams& p0, cudaStream_t s) {
  GemmParams p = p0;
  const int cs = ((EPI == EPI_RESID_LN || EPI == EPI_HEAD) && p.cs > 1) ? p.cs : 1;
  p.cs = cs;
  const int sms = g_num_sms > 0 ? g_num_sms : 148;
  const long long tiles = (long long)((p.rows + BM - 1) / BM) * (p.N / p.BN);
  constexpr int NA = EPI == EPI_LN_FOLD ? 1 : 2;
  const size_t stage = (size_t)NA * kATile + (size_t)p.nb * p.BN * BK * 2;
  // At most two waves of tiles: two CTAs per SM, one accumulator each, so the
  // co-resident CTAs overlap each other's loads, MMAs and epilogues.
  // Otherwise: one persistent CTA per SM with a double-buffered accumulator.
  int per_sm = 1;
  const int st2 = (int)((kSmemPerSM / 2 - 1024 - kSmemFixed - red_bytes(cs)) / stage);
  if (tiles <= 2LL * sms && st2 >= 1 && 2 * pow2_cols(p.BN) <= 512 && g_two_per_sm[EPI][NB - 1]) {
    per_sm = 2;
    p.nacc = 1;
    p.stages = st2 < kMaxStages ? st2 : kMaxStages;
  } else {
    p.nacc = 2 * p.BN <= 512 ? 2 : 1;
    p.stages = gemm_max_stages(p.BN, p.nb, p.K_pad, cs, NA);
  }
  size_t smem = gemm_smem_bytes(p.BN, p.nb, p.stages, cs, NA);
  // (CTAs resident per SM) x (TMEM columns per CTA) <= 512: no CTA ever waits in
  // tcgen05.alloc for a co-resident one
  const size_t max_ctas = 512 / pow2_cols(p.nacc * p.BN);
  const size_t floor_bytes = kSmemPerSM / (max_ctas + 1) + 1;
  if (smem < floor_bytes) smem = floor_bytes;
  if (smem > kSmemMaxBlock) smem = kSmemMaxBlock;
  if (cs > 1) {
    // as many whole clusters as can be resident at once (the CTAs of a cluster
    // share a GPC), persistent over the row tiles; tiles is a multiple of cs
    if (p.N != cs * p.BN || p.BN > 128 || cs > kMaxCluster) return cudaErrorInvalidValue;
    long long nclu = g_cluster_cap[per_sm - 1][cs];
    if (nclu < 1) return cudaErrorInvalidConfiguration;
    if (g_cluster_limit > 0 && nclu > g_cluster_limit) nclu = g_cluster_limit;
    long long grid = nclu * cs;
    if (grid > tiles) grid = tiles;
    return launch_kc(gemm_kernel<EPI, NB>, dim3((unsigned)grid), dim3(kThreads), smem, s, cs, *a_h, *a_l, *b_h,
                     *b_l, o_h ? *o_h : *a_h, o_l ? *o_l : *a_l, o_x ? *o_x : *a_h, p);
  }
  long long grid = (long long)sms * per_sm;
  if (grid > tiles) grid = tiles;
  return launch_k(gemm_kernel<EPI, NB>, dim3((unsigned)grid), dim3(kThreads), smem, s, *a_h, *a_l, *b_h, *b_l,
                  o_h ? *o_h : *a_h, o_l ? *o_l : *a_l, o_x ? *o_x : *a_h, p);
}

cudaError_t gemm_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
  auto attr = [&](const void* f) {
    if (e == cudaSuccess) e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMaxBlock);
  };
  attr((const void*)gemm_kernel<EPI_STORE, 1>);
  attr((const void*)gemm_kernel<EPI_STORE, 2>);
  attr((const void*)gemm_kernel<EPI_RESID_LN, 1>);
  attr((const void*)gemm_kernel<EPI_RESID_LN, 2>);
  attr((const void*)gemm_kernel<EPI_HEAD, 1>);
  attr((const void*)gemm_kernel<EPI_HEAD, 2>);
  attr((const void*)gemm_kernel<EPI_LN_FOLD, 1>);
  attr((const void*)gemm_kernel<EPI_LN_FOLD, 2>);
  auto two_fit = [&](const void* f) {
    int n = 0;
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, f, kThreads, kSmemPerSM / 2 - 1024);
    return n >= 2;
  };
  g_two_per_sm[EPI_STORE][0] = two_fit((const void*)gemm_kernel<EPI_STORE, 1>);
  g_two_per_sm[EPI_STORE][1] = two_fit((const void*)gemm_kernel<EPI_STORE, 2>);
  g_two_per_sm[EPI_RESID_LN][0] = two_fit((const void*)gemm_kernel<EPI_RESID_LN, 1>);
  g_two_per_sm[EPI_RESID_LN][1] = two_fit((const void*)gemm_kernel<EPI_RESID_LN, 2>);
  g_two_per_sm[EPI_HEAD][0] = two_fit((const void*)gemm_kernel<EPI_HEAD, 1>);
  g_two_per_sm[EPI_HEAD][1] = two_fit((const void*)gemm_kernel<EPI_HEAD, 2>);
  g_two_per_sm[EPI_LN_FOLD][0] = two_fit((const void*)gemm_kernel<EPI_LN_FOLD, 1>);
  g_two_per_sm[EPI_LN_FOLD][1] = two_fit((const void*)gemm_kernel<EPI_LN_FOLD, 2>);
  if (g_cluster_limit < 0) {
    const char* v = std::getenv("FE_GEMM_CLUSTERS");
    g_cluster_limit = v && *v ? std::atoi(v) : 0x7fffffff;
  }
  // resident clusters per size, for one CTA per SM (all the shared memory) and two
  for (int two = 0; two < 2 && e == cudaSuccess; ++two) {
    for (int cs = 2; cs <= kMaxCluster; cs *= 2) {
      int n1 = 0, n2 = 0;
      for (int nbv = 1; nbv <= 2; ++nbv) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)cs);
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = two ? kSmemPerSM / 2 - 1024 : kSmemMaxBlock;
        cudaLaunchAttribute a[1];
        a[0].id = cudaLaunchAttributeClusterDimension;
        a[0].val.clusterDim.x = (unsigned)cs;
        a[0].val.clusterDim.y = 1;
        a[0].val.clusterDim.z = 1;
        cfg.attrs = a;
        cfg.numAttrs = 1;
        int n = 0;
        // the LayerNorm and head instantiations: the smaller capacity
        const void* f = nbv == 1 ? (const void*)gemm_kernel<EPI_RESID_LN, 1> : (const void*)gemm_kernel<EPI_RESID_LN, 2>;
        const void* fh = nbv == 1 ? (const void*)gemm_kernel<EPI_HEAD, 1> : (const void*)gemm_kernel<EPI_HEAD, 2>;
        int nh = 0;
        if (cudaOccupancyMaxActiveClusters(&n, f, &cfg) != cudaSuccess ||
            cudaOccupancyMaxActiveClusters(&nh, fh, &cfg) != cudaSuccess) {
          (void)cudaGetLastError();
          n = nh = 0;
        }
        (nbv == 1 ? n1 : n2) = n < nh ? n : nh;
      }
      g_cluster_cap[two][cs] = g_cluster_limit == 0 ? 0 : (n1 < n2 ? n1 : n2);
    }
  }
  return e;
}

int gemm_cluster_capacity(int cs) {
  return (cs >= 2 && cs <= kMaxCluster) ? g_cluster_cap[0][cs] : 0;
}

cudaError_t gemm_launch(int epi, const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* b_h,
                        const CUtensorMap* b_l, const CUtensorMap* o_h, const CUtensorMap* o_l,
                        const CUtensorMap* o_x, const GemmParams& p, cudaStream_t s) {
  if (p.rows <= 0) return cudaSuccess;
  const bool two = p.nb > 1;
  switch (epi) {
    case EPI_STORE:
      return two ? launch_t<EPI_STORE, 2>(a_h, a_l, b_h, b_l, o_h, o_l, o_x, p, s)
                 : launch_t<EPI_STORE, 1>(a_h, a_l, b_h, b_l, o_h, o_l, o_x, p, s);
    case EPI_RESID_LN:
      return two ? launch_t<EPI_RESID_LN, 2>(a_h, a_l, b_h, b_l, o_h, o_l, o_x, p, s)
                 : launch_t<EPI_RESID_LN, 1>(a_h, a_l, b_h, b_l, o_h, o_l, o_x, p, s);
    case EPI_LN_FOLD:
      return two ? launch_t<EPI_LN_FOLD, 2>(a_h, a_l, b_h, b_l, o_h, o_l, o_x, p, s)
                 : launch_t<EPI_LN_FOLD, 1>(a_h, a_l, b_h, b_l, o_h, o_l, o_x, p, s);
    default:
      return two ? launch_t<EPI_HEAD, 2>(a_h, a_l, b_h, b_l, o_h, o_l, o_x, p, s)
                 : launch_t<EPI_HEAD, 1>(a_h, a_l, b_h, b_l, o_h, o_l, o_x, p, s);
  }
}

}  // namespace fe
