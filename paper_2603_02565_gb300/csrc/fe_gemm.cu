// tcgen05 GEMM of the joint evaluator with fused epilogues.
//
// Every dense product of the model (context K/V projection and element
// WQ / WO / FFN of Section 4.2, SeqEnc and cross-sequence projections of
// Sections 4.3-4.4, the score head) is  act[rows, K] x W[K, N]  with a small
// K (d or F).  One CTA computes a 128-row x BN-column tile:
//   warp 0 lane 0  : TMA producer (A hi/lo tiles + weight tiles per 64-wide k block)
//   warp 1 lane 0  : tcgen05.mma issuer, fp32 accumulator in TMEM
//   warps 0-3      : epilogue, thread t owns tile row t (TMEM lane t)
// The activation is a split pair (hi + lo bf16); the product is
// A_hi W_hi + A_lo W_hi (+ A_hi W_lo when the weights carry a lo plane).
#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {
constexpr int BM = 128;
constexpr int BK = 64;                               // one 128-byte swizzle row of bf16
constexpr uint32_t kATile = BM * BK * 2;             // 16 KB per activation plane
constexpr size_t kSmemPerSM = 233472;                // 228 KB
constexpr size_t kSmemMaxBlock = 232448;             // 227 KB opt-in per block
constexpr size_t kSmemExtra = 1024 + 256;            // alignment slack + barriers

uint32_t tmem_cols_for(int BN) {
  return BN <= 32 ? 32u : BN <= 64 ? 64u : BN <= 128 ? 128u : BN <= 256 ? 256u : 512u;
}
}  // namespace

size_t gemm_smem_bytes(int BN, int nb, int stages) {
  const size_t stage = 2 * (size_t)kATile + (size_t)nb * BN * BK * 2;
  return (size_t)stages * stage + kSmemExtra;
}

int gemm_max_stages(int BN, int nb, int K_pad) {
  const size_t stage = 2 * (size_t)kATile + (size_t)nb * BN * BK * 2;
  int s = (int)((kSmemMaxBlock - kSmemExtra) / stage);
  const int nk = K_pad / BK;
  if (s > 4) s = 4;
  if (s > nk) s = nk;
  return s < 1 ? 1 : s;
}

template <int EPI>
__global__ void __launch_bounds__(128, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tA_h, const __grid_constant__ CUtensorMap tA_l,
                const __grid_constant__ CUtensorMap tB_h, const __grid_constant__ CUtensorMap tB_l,
                const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);

  const int BN = p.BN, nb = p.nb, S = p.stages;
  const uint32_t b_bytes = (uint32_t)BN * BK * 2;
  const uint32_t stage_bytes = 2 * kATile + (uint32_t)nb * b_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)S * stage_bytes);
  uint64_t* empty = full + S;
  uint64_t* done = empty + S;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row0 = blockIdx.x * BM;
  const int n0 = blockIdx.y * BN;
  int rows_valid = p.rows;
  if (p.rows_dev) rows_valid = min(*p.rows_dev, p.rows);
  if (row0 >= rows_valid) return;  // whole CTA past the valid rows

  const uint32_t ncols = BN <= 32 ? 32u : BN <= 64 ? 64u : BN <= 128 ? 128u : BN <= 256 ? 256u : 512u;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    mbar_init(done, 1);
    fence_mbar_init();
    prefetch_tmap(&tA_h);
    prefetch_tmap(&tA_l);
    prefetch_tmap(&tB_h);
    if (nb > 1) prefetch_tmap(&tB_l);
  }
  if (warp == 0) tmem_alloc(tmem_slot, ncols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int nk = p.K_pad / BK;

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % S;
      if (kb >= S && !mbar_wait_bounded(empty + s, ((kb / S) & 1) ^ 1, p.status)) break;
      uint8_t* st = smem + (size_t)s * stage_bytes;
      mbar_arrive_expect_tx(full + s, stage_bytes);
      tma_load_2d(st, &tA_h, kb * BK, row0, full + s);
      tma_load_2d(st + kATile, &tA_l, kb * BK, row0, full + s);
      for (int q = 0; q < nb; ++q) {
        const CUtensorMap* tb = q ? &tB_l : &tB_h;
        for (int h = 0; h < BN; h += 256)
          tma_load_2d(st + 2 * kATile + q * b_bytes + (uint32_t)h * BK * 2, tb, kb * BK, n0 + h, full + s);
      }
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    const int nmma = BN > 256 ? 256 : BN;
    const uint32_t idesc = umma_idesc_bf16(BM, nmma);
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % S;
      if (!mbar_wait_bounded(full + s, (kb / S) & 1, p.status)) break;
      tc_fence_after();
      const uint32_t st = smem_u32(smem + (size_t)s * stage_bytes);
#pragma unroll 1
      for (int kk = 0; kk < BK / 16; ++kk) {
        // (A_hi, W_hi), (A_lo, W_hi), (A_hi, W_lo)
        for (int pr = 0; pr < 1 + nb; ++pr) {
          const uint32_t a = st + (pr == 1 ? kATile : 0u) + (uint32_t)kk * 32;
          const uint32_t b = st + 2 * kATile + (pr == 2 ? b_bytes : 0u) + (uint32_t)kk * 32;
          const uint64_t ad = umma_desc_sw128(a);
          for (int h = 0; h < BN; h += 256) {
            const uint64_t bd = umma_desc_sw128(b + (uint32_t)h * BK * 2);
            umma_bf16(tmem + (uint32_t)h, ad, bd, idesc, (kb | kk | pr) != 0 ? 1u : 0u);
          }
        }
      }
      umma_commit(empty + s);  // frees this stage once its MMAs complete
    }
    umma_commit(done);
  }
  __syncwarp();

  // ---------------- epilogue ----------------
  mbar_wait_bounded(done, 0, p.status);
  tc_fence_after();
  const int r = warp * 32 + lane;
  const int grow = row0 + r;
  const bool valid = grow < rows_valid;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);

  if (EPI == EPI_STORE) {
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      tmem_ld32(trow + (uint32_t)c, v);
      const int col = n0 + c;
      if (valid) {
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          float x0 = v[i], x1 = v[i + 1];
          if (p.bias) {
            x0 += p.bias[col + i];
            x1 += p.bias[col + i + 1];
          }
          if (p.relu) {
            x0 = fmaxf(x0, 0.f);
            x1 = fmaxf(x1, 0.f);
          }
          split2(x0, x1, hi[i / 2], lo[i / 2]);
        }
        uint4* dh = reinterpret_cast<uint4*>(p.out_h + (size_t)grow * p.ldo + col);
        uint4* dl = reinterpret_cast<uint4*>(p.out_l + (size_t)grow * p.ldo + col);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          dh[j] = make_uint4(hi[4 * j], hi[4 * j + 1], hi[4 * j + 2], hi[4 * j + 3]);
          dl[j] = make_uint4(lo[4 * j], lo[4 * j + 1], lo[4 * j + 2], lo[4 * j + 3]);
        }
      }
    }
  } else if (EPI == EPI_RESID_LN) {
    // pass 1: x = resid + acc + bias, written out and kept in TMEM
    float sum = 0.f;
    const float* rrow = p.resid + (p.ldr ? (size_t)grow * p.ldr : (size_t)0);
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      tmem_ld32(trow + (uint32_t)c, v);
      if (valid) {
        const float4* rr = reinterpret_cast<const float4*>(rrow + c);
        float4* xo = reinterpret_cast<float4*>(p.x_out + (size_t)grow * p.ldx + c);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float4 q = rr[j];
          float4 x;
          x.x = v[4 * j + 0] + q.x;
          x.y = v[4 * j + 1] + q.y;
          x.z = v[4 * j + 2] + q.z;
          x.w = v[4 * j + 3] + q.w;
          if (p.bias) {
            x.x += p.bias[c + 4 * j + 0];
            x.y += p.bias[c + 4 * j + 1];
            x.z += p.bias[c + 4 * j + 2];
            x.w += p.bias[c + 4 * j + 3];
          }
          v[4 * j + 0] = x.x;
          v[4 * j + 1] = x.y;
          v[4 * j + 2] = x.z;
          v[4 * j + 3] = x.w;
          sum += (x.x + x.y) + (x.z + x.w);
          xo[j] = x;
        }
      }
      tmem_st32(trow + (uint32_t)c, v);
    }
    const float mean = sum / (float)BN;
    // pass 2: biased variance about the mean
    float var = 0.f;
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      tmem_ld32(trow + (uint32_t)c, v);
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float dv = v[i] - mean;
        var = fmaf(dv, dv, var);
      }
    }
    const float rstd = 1.0f / sqrtf(var / (float)BN + p.eps);
    // pass 3: LN(x) as split planes
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      tmem_ld32(trow + (uint32_t)c, v);
      if (valid) {
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) split2((v[i] - mean) * rstd, (v[i + 1] - mean) * rstd, hi[i / 2], lo[i / 2]);
        uint4* dh = reinterpret_cast<uint4*>(p.ln_h + (size_t)grow * p.ldln + c);
        uint4* dl = reinterpret_cast<uint4*>(p.ln_l + (size_t)grow * p.ldln + c);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          dh[j] = make_uint4(hi[4 * j], hi[4 * j + 1], hi[4 * j + 2], hi[4 * j + 3]);
          dl[j] = make_uint4(lo[4 * j], lo[4 * j + 1], lo[4 * j + 2], lo[4 * j + 3]);
        }
      }
    }
  } else {  // EPI_HEAD
    float acc = 0.f;
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      tmem_ld32(trow + (uint32_t)c, v);
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float x = fmaxf(v[i] + p.bias[c + i], 0.f);
        acc = fmaf(x, p.w2[c + i], acc);
      }
    }
    if (valid) p.scores[grow] = acc + p.b2[0];
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, ncols);
}

static size_t gemm_launch_smem(int BN, int nb, int stages) {
  size_t smem = gemm_smem_bytes(BN, nb, stages);
  // Keep (CTAs resident per SM) x (TMEM columns per CTA) <= 512 so that no CTA
  // waits in tcgen05.alloc for a co-resident CTA.
  const size_t max_ctas = 512 / tmem_cols_for(BN);
  const size_t floor_bytes = kSmemPerSM / (max_ctas + 1) + 1;
  if (smem < floor_bytes) smem = floor_bytes;
  if (smem > kSmemMaxBlock) smem = kSmemMaxBlock;
  return smem;
}

template <int EPI>
static cudaError_t launch_t(const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* b_h,
                            const CUtensorMap* b_l, const GemmParams& p, cudaStream_t s) {
  const size_t smem = gemm_launch_smem(p.BN, p.nb, p.stages);
  dim3 grid((unsigned)((p.rows + BM - 1) / BM), (unsigned)(p.N / p.BN));
  gemm_kernel<EPI><<<grid, 128, smem, s>>>(*a_h, *a_l, *b_h, *b_l, p);
  return cudaGetLastError();
}

cudaError_t gemm_prepare() {
  cudaError_t e = cudaFuncSetAttribute(gemm_kernel<EPI_STORE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kSmemMaxBlock);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(gemm_kernel<EPI_RESID_LN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSmemMaxBlock);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(gemm_kernel<EPI_HEAD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSmemMaxBlock);
  return e;
}

cudaError_t gemm_launch(int epi, const CUtensorMap* a_h, const CUtensorMap* a_l, const CUtensorMap* b_h,
                        const CUtensorMap* b_l, const GemmParams& p, cudaStream_t s) {
  if (p.rows <= 0) return cudaSuccess;
  switch (epi) {
    case EPI_STORE: return launch_t<EPI_STORE>(a_h, a_l, b_h, b_l, p, s);
    case EPI_RESID_LN: return launch_t<EPI_RESID_LN>(a_h, a_l, b_h, b_l, p, s);
    default: return launch_t<EPI_HEAD>(a_h, a_l, b_h, b_l, p, s);
  }
}

}  // namespace fe
