// Flash-style multi-head attention over request segments, on tcgen05.
//
// Used twice in the evaluator:
//  * element -> context cross-attention (Section 4.2): the query rows are the
//    distinct elements of request b, the keys/values its C context rows, so
//    the context K/V computed once per request serve every element;
//  * cross-sequence self-attention (Section 4.4) over the K sequence vectors.
//
// Persistent CTAs walk units (segment b, head h, 128-row query tile).  Per
// unit the keys stream in chunks of CK (64 for d_h = 32, 128 for d_h = 64):
//   warp 0 lane 0 : TMA producer -- Q tile (two buffers, one per unit in
//                   flight) and K/V chunks of CK keys (8 stages for d_h = 32,
//                   4 for d_h = 64)
//   warp 1 lane 0 : tcgen05.mma -- S_j = Q K_j^T into TMEM tile j % 2, then
//                   PV_j = P_j V_j with P_j read from that same TMEM tile
//                   into PV buffer j % 2
//   warps 2..     : online softmax from TMEM, one query row per lane; with
//                   d_h = 64, warps w and w+4 share TMEM lane quadrant w % 4
//                   and each take half of the chunk's keys and half of the
//                   output columns.  P_j is written back over S_j as f16;
//                   PV_{j-1} is folded into the register output after P_j is
//                   handed over, so the softmax never waits for the PV
//                   product of the chunk it has just finished
// Q, K, V and P are single f16 planes (unit roundoff 2^-11; Q and K come
// from LayerNorm'd rows times weights of magnitude well inside the f16
// range, P lies in [0, 1]); accumulation, softmax statistics and the output
// are fp32, the output leaves as a bf16 hi/lo pair.
#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {

constexpr int BQ = 128;     // query rows per unit (TMEM lanes)

// d_h = 32: 64-key chunks and 4 softmax warps, small enough for two CTAs per SM.
// d_h = 64: 128-key chunks and 8 softmax warps (two per TMEM lane quadrant).
template <int DH>
struct AttnCfg {
  static constexpr int CK = DH == 32 ? 64 : 128;                // keys per chunk
  static constexpr int kSoftmaxWarps = DH == 32 ? 4 : 8;
  static constexpr int kHalves = kSoftmaxWarps / 4;              // warps sharing one lane quadrant
  static constexpr int kThreads = 64 + 32 * kSoftmaxWarps;
  static constexpr int kCtasPerSM = DH == 32 ? 2 : 1;
  // TMEM: S/P tiles at [0, CK) and [CK, 2CK), PV buffers at [2CK, 2CK + 2DH)
  static constexpr uint32_t kTmemCols = DH == 32 ? 256 : 512;
  static constexpr uint32_t kRowBytes = DH * 2;                 // one row of a Q/K/V tile
  static constexpr uint32_t kQBytes = 128 * kRowBytes;          // Q tile: 128 rows
  static constexpr uint32_t kKVTile = CK * kRowBytes;           // K or V chunk: CK rows
  static constexpr uint32_t kSwz = DH == 32 ? 4u : 2u;          // descriptor swizzle code (64 B / 128 B)
  static constexpr uint32_t kSbo = 8 * kRowBytes;               // 8-row swizzle atom
  static constexpr uint32_t kKVBytes = 2 * kKVTile;             // K, V
  static constexpr int kKVStages = DH == 32 ? 8 : 4;
  static constexpr uint32_t kRed = 2 * 2 * 2 * 128 * 4;       // [max|sum][parity][half][row]
  static constexpr size_t kSmem = 1024 + 2 * kQBytes + kKVStages * kKVBytes + 256 + kRed;
};

__device__ __forceinline__ uint64_t desc_sw(uint32_t saddr, uint32_t sbo, uint32_t swz) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;                       // leading byte offset (unused: one atom wide)
  d |= (uint64_t)(sbo >> 4) << 32;              // stride byte offset: next 8-row atom
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)swz << 61;
  return d;
}

__device__ __forceinline__ void mbar_arrive1(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

}  // namespace

template <int DH>
__global__ void __launch_bounds__(AttnCfg<DH>::kThreads, AttnCfg<DH>::kCtasPerSM)
    attn_kernel(const __grid_constant__ CUtensorMap tQ, const __grid_constant__ CUtensorMap tK,
                const __grid_constant__ CUtensorMap tV, const AttnParams p) {
  using Cfg = AttnCfg<DH>;
  constexpr int CK = Cfg::CK;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  uint8_t* sQ = smem;                                   // [2 buffers]
  uint8_t* sKV = sQ + 2 * Cfg::kQBytes;                 // [stages][K, V]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sKV + Cfg::kKVStages * Cfg::kKVBytes);
  uint64_t* q_full = bars;        // [2]
  uint64_t* q_empty = bars + 2;   // [2]
  uint64_t* kv_full = bars + 4;   // [stages]
  uint64_t* kv_empty = bars + 12; // [stages]
  uint64_t* s_full = bars + 20;   // [2] S_j complete in TMEM tile j % 2
  uint64_t* p_full = bars + 22;   // [2] P_j written over S_j
  uint64_t* pv_full = bars + 24;  // [2] PV_j complete in PV buffer j % 2
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 26);
  float* red = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);  // row-statistic exchange

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qtiles = p.max_q_tiles;
  const int units = p.n_segments * p.n_heads * qtiles;
  const int nch = (p.kv_cnt + CK - 1) / CK;
  if ((int)blockIdx.x >= units) return;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(q_full + i, 1);
      mbar_init(q_empty + i, 1);
      mbar_init(s_full + i, 1);
      mbar_init(p_full + i, 32 * Cfg::kSoftmaxWarps);
      mbar_init(pv_full + i, 1);
    }
    for (int i = 0; i < Cfg::kKVStages; ++i) {
      mbar_init(kv_full + i, 1);
      mbar_init(kv_empty + i, 1);
    }
    fence_mbar_init();
    prefetch_tmap(&tQ);
    prefetch_tmap(&tK);
    prefetch_tmap(&tV);
  }
  if (warp == 0) tmem_alloc(tmem_slot, Cfg::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // the set-up above reads nothing written by earlier kernels; from here on
  // the segment offsets, counts and operands are
  pdl_trigger();
  pdl_wait();

  // unit u -> (segment, head, query tile); query tile fastest
  auto unit_info = [&](int u, int& b, int& h, int& q0, int& qcnt, int& qoff) {
    const int qt = u % qtiles;
    h = (u / qtiles) % p.n_heads;
    b = u / (qtiles * p.n_heads);
    qcnt = p.q_cnt_dev ? p.q_cnt_dev[b] : p.q_cnt_fixed;
    qoff = p.q_off_dev ? p.q_off_dev[b] : b * p.q_stride;
    q0 = qt * BQ;
  };

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int ui = 0, gc = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        int b, h, q0, qcnt, qoff;
        unit_info(u, b, h, q0, qcnt, qoff);
        if (q0 >= qcnt) continue;
        const int qb = ui & 1;
        if (ui >= 2 && !mbar_wait_bounded(q_empty + qb, ((ui >> 1) - 1) & 1, p.status)) break;
        uint8_t* q = sQ + qb * Cfg::kQBytes;
        mbar_arrive_expect_tx(q_full + qb, Cfg::kQBytes);
        tma_load_2d(q, &tQ, p.q_col + h * DH, qoff + q0, q_full + qb);
        for (int j = 0; j < nch; ++j, ++gc) {
          const int ks = gc % Cfg::kKVStages;
          if (gc >= Cfg::kKVStages &&
              !mbar_wait_bounded(kv_empty + ks, ((gc / Cfg::kKVStages) - 1) & 1, p.status)) {
            ok = false;
            break;
          }
          uint8_t* kv = sKV + ks * Cfg::kKVBytes;
          const int row = b * p.kv_stride + j * CK;
          mbar_arrive_expect_tx(kv_full + ks, Cfg::kKVBytes);
          tma_load_2d(kv, &tK, p.k_col + h * DH, row, kv_full + ks);
          tma_load_2d(kv + Cfg::kKVTile, &tV, p.v_col + h * DH, row, kv_full + ks);
        }
        ++ui;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc_s = umma_idesc_f16(BQ, CK);
      const uint32_t idesc_pv = umma_idesc_f16(BQ, DH) | (1u << 16);  // B (V) is MN-major
      int ui = 0, gc = 0;
      bool ok = true;
      // S = Q K^T of global chunk gcc into TMEM tile gcc % 2, the unit's Q in buffer qb
      auto issue_s = [&](int qb, int gcc) -> bool {
        // the tile is free once PV_{gcc-2}, which reads P_{gcc-2} from it, has completed
        if (gcc >= 2 && !mbar_wait_bounded(pv_full + (gcc & 1), ((gcc - 2) >> 1) & 1, p.status)) return false;
        const int ks = gcc % Cfg::kKVStages;
        if (!mbar_wait_bounded(kv_full + ks, (gcc / Cfg::kKVStages) & 1, p.status)) return false;
        tc_fence_after();
        const uint32_t q = smem_u32(sQ + qb * Cfg::kQBytes);
        const uint32_t k = smem_u32(sKV + ks * Cfg::kKVBytes);
        const uint32_t dst = tmem + (uint32_t)((gcc & 1) * CK);
        const uint64_t q0d = desc_sw(q, Cfg::kSbo, Cfg::kSwz), k0d = desc_sw(k, Cfg::kSbo, Cfg::kSwz);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk)
          umma_bf16(dst, desc_adv(q0d, kk * 32), desc_adv(k0d, kk * 32), idesc_s, kk != 0 ? 1u : 0u);
        umma_commit(s_full + (gcc & 1));
        return true;
      };
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        int b, h, q0, qcnt, qoff;
        unit_info(u, b, h, q0, qcnt, qoff);
        if (q0 >= qcnt) continue;
        const int qb = ui & 1;
        if (!mbar_wait_bounded(q_full + qb, (ui >> 1) & 1, p.status)) break;
        for (int j = 0; j < nch; ++j, ++gc) {
          // S_{j+1} is issued ahead so that it overlaps the softmax of chunk j
          if ((j == 0 && !issue_s(qb, gc)) || (j + 1 < nch && !issue_s(qb, gc + 1))) {
            ok = false;
            break;
          }
          if (j + 1 == nch) umma_commit(q_empty + qb);  // every S of this unit issued: Q buffer frees on completion
          if (!mbar_wait_bounded(p_full + (gc & 1), (gc >> 1) & 1, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // PV_j: A = P_j from TMEM tile j % 2, each key block of 64 as 32
          // columns of f16 pairs at the start of its 64 S columns
          const int ks = gc % Cfg::kKVStages;
          const uint32_t v = smem_u32(sKV + ks * Cfg::kKVBytes + Cfg::kKVTile);
          const uint32_t pt = tmem + (uint32_t)((gc & 1) * CK);
          const uint32_t dst = tmem + (uint32_t)(2 * CK + (gc & 1) * DH);
          const uint64_t v0d = desc_sw(v, Cfg::kSbo, Cfg::kSwz);
#pragma unroll
          for (int kk = 0; kk < CK / 16; ++kk)
            umma_bf16_tmem_a(dst, pt + (uint32_t)((kk >> 2) * 64 + (kk & 3) * 8),
                             desc_adv(v0d, (uint32_t)kk * 16 * Cfg::kRowBytes), idesc_pv, kk != 0 ? 1u : 0u);
          umma_commit(pv_full + (gc & 1));
          umma_commit(kv_empty + ks);
        }
        ++ui;
      }
    }
  } else {
    // ---------------- softmax / output (warps 2..9) ----------------
    constexpr int DO = DH / Cfg::kHalves;  // output columns per warp
    constexpr int KW = CK / Cfg::kHalves;  // keys per warp and chunk (64)
    const int sw = warp - 2;
    const int q4 = warp & 3;
    const int half = sw >> 2;     // keys [KW half, KW half + KW) of each chunk, output columns [DO half, DO half + DO)
    const int r = q4 * 32 + lane; // query row of the tile = TMEM lane
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    float* red_max = red;         // [parity][half][128]
    float* red_sum = red + 512;
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + q4) : "memory"); };
    // fold PV_g (PV buffer g % 2) into the register output: o = o * c + PV_g
    auto fold = [&](int g, float c, float* o) -> bool {
      if (!mbar_wait_bounded(pv_full + (g & 1), (g >> 1) & 1, p.status)) return false;
      tc_fence_after();
      float pv[DO];
      const uint32_t src = tmem + lane_off + (uint32_t)(2 * CK + (g & 1) * DH + half * DO);
      if (DO == 16) {
        tmem_ld16(src, pv);
      } else {
#pragma unroll
        for (int cc = 0; cc < DO; cc += 32) tmem_ld32(src + (uint32_t)cc, pv + cc);
      }
#pragma unroll
      for (int i = 0; i < DO; ++i) o[i] = o[i] * c + pv[i];
      return true;
    };
    int gc = 0, ui = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      int b, h, q0, qcnt, qoff;
      unit_info(u, b, h, q0, qcnt, qoff);
      if (q0 >= qcnt) continue;
      float m = -INFINITY, l = 0.f, corr_prev = 1.f;
      float o[DO];
#pragma unroll
      for (int i = 0; i < DO; ++i) o[i] = 0.f;
      // a warp whose 32 query rows all lie past the segment's end only keeps
      // the barrier protocol; those rows of P and of the output are never used
      const bool active = q0 + q4 * 32 < qcnt;
      for (int j = 0; j < nch; ++j, ++gc) {
        if (!mbar_wait_bounded(s_full + (gc & 1), (gc >> 1) & 1, p.status)) {
          ok = false;
          break;
        }
        float corr = 1.f;
        if (active) {
          tc_fence_after();
          const uint32_t tile = tmem + lane_off + (uint32_t)((gc & 1) * CK + half * KW);
          float v[64];
          tmem_ld64(tile, v);
          const int kvalid = p.kv_cnt - j * CK - half * KW;  // valid keys among this warp's 64
          float mx = -INFINITY;
          if (kvalid >= 64) {
#pragma unroll
            for (int i = 0; i < 64; ++i) mx = fmaxf(mx, v[i]);
          } else {
#pragma unroll
            for (int i = 0; i < 64; ++i)
              if (i < kvalid) mx = fmaxf(mx, v[i]);
          }
          mx *= p.scale_log2;
          if (Cfg::kHalves == 2) {
            float* rm = red_max + (gc & 1) * 256;
            rm[half * 128 + r] = mx;
            pair_sync();
            mx = fmaxf(rm[r], rm[128 + r]);
          }
          const float mn = fmaxf(m, mx);
          corr = ex2_approx(m - mn);
          m = mn;
          // P = 2^(s * scale - m) as f16 over the first 32 of this warp's 64
          // S columns (all 64 already in registers): keys 2c, 2c+1 in column
          // c; keys past kv_cnt get 0
          const float sc = p.scale_log2, nm = -mn;
          float sum = 0.f;
          auto emit = [&](auto full) {
#pragma unroll
            for (int hb = 0; hb < 2; ++hb) {
              uint32_t pk[16];
#pragma unroll
              for (int i = 0; i < 32; i += 2) {
                const int k = 32 * hb + i;
                float p0 = ex2_approx(fmaf(v[k], sc, nm));
                float p1 = ex2_approx(fmaf(v[k + 1], sc, nm));
                if (!decltype(full)::value) {
                  p0 = k < kvalid ? p0 : 0.f;
                  p1 = k + 1 < kvalid ? p1 : 0.f;
                }
                sum += p0 + p1;
                pk[i / 2] = pack_f16x2(p0, p1);
              }
              tmem_st16_nowait(tile + (uint32_t)(16 * hb), pk);
            }
          };
          if (kvalid >= 64) emit(std::true_type{});
          else emit(std::false_type{});
          l = l * corr + sum;
          tmem_st_wait();
          tc_fence_before();
        }
        mbar_arrive1(p_full + (gc & 1));
        // the previous chunk's PV is folded while PV_j runs
        if (j > 0 && active && !fold(gc - 1, corr_prev, o)) {
          ok = false;
          break;
        }
        corr_prev = corr;
      }
      if (!ok) break;
      if (active && !fold(gc - 1, corr_prev, o)) break;
      // row sum over both halves, then O / l as a split pair
      float ltot = l;
      if (Cfg::kHalves == 2) {
        float* rs = red_sum + (ui & 1) * 256;
        rs[half * 128 + r] = l;
        pair_sync();
        ltot = rs[r] + rs[128 + r];
      }
      ++ui;
      if (q0 + r < qcnt) {
        const float inv = 1.f / ltot;
        const size_t go = (size_t)(qoff + q0 + r) * p.ldo + p.o_col + h * DH + half * DO;
#pragma unroll
        for (int c = 0; c < DO; c += 8) {
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int i = 0; i < 8; i += 2) split2(o[c + i] * inv, o[c + i + 1] * inv, hi[i / 2], lo[i / 2]);
          *reinterpret_cast<uint4*>(p.o_h + go + c) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
          *reinterpret_cast<uint4*>(p.o_l + go + c) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, Cfg::kTmemCols);
}

namespace {
int g_attn_sms = 0;
}

cudaError_t attn_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_attn_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)AttnCfg<32>::kSmem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)AttnCfg<64>::kSmem);
  return e;
}

cudaError_t attn_launch(int dh, const CUtensorMap* q, const CUtensorMap* k, const CUtensorMap* v, const AttnParams& p0,
                        cudaStream_t s) {
  if (p0.n_segments <= 0 || p0.max_q <= 0 || p0.kv_cnt <= 0) return cudaSuccess;
  AttnParams p = p0;
  p.max_q_tiles = (p.max_q + BQ - 1) / BQ;
  const long long units = (long long)p.n_segments * p.n_heads * p.max_q_tiles;
  const long long sms = g_attn_sms > 0 ? g_attn_sms : 148;
  if (dh == 32) {
    const long long grid = units < sms * AttnCfg<32>::kCtasPerSM ? units : sms * AttnCfg<32>::kCtasPerSM;
    return launch_k(attn_kernel<32>, dim3((unsigned)grid), dim3(AttnCfg<32>::kThreads), AttnCfg<32>::kSmem, s, *q, *k,
                    *v, p);
  }
  const long long grid = units < sms * AttnCfg<64>::kCtasPerSM ? units : sms * AttnCfg<64>::kCtasPerSM;
  return launch_k(attn_kernel<64>, dim3((unsigned)grid), dim3(AttnCfg<64>::kThreads), AttnCfg<64>::kSmem, s, *q, *k,
                  *v, p);
}

}  // namespace fe
