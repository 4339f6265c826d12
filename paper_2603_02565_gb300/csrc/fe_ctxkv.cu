// Query Context Module of Section 4.2 in one kernel: X = LN(context rows),
// [K_0 | V_0 | K_1 | V_1 ...] = X [WK_0 | WV_0 | ...], for rows of width
// d <= 128 with bf16 inputs and bf16-exact weights.  LN(context) never
// reaches memory; K/V leave as one f16 plane (the attention operand).
//
// The LayerNorm has no affine parameters, so with mu and rstd the row's mean
// and 1 / sqrt(var + eps),
//     LN(x) W = rstd (x W) - rstd mu (1^T W):
// the MMA multiplies the raw bf16 rows as they arrive (one exact bf16 plane,
// no normalised operand tile), and the epilogue applies each row's rstd and
// -rstd mu with the column sums of W before rounding to f16.
//
// The N = 2 * n_layers * d output columns are split in two halves; CTA c
// owns half c % 2 (its slice of W^T stays resident in shared memory) and
// walks 128-row blocks of context rows:
//   warp 0 lane 0 : TMA -- the resident weight half once, then the raw
//                   context block of every tile into one of two staging
//                   buffers
//   warp 1 lane 0 : tcgen05.mma -- X W_half (N/2 <= 256 columns) from the
//                   staged raw block into one of two TMEM accumulators, so the
//                   epilogue drains one tile while the next is multiplied
//   warps 2-9     : LayerNorm statistics, two threads per context row (each
//                   half of every 64-column k block, partial sums exchanged by
//                   shuffle), from the staged raw block
//   warps 10-17   : epilogue -- column sums of the weight half once; per tile
//                   TMEM -> rstd acc - rstd mu colsum -> f16 -> 32 x 32 staging
//                   blocks -> TMA tensor stores; warps w and w+4 on TMEM lane
//                   quadrant w % 4, alternating 32-column chunks
// The raw rows are bf16, so each column half's second reading of them costs
// d * 2 bytes per row.
//
// Linear-attention state mode (STATE, two layers, C a multiple of 128): the
// half of CTA c is layer c % 2, [K_l | V_l].  K/V never leave the chip: the
// epilogue writes phi(K) (phi(x) = elu(x) + 1) and V of the 128-row tile as
// MN-major 128-byte-swizzled operand tiles, V followed by 16 columns of ones,
// and one epilogue thread issues phi(K)^T [V | 1] (M = 128, N = d + 16, K = the
// tile's rows) into TMEM, so that the ones columns accumulate z = sum of
// phi(K) over the rows, accumulating over the C / 128
// row blocks of the segment, which the CTA pair takes in a row; after the
// last one each head's diagonal d_h x d_h block and z are stored.  The K/V
// accumulator is single-buffered to leave TMEM for the state.
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
constexpr int kStgBufs = 4;                                  // staging buffers per epilogue warp (stores in flight)
constexpr size_t kSmemMaxBlock = 232448;

constexpr uint32_t kStateTile = 2 * 16384;  // a 128 x 128 f16 MN-major operand: two 64-wide atoms of 128 rows

struct CtxKvLayout {
  uint32_t w_bytes, aux_bytes, raw_bytes, nraw, tail_bytes;
  size_t smem;
};

// tail: the store staging (plain mode) or the phi(K) and V operand tiles of
// the state product (state mode, which also keeps a single raw buffer)
__host__ __device__ inline CtxKvLayout ctxkv_layout(int d_pad, int N, bool state) {
  CtxKvLayout L;
  L.w_bytes = (uint32_t)(d_pad / BK) * (uint32_t)(N / 2) * (BK * 2);  // [kb][N/2 rows x 128 B]
  L.aux_bytes = 4096;  // column sums of the weight half [256] fp32, row statistics [2][128] float2
  L.raw_bytes = (uint32_t)(d_pad / BK) * kPlane;                      // one raw block [kb]
  L.nraw = state ? 1u : 2u;
  // (state mode: the V tile has a third 64-feature atom for the ones columns of z)
  L.tail_bytes = state ? 2u * kStateTile + 16384u : (uint32_t)kEpiWarps * (uint32_t)kStgBufs * kStage;
  L.smem = 1024 + (size_t)L.w_bytes + L.aux_bytes + L.nraw * (size_t)L.raw_bytes + L.tail_bytes + 256;
  return L;
}

// MN-major shared-memory descriptor, 128-byte swizzle: atoms of 64 elements
// (M or N) x 8 rows (K); `lbo` = bytes between atoms along M/N, 1024 bytes
// between 8-row groups along K
__device__ __forceinline__ uint64_t desc_mn128(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// elu(x) + 1 (the linear-attention feature map)
__device__ __forceinline__ float phi_elu1(float x) { return x > 0.f ? x + 1.f : __expf(x); }

__device__ __forceinline__ void arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

// Column i of the weight half, summed over its rows (row i of the resident
// W^T slice [kb][Nh rows x 128 B]; the swizzle only permutes a row's pieces).
__device__ __forceinline__ float weight_colsum(const uint8_t* sW, int Nh, int nkb, int i) {
  float s = 0.f;
  for (int kb = 0; kb < nkb; ++kb) {
    const uint8_t* row = sW + ((size_t)kb * Nh + i) * 128u;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const uint4 q = *reinterpret_cast<const uint4*>(row + 16 * j);
      s += (bf16_lo(q.x) + bf16_hi(q.x)) + (bf16_lo(q.y) + bf16_hi(q.y)) + (bf16_lo(q.z) + bf16_hi(q.z)) +
           (bf16_lo(q.w) + bf16_hi(q.w));
    }
  }
  return s;
}
}  // namespace

template <int NKB, bool STATE>
__global__ void __launch_bounds__(kThreads, 1)
    ctxkv_kernel(const __grid_constant__ CUtensorMap tX, const __grid_constant__ CUtensorMap tW,
                 const __grid_constant__ CUtensorMap tO, const CtxKvParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  const int Nh = p.N / 2, d = p.d;
  const CtxKvLayout LY = ctxkv_layout(NKB * BK, p.N, STATE);
  constexpr int NRAW = STATE ? 1 : 2;                 // raw context buffers
  constexpr int NACC = STATE ? 1 : 2;                 // K/V accumulators in TMEM
  uint8_t* sW = smem;                                 // [kb][Nh rows x 128 B]
  float* wsum = reinterpret_cast<float*>(sW + LY.w_bytes);  // [Nh] column sums of the weight half
  float2* stats = reinterpret_cast<float2*>(wsum + 256);    // [NACC][128] (rstd, -rstd mu) per row
  uint8_t* sRaw = sW + LY.w_bytes + LY.aux_bytes;     // [NRAW buffers][kb]: the MMA's A operand
  uint8_t* sStg = sRaw + NRAW * (size_t)LY.raw_bytes;  // plain: [epilogue warp][kStgBufs][2 KB]; state: phi(K) tile, V tile
  uint64_t* bars = reinterpret_cast<uint64_t*>(sStg + LY.tail_bytes);
  uint64_t* w_full = bars;         // resident weight half loaded
  uint64_t* raw_full = bars + 1;   // [2] raw context block staged
  uint64_t* raw_empty = bars + 3;  // [2] the LayerNorm threads and the MMAs are done with it
  uint64_t* acc_full = bars + 7;   // [2] accumulator complete in TMEM
  uint64_t* acc_empty = bars + 9;  // [2] accumulator drained
  uint64_t* st_full = bars + 11;   // state mode: the state product of the tile complete
  uint64_t* stats_full = bars + 12;  // [2] row statistics of the tile written
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 16);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(w_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(raw_full + i, 1);
      mbar_init(raw_empty + i, 32 * kLnWarps + 1);  // + the MMA commit
      mbar_init(stats_full + i, 32 * kLnWarps);
      mbar_init(acc_full + i, 1);
      mbar_init(acc_empty + i, kEpiWarps);
    }
    mbar_init(st_full, 1);
    fence_mbar_init();
    prefetch_tmap(&tX);
    prefetch_tmap(&tW);
    prefetch_tmap(&tO);
  }
  // TMEM: K/V accumulator i at columns [256 i, 256 i + Nh); state mode: one
  // K/V accumulator at [0, Nh), the state product at [256, 384)
  if (warp == 0) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // CTA c: column half c % 2, row blocks c / 2, c / 2 + G, ... with G = gridDim.x / 2;
  // state mode: the row blocks of segments c / 2, c / 2 + G, ..., each segment's
  // C / 128 blocks in a row, so its state accumulates in TMEM
  const int half = blockIdx.x & 1, G = gridDim.x >> 1;
  const int nblk = (p.rows + BM - 1) / BM;
  const int first = blockIdx.x >> 1;
  const int Ts = STATE ? p.C / BM : 1;  // row blocks per segment
  auto tile_at = [&](int i) -> int {    // this CTA's i-th row block, -1 past the last
    const int seg = first + (i / Ts) * G;
    const int t = seg * Ts + i % Ts;
    return t < nblk ? t : -1;
  };
  const int n_off = half * Nh;  // this CTA's output columns
  // the weight is a parameter: its load may start before the dependency wait
  if (warp == 0 && lane == 0 && tile_at(0) >= 0) {
    mbar_arrive_expect_tx(w_full, LY.w_bytes);
    for (int kb = 0; kb < NKB; ++kb)
      for (int n0 = 0; n0 < Nh; n0 += BM)
        tma_load_2d(sW + (size_t)kb * Nh * (BK * 2) + (size_t)n0 * (BK * 2), &tW, kb * BK, n_off + n0, w_full);
  }
  pdl_trigger();
  pdl_wait();
  if (tile_at(0) < 0) {
    if (warp == 0) tmem_dealloc(tmem, 512);
    return;
  }

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA: raw context blocks ----------------
      int it = 0;
      for (int t = tile_at(it); t >= 0; t = tile_at(++it)) {
        const int rb = it % NRAW;
        if (it >= NRAW && !mbar_wait_bounded(raw_empty + rb, ((it / NRAW) - 1) & 1, p.status)) break;
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
      for (int t = tile_at(it); t >= 0 && ok; t = tile_at(++it)) {
        const int ab = it % NACC;
        if (it >= NACC && !mbar_wait_bounded(acc_empty + ab, ((it / NACC) - 1) & 1, p.status)) break;
        const int rb = it % NRAW;
        if (!mbar_wait_bounded(raw_full + rb, (it / NRAW) & 1, p.status)) break;
        tc_fence_after();
        const uint32_t dst = tmem + (uint32_t)(256 * ab);
        const uint64_t a0 = umma_desc_sw128(smem_u32(sRaw + (size_t)rb * LY.raw_bytes));
        const uint64_t w0 = umma_desc_sw128(smem_u32(sW));
#pragma unroll
        for (int kb = 0; kb < NKB; ++kb) {
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint64_t ah = desc_adv(a0, (uint32_t)kb * kPlane + kk * 32);
            const uint64_t wh = desc_adv(w0, (uint32_t)kb * (uint32_t)Nh * (BK * 2) + kk * 32);
            umma_bf16(dst, ah, wh, idesc, (kb | kk) != 0 ? 1u : 0u);
          }
        }
        umma_commit(raw_empty + rb);  // the raw block frees once these MMAs (and the statistics) are done
        umma_commit(acc_full + ab);
      }
    }
  } else if (warp < 2 + kLnWarps) {
    // ---------------- LayerNorm statistics: two threads per row ----------------
    // lanes l and l ^ 16 share row r; of each 64-column k block part 0 takes
    // the first four 16-byte pieces, part 1 the last four
    const int r = (warp - 2) * 16 + (lane & 15), part = lane >> 4;
    constexpr int kPieces = 4 * NKB;  // 16-byte pieces (8 columns) per thread
    int it = 0;
    for (int t = tile_at(it); t >= 0; t = tile_at(++it)) {
      const int rb = it % NRAW;
      if (!mbar_wait_bounded(raw_full + rb, (it / NRAW) & 1, p.status)) break;
      const uint8_t* raw = sRaw + (size_t)rb * LY.raw_bytes;
      // piece j of this thread: global piece g, column 8 g, 128-byte-swizzled
      // within its 64-column block
      auto gpiece = [&](int j) { return (j >> 2) * 8 + part * 4 + (j & 3); };
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
      // the statistics slot: the epilogue must be done with the tile it held
      const int sl = it % NACC;
      if (it >= NACC && !mbar_wait_bounded(acc_empty + sl, ((it / NACC) - 1) & 1, p.status)) break;
      if (part == 0) stats[sl * 128 + r] = make_float2(rstd, -mean * rstd);
      arrive(stats_full + sl);
      arrive(raw_empty + rb);
    }
  } else if constexpr (STATE) {
    // ---------------- epilogue, state mode ----------------
    const int ew = warp - 2 - kLnWarps;  // 0..7
    const int q = warp & 3;              // TMEM lane quadrant: tile rows 32 q .. 32 q + 31
    const int sub = ew >> 2;             // alternate 32-column chunks
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const int r = q * 32 + lane;         // this thread's row of the tile
    const int d = p.d, dh = p.dh, H = p.d / p.dh, l = half;
    const int SB = dh * dh + dh;
    uint8_t* sPK = sStg;                 // phi(K)[row][feature]: MN-major, two 64-feature atoms
    uint8_t* sPV = sStg + kStateTile;    // V[row][feature], then 16 feature columns of ones
    auto epi_sync = [&]() { asm volatile("bar.sync 5, 256;" ::: "memory"); };
    // d = 64: features 64..127 of the phi(K) operand stay zero
    if (d < 128) {
      for (int i = (ew * 32 + lane) * 16; i < (int)kStateTile; i += 256 * 16)
        if ((i / 16384) * 64 >= d) *reinterpret_cast<uint4*>(sPK + i) = make_uint4(0u, 0u, 0u, 0u);
    }
    // 16-byte piece of (row, feature m..m+7) in an MN-major tile
    auto piece = [&](int m) {
      return (uint32_t)(m >> 6) * 16384u + (uint32_t)r * 128u + ((((uint32_t)(m & 63) >> 3) ^ (uint32_t)(r & 7)) << 4);
    };
    // V features d .. d + 15 are ones (f16 1.0), so the state product's columns
    // d .. d + 15 accumulate z = sum over rows of phi(K), on the tensor core and
    // from the same f16 phi(K) as S
    if (sub == 0) {
      *reinterpret_cast<uint4*>(sPV + piece(d)) = make_uint4(0x3C003C00u, 0x3C003C00u, 0x3C003C00u, 0x3C003C00u);
      *reinterpret_cast<uint4*>(sPV + piece(d + 8)) = make_uint4(0x3C003C00u, 0x3C003C00u, 0x3C003C00u, 0x3C003C00u);
    }
    const uint32_t idesc = umma_idesc_f16(BM, d + 16) | (1u << 15) | (1u << 16);  // A and B MN-major
    const bool wok = mbar_wait_bounded(w_full, 0, p.status);
    if (wok && ew * 32 + lane < Nh) wsum[ew * 32 + lane] = weight_colsum(sW, Nh, NKB, ew * 32 + lane);
    epi_sync();
    int it = 0;
    for (int t = tile_at(it); t >= 0 && wok; t = tile_at(++it)) {
      const int pos = it % Ts;   // row block of the segment
      if (!mbar_wait_bounded(acc_full, it & 1, p.status)) break;
      if (!mbar_wait_bounded(stats_full, it & 1, p.status)) break;
      tc_fence_after();
      const float2 st = stats[r];  // rstd, -rstd mu of this thread's row
      for (int c = 32 * sub; c < 2 * d; c += 64) {
        float v[32];
        tmem_ld32(tmem + lane_off + (uint32_t)c, v);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = fmaf(st.x, v[i], st.y * wsum[c + i]);  // LN(x) W
        const bool isk = c < d;
        const int m0 = isk ? c : c - d;
        if (isk) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = phi_elu1(v[i]);
        }
        // the previous row block's state product must be done reading the operand tiles
        if (c < 64 && it > 0 && !mbar_wait_bounded(st_full, (it - 1) & 1, p.status)) break;
        uint8_t* buf = isk ? sPK : sPV;
#pragma unroll
        for (int j = 0; j < 4; ++j)
          *reinterpret_cast<uint4*>(buf + piece(m0 + 8 * j)) =
              make_uint4(pack_f16x2(v[8 * j], v[8 * j + 1]), pack_f16x2(v[8 * j + 2], v[8 * j + 3]),
                         pack_f16x2(v[8 * j + 4], v[8 * j + 5]), pack_f16x2(v[8 * j + 6], v[8 * j + 7]));
      }
      // the K/V accumulator is read: it may take the next tile
      tc_fence_before();
      __syncwarp();
      if (lane == 0) arrive(acc_empty);
      fence_async_shared();  // the operand tiles, visible to the tensor core
      epi_sync();
      if (ew == 0 && lane == 0) {
        tc_fence_after();
        const uint64_t ad = desc_mn128(smem_u32(sPK), 16384u), bd = desc_mn128(smem_u32(sPV), 16384u);
#pragma unroll
        for (int kk = 0; kk < BM / 16; ++kk)
          umma_bf16(tmem + 256u, desc_adv(ad, (uint32_t)kk * 16u * 128u), desc_adv(bd, (uint32_t)kk * 16u * 128u),
                    idesc, (kk != 0 || pos != 0) ? 1u : 0u);  // accumulate over the segment's row blocks
        umma_commit(st_full);
      }
      if (pos + 1 < Ts) continue;
      // the segment's last row block: its state, S of each head from the
      // diagonal blocks and z, stored (one segment per CTA pair: no atomics)
      if (!mbar_wait_bounded(st_full, it & 1, p.status)) break;
      tc_fence_after();
      const int seg = (t * BM) / p.C;
      float* st_seg = p.states + ((size_t)seg * 2 + l) * H * SB;
      const int m = 32 * q + lane;  // this lane's feature of K
      if (m < d && (sub == 0 || dh == 64)) {
        const int h = m / dh, i = m % dh, j0 = dh == 64 ? 32 * sub : 0;
        float sv[32];
        tmem_ld32(tmem + lane_off + 256u + (uint32_t)(h * dh + j0), sv);
        float* dst = st_seg + (size_t)h * SB + (size_t)i * dh + j0;
#pragma unroll
        for (int jj = 0; jj < 32; jj += 4)
          *reinterpret_cast<float4*>(dst + jj) = make_float4(sv[jj], sv[jj + 1], sv[jj + 2], sv[jj + 3]);
      }
      // z of feature m: column d of the state accumulator (any of the ones columns)
      if (sub == 0 && 32 * q < d) {
        float zz[16];
        tmem_ld16(tmem + lane_off + 256u + (uint32_t)d, zz);
        st_seg[(size_t)(m / dh) * SB + dh * dh + (m % dh)] = zz[0];
      }
      tc_fence_before();
      epi_sync();  // the state accumulator is read before the next segment's first product
    }
  } else {
    // ---------------- epilogue: TMEM -> f16 -> TMA stores ----------------
    const int ew = warp - 2 - kLnWarps;  // 0..7
    const int q = warp & 3;              // TMEM lane quadrant this warp may access
    const int sub = ew >> 2;             // alternate 32-column chunks
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    uint8_t* stg0 = sStg + (size_t)ew * kStgBufs * kStage;
    const int r = q * 32 + lane;  // this thread's row of the tile
    const bool wok = mbar_wait_bounded(w_full, 0, p.status);
    if (wok && ew * 32 + lane < Nh) wsum[ew * 32 + lane] = weight_colsum(sW, Nh, NKB, ew * 32 + lane);
    asm volatile("bar.sync 5, 256;" ::: "memory");  // the eight epilogue warps: column sums written
    int nstore = 0;
    int it = 0;
    for (int t = tile_at(it); t >= 0 && wok; t = tile_at(++it)) {
      const int ab = it & 1;
      if (!mbar_wait_bounded(acc_full + ab, (it >> 1) & 1, p.status)) break;
      if (!mbar_wait_bounded(stats_full + ab, (it >> 1) & 1, p.status)) break;
      tc_fence_after();
      const float2 st = stats[ab * 128 + r];  // rstd, -rstd mu of this thread's row
      const int srow = t * BM + q * 32;
      for (int c = 32 * sub; c < Nh; c += 64) {
        float v[32];
        tmem_ld32(tmem + lane_off + (uint32_t)(256 * ab + c), v);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = fmaf(st.x, v[i], st.y * wsum[c + i]);  // LN(x) W
        // rotating staging buffers: the one written kStgBufs stores ago must have been read
        uint8_t* b = stg0 + (size_t)(nstore % kStgBufs) * kStage;
        if (lane == 0 && nstore >= kStgBufs)
          asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(kStgBufs - 1) : "memory");
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

  __syncwarp();  // each warp arrives whole: single lanes ran the producer and MMA loops
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
  return ctxkv_layout(d_pad, N, false).smem <= kSmemMaxBlock;
}

bool ctxkv_state_supported(int d, int d_pad, int N, int dh, int C) {
  if (d != 64 && d != 128) return false;
  if (N != 4 * d) return false;  // two layers: each column half is one layer's [K | V]
  if (dh != 32 && dh != 64) return false;
  if (C <= 0 || C % BM) return false;  // a 128-row tile lies in one segment
  return ctxkv_layout(d_pad, N, true).smem <= kSmemMaxBlock;
}

cudaError_t ctxkv_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_ctxkv_sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(ctxkv_kernel<1, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMaxBlock);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(ctxkv_kernel<2, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMaxBlock);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(ctxkv_kernel<1, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMaxBlock);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(ctxkv_kernel<2, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMaxBlock);
  return e;
}

cudaError_t ctxkv_launch(const CUtensorMap* x, const CUtensorMap* w, const CUtensorMap* o, int d_pad,
                         const CtxKvParams& p, cudaStream_t s) {
  if (p.rows <= 0) return cudaSuccess;
  const bool state = p.states != nullptr;
  const CtxKvLayout LY = ctxkv_layout(d_pad, p.N, state);
  const long long nblk = (p.rows + BM - 1) / BM;
  // an even grid: CTA pairs (2i, 2i+1) take the two column halves of the same row blocks
  long long grid = g_ctxkv_sms > 0 ? g_ctxkv_sms : 148;
  if (grid > 2 * nblk) grid = 2 * nblk;
  grid &= ~1LL;
  const dim3 g((unsigned)grid), b(kThreads);
  if (state)
    return d_pad > BK ? launch_k(ctxkv_kernel<2, true>, g, b, LY.smem, s, *x, *w, *o, p)
                      : launch_k(ctxkv_kernel<1, true>, g, b, LY.smem, s, *x, *w, *o, p);
  return d_pad > BK ? launch_k(ctxkv_kernel<2, false>, g, b, LY.smem, s, *x, *w, *o, p)
                    : launch_k(ctxkv_kernel<1, false>, g, b, LY.smem, s, *x, *w, *o, p);
}

}  // namespace fe
