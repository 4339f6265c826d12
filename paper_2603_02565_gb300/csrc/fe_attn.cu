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
//   tcgen05.mma   : S_j = Q K_j^T into TMEM tile j % 3 (three S/P tiles let
//                   S_{j+1} and S_{j+2} run ahead of PV_j), and PV_j = P_j V_j
//                   with P_j read from the same TMEM tile, accumulated into the
//                   unit's output accumulator in TMEM (two, alternating by
//                   unit).  One commit per PV_j, on the K/V stage's empty
//                   barrier, tells every role that PV_j is complete.  Each
//                   tcgen05.mma costs its issuing thread a fixed latency
//                   (about 45 ns, whatever N), so a CTA that walks many chunks
//                   issues S from warp 1 and PV from warp 2 (SPLIT); a short
//                   launch keeps one issuer (warp 1) and one warp fewer
//   the other 8   : online softmax from TMEM, one query row per lane; warps
//                   w and w+4 share TMEM lane quadrant w % 4 and each take
//                   half of the chunk's keys and half of the output columns
//                   (row maxima and sums exchanged through shared memory).
//                   P_j is written back over S_j as f16 against a running
//                   maximum that moves only when a chunk exceeds it by more
//                   than 8 (log2 units), when the output accumulator is
//                   rescaled in TMEM; otherwise the softmax never reads the PV
//                   products until the unit's output is stored (for d_h = 64
//                   staged through shared memory, so that the stores write
//                   whole rows)
// Q, K, V and P are single f16 planes (unit roundoff 2^-11; Q and K come
// from LayerNorm'd rows times weights of magnitude well inside the f16
// range, P lies in [0, 2^8]); accumulation, softmax statistics and the output
// are fp32, the output leaves as a bf16 hi/lo pair.
#include <cstdlib>

#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {

constexpr int BQ = 128;     // query rows per unit (TMEM lanes)

// d_h = 32: 64-key chunks, 32 keys per softmax warp, small enough for two CTAs per SM.
// d_h = 64: 128-key chunks and 8 softmax warps (two per TMEM lane quadrant).
template <int DH>
struct AttnCfg {
  static constexpr int CK = DH == 32 ? 64 : 128;                // keys per chunk
  static constexpr int kSoftmaxWarps = 8;
  static constexpr int kHalves = kSoftmaxWarps / 4;              // warps sharing one lane quadrant
  static_assert(kHalves == 2, "two softmax warps per TMEM lane quadrant");
  static constexpr int KW = CK / kHalves;                        // keys per softmax warp and chunk
  static constexpr int kCtasPerSM = DH == 32 ? 2 : 1;
  // TMEM: S/P tiles at [t CK, t CK + CK), t < 3; the output accumulators of
  // consecutive units (alternating) at [3CK, 3CK + 2DH)
  static constexpr int kTiles = 3;
  static constexpr uint32_t kTmemCols = DH == 32 ? 256 : 512;
  static_assert(kTiles * CK + 2 * DH <= (int)kTmemCols, "TMEM budget");
  static constexpr uint32_t kRowBytes = DH * 2;                 // one row of a Q/K/V tile
  static constexpr uint32_t kQBytes = 128 * kRowBytes;          // Q tile: 128 rows
  static constexpr uint32_t kKVTile = CK * kRowBytes;           // K or V chunk: CK rows
  static constexpr uint32_t kSwz = DH == 32 ? 4u : 2u;          // descriptor swizzle code (64 B / 128 B)
  static constexpr uint32_t kSbo = 8 * kRowBytes;               // 8-row swizzle atom
  static constexpr uint32_t kKVBytes = 2 * kKVTile;             // K, V
  static constexpr int kKVStages = DH == 32 ? 8 : 4;
  static constexpr uint32_t kRed = 2 * 2 * 2 * 128 * 4;       // [max|sum][parity][half][row]
  // output staging for d_h = 64, per TMEM lane quadrant: [plane hi|lo][32 rows][NC 16-byte chunks]
  // (for d_h = 32 the direct stores measured faster: 32-byte row pieces, and
  // the unit's end waits on its last PV anyway)
  static constexpr bool kStageOut = DH == 64;
  static constexpr int NC = DH / 8;                            // 16-byte chunks in a row of one plane
  static constexpr uint32_t kStageQuad = kStageOut ? 2 * 32 * NC * 16 : 0;
  static constexpr size_t kSmem = 1024 + 2 * kQBytes + kKVStages * kKVBytes + 256 + kRed + 4 * kStageQuad;
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

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// maximum of 32 values as a tree of three-input maxima
__device__ __forceinline__ float max32(const float* v) {
  float a[11];
#pragma unroll
  for (int i = 0; i < 10; ++i) a[i] = max3f(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
  a[10] = fmaxf(v[30], v[31]);
  return fmaxf(max3f(max3f(a[0], a[1], a[2]), max3f(a[3], a[4], a[5]), max3f(a[6], a[7], a[8])),
               fmaxf(a[9], a[10]));
}

// Non-blocking probe of an mbarrier phase, for waits that are normally
// already satisfied when reached (the issuer's K/V and tile checks).
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_wait_ready(uint64_t* bar, uint32_t parity, int* status) {
  if (mbar_test(bar, parity)) return true;
  return mbar_wait_slow(bar, parity, status);
}

__device__ __forceinline__ void mbar_arrive1(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Unit cursor: unit u -> (segment b, head h, query tile t); query tile fastest.
// Every role walks its CTA's units u = blockIdx.x + i * gridDim.x and skips
// tiles that start past their segment's end.  The position of u + gridDim.x
// follows from that of u by adding gridDim.x's digits in the same mixed radix
// (tiles, heads), kept in shared memory, so that a role moving to its next
// unit does not divide (an integer division is a long serial chain on the
// issuing thread, whose pace sets the kernel's).  The segment count and offset
// of the next candidate unit are loaded one unit ahead, so a role crossing into
// its next unit does not wait on a global load.
struct Cursor {
  int u, b, h, q0, qcnt, qoff;
  int pcnt, poff;  // q_cnt / q_off of unit u + gridDim.x
};

// (b, h, q0) += the digits of gridDim.x (step[0..2] = segments, heads, tiles)
__device__ __forceinline__ void pos_add(const AttnParams& p, const int* step, int& b, int& h, int& q0) {
  int t = (q0 / BQ) + step[2];
  int c = t >= p.max_q_tiles ? 1 : 0;
  q0 = (t - c * p.max_q_tiles) * BQ;
  h += step[1] + c;
  c = h >= p.n_heads ? 1 : 0;
  h -= c * p.n_heads;
  b += step[0] + c;
}

__device__ __forceinline__ void pos_of(const AttnParams& p, int u, int& b, int& h, int& q0) {
  b = u / (p.max_q_tiles * p.n_heads);
  h = (u / p.max_q_tiles) % p.n_heads;
  q0 = (u % p.max_q_tiles) * BQ;
}

__device__ __forceinline__ void cur_fetch(const AttnParams& p, int b, int& cnt, int& off) {
  cnt = p.q_cnt_dev ? __ldg(p.q_cnt_dev + b) : p.q_cnt_fixed;
  off = p.q_off_dev ? __ldg(p.q_off_dev + b) : b * p.q_stride;
}

// settle on the first unit at or after c.u whose tile holds query rows, then
// load the counts of the unit after it
__device__ __forceinline__ void cur_settle(const AttnParams& p, const int* step, int units, Cursor& c) {
  while (c.u < units && c.q0 >= c.qcnt) {
    c.u += gridDim.x;
    if (c.u < units) {
      pos_add(p, step, c.b, c.h, c.q0);
      cur_fetch(p, c.b, c.qcnt, c.qoff);
    }
  }
  if (c.u < units && c.u + (int)gridDim.x < units) {
    int nb = c.b, nh = c.h, nq = c.q0;
    pos_add(p, step, nb, nh, nq);
    cur_fetch(p, nb, c.pcnt, c.poff);
  }
}

__device__ __forceinline__ void cur_first(const AttnParams& p, const int* step, int units, Cursor& c) {
  c.u = blockIdx.x;
  pos_of(p, c.u, c.b, c.h, c.q0);
  cur_fetch(p, c.b, c.qcnt, c.qoff);
  cur_settle(p, step, units, c);
}

__device__ __forceinline__ void cur_next(const AttnParams& p, const int* step, int units, Cursor& c) {
  c.u += gridDim.x;
  if (c.u >= units) return;
  pos_add(p, step, c.b, c.h, c.q0);
  c.qcnt = c.pcnt;
  c.qoff = c.poff;
  cur_settle(p, step, units, c);
}

}  // namespace

// Zero bytes [o0, end) of a shared-memory tile (one thread, 16-byte stores),
// then order the writes before this thread's next tensor-core operations.
__device__ __noinline__ void zero_tail(uint8_t* t, int o0, int end) {
  for (int o = o0; o < end; o += 16) *reinterpret_cast<uint4*>(t + o) = make_uint4(0u, 0u, 0u, 0u);
  fence_async_shared();
}

// Warps ahead of the softmax warps: the producer and one MMA issuer, or the
// producer and separate S and PV issuers.
template <bool SPLIT>
__host__ __device__ constexpr int attn_role_warps() { return SPLIT ? 3 : 2; }
template <int DH, bool SPLIT>
__host__ __device__ constexpr int attn_threads() { return 32 * (attn_role_warps<SPLIT>() + AttnCfg<DH>::kSoftmaxWarps); }

template <int DH, bool SPLIT>
__global__ void __launch_bounds__(attn_threads<DH, SPLIT>(), AttnCfg<DH>::kCtasPerSM)
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
  uint64_t* kv_empty = bars + 12; // [stages] PV_j (and everything issued before it) complete
  uint64_t* s_full = bars + 20;     // [3] S_j complete in TMEM tile j % 3
  uint64_t* p_full = bars + 23;     // [3] P_j written over S_j
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 26);
  int* step = reinterpret_cast<int*>(bars + 27);  // digits of gridDim.x: segments, heads, query tiles
  float* red = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);  // row-statistic exchange
  uint8_t* stage = reinterpret_cast<uint8_t*>(bars) + 256 + Cfg::kRed;             // output staging

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qtiles = p.max_q_tiles;
  const int units = p.n_segments * p.n_heads * qtiles;
  // keys of a unit's segment: a fixed count at a fixed stride, or, for
  // self-attention within segments, the segment's own query rows
  auto kv_count = [&](const Cursor& c) { return p.kv_self ? c.qcnt : p.kv_cnt; };
  auto kv_base = [&](const Cursor& c) { return p.kv_self ? c.qoff : c.b * p.kv_stride; };
  auto chunks = [&](const Cursor& c) { return (kv_count(c) + CK - 1) / CK; };
  if ((int)blockIdx.x >= units) return;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(q_full + i, 1);
      mbar_init(q_empty + i, 1);
    }
    for (int i = 0; i < Cfg::kTiles; ++i) {
      mbar_init(s_full + i, 1);
      mbar_init(p_full + i, 32 * Cfg::kSoftmaxWarps);
    }
    for (int i = 0; i < Cfg::kKVStages; ++i) {
      mbar_init(kv_full + i, 1);
      mbar_init(kv_empty + i, 1);
    }
    fence_mbar_init();
    pos_of(p, (int)gridDim.x, step[0], step[1], step[2]);
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

  // Two CTAs share an SM in the d_h = 32 launches, and a grid of two per SM
  // places the second half of the grid second on each SM: there the role warps
  // rotate (one issuer: producer and issuer swap; two issuers: producer, S and
  // PV issuers move to warps 2, 0, 1), so that the two CTAs' issuing threads
  // sit on different SM sub-partitions (warp w runs on sub-partition w % 4)
  // instead of competing for one's issue slots
  const bool second = Cfg::kCtasPerSM == 2 && (int)blockIdx.x >= (int)(gridDim.x >> 1);
  const int w_prod = second ? (SPLIT ? 2 : 1) : 0;
  const int w_mma = second ? 0 : 1;             // one issuer; with two, the S issuer
  const int w_pv = second ? 1 : 2;              // two issuers: the PV issuer
  if (warp == w_prod) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int ui = 0, gc = 0;
      bool ok = true;
      Cursor c;
      for (cur_first(p, step, units, c); c.u < units && ok; cur_next(p, step, units, c)) {
        const int qb = ui & 1;
        if (ui >= 2 && !mbar_wait_compact(q_empty + qb, ((ui >> 1) - 1) & 1, p.status)) break;
        uint8_t* q = sQ + qb * Cfg::kQBytes;
        mbar_arrive_expect_tx(q_full + qb, Cfg::kQBytes);
        tma_load_2d(q, &tQ, p.q_col + c.h * DH, c.qoff + c.q0, q_full + qb);
        const int nch = chunks(c);
        for (int j = 0; j < nch; ++j, ++gc) {
          const int ks = gc % Cfg::kKVStages;
          if (gc >= Cfg::kKVStages &&
              !mbar_wait_compact(kv_empty + ks, ((gc / Cfg::kKVStages) - 1) & 1, p.status)) {
            ok = false;
            break;
          }
          uint8_t* kv = sKV + ks * Cfg::kKVBytes;
          const int row = kv_base(c) + j * CK;
          mbar_arrive_expect_tx(kv_full + ks, Cfg::kKVBytes);
          if (p.kv3d) {  // head-major K/V: one contiguous block per head
            tma_load_3d(kv, &tK, 0, row, (p.k_col + c.h * DH) / DH, kv_full + ks);
            tma_load_3d(kv + Cfg::kKVTile, &tV, 0, row, (p.v_col + c.h * DH) / DH, kv_full + ks);
          } else {
            tma_load_2d(kv, &tK, p.k_col + c.h * DH, row, kv_full + ks);
            if (p.kv_seg)  // rows past the segment's kv_cnt keys are outside the map: zeros
              tma_load_3d(kv + Cfg::kKVTile, &tV, p.v_col + c.h * DH, j * CK, c.b, kv_full + ks);
            else
              tma_load_2d(kv + Cfg::kKVTile, &tV, p.v_col + c.h * DH, row, kv_full + ks);
          }
        }
        ++ui;
      }
    }
  } else if (!SPLIT && warp == w_mma) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      // The chunks of all this CTA's units form one stream g = 0, 1, ...;
      // S_{g+1} is issued before PV_g, across unit boundaries too, so the
      // softmax finds the next unit's first S ready when it gets there.  The
      // loop is this one thread's serial path and sets the pace of the
      // kernel: running indices instead of divisions, descriptors as a base
      // plus an offset, and one commit per product.
      constexpr int NS = Cfg::kKVStages;
      static_assert((NS & (NS - 1)) == 0, "K/V stages: a power of two");
      const uint32_t idesc_s = umma_idesc_f16(BQ, CK);
      const uint32_t idesc_pv = umma_idesc_f16(BQ, DH) | (1u << 16);  // B (V) is MN-major
      // only a variable key count or one that is not a multiple of CK leaves a
      // partial chunk, whose V rows a segmented map already reads as zeros
      const bool pad_v = p.kv_self || (p.kv_cnt % CK != 0 && !p.kv_seg);
      const uint64_t qd0 = desc_sw(smem_u32(sQ), Cfg::kSbo, Cfg::kSwz);
      const uint64_t kd0 = desc_sw(smem_u32(sKV), Cfg::kSbo, Cfg::kSwz);
      Cursor sc;             // unit of the next S
      int sj = 0, sui = 0;   // its chunk and its unit counter (Q buffer sui % 2)
      int s_nch = 0;         // that unit's chunk count
      int g_s = 0;           // S products issued
      int t_s = 0;           // TMEM tile of the next S (g_s % 3)
      // per chunk g (g % 4; at most two chunks separate S and PV): its unit
      // counter's parity (the output accumulator) and whether it opens the unit
      uint32_t pv_info = 0;
      cur_first(p, step, units, sc);
      if (sc.u < units) s_nch = chunks(sc);
      // S = Q K^T of the chunk at the S cursor into TMEM tile t_s, then advance the cursor
      auto issue_next_s = [&]() -> bool {
        if (sc.u >= units) return true;
        const int qb = sui & 1;
        if (sj == 0 && !mbar_wait_compact(q_full + qb, (sui >> 1) & 1, p.status)) return false;
        // the tile is free once PV_{g_s-3}, which reads P_{g_s-3} from it, has completed
        if (g_s >= Cfg::kTiles) {
          const int gp = g_s - Cfg::kTiles;
          if (!mbar_wait_ready(kv_empty + (gp & (NS - 1)), (uint32_t)(gp / NS) & 1u, p.status)) return false;
        }
        const int ks = g_s & (NS - 1);
        if (!mbar_wait_ready(kv_full + ks, (uint32_t)(g_s / NS) & 1u, p.status)) return false;
        tc_fence_after();
        const uint32_t dst = tmem + (uint32_t)(t_s * CK);
        const uint64_t qd = qd0 + (uint64_t)((qb * Cfg::kQBytes) >> 4);
        const uint64_t kd = kd0 + (uint64_t)((ks * Cfg::kKVBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk)
          umma_bf16(dst, qd + (uint64_t)(kk * 2), kd + (uint64_t)(kk * 2), idesc_s, kk != 0 ? 1u : 0u);
        umma_commit(s_full + t_s);
        pv_info = (pv_info & ~(3u << (2 * (g_s & 3)))) | ((uint32_t)(((sui & 1) << 1) | (sj == 0 ? 1 : 0)) << (2 * (g_s & 3)));
        // The V rows of a partial chunk past the key count belong to the next
        // segment: their P is 0, but 0 x NaN is NaN, so they are zeroed here
        // (the chunk has landed; PV_{g_s}, issued later by this thread, reads them)
        if (pad_v) {
          const int kval = kv_count(sc) - sj * CK;
          if (kval < CK) zero_tail(sKV + ks * Cfg::kKVBytes + Cfg::kKVTile, kval * (int)Cfg::kRowBytes, (int)Cfg::kKVTile);
        }
        ++g_s;
        t_s = t_s == Cfg::kTiles - 1 ? 0 : t_s + 1;
        if (++sj == s_nch) {  // every S of this unit issued: its Q buffer frees on completion
          umma_commit(q_empty + qb);
          sj = 0;
          ++sui;
          cur_next(p, step, units, sc);
          if (sc.u < units) s_nch = chunks(sc);
        }
        return true;
      };
      bool ok = issue_next_s();
      int t = 0;
      uint32_t p_par = 0;  // parity of P_g's phase on p_full[t]: (g / 3) & 1
      for (int g = 0; ok && g < g_s; ++g) {
        if (!issue_next_s()) break;
        if (!mbar_wait_compact(p_full + t, p_par, p.status)) break;
        tc_fence_after();
        // PV_g: A = P_g from TMEM tile g % 3, each softmax warp's KW keys as
        // KW/2 columns of f16 pairs at the start of its KW S columns
        const int ks = g & (NS - 1);
        const uint64_t vd = kd0 + (uint64_t)((ks * Cfg::kKVBytes + Cfg::kKVTile) >> 4);
        const uint32_t pt = tmem + (uint32_t)(t * CK);
        // PV accumulates into the unit's output accumulator (unit parity), from zero at its first chunk
        const uint32_t info = (pv_info >> (2 * (g & 3))) & 3u;
        const uint32_t dst = tmem + (uint32_t)(Cfg::kTiles * CK + (int)(info >> 1) * DH);
#pragma unroll
        for (int kk = 0; kk < CK / 16; ++kk)
          umma_bf16_tmem_a(dst, pt + (uint32_t)((kk / (Cfg::KW / 16)) * Cfg::KW + (kk % (Cfg::KW / 16)) * 8),
                           vd + (uint64_t)((kk * 16 * Cfg::kRowBytes) >> 4), idesc_pv,
                           (kk != 0 || !(info & 1u)) ? 1u : 0u);
        umma_commit(kv_empty + ks);
        if (++t == Cfg::kTiles) {
          t = 0;
          p_par ^= 1u;
        }
      }
    }
  } else if (SPLIT && warp == w_mma) {
    if (lane == 0) {
      // ---------------- S issuer ----------------
      // The chunks of all this CTA's units form one stream g = 0, 1, ...; S_g
      // goes into TMEM tile g % 3 as soon as its K chunk has landed and PV_{g-3}
      // has released the tile, across unit boundaries too, so the softmax finds
      // the next S ready when it gets there.  Running indices and descriptors
      // as a base plus an offset keep this thread's serial path short.
      constexpr int NS = Cfg::kKVStages;
      static_assert((NS & (NS - 1)) == 0, "K/V stages: a power of two");
      const uint32_t idesc_s = umma_idesc_f16(BQ, CK);
      const uint64_t qd0 = desc_sw(smem_u32(sQ), Cfg::kSbo, Cfg::kSwz);
      const uint64_t kd0 = desc_sw(smem_u32(sKV), Cfg::kSbo, Cfg::kSwz);
      int g_s = 0, t_s = 0, sui = 0;
      Cursor sc;
      bool ok = true;
      for (cur_first(p, step, units, sc); sc.u < units && ok; cur_next(p, step, units, sc)) {
        const int qb = sui & 1;
        if (!mbar_wait_compact(q_full + qb, (sui >> 1) & 1, p.status)) break;
        const uint64_t qd = qd0 + (uint64_t)((qb * Cfg::kQBytes) >> 4);
        const int nch = chunks(sc);
        for (int j = 0; j < nch; ++j) {
          // the tile is free once PV_{g_s-3}, which reads P_{g_s-3} from it, has completed
          if (g_s >= Cfg::kTiles) {
            const int gp = g_s - Cfg::kTiles;
            if (!mbar_wait_ready(kv_empty + (gp & (NS - 1)), (uint32_t)(gp / NS) & 1u, p.status)) {
              ok = false;
              break;
            }
          }
          const int ks = g_s & (NS - 1);
          if (!mbar_wait_ready(kv_full + ks, (uint32_t)(g_s / NS) & 1u, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t dst = tmem + (uint32_t)(t_s * CK);
          const uint64_t kd = kd0 + (uint64_t)((ks * Cfg::kKVBytes) >> 4);
#pragma unroll
          for (int kk = 0; kk < DH / 16; ++kk)
            umma_bf16(dst, qd + (uint64_t)(kk * 2), kd + (uint64_t)(kk * 2), idesc_s, kk != 0 ? 1u : 0u);
          umma_commit(s_full + t_s);
          ++g_s;
          t_s = t_s == Cfg::kTiles - 1 ? 0 : t_s + 1;
        }
        if (!ok) break;
        umma_commit(q_empty + qb);  // every S of this unit issued: its Q buffer frees on completion
        ++sui;
      }
    }
  } else if (SPLIT && warp == w_pv) {
    if (lane == 0) {
      // ---------------- PV issuer ----------------
      // PV_g = P_g V_g, P_g read from TMEM tile g % 3 once the softmax has
      // written it, accumulated into the unit's output accumulator (two,
      // alternating by unit), from zero at the unit's first chunk.  One commit
      // per product, on the K/V stage's empty barrier, tells every role that
      // PV_g is complete: the producer may refill the stage, the S issuer may
      // write S_{g+3} over P_g, the softmax may rescale or read the output.
      constexpr int NS = Cfg::kKVStages;
      const uint32_t idesc_pv = umma_idesc_f16(BQ, DH) | (1u << 16);  // B (V) is MN-major
      // only a variable key count or one that is not a multiple of CK leaves a
      // partial chunk, whose V rows a segmented map already reads as zeros
      const bool pad_v = p.kv_self || (p.kv_cnt % CK != 0 && !p.kv_seg);
      const uint64_t vd0 = desc_sw(smem_u32(sKV + Cfg::kKVTile), Cfg::kSbo, Cfg::kSwz);
      int g = 0, t = 0, ui = 0;
      uint32_t p_par = 0;  // parity of P_g's phase on p_full[t]: (g / 3) & 1
      Cursor c;
      bool ok = true;
      for (cur_first(p, step, units, c); c.u < units && ok; cur_next(p, step, units, c)) {
        const uint32_t dst = tmem + (uint32_t)(Cfg::kTiles * CK + (ui & 1) * DH);
        const int nch = chunks(c);
        for (int j = 0; j < nch; ++j, ++g) {
          if (!mbar_wait_compact(p_full + t, p_par, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int ks = g & (NS - 1);
          // The V rows of a partial chunk past the key count belong to the
          // next segment: their P is 0, but 0 x NaN is NaN, so they are zeroed
          // (the chunk landed before S_g, which P_g follows)
          if (pad_v) {
            const int kval = kv_count(c) - j * CK;
            if (kval < CK) zero_tail(sKV + ks * Cfg::kKVBytes + Cfg::kKVTile, kval * (int)Cfg::kRowBytes, (int)Cfg::kKVTile);
          }
          // A = P_g from the tile: each softmax warp's KW keys as KW/2 columns
          // of f16 pairs at the start of its KW S columns
          const uint64_t vd = vd0 + (uint64_t)((ks * Cfg::kKVBytes) >> 4);
          const uint32_t pt = tmem + (uint32_t)(t * CK);
#pragma unroll
          for (int kk = 0; kk < CK / 16; ++kk)
            umma_bf16_tmem_a(dst, pt + (uint32_t)((kk / (Cfg::KW / 16)) * Cfg::KW + (kk % (Cfg::KW / 16)) * 8),
                             vd + (uint64_t)((kk * 16 * Cfg::kRowBytes) >> 4), idesc_pv,
                             (kk != 0 || j != 0) ? 1u : 0u);
          umma_commit(kv_empty + ks);
          if (++t == Cfg::kTiles) {
            t = 0;
            p_par ^= 1u;
          }
        }
        ++ui;
      }
    }
  } else {
    // ---------------- softmax / output (the last eight warps) ----------------
    constexpr int DO = DH / Cfg::kHalves;  // output columns per warp
    constexpr int KW = Cfg::KW;            // keys per warp and chunk (32 for d_h = 32, 64 for d_h = 64)
    const int sw = warp - attn_role_warps<SPLIT>();
    const int q4 = warp & 3;
    const int half = sw >> 2;     // keys [KW half, KW half + KW) of each chunk, output columns [DO half, DO half + DO)
    const int r = q4 * 32 + lane; // query row of the tile = TMEM lane
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    float* red_max = red;         // [parity][half][128]
    float* red_sum = red + 512;
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + q4) : "memory"); };
    // this warp's DO columns of the output accumulator of unit counter ui
    auto o_cols = [&](int ui) {
      return tmem + lane_off + (uint32_t)(Cfg::kTiles * CK + (ui & 1) * DH + half * DO);
    };
    // o (this warp's DO columns, DO = 16 or 32) from / to TMEM
    auto o_load = [&](uint32_t a, float* o) {
      if constexpr (DO == 16)
        tmem_ld16(a, o);
      else
        tmem_ld32(a, o);
    };
    // the finished unit whose output is still to be normalised and stored
    struct Done {
      int h, q0, qcnt, qoff, ui, g;  // g: its last chunk
      float l;
      bool active;
    } dn{};
    bool have_done = false;
    // once the unit's last PV has completed: O / l (l summed over both key
    // halves) as a split pair.  Each lane holds one query row.  For d_h = 64
    // the two warps of a lane quadrant stage their halves of the quadrant's
    // 32 rows in shared memory (16-byte chunks XOR-swizzled by row: no bank
    // conflicts on either side) and then each stores one plane, a lane per
    // chunk, so that a warp instruction writes whole 128-byte rows instead of
    // touching 32 rows
    constexpr int NC = Cfg::NC;
    auto swz = [](int row) { return NC == 8 ? (row & 7) : ((row >> 1) & 3); };
    auto finish = [&]() -> bool {
      float* rs = red_sum + (dn.ui & 1) * 256;
      rs[half * 128 + r] = dn.l;
      pair_sync();
      const float ltot = rs[r] + rs[128 + r];
      if (!dn.active) return true;
      // with staging, both warps of the pair meet at the second barrier below, also after a timed-out wait
      const bool okw = mbar_wait_compact(kv_empty + (dn.g % Cfg::kKVStages),
                                         (uint32_t)(dn.g / Cfg::kKVStages) & 1u, p.status);
      if constexpr (!Cfg::kStageOut) {
        if (!okw) return false;
        tc_fence_after();
        float o[DO];
        o_load(o_cols(dn.ui), o);
        if (dn.q0 + r < dn.qcnt) {
          const float inv = 1.f / ltot;
          const size_t go = (size_t)(dn.qoff + dn.q0 + r) * p.ldo + p.o_col + dn.h * DH + half * DO;
#pragma unroll
          for (int c = 0; c < DO; c += 8) {
            uint32_t hi[4], lo[4];
#pragma unroll
            for (int i = 0; i < 8; i += 2) split2(o[c + i] * inv, o[c + i + 1] * inv, hi[i / 2], lo[i / 2]);
            *reinterpret_cast<uint4*>(p.o_h + go + c) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
            *reinterpret_cast<uint4*>(p.o_l + go + c) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
          }
        }
        return true;
      } else {
        uint8_t* st = stage + q4 * Cfg::kStageQuad;
        if (okw) {
          tc_fence_after();
          float o[DO];
          o_load(o_cols(dn.ui), o);
          const float inv = 1.f / ltot;
#pragma unroll
          for (int c = 0; c < DO; c += 8) {
            uint32_t hi[4], lo[4];
#pragma unroll
            for (int i = 0; i < 8; i += 2) split2(o[c + i] * inv, o[c + i + 1] * inv, hi[i / 2], lo[i / 2]);
            const int pc = (half * (DO / 8) + c / 8) ^ swz(lane);
            *reinterpret_cast<uint4*>(st + (lane * NC + pc) * 16) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
            *reinterpret_cast<uint4*>(st + ((32 + lane) * NC + pc) * 16) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
          }
        }
        pair_sync();
        if (!okw) return false;
        // warp `half` stores plane `half` (hi, lo) of the quadrant's rows
        const uint8_t* src = st + half * 32 * NC * 16;
        bf16* dst = half ? p.o_l : p.o_h;
        const int row0 = dn.q0 + q4 * 32;
#pragma unroll
        for (int i = 0; i < NC; ++i) {
          const int idx = i * 32 + lane;
          const int row = idx / NC, ch = idx % NC;
          if (row0 + row < dn.qcnt) {
            const uint4 v = *reinterpret_cast<const uint4*>(src + (row * NC + (ch ^ swz(row))) * 16);
            *reinterpret_cast<uint4*>(dst + (size_t)(dn.qoff + row0 + row) * p.ldo + p.o_col + dn.h * DH + ch * 8) = v;
          }
        }
        return true;
      }
    };
    int gc = 0, ui = 0;
    bool ok = true;
    Cursor c;
    for (cur_first(p, step, units, c); c.u < units && ok; cur_next(p, step, units, c)) {
      // the running maximum m that P is taken against moves only when a chunk's
      // maximum exceeds it by more than kSlack (log2 units; P <= 2^kSlack stays
      // far inside f16), and then the unit's output accumulator in TMEM is
      // rescaled: most chunks need no correction at all
      constexpr float kSlack = 8.f;
      float m = -INFINITY, l = 0.f;
      // a warp whose 32 query rows all lie past the segment's end only keeps
      // the barrier protocol; those rows of P and of the output are never used
      const bool active = c.q0 + q4 * 32 < c.qcnt;
      const int nch = chunks(c);
      for (int j = 0; j < nch; ++j, ++gc) {
        const int t = gc % Cfg::kTiles;
        if (!mbar_wait_compact(s_full + t, (gc / Cfg::kTiles) & 1, p.status)) {
          ok = false;
          break;
        }
        if (active) {
          tc_fence_after();
          const uint32_t tile = tmem + lane_off + (uint32_t)(t * CK + half * KW);
          float v[KW];
          if constexpr (KW == 64)
            tmem_ld64(tile, v);
          else
            tmem_ld32(tile, v);
          // keys past kv_cnt take no part: -inf gives them P = 0
          const int kvalid = kv_count(c) - j * CK - half * KW;  // valid keys among this warp's KW
          if (kvalid < KW) {
#pragma unroll
            for (int i = 0; i < KW; ++i)
              if (i >= kvalid) v[i] = -INFINITY;
          }
          float mx = max32(v);
          if constexpr (KW == 64) mx = fmaxf(mx, max32(v + 32));
          mx *= p.scale_log2;
          if (Cfg::kHalves == 2) {
            float* rm = red_max + (gc & 1) * 256;
            rm[half * 128 + r] = mx;
            pair_sync();
            mx = fmaxf(rm[r], rm[128 + r]);
          }
          if (j == 0) {
            m = mx;  // the unit's first PV overwrites the accumulator
          } else {
            const bool up = mx > m + kSlack;
            if (__any_sync(0xffffffffu, up)) {
              // the accumulator holds PV up to chunk gc - 1: scale it (and l) to the new maximum
              if (!mbar_wait_compact(kv_empty + ((gc - 1) % Cfg::kKVStages), (uint32_t)((gc - 1) / Cfg::kKVStages) & 1u,
                                     p.status)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const float corr = up ? ex2_approx(m - mx) : 1.f;
              if (up) m = mx;
              l *= corr;
              float o[DO];
              const uint32_t oa = o_cols(ui);
              o_load(oa, o);
#pragma unroll
              for (int i = 0; i < DO; ++i) o[i] *= corr;
              if constexpr (DO == 16) {
                uint32_t ou[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) ou[i] = __float_as_uint(o[i]);
                tmem_st16_nowait(oa, ou);
              } else {
                tmem_st32(oa, o);
              }
            }
          }
          // P = 2^(s * scale - m) as f16 over the first KW/2 of this warp's KW
          // S columns (all of them already in registers): keys 2c, 2c+1 in
          // column c
          const float sc = p.scale_log2, nm = -m;
          float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int hb = 0; hb < KW / 32; ++hb) {
            uint32_t pk[16];
#pragma unroll
            for (int i = 0; i < 32; i += 2) {
              const int k = 32 * hb + i;
              const float p0 = ex2_approx(fmaf(v[k], sc, nm));
              const float p1 = ex2_approx(fmaf(v[k + 1], sc, nm));
              s4[(i >> 1) & 3] += p0 + p1;
              pk[i / 2] = pack_f16x2(p0, p1);
            }
            tmem_st16_nowait(tile + (uint32_t)(16 * hb), pk);
          }
          l += (s4[0] + s4[1]) + (s4[2] + s4[3]);
          tmem_st_wait();
          tc_fence_before();
        }
        mbar_arrive1(p_full + t);
        // at a unit's first chunk, the previous unit's output is stored (its
        // last PV has completed or is about to)
        if (j == 0 && have_done && !finish()) {
          ok = false;
          break;
        }
      }
      if (!ok) break;
      dn.h = c.h;
      dn.q0 = c.q0;
      dn.qcnt = c.qcnt;
      dn.qoff = c.qoff;
      dn.ui = ui;
      dn.g = gc - 1;
      dn.l = l;
      dn.active = active;
      have_done = true;
      ++ui;
    }
    if (ok && have_done) finish();
  }

  __syncwarp();  // each warp arrives whole: single lanes ran the producer and MMA loops
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, Cfg::kTmemCols);
}

namespace {
int g_attn_sms = 0;
// a launch whose CTAs each walk at least this many key chunks takes the split issuers
constexpr long long kSplitChunks = 32;
int g_attn_split = -1;  // FE_ATTN_SPLIT for d_h = 32: 0 one issuer, 1 split issuers, unset by chunks per CTA
}

cudaError_t attn_prepare() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_attn_sms, cudaDevAttrMultiProcessorCount, dev);
  if (g_attn_split < 0) {
    const char* v = std::getenv("FE_ATTN_SPLIT");
    g_attn_split = v && *v ? (std::atoi(v) != 0 ? 1 : 0) : 2;
  }
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<32, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)AttnCfg<32>::kSmem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<32, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)AttnCfg<32>::kSmem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<64, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)AttnCfg<64>::kSmem);
  return e;
}

int attn_chunk_keys(int dh) { return dh == 32 ? AttnCfg<32>::CK : AttnCfg<64>::CK; }

cudaError_t attn_launch(int dh, const CUtensorMap* q, const CUtensorMap* k, const CUtensorMap* v, const AttnParams& p0,
                        cudaStream_t s) {
  if (p0.n_segments <= 0 || p0.max_q <= 0 || (!p0.kv_self && p0.kv_cnt <= 0)) return cudaSuccess;
  AttnParams p = p0;
  p.max_q_tiles = (p.max_q + BQ - 1) / BQ;
  const long long units = (long long)p.n_segments * p.n_heads * p.max_q_tiles;
  const long long sms = g_attn_sms > 0 ? g_attn_sms : 148;
  const int ck = attn_chunk_keys(dh);
  const long long grid_max = sms * (dh == 32 ? AttnCfg<32>::kCtasPerSM : AttnCfg<64>::kCtasPerSM);
  const long long grid = units < grid_max ? units : grid_max;
  // key chunks per CTA: the split issuers pay off once each CTA walks many
  const long long keys = p.kv_self ? p.max_q : p.kv_cnt;
  const long long per_cta = units * ((keys + ck - 1) / ck) / grid;
  const bool split = g_attn_split == 2 ? per_cta >= kSplitChunks : g_attn_split == 1;  // d_h = 64 always splits
  const dim3 g((unsigned)grid);
  if (dh == 32) {
    if (split)
      return launch_k(attn_kernel<32, true>, g, dim3(attn_threads<32, true>()), AttnCfg<32>::kSmem, s, *q, *k, *v, p);
    return launch_k(attn_kernel<32, false>, g, dim3(attn_threads<32, false>()), AttnCfg<32>::kSmem, s, *q, *k, *v, p);
  }
  return launch_k(attn_kernel<64, true>, g, dim3(attn_threads<64, true>()), AttnCfg<64>::kSmem, s, *q, *k, *v, p);
}

}  // namespace fe
