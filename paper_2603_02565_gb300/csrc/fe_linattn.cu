// Linear-attention context module.
//
// The online deployment of the paper (Appendix B.3) serves 1,000-interaction
// contexts with linear attention (Katharopoulos et al., 2020).  Here it
// replaces the softmax in the element -> context cross-attention of Section
// 4.2: with the feature map phi(x) = elu(x) + 1, non-causal over the
// context, the context of a request reduces, per layer l and head h, to the
// state
//     S = sum_c phi(K_l[c, h]) V_l[c, h]^T   [d_h, d_h],   z = sum_c phi(K_l[c, h])   [d_h],
// computed once per request (the QKV-Cache idea with a constant-size state
// instead of C key/value rows), and an element query q reads
//     a = phi(q) S / (phi(q) . z).
//
//   lin_state_kernel : one CTA per (segment, layer x head); streams the
//                      segment's C key/value rows through shared memory in
//                      64-row chunks (16-byte loads of the next chunk in
//                      flight while the current one is multiplied), every
//                      thread owning a 2x2 (d_h = 32) or 4x4 (d_h = 64) tile
//                      of S
//   lin_attn_kernel  : one CTA per segment; the segment's states of one layer
//                      (all heads) and phi(q) of 32-row blocks in shared
//                      memory, one warp per (head, 16 rows), a lane per
//                      output column and 16 rows of accumulators in registers
#include <cuda_fp16.h>

#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {

// elu(x) + 1; the exponential branch (x <= 0, result in (0, 1]) through the
// hardware exponent unit, whose relative error is far below the f16 rounding
// of the keys and queries it is applied to
__device__ __forceinline__ float phi(float x) { return x > 0.f ? x + 1.f : __expf(x); }

__device__ __forceinline__ float warp_sum32(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}

constexpr int kChunk = 64;  // context rows per shared-memory chunk

}  // namespace

// Context states.  A CTA takes one segment, one layer and one group of FG
// features (FG = min(d, 128): the heads [g FG / DH, (g + 1) FG / DH)); every
// thread owns a TI x TJ tile of one head's S, so a context row costs it one
// 16-byte load of phi(K) and TJ / 4 of V for TI * TJ multiply-adds.
template <int DH, int FG>
__global__ void __launch_bounds__(256) lin_state_kernel(const __half* __restrict__ kv, int hm, int rows_alloc, int ld,
                                                        int C, int d, int H, float* __restrict__ states) {
  constexpr int HG = FG / DH;               // heads per group
  constexpr int TI = 4;
  constexpr int TJ = DH == 32 ? 4 : 8;
  constexpr int TPH = DH * DH / (TI * TJ);  // threads per head (64 or 128); HG * TPH <= 256 are active
  constexpr int NJT = DH / TJ;              // tiles along j
  constexpr int SB = DH * DH + DH;
  constexpr int RC = 32;                    // context rows per chunk
  constexpr int NP = RC * FG / 8;           // 16-byte pieces of a chunk, for K and for V
  constexpr int P8 = (NP + 255) / 256;      // per thread
  static_assert(HG * TPH <= 256, "tiling");
  __shared__ __align__(16) float sK[RC][FG];  // phi(K) rows of the chunk
  __shared__ __align__(16) float sV[RC][FG];
  const int s = blockIdx.x, G = d / FG, l = blockIdx.y / G, g = blockIdx.y % G;
  const int kcol = 2 * l * d + g * FG, vcol = (2 * l + 1) * d + g * FG;
  const size_t row0 = (size_t)s * C;
  // element (row, col) of K/V: head-major blocks [col / DH][rows_alloc][DH], or row-major [rows][ld]
  auto at = [&](size_t row, int col) -> size_t {
    return hm ? ((size_t)(col / DH) * rows_alloc + row) * DH + (col % DH) : row * ld + col;
  };
  const int t = threadIdx.x, hh = t / TPH, tl = t % TPH;
  const bool active = hh < HG;
  const int fi = hh * DH + (tl / NJT) * TI;   // feature of S's first row in this tile
  const int fj = hh * DH + (tl % NJT) * TJ;   // feature of its first column
  const bool zrow = (tl % NJT) == 0;          // one column of tiles also sums phi(K) into z
  float acc[TI][TJ];
#pragma unroll
  for (int x = 0; x < TI; ++x)
#pragma unroll
    for (int y = 0; y < TJ; ++y) acc[x][y] = 0.f;
  float zacc[TI] = {0.f, 0.f, 0.f, 0.f};
  uint4 kr[P8], vr[P8];
  // the 16-byte pieces of a chunk this thread loads; rows past C read as zero
  auto load = [&](int r0) {
#pragma unroll
    for (int q = 0; q < P8; ++q) {
      const int idx = t + 256 * q, r = idx / (FG / 8), c8 = (idx % (FG / 8)) * 8;
      if (idx < NP && r0 + r < C) {
        kr[q] = *reinterpret_cast<const uint4*>(kv + at(row0 + r0 + r, kcol + c8));
        vr[q] = *reinterpret_cast<const uint4*>(kv + at(row0 + r0 + r, vcol + c8));
      } else {
        kr[q] = make_uint4(0u, 0u, 0u, 0u);
        vr[q] = kr[q];
      }
    }
  };
  pdl_wait();
  pdl_trigger();
  load(0);
  for (int r0 = 0; r0 < C; r0 += RC) {
    const int nr = min(RC, C - r0);
    __syncthreads();  // the previous chunk is consumed
#pragma unroll
    for (int q = 0; q < P8; ++q) {
      const int idx = t + 256 * q, r = idx / (FG / 8), c8 = (idx % (FG / 8)) * 8;
      if (idx >= NP) continue;
      const __half* hk = reinterpret_cast<const __half*>(&kr[q]);
      const __half* hv = reinterpret_cast<const __half*>(&vr[q]);
      const bool valid = r < nr;
      float4 k0, k1, v0, v1;
      k0.x = valid ? phi(__half2float(hk[0])) : 0.f;  // a missing row adds nothing
      k0.y = valid ? phi(__half2float(hk[1])) : 0.f;
      k0.z = valid ? phi(__half2float(hk[2])) : 0.f;
      k0.w = valid ? phi(__half2float(hk[3])) : 0.f;
      k1.x = valid ? phi(__half2float(hk[4])) : 0.f;
      k1.y = valid ? phi(__half2float(hk[5])) : 0.f;
      k1.z = valid ? phi(__half2float(hk[6])) : 0.f;
      k1.w = valid ? phi(__half2float(hk[7])) : 0.f;
      v0 = make_float4(__half2float(hv[0]), __half2float(hv[1]), __half2float(hv[2]), __half2float(hv[3]));
      v1 = make_float4(__half2float(hv[4]), __half2float(hv[5]), __half2float(hv[6]), __half2float(hv[7]));
      *reinterpret_cast<float4*>(&sK[r][c8]) = k0;
      *reinterpret_cast<float4*>(&sK[r][c8 + 4]) = k1;
      *reinterpret_cast<float4*>(&sV[r][c8]) = v0;
      *reinterpret_cast<float4*>(&sV[r][c8 + 4]) = v1;
    }
    __syncthreads();
    if (r0 + RC < C) load(r0 + RC);  // in flight during the products below
#pragma unroll 4
    for (int r = 0; r < (active ? nr : 0); ++r) {
      const float4 ka = *reinterpret_cast<const float4*>(&sK[r][fi]);
      const float a[4] = {ka.x, ka.y, ka.z, ka.w};
      float b[TJ];
#pragma unroll
      for (int y = 0; y < TJ; y += 4) {
        const float4 vb = *reinterpret_cast<const float4*>(&sV[r][fj + y]);
        b[y] = vb.x;
        b[y + 1] = vb.y;
        b[y + 2] = vb.z;
        b[y + 3] = vb.w;
      }
#pragma unroll
      for (int x = 0; x < TI; ++x)
#pragma unroll
        for (int y = 0; y < TJ; ++y) acc[x][y] = fmaf(a[x], b[y], acc[x][y]);
      if (zrow) {
#pragma unroll
        for (int x = 0; x < TI; ++x) zacc[x] += a[x];
      }
    }
  }
  if (!active) return;
  const int h = g * HG + hh;
  const int Ly = gridDim.y / G;
  float* st = states + (((size_t)s * Ly + l) * H + h) * SB;  // S row-major, then z
  const int i0 = fi - hh * DH, j0 = fj - hh * DH;
#pragma unroll
  for (int x = 0; x < TI; ++x)
#pragma unroll
    for (int y = 0; y < TJ; y += 4)
      *reinterpret_cast<float4*>(st + (i0 + x) * DH + j0 + y) =
          make_float4(acc[x][y], acc[x][y + 1], acc[x][y + 2], acc[x][y + 3]);
  if (zrow) {
#pragma unroll
    for (int x = 0; x < TI; ++x) st[DH * DH + i0 + x] = zacc[x];
  }
}

namespace {
constexpr int kRowBlock = 32;  // element rows staged per block of lin_attn_kernel
constexpr int kRowTask = 16;   // rows per warp task (a task: one head, kRowTask rows)
}

template <int DH>
__global__ void __launch_bounds__(256) lin_attn_kernel(const __half* __restrict__ q, int ldq, int d,
                                                       const float* __restrict__ states, int Ly, int l, int H,
                                                       const int* __restrict__ off_dev, const int* __restrict__ cnt_dev,
                                                       int stride, int cnt_fixed, bf16* o_h, bf16* o_l, int ldo) {
  constexpr int SB = DH * DH + DH;
  constexpr int NJ = DH / 32;           // output columns per lane
  extern __shared__ __align__(16) float sm[];
  float* sst = sm;                      // [H][SB]: layer l's states of this segment
  float* sq = sm + H * SB;              // [kRowBlock][d + 4]: phi(q) of a block of rows (padded rows)
  const int ldq_s = d + 4;
  const int s = blockIdx.x;
  pdl_wait();
  pdl_trigger();
  // the states, four 16-byte loads in flight per thread at a time
  {
    const float4* src = reinterpret_cast<const float4*>(states + ((size_t)s * Ly + l) * H * SB);
    float4* dst = reinterpret_cast<float4*>(sst);
    const int n4 = H * SB / 4;
    for (int i0 = threadIdx.x; i0 < n4; i0 += 1024) {
      float4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + 256 * u < n4) v[u] = src[i0 + 256 * u];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + 256 * u < n4) dst[i0 + 256 * u] = v[u];
    }
  }
  const int off = off_dev ? off_dev[s] : s * stride;
  const int cnt = cnt_dev ? cnt_dev[s] : cnt_fixed;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int d8 = d / 8;
  for (int rb = 0; rb < cnt; rb += kRowBlock) {
    const int nr = min(kRowBlock, cnt - rb);
    __syncthreads();  // the previous block (and, the first time, the states) consumed / written
    for (int i0 = threadIdx.x; i0 < nr * d8; i0 += 1024) {
      uint4 raw[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int idx = i0 + 256 * u;
        if (idx < nr * d8) raw[u] = *reinterpret_cast<const uint4*>(q + (size_t)(off + rb + idx / d8) * ldq + (idx % d8) * 8);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int idx = i0 + 256 * u;
        if (idx < nr * d8) {
          const int r = idx / d8, c8 = (idx % d8) * 8;
          const __half* hq = reinterpret_cast<const __half*>(&raw[u]);
#pragma unroll
          for (int e = 0; e < 8; ++e) sq[r * ldq_s + c8 + e] = phi(__half2float(hq[e]));
        }
      }
    }
    __syncthreads();
    // warp tasks (head, kRowTask rows of the block): lane j owns output
    // column j (and j + 32) of every row of its task
    const int nsub = (nr + kRowTask - 1) / kRowTask;
    for (int task = warp; task < H * nsub; task += 8) {
      const int h = task % H, sr = (task / H) * kRowTask;
      const float* S = sst + h * SB;
      const float* z = S + DH * DH;
      const float* qh = sq + sr * ldq_s + h * DH;
      const int tn = min(kRowTask, nr - sr);
      float acc[kRowTask][NJ];
#pragma unroll
      for (int r = 0; r < kRowTask; ++r)
#pragma unroll
        for (int jj = 0; jj < NJ; ++jj) acc[r][jj] = 0.f;
#pragma unroll 1
      for (int i = 0; i < DH; i += 4) {
        float sv[4][NJ];
#pragma unroll
        for (int ii = 0; ii < 4; ++ii)
#pragma unroll
          for (int jj = 0; jj < NJ; ++jj) sv[ii][jj] = S[(i + ii) * DH + lane + 32 * jj];
#pragma unroll
        for (int r = 0; r < kRowTask; ++r) {
          const float4 f = *reinterpret_cast<const float4*>(qh + r * ldq_s + i);  // one address: broadcast
#pragma unroll
          for (int jj = 0; jj < NJ; ++jj) {
            acc[r][jj] = fmaf(f.x, sv[0][jj], acc[r][jj]);
            acc[r][jj] = fmaf(f.y, sv[1][jj], acc[r][jj]);
            acc[r][jj] = fmaf(f.z, sv[2][jj], acc[r][jj]);
            acc[r][jj] = fmaf(f.w, sv[3][jj], acc[r][jj]);
          }
        }
      }
      // lane r: the normaliser phi(q_r) . z of row r (padded rows: conflict-free)
      float den = 0.f;
      if (lane < tn) {
#pragma unroll 4
        for (int i = 0; i < DH; i += 4) {
          const float4 f = *reinterpret_cast<const float4*>(qh + lane * ldq_s + i);
          den = fmaf(f.x, z[i], den);
          den = fmaf(f.y, z[i + 1], den);
          den = fmaf(f.z, z[i + 2], den);
          den = fmaf(f.w, z[i + 3], den);
        }
      }
#pragma unroll
      for (int r = 0; r < kRowTask; ++r) {
        const float inv = 1.f / __shfl_sync(0xFFFFFFFFu, den, r);
        if (r < tn) {
          const size_t row = (size_t)(off + rb + sr + r);
#pragma unroll
          for (int jj = 0; jj < NJ; ++jj) {
            const float x = acc[r][jj] * inv;
            const __nv_bfloat16 hi = __float2bfloat16_rn(x);
            const __nv_bfloat16 lo = __float2bfloat16_rn(x - __bfloat162float(hi));
            const size_t o = row * ldo + h * DH + lane + 32 * jj;
            o_h[o] = hi;
            o_l[o] = lo;
          }
        }
      }
    }
  }
}

namespace {
// H <= 8 heads of d_h = 64, and a block of rows of width d <= 512
constexpr int kLinAttnSmemMax = 8 * (64 * 64 + 64) * 4 + kRowBlock * (512 + 4) * 4;
}

cudaError_t linattn_prepare() {
  cudaError_t e = cudaFuncSetAttribute(lin_attn_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       kLinAttnSmemMax);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(lin_attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, kLinAttnSmemMax);
  return e;
}

cudaError_t lin_state_launch(const bf16* kv, int hm, int rows_alloc, int ld, int n_seg, int C, int d, int dh, int Ly,
                             int H, float* states, cudaStream_t s) {
  if (n_seg <= 0 || C <= 0) return cudaSuccess;
  const int FG = d < 128 ? d : 128;
  const dim3 grid((unsigned)n_seg, (unsigned)(Ly * (d / FG)));
  const __half* k = reinterpret_cast<const __half*>(kv);
  if (dh == 32 && FG == 128)
    return launch_k(lin_state_kernel<32, 128>, grid, dim3(256), 0, s, k, hm, rows_alloc, ld, C, d, H, states);
  if (dh == 32 && FG == 64)
    return launch_k(lin_state_kernel<32, 64>, grid, dim3(256), 0, s, k, hm, rows_alloc, ld, C, d, H, states);
  if (dh == 64 && FG == 128)
    return launch_k(lin_state_kernel<64, 128>, grid, dim3(256), 0, s, k, hm, rows_alloc, ld, C, d, H, states);
  if (dh == 64 && FG == 64)
    return launch_k(lin_state_kernel<64, 64>, grid, dim3(256), 0, s, k, hm, rows_alloc, ld, C, d, H, states);
  if (dh == 32 && FG == 32)
    return launch_k(lin_state_kernel<32, 32>, grid, dim3(256), 0, s, k, hm, rows_alloc, ld, C, d, H, states);
  return cudaErrorInvalidValue;
}

cudaError_t lin_attn_launch(const bf16* q, int ldq, const float* states, int n_seg, int Ly, int l, int H, int dh,
                            const int* off_dev, const int* cnt_dev, int stride, int cnt_fixed, bf16* o_h, bf16* o_l,
                            int ldo, cudaStream_t s) {
  if (n_seg <= 0) return cudaSuccess;
  const int d = H * dh;
  const size_t smem = ((size_t)H * (dh * dh + dh) + (size_t)kRowBlock * (d + 4)) * sizeof(float);
  if (smem > (size_t)kLinAttnSmemMax) return cudaErrorInvalidValue;
  const __half* qh = reinterpret_cast<const __half*>(q);
  if (dh == 32)
    return launch_k(lin_attn_kernel<32>, dim3((unsigned)n_seg), dim3(256), smem, s, qh, ldq, d, states, Ly, l, H, off_dev,
                    cnt_dev, stride, cnt_fixed, o_h, o_l, ldo);
  if (dh == 64)
    return launch_k(lin_attn_kernel<64>, dim3((unsigned)n_seg), dim3(256), smem, s, qh, ldq, d, states, Ly, l, H, off_dev,
                    cnt_dev, stride, cnt_fixed, o_h, o_l, ldo);
  return cudaErrorInvalidValue;
}

}  // namespace fe
