// Memory-bound kernels of the joint evaluator: distinct-element compaction
// (Section 4.1), LayerNorm / gather of the element rows (Section 4.2),
// index-based assembly with the [CLS]-pooled SeqEnc attention (Section 4.3),
// the argmax of Eq. 1, and init-time weight preparation.
#include <climits>
#include <cstdlib>

#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {

// ---------------------------------------------------------------------------
// small helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Block-wide exclusive scan of one int per thread (blockDim.x == 256).
__device__ int block_excl_scan_256(int v, int* total) {
  __shared__ int warp_tot[8];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[warp] = x;
  __syncthreads();
  int base = 0, all = 0;
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    if (w < warp) base += warp_tot[w];
    all += warp_tot[w];
  }
  __syncthreads();
  *total = all;
  return base + x - v;
}

// DPL consecutive elements of type T -> float
template <int DPL, typename T>
__device__ __forceinline__ void load_vec(const T* src, float* out) {
  if constexpr (sizeof(T) == 4) {
    if constexpr (DPL % 4 == 0) {
#pragma unroll
      for (int i = 0; i < DPL; i += 4) {
        const float4 q = *reinterpret_cast<const float4*>(src + i);
        out[i] = q.x;
        out[i + 1] = q.y;
        out[i + 2] = q.z;
        out[i + 3] = q.w;
      }
    } else {
#pragma unroll
      for (int i = 0; i < DPL; ++i) out[i] = reinterpret_cast<const float*>(src)[i];
    }
  } else {
    if constexpr (DPL % 8 == 0) {
#pragma unroll
      for (int i = 0; i < DPL; i += 8) {
        const uint4 q = *reinterpret_cast<const uint4*>(src + i);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          out[i + 2 * j] = bf16lo_f(w[j]);
          out[i + 2 * j + 1] = bf16hi_f(w[j]);
        }
      }
    } else if constexpr (DPL % 2 == 0) {
#pragma unroll
      for (int i = 0; i < DPL; i += 2) {
        const uint32_t w = *reinterpret_cast<const uint32_t*>(src + i);
        out[i] = bf16lo_f(w);
        out[i + 1] = bf16hi_f(w);
      }
    } else {
#pragma unroll
      for (int i = 0; i < DPL; ++i) out[i] = __bfloat162float(src[i]);
    }
  }
}

// split pair of DPL consecutive bf16 (hi plane + lo plane) -> float
template <int DPL>
__device__ __forceinline__ void load_split(const bf16* h, const bf16* l, float* out) {
  float a[DPL], b[DPL];
  load_vec<DPL>(h, a);
  load_vec<DPL>(l, b);
#pragma unroll
  for (int i = 0; i < DPL; ++i) out[i] = a[i] + b[i];
}

// DPL floats -> split planes
template <int DPL>
__device__ __forceinline__ void store_split(const float* x, bf16* h, bf16* l) {
  if constexpr (DPL % 2 == 0) {
    uint32_t hw[DPL / 2], lw[DPL / 2];
#pragma unroll
    for (int i = 0; i < DPL; i += 2) split2(x[i], x[i + 1], hw[i / 2], lw[i / 2]);
    if constexpr (DPL % 8 == 0) {
#pragma unroll
      for (int i = 0; i < DPL / 2; i += 4) {
        *reinterpret_cast<uint4*>(h + 2 * i) = make_uint4(hw[i], hw[i + 1], hw[i + 2], hw[i + 3]);
        *reinterpret_cast<uint4*>(l + 2 * i) = make_uint4(lw[i], lw[i + 1], lw[i + 2], lw[i + 3]);
      }
    } else {
#pragma unroll
      for (int i = 0; i < DPL / 2; ++i) {
        *reinterpret_cast<uint32_t*>(h + 2 * i) = hw[i];
        *reinterpret_cast<uint32_t*>(l + 2 * i) = lw[i];
      }
    }
  } else {
#pragma unroll
    for (int i = 0; i < DPL; ++i) split_bf16(x[i], h[i], l[i]);
  }
}

// LN of a row distributed over a warp, DPL values per lane (biased variance, two passes)
template <int DPL>
__device__ __forceinline__ void warp_layer_norm(float* x, int d, float eps) {
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < DPL; ++i) s += x[i];
  const float mean = warp_sum(s) / (float)d;
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < DPL; ++i) {
    const float t = x[i] - mean;
    q = fmaf(t, t, q);
  }
  const float rstd = 1.0f / sqrtf(warp_sum(q) / (float)d + eps);
#pragma unroll
  for (int i = 0; i < DPL; ++i) x[i] = (x[i] - mean) * rstd;
}

}  // namespace

// ---------------------------------------------------------------------------
// distinct-element compaction, one CTA (256 threads) per request.  It reads
// only the batch's candidate indices and writes only the layout, so it waits
// for the kernel before it (the context kernel) at its end rather than its
// start: it runs beside that kernel, and still completes after it, so the
// kernels after it see both.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) compact_kernel(const int32_t* __restrict__ cand, int B, int M, int K,
                                                      int L, int cap, int* U, int* off, int* bad, int* slot_local,
                                                      int* list, int* status, unsigned* ticket) {
  extern __shared__ uint32_t csm[];
  const int W = (M + 31) >> 5;
  uint32_t* bits = csm;
  int* pre = reinterpret_cast<int*>(csm + W);
  __shared__ int s_bad;
  __shared__ int s_last;
  const int b = blockIdx.x, tid = threadIdx.x;
  const int n = K * L;
  const int32_t* cb = cand + (size_t)b * n;
  pdl_trigger();

  for (int w = tid; w < W; w += 256) bits[w] = 0u;
  if (tid == 0) s_bad = 0;
  __syncthreads();
  for (int i = tid; i < n; i += 256) {
    const int m = cb[i];
    if (m < 0 || m >= M)
      s_bad = 1;
    else
      atomicOr(&bits[m >> 5], 1u << (m & 31));
  }
  __syncthreads();
  if (s_bad) {
    for (int i = tid; i < n; i += 256) slot_local[(size_t)b * n + i] = -1;
    if (tid == 0) {
      U[b] = 0;
      bad[b] = 1;
      atomicOr(status, ST_INDEX);
    }
  } else {
    const int per = (W + 255) / 256;
    const int w0 = min(W, tid * per), w1 = min(W, w0 + per);
    int local = 0;
    for (int w = w0; w < w1; ++w) local += __popc(bits[w]);
    int total;
    int run = block_excl_scan_256(local, &total);
    for (int w = w0; w < w1; ++w) {
      pre[w] = run;
      run += __popc(bits[w]);
    }
    __syncthreads();
    if (tid == 0) {
      U[b] = total;
      bad[b] = 0;
    }
    for (int w = tid; w < W; w += 256) {
      uint32_t x = bits[w];
      int r = pre[w];
      while (x) {
        const int bit = __ffs(x) - 1;
        list[(size_t)b * cap + r++] = w * 32 + bit;
        x &= x - 1;
      }
    }
    for (int i = tid; i < n; i += 256) {
      const int m = cb[i];
      slot_local[(size_t)b * n + i] = pre[m >> 5] + __popc(bits[m >> 5] & ((1u << (m & 31)) - 1u));
    }
  }
  // the last CTA to finish turns the counts into offsets (no CTA waits on another)
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(ticket, 1u) == gridDim.x - 1);
  __syncthreads();
  if (s_last) {
    __threadfence();
    const int per = (B + 255) / 256;
    const int b0 = min(B, tid * per), b1 = min(B, b0 + per);
    int local = 0;
    for (int i = b0; i < b1; ++i) local += __ldcg(U + i);
    int total;
    int run = block_excl_scan_256(local, &total);
    for (int i = b0; i < b1; ++i) {
      off[i] = run;
      run += __ldcg(U + i);
    }
    if (tid == 0) {
      off[B] = total;
      *ticket = 0u;
    }
  }
  pdl_wait();  // complete no earlier than the kernel before this one
}

cudaError_t compact_launch(const int32_t* cand, int B, int M, int K, int L, int cap, int* U, int* off,
                           int* bad, int* slot_local, int* list, int* status, unsigned* ticket,
                           cudaStream_t s) {
  const size_t smem = (size_t)2 * ((M + 31) / 32) * sizeof(uint32_t);
  return launch_k(compact_kernel, dim3(B), dim3(256), smem, s, cand, B, M, K, L, cap, U, off, bad, slot_local, list,
                  status, ticket);
}

// ---------------------------------------------------------------------------
// candidate-factorized layout: one CTA (256 threads) per request
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) identity_layout_kernel(const int32_t* __restrict__ cand, int B, int M, int KL,
                                                              int* U, int* off, int* bad, int* slot, int* list,
                                                              int* status) {
  const int b = blockIdx.x;
  pdl_wait();
  pdl_trigger();
  const int32_t* cb = cand + (size_t)b * KL;
  int any_bad = 0;
  for (int i = threadIdx.x; i < KL; i += blockDim.x) {
    const int v = cb[i];
    any_bad |= (v < 0 || v >= M);
  }
  any_bad = __syncthreads_or(any_bad);
  for (int i = threadIdx.x; i < KL; i += blockDim.x) {
    list[(size_t)b * KL + i] = any_bad ? 0 : cb[i];
    slot[(size_t)b * KL + i] = any_bad ? -1 : i;
  }
  if (threadIdx.x == 0) {
    U[b] = KL;
    off[b] = b * KL;
    bad[b] = any_bad;
    if (any_bad) atomicOr(status, ST_INDEX);
    if (b == B - 1) off[B] = B * KL;
  }
}

cudaError_t identity_layout_launch(const int32_t* cand, int B, int M, int KL, int* U, int* off, int* bad,
                                   int* slot, int* list, int* status, cudaStream_t s) {
  if (B <= 0) return cudaSuccess;
  return launch_k(identity_layout_kernel, dim3(B), dim3(256), 0, s, cand, B, M, KL, U, off, bad, slot, list, status);
}

// Whole-pool layout (Section 4.1's alternative U(z) = C(x), U = M): every pool
// row of request b is an element, list[b*M + i] = i, slot[b, i] = cand[b, i];
// a request with an index outside [0, M) gets bad[b] = 1 and slots -1.
__global__ void __launch_bounds__(256) pool_layout_kernel(const int32_t* __restrict__ cand, int B, int M, int KL,
                                                          int* U, int* off, int* bad, int* slot, int* list,
                                                          int* status) {
  const int b = blockIdx.x;
  pdl_wait();
  pdl_trigger();
  const int32_t* cb = cand + (size_t)b * KL;
  int any_bad = 0;
  for (int i = threadIdx.x; i < KL; i += blockDim.x) {
    const int v = cb[i];
    any_bad |= (v < 0 || v >= M);
  }
  any_bad = __syncthreads_or(any_bad);
  for (int i = threadIdx.x; i < KL; i += blockDim.x) slot[(size_t)b * KL + i] = any_bad ? -1 : cb[i];
  for (int i = threadIdx.x; i < M; i += blockDim.x) list[(size_t)b * M + i] = i;
  if (threadIdx.x == 0) {
    U[b] = M;
    off[b] = b * M;
    bad[b] = any_bad;
    if (any_bad) atomicOr(status, ST_INDEX);
    if (b == B - 1) off[B] = B * M;
  }
}

cudaError_t pool_layout_launch(const int32_t* cand, int B, int M, int KL, int* U, int* off, int* bad, int* slot,
                               int* list, int* status, cudaStream_t s) {
  if (B <= 0) return cudaSuccess;
  return launch_k(pool_layout_kernel, dim3(B), dim3(256), 0, s, cand, B, M, KL, U, off, bad, slot, list, status);
}

// ---------------------------------------------------------------------------
// LN of context rows -> split planes (one warp per row)
// ---------------------------------------------------------------------------
template <int DPL, typename T>
__global__ void __launch_bounds__(256) ctx_ln_kernel(const T* __restrict__ x, int rows, float eps,
                                                     bf16* out_h, bf16* out_l, int ldo) {
  constexpr int d = DPL * 32;
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5);
  pdl_wait();
  pdl_trigger();
  if (r >= rows) return;
  float v[DPL];
  load_vec<DPL>(x + (size_t)r * d + lane * DPL, v);
  warp_layer_norm<DPL>(v, d, eps);
  store_split<DPL>(v, out_h + (size_t)r * ldo + lane * DPL, out_l + (size_t)r * ldo + lane * DPL);
}

// ---------------------------------------------------------------------------
// gather the distinct pool rows -> h (fp32) and LN(h) planes (one warp per row)
// ---------------------------------------------------------------------------
template <int DPL, typename T>
__global__ void __launch_bounds__(256) gather_ln_kernel(const T* __restrict__ pool, int B, int M, int cap,
                                                        const int* __restrict__ off, const int* __restrict__ list,
                                                        int max_rows, float eps, float* h, int ldh, bf16* ln_h,
                                                        bf16* ln_l, int ldln) {
  constexpr int d = DPL * 32, RPW = 4;  // four consecutive rows per warp, their loads issued together
  const int lane = threadIdx.x & 31;
  const int r0 = (blockIdx.x * 8 + (threadIdx.x >> 5)) * RPW;
  pdl_wait();
  pdl_trigger();
  const int nrow = min(max_rows, off[B]);
  if (r0 >= nrow) return;
  // the largest b with off[b] <= r0, by the warp: each round the 32 lanes probe
  // 32 evenly spaced candidates of the range [lo, hi) (off[lo] <= r0 holds) and
  // keep the span after the last one that passes, so that B = 1024 takes two
  // rounds of loads instead of ten dependent ones
  int lo = 0, hi = B;
  while (hi - lo > 1) {
    const int step = (hi - lo + 31) / 32;
    const int idx = lo + lane * step;
    const unsigned pass = __ballot_sync(0xffffffffu, idx < hi && off[idx] <= r0);
    lo += (31 - __clz(pass)) * step;
    hi = min(lo + step, hi);
  }
  // the following rows: the same request, or a later one
  int bs[RPW], ms[RPW];
  int b = lo, b_end = off[b + 1];
#pragma unroll
  for (int u = 0; u < RPW; ++u) {
    const int r = r0 + u;
    bs[u] = -1;
    if (r < nrow) {
      while (b_end <= r) b_end = off[++b + 1];
      bs[u] = b;
      ms[u] = list[(size_t)b * cap + (r - off[b])];
    }
  }
  float v[RPW][DPL];
#pragma unroll
  for (int u = 0; u < RPW; ++u)
    if (bs[u] >= 0) load_vec<DPL>(pool + ((size_t)bs[u] * M + ms[u]) * d + lane * DPL, v[u]);
#pragma unroll
  for (int u = 0; u < RPW; ++u) {
    if (bs[u] < 0) break;
    const int r = r0 + u;
    float* hr = h + (size_t)r * ldh + lane * DPL;
    if constexpr (DPL % 4 == 0) {
#pragma unroll
      for (int i = 0; i < DPL; i += 4)
        *reinterpret_cast<float4*>(hr + i) = make_float4(v[u][i], v[u][i + 1], v[u][i + 2], v[u][i + 3]);
    } else {
#pragma unroll
      for (int i = 0; i < DPL; ++i) hr[i] = v[u][i];
    }
    warp_layer_norm<DPL>(v[u], d, eps);
    store_split<DPL>(v[u], ln_h + (size_t)r * ldln + lane * DPL, ln_l + (size_t)r * ldln + lane * DPL);
  }
}

template <typename T>
static cudaError_t ctx_ln_t(const T* x, int rows, int d, float eps, bf16* oh, bf16* ol, int ldo, cudaStream_t s) {
  const unsigned g = (unsigned)((rows + 7) / 8);
  switch (d) {
    case 32: return launch_k(ctx_ln_kernel<1, T>, dim3(g), dim3(256), 0, s, x, rows, eps, oh, ol, ldo);
    case 64: return launch_k(ctx_ln_kernel<2, T>, dim3(g), dim3(256), 0, s, x, rows, eps, oh, ol, ldo);
    case 128: return launch_k(ctx_ln_kernel<4, T>, dim3(g), dim3(256), 0, s, x, rows, eps, oh, ol, ldo);
    case 256: return launch_k(ctx_ln_kernel<8, T>, dim3(g), dim3(256), 0, s, x, rows, eps, oh, ol, ldo);
    case 512: return launch_k(ctx_ln_kernel<16, T>, dim3(g), dim3(256), 0, s, x, rows, eps, oh, ol, ldo);
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

// (mean, rstd) of a row: four rows per warp, their loads issued together, then
// two passes over each row in registers
template <int DPL>
__global__ void __launch_bounds__(256) row_stats_kernel(const bf16* __restrict__ x, int rows, float eps,
                                                        float2* __restrict__ out) {
  constexpr int d = DPL * 32, RPW = 4;
  const int lane = threadIdx.x & 31;
  const int r0 = (blockIdx.x * 8 + (threadIdx.x >> 5)) * RPW;
  pdl_wait();
  pdl_trigger();
  if (r0 >= rows) return;
  float v[RPW][DPL];
#pragma unroll
  for (int u = 0; u < RPW; ++u) {
    if (r0 + u < rows) {
      load_vec<DPL>(x + (size_t)(r0 + u) * d + lane * DPL, v[u]);
    } else {
#pragma unroll
      for (int i = 0; i < DPL; ++i) v[u][i] = 0.f;
    }
  }
#pragma unroll
  for (int u = 0; u < RPW; ++u) {
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < DPL; ++i) s += v[u][i];
    const float mean = warp_sum(s) / (float)d;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < DPL; ++i) {
      const float t = v[u][i] - mean;
      q = fmaf(t, t, q);
    }
    const float rstd = 1.0f / sqrtf(warp_sum(q) / (float)d + eps);
    if (lane == 0 && r0 + u < rows) out[r0 + u] = make_float2(mean, rstd);
  }
}

cudaError_t row_stats_launch(const bf16* x, int rows, int d, float eps, float2* out, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  const unsigned g = (unsigned)((rows + 31) / 32);
  switch (d) {
    case 32: return launch_k(row_stats_kernel<1>, dim3(g), dim3(256), 0, s, x, rows, eps, out);
    case 64: return launch_k(row_stats_kernel<2>, dim3(g), dim3(256), 0, s, x, rows, eps, out);
    case 128: return launch_k(row_stats_kernel<4>, dim3(g), dim3(256), 0, s, x, rows, eps, out);
    case 256: return launch_k(row_stats_kernel<8>, dim3(g), dim3(256), 0, s, x, rows, eps, out);
    case 512: return launch_k(row_stats_kernel<16>, dim3(g), dim3(256), 0, s, x, rows, eps, out);
    default: return cudaErrorInvalidValue;
  }
}

// column sums of a weight (init time): one warp per output column n
__global__ void colsum_kernel(const bf16* w_h, const bf16* w_l, int ld, int N, int K, float* out) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (n >= N) return;
  float a = 0.f;
  for (int k = lane; k < K; k += 32) {
    a += __bfloat162float(w_h[(size_t)n * ld + k]);
    if (w_l) a += __bfloat162float(w_l[(size_t)n * ld + k]);
  }
  a = warp_sum(a);
  if (lane == 0) out[n] = a;
}

cudaError_t colsum_launch(const bf16* w_h, const bf16* w_l, int ld, int N, int K, float* out, cudaStream_t s) {
  if (N <= 0) return cudaSuccess;
  colsum_kernel<<<(N + 7) / 8, 256, 0, s>>>(w_h, w_l, ld, N, K, out);
  return cudaGetLastError();
}

cudaError_t ctx_ln_launch(const void* x, int io_f32, int rows, int d, float eps, bf16* out_h, bf16* out_l,
                          int ldo, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (io_f32) return ctx_ln_t(static_cast<const float*>(x), rows, d, eps, out_h, out_l, ldo, s);
  return ctx_ln_t(static_cast<const bf16*>(x), rows, d, eps, out_h, out_l, ldo, s);
}

template <typename T>
static cudaError_t gather_t(const T* pool, int B, int M, int d, int cap, const int* off, const int* list,
                            int max_rows, float eps, float* h, int ldh, bf16* lh, bf16* ll, int ldln,
                            cudaStream_t s) {
  const unsigned g = (unsigned)((max_rows + 31) / 32);
#define FE_GATHER(DPL)                                                                                      \
  return launch_k(gather_ln_kernel<DPL, T>, dim3(g), dim3(256), 0, s, pool, B, M, cap, off, list, max_rows, eps, h, \
                  ldh, lh, ll, ldln)
  switch (d) {
    case 32: FE_GATHER(1); break;
    case 64: FE_GATHER(2); break;
    case 128: FE_GATHER(4); break;
    case 256: FE_GATHER(8); break;
    case 512: FE_GATHER(16); break;
    default: return cudaErrorInvalidValue;
  }
#undef FE_GATHER
  return cudaGetLastError();
}

cudaError_t gather_ln_launch(const void* pool, int io_f32, int B, int M, int d, int cap, const int* off,
                             const int* list, int max_rows, float eps, float* h, int ldh, bf16* ln_h,
                             bf16* ln_l, int ldln, cudaStream_t s) {
  if (max_rows <= 0) return cudaSuccess;
  if (io_f32)
    return gather_t(static_cast<const float*>(pool), B, M, d, cap, off, list, max_rows, eps, h, ldh, ln_h, ln_l,
                    ldln, s);
  return gather_t(static_cast<const bf16*>(pool), B, M, d, cap, off, list, max_rows, eps, h, ldh, ln_h, ln_l,
                  ldln, s);
}

// ---------------------------------------------------------------------------
// SeqEnc [CLS] attention: W = 1, 2, 4 or 8 warps per sequence (b, k) and 8 / W
// sequences per CTA.  Tokens are [CLS] and the L indexed elements, whose keys
// and values are the cached element projections plus the position projections
// (x_j W = H[i] W + P[j-1] W; positions added after indexing).  Only the [CLS]
// query is needed, so a key enters through its logit
//   q0 . (H[i] WKs + P[j-1] WKs) = sum of the element's per-chunk partials
//                                  q0 . (H[i] WKs) + a per-position constant,
// and a key costs its value row (and the position's value row) only.  Warp w of
// a sequence takes the keys j = w, w + W, ... with its own running maximum and
// sum per head and its own output row; with W > 1 the W partial results are
// merged in shared memory (softmax over all keys = the partial sums rescaled to
// the largest partial maximum), so that few long sequences still give every SM
// several warps.  Short position tables (L d <= kVpStage) are staged in shared
// memory once per CTA.
// ---------------------------------------------------------------------------
constexpr int kVpStage = 6144;  // floats

template <int DPL>
__global__ void __launch_bounds__(256) cls_attn_kernel(const ClsParams p, int W) {
  extern __shared__ float cls_sm[];  // W > 1: [8][d] partial rows, [8][32] maxima, [8][32] sums; then P WVs
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int seq = blockIdx.x * (8 / W) + warp / W;
  const int wi = warp % W;  // this warp's share of the keys
  const int d = p.d;
  const int lph = 32 / p.H;  // lanes per head
  const int hd = lane / lph;  // this lane's head
  const int cph = (d / p.H) / 32;  // logit chunks per head (1 or 2)
  const int nch = d / 32;
  const int d0 = lane * DPL;
  // P WVs rows are parameters: staged before the programmatic wait
  const bool vp_smem = p.L * d <= kVpStage;
  float* svp = cls_sm + (W > 1 ? 8 * d + 512 : 0);
  if (vp_smem) {
    const float4* src = reinterpret_cast<const float4*>(p.vP);
    for (int i = threadIdx.x; i < p.L * d / 4; i += blockDim.x) reinterpret_cast<float4*>(svp)[i] = src[i];
  }
  const float* vpb = vp_smem ? svp : p.vP;
  pdl_wait();
  pdl_trigger();
  if (vp_smem) __syncthreads();
  const bool live = seq < p.B * p.K;
  float o[DPL];
  float m = -INFINITY, l = 0.f;
#pragma unroll
  for (int i = 0; i < DPL; ++i) o[i] = 0.f;
  if (live) {
    const int b = seq / p.K;
    if (wi == 0) {  // token 0: [CLS]
      m = p.qk0[hd] * p.scale;
      l = 1.f;
      load_vec<DPL>(p.v0 + d0, o);
    }
    const int L = p.bad[b] ? 0 : p.L;
    const int base = p.off[b];
    const int* sl = p.slot_local + (size_t)seq * p.L;
    const int nk = L > wi ? (L - wi + W - 1) / W : 0;  // keys of this warp
    // lane i holds the slot of the warp's key i (one load for its first 32 keys),
    // so a key's rows are requested without first waiting for its slot index
    const int my_slot = lane < nk ? sl[wi + lane * W] : 0;
    for (int i = 0; i < nk; ++i) {
      const int j = wi + i * W;
      const int slot = i < 32 ? __shfl_sync(0xffffffffu, my_slot, i) : sl[j];
      const size_t er = (size_t)(base + slot);
      const float* lg = p.elog + er * nch + (size_t)(hd * cph);
      float s = lg[0];
      if (cph > 1) s += lg[1];
      s = (s + p.qkP[j * p.H + hd]) * p.scale;
      float vx[DPL], vp[DPL];
      load_split<DPL>(p.kv_h + er * p.ldkv + d + d0, p.kv_l + er * p.ldkv + d + d0, vx);
      load_vec<DPL>(vpb + (size_t)j * d + d0, vp);
      const float mn = fmaxf(m, s);
      const float c = expf(m - mn);  // 0 while m is -inf (a warp's first key)
      const float e = expf(s - mn);
      l = l * c + e;
#pragma unroll
      for (int t = 0; t < DPL; ++t) o[t] = o[t] * c + e * (vx[t] + vp[t]);
      m = mn;
    }
  }
  if (W == 1) {
    if (live) {
      const float inv = 1.f / l;
#pragma unroll
      for (int i = 0; i < DPL; ++i) o[i] *= inv;
      store_split<DPL>(o, p.o_h + (size_t)seq * p.ldo + d0, p.o_l + (size_t)seq * p.ldo + d0);
    }
    return;
  }
  float* so = cls_sm;             // [8][d]
  float* sm = cls_sm + 8 * d;     // [8][32]
  float* ss = sm + 256;           // [8][32]
#pragma unroll
  for (int i = 0; i < DPL; ++i) so[warp * d + d0 + i] = o[i];
  sm[warp * 32 + lane] = m;
  ss[warp * 32 + lane] = l;
  __syncthreads();
  if (!live) return;
  // the sequence's W warps merge its row, two adjacent columns per thread; a
  // column's maximum and sum are those of the lane that owns it (equal on all
  // lanes of a head); warp 0 of the sequence holds [CLS], so the maximum is finite
  const int g0 = warp - wi;
  for (int c = 2 * (wi * 32 + lane); c < d; c += 64 * W) {
    float r[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int ln = (c + u) / DPL;
      float M = -INFINITY;
      for (int w = 0; w < W; ++w) M = fmaxf(M, sm[(g0 + w) * 32 + ln]);
      float sum = 0.f, acc = 0.f;
      for (int w = 0; w < W; ++w) {
        const float e = expf(sm[(g0 + w) * 32 + ln] - M);
        sum = fmaf(ss[(g0 + w) * 32 + ln], e, sum);
        acc = fmaf(so[(g0 + w) * d + c + u], e, acc);
      }
      r[u] = acc / sum;
    }
    uint32_t hw, lw;
    split2(r[0], r[1], hw, lw);
    *reinterpret_cast<uint32_t*>(p.o_h + (size_t)seq * p.ldo + c) = hw;
    *reinterpret_cast<uint32_t*>(p.o_l + (size_t)seq * p.ldo + c) = lw;
  }
}

cudaError_t cls_attn_launch(const ClsParams& p, cudaStream_t s) {
  const int n = p.B * p.K;
  if (n <= 0) return cudaSuccess;
  // warps per sequence: enough warps in flight (about 4096) for the latency of
  // the gathered rows, at least two keys per warp
  int W = 1;
  while (W < 8 && 2 * W <= p.L && (long long)n * W < 4096) W *= 2;
  const unsigned g = (unsigned)((n + 8 / W - 1) / (8 / W));
  const size_t smem = ((W > 1 ? (size_t)(8 * p.d + 512) : 0) + (p.L * p.d <= kVpStage ? (size_t)p.L * p.d : 0)) *
                      sizeof(float);
  switch (p.d) {
    case 32: return launch_k(cls_attn_kernel<1>, dim3(g), dim3(256), smem, s, p, W);
    case 64: return launch_k(cls_attn_kernel<2>, dim3(g), dim3(256), smem, s, p, W);
    case 128: return launch_k(cls_attn_kernel<4>, dim3(g), dim3(256), smem, s, p, W);
    case 256: return launch_k(cls_attn_kernel<8>, dim3(g), dim3(256), smem, s, p, W);
    case 512: return launch_k(cls_attn_kernel<16>, dim3(g), dim3(256), smem, s, p, W);
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

__global__ void cls_consts_kernel(const float* q0, const float* k0, const float* kP, int max_L, int d, int H,
                                  float* out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (max_L + 1) * H) return;
  const int j = i / H, h = i % H, dh = d / H;
  const float* kv = j < max_L ? kP + (size_t)j * d : k0;
  float acc = 0.f;
  for (int c = h * dh; c < h * dh + dh; ++c) acc = fmaf(q0[c], kv[c], acc);
  out[i] = acc;
}

cudaError_t cls_consts_launch(const float* q0, const float* k0, const float* kP, int max_L, int d, int H, float* qk,
                              cudaStream_t s) {
  const int n = (max_L + 1) * H;
  cls_consts_kernel<<<(n + 127) / 128, 128, 0, s>>>(q0, k0, kP, max_L, d, H, qk);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// init-time weight preparation
// ---------------------------------------------------------------------------
__global__ void transpose_split_kernel(const float* __restrict__ W, int Kin, int N, bf16* out_h, bf16* out_l,
                                       int ldo, int row0) {
  const size_t total = (size_t)Kin * N;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total; i += (size_t)gridDim.x * blockDim.x) {
    const int n = (int)(i % N), k = (int)(i / N);
    bf16 h, l;
    split_bf16(W[i], h, l);
    const size_t o = (size_t)(row0 + n) * ldo + k;
    out_h[o] = h;
    if (out_l) out_l[o] = l;
  }
}

cudaError_t transpose_split_launch(const float* W, int Kin, int N, bf16* out_h, bf16* out_l, int ldo, int row0,
                                   cudaStream_t s) {
  transpose_split_kernel<<<256, 256, 0, s>>>(W, Kin, N, out_h, out_l, ldo, row0);
  return cudaGetLastError();
}

__global__ void small_matmul_kernel(const float* __restrict__ X, int R, int Kd, const float* __restrict__ W, int N,
                                    float* out) {
  const size_t total = (size_t)R * N;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total; i += (size_t)gridDim.x * blockDim.x) {
    const int n = (int)(i % N), r = (int)(i / N);
    float acc = 0.f;
    for (int k = 0; k < Kd; ++k) acc = fmaf(X[(size_t)r * Kd + k], W[(size_t)k * N + n], acc);
    out[i] = acc;
  }
}

cudaError_t small_matmul_launch(const float* X, int R, int Kd, const float* W, int N, float* out, cudaStream_t s) {
  if (R <= 0) return cudaSuccess;
  small_matmul_kernel<<<128, 256, 0, s>>>(X, R, Kd, W, N, out);
  return cudaGetLastError();
}

// A bounded wait that nothing completes: one thread initialises an mbarrier
// with an arrival count of one, never arrives on it and waits for its first
// phase through the batch kernels' bounded wait, with a limit of limit_ns.
// No copy and no tensor-core work is in flight, so giving up is always safe.
// Launched only by the wait test hook (fe_debug_wait_probe).
__global__ void wait_probe_kernel(int* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_mbar_init();
  mbar_wait_bounded_ns(&bar, 0, status, limit_ns);
}

cudaError_t wait_probe_launch(int* status, uint64_t limit_ns, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(status, limit_ns);
  return cudaGetLastError();
}

bool pdl_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("FE_NO_PDL");
    return !(v && v[0] == '1');
  }();
  return on;
}

cudaError_t misc_prepare() {
  return cudaFuncSetAttribute(compact_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 65536 + 1024);
}

}  // namespace fe
