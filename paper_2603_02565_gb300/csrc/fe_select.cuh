// Eq. 1's argmax over each request's K candidate scores, fused into the
// kernel that computes the scores (the score head's epilogue).
//
// Row s is sequence k = s % K of request b = s / K.  Every row folds its score
// into a per-request 64-bit atomicMax of (order-preserving score bits << 32 |
// ~k), so that the largest score wins and ties go to the smaller k; a NaN
// score sets the request's flag instead; a rejected request (bad[b]) gets NaN
// scores.  Every CTA of the launch then takes a ticket (atomic count, no
// waits); the last one writes best (-1 for a rejected request or a NaN
// score, with ST_NUMERIC for the latter), copies the batch status word into
// the page-locked host word and clears the status, the keys, the flags and the
// ticket for the next batch.
#pragma once
#include <cstdint>

#include "fe_kernels.h"

namespace fe {


// Order-preserving map of a (non-NaN) float to 32 bits: a > b iff key(a) > key(b).
__device__ __forceinline__ uint32_t sel_ordered_bits(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Row `row`'s score f folded into its request's maximum (NaN for a rejected
// request), for the 32 rows of a warp (all lanes call it, `valid` per lane):
// lanes of the same request (contiguous rows) first take their maximum by a
// segmented shuffle reduction, so that each request sees one atomic per warp.
__device__ __forceinline__ void sel_fold_warp(const SelArgs& s, int row, float& f, bool valid) {
  const int lane = threadIdx.x & 31;
  const int b = valid ? row / s.K : -1;
  unsigned long long key = 0ull;
  if (valid) {
    const int k = row - b * s.K;
    if (s.bad[b])
      f = __int_as_float(0x7fc00000);
    else if (f != f)
      atomicOr(s.nan + b, 1);
    else
      key = ((unsigned long long)sel_ordered_bits(f) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)k);
  }
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {  // lane i: maximum over [i, i + 2 off) within its request
    const unsigned long long ok = __shfl_down_sync(0xffffffffu, key, off);
    const int ob = __shfl_down_sync(0xffffffffu, b, off);
    if (lane + off < 32 && ob == b && ok > key) key = ok;
  }
  const int pb = __shfl_up_sync(0xffffffffu, b, 1);
  if (valid && key != 0ull && (lane == 0 || pb != b)) atomicMax(s.keys + b, key);  // the request's first lane
}

static __device__ void sel_finish(const SelArgs& s) {
  __threadfence();
  for (int b = threadIdx.x; b < s.B; b += blockDim.x) {
    const unsigned long long key = atomicExch(s.keys + b, 0ull);  // through L2
    const int nan = atomicExch(s.nan + b, 0);
    int best = -1;
    if (!s.bad[b] && !nan && key != 0ull) best = (int)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
    if (!s.bad[b] && nan) atomicOr(s.status, ST_NUMERIC);
    s.best[b] = best;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int st = atomicExch(s.status, 0);
    *s.ticket = 0u;
    *reinterpret_cast<volatile int*>(s.host_status) = st;
    __threadfence_system();
  }
}

// Called by every thread of every CTA once its rows are folded; `flag` is a
// shared word the CTA no longer uses.
static __device__ void sel_ticket(const SelArgs& s, volatile uint32_t* flag) {
  __threadfence();  // this thread's folds before the count
  __syncthreads();
  if (threadIdx.x == 0) *flag = atomicAdd(s.ticket, 1u) == gridDim.x - 1 ? 1u : 0u;
  __syncthreads();
  if (*flag) sel_finish(s);
}

}  // namespace fe
