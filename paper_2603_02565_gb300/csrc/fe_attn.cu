// Flash-style multi-head attention over request segments.
//
// Used twice per layer structure of the evaluator:
//  * element -> context cross-attention (Section 4.2): the query rows are the
//    distinct elements of request b, the keys/values its C context rows, so
//    the context K/V computed once per request serve every element;
//  * cross-sequence self-attention (Section 4.4) over the K sequence vectors.
// One CTA = 4 warps = 64 query rows of one (segment, head); the keys stream
// through shared memory in blocks of 64 with an online softmax in fp32.
// Operands are split pairs (hi + lo bf16); S = Qh Kh + Qh Kl + Ql Kh and
// O = Ph Vh + Ph Vl + Pl Vh, fp32 accumulation.
#include "fe_common.cuh"
#include "fe_kernels.h"

namespace fe {

namespace {

constexpr int BQ = 64;
constexpr int BKV = 64;

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t* r, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t* r, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}

__device__ __forceinline__ void mma16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int DH>
__host__ __device__ constexpr int pitch() { return DH + 8; }  // bf16 per shared row (16 B pad: conflict-free ldmatrix)

template <int DH>
constexpr size_t attn_smem() { return (size_t)(2 * BQ + 8 * BKV) * pitch<DH>() * 2; }

}  // namespace

template <int DH>
__global__ void __launch_bounds__(128) attn_kernel(const AttnParams p) {
  constexpr int P = pitch<DH>();
  constexpr int CH = DH / 8;  // 16-byte chunks per row
  extern __shared__ __align__(16) uint8_t smem_raw[];
  bf16* sQh = reinterpret_cast<bf16*>(smem_raw);
  bf16* sQl = sQh + BQ * P;
  bf16* sKV = sQl + BQ * P;  // [buffer 2][plane 4: Kh Kl Vh Vl][BKV * P]

  const int b = blockIdx.z, head = blockIdx.y;
  pdl_wait();
  pdl_trigger();
  const int q_cnt = p.q_cnt_dev ? p.q_cnt_dev[b] : p.q_cnt_fixed;
  const int q_begin = blockIdx.x * BQ;
  if (q_begin >= q_cnt) return;
  const int q_off = p.q_off_dev ? p.q_off_dev[b] : b * p.q_stride;
  const int kv_off = b * p.kv_stride;
  const int kv_cnt = p.kv_cnt;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int col0 = head * DH;

  for (int i = tid; i < BQ * CH; i += 128) {
    const int r = i / CH, c = i % CH;
    const bool v = q_begin + r < q_cnt;
    const size_t go = (size_t)(q_off + q_begin + (v ? r : 0)) * p.ldq + col0 + c * 8;
    cp_async16(sQh + r * P + c * 8, p.q_h + go, v);
    cp_async16(sQl + r * P + c * 8, p.q_l + go, v);
  }
  auto load_kv = [&](int kb, int buf) {
    bf16* base = sKV + buf * 4 * BKV * P;
    for (int i = tid; i < BKV * CH; i += 128) {
      const int r = i / CH, c = i % CH;
      const int key = kb * BKV + r;
      const bool v = key < kv_cnt;
      const size_t go = (size_t)(kv_off + (v ? key : 0)) * p.ldkv + col0 + c * 8;
      const int so = r * P + c * 8;
      cp_async16(base + 0 * BKV * P + so, p.k_h + go, v);
      cp_async16(base + 1 * BKV * P + so, p.k_l + go, v);
      cp_async16(base + 2 * BKV * P + so, p.v_h + go, v);
      cp_async16(base + 3 * BKV * P + so, p.v_l + go, v);
    }
  };
  load_kv(0, 0);
  cp_async_commit();

  const int nkb = (kv_cnt + BKV - 1) / BKV;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[DH / 8][4];
#pragma unroll
  for (int i = 0; i < DH / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  uint32_t qh[DH / 16][4], ql[DH / 16][4];

  for (int kb = 0; kb < nkb; ++kb) {
    const int buf = kb & 1;
    if (kb + 1 < nkb) {
      load_kv(kb + 1, buf ^ 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (kb == 0) {
#pragma unroll
      for (int kc = 0; kc < DH / 16; ++kc) {
        const int off = (warp * 16 + (lane & 15)) * P + kc * 16 + (lane >> 4) * 8;
        ldsm_x4(qh[kc], sQh + off);
        ldsm_x4(ql[kc], sQl + off);
      }
    }
    const bf16* sKh = sKV + buf * 4 * BKV * P;
    const bf16* sKl = sKh + BKV * P;
    const bf16* sVh = sKl + BKV * P;
    const bf16* sVl = sVh + BKV * P;

    // S = Q K^T over 64 keys: 8 n-blocks of 8 keys
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kc = 0; kc < DH / 16; ++kc) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int off = (np * 16 + (lane & 7) + ((lane >> 4) << 3)) * P + kc * 16 + ((lane >> 3) & 1) * 8;
        uint32_t kh[4], kl[4];
        ldsm_x4(kh, sKh + off);
        ldsm_x4(kl, sKl + off);
        mma16816(s[2 * np], qh[kc], kh[0], kh[1]);
        mma16816(s[2 * np], qh[kc], kl[0], kl[1]);
        mma16816(s[2 * np], ql[kc], kh[0], kh[1]);
        mma16816(s[2 * np + 1], qh[kc], kh[2], kh[3]);
        mma16816(s[2 * np + 1], qh[kc], kl[2], kl[3]);
        mma16816(s[2 * np + 1], ql[kc], kh[2], kh[3]);
      }
    }
    // scale (log2 domain) and mask keys past the segment
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
      const int key = kb * BKV + nb * 8 + 2 * (lane & 3);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const bool v = key + (e & 1) < kv_cnt;
        s[nb][e] = v ? s[nb][e] * p.scale_log2 : -INFINITY;
      }
      mx0 = fmaxf(mx0, fmaxf(s[nb][0], s[nb][1]));
      mx1 = fmaxf(mx1, fmaxf(s[nb][2], s[nb][3]));
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float c0 = exp2f(m0 - mn0), c1 = exp2f(m1 - mn1);
    m0 = mn0;
    m1 = mn1;
    float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) {
      s[nb][0] = exp2f(s[nb][0] - mn0);
      s[nb][1] = exp2f(s[nb][1] - mn0);
      s[nb][2] = exp2f(s[nb][2] - mn1);
      s[nb][3] = exp2f(s[nb][3] - mn1);
      rs0 += s[nb][0] + s[nb][1];
      rs1 += s[nb][2] + s[nb][3];
    }
    l0 = l0 * c0 + rs0;
    l1 = l1 * c1 + rs1;
#pragma unroll
    for (int i = 0; i < DH / 8; ++i) {
      o[i][0] *= c0;
      o[i][1] *= c0;
      o[i][2] *= c1;
      o[i][3] *= c1;
    }
    // O += P V, P as split A fragments (16 keys per k-chunk)
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      uint32_t ph[4], pl[4];
      split2(s[2 * kc][0], s[2 * kc][1], ph[0], pl[0]);
      split2(s[2 * kc][2], s[2 * kc][3], ph[1], pl[1]);
      split2(s[2 * kc + 1][0], s[2 * kc + 1][1], ph[2], pl[2]);
      split2(s[2 * kc + 1][2], s[2 * kc + 1][3], ph[3], pl[3]);
#pragma unroll
      for (int dp = 0; dp < DH / 16; ++dp) {
        const int off = (kc * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * P + dp * 16 + (lane >> 4) * 8;
        uint32_t vh[4], vl[4];
        ldsm_x4_t(vh, sVh + off);
        ldsm_x4_t(vl, sVl + off);
        mma16816(o[2 * dp], ph, vh[0], vh[1]);
        mma16816(o[2 * dp], ph, vl[0], vl[1]);
        mma16816(o[2 * dp], pl, vh[0], vh[1]);
        mma16816(o[2 * dp + 1], ph, vh[2], vh[3]);
        mma16816(o[2 * dp + 1], ph, vl[2], vl[3]);
        mma16816(o[2 * dp + 1], pl, vh[2], vh[3]);
      }
    }
    __syncthreads();  // buffer `buf` is refilled two iterations later
  }

  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float i0 = 1.f / l0, i1 = 1.f / l1;
  const int r0 = q_begin + warp * 16 + (lane >> 2);
  const int r1 = r0 + 8;
#pragma unroll
  for (int nb = 0; nb < DH / 8; ++nb) {
    const int c = col0 + nb * 8 + 2 * (lane & 3);
    uint32_t hi, lo;
    if (r0 < q_cnt) {
      split2(o[nb][0] * i0, o[nb][1] * i0, hi, lo);
      const size_t go = (size_t)(q_off + r0) * p.ldo + c;
      *reinterpret_cast<uint32_t*>(p.o_h + go) = hi;
      *reinterpret_cast<uint32_t*>(p.o_l + go) = lo;
    }
    if (r1 < q_cnt) {
      split2(o[nb][2] * i1, o[nb][3] * i1, hi, lo);
      const size_t go = (size_t)(q_off + r1) * p.ldo + c;
      *reinterpret_cast<uint32_t*>(p.o_h + go) = hi;
      *reinterpret_cast<uint32_t*>(p.o_l + go) = lo;
    }
  }
}

cudaError_t attn_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)attn_smem<32>());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)attn_smem<64>());
  return e;
}

cudaError_t attn_launch(int dh, int n_heads, int n_segments, int max_q, const AttnParams& p, cudaStream_t s) {
  if (n_segments <= 0 || max_q <= 0 || p.kv_cnt <= 0) return cudaSuccess;
  dim3 grid((unsigned)((max_q + BQ - 1) / BQ), (unsigned)n_heads, (unsigned)n_segments);
  if (dh == 32) return launch_k(attn_kernel<32>, grid, dim3(128), attn_smem<32>(), s, p);
  return launch_k(attn_kernel<64>, grid, dim3(128), attn_smem<64>(), s, p);
}

}  // namespace fe
