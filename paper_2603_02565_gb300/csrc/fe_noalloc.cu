// Distinct-element layout for callers that must not allocate device memory.
//
// fe_distinct_layout_noalloc runs the same compaction as the first stage of
// fe_evaluate (|U(z_b)| and each occurrence's rank among the distinct pool
// rows of its request), but its scratch -- the per-request offsets, the
// bad-request flags, the distinct-row lists, the status word and the
// last-block ticket -- lives in one file-scope __device__ array instead of a
// workspace obtained with cudaMalloc.  The array is part of the library's
// device image: every GPU that loads the library holds it until the process
// exits, and every call on that GPU shares it.
#include <mutex>

#include "fe_common.cuh"
#include "fe_kernels.h"

namespace {

constexpr int kMaxRequests = 65536;        // B limit
constexpr int kMaxDistinctRows = 1 << 20;  // limit on B * min(M, K * L)
constexpr int kMaxPool = 262144;           // M limit (shared-memory bitmap of the kernel)
// [status][ticket][off: B+1][bad: B][list: B * min(M, K*L)]
constexpr size_t kScratchInts = 2 + (size_t)(kMaxRequests + 1) + kMaxRequests + kMaxDistinctRows;

static __device__ __align__(256) int g_layout_scratch[kScratchInts];

constexpr int kMaxDevices = 64;
int* g_scratch_addr[kMaxDevices] = {};
std::once_flag g_setup_once[kMaxDevices];
cudaError_t g_setup_err[kMaxDevices] = {};

// Once per device, with that device current: the device address of the
// scratch array (host code only sees a stand-in symbol, never a usable
// pointer) and the kernel's shared-memory limit.  Neither call allocates.
cudaError_t setup_device(int dev) {
  std::call_once(g_setup_once[dev], [dev]() {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_layout_scratch);
    if (e == cudaSuccess) e = fe::misc_prepare();
    if (e == cudaSuccess) g_scratch_addr[dev] = static_cast<int*>(p);
    g_setup_err[dev] = e;
  });
  return g_setup_err[dev];
}

}  // namespace

extern "C" int fe_distinct_layout_noalloc(const int32_t* cand_idx, int B, int M, int K, int L, int32_t* U_out,
                                          int32_t* slot_out, void* stream) {
  if (B < 0 || M < 0 || K < 0 || L < 0) return FE_ERR_INVALID_ARG;
  const long long cap = (M < (long long)K * L) ? M : (long long)K * L;
  if (B > kMaxRequests || M > kMaxPool || (long long)B * cap > kMaxDistinctRows ||
      (long long)B * K * L > (1ll << 31) - 1)
    return FE_ERR_UNSUPPORTED;
  if (B == 0) return FE_OK;
  if (!U_out || (K * L > 0 && (!cand_idx || !slot_out))) return FE_ERR_INVALID_ARG;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FE_ERR_CUDA;
  if (setup_device(dev) != cudaSuccess) return FE_ERR_CUDA;
  int* base = g_scratch_addr[dev];
  int* status = base;
  unsigned* ticket = reinterpret_cast<unsigned*>(base + 1);
  int* off = base + 2;
  int* bad = off + (B + 1);
  int* list = bad + B;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the status word and the last-block ticket must start at zero every call
  e = cudaMemsetAsync(base, 0, 2 * sizeof(int), s);
  if (e == cudaSuccess)
    e = fe::compact_launch(cand_idx, B, M, K, L, (int)cap, U_out, off, bad, slot_out, list, status, ticket, s);
  return e == cudaSuccess ? FE_OK : FE_ERR_CUDA;
}
