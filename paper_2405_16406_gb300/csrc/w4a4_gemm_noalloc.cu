// w4a4_gemm_noalloc.cu -- spinq_w4a4_gemm_noalloc: the split-K W4A4 GEMM with
// its workspace in a fixed device array that the library itself owns, so the
// caller passes only inputs and outputs.
//
// Who needs this: code that must not allocate device memory at the point
// where it runs the layer.  Examples are serving runtimes that reserve their
// whole memory budget at start-up and forbid later allocations, code running
// on threads that may not call into an allocator while other streams are
// being captured into CUDA graphs, and embedders that have no device
// allocator of their own to hand a workspace from.
//
// The scratch is the static array below (kNoAllocScratchBytes); every GPU
// that loads the library holds it until the process exits.  Host code cannot
// use the array's name as a device address, so the address is looked up once
// per device, with that device current, through cudaGetSymbolAddress.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/spinq.h"
#include "spinq_internal.h"

namespace {

constexpr int64_t kNoAllocScratchBytes = int64_t(8) << 20;   // 8 MiB

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_scratch_mu;
void* g_scratch_addr[64] = {nullptr};

// Device address of g_noalloc_scratch on the current device (looked up on the
// first call for that device).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

bool is_aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" spinq_status spinq_w4a4_gemm_noalloc(const uint8_t* a_codes, const float* a_scale,
                                                const float* a_zero, const uint8_t* w_codes,
                                                const float* w_scale, const int32_t* w_rowsum,
                                                int64_t M, int64_t N, int64_t K, void* y_f16,
                                                int32_t* acc_out, void* stream) {
  if (M < 0 || N < 0 || K <= 0) return SPINQ_EINVAL;
  if (M > 0 && N > 0 && (!a_codes || !a_scale || !w_codes || !w_scale || !w_rowsum || !y_f16))
    return SPINQ_EINVAL;
  if (K % 128 != 0 || N % 16 != 0) return SPINQ_EINVAL;
  if (!is_aligned16(a_codes) || !is_aligned16(w_codes) || !is_aligned16(y_f16) || !is_aligned16(w_scale) ||
      !is_aligned16(w_rowsum) || (acc_out && !is_aligned16(acc_out)))
    return SPINQ_EINVAL;
  if (K > 65536 || M > INT32_MAX || N > INT32_MAX) return SPINQ_EUNSUPPORTED;
  if (M == 0 || N == 0) return SPINQ_OK;
  // a split whose partial sums do not fit the scratch is not taken: the
  // tiles then keep their whole K range
  int64_t need = spinq::w4a4_gemm_workspace_bytes(M, N, K);
  if (need > kNoAllocScratchBytes) need = 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  void* ws = nullptr;
  if (need > 0) {
    if (scratch_address(&ws) != cudaSuccess) return SPINQ_ECUDA;
    // the array still holds what the previous call left in it: the partial
    // accumulators and tile counters must start at zero
    if (cudaMemsetAsync(ws, 0, (size_t)need, s) != cudaSuccess) return SPINQ_ECUDA;
  }
  const spinq::GemmArgs g{a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y_f16, acc_out};
  const cudaError_t e = spinq::launch_w4a4_gemm_splitk(g, ws, need, s);
  if (e == cudaSuccess) return SPINQ_OK;
  return e == cudaErrorNotSupported ? SPINQ_EUNSUPPORTED : SPINQ_ECUDA;
}
