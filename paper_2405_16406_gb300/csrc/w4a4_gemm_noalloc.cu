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
// use the array's name as a device address, so the address is looked up with
// cudaGetSymbolAddress, with the device current, on the first call in each
// CUDA context (a context destroyed by cudaDeviceReset and created again
// loads the module again, so the address is looked up again).
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/spinq.h"
#include "spinq_internal.h"

namespace {

constexpr int64_t kNoAllocScratchBytes = SPINQ_NOALLOC_SCRATCH_BYTES;   // 8 MiB

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);

// cuCtxGetCurrent through the runtime's driver entry-point query (the
// library does not link against libcuda); null if the driver lacks it.
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  });
  return fn;
}

struct ScratchSlot {
  CUcontext ctx;
  void* addr;
};

std::mutex g_scratch_mu;
ScratchSlot g_scratch[64] = {};

// Device address of g_noalloc_scratch in the current device's context.
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  CtxGetCurrentFn get = ctx_get_current();
  if (!get) return cudaErrorDeviceUninitialized;
  CUcontext ctx = nullptr;
  if (get(&ctx) != CUDA_SUCCESS) return cudaErrorDeviceUninitialized;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (ctx != nullptr && g_scratch[dev].addr != nullptr && g_scratch[dev].ctx == ctx) {
    *out = g_scratch[dev].addr;
    return cudaSuccess;
  }
  // first call in this context (or no context yet on this thread: the
  // lookup makes the device's primary context current)
  void* p = nullptr;
  if ((e = cudaGetSymbolAddress(&p, g_noalloc_scratch)) != cudaSuccess) return e;
  if (get(&ctx) != CUDA_SUCCESS || ctx == nullptr) return cudaErrorDeviceUninitialized;
  g_scratch[dev] = ScratchSlot{ctx, p};
  *out = p;
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
  // the scratch this request needs under the current plan (0 when its plan
  // does not split K); a request beyond the fixed array is refused
  const int64_t need = spinq::w4a4_gemm_workspace_bytes(M, N, K);
  if (need > kNoAllocScratchBytes) return SPINQ_ESCRATCH;
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
