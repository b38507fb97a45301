// launch_util.h -- cached launch-configuration queries.  Each is computed once
// per (device, kernel, dynamic shared memory) and then served from a table, so
// launchers make no device queries on the hot path and stay usable while a
// stream is being captured into a CUDA graph.
#pragma once

#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <map>
#include <mutex>
#include <tuple>
#include <utility>

namespace spinq {

inline int device_sm_count() {
  static int cache[64] = {0};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return 1;
  if (cache[dev] == 0) {
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cache[dev] = sms > 0 ? sms : 1;
  }
  return cache[dev];
}

// Makes sure the kernel may use `smem` bytes of dynamic shared memory and
// returns the number of resident blocks per SM for this launch shape (at
// least 1).  The kernel's limit only ever grows (one kernel is launched with
// several sizes: lowering it for a small launch would make a larger size that
// is already cached fail to launch).
template <typename Kern>
cudaError_t prepare_launch(Kern kern, int threads, size_t smem, int* blocks_per_sm) {
  static std::mutex mu;
  static std::map<std::tuple<int, const void*, size_t, int>, int> occ;
  static std::map<std::pair<int, const void*>, size_t> limit;   // per device and kernel
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_tuple(dev, reinterpret_cast<const void*>(kern), smem, threads);
  std::lock_guard<std::mutex> lock(mu);
  auto it = occ.find(key);
  if (it != occ.end()) {
    *blocks_per_sm = it->second;
    return cudaSuccess;
  }
  size_t& lim = limit[std::make_pair(dev, reinterpret_cast<const void*>(kern))];
  if (smem > 48 * 1024 && smem > lim) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    lim = smem;
  }
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  occ[key] = per_sm;
  *blocks_per_sm = per_sm;
  return cudaSuccess;
}

// prepare_launch for a kernel that allocates `tmem_cols` columns of tensor
// memory per block.  The occupancy query answers one block per SM for every
// kernel that allocates tensor memory (measured on GB300), so the resident
// blocks come from the per-SM limits instead: shared memory (with the
// per-block reservation), registers (whole warps, 256-register granules),
// threads, and the SM's 512 tensor-memory columns.
// The answer is cached per device, kernel and launch shape (the cost models
// ask on every call).
template <typename Kern>
cudaError_t prepare_launch_tmem(Kern kern, int threads, size_t smem, int tmem_cols, int* blocks_per_sm) {
  static std::mutex mu;
  static std::map<std::tuple<int, const void*, size_t, int, int>, int> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_tuple(dev, reinterpret_cast<const void*>(kern), smem, threads, tmem_cols);
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      *blocks_per_sm = it->second;
      return cudaSuccess;
    }
  }
  int q = 0;
  cudaError_t e = prepare_launch(kern, threads, smem, &q);
  if (e != cudaSuccess) return e;
  int smem_sm = 0, smem_rsv = 0, regs_sm = 0, thr_sm = 0;
  cudaFuncAttributes fa;
  if ((e = cudaFuncGetAttributes(&fa, kern)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev)) != cudaSuccess ||
      (e = cudaDeviceGetAttribute(&smem_rsv, cudaDevAttrReservedSharedMemoryPerBlock, dev)) != cudaSuccess ||
      (e = cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev)) != cudaSuccess ||
      (e = cudaDeviceGetAttribute(&thr_sm, cudaDevAttrMaxThreadsPerMultiProcessor, dev)) != cudaSuccess)
    return e;
  const int warps = (threads + 31) / 32;
  const int regs_warp = (fa.numRegs * 32 + 255) / 256 * 256;
  int n = (int)((size_t)smem_sm / (smem + fa.sharedSizeBytes + (size_t)smem_rsv));
  if (regs_warp > 0) n = std::min(n, regs_sm / (warps * regs_warp));
  n = std::min(n, thr_sm / (warps * 32));
  if (tmem_cols > 0) n = std::min(n, 512 / tmem_cols);
  *blocks_per_sm = std::max(1, std::min(n, 32));
  std::lock_guard<std::mutex> lock(mu);
  cache[key] = *blocks_per_sm;
  return cudaSuccess;
}

// Launches still to be refused with cudaErrorLaunchOutOfResources without
// reaching the driver (a host-side fake of a failing launch, set by tests
// through spinq_debug_fail_launches; 0 in normal use).
extern std::atomic<int> g_fail_launches;

// Launch with programmatic stream serialization: the kernel may begin while
// the previous kernel in the stream finishes (it waits with griddepcontrol
// before touching global memory).  `cluster_x` > 1 adds a cluster dimension.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       int cluster_x, Args&&... args) {
  if (g_fail_launches.load(std::memory_order_relaxed) > 0 &&
      g_fail_launches.fetch_sub(1, std::memory_order_relaxed) > 0)
    return cudaErrorLaunchOutOfResources;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  int n = 1;
  if (cluster_x > 1) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)cluster_x;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    n = 2;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

}  // namespace spinq
