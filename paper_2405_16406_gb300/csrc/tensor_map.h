// tensor_map.h -- host access to cuTensorMapEncodeTiled through the runtime's
// driver entry-point query, so the library needs no link against libcuda.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include <stdint.h>

#include <mutex>

namespace spinq {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

// The encoder, looked up once; null when the driver does not provide it.
inline EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// Packed 4-bit code matrix [rows][K/2] bytes, boxes of 64 bytes x box_rows.
bool encode_packed_map(CUtensorMap* map, const void* ptr, int64_t rows, int64_t K, int box_rows);
// y [M][N] fp16 for the GEMM epilogues' TMA stores: 32 x 32 boxes, 64-byte swizzle.
bool encode_y_map(CUtensorMap* map, void* y, int64_t M, int64_t N);

}  // namespace spinq
