// quant_common.cuh -- device pieces of the Eq. 1 quantizer shared by the
// activation kernels: the row-range reduction (absmax for the symmetric
// form, min and max for the asymmetric form) and the per-row constants.
#pragma once

#include <float.h>

#include "spinq_device.cuh"

namespace spinq {

template <bool SYM>
struct Range {
  float hi, lo;
  __device__ __forceinline__ Range() : hi(SYM ? 0.f : -FLT_MAX), lo(FLT_MAX) {}
  __device__ __forceinline__ void add(float v) {
    if (SYM) {
      hi = fmaxf(hi, fabsf(v));
    } else {
      hi = fmaxf(hi, v);
      lo = fminf(lo, v);
    }
  }
  __device__ __forceinline__ void warp_reduce() {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
      if (!SYM) lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    }
  }
};

// Row-wide range over the W warps of the CTA (red: 2*W floats).
template <bool SYM, int W>
__device__ __forceinline__ void block_range(Range<SYM>& r, float* red) {
  r.warp_reduce();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (W > 1) {
    if (lane == 0) {
      red[w] = r.hi;
      red[W + w] = r.lo;
    }
    __syncthreads();
    r.hi = red[0];
    r.lo = red[W];
#pragma unroll
    for (int i = 1; i < W; ++i) {
      r.hi = fmaxf(r.hi, red[i]);
      if (!SYM) r.lo = fminf(r.lo, red[W + i]);
    }
  }
}

// Quantizer constants of Eq. 1 for the (unnormalised) row range.
template <bool SYM>
struct QParams {
  float inv, off, alpha, beta;
  __device__ __forceinline__ QParams(const Range<SYM>& r, float clip) {
    if (SYM) {
      const float m = clip * r.hi;
      alpha = m / 7.f;
      inv = m > 0.f ? 7.f / m : 0.f;
      off = 0.f;
      beta = 0.f;
    } else {
      const float h2 = clip * r.hi, l2 = clip * r.lo;
      alpha = (h2 - l2) / 15.f;
      inv = h2 > l2 ? 15.f / (h2 - l2) : 0.f;
      beta = l2;
      off = -l2 * inv;
    }
  }
  template <bool CLAMP>
  __device__ __forceinline__ uint32_t code_bits(float v) const {
    float t = fmaf(v, inv, off);
    if (CLAMP) t = SYM ? fminf(fmaxf(t, -8.f), 7.f) : fminf(fmaxf(t, 0.f), 15.f);
    return round_bits(t);
  }
};

}  // namespace spinq
