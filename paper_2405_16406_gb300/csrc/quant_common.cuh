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
  // two values at once with the 3-input min/max of sm_100+
  __device__ __forceinline__ void add2(float a, float b) {
    if (SYM) {
      asm("max.f32 %0, %0, %1, %2;" : "+f"(hi) : "f"(fabsf(a)), "f"(fabsf(b)));
    } else {
      asm("max.f32 %0, %0, %1, %2;" : "+f"(hi) : "f"(a), "f"(b));
      asm("min.f32 %0, %0, %1, %2;" : "+f"(lo) : "f"(a), "f"(b));
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
    if (SYM && !CLAMP) return __float_as_uint(fmaf(v, inv, kRoundMagic));  // one rounding: rint(v/alpha)
    float t = fmaf(v, inv, off);
    if (CLAMP) t = SYM ? fminf(fmaxf(t, -8.f), 7.f) : fminf(fmaxf(t, 0.f), 15.f);
    return round_bits(t);
  }
};

// ---------------------------------------------------------------------------
// RowStream: rows of a row-major fp16 matrix streamed into shared memory with
// TMA bulk copies, NST rows ahead, for a CTA that walks rows r0, r0 + G, ...
// Thread 0 issues; every thread waits.  A stage is refilled (release) once
// the CTA has read it.  Waits are bounded in time and set `*abort` on expiry.
// ---------------------------------------------------------------------------
template <int NST>
struct RowStream {
  uint8_t* stage0;      // NST stages of `stage_bytes`
  uint32_t stage_bytes;
  uint64_t* bars;       // NST mbarriers
  const uint8_t* src;   // matrix base
  int64_t row_bytes;    // pitch
  uint32_t copy_bytes;  // bytes copied per row (multiple of 16)
  int64_t rows, r0, G;
  int issued;           // iterations issued so far (thread 0)

  __device__ __forceinline__ void init() {
    if (threadIdx.x == 0)
      for (int s = 0; s < NST; ++s) mbar_init(&bars[s], 1);
  }
  __device__ __forceinline__ void issue(int iter) {
    const int64_t row = r0 + (int64_t)iter * G;
    if (row >= rows) return;
    const int s = iter % NST;
    fence_proxy_async_smem();
    mbar_arrive_expect_tx(&bars[s], copy_bytes);
    bulk_load(stage0 + (size_t)s * stage_bytes, src + row * row_bytes, copy_bytes, &bars[s]);
    issued = iter + 1;
  }
  // thread 0, after init() and a CTA barrier
  __device__ __forceinline__ void prologue() {
    issued = 0;
    if (threadIdx.x == 0)
      for (int i = 0; i < NST; ++i) issue(i);
  }
  __device__ __forceinline__ uint8_t* stage(int iter) const { return stage0 + (size_t)(iter % NST) * stage_bytes; }
  // every thread; false on timeout or abort
  __device__ __forceinline__ bool wait(int iter, volatile int* abort, uint64_t limit_ns) {
    const uint32_t par = (uint32_t)(iter / NST) & 1u;
    if (mbar_try_wait(&bars[iter % NST], par)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(&bars[iter % NST], par)) {
      if (*abort || globaltimer_ns() - t0 > limit_ns) {
        *abort = 1;
        return false;
      }
    }
    return true;
  }
  // thread 0, after the CTA has finished reading stage(iter)
  __device__ __forceinline__ void release(int iter) {
    if (threadIdx.x == 0) issue(iter + NST);
  }
  // thread 0: let copies in flight land before the CTA exits (abort path)
  __device__ __forceinline__ void drain(int iter, uint64_t limit_ns) {
    if (threadIdx.x != 0) return;
    for (int j = iter; j < issued; ++j) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&bars[j % NST], (j / NST) & 1) && globaltimer_ns() - t0 < limit_ns) {
      }
    }
  }
};

}  // namespace spinq
