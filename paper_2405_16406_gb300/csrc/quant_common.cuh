// quant_common.cuh -- device pieces of the Eq. 1 quantizer shared by the
// activation kernels: the row-range reduction (absmax for the symmetric
// form, min and max for the asymmetric form) and the per-row constants.
#pragma once

#include <float.h>

#include "spinq_device.cuh"
#include "spinq_internal.h"

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
  __device__ __forceinline__ void add_pair(F2 v) {
    float a, b;
    f2_split(v, a, b);
    add2(a, b);
  }
  // over the 32 lanes of a converged warp, with the float warp reductions of
  // sm_100+ (max and min are exact, so this equals the shuffle tree)
  __device__ __forceinline__ void warp_reduce() {
    asm volatile("redux.sync.max.f32 %0, %0, 0xffffffff;" : "+f"(hi));
    if (!SYM) asm volatile("redux.sync.min.f32 %0, %0, 0xffffffff;" : "+f"(lo));
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
  F2 inv2, bias2;  // (inv, inv); (magic, magic) for SYM, (off, off) otherwise
  __device__ __forceinline__ QParams(const Range<SYM>& r, float clip) {
    // alpha is a scale factor (a product, no division needed); the codes use
    // the correctly rounded reciprocal step inv
    if (SYM) {
      const float m = clip * r.hi;
      alpha = m * (1.f / 7.f);
      inv = m > 0.f ? 7.f / m : 0.f;
      off = 0.f;
      beta = 0.f;
    } else {
      const float h2 = clip * r.hi, l2 = clip * r.lo;
      alpha = (h2 - l2) * (1.f / 15.f);
      inv = h2 > l2 ? 15.f / (h2 - l2) : 0.f;
      beta = l2;
      off = -l2 * inv;
    }
    inv2 = f2_make(inv, inv);
    bias2 = SYM ? f2_make(kRoundMagic, kRoundMagic) : f2_make(off, off);
  }
  template <bool CLAMP>
  __device__ __forceinline__ uint32_t code_bits(float v) const {
    if (SYM && !CLAMP) return __float_as_uint(fmaf(v, inv, kRoundMagic));  // one rounding: rint(v/alpha)
    float t = fmaf(v, inv, off);
    if (CLAMP) t = SYM ? fminf(fmaxf(t, -8.f), 7.f) : fminf(fmaxf(t, 0.f), 15.f);
    return round_bits(t);
  }
  // code_bits() of both lanes of a pair, on the packed fp32 pipe: the same
  // operations in the same order, so the same bits
  template <bool CLAMP>
  __device__ __forceinline__ void code_bits2(F2 v, uint32_t& b0, uint32_t& b1) const {
    float x0, x1;
    if (CLAMP) {
      f2_split(v, x0, x1);
      b0 = code_bits<true>(x0);
      b1 = code_bits<true>(x1);
      return;
    }
    F2 t = f2_fma(v, inv2, bias2);
    if (!SYM) t = f2_add(t, f2_make(kRoundMagic, kRoundMagic));
    f2_split(t, x0, x1);
    b0 = __float_as_uint(x0);
    b1 = __float_as_uint(x1);
  }
};

__device__ __forceinline__ uint32_t e4m3x2_bits(float lo, float hi) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}

// The 8-bit quantizers of rotate_quant_8bit.cu (unclipped forms) on a row
// range: E4M3 codes x / alpha with alpha = max|x| / 448; int8 codes
// c = rint(x / alpha) (symmetric, alpha = max|x| / 127) or rint((x - beta) /
// alpha) - 128 (asymmetric, alpha = (max - min) / 255), stored as the planes
// E4M3(16 floor(c / 16)) and E4M3(c mod 16).  rint is the 1.5 2^23 rounding
// (to nearest even, as the other kernel's conversion), floor(c / 16) is
// rint((c - 7.5) / 16), exact for integer c; every value is exact in E4M3.
template <bool SYM>
struct Quant8 {
  float inv, off, alpha, beta;
  __device__ __forceinline__ Quant8(const Range<SYM>& r, float clip, bool e4m3) {
    off = 0.f;
    beta = 0.f;
    if (e4m3) {
      const float m = clip * r.hi;
      alpha = m * (1.f / 448.f);
      inv = m > 0.f ? 448.f / m : 0.f;
    } else if (SYM) {
      const float m = clip * r.hi;
      alpha = m / 127.f;
      inv = m > 0.f ? 127.f / m : 0.f;
    } else {
      const float h2 = clip * r.hi, l2 = clip * r.lo;
      alpha = (h2 - l2) / 255.f;
      inv = h2 > l2 ? 255.f / (h2 - l2) : 0.f;
      beta = l2;
      off = -l2 * inv;
    }
  }
  // the codes of 8 consecutive elements (4 pairs): E4M3 bytes in `hi`, or the
  // two planes in `hi` (16 floor(c / 16)) and `lo` (c mod 16)
  template <int F8>
  __device__ __forceinline__ void codes8(const F2 (&v)[4], uint2& hi, uint2& lo) const {
    uint32_t hb[4], lb[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float x0, x1;
      f2_split(v[q], x0, x1);
      if (F8 == kFmtE4M3) {
        hb[q] = e4m3x2_bits(fmaf(x0, inv, off), fmaf(x1, inv, off));
        lb[q] = 0;
      } else {
        float c0 = (fmaf(x0, inv, off) + kRoundMagic) - kRoundMagic;
        float c1 = (fmaf(x1, inv, off) + kRoundMagic) - kRoundMagic;
        if (!SYM) c0 -= 128.f, c1 -= 128.f;
        const float q0 = (fmaf(c0, 0.0625f, -0.46875f) + kRoundMagic) - kRoundMagic;
        const float q1 = (fmaf(c1, 0.0625f, -0.46875f) + kRoundMagic) - kRoundMagic;
        hb[q] = e4m3x2_bits(16.f * q0, 16.f * q1);
        lb[q] = e4m3x2_bits(fmaf(-16.f, q0, c0), fmaf(-16.f, q1, c1));
      }
    }
    hi = make_uint2(hb[0] | (hb[1] << 16), hb[2] | (hb[3] << 16));
    lo = make_uint2(lb[0] | (lb[1] << 16), lb[2] | (lb[3] << 16));
  }
};

// ---------------------------------------------------------------------------
// RowStream: rows of a row-major fp16 matrix streamed into shared memory with
// TMA bulk copies, NST rows ahead, for a CTA that walks rows r0, r0 + G, ...
// A row is copied as `nseg` segments of `seg_bytes` (consecutive in global
// memory, `seg_stride` bytes apart in shared memory, so that a kernel can pad
// its segments).  Every thread waits; a stage is refilled once the CTA has
// read it, by whichever warp reads it last (release_warp) or by thread 0
// after a CTA barrier (release).  Waits are bounded in time and set `*abort`
// on expiry.
// ---------------------------------------------------------------------------
template <int NST>
struct RowStream {
  uint8_t* stage0;      // NST stages of `stage_bytes`
  uint32_t stage_bytes;
  uint64_t* bars;       // NST mbarriers
  const uint8_t* src;   // matrix base
  int64_t row_bytes;    // pitch
  uint32_t seg_bytes;   // bytes per segment (multiple of 16)
  uint32_t nseg;        // segments per row
  uint32_t seg_stride;  // shared-memory distance of consecutive segments
  int64_t rows, r0, G;

  __device__ __forceinline__ void init() {
    if (threadIdx.x == 0)
      for (int s = 0; s < NST; ++s) mbar_init(&bars[s], 1);
  }
  __device__ __forceinline__ bool has(int iter) const { return r0 + (int64_t)iter * G < rows; }
  __device__ __forceinline__ void issue(int iter) {
    if (!has(iter)) return;
    const int64_t row = r0 + (int64_t)iter * G;
    const int s = iter % NST;
    uint8_t* dst = stage0 + (size_t)s * stage_bytes;
    const uint8_t* from = src + row * row_bytes;
    fence_proxy_async_smem();
    mbar_arrive_expect_tx(&bars[s], seg_bytes * nseg);
#pragma unroll 1
    for (uint32_t i = 0; i < nseg; ++i) bulk_load(dst + i * seg_stride, from + (size_t)i * seg_bytes, seg_bytes, &bars[s]);
  }
  // thread 0, after init() and a CTA barrier
  __device__ __forceinline__ void prologue() {
    if (threadIdx.x == 0)
      for (int i = 0; i < NST; ++i) issue(i);
  }
  __device__ __forceinline__ uint8_t* stage(int iter) const { return stage0 + (size_t)(iter % NST) * stage_bytes; }
  // every thread; false on timeout or abort
  __device__ __forceinline__ bool wait(int iter, volatile int* abort, uint64_t limit_ns) {
    return mbar_wait_backoff(&bars[iter % NST], (uint32_t)(iter / NST) & 1u, abort, limit_ns);
  }
  // thread 0, after a CTA barrier that follows the last read of stage(iter)
  __device__ __forceinline__ void release(int iter) {
    if (threadIdx.x == 0) issue(iter + NST);
  }
  // every warp, once it has finished reading stage(iter) (its loads have
  // returned); the last of `nwarps` warps to get here refills the stage.
  // `count` is a shared-memory word that starts at 0 and is left at 0.
  __device__ __forceinline__ void release_warp(int iter, int* count, int nwarps) {
    __syncwarp();
    if ((threadIdx.x & 31) == 0) {
      __threadfence_block();
      if (atomicAdd(count, 1) == nwarps - 1) {
        *count = 0;
        issue(iter + NST);
      }
    }
  }
  // thread 0 on the abort path at iteration `iter` (every earlier stage was
  // released, so the copies of iter .. iter + NST - 1 may be in flight): let
  // them land before the CTA exits
  __device__ __forceinline__ void drain(int iter, uint64_t limit_ns) {
    if (threadIdx.x != 0) return;
    for (int j = iter; j < iter + NST; ++j) {
      if (!has(j)) break;
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&bars[j % NST], (j / NST) & 1) && globaltimer_ns() - t0 < limit_ns) {
      }
    }
  }
};

}  // namespace spinq
