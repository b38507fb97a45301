// rotate_quant_8bit.cu -- the quantizers of the 8-bit linears (main results
// table, 4-8-x rows; appendix "Latency measurement on GPU", FP8 setting):
// the online rotation x R (Sec. 3.1, skipped when there is none) followed by
//
//   kFmtInt8Planes  Eq. 1 with N = 8 (per token): code c = q (symmetric) or
//                   u - 128 (asymmetric), stored as the two E4M3 planes the
//                   W4A8 GEMM reads: row [2K] bytes, byte k = E4M3(16 (c >> 4)),
//                   byte K + k = E4M3(c & 15) (both exact);
//   kFmtE4M3        per-row FP8: alpha = clip max|x| / 448, code =
//                   E4M3(x / alpha) rounded to nearest even, saturating;
//   kFmtInt4Bytes   Eq. 1 with N = 4, symmetric per output channel (weights of
//                   the W4A8 linear): each 4-bit code stored as one E4M3 byte,
//                   plus the row sum of the codes.
//
// One CTA of 256 threads per row (persistent over rows).  The row is held in
// shared memory as fp32; the power-of-two factor is a radix-2 FWHT over the
// fast index, the small Paley factor a dense +-1 product over the slow index.
// Codes are taken on the unnormalised row; alpha and beta carry 1/sqrt(K).
#include <cuda_fp16.h>
#include <float.h>

#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ uint32_t e4m3x2(float lo, float hi) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}

template <int FMT, bool SYM, bool CLAMP, int NS>
__global__ void __launch_bounds__(kThreads) rq8_rows_kernel(Rq8Args a) {
  extern __shared__ float s[];
  __shared__ float red_hi[kThreads / 32], red_lo[kThreads / 32];
  __shared__ int red_sum[kThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int K = (int)a.K;
  const int P = a.n_pow2;
  const int log2P = a.n_small ? 31 - __clz(P) : 0;
  const __half* __restrict__ x = reinterpret_cast<const __half*>(a.x);
  pdl_wait();
  pdl_trigger();

  for (int64_t row = blockIdx.x; row < a.rows; row += gridDim.x) {
    const __half* xr = x + row * a.ldx;
    for (int c = tid; c < K / 8; c += kThreads) {
      const uint4 v = __ldg(reinterpret_cast<const uint4*>(xr) + c);
      const __half2* h = reinterpret_cast<const __half2*>(&v);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = __half22float2(h[e]);
        *reinterpret_cast<float2*>(s + 8 * c + 2 * e) = f;
      }
    }
    __syncthreads();
    if (a.n_small) {
      for (int lh = 0; lh < log2P; ++lh) {
        const int h = 1 << lh;
        for (int p = tid; p < K / 2; p += kThreads) {
          const int seg = p >> (log2P - 1);
          const int l = p & ((P >> 1) - 1);
          const int j = ((l >> lh) << (lh + 1)) | (l & (h - 1));
          const int i0 = seg * P + j;
          const float u = s[i0], w = s[i0 + h];
          s[i0] = u + w;
          s[i0 + h] = u - w;
        }
        __syncthreads();
      }
      if constexpr (NS > 1) {
        // the small factor, unrolled at its compile-time order (registers only)
        uint32_t neg[NS];
#pragma unroll
        for (int ip = 0; ip < NS; ++ip) neg[ip] = a.hs.neg[ip];
        for (int j = tid; j < P; j += kThreads) {
          float t[NS];
#pragma unroll
          for (int ip = 0; ip < NS; ++ip) t[ip] = s[ip * P + j];
#pragma unroll
          for (int i = 0; i < NS; ++i) {
            float acc = 0.f;
#pragma unroll
            for (int ip = 0; ip < NS; ++ip) acc += ((neg[ip] >> i) & 1u) ? -t[ip] : t[ip];
            s[i * P + j] = acc;
          }
        }
        __syncthreads();
      }
    }
    // row range
    float hi = SYM ? 0.f : -FLT_MAX, lo = FLT_MAX;
    for (int k = tid; k < K; k += kThreads) {
      const float v = s[k];
      if (SYM) {
        hi = fmaxf(hi, fabsf(v));
      } else {
        hi = fmaxf(hi, v);
        lo = fminf(lo, v);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    }
    if (lane == 0) {
      red_hi[warp] = hi;
      red_lo[warp] = lo;
    }
    __syncthreads();
    hi = red_hi[0];
    lo = red_lo[0];
    for (int w = 1; w < kThreads / 32; ++w) {
      hi = fmaxf(hi, red_hi[w]);
      lo = fminf(lo, red_lo[w]);
    }
    // per-row constants (unnormalised row)
    float inv, off = 0.f, alpha, beta = 0.f;
    if (FMT == kFmtE4M3) {
      const float m = a.clip * hi;
      alpha = m * (1.f / 448.f);
      inv = m > 0.f ? 448.f / m : 0.f;
    } else {
      const float qmax = FMT == kFmtInt8Planes ? 127.f : 7.f;
      if (SYM) {
        const float m = a.clip * hi;
        alpha = m / qmax;
        inv = m > 0.f ? qmax / m : 0.f;
      } else {
        const float h2 = a.clip * hi, l2 = a.clip * lo;
        alpha = (h2 - l2) / 255.f;
        inv = h2 > l2 ? 255.f / (h2 - l2) : 0.f;
        beta = l2;
        off = -l2 * inv;
      }
    }
    int csum = 0;
    uint8_t* out = a.codes + row * (FMT == kFmtInt8Planes ? 2 * a.K : a.K);
    for (int c = tid; c < K / 8; c += kThreads) {
      uint32_t w0[2] = {0, 0}, w1[2] = {0, 0};
#pragma unroll
      for (int e = 0; e < 8; e += 2) {
        float t0 = fmaf(s[8 * c + e], inv, off), t1 = fmaf(s[8 * c + e + 1], inv, off);
        uint32_t b0, b1;
        if (FMT == kFmtE4M3) {
          b0 = e4m3x2(t0, t1);   // both bytes at once: lo element in the low byte
          b1 = 0;
        } else {
          if (FMT == kFmtInt8Planes) {
            if (CLAMP) {
              t0 = SYM ? fminf(fmaxf(t0, -128.f), 127.f) : fminf(fmaxf(t0, 0.f), 255.f);
              t1 = SYM ? fminf(fmaxf(t1, -128.f), 127.f) : fminf(fmaxf(t1, 0.f), 255.f);
            }
            const int c0 = __float2int_rn(t0) - (SYM ? 0 : 128), c1 = __float2int_rn(t1) - (SYM ? 0 : 128);
            b0 = e4m3x2((float)(16 * (c0 >> 4)), (float)(16 * (c1 >> 4)));
            b1 = e4m3x2((float)(c0 & 15), (float)(c1 & 15));
          } else {   // kFmtInt4Bytes: symmetric 4-bit codes, one per byte
            if (CLAMP) {
              t0 = fminf(fmaxf(t0, -8.f), 7.f);
              t1 = fminf(fmaxf(t1, -8.f), 7.f);
            }
            const int c0 = __float2int_rn(t0), c1 = __float2int_rn(t1);
            csum += c0 + c1;
            b0 = e4m3x2((float)c0, (float)c1);
            b1 = 0;
          }
        }
        w0[e >> 2] |= b0 << (8 * (e & 3));
        w1[e >> 2] |= b1 << (8 * (e & 3));
      }
      *reinterpret_cast<uint2*>(out + 8 * c) = make_uint2(w0[0], w0[1]);
      if (FMT == kFmtInt8Planes) *reinterpret_cast<uint2*>(out + a.K + 8 * c) = make_uint2(w1[0], w1[1]);
    }
    if (FMT == kFmtInt4Bytes) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) csum += __shfl_xor_sync(0xffffffffu, csum, o);
      if (lane == 0) red_sum[warp] = csum;
    }
    __syncthreads();
    if (tid == 0) {
      a.scale[row] = alpha * a.norm;
      if (!SYM && FMT == kFmtInt8Planes) a.zero[row] = beta * a.norm;
      if (FMT == kFmtInt4Bytes && a.rowsum) {
        int tot = 0;
        for (int w = 0; w < kThreads / 32; ++w) tot += red_sum[w];
        a.rowsum[row] = tot;
      }
    }
    __syncthreads();
  }
}

template <int FMT, bool SYM, bool CLAMP, int NS>
cudaError_t launch_ns(const Rq8Args& a, cudaStream_t stream) {
  const size_t smem = sizeof(float) * (size_t)a.K;
  auto kern = rq8_rows_kernel<FMT, SYM, CLAMP, NS>;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, kThreads, smem, &per_sm);
  if (e != cudaSuccess) return e;
  const int64_t cap = (int64_t)device_sm_count() * per_sm;
  const int64_t grid = a.rows < cap ? a.rows : cap;
  e = launch_pdl(kern, dim3((unsigned)grid), dim3(kThreads), smem, stream, 1, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int FMT, bool SYM, bool CLAMP>
cudaError_t launch_t(const Rq8Args& a, cudaStream_t stream) {
  switch (a.n_small) {
    case 12: return launch_ns<FMT, SYM, CLAMP, 12>(a, stream);
    case 20: return launch_ns<FMT, SYM, CLAMP, 20>(a, stream);
    case 28: return launch_ns<FMT, SYM, CLAMP, 28>(a, stream);
  }
  return launch_ns<FMT, SYM, CLAMP, 1>(a, stream);
}

template <int FMT>
cudaError_t launch_fmt(const Rq8Args& a, cudaStream_t stream) {
  const bool clamp = a.clip < 1.0f;
  if (a.symmetric) return clamp ? launch_t<FMT, true, true>(a, stream) : launch_t<FMT, true, false>(a, stream);
  return clamp ? launch_t<FMT, false, true>(a, stream) : launch_t<FMT, false, false>(a, stream);
}

}  // namespace

cudaError_t launch_rotate_quant_8bit(const Rq8Args& a, cudaStream_t stream) {
  if (a.rows == 0) return cudaSuccess;
  // a Paley rotation with the unclipped activation formats: the Paley kernel
  bool handled = false;
  const cudaError_t ep = launch_rotate_quant_8bit_paley(a, stream, &handled);
  if (ep != cudaSuccess || handled) return ep;
  switch (a.format) {
    case kFmtInt8Planes: return launch_fmt<kFmtInt8Planes>(a, stream);
    case kFmtE4M3: return a.symmetric ? launch_fmt<kFmtE4M3>(a, stream) : cudaErrorInvalidValue;
    case kFmtInt4Bytes: return a.symmetric ? launch_fmt<kFmtInt4Bytes>(a, stream) : cudaErrorInvalidValue;
  }
  return cudaErrorNotSupported;
}

}  // namespace spinq
