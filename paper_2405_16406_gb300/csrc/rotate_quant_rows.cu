// rotate_quant_rows.cu -- one CTA per row: rotation x R (Sec. 3.1, R4 and the
// weight merge W' = W R) followed by the Eq. 1 quantizer of the whole row.
//
// The row is held in shared memory as fp32 (K <= 32768 -> 128 KB).  The
// power-of-two factor is a radix-2 FWHT over the fast index, one butterfly
// stage per barrier; the small Paley factor is a dense +-1 product over the
// slow index, one column per thread.  The 1/sqrt(K) normalization is not
// applied to the elements: Eq. 1 codes do not change when a row is scaled,
// so only alpha and beta are multiplied by it.
//
// This kernel serves the offline weight path (any supported size) and every
// activation shape that the specialised kernel does not cover.
#include <cuda_fp16.h>
#include <float.h>

#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <bool SYM, bool ROWSUM, bool CLAMP>
__global__ void __launch_bounds__(kThreads) rotate_quant_rows_kernel(RotQuantArgs a) {
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
      const uint32_t sb = a.signs ? a.signs[c] : 0u;   // random signs of R = S H (bit e: element 8c + e)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = __half22float2(h[e]);
        s[8 * c + 2 * e] = (sb >> (2 * e)) & 1u ? -f.x : f.x;
        s[8 * c + 2 * e + 1] = (sb >> (2 * e + 1)) & 1u ? -f.y : f.y;
      }
    }
    __syncthreads();

    if (a.n_small) {
      // x[i][:] <- x[i][:] H_P for every slow index i (radix-2 stages)
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
      // y[i][j] = sum_i' x[i'][j] H_s[i'][i]
      const int ns = a.n_small;
      if (ns > 1) {
        for (int j = tid; j < P; j += kThreads) {
          float t[32];
          for (int ip = 0; ip < ns; ++ip) t[ip] = s[ip * P + j];
          for (int i = 0; i < ns; ++i) {
            float acc = 0.f;
            for (int ip = 0; ip < ns; ++ip) acc += ((a.hs.neg[ip] >> i) & 1u) ? -t[ip] : t[ip];
            s[i * P + j] = acc;  // column j only read above by this thread
          }
        }
        __syncthreads();
      }
    }

    // range of the row
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
    hi = warp_max(hi);
    if (!SYM) lo = warp_min(lo);
    if (lane == 0) {
      red_hi[warp] = hi;
      red_lo[warp] = lo;
    }
    __syncthreads();
    hi = red_hi[0];
    lo = red_lo[0];
    for (int w = 1; w < kThreads / 32; ++w) {
      hi = fmaxf(hi, red_hi[w]);
      if (!SYM) lo = fminf(lo, red_lo[w]);
    }
    // Eq. 1 on the unnormalised row; alpha and beta carry the normalisation.
    float inv, off, alpha, beta = 0.f;
    if (SYM) {
      const float m = a.clip * hi;
      alpha = m / 7.f;
      inv = m > 0.f ? 7.f / m : 0.f;
      off = 0.f;
    } else {
      const float h2 = a.clip * hi, l2 = a.clip * lo;
      alpha = (h2 - l2) / 15.f;
      inv = h2 > l2 ? 15.f / (h2 - l2) : 0.f;
      beta = l2;
      off = -l2 * inv;
    }

    int csum = 0;
    uint32_t* out = reinterpret_cast<uint32_t*>(a.codes + row * (a.K / 2));
    for (int c = tid; c < K / 8; c += kThreads) {
      uint32_t r[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        float t = fmaf(s[8 * c + e], inv, off);
        if (CLAMP) t = SYM ? fminf(fmaxf(t, -8.f), 7.f) : fminf(fmaxf(t, 0.f), 15.f);
        r[e] = round_bits(t);
        if (ROWSUM) csum += (int)(r[e] - __float_as_uint(kRoundMagic));
      }
      out[c] = pack8_nibbles(r);
    }
    if (ROWSUM) {
      csum = warp_sum(csum);
      if (lane == 0) red_sum[warp] = csum;
    }
    __syncthreads();
    if (tid == 0) {
      a.scale[row] = alpha * a.norm;
      if (!SYM) a.zero[row] = beta * a.norm;
      if (ROWSUM) {
        int tot = 0;
        for (int w = 0; w < kThreads / 32; ++w) tot += red_sum[w];
        a.rowsum[row] = tot;
      }
    }
    __syncthreads();
  }
}

template <bool SYM, bool ROWSUM, bool CLAMP>
cudaError_t launch_t(const RotQuantArgs& a, cudaStream_t stream) {
  const size_t smem = sizeof(float) * (size_t)a.K;
  auto kern = rotate_quant_rows_kernel<SYM, ROWSUM, CLAMP>;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, kThreads, smem, &per_sm);
  if (e != cudaSuccess) return e;
  const int64_t cap = (int64_t)device_sm_count() * per_sm * 4;
  const int64_t grid = a.rows < cap ? a.rows : cap;
  e = launch_pdl(kern, dim3((unsigned)grid), dim3(kThreads), smem, stream, 1, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rotate_quant_rows(const RotQuantArgs& a, cudaStream_t stream) {
  if (a.rows == 0) return cudaSuccess;
  bool handled = false;
  cudaError_t e = launch_rotate_quant_act_fast(a, stream, &handled);
  if (handled || e != cudaSuccess) return e;
  e = launch_rotate_quant_act_paley(a, stream, &handled);
  if (handled || e != cudaSuccess) return e;
  const bool clamp = a.clip < 1.0f;
  if (a.symmetric) {
    if (a.rowsum) return clamp ? launch_t<true, true, true>(a, stream) : launch_t<true, true, false>(a, stream);
    return clamp ? launch_t<true, false, true>(a, stream) : launch_t<true, false, false>(a, stream);
  }
  if (a.rowsum) return cudaErrorInvalidValue;
  return clamp ? launch_t<false, false, true>(a, stream) : launch_t<false, false, false>(a, stream);
}

}  // namespace spinq
