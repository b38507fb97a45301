// w4a4_gemv.cu -- the W4A4 GEMM for a handful of tokens (decode, M <= 4).
//
// y[m][n] = s_n (alpha_m acc[m][n] + beta'_m rowsum_n), acc = sum_k a_mk q_nk,
// as in w4a4_gemm.cu.  With a few tokens the product is bound by streaming the
// packed weights from HBM (N K / 2 bytes); the tensor-core kernels stage every
// weight tile through shared memory and reduce K slices across CTAs, which
// costs several microseconds of latency for a few microseconds of streaming.
// Here each warp owns whole output channels: lanes load 16-byte chunks of a
// weight row straight from global memory (512 contiguous bytes per warp load),
// expand the nibbles to unsigned bytes in registers and take exact integer dot
// products (dp4a) against the tokens' codes, which the CTA expanded once into
// shared memory.  A warp reduction (redux) finishes each channel; no
// workspace, no atomics.
//
// Codes are made unsigned as in the tensor-core path (u = code ^ 8 for two's
// complement codes, u = code for asymmetric activations), so
//   acc = sum u_a u_w - 8 sum_k u_a - 8 sum_k u_w + 64 K
// with sum_k u_w = rowsum_n + 8 K: every term is an exact int32.
#include <cuda_fp16.h>

#include "../../include/spinq.h"
#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

constexpr int kGemvThreads = 512;
constexpr int kGemvWarps = kGemvThreads / 32;

// 32 packed codes -> their unsigned bytes: lo[j] holds the low nibbles of
// word j (even k), hi[j] the high nibbles (odd k).
__device__ __forceinline__ void expand16(const uint4 w, uint32_t x, uint32_t lo[4], uint32_t hi[4]) {
  const uint32_t v[4] = {w.x ^ x, w.y ^ x, w.z ^ x, w.w ^ x};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    lo[j] = v[j] & 0x0F0F0F0Fu;
    hi[j] = (v[j] >> 4) & 0x0F0F0F0Fu;
  }
}

__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

__device__ __forceinline__ uint32_t dp4a_u(uint32_t a, uint32_t b, uint32_t c) {
  return __dp4a(a, b, c);
}

// Shared memory: the tokens' expanded codes as pairs (lo_j, hi_j) at
// [(m * 4 + j) * NQ + q] (q = 16-byte chunk of the row), so the lanes of a warp,
// which take consecutive chunks, read consecutive 8-byte words; then the
// tokens' sums of unsigned codes.
template <int MT, bool ASYM, bool ACC_OUT>
__global__ void __launch_bounds__(kGemvThreads) w4a4_gemv_kernel(GemmArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int M = (int)a.M, NQ = (int)(a.K / 32);
  const int64_t kh = a.K / 2;
  uint2* As = reinterpret_cast<uint2*>(smem);
  int* su = reinterpret_cast<int*>(smem + (size_t)M * 4 * NQ * 8);
  const uint32_t xa = ASYM ? 0u : 0x88888888u;

  if (tid < MT) su[tid] = 0;
  // The weight row of this warp's first channel into L2 while the previous
  // kernel may still run: L2 is coherent with that kernel's stores, and
  // nothing is read into registers before griddepcontrol.wait.
  {
    const int64_t n = (int64_t)blockIdx.x * kGemvWarps + warp;
    if (n < a.N) {
      const char* row = reinterpret_cast<const char*>(a.w_codes) + n * kh;
      for (int64_t off = (int64_t)lane * 128; off < kh; off += 32 * 128) prefetch_l2(row + off);
    }
  }
  __syncthreads();
  pdl_wait();
  pdl_trigger();
  // expand the tokens' codes once per CTA
  for (int idx = tid; idx < M * NQ; idx += kGemvThreads) {
    const int m = idx / NQ, q = idx - m * NQ;
    const uint4 w = __ldg(reinterpret_cast<const uint4*>(a.a_codes + (int64_t)m * kh) + q);
    uint32_t lo[4], hi[4];
    expand16(w, xa, lo, hi);
    uint32_t s = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      As[(m * 4 + j) * NQ + q] = make_uint2(lo[j], hi[j]);
      s = dp4a_u(lo[j], 0x01010101u, dp4a_u(hi[j], 0x01010101u, s));
    }
    atomicAdd(&su[m], (int)s);
  }
  __syncthreads();

  const int64_t tw = (int64_t)gridDim.x * kGemvWarps;
  const uint4* W = reinterpret_cast<const uint4*>(a.w_codes);
  for (int64_t n = (int64_t)blockIdx.x * kGemvWarps + warp; n < a.N; n += tw) {
    const uint4* wrow = W + n * (kh / 16);
    uint32_t acc[MT];
#pragma unroll
    for (int m = 0; m < MT; ++m) acc[m] = 0;
    // four chunks per lane in flight per batch
    for (int q0 = 0; q0 < NQ; q0 += 4 * 32) {
      uint4 wv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int q = q0 + lane + 32 * i;
        wv[i] = q < NQ ? __ldcs(wrow + q) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int q = q0 + lane + 32 * i;
        if (q >= NQ) break;
        uint32_t lo[4], hi[4];
        expand16(wv[i], 0x88888888u, lo, hi);
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          if (m >= M) break;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint2 av = As[(m * 4 + j) * NQ + q];
            acc[m] = dp4a_u(lo[j], av.x, dp4a_u(hi[j], av.y, acc[m]));
          }
        }
      }
    }
    const float sn = __ldg(a.w_scale + n);
    const int rw = __ldg(a.w_rowsum + n);
    const int sw = rw + 8 * (int)a.K;          // sum_k u_w
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      if (m >= M) break;
      const int s = (int)__reduce_add_sync(0xffffffffu, acc[m]);
      if (lane == m) {
        const int accm = s - 8 * su[m] - 8 * sw + 64 * (int)a.K;
        const float alpha = __ldg(a.a_scale + m);
        const float bp = ASYM ? __ldg(a.a_zero + m) + 8.f * alpha : 0.f;
        reinterpret_cast<__half*>(a.y)[(int64_t)m * a.N + n] =
            __float2half_rn(sn * fmaf(alpha, (float)accm, bp * (float)rw));
        if (ACC_OUT) a.acc_out[(int64_t)m * a.N + n] = accm;
      }
    }
  }
}

template <int MT, bool ASYM, bool ACC_OUT>
cudaError_t launch_gemv_t(const GemmArgs& a, cudaStream_t stream) {
  auto kern = w4a4_gemv_kernel<MT, ASYM, ACC_OUT>;
  const size_t smem = (size_t)a.M * (size_t)(a.K / 32) * 32 + 16 * sizeof(int);
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, kGemvThreads, smem, &per_sm);
  if (e != cudaSuccess) return e;
  const int64_t warps_needed = a.N;
  int64_t grid = (int64_t)device_sm_count() * per_sm;
  const int64_t by_n = (warps_needed + kGemvWarps - 1) / kGemvWarps;
  if (grid > by_n) grid = by_n;
  e = launch_pdl(kern, dim3((unsigned)grid), dim3(kGemvThreads), smem, stream, 1, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int MT>
cudaError_t launch_gemv_mt(const GemmArgs& a, cudaStream_t stream) {
  const bool asym = a.a_zero != nullptr, acc = a.acc_out != nullptr;
  if (asym) return acc ? launch_gemv_t<MT, true, true>(a, stream) : launch_gemv_t<MT, true, false>(a, stream);
  return acc ? launch_gemv_t<MT, false, true>(a, stream) : launch_gemv_t<MT, false, false>(a, stream);
}

}  // namespace

int64_t w4a4_gemv_smem_bytes(int64_t M, int64_t K) { return M * K + 16 * (int64_t)sizeof(int); }

cudaError_t launch_w4a4_gemv(const GemmArgs& a, cudaStream_t stream, bool* handled) {
  *handled = false;
  if (a.N == 0 || !w4a4_gemv_fits(a.M, a.K)) return cudaSuccess;
  *handled = true;
  static_assert(kGemvMaxM <= 4, "instances up to four tokens");
  if (a.M <= 1) return launch_gemv_mt<1>(a, stream);
  if (a.M <= 2) return launch_gemv_mt<2>(a, stream);
  return launch_gemv_mt<4>(a, stream);
}

}  // namespace spinq
