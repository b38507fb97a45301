// cayley_step.cu -- spinq_cayley_step: one Cayley SGD update of a batch of
// n x n rotations (Sec. 3.2), n in {16, 32, 64, 128} (R2 is head_dim x
// head_dim, one per layer), one CTA per rotation.
//
//   G_hat = G R^T - 1/2 R R^T G R^T,   Y = G_hat - G_hat^T,
//   R' = (I - a/2 Y)^-1 (I + a/2 Y) R  by the fixed-point iteration
//   R'_0 = R + a Y R,  R'_{k+1} = R + (a/2) Y (R + R'_k).
//
// G is the negative of the loss gradient the caller passes (the printed update
// with G = +grad climbs the loss; the cited Cayley SGD forms G_hat from the
// negative gradient).  With D_k = R'_k - R the iteration reads
// D_0 = M = a Y R, D_{k+1} = M + (a/2) Y D_k, and R' = R + D_iters: M stays in
// registers, so three n x n fp32 buffers in shared memory suffice
// (3 * 128 * 132 * 4 = 203 KB at n = 128):
//
//   buf0 = R^T, buf1 = -grad         (loaded)
//   buf2 = A = G R^T                 [G buf1, R^T buf0]
//   buf1 = C = R^T A                 [R^T buf0, A buf2]
//   buf2 = G_hat = A - 1/2 R C       [R = buf0 read transposed, C buf1]
//   buf1 = Y = G_hat - G_hat^T;  buf0 transposed in place to R
//   M = a Y R (registers), buf2 = D_0 = M
//   D_{k+1} = M + (a/2) Y D_k        ping-pong between buf0 and buf2
//   R_out = R + D_iters              (R re-read from global memory)
//
// Thread (rg, cg) owns rows i0 = TR rg .. and columns 4 cg .. 4 cg + 3 and
// N/2 + 4 cg .. + 3 of every product (so that the 16-byte operand loads of a
// quarter warp are contiguous); the products run on packed fp32 pairs
// (fma.rn.f32x2), the column pairs of a row in one register pair.
#include <cuda_runtime.h>

#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

template <int N>
struct CayleyShape {
  static constexpr int TR = N >= 128 ? 4 : (N >= 64 ? 2 : 1);  // rows per thread
  static constexpr int CG = N / 8;                              // column groups of 8
  static constexpr int RG = N / TR;                             // row groups
  static constexpr int THREADS = CG * RG;
  static constexpr int S = N + 4;                               // row stride in floats
  static constexpr int BUF = N * S;
  static constexpr int BYTES = 3 * BUF * 4;
  static_assert(THREADS <= 1024 && THREADS % 32 == 0, "block shape");
};

template <int N>
using Acc = F2[CayleyShape<N>::TR][4];

// acc[r][c] += sum_k X(i0 + r, k) * B[k][col 2c, 2c + 1 of the thread], with
// X(i, k) = X[i][k], or X[k][i] when XT.
template <int N, bool XT>
__device__ __forceinline__ void mm_acc(const float* X, const float* B, int i0, int ja, int jb, Acc<N>& acc) {
  using S = CayleyShape<N>;
#pragma unroll 2
  for (int k = 0; k < N; ++k) {
    float xv[S::TR];
    if (XT) {
      if constexpr (S::TR == 4) {
        const float4 t = *reinterpret_cast<const float4*>(X + k * S::S + i0);
        xv[0] = t.x, xv[1] = t.y, xv[2] = t.z, xv[3] = t.w;
      } else if constexpr (S::TR == 2) {
        const float2 t = *reinterpret_cast<const float2*>(X + k * S::S + i0);
        xv[0] = t.x, xv[1] = t.y;
      } else {
        xv[0] = X[k * S::S + i0];
      }
    } else {
#pragma unroll
      for (int r = 0; r < S::TR; ++r) xv[r] = X[(i0 + r) * S::S + k];
    }
    const float4 b0 = *reinterpret_cast<const float4*>(B + k * S::S + ja);
    const float4 b1 = *reinterpret_cast<const float4*>(B + k * S::S + jb);
    const F2 bp[4] = {f2_make(b0.x, b0.y), f2_make(b0.z, b0.w), f2_make(b1.x, b1.y), f2_make(b1.z, b1.w)};
#pragma unroll
    for (int r = 0; r < S::TR; ++r) {
      const F2 xx = f2_make(xv[r], xv[r]);
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = f2_fma(xx, bp[c], acc[r][c]);
    }
  }
}

template <int N>
__device__ __forceinline__ void acc_zero(Acc<N>& acc) {
#pragma unroll
  for (int r = 0; r < CayleyShape<N>::TR; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = f2_make(0.f, 0.f);
}

template <int N>
__device__ __forceinline__ void tile_store(float* dst, int i0, int ja, int jb, const Acc<N>& acc) {
  using S = CayleyShape<N>;
#pragma unroll
  for (int r = 0; r < S::TR; ++r) {
    float v[8];
#pragma unroll
    for (int c = 0; c < 4; ++c) f2_split(acc[r][c], v[2 * c], v[2 * c + 1]);
    *reinterpret_cast<float4*>(dst + (i0 + r) * S::S + ja) = make_float4(v[0], v[1], v[2], v[3]);
    *reinterpret_cast<float4*>(dst + (i0 + r) * S::S + jb) = make_float4(v[4], v[5], v[6], v[7]);
  }
}

template <int N>
__global__ void __launch_bounds__(CayleyShape<N>::THREADS, 1)
    cayley_step_kernel(const float* __restrict__ R, const float* __restrict__ grad, float alpha, int iters,
                       float* R_out, float* Y_out) {
  using S = CayleyShape<N>;
  extern __shared__ __align__(16) float sm[];
  float* buf0 = sm;
  float* buf1 = sm + S::BUF;
  float* buf2 = sm + 2 * S::BUF;
  const int tid = threadIdx.x;
  const int cg = tid % S::CG, rg = tid / S::CG;
  // columns 4 cg .. + 3 and N/2 + 4 cg .. + 3: the 16-byte operand loads of
  // a quarter warp (cg = 0..7, one rg) cover 128 contiguous bytes
  const int i0 = rg * S::TR, ja = 4 * cg, jb = N / 2 + 4 * cg;
  const size_t base = (size_t)blockIdx.x * N * N;
  pdl_wait();
  pdl_trigger();

  // buf0 = R^T, buf1 = G = -grad
#pragma unroll
  for (int r = 0; r < S::TR; ++r) {
    const float4 a0 = *reinterpret_cast<const float4*>(R + base + (size_t)(i0 + r) * N + ja);
    const float4 a1 = *reinterpret_cast<const float4*>(R + base + (size_t)(i0 + r) * N + jb);
    const float v[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
    for (int c = 0; c < 8; ++c) buf0[(c < 4 ? ja + c : jb + c - 4) * S::S + i0 + r] = v[c];
    const float4 g0 = *reinterpret_cast<const float4*>(grad + base + (size_t)(i0 + r) * N + ja);
    const float4 g1 = *reinterpret_cast<const float4*>(grad + base + (size_t)(i0 + r) * N + jb);
    *reinterpret_cast<float4*>(buf1 + (i0 + r) * S::S + ja) = make_float4(-g0.x, -g0.y, -g0.z, -g0.w);
    *reinterpret_cast<float4*>(buf1 + (i0 + r) * S::S + jb) = make_float4(-g1.x, -g1.y, -g1.z, -g1.w);
  }
  __syncthreads();

  Acc<N> acc;
  // A = G R^T -> buf2
  acc_zero<N>(acc);
  mm_acc<N, false>(buf1, buf0, i0, ja, jb, acc);
  tile_store<N>(buf2, i0, ja, jb, acc);
  __syncthreads();
  // C = R^T A -> buf1
  acc_zero<N>(acc);
  mm_acc<N, false>(buf0, buf2, i0, ja, jb, acc);
  tile_store<N>(buf1, i0, ja, jb, acc);
  __syncthreads();
  // G_hat = A - 1/2 R C -> buf2
  acc_zero<N>(acc);
  mm_acc<N, true>(buf0, buf1, i0, ja, jb, acc);
  const F2 mhalf = f2_make(-0.5f, -0.5f);
#pragma unroll
  for (int r = 0; r < S::TR; ++r) {
    const float* at = buf2 + (i0 + r) * S::S;   // this thread's own tile of A
    const float4 t0 = *reinterpret_cast<const float4*>(at + ja);
    const float4 t1 = *reinterpret_cast<const float4*>(at + jb);
    const F2 av[4] = {f2_make(t0.x, t0.y), f2_make(t0.z, t0.w), f2_make(t1.x, t1.y), f2_make(t1.z, t1.w)};
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[r][c] = f2_fma(acc[r][c], mhalf, av[c]);
  }
  tile_store<N>(buf2, i0, ja, jb, acc);
  __syncthreads();
  // Y = G_hat - G_hat^T -> buf1 (and Y_out); buf0 transposed in place to R
#pragma unroll
  for (int r = 0; r < S::TR; ++r) {
    const int i = i0 + r;
    float y[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const int j = c < 4 ? ja + c : jb + c - 4;
      y[c] = buf2[i * S::S + j] - buf2[j * S::S + i];
      buf1[i * S::S + j] = y[c];
      if (i < j) {
        const float t = buf0[i * S::S + j];
        buf0[i * S::S + j] = buf0[j * S::S + i];
        buf0[j * S::S + i] = t;
      }
    }
    if (Y_out) {
      *reinterpret_cast<float4*>(Y_out + base + (size_t)i * N + ja) = make_float4(y[0], y[1], y[2], y[3]);
      *reinterpret_cast<float4*>(Y_out + base + (size_t)i * N + jb) = make_float4(y[4], y[5], y[6], y[7]);
    }
  }
  __syncthreads();
  // M = a Y R (registers), D_0 = M -> buf2
  Acc<N> m;
  acc_zero<N>(acc);
  mm_acc<N, false>(buf1, buf0, i0, ja, jb, acc);
  const F2 a2 = f2_make(alpha, alpha), h2 = f2_make(0.5f * alpha, 0.5f * alpha), zero2 = f2_make(0.f, 0.f);
#pragma unroll
  for (int r = 0; r < S::TR; ++r)
#pragma unroll
    for (int c = 0; c < 4; ++c) m[r][c] = f2_fma(acc[r][c], a2, zero2);
  if (iters > 0) tile_store<N>(buf2, i0, ja, jb, m);
  // D_{k+1} = M + (a/2) Y D_k, left in acc (D_0 = M when iters = 0)
  float* cur = buf2;
  float* nxt = buf0;
  for (int k = 0; k < iters; ++k) {
    __syncthreads();
    acc_zero<N>(acc);
    mm_acc<N, false>(buf1, cur, i0, ja, jb, acc);
#pragma unroll
    for (int r = 0; r < S::TR; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = f2_fma(acc[r][c], h2, m[r][c]);
    if (k + 1 < iters) tile_store<N>(nxt, i0, ja, jb, acc);
    float* t = cur;
    cur = nxt;
    nxt = t;
  }
  if (iters == 0) {
#pragma unroll
    for (int r = 0; r < S::TR; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = m[r][c];
  }
  // R' = R + D
#pragma unroll
  for (int r = 0; r < S::TR; ++r) {
    const size_t off = base + (size_t)(i0 + r) * N;
    const float4 a0 = *reinterpret_cast<const float4*>(R + off + ja);
    const float4 a1 = *reinterpret_cast<const float4*>(R + off + jb);
    float v[8];
#pragma unroll
    for (int c = 0; c < 4; ++c) f2_split(acc[r][c], v[2 * c], v[2 * c + 1]);
    *reinterpret_cast<float4*>(R_out + off + ja) = make_float4(a0.x + v[0], a0.y + v[1], a0.z + v[2], a0.w + v[3]);
    *reinterpret_cast<float4*>(R_out + off + jb) = make_float4(a1.x + v[4], a1.y + v[5], a1.z + v[6], a1.w + v[7]);
  }
}

template <int N>
cudaError_t launch_cayley_n(const CayleyArgs& a, cudaStream_t stream) {
  using S = CayleyShape<N>;
  auto kern = cayley_step_kernel<N>;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, S::THREADS, S::BYTES, &per_sm);
  if (e != cudaSuccess) return e;
  e = launch_pdl(kern, dim3((unsigned)a.batch), dim3(S::THREADS), S::BYTES, stream, 1, a.R, a.grad, a.alpha,
                 a.iters, a.R_out, a.Y_out);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_cayley_step(const CayleyArgs& a, cudaStream_t stream) {
  switch (a.n) {
    case 16: return launch_cayley_n<16>(a, stream);
    case 32: return launch_cayley_n<32>(a, stream);
    case 64: return launch_cayley_n<64>(a, stream);
    case 128: return launch_cayley_n<128>(a, stream);
  }
  return cudaErrorNotSupported;
}

}  // namespace spinq
