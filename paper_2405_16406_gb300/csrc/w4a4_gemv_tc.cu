// w4a4_gemv_tc.cu -- the W4A4 GEMM for up to 16 tokens (decode) on the
// tensor core, streaming the weights through per-warp shared-memory stages.
//
// y[m][n] = s_n (alpha_m acc[m][n] + beta'_m rowsum_n), acc = sum_k a_mk q_nk,
// as in w4a4_gemm.cu.  With a few tokens the product streams the packed
// weights from HBM (N K / 2 bytes), so the loads of every warp must stay in
// flight back to back: a CTA owns 16 output channels for the whole K range,
// its WK warps each take a contiguous run of 128-deep K blocks (WK chosen at
// launch so that the N / 16 CTAs fill the GPU in one wave), and each warp
// streams its run through two shared-memory stages of 8 K blocks (512
// contiguous bytes of each of its 16 weight rows and of each token row below
// M, one row per copy instruction of the whole warp, as the weight stream of
// the GEMV kernel), one stage in flight while the other is used.  The partial sums meet in shared memory at the end (no workspace,
// no atomics, no second pass).
//
// Products on the tensor core, m16n8k16 with fp16 operands and fp32
// accumulation; M = 16 channels, N = 8 tokens.  Per K block, lane (g, c)
// (g = lane / 4, c = lane % 4) takes bytes [16 c, 16 c + 16) of the block of
// weight rows g and g + 8 and of its tokens' rows.  One mask turns a word of
// 8 unsigned codes into fp16 pairs: the codes at bits 0-3 and 16-19 read as
// fp16 bit patterns are the subnormals u 2^-24, those at bits 4-7 and 20-23
// are 16 u 2^-24 (the codes of bytes 1 and 3 after a shift by 8).  The
// tensor core multiplies subnormal operands exactly, so per word one MMA
// takes the low-nibble codes of both operands (products u_a u_w 2^-48) and
// one the high-nibble codes (256 u_a u_w 2^-48), each into an accumulator of
// its own: every partial sum is a multiple of 2^-48 (resp. 2^-40) below 2^23
// of those units for K <= 65536, hence exact.  The MMA's k index takes the
// lane's codes in the same order on both operands, a permutation of the
// sum's terms.  Two more MMAs against a constant fragment of ones give each
// token's sum of codes.
//
// Codes are made unsigned as in the other kernels (u = code ^ 8 for two's
// complement codes, u = code for asymmetric activations), so
//   acc = S - 8 sum_k u_a - 8 sum_k u_w + 64 K = S - 8 sum_k u_a - 8 rowsum_n
// with S = sum_k u_a u_w.  The epilogue is the one of the other kernels, so
// the outputs are bit-identical.
#include <cuda_fp16.h>

#include "../../include/spinq.h"
#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

constexpr int kTcMaxWarps = 16;    // warps per CTA at most (the K split of one channel group)
constexpr int kTcSmemPerSm = 196 * 1024;   // shared memory per SM the stages may take

__device__ __forceinline__ void cp16_stream(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global.L2::128B [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
// 16 bytes of token codes, kept in L1: the CTAs on an SM read the same ones
__device__ __forceinline__ void cp16_shared_l1(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// Stage geometry: U = 8 K blocks of 16 weight rows and 8 NT token rows, 512
// bytes each, packed (a quarter warp's fragment reads meet 2-way bank
// conflicts); S = 2 stages: 24 KB (NT = 1) or 32 KB (NT = 2) per warp.
template <int NT>
struct TcStage {
  static constexpr int U = 8, RS = 512, S = 2, ROWS = 16 + 8 * NT;
  static constexpr int BYTES = ROWS * RS;
  static constexpr int WARP = S * BYTES;
};

__device__ __forceinline__ uint32_t word(const uint4& v, int s) {
  return s == 0 ? v.x : (s == 1 ? v.y : (s == 2 ? v.z : v.w));
}

// NT n8 tiles of tokens (M <= 8 NT).
template <int NT, bool ASYM, bool ACC_OUT>
__global__ void __launch_bounds__(kTcMaxWarps * 32) w4a4_gemv_tc_kernel(GemmArgs a) {
  using R = TcStage<NT>;
  constexpr int U = R::U, RS = R::RS, S = R::S, TOK = 8 * NT;
  extern __shared__ __align__(16) uint8_t tc_smem[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int WK = blockDim.x >> 5;
  const int g = lane >> 2, c = lane & 3;
  const int64_t n0 = (int64_t)blockIdx.x * 16;
  const int nkb = (int)(a.K / 128);
  const size_t rowb = (size_t)(a.K / 2);
  // this warp's run of K blocks, in stages of U
  const int per = (nkb + WK - 1) / WK;
  const int kbeg = warp * per, kend = kbeg + per < nkb ? kbeg + per : nkb;
  const int nst = kend > kbeg ? (kend - kbeg + U - 1) / U : 0;
  // token rows copied: those below M (the slots of the others hold whatever
  // they hold, which unpacks to finite codes; those columns are never stored)
  const int mrow = (int)(a.M < TOK ? a.M : TOK);
  // copy role: the whole warp takes one row per instruction, 16 bytes a lane
  const int off16 = lane * 16;
  const uint8_t* wrow = a.w_codes + (size_t)n0 * rowb;   // weight row r at wrow + r rowb (N is a multiple of 16)
  // the first stage's weights do not depend on the previous kernel: fetch
  // them into L2 before waiting for it
  if (nst > 0 && lane < 16 && (size_t)kbeg * 64 + (size_t)(lane & 3) * 128 < (size_t)kend * 64)
    for (int r4 = 0; r4 < 4; ++r4)
      asm volatile("prefetch.global.L2 [%0];" ::"l"(wrow + (size_t)(4 * r4 + (lane >> 2)) * rowb + (size_t)kbeg * 64 +
                                                        (size_t)(lane & 3) * 128));
  pdl_wait();
  pdl_trigger();
  uint8_t* ring = tc_smem + (size_t)warp * R::WARP;
  const uint32_t ring_a = smem_u32(ring);
  auto issue = [&](int i) {
    if (i < nst) {
      const int kb = kbeg + U * i;
      const int nbytes = (kend - kb < U ? kend - kb : U) * 64;
      const uint32_t st = ring_a + (uint32_t)(i % S) * R::BYTES;
      if (off16 < nbytes) {
#pragma unroll
        for (int r = 0; r < 16; ++r)
          cp16_stream(st + r * RS + off16, wrow + (size_t)r * rowb + (size_t)kb * 64 + off16);
        for (int m = 0; m < mrow; ++m)
          cp16_shared_l1(st + (16 + m) * RS + off16, a.a_codes + (size_t)m * rowb + (size_t)kb * 64 + off16);
      }
    }
    cp_commit();   // an empty group past the end keeps the wait count uniform
  };
#pragma unroll
  for (int i = 0; i < S - 1; ++i) issue(i);

  const uint32_t xw = 0x88888888u, xa = ASYM ? 0u : 0x88888888u;
  // the ones fragment: A = 1 2^-24 everywhere
  const uint32_t ones[4] = {0x00010001u, 0x00010001u, 0x00010001u, 0x00010001u};
  // lo / hi: the low- and high-nibble products; olo / ohi: the tokens' code sums
  float lo[NT][4], hi[NT][4], olo[NT][4], ohi[NT][4];
#pragma unroll
  for (int t = 0; t < NT; ++t)
#pragma unroll
    for (int e = 0; e < 4; ++e) lo[t][e] = hi[t][e] = olo[t][e] = ohi[t][e] = 0.f;
  for (int i = 0; i < nst; ++i) {
    issue(i + S - 1);
    cp_wait<S - 1>();   // this lane's copies of stage i have landed
    __syncwarp();       // and every other lane's
    const uint8_t* st = ring + (size_t)(i % S) * R::BYTES + 16 * c;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (kbeg + U * i + u >= kend) break;   // warp-uniform
      const uint4 wa = *reinterpret_cast<const uint4*>(st + g * RS + 64 * u);
      const uint4 wb = *reinterpret_cast<const uint4*>(st + (g + 8) * RS + 64 * u);
      uint4 ta[NT];
#pragma unroll
      for (int t = 0; t < NT; ++t) ta[t] = *reinterpret_cast<const uint4*>(st + (16 + 8 * t + g) * RS + 64 * u);
#pragma unroll
      for (int s4 = 0; s4 < 4; ++s4) {
        // rows g (x0) and g + 8 (x1): bytes 0, 2 (k = 2c, 2c+1) and, after
        // the shift, bytes 1, 3 (k = 2c+8, 2c+9)
        const uint32_t x0 = word(wa, s4) ^ xw, x1 = word(wb, s4) ^ xw, y0 = x0 >> 8, y1 = x1 >> 8;
        const uint32_t al[4] = {x0 & 0x000F000Fu, x1 & 0x000F000Fu, y0 & 0x000F000Fu, y1 & 0x000F000Fu};
        const uint32_t ah[4] = {x0 & 0x00F000F0u, x1 & 0x00F000F0u, y0 & 0x00F000F0u, y1 & 0x00F000F0u};
#pragma unroll
        for (int t = 0; t < NT; ++t) {
          const uint32_t v = word(ta[t], s4) ^ xa, v8 = v >> 8;
          const uint32_t bl0 = v & 0x000F000Fu, bl1 = v8 & 0x000F000Fu;
          const uint32_t bh0 = v & 0x00F000F0u, bh1 = v8 & 0x00F000F0u;
          mma_16816_f16_f32_acc(lo[t], al, bl0, bl1);
          mma_16816_f16_f32_acc(hi[t], ah, bh0, bh1);
          mma_16816_f16_f32_acc(olo[t], ones, bl0, bl1);
          mma_16816_f16_f32_acc(ohi[t], ones, bh0, bh1);
        }
      }
    }
    __syncwarp();   // every lane is done with the stage before it is refilled
  }
  cp_wait<0>();
  __syncthreads();   // every warp is done with its stages: the reduction reuses them
  // ---- partial sums: tile t gives (channel g, tokens 8t + 2c, 2c + 1) and
  // (channel g + 8, same), as integers (exact: every value is a whole number
  // of its unit below 2^24); the token sums are the same in every row
  int* red = reinterpret_cast<int*>(tc_smem);                          // [WK][16][TOK + 1]
  int* sua = red + (size_t)WK * 16 * (TOK + 1);                        // [WK][TOK]
  int* rwp = red + (size_t)warp * 16 * (TOK + 1);
#pragma unroll
  for (int t = 0; t < NT; ++t)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int ch = g + 8 * (e >> 1), m = 8 * t + 2 * c + (e & 1);
      // lo holds sum u_w u_a 2^-48, hi (16 u_w)(16 u_a) 2^-48 = u_w u_a 2^-40
      rwp[ch * (TOK + 1) + m] =
          __float2int_rn(lo[t][e] * 281474976710656.0f) + __float2int_rn(hi[t][e] * 1099511627776.0f);
      if (g == 0 && e < 2)   // olo holds sum u_a 2^-48, ohi sum (16 u_a) 2^-48 = sum u_a 2^-44
        sua[warp * TOK + m] =
            __float2int_rn(olo[t][e] * 281474976710656.0f) + __float2int_rn(ohi[t][e] * 17592186044416.0f);
    }
  __syncthreads();
  // ---- epilogue: one (channel, token) per thread and round
  for (int e = threadIdx.x; e < 16 * TOK; e += WK * 32) {
    const int ch = e & 15, m = e >> 4;
    if (m >= a.M) continue;
    int sf = 0, sa = 0;
    for (int w = 0; w < WK; ++w) {
      sf += red[((size_t)w * 16 + ch) * (TOK + 1) + m];
      sa += sua[w * TOK + m];
    }
    const int64_t n = n0 + ch;
    const int rw = __ldg(a.w_rowsum + n);
    const int accm = sf - 8 * sa - 8 * rw;
    const float alpha = __ldg(a.a_scale + m);
    const float bp = ASYM ? __ldg(a.a_zero + m) + 8.f * alpha : 0.f;
    const float sn = __ldg(a.w_scale + n);
    reinterpret_cast<__half*>(a.y)[(int64_t)m * a.N + n] = __float2half_rn(sn * fmaf(alpha, (float)accm, bp * (float)rw));
    if (ACC_OUT) a.acc_out[(int64_t)m * a.N + n] = accm;
  }
}

template <int NT, bool ASYM, bool ACC_OUT>
cudaError_t launch_tc_t(const GemmArgs& a, cudaStream_t stream) {
  auto kern = w4a4_gemv_tc_kernel<NT, ASYM, ACC_OUT>;
  const int64_t grid = a.N / 16;
  // warps per CTA: the largest power of two up to 16 (and up to the K blocks)
  // with which the grid's warps fit the GPU's resident warps in one wave
  // (and within the shared-memory budget of one CTA)
  const int64_t slots = (int64_t)device_sm_count() * (kTcSmemPerSm / TcStage<NT>::WARP);
  int wk = kTcMaxWarps;
  while (wk > 1 && (grid * wk > slots || wk > a.K / 128 || (int64_t)wk * TcStage<NT>::WARP > kTcSmemPerSm)) wk >>= 1;
  const size_t smem = (size_t)wk * TcStage<NT>::WARP;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, wk * 32, smem, &per_sm);
  if (e != cudaSuccess) return e;
  e = launch_pdl(kern, dim3((unsigned)grid), dim3(wk * 32), smem, stream, 1, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int NT>
cudaError_t launch_tc_nt(const GemmArgs& a, cudaStream_t stream) {
  const bool asym = a.a_zero != nullptr, acc = a.acc_out != nullptr;
  if (asym) return acc ? launch_tc_t<NT, true, true>(a, stream) : launch_tc_t<NT, true, false>(a, stream);
  return acc ? launch_tc_t<NT, false, true>(a, stream) : launch_tc_t<NT, false, false>(a, stream);
}

}  // namespace

cudaError_t launch_w4a4_gemv_tc(const GemmArgs& a, cudaStream_t stream, bool* handled) {
  *handled = false;
  if (a.N == 0 || !w4a4_gemv_tc_fits(a.M, a.N, a.K)) return cudaSuccess;
  *handled = true;
  static_assert(kGemvTcMaxM <= 16, "instances up to two token tiles");
  if (a.M <= 8) return launch_tc_nt<1>(a, stream);
  return launch_tc_nt<2>(a, stream);
}

}  // namespace spinq
