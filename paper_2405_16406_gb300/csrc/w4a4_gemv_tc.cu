// w4a4_gemv_tc.cu -- the W4A4 GEMM for up to 16 tokens (decode) on the
// tensor core, in two forms.
//
// y[m][n] = s_n (alpha_m acc[m][n] + beta'_m rowsum_n), acc = sum_k a_mk q_nk,
// as in w4a4_gemm.cu.  With a few tokens the product streams the packed
// weights from HBM (N K / 2 bytes), so the loads of every warp must stay in
// flight back to back.
//
// Register-streamed form (K = 128 NKW W, NKW in {1, 2, 4, 8}, W <= 16): one
// CTA per SM, its W warps split K and load the weights straight into a ring
// of registers; described at w4a4_decode_rs_kernel below.
//
// Shared-memory stage form (every other K up to 65536): a CTA owns 16 output
// channels for the whole K range, its WK warps each take a contiguous run of
// 128-deep K blocks (WK chosen at launch so that the N / 16 CTAs fill the GPU
// in one wave), and each warp streams its run through two shared-memory
// stages of 8 K blocks (512 contiguous bytes of each of its 16 weight rows
// and of each token row below M, one row per copy instruction of the whole
// warp, as the weight stream of the GEMV kernel), one stage in flight while
// the other is used.  The partial sums meet in shared memory at the end (no
// workspace, no atomics, no second pass).
//
// Its products on the tensor core, m16n8k16 with fp16 operands and fp32
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

#include <utility>

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

// ---------------------------------------------------------------------------
// Register-streamed form, for K = 128 NKW W with W <= 16 warps.
//
// A tile is 16 output channels (the MMA's M side) by the tokens (NT n8 tiles,
// columns past M zero).  Warp w of a CTA owns K blocks [NKW w, NKW w + NKW)
// of every tile the CTA takes; its tokens' words for those blocks sit in
// shared memory for the whole kernel, and it streams the weights of block
// (tile, kb) straight from global memory into a ring of kRsDepth blocks of
// registers (lane (g, c) loads 16 bytes of channel rows g and g + 8, chunk c
// of the block), with no copy stage and no copy waits: the loads of all
// warps stay in flight back to back.
//
// One accumulator unit for both nibbles: a weight word masked at bits 0-3 /
// 16-19 reads as u 2^-24 and at bits 4-7 / 20-23 as 16 u 2^-24 = u 2^-20; the
// token words are stored nibble-swapped, so the same masks give the token
// code of a low-nibble weight position as u 2^-20 and that of a high-nibble
// position as u 2^-24.  Every product is u_a u_w 2^-44, every partial sum a
// whole number of 2^-44 below 225 K < 2^24 of them: exact in fp32.  The MMA's
// k index takes each word's codes in the same order on both operands.  The
// weights' two's complement codes become u = code ^ 8 inside the mask
// instruction ((x & m) ^ x8, one three-input logic operation).
//
// A tile's K blocks meet in shared memory: each warp adds its exact partial
// sums (as integers) into one of kRsSlots slots and arrives on the slot's
// `full` barrier; the tile's epilogue warp (tiles w, w + W, ... go to warp w)
// waits on it, applies the epilogue of the other kernels (bit-identical
// outputs), clears the slot and arrives on `empty`, which a warp waits on
// before it adds tile ti + kRsSlots into the same slot.  Every wait is
// bounded; one that gives up records SPINQ_ETIMEOUT and every warp leaves at
// its next wait.
constexpr int kRsMaxWarps = 16;
constexpr int kRsDepth = 4;       // K blocks of weights (2 x 16 bytes each) in flight per lane
constexpr int kRsSlots = 4;       // shared-memory slots of tiles being reduced (a power of two)
constexpr int kRsSite = 30;       // wait site recorded on a time-out
constexpr int kRsCtasPerSm = 1;   // one CTA per SM (up to 16 warps of up to 128 registers)
constexpr uint64_t kRsWaitNs = 2000000000ull;

// weights are read once: keep them out of L1
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ uint32_t nibble_swap(uint32_t x) {
  return ((x & 0x0F0F0F0Fu) << 4) | ((x >> 4) & 0x0F0F0F0Fu);
}

// (x & m) ^ f in one instruction (m and f in registers)
__device__ __forceinline__ uint32_t and_xor(uint32_t x, uint32_t m, uint32_t f) {
  uint32_t r;
  asm("lop3.b32 %0, %1, %2, %3, 0x6A;" : "=r"(r) : "r"(x), "r"(m), "r"(f));
  return r;
}

template <int NKW, int NT, bool ASYM, bool ACC_OUT>
__global__ void __launch_bounds__(kRsMaxWarps * 32, 1) w4a4_decode_rs_kernel(GemmArgs a, int* status) {
  // ring depth: a whole number of tiles' K blocks (RT) or a divisor of a
  // tile's K blocks; TG tiles per turn of the ring
  constexpr bool RT = NKW < kRsDepth;
  constexpr int D = RT ? kRsDepth - kRsDepth % NKW : kRsDepth;
  constexpr int TG = RT ? D / NKW : 1;
  static_assert(RT || NKW % D == 0, "a tile's K blocks fill whole turns of the ring");
  constexpr int TOK = 8 * NT;
  __shared__ int acc_s[kRsSlots][16 * TOK];   // [slot][token 16 + channel]
  __shared__ int cnt_s[kRsSlots];                 // warps done with the slot's tile
  __shared__ int sa_s[16];                    // the tokens' code sums
  __shared__ float al_s[16], bp_s[16];        // alpha_m and beta'_m = zero_m + 8 alpha_m (asymmetric)
  __shared__ __align__(8) uint64_t empty[kRsSlots];
  __shared__ int abort_s;
  // dynamic: the warps' token words [warp][j][nt][lane], then the channel
  // scales and row sums of this CTA's tiles
  extern __shared__ __align__(16) uint4 tok_s[];
  volatile int* abort_flag = &abort_s;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, W = blockDim.x >> 5;
  const int g = lane >> 2, c = lane & 3;
  const int M = (int)a.M;
  const int64_t ntiles = a.N / 16, G = gridDim.x;
  const int nt_cta = ntiles > (int64_t)blockIdx.x ? (int)((ntiles - blockIdx.x + G - 1) / G) : 0;
  const size_t rowb = (size_t)(a.K / 2);
  const int kb0 = warp * NKW;
  // K block j of tile u of this CTA: this lane's 16 bytes of row g at
  // w0 + u tstride + j 64, those of row g + 8 a further 8 rowb on
  const uint8_t* w0 = a.w_codes + (size_t)(16 * blockIdx.x + g) * rowb + (size_t)kb0 * 64 + 16 * c;
  const size_t tstride = (size_t)(16 * G) * rowb, r8 = 8 * rowb;
  if (threadIdx.x == 0) {
    for (int k = 0; k < kRsSlots; ++k) {
      mbar_init(&empty[k], 1);
      cnt_s[k] = 0;
    }
    abort_s = 0;
    fence_mbar_init();
  }
  for (int e = threadIdx.x; e < kRsSlots * 16 * TOK; e += blockDim.x) (&acc_s[0][0])[e] = 0;
  if (threadIdx.x < 16) sa_s[threadIdx.x] = 0;
  if (threadIdx.x >= 32 * (W - 1) && lane < 16) {   // the last warp: the tokens' scales
    const float al = lane < M ? __ldg(a.a_scale + lane) : 0.f;
    al_s[lane] = al;
    bp_s[lane] = (ASYM && lane < M) ? __ldg(a.a_zero + lane) + 8.f * al : 0.f;
  }
  // the weights do not depend on the previous kernel: every 128-byte line
  // this warp will read goes into L2 before it waits for that kernel, so
  // the register loads below meet L2 latency instead of DRAM latency (lane
  // l takes row l % 16 of every other tile)
  {
    const int nl = NKW >= 2 ? NKW / 2 : 1;   // lines per row of this warp's K range
    const uint8_t* p = a.w_codes + (size_t)(16 * blockIdx.x + (lane & 15)) * rowb + (size_t)kb0 * 64;
    for (int ti = lane >> 4; ti < nt_cta; ti += 2)
      for (int l = 0; l < nl; ++l) asm volatile("prefetch.global.L2 [%0];" ::"l"(p + (size_t)ti * tstride + l * 128));
  }
  __syncthreads();
  pdl_wait();
  pdl_trigger();
  uint4 ra[D], rb[D];   // rows g and g + 8
#pragma unroll
  for (int d = 0; d < D; ++d)
    if (d / NKW < nt_cta) {
      const uint8_t* p = w0 + (size_t)(d / NKW) * tstride + (size_t)(d % NKW) * 64;
      ra[d] = ldg_stream(p);
      rb[d] = ldg_stream(p + r8);
    }
  // the channel constants of every tile of this CTA: loaded now, stored
  // after the token words below, so that the two loads' latencies overlap
  const int nch = 16 * nt_cta;
  float csn[2];
  int crw[2];
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int e = threadIdx.x + k * blockDim.x;
    if (e < nch) {
      const int64_t n = 16 * (blockIdx.x + (int64_t)(e >> 4) * G) + (e & 15);
      csn[k] = __ldg(a.w_scale + n);
      crw[k] = __ldg(a.w_rowsum + n);
    }
  }
  // this warp's token words: token 8 nt + g, its K blocks, chunk c; made
  // unsigned (u = code ^ 8 for two's complement codes) and nibble-swapped;
  // tokens past M are zero
  const uint32_t xa = ASYM ? 0u : 0x88888888u;
  uint4* tw = tok_s + (size_t)warp * NKW * NT * 32 + lane;   // [j][nt] at (j NT + nt) 32
  uint32_t su[NT];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) su[nt] = 0u;
#pragma unroll
  for (int j = 0; j < NKW; ++j)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int m = 8 * nt + g;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (m < M) v = __ldg(reinterpret_cast<const uint4*>(a.a_codes + (size_t)m * rowb + (size_t)(kb0 + j) * 64 + 16 * c));
      uint32_t sw[4];
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        const uint32_t u = word(v, s) ^ xa;
        su[nt] = __dp4a((u & 0x0F0F0F0Fu) + ((u >> 4) & 0x0F0F0F0Fu), 0x01010101u, su[nt]);
        sw[s] = m < M ? nibble_swap(u) : 0u;
      }
      tw[(j * NT + nt) * 32] = make_uint4(sw[0], sw[1], sw[2], sw[3]);
    }
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    su[nt] += __shfl_xor_sync(0xffffffffu, su[nt], 1);
    su[nt] += __shfl_xor_sync(0xffffffffu, su[nt], 2);
    if (c == 0 && 8 * nt + g < M) atomicAdd(&sa_s[8 * nt + g], (int)su[nt]);
  }
  // the channel constants of every tile of this CTA
  float* sn_s = reinterpret_cast<float*>(tok_s + (size_t)W * NKW * NT * 32);
  int* rw_s = reinterpret_cast<int*>(sn_s + 16 * nt_cta);
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    const int e = threadIdx.x + k * blockDim.x;
    if (e < nch) {
      sn_s[e] = csn[k];
      rw_s[e] = crw[k];
    }
  }
  for (int e = threadIdx.x + 2 * blockDim.x; e < nch; e += blockDim.x) {
    const int64_t n = 16 * (blockIdx.x + (int64_t)(e >> 4) * G) + (e & 15);
    sn_s[e] = __ldg(a.w_scale + n);
    rw_s[e] = __ldg(a.w_rowsum + n);
  }
  __syncthreads();   // the token sums, scales and channel constants are complete
  // masks and sign flips of the weight words, in registers for and_xor
  uint32_t mlo = 0x000F000Fu, mhi = 0x00F000F0u, flo = 0x00080008u, fhi = 0x00800080u;
  asm volatile("" : "+r"(mlo), "+r"(mhi), "+r"(flo), "+r"(fhi));
  // per token tile, two accumulators (bytes 0 and 2 / bytes 1 and 3 of each
  // word) keep the MMA chains short; their sum is exact too
  float d0[NT][4], d1[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) d0[nt][e] = d1[nt][e] = 0.f;
  const uint8_t* wp = w0 + (size_t)TG * tstride;          // tile ti + TG
  // One tile: its K blocks (ring slots from the compile-time position U of
  // the tile in the ring's turn), then its share of the reduction.  `refill`
  // is false only for the last TG tiles (nothing further to load).
  auto do_tile = [&](auto U, int ti, bool refill) -> bool {
    constexpr int u = decltype(U)::value;
#pragma unroll
    for (int j = 0; j < NKW; ++j) {
      const int dd = (u * NKW + j) % D;
      const uint4 wa = ra[dd], wb = rb[dd];
      uint4 tv[NT];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) tv[nt] = tw[(j * NT + nt) * 32];
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        const uint32_t x0 = word(wa, s), x1 = word(wb, s), y0 = x0 >> 8, y1 = x1 >> 8;
        const uint32_t a1[4] = {and_xor(x0, mlo, flo), and_xor(x1, mlo, flo), and_xor(x0, mhi, fhi),
                                and_xor(x1, mhi, fhi)};
        const uint32_t a2[4] = {and_xor(y0, mlo, flo), and_xor(y1, mlo, flo), and_xor(y0, mhi, fhi),
                                and_xor(y1, mhi, fhi)};
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          const uint32_t t0 = word(tv[nt], s), t8 = t0 >> 8;
          mma_16816_f16_f32_acc(d0[nt], a1, t0 & 0x00F000F0u, t0 & 0x000F000Fu);
          mma_16816_f16_f32_acc(d1[nt], a2, t8 & 0x00F000F0u, t8 & 0x000F000Fu);
        }
      }
      // refill the slot with the block D ahead: tile ti + TG, block j (RT);
      // block j + D of this tile, or block j + D - NKW of the next one
      const uint8_t* q = RT ? wp + j * 64 : (j + D < NKW ? wp - tstride + (j + D) * 64 : wp + (j + D - NKW) * 64);
      if ((!RT && j + D < NKW) || refill) {
        ra[dd] = ldg_stream(q);
        rb[dd] = ldg_stream(q + r8);
      }
    }
    wp += tstride;
    // ---- this warp's share of tile ti is done
    const int slot = ti & (kRsSlots - 1);
    if (ti >= kRsSlots &&
        !__all_sync(0xffffffffu, mbar_wait_suspend(&empty[slot], (uint32_t)((ti / kRsSlots) - 1) & 1u, abort_flag,
                                                   kRsWaitNs)))
      return false;
    // lane (g, c): channels g and g + 8, tokens 8 nt + 2c and 8 nt + 2c + 1;
    // exact integers (whole numbers of 2^-44 below 2^24 of them); the sums
    // of tokens past M are zero (their words are), so every lane adds
    const float unit = 17592186044416.0f;   // 2^44
    int* accp = &acc_s[slot][(2 * c) * 16 + g];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        atomicAdd(accp + (8 * nt + (e & 1)) * 16 + 8 * (e >> 1), __float2int_rn((d0[nt][e] + d1[nt][e]) * unit));
        d0[nt][e] = d1[nt][e] = 0.f;
      }
    // the last warp to finish the tile applies the epilogue (the fence
    // orders each warp's adds before its count)
    __threadfence_block();
    __syncwarp();
    int last = 0;
    if (lane == 0) last = atomicAdd(&cnt_s[slot], 1) == W - 1;
    if (!__shfl_sync(0xffffffffu, last, 0)) return true;
    __threadfence_block();
    const int ch = lane & 15;
    const int64_t n = 16 * (blockIdx.x + (int64_t)ti * G) + ch;
    const float sn = sn_s[16 * ti + ch];
    const int rw = rw_s[16 * ti + ch];
#pragma unroll
    for (int q = 0; q < TOK / 2; ++q) {
      const int idx = lane + 32 * q, m = idx >> 4;
      const int v = acc_s[slot][idx];
      acc_s[slot][idx] = 0;
      if (m < M) {
        const int accm = v - 8 * sa_s[m] - 8 * rw;
        reinterpret_cast<__half*>(a.y)[(int64_t)m * a.N + n] =
            __float2half_rn(sn * fmaf(al_s[m], (float)accm, bp_s[m] * (float)rw));
        if (ACC_OUT) a.acc_out[(int64_t)m * a.N + n] = accm;
      }
    }
    __syncwarp();
    if (lane == 0) {
      cnt_s[slot] = 0;
      mbar_arrive(&empty[slot]);   // release: the cleared slot is ordered before it
    }
    return true;
  };
  bool ok = true;
  int t = 0;
  static_assert(TG <= 4, "tiles per turn of the ring");
  // tile U of the turn starting at t (U < TG); `tail`: the last turns, where
  // tiles past nt_cta are skipped and the last TG load nothing more
  auto turn_tile = [&](auto U, bool tail) {
    constexpr int u = decltype(U)::value;
    if constexpr (u < TG) {
      if (ok && (!tail || t + u < nt_cta)) ok = do_tile(U, t + u, !tail || t + u + TG < nt_cta);
    }
  };
  // whole turns of the ring whose tiles all refill it
  for (; t + 2 * TG <= nt_cta && ok; t += TG) {
    turn_tile(std::integral_constant<int, 0>{}, false);
    turn_tile(std::integral_constant<int, 1>{}, false);
    turn_tile(std::integral_constant<int, 2>{}, false);
    turn_tile(std::integral_constant<int, 3>{}, false);
  }
  for (; t < nt_cta && ok; t += TG) {
    turn_tile(std::integral_constant<int, 0>{}, true);
    turn_tile(std::integral_constant<int, 1>{}, true);
    turn_tile(std::integral_constant<int, 2>{}, true);
    turn_tile(std::integral_constant<int, 3>{}, true);
  }
  if (!ok && threadIdx.x % 32 == 0 && status && atomicCAS(status, 0, (int)SPINQ_ETIMEOUT) == 0)
    atomicExch(status + 1, kRsSite);
}

// K blocks per warp for the register-streamed form (0: the shape is not its own)
inline int rs_blocks_per_warp(int64_t K) {
  const int64_t nkb = K / 128;
  for (int nkw = 1; nkw <= 8; nkw *= 2)
    if (nkb % nkw == 0 && nkb / nkw <= kRsMaxWarps) return nkw;
  return 0;
}

template <int NKW, int NT, bool ASYM, bool ACC_OUT>
cudaError_t launch_rs_t(const GemmArgs& a, cudaStream_t stream) {
  auto kern = w4a4_decode_rs_kernel<NKW, NT, ASYM, ACC_OUT>;
  const int warps = (int)(a.K / 128 / NKW);
  const int64_t tiles = a.N / 16, slots = (int64_t)device_sm_count() * kRsCtasPerSm;
  const int64_t grid = tiles < slots ? tiles : slots;
  // the warps' token words and the channel constants of a CTA's tiles
  const size_t smem = (size_t)warps * NKW * NT * 32 * 16 + (size_t)((tiles + grid - 1) / grid) * 16 * 8;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, warps * 32, smem, &per_sm);
  if (e != cudaSuccess) return e;
  e = launch_pdl(kern, dim3((unsigned)grid), dim3(warps * 32), smem, stream, 1, a, device_status_word());
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int NKW, int NT>
cudaError_t launch_rs_nt(const GemmArgs& a, cudaStream_t stream) {
  const bool asym = a.a_zero != nullptr, acc = a.acc_out != nullptr;
  if (asym) return acc ? launch_rs_t<NKW, NT, true, true>(a, stream) : launch_rs_t<NKW, NT, true, false>(a, stream);
  return acc ? launch_rs_t<NKW, NT, false, true>(a, stream) : launch_rs_t<NKW, NT, false, false>(a, stream);
}

template <int NKW>
cudaError_t launch_rs_nkw(const GemmArgs& a, cudaStream_t stream) {
  return a.M <= 8 ? launch_rs_nt<NKW, 1>(a, stream) : launch_rs_nt<NKW, 2>(a, stream);
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

bool w4a4_gemv_tc_streamed(int64_t K) { return K >= 128 && K % 128 == 0 && rs_blocks_per_warp(K) != 0; }

cudaError_t launch_w4a4_gemv_tc(const GemmArgs& a, cudaStream_t stream, bool* handled) {
  *handled = false;
  if (a.N == 0 || !w4a4_gemv_tc_fits(a.M, a.N, a.K)) return cudaSuccess;
  *handled = true;
  static_assert(kGemvTcMaxM <= 16, "instances up to two token tiles");
  switch (rs_blocks_per_warp(a.K)) {
    case 1: return launch_rs_nkw<1>(a, stream);
    case 2: return launch_rs_nkw<2>(a, stream);
    case 4: return launch_rs_nkw<4>(a, stream);
    case 8: return launch_rs_nkw<8>(a, stream);
    default: break;
  }
  if (a.M <= 8) return launch_tc_nt<1>(a, stream);
  return launch_tc_nt<2>(a, stream);
}

}  // namespace spinq
