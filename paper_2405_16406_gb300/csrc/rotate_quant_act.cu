// rotate_quant_act.cu -- activation kernels of spinq_rotate_quant_act:
// the online rotation R4 (Sec. 3.1) fused with the per-token Eq. 1 quantizer,
// for a power-of-two rotation size 512 <= P <= 16384, and the quantizer alone
// when there is no online rotation.
//
// One CTA of W warps owns one row at a time (persistent over rows).
//
// Phase 1 (registers).  Lane `lane` of warp w loads the 16-byte chunks
// ch = lane + 32 (w + W v), v < V, so every load instruction is coalesced.
// Element index bits: e (0..2, inside a chunk), c = lane & 3 (3..4),
// g = lane >> 2 (5..7), w (8 .. 8+LW-1), v (8+LW ..).
// A tensor-core m16n8k16 with B = the 16-point Sylvester matrix contracts the
// bits {e0, e2, c0, c1} of the RAW fp16 input (entries +-1: exact products,
// fp32 sums) and returns fp32 in the lane that supplied the data, at the same
// element positions (the chunk's four 32-bit words are the A fragment as they
// are: words 0/2 are rows g, words 1/3 rows g + 8, so e1 is the row bit).
// Radix-2 butterflies inside the lane then cover e1 and the v bits.
//
// Transpose.  The rows go through shared memory once as fp32 (16-byte chunks
// XOR-swizzled so that both the phase-1 stores and the phase-2 loads are free
// of bank conflicts).
//
// Phase 2 (registers).  Thread t owns the remaining bits (g and w: 3 + LW
// bits) for 2^L consecutive elements, finishes the butterflies, joins the
// row-wide range reduction and writes its packed codes (2^L nibbles).
//
// Eq. 1 is applied to the unnormalised row; alpha and beta carry 1/sqrt(K).
#include <cuda_fp16.h>
#include <float.h>

#include "launch_util.h"
#include "quant_common.cuh"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

__device__ __forceinline__ uint32_t h16_entry_pair(int k0, int k1, int n, bool hadamard) {
  float v0, v1;
  if (hadamard) {
    v0 = (__popc(k0 & n) & 1) ? -1.f : 1.f;
    v1 = (__popc(k1 & n) & 1) ? -1.f : 1.f;
  } else {
    v0 = k0 == n ? 1.f : 0.f;
    v1 = k1 == n ? 1.f : 0.f;
  }
  return pack_half2_bits(v0, v1);
}

// B fragments of the 16 x 16 Sylvester matrix (hadamard) or identity, for the
// two n-tiles n = g and n = g + 8.
__device__ __forceinline__ void make_b16(uint32_t b[2][2], bool hadamard) {
  const int lane = threadIdx.x & 31, g = lane >> 2, c = lane & 3;
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
    const int n = g + 8 * nt;
    b[nt][0] = h16_entry_pair(2 * c, 2 * c + 1, n, hadamard);
    b[nt][1] = h16_entry_pair(2 * c + 8, 2 * c + 9, n, hadamard);
  }
}

// One 16-byte chunk (8 fp16) through the tensor core: the results y[e],
// e = 0..7, come back as the pairs y2[q] = (y[2q], y[2q + 1]).  The words of
// the chunk are the A fragment in their own order (k = e0 + 2c + 8 e2, row
// g + 8 e1), so no register moves are needed.
__device__ __forceinline__ void chunk_mma(const uint4 in, const uint32_t b[2][2], F2 y2[4]) {
  const uint32_t A[4] = {in.x, in.y, in.z, in.w};
  mma_16816_f16_f32_pairs(y2[0], y2[1], A, b[0][0], b[0][1]);
  mma_16816_f16_f32_pairs(y2[2], y2[3], A, b[1][0], b[1][1]);
}

// ------------------------------------------------------------------------
// power-of-two rotation
// ------------------------------------------------------------------------
template <int LW, int L>
struct Pow2Shape {
  static constexpr int W = 1 << LW;
  static constexpr int T = 32 * W;
  static constexpr int LV = LW + L;
  static constexpr int V = 1 << LV;
  static constexpr int P = 256 * W * V;
  static constexpr int NG = 1 << (3 + LW);  // phase-2 groups per thread
  static constexpr int GL = 1 << L;         // consecutive elements per group
};

constexpr uint64_t kRowWaitLimitNs = 2000000000ull;

// fp32 transpose buffer: two planes, element p -> plane (p >> 2) & 1,
// word 4 (p >> 3) + (p & 3); plane 1 starts 16 words (64 B) after the end of
// plane 0 so that the two planes map to opposite halves of the bank space.
// Phase 1 stores each chunk as one float4 per plane (8 lanes = 128 contiguous
// bytes); phase 2 reads 2 or 4 consecutive elements whose word offsets are a
// per-thread base plus compile-time constants.
template <int P>
__device__ __forceinline__ uint32_t plane_word(uint32_t p) {
  return ((p >> 2) & 1u) * (P / 2 + 16) + ((p >> 3) << 2) + (p & 3u);
}

template <int LW, int L>
struct Pow2Smem {
  using S = Pow2Shape<LW, L>;
  static constexpr int NST = S::P >= 4096 ? 1 : 2;     // fp16 rows staged ahead
  static constexpr int OFF_F32 = 0;                     // two planes
  static constexpr int OFF_STAGE = (S::P + 32) * 4;
  static constexpr int OFF_BAR = OFF_STAGE + NST * S::P * 2;
  static constexpr int OFF_MISC = OFF_BAR + NST * 8;   // abort flag + range scratch
  static constexpr int BYTES = OFF_MISC + 16 + 2 * S::W * 4;
};

template <int LW, int L, bool SYM, bool CLAMP, bool SG>
__global__ void __launch_bounds__(32 << LW) rq_pow2_kernel(RotQuantArgs a) {
  using S = Pow2Shape<LW, L>;
  using SM = Pow2Smem<LW, L>;
  static_assert(L == 1 || L == 2, "phase-2 group of 2 or 4 elements");
  extern __shared__ __align__(128) uint8_t smem[];
  float* sm = reinterpret_cast<float*>(smem + SM::OFF_F32);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + SM::OFF_MISC);
  float* red = reinterpret_cast<float*>(smem + SM::OFF_MISC + 16);
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  uint32_t bh[2][2];
  make_b16(bh, true);

  int* release_count = reinterpret_cast<int*>(smem + SM::OFF_MISC + 4);
  RowStream<SM::NST> rs{smem + SM::OFF_STAGE, (uint32_t)(S::P * 2),
                        reinterpret_cast<uint64_t*>(smem + SM::OFF_BAR),
                        reinterpret_cast<const uint8_t*>(a.x), a.ldx * 2, (uint32_t)(S::P * 2), 1u, 0u,
                        a.rows, (int64_t)blockIdx.x, (int64_t)gridDim.x};
  rs.init();
  if (tid == 0) {
    *abort_flag = 0;
    *release_count = 0;
    fence_mbar_init();
  }
  __syncthreads();
  pdl_wait();
  pdl_trigger();
  rs.prologue();
  // Random signs (R = S H): chunk v of this lane is chunk ch of every row,
  // whose 8 sign bits are byte ch of the bit mask; gathered once.
  uint32_t sgb[(S::V + 3) / 4];
#pragma unroll
  for (int t = 0; t < (S::V + 3) / 4; ++t) sgb[t] = 0;
  if constexpr (SG) {
#pragma unroll
    for (int v = 0; v < S::V; ++v)
      sgb[v >> 2] |= (uint32_t)a.signs[lane + 32 * (w + S::W * v)] << (8 * (v & 3));
  }

  // phase-2 fixed element bits of this thread: {L..2}, {3, 4}, v bits
  const uint32_t t_lo = (uint32_t)tid & ((1u << (3 - L)) - 1u);
  const uint32_t t_c = ((uint32_t)tid >> (3 - L)) & 3u;
  const uint32_t t_v = (uint32_t)tid >> (5 - L);
  const uint32_t fixed = (t_lo << L) | (t_c << 3) | (t_v << (8 + LW));
  const float* zbase = sm + plane_word<S::P>(fixed);   // group m adds 4 * (m << 2) words
  uint8_t* const codes0 = a.codes + (fixed >> 1);

  int it = 0;
  for (int64_t row = blockIdx.x; row < a.rows; row += gridDim.x, ++it) {
    rs.wait(it, abort_flag, kRowWaitLimitNs);
    __syncthreads();
    if (*abort_flag) break;
    // ---------------- phase 1
    const uint4* src = reinterpret_cast<const uint4*>(rs.stage(it));
    F2 y[S::V][4];  // y[v][q] = elements (2q, 2q + 1) of chunk v
#pragma unroll
    for (int v = 0; v < S::V; ++v) {
      uint4 in = src[lane + 32 * (w + S::W * v)];
      if constexpr (SG) {   // negate the fp16 elements whose sign bit is set
        const uint32_t B = sgb[v >> 2] >> (8 * (v & 3));
        in.x ^= ((B & 1u) << 15) | ((B & 2u) << 30);
        in.y ^= ((B & 4u) << 13) | ((B & 8u) << 28);
        in.z ^= ((B & 16u) << 11) | ((B & 32u) << 26);
        in.w ^= ((B & 64u) << 9) | ((B & 128u) << 24);
      }
      chunk_mma(in, bh, y[v]);
    }
    rs.release_warp(it, release_count, S::W);  // the next copy into this stage overlaps the rest of the row
#pragma unroll
    for (int v = 0; v < S::V; ++v) {  // e1
      f2_bfly(y[v][0], y[v][1]);
      f2_bfly(y[v][2], y[v][3]);
    }
#pragma unroll
    for (int bit = 1; bit < S::V; bit <<= 1)
#pragma unroll
      for (int v = 0; v < S::V; ++v)
        if (!(v & bit)) {
#pragma unroll
          for (int q = 0; q < 4; ++q) f2_bfly(y[v][q], y[v | bit][q]);
        }
#pragma unroll
    for (int v = 0; v < S::V; ++v) {
      const uint32_t ch = (uint32_t)(lane + 32 * (w + S::W * v));
      // 8-byte stores of whole pairs: a 16-byte store would need the two
      // pairs in four consecutive registers
      unsigned long long* p0 = reinterpret_cast<unsigned long long*>(sm + 4 * ch);
      unsigned long long* p1 = reinterpret_cast<unsigned long long*>(sm + S::P / 2 + 16 + 4 * ch);
      p0[0] = y[v][0].u;
      p0[1] = y[v][1].u;
      p1[0] = y[v][2].u;
      p1[1] = y[v][3].u;
    }
    __syncthreads();

    // ---------------- phase 2: groups m cover element bits 5.. (g, then w)
    constexpr int GP = S::GL / 2;  // pairs per group
    F2 z[S::NG][GP];
#pragma unroll
    for (int m = 0; m < S::NG; ++m) {
      if constexpr (GP == 2) {
        const ulonglong2 u = *reinterpret_cast<const ulonglong2*>(zbase + 16 * m);
        z[m][0].u = u.x;
        z[m][GP - 1].u = u.y;
      } else {
        z[m][0].u = *reinterpret_cast<const unsigned long long*>(zbase + 16 * m);
      }
    }
#pragma unroll
    for (int bit = 1; bit < S::NG; bit <<= 1)
#pragma unroll
      for (int m = 0; m < S::NG; ++m)
        if (!(m & bit)) {
#pragma unroll
          for (int q = 0; q < GP; ++q) f2_bfly(z[m][q], z[m | bit][q]);
        }
    Range<SYM> r;
#pragma unroll
    for (int m = 0; m < S::NG; ++m)
#pragma unroll
      for (int q = 0; q < GP; ++q) r.add_pair(z[m][q]);
    block_range<SYM, S::W>(r, red);
    const QParams<SYM> qp(r, a.clip);

    uint8_t* out = codes0 + row * (a.K / 2);
#pragma unroll
    for (int m = 0; m < S::NG; ++m) {
      // element offset of group m is 32 m (bits 5..), i.e. 16 m bytes of codes
      uint32_t rb[4];
      qp.template code_bits2<CLAMP>(z[m][0], rb[0], rb[1]);
      if constexpr (GP == 2) {
        qp.template code_bits2<CLAMP>(z[m][GP - 1], rb[2], rb[3]);
        *reinterpret_cast<uint16_t*>(out + 16 * m) = (uint16_t)pack4_nibbles(rb[0], rb[1], rb[2], rb[3]);
      } else {
        out[16 * m] = (uint8_t)pack2_nibbles(rb[0], rb[1]);
      }
    }
    if (tid == 0) {
      a.scale[row] = qp.alpha * a.norm;
      if (!SYM) a.zero[row] = qp.beta * a.norm;
    }
    __syncthreads();  // the transpose buffer and `red` are reused by the next row
  }
  if (*abort_flag) rs.drain(it, kRowWaitLimitNs);
}

// ------------------------------------------------------------------------
// quantizer only (no online rotation): one CTA of W warps per row.  Every
// lane loads its (up to kNoRotCPT) 16-byte chunks straight into registers with
// streaming loads issued back to back, so a whole row is in flight at once
// and, with every CTA of the grid resident, so is the whole matrix.  The row
// range is taken on the fp16 values themselves (max and min of fp16 numbers
// are exact, and equal the range of their fp32 values); then the tensor core
// widens each chunk to fp32 exactly (B = I16) for Eq. 1.
// ------------------------------------------------------------------------
constexpr int kNoRotCPT = 8;   // chunks per lane

__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ uint32_t h2_absmax(uint32_t m, uint32_t x) {
  uint32_t r;
  asm("{\n .reg .b32 t;\n abs.f16x2 t, %2;\n max.f16x2 %0, %1, t;\n}\n" : "=r"(r) : "r"(m), "r"(x));
  return r;
}
__device__ __forceinline__ uint32_t h2_max(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
__device__ __forceinline__ uint32_t h2_min(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("min.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
__device__ __forceinline__ float h2_hi_lo_max(uint32_t v) {
  const __half2 h = *reinterpret_cast<const __half2*>(&v);
  return fmaxf(__low2float(h), __high2float(h));
}
__device__ __forceinline__ float h2_hi_lo_min(uint32_t v) {
  const __half2 h = *reinterpret_cast<const __half2*>(&v);
  return fminf(__low2float(h), __high2float(h));
}

template <bool SYM, bool CLAMP>
__global__ void __launch_bounds__(512) rq_norot_kernel(RotQuantArgs a) {
  __shared__ float red[2 * 16];
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5, W = (int)(blockDim.x >> 5);
  const int64_t row = blockIdx.x;
  const int nchunk = (int)(a.K / 8);
  uint32_t bi[2][2];
  make_b16(bi, false);
  pdl_wait();
  pdl_trigger();
  const uint8_t* src = reinterpret_cast<const uint8_t*>(a.x) + row * a.ldx * 2;
  uint4 c[kNoRotCPT];
#pragma unroll
  for (int v = 0; v < kNoRotCPT; ++v) {
    const int ch = lane + 32 * (w + W * v);
    c[v] = ch < nchunk ? ld_stream_v4(src + (size_t)ch * 16) : make_uint4(0, 0, 0, 0);
  }
  // row range on the fp16 values: +-inf start values for the asymmetric
  // form, absolute values from 0 for the symmetric one
  uint32_t hi2 = SYM ? 0u : 0xFC00FC00u, lo2 = 0x7C007C00u;
#pragma unroll
  for (int v = 0; v < kNoRotCPT; ++v) {
    if (lane + 32 * (w + W * v) < nchunk) {
      const uint32_t q[4] = {c[v].x, c[v].y, c[v].z, c[v].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (SYM) {
          hi2 = h2_absmax(hi2, q[e]);
        } else {
          hi2 = h2_max(hi2, q[e]);
          lo2 = h2_min(lo2, q[e]);
        }
      }
    }
  }
  Range<SYM> r;
  r.hi = h2_hi_lo_max(hi2);
  if (!SYM) r.lo = h2_hi_lo_min(lo2);
  r.warp_reduce();
  if (W > 1) {
    if (lane == 0) {
      red[w] = r.hi;
      red[16 + w] = r.lo;
    }
    __syncthreads();
    r.hi = red[0];
    r.lo = red[16];
    for (int i = 1; i < W; ++i) {
      r.hi = fmaxf(r.hi, red[i]);
      if (!SYM) r.lo = fminf(r.lo, red[16 + i]);
    }
  }
  const QParams<SYM> qp(r, a.clip);
  uint32_t* out = reinterpret_cast<uint32_t*>(a.codes + row * (a.K / 2));
#pragma unroll
  for (int v = 0; v < kNoRotCPT; ++v) {
    const int ch = lane + 32 * (w + W * v);
    F2 y[4];
    chunk_mma(c[v], bi, y);   // exact fp16 -> fp32 (all lanes take part)
    uint32_t rb[8];
#pragma unroll
    for (int q = 0; q < 4; ++q) qp.template code_bits2<CLAMP>(y[q], rb[2 * q], rb[2 * q + 1]);
    if (ch < nchunk) out[ch] = pack8_nibbles(rb);
  }
  if (tid == 0) {
    a.scale[row] = qp.alpha * a.norm;
    if (!SYM) a.zero[row] = qp.beta * a.norm;
  }
}

template <typename Kern>
cudaError_t launch_rows(Kern kern, int threads, size_t smem, const RotQuantArgs& a, cudaStream_t stream) {
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, threads, smem, &per_sm);
  if (e != cudaSuccess) return e;
  const int64_t cap = (int64_t)device_sm_count() * per_sm;
  const int64_t grid = a.rows < cap ? a.rows : cap;
  e = launch_pdl(kern, dim3((unsigned)grid), dim3(threads), smem, stream, 1, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int LW, int L, bool SYM, bool CLAMP, bool SG>
cudaError_t launch_pow2(const RotQuantArgs& a, cudaStream_t stream) {
  using S = Pow2Shape<LW, L>;
  return launch_rows(rq_pow2_kernel<LW, L, SYM, CLAMP, SG>, S::T, Pow2Smem<LW, L>::BYTES, a, stream);
}

template <bool SYM, bool CLAMP, bool SG = false>
cudaError_t launch_pow2_for(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  *handled = true;
  switch (a.n_pow2) {
    case 512: return launch_pow2<0, 1, SYM, CLAMP, SG>(a, stream);
    case 1024: return launch_pow2<0, 2, SYM, CLAMP, SG>(a, stream);
    case 2048: return launch_pow2<1, 1, SYM, CLAMP, SG>(a, stream);
    case 4096: return launch_pow2<1, 2, SYM, CLAMP, SG>(a, stream);
    case 8192: return launch_pow2<2, 1, SYM, CLAMP, SG>(a, stream);
    case 16384: return launch_pow2<2, 2, SYM, CLAMP, SG>(a, stream);
  }
  *handled = false;
  return cudaSuccess;
}

template <bool SYM, bool CLAMP>
cudaError_t launch_norot_for(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  const int64_t nchunk = a.K / 8;
  const int64_t warps = (nchunk + 32 * kNoRotCPT - 1) / (32 * kNoRotCPT);
  *handled = warps <= 16;
  if (!*handled) return cudaSuccess;
  // one CTA per row, no persistence: every row's loads are in flight at once
  // when the grid is resident (2048 rows of 4096 need 2048 CTAs of 64 threads)
  auto kern = rq_norot_kernel<SYM, CLAMP>;
  const int threads = (int)(32 * warps);
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, threads, 0, &per_sm);
  if (e != cudaSuccess) return e;
  e = launch_pdl(kern, dim3((unsigned)a.rows), dim3(threads), 0, stream, 1, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rotate_quant_act_fast(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  *handled = false;
  if (a.rows == 0 || a.rowsum) return cudaSuccess;
  const bool clamp = a.clip < 1.0f;
  if (a.n_small == 0) {
    if (a.symmetric)
      return clamp ? launch_norot_for<true, true>(a, stream, handled) : launch_norot_for<true, false>(a, stream, handled);
    return clamp ? launch_norot_for<false, true>(a, stream, handled) : launch_norot_for<false, false>(a, stream, handled);
  }
  if (a.n_small == 1 && a.signs) {   // random signs: the unclipped forms (clipped ones take the generic kernel)
    if (clamp) return cudaSuccess;
    return a.symmetric ? launch_pow2_for<true, false, true>(a, stream, handled)
                       : launch_pow2_for<false, false, true>(a, stream, handled);
  }
  if (a.n_small == 1) {
    const cudaError_t e = launch_rotate_quant_act_tc(a, stream, handled);
    if (*handled || e != cudaSuccess) return e;
    if (a.symmetric)
      return clamp ? launch_pow2_for<true, true>(a, stream, handled) : launch_pow2_for<true, false>(a, stream, handled);
    return clamp ? launch_pow2_for<false, true>(a, stream, handled) : launch_pow2_for<false, false>(a, stream, handled);
  }
  return cudaSuccess;
}

}  // namespace spinq
