// decode_attention.cu -- spinq_decode_attention_kv4: attention of one decode
// query per (batch, query head) over the 4-bit KV cache that
// spinq_rotate_quant_kv writes (Sec. 3.1: R3 rotates Q and K over head_dim so
// that Q K^T is unchanged while the cache quantizes to 4 bits; appendix
// "Latency measurement on GPU": the time per generated token).
//
//   s_t = scale * q . k_t,   k_t = alpha_t u_t + beta_t (asymmetric Eq. 1),
//   o   = sum_t softmax_t(s)_t v_t,  v_t = alpha'_t u'_t + beta'_t,
// for t < lens[b]; query head h reads kv head h / G (G = Hq / Hkv).
//
// The codes are never expanded to memory: the score is
//   s_t = scale * (alpha_t (q . u_t) + beta_t sum_d q_d),
// and the value sum is
//   o = sum_t p_t (alpha'_t u'_t + beta'_t)
//     = r * sum_t (p_t alpha'_t / r) u'_t + sum_t p_t beta'_t,
// so both products take the raw codes u as fp16 operands of the tensor core
// (mma.sync m16n8k16, fp32 accumulation).  A code is unpacked by one mask:
// read as an fp16 bit pattern it is the subnormal u 2^-24 (or 16 u 2^-24),
// which the tensor core multiplies exactly, and the product with an fp16
// query element or weight is exact in fp32.  r is the maximum value scale of
// the warp's tokens and the softmax maximum moves only in steps of more than
// 2^8, so the fp16 weights p alpha' / r stay within [0, 256].
// Split over the cache length (flash decoding):
//
//   partial kernel  grid (chunk, kv head, batch), 4 warps; a warp takes steps
//     of 16 tokens.  Both products put the G query heads of the kv head on
//     the MMA's N side (8 columns, columns >= G zero), so no accumulator
//     register holds padding.  Scores S^T = K q^T: M = the 16 tokens,
//     K = head_dim.  Lane (g, c) (g = lane / 4, c = lane % 4) loads bytes
//     [c D/8, (c+1) D/8) of key rows g and g + 8, and the order in which
//     head_dim meets the MMA's k index is chosen so that those bytes are
//     exactly the lane's A fragments (the query fragments use the same
//     order).  Values O^T = V^T P^T: M = 16 of head_dim, K = the 16 tokens;
//     the weights' fp16 pairs (one token, two heads) become the B fragment
//     (one head, two tokens) by an 8x8 transpose (movmatrix), and lane (g, c)
//     loads bytes [g D/16, (g+1) D/16) of value rows 2c, 2c+1, 2c+8, 2c+9,
//     pairing two tokens' codes per fp16x2 register with a byte permute.
//     Online softmax per step in base 2; the 4 warps merge at the end and
//     write (max, sum, o[D]) of the chunk to the workspace.
//   combine kernel  one warp per (batch, query head) merges the chunks.
#include <cuda_fp16.h>
#include <float.h>

#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

constexpr int kAttnWarps = 4;
constexpr int kAttnCtasPerSm = 4;   // resident CTAs per SM the chunking plans for
constexpr int kAttnStages = 4;      // 16-token stages in each warp's copy ring
constexpr float kLog2e = 1.4426950408889634f;

// Two codes of a word as an fp16 pair by one mask: the codes at bits 0-3 and
// 16-19 read as fp16 bit patterns are the subnormals u 2^-24, those at bits
// 4-7 and 20-23 are 16 u 2^-24.  The tensor core multiplies subnormal fp16
// operands exactly; the factors 2^24 and 16 are taken out of the products'
// other operand or of the accumulators.
__device__ __forceinline__ uint32_t codes_lo(uint32_t x) { return x & 0x000F000Fu; }
__device__ __forceinline__ uint32_t codes_hi(uint32_t x) { return x & 0x00F000F0u; }
constexpr float kCodeScale = 16777216.f;   // 2^24

// 2^x (ex2.approx.ftz: relative error below 2^-22; -inf and large negative x
// give +0)
__device__ __forceinline__ float exp2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
  return y;
}

// 8x8 transpose of fp16 pairs across the warp: lane (g, c) gives elements
// (g, 2c), (g, 2c+1) and gets (2c, g), (2c+1, g).
__device__ __forceinline__ uint32_t transpose8x8(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;\n" : "=r"(y) : "r"(x));
  return y;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// Shared-memory ring of one warp: kAttnStages stages of 16 tokens, each the
// key and value code rows (D/2 bytes, rows RSB = D/2 + 16 bytes apart, which
// spreads the lanes' fragment reads evenly over the banks) and per token the
// four scales (key scale, key zero, value scale, value zero).
template <int D>
struct AttnRing {
  static constexpr int RSB = D / 2 + 16;
  static constexpr int KOFF = 0, VOFF = 16 * RSB, SOFF = 32 * RSB;
  static constexpr int STAGE = 32 * RSB + 16 * 16;
  static constexpr int WARP = kAttnStages * STAGE;
};

// index of element d of head h in a warp's output staging (which reuses the
// ring once the loop is done): one word of padding per 16 and 4 per head make
// the lanes' stores (heads 2c + e, dims 16g + j for D = 128) fall in 32
// different banks
template <int D>
__device__ __forceinline__ int stage_idx(int h, int d) {
  return h * (D + D / 16 + 4) + d + d / 16;
}

template <int D, int G>
__global__ void __launch_bounds__(kAttnWarps * 32, kAttnCtasPerSm) attn_partial_kernel(AttnArgs a, int chunk_len,
                                                                                       int nchunk) {
  constexpr int KW = D / 32;   // words of key codes per lane and token row (D/8 bytes)
  constexpr int VW = D / 64;   // words of value codes per lane and token row (D/16 bytes)
  constexpr int NS = D / 16;   // k16 slices of the score product
  constexpr int NM = D / 16;   // m16 tiles of head_dim in the value product
  constexpr int CPR = D / 32;  // 16-byte chunks per code row
  constexpr int NCP = CPR / 2; // 16-byte copies per lane and code matrix
  using Ring = AttnRing<D>;
  static_assert(G >= 1 && G <= 8, "at most 8 query heads per kv head");
  static_assert(G * (D + D / 16 + 4) * 4 <= Ring::WARP, "output staging fits in the warp's ring");
  __shared__ __align__(16) unsigned char ring_s[kAttnWarps][Ring::WARP];
  __shared__ float m_s[kAttnWarps][G], l_s[kAttnWarps][G];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, c = lane & 3;
  const int chunk = blockIdx.x, hk = blockIdx.y, b = blockIdx.z;
  pdl_wait();
  pdl_trigger();
  int64_t L = a.lens ? (int64_t)a.lens[b] : a.S;
  L = L < 0 ? 0 : (L > a.S ? a.S : L);
  const int64_t t0 = (int64_t)chunk * chunk_len;
  const int64_t t1 = t0 + chunk_len < L ? t0 + chunk_len : L;
  const int span = t1 > t0 ? (int)(t1 - t0) : 0;   // tokens of the chunk
  // this warp's steps: 16 tokens each, steps warp, warp + 4, ... of the chunk
  const int nstep_chunk = (span + 15) / 16;
  const int nstep = nstep_chunk > warp ? (nstep_chunk - warp + kAttnWarps - 1) / kAttnWarps : 0;

  // Copy sources.  A step's rows past the chunk are still copied (their
  // scores are masked and their value scales zeroed below), clamped to the
  // batch's last cache row so that every address lies inside the cache.
  // Offsets within a batch's cache fit in 31 bits (checked by the caller).
  const uint32_t row = (uint32_t)a.Hkv * (D / 2);   // bytes between consecutive tokens' codes
  const size_t tok0 = (size_t)b * a.S * a.Hkv + hk + (size_t)t0 * a.Hkv;   // scale index of token t0
  const int last = (int)(a.S - 1 - t0);                                     // last cache row, from t0
  const uint8_t* kb = a.k_codes + tok0 * (D / 2);
  const uint8_t* vb = a.v_codes + tok0 * (D / 2);
  const int ch = lane % CPR;
  const int ts = lane & 15;   // this lane's token of the scale copies
  const float* sb0 = (lane < 16 ? a.k_scale : a.v_scale) + tok0;
  const float* sb1 = (lane < 16 ? a.k_zero : a.v_zero) + tok0;
  const uint32_t ring = smem_u32(ring_s[warp]);
  const uint32_t sdst = Ring::SOFF + 16 * ts + 8 * (lane >> 4);
  // copies of step i into stage i % kAttnStages: lane j moves 16-byte chunks
  // j, j + 32, ... of the 16 x CPR chunks of each code matrix and two of the
  // 64 scales
  auto issue = [&](int i) {
    if (i < nstep) {
      const int tb = 16 * (warp + kAttnWarps * i);   // first token of the step, from t0
      const uint32_t st = ring + (uint32_t)(i % kAttnStages) * Ring::STAGE;
      if (tb + 15 <= last) {   // the whole step inside the cache
#pragma unroll
        for (int k = 0; k < NCP; ++k) {
          const int rr = (lane + 32 * k) / CPR;
          const uint32_t off = (uint32_t)(tb + rr) * row + 16 * ch;
          cp_async16(st + Ring::KOFF + rr * Ring::RSB + 16 * ch, kb + off);
          cp_async16(st + Ring::VOFF + rr * Ring::RSB + 16 * ch, vb + off);
        }
        const uint32_t so = (uint32_t)(tb + ts) * (uint32_t)a.Hkv;
        cp_async4(st + sdst, sb0 + so);
        cp_async4(st + sdst + 4, sb1 + so);
      } else {
#pragma unroll
        for (int k = 0; k < NCP; ++k) {
          const int rr = (lane + 32 * k) / CPR;
          const uint32_t off = (uint32_t)min(tb + rr, last) * row + 16 * ch;
          cp_async16(st + Ring::KOFF + rr * Ring::RSB + 16 * ch, kb + off);
          cp_async16(st + Ring::VOFF + rr * Ring::RSB + 16 * ch, vb + off);
        }
        const uint32_t so = (uint32_t)min(tb + ts, last) * (uint32_t)a.Hkv;
        cp_async4(st + sdst, sb0 + so);
        cp_async4(st + sdst + 4, sb1 + so);
      }
    }
    cp_async_commit();   // an empty group past the end keeps the wait count uniform
  };
  // pairs of steps: while pair j is computed, pair j + 1 is in flight
  static_assert(kAttnStages == 4, "two pairs of stages");
  issue(0);
  issue(1);

  // value-scale reference of this warp: r = max alpha' over its tokens (the
  // fp16 weights p alpha' / r stay within [0, 256]); the loads overlap the
  // copies in flight
  float r = 0.f;
  for (int j = lane; j < 16 * nstep; j += 32) {
    const int t = 16 * (warp + kAttnWarps * (j >> 4)) + (j & 15);
    if (t < span) r = fmaxf(r, __ldg(a.v_scale + tok0 + (size_t)t * a.Hkv));
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) r = fmaxf(r, __shfl_xor_sync(0xffffffffu, r, off));
  const float rinv = r > 0.f ? 1.f / r : 0.f;

  // B fragments of query head g (zero for g >= G) in the order the key codes
  // meet the MMA: slice 2w + e, k = 2c, 2c+1 take dimensions 2(cD/8 + 4w + e)
  // and that + 4 (low nibbles of the lane's bytes 4w + e and 4w + e + 2),
  // k = 2c+8, 2c+9 the same plus one (high nibbles).
  uint32_t qb[NS][2];
  float qs = 0.f;
  {
    const __half* qh =
        reinterpret_cast<const __half*>(a.q) + ((size_t)b * a.Hq + (size_t)hk * G + (g < G ? g : 0)) * D;
    // slices 2w and 2w + 1 take the lane's dimensions cD/4 + 8w .. + 7: one
    // 16-byte load
#pragma unroll
    for (int w = 0; w < KW; ++w) {
      uint4 raw = *reinterpret_cast<const uint4*>(qh + c * (D / 4) + 8 * w);
      if (g >= G) raw = make_uint4(0u, 0u, 0u, 0u);
      const __half* hv = reinterpret_cast<const __half*>(&raw);
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const __half x0 = hv[2 * e], x1 = hv[2 * e + 4], y0 = hv[2 * e + 1], y1 = hv[2 * e + 5];
        // the high-nibble positions meet codes 16 u 2^-24: their query
        // elements are divided by 16 (exact in fp16 above 2^-10)
        const __half2 lo = __halves2half2(x0, x1);
        const __half2 hi = __hmul2(__halves2half2(y0, y1), __float2half2_rn(0.0625f));
        qb[2 * w + e][0] = *reinterpret_cast<const uint32_t*>(&lo);
        qb[2 * w + e][1] = *reinterpret_cast<const uint32_t*>(&hi);
        qs += (__half2float(x0) + __half2float(x1)) + (__half2float(y0) + __half2float(y1));
      }
    }
    qs += __shfl_xor_sync(0xffffffffu, qs, 1);
    qs += __shfl_xor_sync(0xffffffffu, qs, 2);
  }
  // this lane's accumulator columns are heads 2c and 2c + 1 (head h's sum sits
  // in lane 4h); the scores carry the factor scale log2 e
  const float ks = a.scale * kLog2e;
  const float qsk[2] = {ks * __shfl_sync(0xffffffffu, qs, 8 * c), ks * __shfl_sync(0xffffffffu, qs, 8 * c + 4)};

  // Running state of heads 2c + e in this lane: the score maximum m (base 2),
  // the lane's share (tokens g, g + 8 of each step) of the weight sum l and of
  // sum p beta', and o[mu] = sum p alpha' u / r for dimensions gD/8 + 2mu
  // (o[mu][e]) and gD/8 + 2mu + 1 (o[mu][2 + e]).
  float o[NM][4];
#pragma unroll
  for (int mu = 0; mu < NM; ++mu) o[mu][0] = o[mu][1] = o[mu][2] = o[mu][3] = 0.f;
  float m[2] = {-FLT_MAX, -FLT_MAX}, l[2] = {0.f, 0.f}, bs[2] = {0.f, 0.f};

  const int npair = (nstep + 1) / 2;
  for (int jp = 0; jp < npair; ++jp) {
    issue(2 * jp + 2);
    issue(2 * jp + 3);
    cp_async_wait<2>();   // this lane's copies of steps 2jp, 2jp + 1 have landed
    __syncwarp();         // and every other lane's
    // Step u of the pair is step 2jp + u of the warp; the second step of the
    // last pair may lie past the chunk (rem <= 0: every token masked, its
    // stage holds stale data that only meets masked weights).
    const unsigned char* st[2];
    int rem[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int i = 2 * jp + u;
      st[u] = ring_s[warp] + (i % kAttnStages) * Ring::STAGE;
      rem[u] = span - 16 * (warp + kAttnWarps * i);
    }
    // ---- scores S^T of both steps (two independent MMA chains)
    uint32_t kx[2][2][KW];
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const unsigned char* p = st[u] + Ring::KOFF + (g + 8 * hf) * Ring::RSB + c * (D / 8);
        if constexpr (KW == 4) {
          const uint4 v = *reinterpret_cast<const uint4*>(p);
          kx[u][hf][0] = v.x, kx[u][hf][1] = v.y, kx[u][hf][2] = v.z, kx[u][hf][3] = v.w;
        } else {
          const uint2 v = *reinterpret_cast<const uint2*>(p);
          kx[u][hf][0] = v.x, kx[u][hf][1] = v.y;
        }
      }
    // four accumulators (step u, slice parity) keep the dependent chains short
    float sacc[2][4], sodd[2][4];
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
      for (int k = 0; k < 4; ++k) sacc[u][k] = sodd[u][k] = 0.f;
#pragma unroll
    for (int w = 0; w < KW; ++w)
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const uint32_t x0 = kx[u][0][w], x1 = kx[u][1][w], y0 = x0 >> 8, y1 = x1 >> 8;
        const uint32_t a0[4] = {codes_lo(x0), codes_lo(x1), codes_hi(x0), codes_hi(x1)};
        mma_16816_f16_f32_acc(sacc[u], a0, qb[2 * w][0], qb[2 * w][1]);
        const uint32_t a1[4] = {codes_lo(y0), codes_lo(y1), codes_hi(y0), codes_hi(y1)};
        mma_16816_f16_f32_acc(sodd[u], a1, qb[2 * w + 1][0], qb[2 * w + 1][1]);
      }
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
      for (int k = 0; k < 4; ++k) sacc[u][k] += sodd[u][k];
    // scores of tokens g (hf 0) and g + 8 (hf 1) of each step for heads 2c + e;
    // tokens past the chunk: score -inf-like, value scale and zero 0 (their
    // rows were copied from the clamped address and may hold anything)
    float sc[2][2][2], wv[2][2], zv[2][2], mx[2] = {-FLT_MAX, -FLT_MAX};
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const float4 f = *reinterpret_cast<const float4*>(st[u] + Ring::SOFF + 16 * (g + 8 * hf));
        const bool in = g + 8 * hf < rem[u];
        const float ka = (ks * kCodeScale) * f.x;
        wv[u][hf] = in ? f.z * rinv : 0.f;
        zv[u][hf] = in ? f.w : 0.f;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          sc[u][hf][e] = in ? fmaf(ka, sacc[u][2 * hf + e], f.y * qsk[e]) : -FLT_MAX;
          mx[e] = fmaxf(mx[e], sc[u][hf][e]);
        }
      }
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      mx[0] = fmaxf(mx[0], __shfl_xor_sync(0xffffffffu, mx[0], off));
      mx[1] = fmaxf(mx[1], __shfl_xor_sync(0xffffffffu, mx[1], off));
    }
    // The running maximum moves only when a score exceeds it by more than 8
    // (base 2), so the weights p stay below 2^8 and the accumulators are
    // rescaled rarely.  The pair's first step holds a token of the chunk, so
    // m is finite from the first pair on and the masked scores give p = 0.
    float p[2][2][2], corr[2];
    bool moved = false;
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const float mnew = mx[e] > m[e] + 8.f ? mx[e] : m[e];
      moved |= mnew != m[e];
      corr[e] = exp2_approx(m[e] - mnew);
      float ps = 0.f, pz = 0.f;
#pragma unroll
      for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          p[u][hf][e] = exp2_approx(sc[u][hf][e] - mnew);
          ps += p[u][hf][e];
          pz = fmaf(p[u][hf][e], zv[u][hf], pz);
        }
      l[e] = fmaf(l[e], corr[e], ps);
      bs[e] = fmaf(bs[e], corr[e], pz);
      m[e] = mnew;
    }
    if (__any_sync(0xffffffffu, moved)) {
#pragma unroll
      for (int mu = 0; mu < NM; ++mu) {
        o[mu][0] *= corr[0], o[mu][2] *= corr[0];
        o[mu][1] *= corr[1], o[mu][3] *= corr[1];
      }
    }
    // ---- o^T += V^T P'^T with P' = p alpha' / r in fp16: the pairs (token,
    // heads 2c, 2c+1) transposed to (head g, tokens 2c, 2c+1) are the B
    // fragment (tokens 0..7 in register 0, 8..15 in register 1)
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const uint32_t pb0 = transpose8x8(pack_half2_bits(p[u][0][0] * wv[u][0], p[u][0][1] * wv[u][0]));
      const uint32_t pb1 = transpose8x8(pack_half2_bits(p[u][1][0] * wv[u][1], p[u][1][1] * wv[u][1]));
      uint32_t vx[4][VW];
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        const unsigned char* q = st[u] + Ring::VOFF + (8 * (rr >> 1) + 2 * c + (rr & 1)) * Ring::RSB + g * (D / 16);
        if constexpr (VW == 2) {
          const uint2 v = *reinterpret_cast<const uint2*>(q);
          vx[rr][0] = v.x, vx[rr][1] = v.y;
        } else {
          vx[rr][0] = *reinterpret_cast<const uint32_t*>(q);
        }
      }
#pragma unroll
      for (int w = 0; w < VW; ++w) {
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          // bytes 2q, 2q+1 of word w of rows 2c | 2c+1 (and 2c+8 | 2c+9): the
          // same dimension of two tokens lands in one fp16 pair; the lane's
          // nibbles 8w + 4q + 2kk go to row g, + 1 to row g + 8
          const uint32_t xa = __byte_perm(vx[0][w], vx[1][w], q ? 0x7632 : 0x5410);
          const uint32_t xb = __byte_perm(vx[2][w], vx[3][w], q ? 0x7632 : 0x5410);
          const uint32_t a0[4] = {codes_lo(xa), codes_hi(xa), codes_lo(xb), codes_hi(xb)};
          mma_16816_f16_f32_acc(o[4 * w + 2 * q], a0, pb0, pb1);
          const uint32_t ya = xa >> 8, yb = xb >> 8;
          const uint32_t a1[4] = {codes_lo(ya), codes_hi(ya), codes_lo(yb), codes_hi(yb)};
          mma_16816_f16_f32_acc(o[4 * w + 2 * q + 1], a1, pb0, pb1);
        }
      }
    }
    __syncwarp();   // every lane is done with the pair's stages before they are refilled
  }
  cp_async_wait<0>();
  __syncwarp();

  // ---- merge the warps and write the chunk's partial result
#pragma unroll
  for (int e = 0; e < 2; ++e)
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      l[e] += __shfl_xor_sync(0xffffffffu, l[e], off);
      bs[e] += __shfl_xor_sync(0xffffffffu, bs[e], off);
    }
  float* o_w = reinterpret_cast<float*>(ring_s[warp]);
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int h = 2 * c + e;
    if (h < G) {
#pragma unroll
      for (int mu = 0; mu < NM; ++mu) {
        const int d = g * (D / 8) + 2 * mu;
        // rows g + 8 took codes 16 u 2^-24, rows g codes u 2^-24
        o_w[stage_idx<D>(h, d)] = fmaf(r * kCodeScale, o[mu][e], bs[e]);
        o_w[stage_idx<D>(h, d + 1)] = fmaf(r * (kCodeScale / 16.f), o[mu][2 + e], bs[e]);
      }
      if (g == 0) {
        m_s[warp][h] = m[e];
        l_s[warp][h] = l[e];
      }
    }
  }
  __syncthreads();
  for (int e = threadIdx.x; e < G * (D + 2); e += kAttnWarps * 32) {
    const int h = e / (D + 2), d = e % (D + 2);
    float M = -FLT_MAX;
#pragma unroll
    for (int w = 0; w < kAttnWarps; ++w) M = fmaxf(M, m_s[w][h]);
    float val = 0.f;
    if (d == 0) {
      val = M;
    } else {
#pragma unroll
      for (int w = 0; w < kAttnWarps; ++w) {
        const float fw = l_s[w][h] > 0.f ? exp2_approx(m_s[w][h] - M) : 0.f;
        val += fw * (d == 1 ? l_s[w][h] : reinterpret_cast<const float*>(ring_s[w])[stage_idx<D>(h, d - 2)]);
      }
    }
    const size_t hq = (size_t)hk * G + h;
    a.workspace[(((size_t)b * a.Hq + hq) * nchunk + chunk) * (D + 2) + d] = val;
  }
}

template <int D>
__global__ void __launch_bounds__(128) attn_combine_kernel(AttnArgs a, int nchunk) {
  constexpr int DPL = D / 32;
  const int lane = threadIdx.x & 31;
  const int64_t bh = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  pdl_wait();
  pdl_trigger();
  if (bh >= a.B * a.Hq) return;
  const float* ws = a.workspace + (size_t)bh * nchunk * (D + 2);
  // the chunks' maxima in parallel over the lanes, then the weighted sums;
  // the loads of up to eight chunks are in flight together
  float M = -FLT_MAX;
  for (int c = lane; c < nchunk; c += 32) M = fmaxf(M, ws[(size_t)c * (D + 2)]);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
  float o[DPL] = {}, den = 0.f;
  for (int c0 = 0; c0 < nchunk; c0 += 32) {
    const int c = c0 + lane;
    float f = 0.f;
    if (c < nchunk) {
      const float lc = ws[(size_t)c * (D + 2) + 1];
      f = lc > 0.f ? exp2_approx(ws[(size_t)c * (D + 2)] - M) : 0.f;
      den = fmaf(f, lc, den);
    }
    const int n = nchunk - c0 < 32 ? nchunk - c0 : 32;
#pragma unroll 8
    for (int j = 0; j < n; ++j) {
      const float fj = __shfl_sync(0xffffffffu, f, j);
      const float2* w = reinterpret_cast<const float2*>(ws + (size_t)(c0 + j) * (D + 2) + 2 + DPL * lane);
#pragma unroll
      for (int i = 0; i < DPL / 2; ++i) {
        const float2 v = w[i];
        o[2 * i] = fmaf(fj, v.x, o[2 * i]);
        o[2 * i + 1] = fmaf(fj, v.y, o[2 * i + 1]);
      }
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) den += __shfl_xor_sync(0xffffffffu, den, off);
  const float inv = den > 0.f ? 1.f / den : 0.f;
  __half* out = reinterpret_cast<__half*>(a.out) + (size_t)bh * D + DPL * lane;
#pragma unroll
  for (int i = 0; i < DPL; i += 2) *reinterpret_cast<__half2*>(out + i) = __floats2half2_rn(o[i] * inv, o[i + 1] * inv);
}

template <int D, int G>
cudaError_t launch_dg(const AttnArgs& a, int nchunk, cudaStream_t stream) {
  const int chunk_len = (int)((a.S + nchunk - 1) / nchunk);
  cudaError_t e = launch_pdl(attn_partial_kernel<D, G>, dim3((unsigned)nchunk, (unsigned)a.Hkv, (unsigned)a.B),
                             dim3(kAttnWarps * 32), 0, stream, 1, a, chunk_len, nchunk);
  if (e != cudaSuccess) return e;
  const int64_t groups = (a.B * a.Hq + 3) / 4;
  e = launch_pdl(attn_combine_kernel<D>, dim3((unsigned)groups), dim3(128), 0, stream, 1, a, nchunk);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_d(const AttnArgs& a, int nchunk, cudaStream_t stream) {
  switch (a.Hq / a.Hkv) {
    case 1: return launch_dg<D, 1>(a, nchunk, stream);
    case 2: return launch_dg<D, 2>(a, nchunk, stream);
    case 4: return launch_dg<D, 4>(a, nchunk, stream);
    case 8: return launch_dg<D, 8>(a, nchunk, stream);
  }
  return cudaErrorNotSupported;
}

}  // namespace

int decode_attention_chunks(int64_t B, int64_t S, int64_t Hkv) {
  // one wave of the resident CTAs (kAttnCtasPerSm per SM), at least 64
  // tokens per chunk
  const int64_t pairs = B * Hkv > 0 ? B * Hkv : 1;
  int64_t n = (int64_t)kAttnCtasPerSm * device_sm_count() / pairs;
  const int64_t by_len = (S + 63) / 64;
  if (n > by_len) n = by_len;
  if (n > 1024) n = 1024;
  return (int)(n < 1 ? 1 : n);
}

cudaError_t launch_decode_attention(const AttnArgs& a, int nchunk, cudaStream_t stream) {
  if (a.D == 128) return launch_d<128>(a, nchunk, stream);
  if (a.D == 64) return launch_d<64>(a, nchunk, stream);
  return cudaErrorNotSupported;
}

}  // namespace spinq
