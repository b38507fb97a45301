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
// so each lane multiplies the raw code values by q, and the value update
// dequantizes in registers.  Split over the cache length (flash decoding):
//
//   partial kernel  grid (chunk, kv head, batch), 4 warps.  Lane l owns the
//     dimensions D/32 * l .. of the head; a warp takes blocks of 32 / G
//     tokens, so that its G query heads x 32 / G tokens are 32 dot products,
//     summed across the warp by a transpose-reduction (after it lane j holds
//     dot product j: 31 shuffles for 32 sums).  The block's softmax weights
//     go through shared memory to every lane for the value update.  Online
//     softmax state per head; the 4 warps merge at the end and write
//     (max, sum, o[D]) of the chunk to the workspace.
//   combine kernel  one warp per (batch, query head) merges the chunks.
#include <cuda_fp16.h>
#include <float.h>

#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

constexpr int kAttnWarps = 4;

__device__ __forceinline__ float nib(uint32_t w, int i) {
  // code i of w as a float: 2^23 + u read as fp32 bits, minus 2^23
  return __uint_as_float(0x4B000000u | ((w >> (4 * i)) & 15u)) - 8388608.f;
}

template <int D, int G>
__global__ void __launch_bounds__(kAttnWarps * 32, 4) attn_partial_kernel(AttnArgs a, int chunk_len, int nchunk) {
  constexpr int DPL = D / 32;                 // dimensions per lane
  constexpr int NT = 32 / G < 8 ? 32 / G : 8; // tokens per block
  constexpr int NV = NT * G;                  // dot products per block (8, 16 or 32)
  constexpr int R = 32 / NV;                  // lanes that end up holding each of them
  __shared__ float p_s[kAttnWarps][32];
  __shared__ float c_s[kAttnWarps][G];
  __shared__ float m_s[kAttnWarps][G], l_s[kAttnWarps][G];
  __shared__ float o_s[kAttnWarps][G][D];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int chunk = blockIdx.x, hk = blockIdx.y, b = blockIdx.z;
  pdl_wait();
  pdl_trigger();
  int64_t L = a.lens ? (int64_t)a.lens[b] : a.S;
  L = L < 0 ? 0 : (L > a.S ? a.S : L);
  const int64_t t0 = (int64_t)chunk * chunk_len;
  const int64_t t1 = t0 + chunk_len < L ? t0 + chunk_len : L;

  // this lane's slice of the G query heads, and each head's sum over D
  float q[G][DPL], qsum[G];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    const __half* qh = reinterpret_cast<const __half*>(a.q) + ((size_t)b * a.Hq + (size_t)hk * G + h) * D;
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < DPL; ++i) {
      q[h][i] = __half2float(qh[DPL * lane + i]);
      s += q[h][i];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    qsum[h] = s;
  }
  float m[G], l[G], acc[G][DPL];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    m[h] = -FLT_MAX;
    l[h] = 0.f;
#pragma unroll
    for (int i = 0; i < DPL; ++i) acc[h][i] = 0.f;
  }
  // this lane's pair of the block: value vi = lane / R, token jt = vi / G,
  // head jh = vi % G
  const int vi = lane / R, jt = vi / G, jh = vi % G;
  const size_t kv_stride = (size_t)a.Hkv;   // rows between consecutive tokens

  // Every load of a block (key and value codes, their scales) is issued
  // before any arithmetic on it: one memory round trip per block.
  struct Blk {
    uint32_t kw[NT], vw[NT];
    float ka, kb;     // key scale / zero of token jt (this lane's pair)
    float va, vb;     // value scale / zero of token (lane % NT)
  };
  auto load = [&](int64_t blk, Blk& x) {
#pragma unroll
    for (int tt = 0; tt < NT; ++tt) {
      const int64_t t = blk + tt;
      const size_t r = ((size_t)b * a.S + t) * kv_stride + hk;
      const uint8_t* kc = a.k_codes + r * (D / 2) + (DPL / 2) * lane;
      const uint8_t* vc = a.v_codes + r * (D / 2) + (DPL / 2) * lane;
      const bool in = t < t1;
      x.kw[tt] = in ? (DPL == 4 ? (uint32_t)*reinterpret_cast<const uint16_t*>(kc) : (uint32_t)*kc) : 0u;
      x.vw[tt] = in ? (DPL == 4 ? (uint32_t)*reinterpret_cast<const uint16_t*>(vc) : (uint32_t)*vc) : 0u;
    }
    const int64_t tk = blk + jt, tv = blk + (lane % NT);
    const size_t rk = ((size_t)b * a.S + tk) * kv_stride + hk, rv = ((size_t)b * a.S + tv) * kv_stride + hk;
    x.ka = tk < t1 ? a.k_scale[rk] : 0.f;
    x.kb = tk < t1 ? a.k_zero[rk] : 0.f;
    x.va = tv < t1 ? a.v_scale[rv] : 0.f;
    x.vb = tv < t1 ? a.v_zero[rv] : 0.f;
  };
  const int64_t step = (int64_t)kAttnWarps * NT;
  Blk cur;
  for (int64_t blk = t0 + (int64_t)warp * NT; blk < t1; blk += step) {
    load(blk, cur);
    // ---- scores: 32 dot products (token, head) of the block
    float v[NV];
#pragma unroll
    for (int tt = 0; tt < NT; ++tt) {
      float u[DPL];
#pragma unroll
      for (int i = 0; i < DPL; ++i) u[i] = nib(cur.kw[tt], i);
#pragma unroll
      for (int h = 0; h < G; ++h) {
        float d = 0.f;
#pragma unroll
        for (int i = 0; i < DPL; ++i) d = fmaf(q[h][i], u[i], d);
        v[tt * G + h] = d;
      }
    }
    // transpose-reduction: halving rounds over the top lane bits, then plain
    // sums over the rest; after it, lane j holds the warp sum of v[j / R]
#pragma unroll
    for (int o = 16, n = NV; n > 1; o >>= 1, n >>= 1) {
      const bool up = (lane & o) != 0;
#pragma unroll
      for (int i = 0; i < n / 2; ++i) {
        const float send = up ? v[i] : v[i + n / 2];
        const float keep = up ? v[i + n / 2] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
      }
    }
#pragma unroll
    for (int o = R / 2; o >= 1; o >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
    const int64_t tj = blk + jt;
    const float s = tj < t1 ? a.scale * fmaf(cur.ka, v[0], cur.kb * qsum[jh]) : -FLT_MAX;
    // block maximum and sum per head: lanes with the same head differ in the bits above log2(G)
    float mx = s;
#pragma unroll
    for (int o = G * R; o < 32; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float mh = m[0];
#pragma unroll
    for (int h = 1; h < G; ++h)
      if (jh == h) mh = m[h];
    const float mnew = fmaxf(mh, mx);
    const float p = tj < t1 ? __expf(s - mnew) : 0.f;
    float ps = p;
#pragma unroll
    for (int o = G * R; o < 32; o <<= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
    if (lane % R == 0) p_s[warp][vi] = p;
    if (jt == 0 && lane % R == 0) c_s[warp][jh] = __expf(mh - mnew);   // lane h R holds head h
    __syncwarp();
    // new per-head state in every lane
#pragma unroll
    for (int h = 0; h < G; ++h) {
      const float corr = c_s[warp][h];
      const float m_h = __shfl_sync(0xffffffffu, mnew, h * R);
      const float s_h = __shfl_sync(0xffffffffu, ps, h * R);
      l[h] = l[h] * corr + s_h;
      m[h] = m_h;
#pragma unroll
      for (int i = 0; i < DPL; ++i) acc[h][i] *= corr;
    }
    // ---- values (weights of masked tokens are 0, their codes 0)
#pragma unroll
    for (int tt = 0; tt < NT; ++tt) {
      const float al = __shfl_sync(0xffffffffu, cur.va, tt), be = __shfl_sync(0xffffffffu, cur.vb, tt);
      float vv[DPL];
#pragma unroll
      for (int i = 0; i < DPL; ++i) vv[i] = fmaf(al, nib(cur.vw[tt], i), be);
#pragma unroll
      for (int h = 0; h < G; ++h) {
        const float pw = p_s[warp][tt * G + h];
#pragma unroll
        for (int i = 0; i < DPL; ++i) acc[h][i] = fmaf(pw, vv[i], acc[h][i]);
      }
    }
    __syncwarp();
  }
  // ---- merge the warps and write the chunk's partial result
#pragma unroll
  for (int h = 0; h < G; ++h) {
    if (lane == 0) {
      m_s[warp][h] = m[h];
      l_s[warp][h] = l[h];
    }
#pragma unroll
    for (int i = 0; i < DPL; ++i) o_s[warp][h][DPL * lane + i] = acc[h][i];
  }
  __syncthreads();
  for (int e = threadIdx.x; e < G * (D + 2); e += kAttnWarps * 32) {
    const int h = e / (D + 2), d = e % (D + 2);
    float M = -FLT_MAX;
    for (int w = 0; w < kAttnWarps; ++w) M = fmaxf(M, m_s[w][h]);
    float val = 0.f;
    if (d == 0) {
      val = M;
    } else {
      for (int w = 0; w < kAttnWarps; ++w) {
        const float f = l_s[w][h] > 0.f ? __expf(m_s[w][h] - M) : 0.f;
        val += f * (d == 1 ? l_s[w][h] : o_s[w][h][d - 2]);
      }
    }
    const size_t hq = (size_t)hk * G + h;
    a.workspace[(((size_t)b * a.Hq + hq) * nchunk + chunk) * (D + 2) + d] = val;
  }
}

template <int D>
__global__ void __launch_bounds__(128) attn_combine_kernel(AttnArgs a, int nchunk) {
  const int lane = threadIdx.x & 31;
  const int64_t bh = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  pdl_wait();
  pdl_trigger();
  if (bh >= a.B * a.Hq) return;
  const float* ws = a.workspace + (size_t)bh * nchunk * (D + 2);
  float M = -FLT_MAX;
  for (int c = 0; c < nchunk; ++c) M = fmaxf(M, ws[(size_t)c * (D + 2)]);
  constexpr int DPL = D / 32;
  float o[DPL] = {}, den = 0.f;
  for (int c = 0; c < nchunk; ++c) {
    const float* w = ws + (size_t)c * (D + 2);
    if (!(w[1] > 0.f)) continue;
    const float f = __expf(w[0] - M);
    den += f * w[1];
#pragma unroll
    for (int i = 0; i < DPL; ++i) o[i] += f * w[2 + DPL * lane + i];
  }
  const float inv = den > 0.f ? 1.f / den : 0.f;
  __half* out = reinterpret_cast<__half*>(a.out) + (size_t)bh * D + DPL * lane;
#pragma unroll
  for (int i = 0; i < DPL; ++i) out[i] = __float2half_rn(o[i] * inv);
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
  // about eight CTAs per SM, at least 32 tokens per chunk
  const int64_t pairs = B * Hkv > 0 ? B * Hkv : 1;
  int64_t n = (8 * (int64_t)device_sm_count() + pairs - 1) / pairs;
  const int64_t by_len = (S + 31) / 32;
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
