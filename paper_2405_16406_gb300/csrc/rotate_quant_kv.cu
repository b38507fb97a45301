// rotate_quant_kv.cu -- R3 on Q and K over head_dim followed by the 4-bit
// asymmetric KV-cache quantizer (Sec. 3.1 R3; Eq. 1; appendix "Quantization
// choice").  V is quantized without rotation (R2 merged into W_v / W_o).
//
// Work unit: one warp, 8 rows of D elements (D = 64 or 128) of one tensor.
// A quad of lanes (g = lane/4 picks the row, c = lane%4) owns one row; lane c
// loads the 8*V consecutive elements [8Vc, 8Vc + 8V) as V 16-byte chunks
// (V = D/32).  Element index bits: e (3 bits, inside a chunk), v (log2 V
// bits, chunk within the lane), c (2 bits, the lane in the quad).
//
// Stage 1 runs on the tensor core, on the raw fp16 input: one m16n8k16 MMA
// per chunk with B = the 16-point Sylvester matrix contracts the 4 bits
// {e0, e2, c0, c1} (k = 2c + e0 + 8 e2); the two A rows g and g+8 carry e1 = 0
// and e1 = 1.  The outputs land in the lane that supplied the inputs, at the
// same element positions, already in fp32 (entries are +-1, so the products
// are exact and the sums are fp32 sums of 16 fp16 values).  The remaining
// bits (e1 and v) are radix-2 butterflies inside the lane.  For V the same
// MMA with B = I16 only widens fp16 to fp32 (exactly).
//
// Eq. 1 on the unnormalised rotated row: the codes do not depend on the
// 1/sqrt(D) factor, which is applied to alpha and beta (and to Q's output).
#include <cuda_fp16.h>
#include <float.h>

#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

constexpr int kWarps = 8;

__device__ __forceinline__ uint32_t h16_pair(int k0, int k1, int n, bool hadamard) {
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

template <int D, bool CLAMP, bool ROPE>
__global__ void __launch_bounds__(kWarps * 32) rotate_quant_kv_kernel(KVArgs a) {
  constexpr int V = D / 32;  // 16-byte chunks per lane
  const int lane = threadIdx.x & 31, g = lane >> 2, c = lane & 3;
  const int warp = threadIdx.x >> 5;

  // B fragments for n-tiles 0 (n = g) and 1 (n = g + 8)
  uint32_t bh[2][2], bi[2][2];
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
    const int n = g + 8 * nt;
    bh[nt][0] = h16_pair(2 * c, 2 * c + 1, n, true);
    bh[nt][1] = h16_pair(2 * c + 8, 2 * c + 9, n, true);
    bi[nt][0] = h16_pair(2 * c, 2 * c + 1, n, false);
    bi[nt][1] = h16_pair(2 * c + 8, 2 * c + 9, n, false);
  }

  pdl_wait();
  pdl_trigger();
  const int64_t gq = (a.rows_q + 7) / 8, gk = (a.rows_kv + 7) / 8;
  const int64_t total = gq + 2 * gk;
  const int64_t stride = (int64_t)gridDim.x * kWarps;
  for (int64_t G = (int64_t)blockIdx.x * kWarps + warp; G < total; G += stride) {
    int kind;  // 0 = Q, 1 = K, 2 = V
    int64_t grp;
    if (G < gq) {
      kind = 0;
      grp = G;
    } else if (G < gq + gk) {
      kind = 1;
      grp = G - gq;
    } else {
      kind = 2;
      grp = G - gq - gk;
    }
    const int64_t rows = kind == 0 ? a.rows_q : a.rows_kv;
    const int64_t row = grp * 8 + g;
    const bool valid = row < rows;
    const __half* src = reinterpret_cast<const __half*>(kind == 0 ? a.q_in : kind == 1 ? a.k_in : a.v_in);
    const uint4* p = reinterpret_cast<const uint4*>(src + row * D) + c * V;

    uint4 in[V];
#pragma unroll
    for (int v = 0; v < V; ++v) in[v] = valid ? __ldg(p + v) : make_uint4(0, 0, 0, 0);

    if (ROPE && kind != 2) {
      // Rotary embedding at the row's token position (rotate-half form), in
      // fp32 from the caller's (cos, sin) table, rounded back to fp16 like the
      // model's activations: y_i = x_i cos - x_{i+D/2} sin and
      // y_{i+D/2} = x_i sin + x_{i+D/2} cos.  Lanes c and c ^ 2 of a quad hold
      // the dimensions i and i + D/2 at the same register positions.
      const int64_t H = kind == 0 ? a.Hq : a.Hkv;
      int64_t pos = valid ? (int64_t)a.positions[row / H] : 0;
      pos = pos < 0 ? 0 : (pos >= a.max_pos ? a.max_pos - 1 : pos);
      const float2* cs = reinterpret_cast<const float2*>(a.cos_sin) + pos * (D / 2);
      // the partner's value enters with sign -1 in the first half and +1 in
      // the second: y = x cos + (-+x') sin, the sign flipped on its fp16 bits
      const uint32_t nsign = c < 2 ? 0x80008000u : 0u;
#pragma unroll
      for (int v = 0; v < V; ++v) {
        uint32_t w[4] = {in[v].x, in[v].y, in[v].z, in[v].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t pw = __shfl_xor_sync(0xffffffffu, w[j], 2) ^ nsign;
          const int f = (8 * V * c + 8 * v + 2 * j) & (D / 2 - 1);
          const float4 t = valid ? __ldg(reinterpret_cast<const float4*>(cs + f)) : make_float4(1.f, 0.f, 1.f, 0.f);
          const float2 x = __half22float2(*reinterpret_cast<const __half2*>(&w[j]));
          const float2 o = __half22float2(*reinterpret_cast<const __half2*>(&pw));
          const float y0 = __fadd_rn(__fmul_rn(x.x, t.x), __fmul_rn(o.x, t.y));
          const float y1 = __fadd_rn(__fmul_rn(x.y, t.z), __fmul_rn(o.y, t.w));
          w[j] = pack_half2_bits(y0, y1);
        }
        in[v] = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }

    float y[V][8];
#pragma unroll
    for (int v = 0; v < V; ++v) {
      // the chunk's words are the A fragment as they are: k = e0 + 2c + 8 e2,
      // row g + 8 e1 (no register moves), so the MMA contracts {e0, e2, c}
      const uint32_t A[4] = {in[v].x, in[v].y, in[v].z, in[v].w};
      float d0[4], d1[4];
      if (kind == 2) {
        mma_16816_f16_f32(d0, A, bi[0][0], bi[0][1]);
        mma_16816_f16_f32(d1, A, bi[1][0], bi[1][1]);
      } else {
        mma_16816_f16_f32(d0, A, bh[0][0], bh[0][1]);
        mma_16816_f16_f32(d1, A, bh[1][0], bh[1][1]);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        y[v][e] = d0[e];
        y[v][e + 4] = d1[e];
      }
    }

    if (kind != 2) {
#pragma unroll
      for (int v = 0; v < V; ++v)
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (!(e & 2)) {  // e1, the bit the MMA leaves
            const float u = y[v][e], w = y[v][e + 2];
            y[v][e] = u + w;
            y[v][e + 2] = u - w;
          }
#pragma unroll
      for (int bit = 1; bit < V; bit <<= 1)
#pragma unroll
        for (int v = 0; v < V; ++v)
          if (!(v & bit)) {
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float u = y[v][e], w = y[v | bit][e];
              y[v][e] = u + w;
              y[v | bit][e] = u - w;
            }
          }
    }

    if (kind == 0) {
      if (valid) {
        uint4* q = reinterpret_cast<uint4*>(reinterpret_cast<__half*>(a.q_out) + row * D) + c * V;
#pragma unroll
        for (int v = 0; v < V; ++v) {
          uint4 o;
          o.x = pack_half2_bits(y[v][0] * a.norm, y[v][1] * a.norm);
          o.y = pack_half2_bits(y[v][2] * a.norm, y[v][3] * a.norm);
          o.z = pack_half2_bits(y[v][4] * a.norm, y[v][5] * a.norm);
          o.w = pack_half2_bits(y[v][6] * a.norm, y[v][7] * a.norm);
          q[v] = o;
        }
      }
      continue;
    }

    // asymmetric Eq. 1 over the row (quad reduction)
    float hi = -FLT_MAX, lo = FLT_MAX;
#pragma unroll
    for (int v = 0; v < V; ++v)
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        hi = fmaxf(hi, y[v][e]);
        lo = fminf(lo, y[v][e]);
      }
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, 1));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, 2));
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, 1));
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, 2));
    const float h2 = a.clip * hi, l2 = a.clip * lo;
    const float inv = h2 > l2 ? 15.f / (h2 - l2) : 0.f;
    const float off = -l2 * inv;
    uint32_t words[V];
#pragma unroll
    for (int v = 0; v < V; ++v) {
      uint32_t r[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        float t = fmaf(y[v][e], inv, off);
        if (CLAMP) t = fminf(fmaxf(t, 0.f), 15.f);
        r[e] = round_bits(t);
      }
      words[v] = pack8_nibbles(r);
    }
    if (valid) {
      const float nrm = kind == 1 ? a.norm : 1.f;
      uint8_t* codes = kind == 1 ? a.k_codes : a.v_codes;
      uint32_t* dst = reinterpret_cast<uint32_t*>(codes + row * (D / 2)) + c * V;
      if (V == 4) {
        *reinterpret_cast<uint4*>(dst) = make_uint4(words[0], words[1], words[2 % V], words[3 % V]);
      } else {
        *reinterpret_cast<uint2*>(dst) = make_uint2(words[0], words[1 % V]);
      }
      if (c == 0) {
        (kind == 1 ? a.k_scale : a.v_scale)[row] = (h2 - l2) / 15.f * nrm;
        (kind == 1 ? a.k_zero : a.v_zero)[row] = l2 * nrm;
      }
    }
  }
}

template <int D, bool CLAMP, bool ROPE>
cudaError_t launch_t(const KVArgs& a, cudaStream_t stream) {
  const int64_t groups = (a.rows_q + 7) / 8 + 2 * ((a.rows_kv + 7) / 8);
  const int sms = device_sm_count();
  int64_t blocks = (groups + kWarps - 1) / kWarps;
  const int64_t cap = (int64_t)sms * 16;  // persistent-style cap: 16 blocks of 8 warps per SM
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  const cudaError_t e = launch_pdl(rotate_quant_kv_kernel<D, CLAMP, ROPE>, dim3((unsigned)blocks),
                                   dim3(kWarps * 32), 0, stream, 1, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rotate_quant_kv(const KVArgs& a, cudaStream_t stream) {
  if (a.rows_q == 0 && a.rows_kv == 0) return cudaSuccess;
  const bool clamp = a.clip < 1.0f;
  if (a.positions) {
    if (a.D == 128) return clamp ? launch_t<128, true, true>(a, stream) : launch_t<128, false, true>(a, stream);
    if (a.D == 64) return clamp ? launch_t<64, true, true>(a, stream) : launch_t<64, false, true>(a, stream);
    return cudaErrorInvalidValue;
  }
  if (a.D == 128) return clamp ? launch_t<128, true, false>(a, stream) : launch_t<128, false, false>(a, stream);
  if (a.D == 64) return clamp ? launch_t<64, true, false>(a, stream) : launch_t<64, false, false>(a, stream);
  return cudaErrorInvalidValue;
}

}  // namespace spinq
