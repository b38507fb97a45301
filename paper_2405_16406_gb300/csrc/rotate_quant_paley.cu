// rotate_quant_paley.cu -- spinq_rotate_quant_act for a rotation with a Paley
// factor: R = (H_s (x) H_P)/sqrt(K), K = n_s * P, n_s in {12, 20, 28},
// P in {128, 256, 512} (Sec. 3.1, R4 of non-power-of-two size), fused with the
// per-token Eq. 1 quantizer.  Element k = i * P + j (i: Paley index).
//
// One CTA (W = P/64 warps) owns one row at a time; rows stream in through
// shared memory with TMA bulk copies, NST rows ahead (one copy per Paley
// segment i, each segment padded by 16 bytes so that ldmatrix is free of bank
// conflicts).
//
// Phase 1 (tensor core, raw fp16).  Y[i][j] = sum_i' X[i'][j] H_s[i'][i] is an
// m16n8k16 MMA per 16 consecutive j: A[m = j][k = i'] comes straight from the
// staged fp16 rows with ldmatrix.trans, B = H_s (+-1, zero-padded to 16/32).
// Lane (g, c) of warp w receives j = 16 (w + W v) + 8 h + g for h in {0, 1},
// v in 0..3 and i = 2c + {0, 1} + 8 nt.  Radix-2 butterflies inside the lane
// cover the j bits of h and v.
//
// Transpose.  Y goes to a padded fp32 buffer (row stride P + 4: conflict-free
// for both the scalar stores here and the 16-byte loads of phase 2).
//
// Phase 2.  A thread owns, for one i, the 8 consecutive j of bits 0..2 for
// each value of the warp bits (8 W values), finishes the butterflies over
// those bits, joins the row-wide range reduction and stores 32-bit words of 8
// packed codes.  Eq. 1 runs on the unnormalised row; alpha and beta carry
// 1/sqrt(K).
#include <cuda_fp16.h>

#include "launch_util.h"
#include "quant_common.cuh"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {
namespace {

constexpr uint64_t kRowWaitLimitNs = 2000000000ull;

template <int NS, int LP>
struct PaleyShape {
  static constexpr int P = 1 << LP;
  static constexpr int W = P / 64;                 // warps
  static constexpr int T = 32 * W;
  static constexpr int KS = (NS + 15) / 16;        // k16 steps over i'
  static constexpr int NT = (NS + 7) / 8;          // n8 tiles over i
  static constexpr int NSP = NS <= 16 ? 16 : 32;   // phase-2 row slots
  static constexpr int NCOMBO = NSP * 8;          // phase-2 (i slot, j group) combos
  static constexpr int NCB = (NCOMBO + T - 1) / T; // combos per thread
  static constexpr int PS = P + 4;                 // fp32 row stride
  static constexpr int SEGB = 2 * P + 16;          // staged fp16 segment stride (bytes)
  static constexpr int ROWB = NS * SEGB;           // staged row (bytes)
  // rows in flight: one staged row for the large shapes so that two CTAs fit
  // on an SM; the next row is requested as soon as phase 1 has consumed the
  // current one, so its copy overlaps phase 2
  static constexpr int NST = NS * P >= 8192 ? 1 : 2;
  // shared memory layout (bytes)
  static constexpr int OFF_STAGE = 0;
  static constexpr int OFF_ZERO = NST * ROWB;
  static constexpr int OFF_F32 = OFF_ZERO + 16;
  static constexpr int OFF_BAR = OFF_F32 + NS * PS * 4;
  static constexpr int OFF_RED = OFF_BAR + NST * 8;
  static constexpr int BYTES = OFF_RED + 2 * W * 4 + 16;
};

template <int NS, int LP, bool SYM, bool CLAMP>
__global__ void __launch_bounds__(32 * ((1 << LP) / 64), 16 / ((1 << LP) / 64)) rq_paley_kernel(RotQuantArgs a) {
  using S = PaleyShape<NS, LP>;
  constexpr int P = S::P, W = S::W;
  extern __shared__ __align__(128) uint8_t smem[];
  float* sf = reinterpret_cast<float*>(smem + S::OFF_F32);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);
  float* red = reinterpret_cast<float*>(smem + S::OFF_RED);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + S::OFF_RED + 2 * W * 4);
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5, g = lane >> 2, c = lane & 3;
  const uint8_t* __restrict__ x = reinterpret_cast<const uint8_t*>(a.x);
  const int64_t row_bytes = a.ldx * 2;

  // B fragments of H_s (k = i', n = i), zero outside NS
  uint32_t bs[S::KS][S::NT][2];
#pragma unroll
  for (int ks = 0; ks < S::KS; ++ks)
#pragma unroll
    for (int nt = 0; nt < S::NT; ++nt) {
      const int n = g + 8 * nt;
#pragma unroll
      for (int hb = 0; hb < 2; ++hb) {
        const int k0 = 2 * c + 8 * hb + 16 * ks;
        float v[2];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int k = k0 + e;
          v[e] = (k < NS && n < NS) ? (((a.hs.neg[k] >> n) & 1u) ? -1.f : 1.f) : 0.f;
        }
        bs[ks][nt][hb] = pack_half2_bits(v[0], v[1]);
      }
    }

  if (tid == 0) {
    for (int s = 0; s < S::NST; ++s) mbar_init(&full[s], 1);
    *reinterpret_cast<uint4*>(smem + S::OFF_ZERO) = make_uint4(0, 0, 0, 0);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  const int64_t r0 = blockIdx.x, G = gridDim.x;
  auto issue = [&](int64_t row, int stage) {
    uint8_t* dst = smem + S::OFF_STAGE + stage * S::ROWB;
    fence_proxy_async_smem();  // earlier ldmatrix reads of this stage precede the copy
    mbar_arrive_expect_tx(&full[stage], (uint32_t)(NS * P * 2));
    const uint8_t* src = x + row * row_bytes;
#pragma unroll 1
    for (int i = 0; i < NS; ++i) bulk_load(dst + i * S::SEGB, src + i * P * 2, P * 2, &full[stage]);
  };
  int issued = 0;  // iterations whose row copy has been issued (thread 0 only)
  if (tid == 0) {
    for (int s = 0; s < S::NST; ++s)
      if (r0 + s * G < a.rows) {
        issue(r0 + s * G, s);
        issued = s + 1;
      }
  }

  // phase-2 identity
  const uint32_t zero_addr = smem_u32(smem + S::OFF_ZERO);
  int it = 0;
  for (int64_t row = r0; row < a.rows; row += G, ++it) {
    const int st = it % S::NST;
    // wait for this row (bounded)
    {
      bool ok = mbar_try_wait(&full[st], (it / S::NST) & 1);
      if (!ok) {
        const uint64_t t0 = globaltimer_ns();
        while (!(ok = mbar_try_wait(&full[st], (it / S::NST) & 1))) {
          if (*abort_flag || globaltimer_ns() - t0 > kRowWaitLimitNs) break;
        }
      }
      if (!ok) *abort_flag = 1;
    }
    __syncthreads();
    if (*abort_flag) break;
    const uint32_t stage_addr = smem_u32(smem + S::OFF_STAGE + st * S::ROWB);

    // ---------------- phase 1: H_s on the tensor core
    float y[S::NT][2][2][4];  // [nt][hi][h][v]
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int jb = 16 * (w + W * v);
      float d[S::NT][4];
#pragma unroll
      for (int nt = 0; nt < S::NT; ++nt) d[nt][0] = d[nt][1] = d[nt][2] = d[nt][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < S::KS; ++ks) {
        const int q = lane >> 3, r = lane & 7;
        const int ip = r + 8 * (q >> 1) + 16 * ks;
        const int js = jb + 8 * (q & 1);
        const uint32_t addr = ip < NS ? stage_addr + (uint32_t)(ip * S::SEGB + js * 2) : zero_addr;
        uint32_t af[4];
        ldmatrix_x4_trans(af, addr);
#pragma unroll
        for (int nt = 0; nt < S::NT; ++nt) mma_16816_f16_f32_acc(d[nt], af, bs[ks][nt][0], bs[ks][nt][1]);
      }
#pragma unroll
      for (int nt = 0; nt < S::NT; ++nt) {
        y[nt][0][0][v] = d[nt][0];
        y[nt][1][0][v] = d[nt][1];
        y[nt][0][1][v] = d[nt][2];
        y[nt][1][1][v] = d[nt][3];
      }
    }
    // butterflies over h (j bit 3) and v (the two highest j bits)
#pragma unroll
    for (int nt = 0; nt < S::NT; ++nt)
#pragma unroll
      for (int hi = 0; hi < 2; ++hi) {
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const float p0 = y[nt][hi][0][v], p1 = y[nt][hi][1][v];
          y[nt][hi][0][v] = p0 + p1;
          y[nt][hi][1][v] = p0 - p1;
        }
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int bit = 1; bit < 4; bit <<= 1)
#pragma unroll
            for (int v = 0; v < 4; ++v)
              if (!(v & bit)) {
                const float p0 = y[nt][hi][h][v], p1 = y[nt][hi][h][v | bit];
                y[nt][hi][h][v] = p0 + p1;
                y[nt][hi][h][v | bit] = p0 - p1;
              }
      }
    // transpose through shared memory
#pragma unroll
    for (int nt = 0; nt < S::NT; ++nt)
#pragma unroll
      for (int hi = 0; hi < 2; ++hi) {
        const int i = 2 * c + 8 * nt + hi;
        if (i < NS) {
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int v = 0; v < 4; ++v) sf[i * S::PS + 16 * (w + W * v) + 8 * h + g] = y[nt][hi][h][v];
        }
      }
    __syncthreads();
    // the staged row is consumed: request the row NST iterations ahead into it
    if (tid == 0) {
      const int64_t nxt = row + (int64_t)S::NST * G;
      if (nxt < a.rows) {
        issue(nxt, st);
        issued = it + S::NST + 1;
      }
    }

    // ---------------- phase 2
    float z[S::NCB][W][8];
    Range<SYM> rg;
#pragma unroll
    for (int k = 0; k < S::NCB; ++k) {
      const int cb = tid + S::T * k;
      const int i2 = cb % S::NSP, jc = cb / S::NSP;
      const int jf = 8 * (jc & 1) + 16 * W * (jc >> 1);
      const bool act = cb < S::NCOMBO && i2 < NS;
      if (act) {
#pragma unroll
        for (int wv = 0; wv < W; ++wv) {
          const float4 u0 = *reinterpret_cast<const float4*>(sf + i2 * S::PS + jf + 16 * wv);
          const float4 u1 = *reinterpret_cast<const float4*>(sf + i2 * S::PS + jf + 16 * wv + 4);
          z[k][wv][0] = u0.x; z[k][wv][1] = u0.y; z[k][wv][2] = u0.z; z[k][wv][3] = u0.w;
          z[k][wv][4] = u1.x; z[k][wv][5] = u1.y; z[k][wv][6] = u1.z; z[k][wv][7] = u1.w;
        }
      } else {
#pragma unroll
        for (int wv = 0; wv < W; ++wv)
#pragma unroll
          for (int e = 0; e < 8; ++e) z[k][wv][e] = 0.f;
      }
#pragma unroll
      for (int bit = 1; bit < 8; bit <<= 1)
#pragma unroll
        for (int wv = 0; wv < W; ++wv)
#pragma unroll
          for (int e = 0; e < 8; ++e)
            if (!(e & bit)) {
              const float p0 = z[k][wv][e], p1 = z[k][wv][e | bit];
              z[k][wv][e] = p0 + p1;
              z[k][wv][e | bit] = p0 - p1;
            }
#pragma unroll
      for (int bit = 1; bit < W; bit <<= 1)
#pragma unroll
        for (int wv = 0; wv < W; ++wv)
          if (!(wv & bit)) {
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float p0 = z[k][wv][e], p1 = z[k][wv | bit][e];
              z[k][wv][e] = p0 + p1;
              z[k][wv | bit][e] = p0 - p1;
            }
          }
      if (act)
#pragma unroll
        for (int wv = 0; wv < W; ++wv)
#pragma unroll
          for (int e = 0; e < 8; ++e) rg.add(z[k][wv][e]);
    }
    block_range<SYM, W>(rg, red);
    const QParams<SYM> qp(rg, a.clip);
    uint8_t* out = a.codes + row * (a.K / 2);
#pragma unroll
    for (int k = 0; k < S::NCB; ++k) {
      const int cb = tid + S::T * k;
      const int i2 = cb % S::NSP, jc = cb / S::NSP;
      const int jf = 8 * (jc & 1) + 16 * W * (jc >> 1);
      if (cb < S::NCOMBO && i2 < NS) {
#pragma unroll
        for (int wv = 0; wv < W; ++wv) {
          uint32_t rb[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) rb[e] = qp.template code_bits<CLAMP>(z[k][wv][e]);
          *reinterpret_cast<uint32_t*>(out + (i2 * P + jf + 16 * wv) / 2) = pack8_nibbles(rb);
        }
      }
    }
    if (tid == 0) {
      a.scale[row] = qp.alpha * a.norm;
      if (!SYM) a.zero[row] = qp.beta * a.norm;
    }
    __syncthreads();  // stage, fp32 buffer and `red` are reused by the next row
  }
  if (*abort_flag && tid == 0) {
    // let the copies still in flight (iterations it .. issued-1) land first
    for (int j = it; j < issued; ++j) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&full[j % S::NST], (j / S::NST) & 1) && globaltimer_ns() - t0 < kRowWaitLimitNs) {
      }
    }
  }
}

template <int NS, int LP, bool SYM, bool CLAMP>
cudaError_t launch_paley(const RotQuantArgs& a, cudaStream_t stream) {
  using S = PaleyShape<NS, LP>;
  auto kern = rq_paley_kernel<NS, LP, SYM, CLAMP>;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, S::T, S::BYTES, &per_sm);
  if (e != cudaSuccess) return e;
  const int64_t cap = (int64_t)device_sm_count() * per_sm;
  const int64_t grid = a.rows < cap ? a.rows : cap;
  kern<<<(unsigned)grid, S::T, S::BYTES, stream>>>(a);
  return cudaGetLastError();
}

template <int NS, bool SYM, bool CLAMP>
cudaError_t launch_ns(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  *handled = true;
  switch (a.n_pow2) {
    case 128: return launch_paley<NS, 7, SYM, CLAMP>(a, stream);
    case 256: return launch_paley<NS, 8, SYM, CLAMP>(a, stream);
    case 512: return launch_paley<NS, 9, SYM, CLAMP>(a, stream);
  }
  *handled = false;
  return cudaSuccess;
}

template <bool SYM, bool CLAMP>
cudaError_t launch_sc(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  switch (a.n_small) {
    case 12: return launch_ns<12, SYM, CLAMP>(a, stream, handled);
    case 20: return launch_ns<20, SYM, CLAMP>(a, stream, handled);
    case 28: return launch_ns<28, SYM, CLAMP>(a, stream, handled);
  }
  *handled = false;
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_rotate_quant_act_paley(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  *handled = false;
  if (a.rows == 0 || a.rowsum || a.n_small <= 1) return cudaSuccess;
  if ((a.ldx * 2) % 16 != 0) return cudaSuccess;
  const bool clamp = a.clip < 1.0f;
  if (a.symmetric) return clamp ? launch_sc<true, true>(a, stream, handled) : launch_sc<true, false>(a, stream, handled);
  return clamp ? launch_sc<false, true>(a, stream, handled) : launch_sc<false, false>(a, stream, handled);
}

}  // namespace spinq
