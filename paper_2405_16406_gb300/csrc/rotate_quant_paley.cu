// rotate_quant_paley.cu -- spinq_rotate_quant_act for a rotation with a Paley
// factor: R = (H_s (x) H_P)/sqrt(K), K = n_s * P, n_s in {12, 20, 28},
// P in {128, 256, 512} (Sec. 3.1, R4 of non-power-of-two size), fused with the
// per-token Eq. 1 quantizer.  Element k = i * P + j (i: Paley index).
//
// A persistent CTA walks rows r0, r0 + G, ... with two warp roles that hand
// work to each other through mbarriers (no CTA-wide barrier in the loop):
//
//  * phase-1 warps (W = P/64): the H_s factor on the tensor core plus the
//    first butterflies, written to one of two fp32 transpose buffers;
//  * phase-2 warps (W): the remaining butterflies, the row range, Eq. 1 and
//    the packed codes.
//
// Rows arrive in a ring of NSTG shared-memory stages, one TMA tensor copy per
// row; the last phase-1 warp to finish reading a stage issues the copy of the
// row NSTG iterations ahead into it.  The tensor map views a row as
// (j_lo = j % 64, i, j_hi = j / 64), so a stage holds 128-byte lines
// l = i + n_s j_hi with the 128-byte swizzle: the 16-byte chunk c of line l
// sits at chunk c ^ (l % 8), which keeps ldmatrix free of bank conflicts.
// Phase 1 of row r + 1 runs while phase 2 of row r runs, and the copies of
// the next rows are in flight meanwhile.
//
// Phase 1 (tensor core, raw fp16).  Y^T[i][j] = sum_i' H_s[i'][i] X[i'][j]
// is an m16n8k16 MMA per 16 Paley rows i and 8 consecutive j: A = H_s^T (+-1,
// zero outside NS), B[k = i'][n = j] straight from the staged fp16 row with
// ldmatrix.trans.  Warp w takes j in [64 w, 64 w + 64); lane (g, c) receives
// the pairs (j, j + 1), j = 64 w + 8 nt + 2c, of rows i = 16 mt + 8 h + g, and
// finishes j bit 0 inside each pair and j bits 3..5 (nt) across its registers.
//
// Transpose.  Y goes to an fp32 buffer with row stride P + 8 in which j sits
// at j with bit 2 flipped by bit 5: the 8-byte pair stores here and the
// 16-byte loads of phase 2 are both free of bank conflicts.
//
// Phase 2.  A thread owns, for one i, the 8 consecutive j of bits 0..2 for
// each value of the bits above 5 (8 W values), finishes the butterflies over
// j bits 1, 2 and 6.. on packed pairs and joins the row-wide range reduction
// (one named barrier over the phase-2 warps).  The 8 lanes of a quarter warp
// share i, so each of their 4-byte code words lands next to the others
// (32 contiguous bytes per store instruction and quarter warp).
// Eq. 1 runs on the unnormalised row; alpha and beta carry 1/sqrt(K).
//
// Every wait is bounded in time (suspended in hardware until the phase
// completes, the limit checked every ~20 us).  A warp that gives up raises the
// CTA's abort flag; the others see it in their own waits, the phase-2 warps agree on it
// through a barrier reduction before any global store, and the phase-1 warps
// let the copies in flight land before they exit.
#include <cuda_fp16.h>

#include "launch_util.h"
#include "quant_common.cuh"
#include "spinq_device.cuh"
#include "spinq_internal.h"
#include "tensor_map.h"

namespace spinq {
namespace {

constexpr uint64_t kWaitLimitNs = 2000000000ull;
// limit of the ordinary waits (kWaitLimitNs unless a test lowers it); the
// drain of copies in flight always uses kWaitLimitNs
__device__ uint64_t g_wait_ns = kWaitLimitNs;
constexpr int kSmemBudget = 232448;  // dynamic shared memory a CTA may opt into
constexpr int kPhase2Bar = 1;        // named barrier of the phase-2 warps
constexpr int kPhase1Bar = 2;        // named barrier of the phase-1 warps (exit only)

template <int NS, int LP>
struct PaleyShape {
  static constexpr int P = 1 << LP;
  static constexpr int W = P / 64;                 // warps per compute role
  static constexpr int T = 32 * W;                 // threads per compute role
  static constexpr int THREADS = 2 * T;            // phase-1 warps, then phase-2 warps
  static constexpr int KS = (NS + 15) / 16;        // k16 steps over i'
  static constexpr int MT = (NS + 15) / 16;        // m16 tiles over i
  static constexpr int NSP = NS <= 16 ? 16 : 32;   // phase-2 row slots
  static constexpr int NCOMBO = NSP * 8;           // phase-2 (i slot, j group) combos
  static constexpr int NCB = (NCOMBO + T - 1) / T; // combos per thread
  static constexpr int PS = P + 8;                 // fp32 row stride (8 mod 32: see the layout note)
  static constexpr int ROWB = NS * P * 2;          // staged row (bytes, a multiple of 1024)
  static constexpr int F32B = NS * PS * 4;         // one transpose buffer (bytes)
  static constexpr int MISC = 4 * 8 + 16 + 2 * 2 * W * 4;  // 4 barriers, flag, range scratch
  static constexpr int NSTG_FIT = (kSmemBudget - 1024 - 2 * F32B - MISC) / (ROWB + 16);  // 16: barrier + counters
  static constexpr int NSTG = NSTG_FIT < 4 ? NSTG_FIT : 4;   // staged rows
  static_assert(NSTG >= 2, "two staged rows must fit");
  static_assert(ROWB % 1024 == 0, "stages keep the 1024-byte alignment of the swizzle pattern");
  static_assert(NS % 4 == 0, "phase-2 warps hold 4 whole Paley rows");
  // shared memory layout (bytes from the 1024-aligned base)
  static constexpr int OFF_STAGE = 0;
  static constexpr int OFF_F32 = NSTG * ROWB;
  static constexpr int OFF_BAR = OFF_F32 + 2 * F32B;   // full[NSTG] bfull[2] bempty[2]
  static constexpr int OFF_CNT = OFF_BAR + (NSTG + 4) * 8;   // int readers[NSTG], int issued[NSTG]
  static constexpr int OFF_FLAG = OFF_CNT + NSTG * 8;
  static constexpr int OFF_RED = OFF_FLAG + 16;    // [2 rows][hi W, lo W]
  static constexpr int BYTES = OFF_RED + 2 * 2 * W * 4 + 1024;  // + alignment slack
  static_assert(BYTES <= kSmemBudget, "shared memory");
};

// Transpose-buffer position (floats from the row start) of element j: j with
// bit 2 flipped by bit 5.  With the row stride P + 8 (8 mod 32) this keeps
// both the phase-1 stores (8-byte pairs (j, j + 1) of 4 Paley rows x 4 lane
// columns per half warp) and the phase-2 loads (16-byte quads of the 8 j
// groups of one Paley row per quarter warp) free of bank conflicts.
__host__ __device__ constexpr int tpos(int j) { return j ^ (((j >> 5) & 1) << 2); }

// Paley row slot of phase-2 combo cb: the 8 lanes of a quarter warp share
// it (cb & 7 is the j group), so a warp covers 4 consecutive slots
__device__ __forceinline__ int combo_i(int cb) {
  return ((cb >> 5) << 2) | ((cb >> 3) & 3);
}

// True when every slot of the warp holding combo cb is padding (>= ns): the
// warp then skips the arithmetic of that combo altogether (warp-uniform).
__device__ __forceinline__ bool combo_warp_idle(int cb, int ns) {
  return ((cb >> 5) << 2) >= ns;
}

// Bounded wait for the phase of `bar` with `parity`.  Returns false when the
// abort flag is up or the limit expired (then it raises the flag).
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
  return mbar_wait_suspend(bar, parity, abort_flag, g_wait_ns);
}

// bar.sync over `nthreads` threads whose result is the OR of `pred` over them.
__device__ __forceinline__ bool named_bar_or(int id, int nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, %2, %3, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

// F8 = 0: 4-bit codes (Eq. 1, N = 4); F8 = kFmtInt8Planes / kFmtE4M3: the
// 8-bit quantizers of the 8-bit linears (codes laid out as in
// rotate_quant_8bit.cu), on the same rotation.
template <int NS, int LP, bool SYM, bool CLAMP, bool SG, int F8 = 0>
__global__ void __launch_bounds__(PaleyShape<NS, LP>::THREADS, 1)
    rq_paley_kernel(const __grid_constant__ CUtensorMap tmx, RotQuantArgs a) {
  using S = PaleyShape<NS, LP>;
  constexpr int P = S::P, W = S::W, T = S::T, NSTG = S::NSTG, PS = S::PS;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-aligned base, derived from the shared array itself so that every
  // access below stays in the shared address space
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);
  uint64_t* bfull = full + NSTG;
  uint64_t* bempty = bfull + 2;
  int* readers = reinterpret_cast<int*>(smem + S::OFF_CNT);  // phase-1 warps done with a stage
  int* issued = readers + NSTG;                              // last iteration copied into a stage
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + S::OFF_FLAG);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r0 = blockIdx.x, G = gridDim.x;
  const int niter = a.rows > r0 ? (int)((a.rows - r0 + G - 1) / G) : 0;
  // copy of iteration `it` into its stage (one thread)
  auto issue = [&](int it) {
    const int s = it % NSTG;
    fence_proxy_async_smem();
    mbar_arrive_expect_tx(&full[s], (uint32_t)S::ROWB);
    tma_load_4d(smem + S::OFF_STAGE + s * S::ROWB, &tmx, &full[s], 0, 0, 0, (int32_t)(r0 + (int64_t)it * G));
    issued[s] = it;
  };

  if (tid == 0) {
    for (int s = 0; s < NSTG; ++s) {
      mbar_init(&full[s], 1);
      readers[s] = 0;
      issued[s] = -1;
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bfull[b], W);   // one arrival per warp, after __syncwarp
      mbar_init(&bempty[b], W);
    }
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmx);
  }
  __syncthreads();  // the last CTA-wide barrier: the roles part here
  pdl_wait();
  pdl_trigger();
  if (tid == 0 && !a.debug_stall)   // a test of the time-outs issues no copies
    for (int it = 0; it < NSTG && it < niter; ++it) issue(it);

  if (warp < W) {
    // ---------------- phase 1: H_s on the tensor core, first butterflies
    // Y^T = H_s^T X as m16n8k16 MMAs: M = i (the Paley index, S::MT tiles),
    // N = 8 consecutive j, K = i'.  Warp w takes j in [64 w, 64 w + 64) (8
    // n-tiles); lane (g, c) ends up with the pairs (j, j + 1) for
    // j = 64 w + 8 nt + 2c and i = 16 mt + 8 h + g.
    const int w = warp, g = lane >> 2, c = lane & 3;
    // A fragments of H_s^T: A[i][i'] = H_s[i'][i], zero outside NS (so the
    // padding rows of the B operand, which read a real row, add nothing)
    uint32_t ah[S::MT][S::KS][4];
#pragma unroll
    for (int mt = 0; mt < S::MT; ++mt)
#pragma unroll
      for (int ks = 0; ks < S::KS; ++ks)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int i = 16 * mt + g + 8 * (q & 1), k0 = 16 * ks + 2 * c + 8 * (q >> 1);
          float v[2];
#pragma unroll
          for (int e = 0; e < 2; ++e)
            v[e] = (i < NS && k0 + e < NS) ? (((a.hs.neg[k0 + e] >> i) & 1u) ? -1.f : 1.f) : 0.f;
          ah[mt][ks][q] = pack_half2_bits(v[0], v[1]);
        }
    // ldmatrix.x4.trans row addresses (from the stage base): matrix q of
    // (ks, ntp) holds i' = 16 ks + 8 (q & 1) + 0..7 (rows) at j = 64 w + 8 nt
    // + 0..7 (columns), nt = 2 ntp + (q >> 1); lane 8q + r gives row r.  The
    // stage holds 128-byte lines l = i' + NS j_hi with chunk c at c ^ (l % 8).
    uint32_t loff[S::KS][4];
    {
      const int q = lane >> 3, r = lane & 7;
#pragma unroll
      for (int ks = 0; ks < S::KS; ++ks)
#pragma unroll
        for (int ntp = 0; ntp < 4; ++ntp) {
          int ip = 16 * ks + 8 * (q & 1) + r;
          ip = ip < NS ? ip : NS - 1;
          const int nt = 2 * ntp + (q >> 1), line = ip + NS * w;
          loff[ks][ntp] = (uint32_t)(line * 128 + ((nt ^ (line & 7)) << 4));
        }
    }
    // Random signs (R = S H): element e of register q of the (ks, ntp)
    // fragment is x[i'][j] with i' = 16 ks + 8 (q & 1) + 2c + e and
    // j = 64 w + 8 (2 ntp + (q >> 1)) + g, the same for every row: this lane
    // gathers those sign bits once, bit ((ks 4 + ntp) 4 + q) 2 + e.
    constexpr int NSB = (S::KS * 4 * 4 * 2 + 31) / 32;
    uint32_t sgn[NSB];
#pragma unroll
    for (int t = 0; t < NSB; ++t) sgn[t] = 0;
    if constexpr (SG) {
#pragma unroll
      for (int ks = 0; ks < S::KS; ++ks)
#pragma unroll
        for (int ntp = 0; ntp < 4; ++ntp)
#pragma unroll
          for (int q = 0; q < 4; ++q)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int ip = 16 * ks + 8 * (q & 1) + 2 * c + e;
              const int j = 64 * w + 8 * (2 * ntp + (q >> 1)) + g;
              const int idx = ((ks * 4 + ntp) * 4 + q) * 2 + e;
              if (ip < NS) {
                const int k = ip * P + j;
                sgn[idx >> 5] |= (uint32_t)((a.signs[k >> 3] >> (k & 7)) & 1) << (idx & 31);
              }
            }
    }
    // transpose-buffer float offsets of this lane's pairs: row g, column
    // tpos(64 w + 8 nt + 2c) = 64 w + 8 nt + (2c ^ 4 (nt >> 2))
    const int sb0 = g * PS + 64 * w + 2 * c, sb1 = g * PS + 64 * w + ((2 * c) ^ 4);
    for (int it = 0; it < niter; ++it) {
      const int s = it % NSTG;
      // warp-uniform decision: the MMAs below need every lane
      if (!__all_sync(0xffffffffu, wait_or_abort(&full[s], (uint32_t)(it / NSTG) & 1u, abort_flag))) break;
      const uint32_t stage_addr = smem_u32(smem + S::OFF_STAGE + s * S::ROWB);
      // y[mt][h][nt] = the pair (j, j + 1), j = 64 w + 8 nt + 2c, of row i = 16 mt + 8 h + g
      F2 y[S::MT][2][8];
#pragma unroll
      for (int ks = 0; ks < S::KS; ++ks)
#pragma unroll
        for (int ntp = 0; ntp < 4; ++ntp) {
          uint32_t bf[4];
          ldmatrix_x4_trans(bf, stage_addr + loff[ks][ntp]);
          if constexpr (SG) {   // negate the fp16 elements whose sign bit is set
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const int idx = ((ks * 4 + ntp) * 4 + q) * 2;
              const uint32_t bb = (sgn[idx >> 5] >> (idx & 31)) & 3u;
              bf[q] ^= ((bb & 1u) << 15) | ((bb & 2u) << 30);
            }
          }
#pragma unroll
          for (int mt = 0; mt < S::MT; ++mt)
#pragma unroll
            for (int hn = 0; hn < 2; ++hn) {
              const int nt = 2 * ntp + hn;
              if (ks == 0)
                mma_16816_f16_f32_pairs(y[mt][0][nt], y[mt][1][nt], ah[mt][ks], bf[2 * hn], bf[2 * hn + 1]);
              else
                mma_16816_f16_f32_pairs_acc(y[mt][0][nt], y[mt][1][nt], ah[mt][ks], bf[2 * hn], bf[2 * hn + 1]);
            }
        }
      __syncwarp();
      if (lane == 0) {
        // this warp no longer reads the stage; the last one refills it
        __threadfence_block();
        if (atom_add_shared(&readers[s], 1u) == (uint32_t)(W - 1)) {
          readers[s] = 0;
          if (it + NSTG < niter) issue(it + NSTG);
        }
      }
      // butterflies over j bit 0 (inside each pair) and j bits 3, 4, 5 (nt);
      // row halves wholly past NS hold zeros and are skipped
#pragma unroll
      for (int mt = 0; mt < S::MT; ++mt)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          if (16 * mt + 8 * h >= NS) continue;
#pragma unroll
          for (int nt = 0; nt < 8; ++nt) f2_bfly_inner(y[mt][h][nt]);
#pragma unroll
          for (int bit = 1; bit < 8; bit <<= 1)
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
              if (!(nt & bit)) f2_bfly(y[mt][h][nt], y[mt][h][nt | bit]);
        }
      const int b = it & 1;
      if (it >= 2 &&
          !__all_sync(0xffffffffu, wait_or_abort(&bempty[b], (uint32_t)((it >> 1) - 1) & 1u, abort_flag)))
        break;
      // transpose through shared memory: one 8-byte store per pair
      float* sf = reinterpret_cast<float*>(smem + S::OFF_F32 + b * S::F32B);
#pragma unroll
      for (int mt = 0; mt < S::MT; ++mt)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          if (16 * mt + 8 * h >= NS) continue;
          if (16 * mt + 8 * h + g < NS) {
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
              *reinterpret_cast<unsigned long long*>(sf + (nt < 4 ? sb0 : sb1) + (16 * mt + 8 * h) * PS + 8 * nt) =
                  y[mt][h][nt].u;
          }
        }
      __syncwarp();
      if (lane == 0) mbar_arrive(&bfull[b]);  // release: the warp's stores above are ordered before it
    }
    // every phase-1 warp has stopped issuing; after an abort, let the copies
    // still in flight land before the CTA can exit
    named_bar_sync(kPhase1Bar, T);
    if (*abort_flag && tid == 0 && a.status && atomicCAS(a.status, 0, (int)4 /* SPINQ_ETIMEOUT */) == 0)
      atomicExch(a.status + 1, 20);   // wait site: the Paley rotate+quant kernel
    if (*abort_flag && tid == 0)
      for (int s = 0; s < NSTG; ++s)
        if (issued[s] >= 0) mbar_wait_bounded(&full[s], (uint32_t)(issued[s] / NSTG) & 1u, kWaitLimitNs);
    return;
  }

  // ---------------- phase 2: remaining butterflies, range, Eq. 1, codes
  // Combo cb = (Paley row i, j group jg = j bits 3..5): the thread holds the
  // 8 consecutive j of bits 0..2 for each value wv of the bits above 5, as
  // z[k][wv][q] = the pair (j, j + 1), j = 64 wv + 8 jg + 2q.  The 8 lanes of
  // a quarter warp share i, so a warp holds 4 whole Paley rows.
  const int t2 = tid - T, w2 = warp - W;
  float* red = reinterpret_cast<float*>(smem + S::OFF_RED);
  int ld0[S::NCB], ld1[S::NCB];   // float offsets of the quads hh = 0, 1 at wv = 0
#pragma unroll
  for (int k = 0; k < S::NCB; ++k) {
    const int cb = t2 + T * k, i2 = combo_i(cb), jg = cb & 7;
    ld0[k] = i2 * PS + tpos(8 * jg);
    ld1[k] = i2 * PS + tpos(8 * jg + 4);
  }
  for (int it = 0; it < niter; ++it) {
    const int64_t row = r0 + (int64_t)it * G;
    const int b = it & 1;
    // on a failed wait the buffer is read anyway (in bounds, discarded below)
    const bool ok = wait_or_abort(&bfull[b], (uint32_t)(it >> 1) & 1u, abort_flag);
    const float* sf = reinterpret_cast<const float*>(smem + S::OFF_F32 + b * S::F32B);
    F2 z[S::NCB][W][4];
#pragma unroll
    for (int k = 0; k < S::NCB; ++k) {
      const int cb = t2 + T * k;
      if (cb < S::NCOMBO && !combo_warp_idle(cb, NS)) {
#pragma unroll
        for (int wv = 0; wv < W; ++wv) {
          const ulonglong2 u0 = *reinterpret_cast<const ulonglong2*>(sf + ld0[k] + 64 * wv);
          const ulonglong2 u1 = *reinterpret_cast<const ulonglong2*>(sf + ld1[k] + 64 * wv);
          z[k][wv][0].u = u0.x;
          z[k][wv][1].u = u0.y;
          z[k][wv][2].u = u1.x;
          z[k][wv][3].u = u1.y;
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&bempty[b]);  // the buffer is in registers: phase 1 may refill it
    Range<SYM> rg;
#pragma unroll
    for (int k = 0; k < S::NCB; ++k) {
      const int cb = t2 + T * k;
      if (cb >= S::NCOMBO || combo_warp_idle(cb, NS)) continue;
#pragma unroll
      for (int wv = 0; wv < W; ++wv) {
        f2_bfly(z[k][wv][0], z[k][wv][1]);   // j bit 1
        f2_bfly(z[k][wv][2], z[k][wv][3]);
        f2_bfly(z[k][wv][0], z[k][wv][2]);   // j bit 2
        f2_bfly(z[k][wv][1], z[k][wv][3]);
      }
#pragma unroll
      for (int bit = 1; bit < W; bit <<= 1)   // j bits 6 ..
#pragma unroll
        for (int wv = 0; wv < W; ++wv)
          if (!(wv & bit)) {
#pragma unroll
            for (int q = 0; q < 4; ++q) f2_bfly(z[k][wv][q], z[k][wv | bit][q]);
          }
#pragma unroll
      for (int wv = 0; wv < W; ++wv)
#pragma unroll
        for (int q = 0; q < 4; ++q) rg.add_pair(z[k][wv][q]);
    }
    // row range over the phase-2 warps (scratch alternates between rows, so
    // one barrier per row suffices); the same barrier settles the abort
    // decision for every phase-2 thread before any global store
    rg.warp_reduce();
    float* rd = red + (it & 1) * 2 * W;
    if (lane == 0) {
      rd[w2] = rg.hi;
      rd[W + w2] = rg.lo;
    }
    if (named_bar_or(kPhase2Bar, T, !ok || *abort_flag)) break;
    rg.hi = rd[0];
    rg.lo = rd[W];
#pragma unroll
    for (int i = 1; i < W; ++i) {
      rg.hi = fmaxf(rg.hi, rd[i]);
      if (!SYM) rg.lo = fminf(rg.lo, rd[W + i]);
    }
    if constexpr (F8 == 0) {
      const QParams<SYM> qp(rg, a.clip);
      uint32_t* out = reinterpret_cast<uint32_t*>(a.codes + row * (a.K / 2));
#pragma unroll
      for (int k = 0; k < S::NCB; ++k) {
        const int cb = t2 + T * k;
        if (cb >= S::NCOMBO || combo_warp_idle(cb, NS)) continue;
        // word 8 wv + jg of segment i2 holds the codes of j = 64 wv + 8 jg .. + 7;
        // a quarter warp writes 32 contiguous bytes per wv
        uint32_t* seg = out + combo_i(cb) * (P / 8) + (cb & 7);
#pragma unroll
        for (int wv = 0; wv < W; ++wv) {
          uint32_t rb[8];
#pragma unroll
          for (int q = 0; q < 4; ++q) qp.template code_bits2<CLAMP>(z[k][wv][q], rb[2 * q], rb[2 * q + 1]);
          seg[8 * wv] = pack8_nibbles(rb);
        }
      }
      if (t2 == 0) {
        a.scale[row] = qp.alpha * a.norm;
        if (!SYM) a.zero[row] = qp.beta * a.norm;
      }
    } else {
      static_assert(!CLAMP, "the 8-bit quantizers run here unclipped");
      const Quant8 q8(rg, a.clip, F8 == kFmtE4M3);
      uint8_t* out = a.codes + row * (F8 == kFmtInt8Planes ? 2 * a.K : a.K);
#pragma unroll
      for (int k = 0; k < S::NCB; ++k) {
        const int cb = t2 + T * k;
        if (cb >= S::NCOMBO || combo_warp_idle(cb, NS)) continue;
        // the 8 bytes of j = 64 wv + 8 jg .. + 7 of segment i2
        uint8_t* seg = out + combo_i(cb) * P + 8 * (cb & 7);
#pragma unroll
        for (int wv = 0; wv < W; ++wv) {
          uint2 hi, lo;
          q8.template codes8<F8>(z[k][wv], hi, lo);
          *reinterpret_cast<uint2*>(seg + 64 * wv) = hi;
          if (F8 == kFmtInt8Planes) *reinterpret_cast<uint2*>(seg + a.K + 64 * wv) = lo;
        }
      }
      if (t2 == 0) {
        a.scale[row] = q8.alpha * a.norm;
        if (!SYM && F8 == kFmtInt8Planes) a.zero[row] = q8.beta * a.norm;
      }
    }
  }
}

template <int NS, int LP, bool SYM, bool CLAMP, bool SG, int F8 = 0>
cudaError_t launch_paley(const RotQuantArgs& a, cudaStream_t stream) {
  using S = PaleyShape<NS, LP>;
  // rows as (j_lo, i, j_hi, row): one copy lands a row as 128-byte swizzled lines i + NS j_hi
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return cudaErrorNotSupported;
  CUtensorMap tmx;
  const cuuint64_t gdim[4] = {64, (cuuint64_t)NS, (cuuint64_t)(S::P / 64), (cuuint64_t)a.rows};
  const cuuint64_t gstride[3] = {(cuuint64_t)(S::P * 2), 128, (cuuint64_t)(a.ldx * 2)};
  const cuuint32_t box[4] = {64, (cuuint32_t)NS, (cuuint32_t)(S::P / 64), 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  if (enc(&tmx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void*>(a.x), gdim, gstride, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorNotSupported;
  auto kern = rq_paley_kernel<NS, LP, SYM, CLAMP, SG, F8>;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, S::THREADS, S::BYTES, &per_sm);
  if (e != cudaSuccess) return e;
  const int64_t cap = (int64_t)device_sm_count() * per_sm;
  const int64_t grid = a.rows < cap ? a.rows : cap;
  RotQuantArgs la = a;
  la.debug_stall = take_debug_stall() ? 1 : 0;
  e = launch_pdl(kern, dim3((unsigned)grid), dim3(S::THREADS), S::BYTES, stream, 1, tmx, la);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int NS, bool SYM, bool CLAMP, bool SG>
cudaError_t launch_ns(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  *handled = true;
  switch (a.n_pow2) {
    case 128: return launch_paley<NS, 7, SYM, CLAMP, SG>(a, stream);
    case 256: return launch_paley<NS, 8, SYM, CLAMP, SG>(a, stream);
    case 512: return launch_paley<NS, 9, SYM, CLAMP, SG>(a, stream);
  }
  *handled = false;
  return cudaSuccess;
}

// H_s (x) H_P with P = 2 Q equals (H_s (x) H_2) (x) H_Q on the same element
// order (k = i P + j = (2 i + j_top) Q + j_low, and the Sylvester H_P is H_2
// on the top bit of j times H_Q on the rest), so a factor of 2 can move from
// the butterflies to the tensor core.  H_12 (x) H_256 runs as H_24 (x) H_128:
// the 24 rows of H_24 fill the MMA's three n8 tiles exactly, where the 12
// rows of H_12 leave a quarter of two tiles empty.
SmallHadamard kron_h2(const SmallHadamard& h) {
  SmallHadamard r;
  r.n = 2 * h.n;
  for (int p = 0; p < h.n; ++p)
    for (int a2 = 0; a2 < 2; ++a2) {
      uint32_t bits = 0;
      for (int q = 0; q < h.n; ++q)
        for (int b2 = 0; b2 < 2; ++b2)
          if ((((h.neg[p] >> q) & 1u) ^ (uint32_t)(a2 & b2)) != 0) bits |= 1u << (2 * q + b2);
      r.neg[2 * p + a2] = bits;
    }
  return r;
}

template <bool SYM, bool CLAMP, bool SG>
cudaError_t launch_sc(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  if (a.n_small == 12 && a.n_pow2 == 256) {
    RotQuantArgs b = a;
    b.hs = kron_h2(a.hs);
    b.n_small = 24;
    b.n_pow2 = 128;
    *handled = true;
    return launch_paley<24, 7, SYM, CLAMP, SG>(b, stream);
  }
  switch (a.n_small) {
    case 12: return launch_ns<12, SYM, CLAMP, SG>(a, stream, handled);
    case 20: return launch_ns<20, SYM, CLAMP, SG>(a, stream, handled);
    case 28: return launch_ns<28, SYM, CLAMP, SG>(a, stream, handled);
  }
  *handled = false;
  return cudaSuccess;
}

// The 8-bit quantizers on a Paley rotation (unclipped forms, no random signs).
template <int F8, bool SYM>
cudaError_t launch8_sc(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  *handled = true;
  if (a.n_small == 12 && a.n_pow2 == 256) {
    RotQuantArgs b = a;
    b.hs = kron_h2(a.hs);
    b.n_small = 24;
    b.n_pow2 = 128;
    return launch_paley<24, 7, SYM, false, false, F8>(b, stream);
  }
#define SPINQ_P8(NS_)                                                      \
  switch (a.n_pow2) {                                                      \
    case 128: return launch_paley<NS_, 7, SYM, false, false, F8>(a, stream); \
    case 256: return launch_paley<NS_, 8, SYM, false, false, F8>(a, stream); \
    case 512: return launch_paley<NS_, 9, SYM, false, false, F8>(a, stream); \
  }                                                                        \
  break;
  switch (a.n_small) {
    case 12: SPINQ_P8(12)
    case 20: SPINQ_P8(20)
    case 28: SPINQ_P8(28)
  }
#undef SPINQ_P8
  *handled = false;
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_rotate_quant_8bit_paley(const Rq8Args& a, cudaStream_t stream, bool* handled) {
  *handled = false;
  if (a.rows == 0 || a.n_small <= 1 || a.clip < 1.0f) return cudaSuccess;
  if (a.format != kFmtE4M3 && a.format != kFmtInt8Planes) return cudaSuccess;
  if (a.format == kFmtE4M3 && !a.symmetric) return cudaSuccess;
  if ((a.ldx * 2) % 16 != 0) return cudaSuccess;
  RotQuantArgs b{};
  b.x = a.x;
  b.rows = a.rows;
  b.K = a.K;
  b.ldx = a.ldx;
  b.n_small = a.n_small;
  b.n_pow2 = a.n_pow2;
  b.hs = a.hs;
  b.symmetric = a.symmetric;
  b.clip = a.clip;
  b.norm = a.norm;
  b.codes = a.codes;
  b.scale = a.scale;
  b.zero = a.zero;
  b.status = device_status_word();
  {
    const cudaError_t e = launch_rotate_quant_8bit_tc(b, a.format, stream, handled);
    if (*handled || e != cudaSuccess) return e;
  }
  if (a.format == kFmtE4M3) return launch8_sc<kFmtE4M3, true>(b, stream, handled);
  return a.symmetric ? launch8_sc<kFmtInt8Planes, true>(b, stream, handled)
                     : launch8_sc<kFmtInt8Planes, false>(b, stream, handled);
}

cudaError_t set_wait_limit_paley(uint64_t ns) {
  const cudaError_t e = cudaMemcpyToSymbol(g_wait_ns, &ns, sizeof(ns));
  return e != cudaSuccess ? e : set_wait_limit_rq_tc(ns);
}

cudaError_t launch_rotate_quant_act_paley(const RotQuantArgs& a0, cudaStream_t stream, bool* handled) {
  RotQuantArgs a = a0;
  a.status = device_status_word();
  a.debug_stall = 0;
  *handled = false;
  if (a.rows == 0 || a.rowsum || a.n_small <= 1) return cudaSuccess;
  if ((a.ldx * 2) % 16 != 0) return cudaSuccess;
  {
    const cudaError_t e = launch_rotate_quant_act_tc(a, stream, handled);
    if (*handled || e != cudaSuccess) return e;
  }
  const bool clamp = a.clip < 1.0f;
  if (a.signs) {   // random signs: the unclipped forms (clipped ones take the generic kernel)
    if (clamp) return cudaSuccess;
    return a.symmetric ? launch_sc<true, false, true>(a, stream, handled)
                       : launch_sc<false, false, true>(a, stream, handled);
  }
  if (a.symmetric)
    return clamp ? launch_sc<true, true, false>(a, stream, handled) : launch_sc<true, false, false>(a, stream, handled);
  return clamp ? launch_sc<false, true, false>(a, stream, handled) : launch_sc<false, false, false>(a, stream, handled);
}

}  // namespace spinq
