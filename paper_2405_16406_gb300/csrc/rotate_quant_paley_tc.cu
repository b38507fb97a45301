// rotate_quant_paley_tc.cu -- spinq_rotate_quant_act for plain rotations R =
// (H_s (x) H_P) / sqrt(K) (Sec. 3.1, R4; H_s a Paley factor, or n_s = 1 for a
// Sylvester rotation of P points), fused with the per-token Eq. 1 4-bit
// quantizer, on the 5th-generation tensor core.  Element k = i P + j.
//
// The Sylvester H_P is H_(P/128) on the top bits of j (jh = j / 128) times
// H_128 on the rest (jl = j % 128), so with the row written as the matrix
// X[a][jl], a = i (P / 128) + jh (F = n_s P / 128 rows of 128 columns),
//
//   Y[a][jl] = sum_jl' ( sum_a' T[a][a'] X[a'][jl'] ) H_128[jl'][jl],
//   T[a][a'] = H_s[i'][i] H_(P/128)[jh'][jh].
//
// The inner sum is one tcgen05 MMA for RPS = 128 / F rows at once (T =
// I_RPS (x) T on the MMA's M = 128 rows, the first MR = RPS F of them
// non-zero; N = 128 columns jl; K = MR in K steps of 16) on the raw fp16
// input: entries +-1, so the products are exact and the sums are fp32 sums of
// fp16 values, as for the H_s stage of the mma.sync kernel.  The accumulator
// lands in tensor memory with (r, a) on lane F r + a and the 128 columns jl
// across 128 columns, so one thread reads the whole 128-point vector of its
// block: the 7 stages of H_128 are butterflies inside the thread (no
// shared-memory transpose), then the row range (over the row's lanes),
// Eq. 1 and 64 contiguous bytes of codes per thread (the codes of elements
// 128 a .. 128 a + 127 of row r); or, for the 8-bit linears, the per-row FP8
// quantizer and 128 bytes of E4M3 codes per thread.
//
// Warp roles (one CTA per SM, rows r0, r0 + G, ...):
//  * warp 0: one thread copies each MMA's RPS rows into a ring of NSTG
//    stages with one TMA tensor copy (the tensor map views them as (jl % 64,
//    a, r, jl / 64): two 64-column atoms of MR 128-byte rows, 128-byte
//    swizzle, the canonical MN-major layout of the MMA's B operand);
//  * warp 1: one thread issues the MMAs of a stage into one of NBUF tensor
//    memory accumulators (128 columns each) and commits them to the stage's
//    `free` barrier and the accumulator's `full` barrier;
//  * NGRP groups of 4 warps (one per tensor-memory lane quadrant) take the
//    accumulators in turn: read one (releasing it for the next MMA), the
//    butterflies, the ranges (per-quadrant partials, or shared-memory
//    atomics where rows share warps, and a named barrier per group), Eq. 1
//    and the codes.
// T is written once per CTA into shared memory (K-major, 128-byte swizzle),
// from the Paley sign words staged in shared memory, after the copy thread
// has issued the first pass over the ring.
//
// Every wait is bounded in time; a wait that gives up raises the CTA's abort
// flag, the others see it at their next wait, the MMA thread drains its MMAs
// and the copy thread lets its copies land before tensor memory is released.
// The quantizer groups poll (a suspended wait woke up late); the copy thread,
// which runs rows ahead, sleeps between polls and leaves the issue slots to
// the groups on its sub-partition, and so does the MMA thread where an MMA
// covers two rows.
#include <cuda_fp16.h>

#include <climits>

#include "../../include/spinq.h"
#include "launch_util.h"
#include "quant_common.cuh"
#include "spinq_device.cuh"
#include "spinq_internal.h"
#include "tensor_map.h"

namespace spinq {
namespace {

constexpr uint64_t kTcWaitLimitNs = 2000000000ull;
// limit of the ordinary waits (kTcWaitLimitNs unless a test lowers it); the
// drains of copies and MMAs in flight always use kTcWaitLimitNs
__device__ uint64_t g_tc_wait_ns = kTcWaitLimitNs;
constexpr int kTcSmemBudget = 232448;
constexpr int kTcSite = 21;   // wait site recorded on a time-out

// A row of K = n_s P elements (n_s = 1 for a Sylvester rotation) is the
// matrix X[a][jl] of F = n_s P / 128 rows a = i (P / 128) + jh (i the Paley
// index, jh = j / 128) and 128 columns jl = j % 128; R = H_s (x) H_P with
// H_P = H_(P/128) (x) H_128, so the factor H_f = H_s (x) H_(P/128) acts on a and
// H_128 on jl.  RPS rows share one MMA: T = I_RPS (x) H_f^T, MR = RPS F lanes.
template <int F, int RPS>
struct RqTc {
  static constexpr int MR = F * RPS;              // live lanes: rows (r, a) of the MMA
  static constexpr int KS = MR / 16;              // MMA K steps
  static constexpr int ATOMB = MR * 128;          // one 64-column atom of a stage
  static constexpr int ROWB = 2 * ATOMB;          // a stage (RPS rows of K fp16)
  static_assert(MR <= 128 && MR % 16 == 0 && ATOMB % 1024 == 0, "MMA shape and the swizzle period");
  static constexpr int NGRP = 2;                  // row groups of GW warps
  static constexpr int GW = 4;                    // one warp per tensor-memory lane quadrant
  static constexpr int NBUF = 4;                  // tensor-memory accumulators (128 columns each)
  static constexpr int TMEM_COLS = NBUF * 128 <= 256 ? 256 : 512;   // allocated (a power of two)
  static constexpr int THREADS = 32 * (2 + GW * NGRP);
  static constexpr int TB = 2 * 128 * 128;        // T: two 64-column K atoms of 128 rows (fp16)
  static constexpr int MISC = 1024;               // barriers, flags, range slots
  static constexpr int NSTG_FIT = (kTcSmemBudget - 1024 - TB - MISC) / ROWB;
  static constexpr int NSTG = NSTG_FIT < 6 ? NSTG_FIT : 6;   // staged MMA inputs
  static_assert(NSTG >= 2, "two stages must fit");
  static_assert(NGRP <= NBUF && NBUF % NGRP == 0, "each accumulator belongs to one group");
  // shared memory (bytes from the 1024-aligned base)
  static constexpr int OFF_T = 0;
  static constexpr int OFF_STG = TB;
  static constexpr int OFF_BAR = OFF_STG + NSTG * ROWB;   // full[NSTG] sfree[NSTG] dfull[NBUF] dfree[NBUF] drain
  static constexpr int OFF_MISC = OFF_BAR + (2 * NSTG + 2 * NBUF + 1) * 8;   // tmem slot, abort flag, issued[NSTG]
  // each warp's lanes belong to one row: per-quadrant partials; else atomics
  static constexpr bool QUADS = RPS == 1 || F % 32 == 0;
  static constexpr int OFF_RED = OFF_MISC + 8 + 4 * NSTG;   // QUADS: float [NGRP][2][hi GW, lo GW]; else int [NGRP][3][RPS][hi, lo]
  static constexpr int REDB = QUADS ? NGRP * 2 * 2 * GW * 4 : NGRP * 3 * RPS * 2 * 4;
  static constexpr int OFF_NEG = OFF_RED + REDB;   // the Paley sign words hs.neg[32]
  static constexpr int BYTES = OFF_NEG + 128 + 1024;
  static_assert(OFF_NEG + 128 <= OFF_BAR + MISC, "misc area");
  static_assert(BYTES <= kTcSmemBudget, "shared memory");
};

// Order-preserving map between float bit patterns and signed ints (an
// involution), so that atomicMax / atomicMin on ints give the float max / min.
__device__ __forceinline__ int f2ord(float f) {
  const int b = __float_as_int(f);
  return b >= 0 ? b : b ^ 0x7FFFFFFF;
}
__device__ __forceinline__ float ord2f(int b) { return __int_as_float(b >= 0 ? b : b ^ 0x7FFFFFFF); }

// byte offset of byte b of row r in a block of 128-byte rows with the 128-byte swizzle
__device__ __forceinline__ uint32_t sw128(uint32_t r, uint32_t b) {
  return r * 128 + ((((b >> 4) ^ (r & 7)) << 4) | (b & 15));
}

// Non-blocking probe of the phase with `parity` (never suspends the thread).
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait that polls: a suspended wait woke up to ~0.5 us after the
// phase completed (measured on the row pipeline of this kernel: 40.8 against
// 36.7 us for H_8192 on 8192 rows), which the quantizer groups pay once per
// row.  The abort flag and the time limit are checked every 256 polls.
__device__ __forceinline__ bool tc_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_test_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t k = 1;; ++k) {
    if (mbar_test_wait(bar, parity)) return true;
    if ((k & 255u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > g_tc_wait_ns) {
        *abort_flag = 1;
        return false;
      }
    }
  }
}

// bar.sync over `nthreads` threads whose result is the OR of `pred` over them.
__device__ __forceinline__ bool tc_bar_or(int id, int nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, %2, %3, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

// F8 = 0: the 4-bit codes (Eq. 1); F8 = kFmtE4M3: the per-row FP8 quantizer
// of the 8-bit linears (unclipped), codes laid out as in rotate_quant_8bit.cu
// (the int8-planes epilogue is written for F8 = kFmtInt8Planes too, but it
// is not instantiated: its two roundings and two conversions per element on
// the quantizer groups made H_28 (x) H_512 slower here, 43.3 against 34.4 us
// on the Paley kernel, while E4M3 went 26.0 -> 19.0 us).
template <int F, int RPS, bool SYM, bool CLAMP, int F8 = 0>
__global__ void __launch_bounds__(RqTc<F, RPS>::THREADS, 1)
    rq_tc_kernel(const __grid_constant__ CUtensorMap tmx, RotQuantArgs a) {
  using S = RqTc<F, RPS>;
  constexpr int MR = S::MR, KS = S::KS, NSTG = S::NSTG, NBUF = S::NBUF, NGRP = S::NGRP;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-aligned base, derived from the shared array itself
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);   // row landed in stage s
  uint64_t* sfree = full + NSTG;                                       // stage s read by its MMAs
  uint64_t* dfull = sfree + NSTG;                                      // accumulator b written
  uint64_t* dfree = dfull + NBUF;                                      // accumulator b read out (4 warps)
  uint64_t* drain = dfree + NBUF;                                      // every MMA issued has completed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + S::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + S::OFF_MISC + 4);
  int* issued = reinterpret_cast<int*>(smem + S::OFF_MISC + 8);      // last iteration copied into stage s
  int* rslot = reinterpret_cast<int*>(smem + S::OFF_RED);            // [group][row % 3][r][hi, lo]
  uint32_t* neg_s = reinterpret_cast<uint32_t*>(smem + S::OFF_NEG);  // H_s sign words (0 for n_s = 1)
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r0 = blockIdx.x, G = gridDim.x;
  const int64_t units = a.rows / RPS;   // MMAs (RPS rows each)
  const int niter = units > r0 ? (int)((units - r0 + G - 1) / G) : 0;

  // one TMA tensor copy: the RPS rows of iteration `it` into stage s
  auto copy_row = [&](int it, int s) {
    mbar_arrive_expect_tx(&full[s], (uint32_t)S::ROWB);
    tma_load_5d(smem + S::OFF_STG + s * S::ROWB, &tmx, &full[s], 0, 0, 0, 0, (int32_t)(r0 + (int64_t)it * G));
    issued[s] = it;
  };
  if (tid == 0) {
    for (int s = 0; s < NSTG; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&sfree[s], 1);
      issued[s] = -1;
    }
    for (int b = 0; b < NBUF; ++b) {
      mbar_init(&dfull[b], 1);
      mbar_init(&dfree[b], S::GW);
    }
    mbar_init(drain, 1);
    if (!S::QUADS)
      for (int e = 0; e < S::REDB / 8; ++e) {   // every slot at its identity
        rslot[2 * e] = SYM ? 0 : INT_MIN;
        rslot[2 * e + 1] = INT_MAX;
      }
    // constant indexes: a lane-dependent index into the parameter space
    // would serialize over the distinct words
#pragma unroll
    for (int q = 0; q < 32; ++q) neg_s[q] = a.n_small > 1 ? a.hs.neg[q] : 0u;
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmx);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, S::TMEM_COLS);
    tmem_relinquish();
  }
  __syncthreads();   // barriers and sign words
  // the first pass over the ring is issued before T is built, so the first
  // rows land while the CTA sets up (measured: issuing two first and the
  // rest once row 0 is in was slower, 18.3 against 17.3 us on 2048 x 14336)
  const int it0 = a.debug_stall ? 0 : (niter < NSTG ? niter : NSTG);
  if (tid == 0) {
    pdl_wait();
    for (int it = 0; it < it0; ++it) copy_row(it, it);
  }

  // T = I_RPS (x) H_f^T in the MMA's A layout (K-major, 128-byte swizzle):
  // element (m, k) at K atom k / 64, row m, bytes 2 (k % 64); m = F r + a,
  // a = i JHB + jh; T[(r, a)][(r, a')] = H_s[i'][i] H_JHB[jh'][jh], zero
  // between different rows r and outside MR.  A warp writes one row m per
  // step, lane l the four k = 4 l .. 4 l + 3 (their terms fixed per lane).
  {
    const int lj = __ffs(a.n_pow2) - 8;   // log2(P / 128): P is a power of two
    const int jm = (1 << lj) - 1;
    uint32_t wk[4];
    int jk[4], rk[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int kk = 4 * lane + q, ak = kk % F;
      wk[q] = neg_s[ak >> lj];
      jk[q] = ak & jm;
      rk[q] = kk < MR ? kk / F : -1;
    }
    uint8_t* tl = smem + S::OFF_T + (lane >> 4) * 16384;
    for (int m = warp; m < 128; m += S::THREADS / 32) {
      const int am = m % F, rm = m < MR ? m / F : -2;
      const int i = am >> lj, jh = am & jm;
      uint32_t h[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint32_t sg = ((wk[q] >> i) ^ (uint32_t)__popc(jh & jk[q])) & 1u;
        h[q] = rk[q] == rm ? (0x3C00u | (sg << 15)) : 0u;   // fp16 +-1 or 0
      }
      *reinterpret_cast<uint2*>(tl + sw128(m, (lane & 15) * 8)) = make_uint2(h[0] | (h[1] << 16), h[2] | (h[3] << 16));
    }
  }
  fence_proxy_async_smem();   // T, written by ordinary stores, is read by the tensor core
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    // ---------------- copies: one TMA tensor copy per row
    if (lane == 0 && !a.debug_stall) {   // a test of the time-outs issues no copies
      for (int it = it0; it < niter; ++it) {
        const int s = it % NSTG;
        if (!mbar_wait_backoff(&sfree[s], (uint32_t)((it / NSTG) - 1) & 1u, abort_flag, g_tc_wait_ns)) break;
        copy_row(it, s);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMAs: T (x) the staged row into accumulator it % NBUF
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_f16_f32_bmn(128, 128);
      const uint32_t tb = smem_u32(smem + S::OFF_T), sb0 = smem_u32(smem + S::OFF_STG);
      // with two rows per MMA this thread sleeps between polls (H_8192 on
      // 8192 x 8192: 33.2 against 36.8 us polling); with one it polls
      // (H_28 (x) H_512 on 2048 x 14336: 17.3 against 17.8 us sleeping)
      auto mma_wait = [&](uint64_t* bar, uint32_t parity) {
        return RPS > 1 ? mbar_wait_backoff(bar, parity, abort_flag, g_tc_wait_ns) : tc_wait(bar, parity, abort_flag);
      };
      for (int it = 0; it < niter; ++it) {
        const int s = it % NSTG, b = it % NBUF;
        if (!mma_wait(&full[s], (uint32_t)(it / NSTG) & 1u)) break;
        if (it >= NBUF && !mma_wait(&dfree[b], (uint32_t)((it / NBUF) - 1) & 1u)) break;
        tc_fence_after();
        const uint32_t sb = sb0 + (uint32_t)(s * S::ROWB);
        // E = T [X0 | X1]: columns 0..63 E0 = T X0, columns 64..127 E1 = T X1
#pragma unroll
        for (int ks = 0; ks < KS; ++ks)
          tc_mma_f16(tmem + (uint32_t)(b * 128), umma_desc_sw128(tb + (ks >> 2) * 16384 + (ks & 3) * 32),
                     umma_desc_sw128_mn(sb + ks * 2048, S::ATOMB, 1024), idesc, ks > 0 ? 1u : 0u);
        tc_commit(&sfree[s]);   // the stage may be refilled once these MMAs have read it
        tc_commit(&dfull[b]);
      }
      // tensor memory is released only after every MMA issued has completed
      tc_commit(drain);
      mbar_wait_bounded(drain, 0, kTcWaitLimitNs);
    }
  } else {
    // ---------------- groups of GW = 4 warps (one per tensor-memory lane
    // quadrant): butterflies, range, Eq. 1, codes
    constexpr int GW = S::GW;
    const int gw = warp - 2, grp = gw / GW, quad = warp & 3;
    const int m = quad * 32 + lane;   // this thread's lane: row r = m / F, block a = m % F
    const bool live = m < MR;
    const int rr_ = live ? m / F : 0;  // its input row within the MMA
    for (int it = grp; it < niter; it += NGRP) {
      const int b = it % NBUF;
      const int64_t row = (r0 + (int64_t)it * G) * RPS + rr_;
      // on a failed wait the accumulator is read anyway (in bounds, discarded below)
      const bool ok = tc_wait(&dfull[b], (uint32_t)(it / NBUF) & 1u, abort_flag);
      __syncwarp();   // the tensor-memory loads below are warp-collective
      tc_fence_after();
      uint32_t r[128];
      const uint32_t ta = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(b * 128);
#pragma unroll
      for (int q = 0; q < 128; q += 32) tmem_ld_32x32b_x32(ta + q, r + q);
#pragma unroll
      for (int q = 0; q < 128; q += 16) tmem_ld_wait(r + q);
      tc_fence_before();
      __syncwarp();
      if (lane == 0 && ok) mbar_arrive(&dfree[b]);   // the accumulator is in registers
      // H_128 over jl: bit 0 inside each pair (jl, jl + 1), bits 1..6 across pairs
      F2 z[64];
#pragma unroll
      for (int p = 0; p < 64; ++p) {
        z[p] = f2_from_bits(r[2 * p], r[2 * p + 1]);
        f2_bfly_inner(z[p]);
      }
#pragma unroll
      for (int h = 1; h < 64; h <<= 1)
#pragma unroll
        for (int p = 0; p < 64; ++p)
          if (!(p & h)) f2_bfly(z[p], z[p | h]);
      // row range: four partial ranges per thread (short dependency chains),
      // then over the row's lanes; the group barrier also settles the abort
      // decision for every thread of the group
      Range<SYM> rg[4];
      if (live) {
#pragma unroll
        for (int p = 0; p < 64; ++p) rg[p & 3].add_pair(z[p]);
      }
#pragma unroll
      for (int q = 1; q < 4; ++q) {
        rg[0].hi = fmaxf(rg[0].hi, rg[q].hi);
        if (!SYM) rg[0].lo = fminf(rg[0].lo, rg[q].lo);
      }
      const int qrow = it / NGRP;
      Range<SYM> rr;
      if constexpr (S::QUADS) {
        // one warp reduction, the partials of the quadrants holding the row
        // (scratch alternates between the group's rows: one barrier per row)
        rg[0].warp_reduce();
        float* rd = reinterpret_cast<float*>(rslot) + (grp * 2 + (qrow & 1)) * 2 * GW;
        if (lane == 0) {
          rd[quad] = rg[0].hi;
          rd[GW + quad] = rg[0].lo;
        }
        if (tc_bar_or(1 + grp, 32 * GW, !ok || *abort_flag)) break;
        const int q_lo = (rr_ * F) / 32, q_hi = ((rr_ + 1) * F - 1) / 32;
        rr.hi = rd[q_lo];
        rr.lo = rd[GW + q_lo];
#pragma unroll
        for (int q = 0; q < GW; ++q)
          if (q > q_lo && q <= q_hi && q * 32 < MR) {
            rr.hi = fmaxf(rr.hi, rd[q]);
            if (!SYM) rr.lo = fminf(rr.lo, rd[GW + q]);
          }
      } else {
        // rows share warps: masked warp reductions per row the warp's lanes
        // span, then shared-memory atomics on order-preserving ints (slot
        // sets rotate over three rows: set q + 1 is reset before this row's
        // barrier, after every thread has read it for row q - 2)
        int* set = rslot + (grp * 3 + qrow % 3) * RPS * 2;
        if (gw % GW == 0 && lane == 0) {
          int* nxt = rslot + (grp * 3 + (qrow + 1) % 3) * RPS * 2;
          for (int r = 0; r < RPS; ++r) {
            nxt[2 * r] = SYM ? 0 : INT_MIN;
            nxt[2 * r + 1] = INT_MAX;
          }
        }
        constexpr int NRW = F >= 32 ? 2 : 3;
        const int row0 = (quad * 32) / F;
#pragma unroll
        for (int k = 0; k < NRW; ++k) {
          const int rk = row0 + k;
          const bool mine = live && rr_ == rk;
          Range<SYM> w;
          if (mine) w = rg[0];
          w.warp_reduce();
          const bool any = __any_sync(0xffffffffu, mine);
          if (lane == 0 && any) {
            if (SYM) {
              atomicMax(&set[2 * rk], __float_as_int(w.hi));   // hi >= 0
            } else {
              atomicMax(&set[2 * rk], f2ord(w.hi));
              atomicMin(&set[2 * rk + 1], f2ord(w.lo));
            }
          }
        }
        if (tc_bar_or(1 + grp, 32 * GW, !ok || *abort_flag)) break;
        rr.hi = SYM ? __int_as_float(set[2 * rr_]) : ord2f(set[2 * rr_]);
        if (!SYM) rr.lo = ord2f(set[2 * rr_ + 1]);
      }
      if constexpr (F8 != 0) {
        // 128 codes of elements 128 a .. 128 a + 127 of row r: one E4M3 byte
        // each, or one byte in each of the two int8 planes (row stride 2K)
        const Quant8<SYM> q8(rr, a.clip, F8 == kFmtE4M3);
        if (live) {
          uint8_t* base = a.codes + row * (F8 == kFmtE4M3 ? a.K : 2 * a.K) + (int64_t)(m % F) * 128;
#pragma unroll
          for (int g = 0; g < 16; g += 2) {
            uint2 h0, l0, h1, l1;
            const F2 v0[4] = {z[4 * g], z[4 * g + 1], z[4 * g + 2], z[4 * g + 3]};
            const F2 v1[4] = {z[4 * g + 4], z[4 * g + 5], z[4 * g + 6], z[4 * g + 7]};
            q8.template codes8<F8>(v0, h0, l0);
            q8.template codes8<F8>(v1, h1, l1);
            *reinterpret_cast<uint4*>(base + g * 8) = make_uint4(h0.x, h0.y, h1.x, h1.y);
            if (F8 == kFmtInt8Planes) *reinterpret_cast<uint4*>(base + a.K + g * 8) = make_uint4(l0.x, l0.y, l1.x, l1.y);
          }
        }
        if (live && m % F == 0) {
          a.scale[row] = q8.alpha * a.norm;
          if (!SYM) a.zero[row] = q8.beta * a.norm;
        }
        continue;
      }
      const QParams<SYM> qp(rr, a.clip);
      if (live) {
        // codes of elements 128 a .. 128 a + 127 of row r: 64 contiguous bytes
        uint4* out = reinterpret_cast<uint4*>(a.codes + row * (a.K / 2) + (int64_t)(m % F) * 64);
#pragma unroll
        for (int w4 = 0; w4 < 4; ++w4) {
          uint32_t wd[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint32_t rb[8];
#pragma unroll
            for (int t = 0; t < 4; ++t) qp.template code_bits2<CLAMP>(z[16 * w4 + 4 * q + t], rb[2 * t], rb[2 * t + 1]);
            wd[q] = pack8_nibbles(rb);
          }
          out[w4] = make_uint4(wd[0], wd[1], wd[2], wd[3]);
        }
      }
      if (live && m % F == 0) {
        a.scale[row] = qp.alpha * a.norm;
        if (!SYM) a.zero[row] = qp.beta * a.norm;
      }
    }
  }
  // after an abort the copies still in flight land before the CTA exits
  if (warp == 0 && lane == 0 && *abort_flag)
    for (int s = 0; s < NSTG; ++s)
      if (issued[s] >= 0) mbar_wait_bounded(&full[s], (uint32_t)(issued[s] / NSTG) & 1u, kTcWaitLimitNs);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (*abort_flag && tid == 0 && a.status && atomicCAS(a.status, 0, (int)SPINQ_ETIMEOUT) == 0)
    atomicExch(a.status + 1, kTcSite);
  if (warp == 1) tmem_dealloc(tmem, S::TMEM_COLS);
}

template <int F, int RPS, bool SYM, bool CLAMP, int F8 = 0>
cudaError_t launch_tc(const RotQuantArgs& a, cudaStream_t stream) {
  using S = RqTc<F, RPS>;
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return cudaErrorNotSupported;
  // RPS rows as (jl % 64, a, r, jl / 64): two 64-column atoms of MR
  // 128-byte rows (r, a) (a indexes the row's 128-element blocks)
  CUtensorMap tmx;
  const cuuint64_t ld = (cuuint64_t)(a.ldx * 2);
  const cuuint64_t gdim[5] = {64, (cuuint64_t)F, (cuuint64_t)RPS, 2, (cuuint64_t)(a.rows / RPS)};
  const cuuint64_t gstr[4] = {256, ld, 128, ld * RPS};
  const cuuint32_t box[5] = {64, (cuuint32_t)F, (cuuint32_t)RPS, 2, 1};
  const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  if (enc(&tmx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 5, const_cast<void*>(a.x), gdim, gstr, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorNotSupported;
  auto kern = rq_tc_kernel<F, RPS, SYM, CLAMP, F8>;
  int per_sm = 0;
  cudaError_t e = prepare_launch_tmem(kern, S::THREADS, S::BYTES, S::TMEM_COLS, &per_sm);
  if (e != cudaSuccess) return e;
  const int64_t units = a.rows / RPS;
  const int64_t cap = (int64_t)device_sm_count() * per_sm;
  const int64_t grid = units < cap ? units : cap;
  RotQuantArgs la = a;
  la.debug_stall = take_debug_stall() ? 1 : 0;
  e = launch_pdl(kern, dim3((unsigned)grid), dim3(S::THREADS), S::BYTES, stream, 1, tmx, la);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int F, int RPS>
cudaError_t launch_tc_f(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  // whole MMAs only, and at least one per SM: below that the per-CTA setup
  // (the constant operand, tensor memory, the pipeline fill) costs more than
  // the row kernels (H_8192 on 8 to 128 tokens: 3.5-3.7 against 2.3-2.5 us)
  *handled = a.rows % RPS == 0 && a.rows / RPS >= device_sm_count();
  if (!*handled) return cudaSuccess;
  const bool clamp = a.clip < 1.0f;
  if (a.symmetric) return clamp ? launch_tc<F, RPS, true, true>(a, stream) : launch_tc<F, RPS, true, false>(a, stream);
  return clamp ? launch_tc<F, RPS, false, true>(a, stream) : launch_tc<F, RPS, false, false>(a, stream);
}

}  // namespace

cudaError_t launch_rotate_quant_8bit_tc(const RotQuantArgs& a, int format, cudaStream_t stream, bool* handled) {
  // the FP8 quantizer on the tcgen05 kernel for H_28 (x) H_512 (the 8-bit
  // linears' down_proj): symmetric, unclipped, no random signs, at least one
  // row per SM
  *handled = false;
  if (format != kFmtE4M3 || !a.symmetric) return cudaSuccess;
  if (a.rows < device_sm_count() || a.signs || a.rowsum || a.clip < 1.0f) return cudaSuccess;
  if (a.n_small != 28 || a.n_pow2 != 512 || a.K != 14336 || (a.ldx * 2) % 16 != 0) return cudaSuccess;
  *handled = true;
  return launch_tc<112, 1, true, false, kFmtE4M3>(a, stream);
}

cudaError_t set_wait_limit_rq_tc(uint64_t ns) { return cudaMemcpyToSymbol(g_tc_wait_ns, &ns, sizeof(ns)); }

cudaError_t launch_rotate_quant_act_tc(const RotQuantArgs& a, cudaStream_t stream, bool* handled) {
  *handled = false;
  if (a.rows == 0 || a.rowsum || a.signs || a.n_small < 1 || a.n_pow2 < 128 || a.n_pow2 % 128 != 0) return cudaSuccess;
  if ((a.ldx * 2) % 16 != 0 || a.K != (int64_t)a.n_small * a.n_pow2) return cudaSuccess;
  // the block counts F = n_s P / 128 with an instance (RPS rows per MMA)
  switch (a.n_small * (a.n_pow2 / 128)) {
    case 112: return launch_tc_f<112, 1>(a, stream, handled);   // H_28 (x) H_512
    case 80: return launch_tc_f<80, 1>(a, stream, handled);     // H_20 (x) H_512
    case 48: return launch_tc_f<48, 2>(a, stream, handled);     // H_12 (x) H_512
    case 24: return launch_tc_f<24, 4>(a, stream, handled);     // H_12 (x) H_256 (19.6 against 20.2 us on 8192 x 3072)
    case 64: return a.n_small == 1 ? launch_tc_f<64, 2>(a, stream, handled) : cudaSuccess;     // H_8192
    case 128: return a.n_small == 1 ? launch_tc_f<128, 1>(a, stream, handled) : cudaSuccess;   // H_16384
  }
  return cudaSuccess;
}

}  // namespace spinq
