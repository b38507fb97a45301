// w4a4_gemm_pair.cu -- the W4A4 prefill GEMM on SM pairs (tcgen05 cta_group::2).
//
// Same arithmetic as w4a4_gemm.cu: the 4-bit codes are made unsigned and read
// as E4M3 bytes (u * 2^-9), the tensor core accumulates S = sum u_a u_w 2^-18
// exactly in fp32, and the epilogue recovers
//   acc = S 2^18 - 8 sum_k u_a - 8 rowsum_n,
//   y   = s_n (alpha_m acc + beta'_m rowsum_n).
//
// Here the two CTAs of a cluster compute one 256 x BN output tile together
// with M = 256 MMAs issued by one thread of CTA 0 (the leader).  CTA rank r
// holds, at the same shared-memory offsets in both CTAs,
//   rows m0 + 128 r .. + 127 of A and rows n0 + (BN/2) r .. of B (unpacked,
//   K-major, 128-byte swizzle),
// and rows m0 + 128 r .. of the accumulator in its own tensor memory (BN fp32
// columns).  Each CTA unpacks only its halves, so an SM unpacks as many bytes
// per flop as in a single-CTA 256 x 256 tile, while its accumulator needs
// only BN columns: two accumulator buffers fit, and the epilogue of one tile
// (TMEM loads, integer recovery, scales, TMA stores of y) runs while the
// tensor core works on the next.
//
// Roles per CTA (704 threads):
//   warp 0       TMA producer of the CTA's packed A and B halves (local ring)
//   warp 1       tensor-memory allocation for the pair (both CTAs); lane 0 of
//                the leader issues the MMAs and commits them to both CTAs
//   warps 2..5   epilogue of the CTA's 128 accumulator rows (TMEM lane
//                quadrant warp % 4), y through swizzled staging and TMA stores
//   warps 6..21  unpack, two groups of 8 warps on alternate K steps
// Signals between the CTAs: the unpack warps of both arrive on the leader's
// full_u (16 arrivals), the epilogues of both on the leader's acc_empty (8);
// the leader's MMA commits arrive, multicast, on empty_u, acc_full and drain
// of both.  Every wait is bounded in time; a wait that gives up records
// SPINQ_ETIMEOUT in the device status word and raises the abort flag of both
// CTAs, so that every role of the pair winds down to the final cluster
// barrier.
#include <cuda.h>
#include <cuda_fp16.h>

#include <map>
#include <mutex>
#include <tuple>

#include "../../include/spinq.h"
#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"
#include "tensor_map.h"

namespace spinq {
namespace {

constexpr int kUnpackWarps = 8;   // per group
constexpr int kUnpackGroups = 2;
constexpr int kEpiWarps = 4;
constexpr int kThreads = (6 + kUnpackGroups * kUnpackWarps) * 32;
constexpr int kFirstUnpackWarp = 6;
constexpr int kFirstEpiWarp = 2;
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint16_t kBothCtas = 0x3;

template <int BN>
struct PairCfg {
  static constexpr int BNH = BN / 2;   // B rows held by each CTA
  static constexpr int NP = 3;         // packed (TMA) stages
  static constexpr int NU = 5;         // unpacked (MMA operand) stages
  static constexpr int NACC = 2;       // accumulator buffers
  static constexpr int TA = 128 * 4 / (kUnpackWarps * 32);   // A chunks per unpack thread
  static constexpr int TB = BNH * 4 / (kUnpackWarps * 32);   // B chunks per unpack thread
  static_assert(TA >= 1 && TB >= 1, "one chunk per unpack thread at least");
  static constexpr uint32_t uA = 0;
  static constexpr uint32_t uB = uA + NU * 128 * 128;
  static constexpr uint32_t pA = uB + NU * BNH * 128;
  static constexpr uint32_t pB = pA + NP * 128 * 64;
  static constexpr uint32_t bars = pB + NP * BNH * 64;
  // full_p[NP] empty_p[NP] full_u[NU] empty_u[NU] acc_full[NACC] acc_empty[NACC]
  // rs_full[2] rs_empty[2] drain
  static constexpr int nbars = 2 * NP + 2 * NU + 2 * NACC + 5;
  static constexpr uint32_t misc = bars + nbars * 8;   // tmem slot, abort flag, scratch
  static constexpr uint32_t rs_a = (misc + 16 + 15) & ~15u;   // [2][groups][128] row sums
  static constexpr uint32_t cols = rs_a + 2 * kUnpackGroups * 128 * 4;   // s_n[BN], (float) rowsum_n[BN]
  static constexpr uint32_t ys = (cols + 2 * BN * 4 + 1023) & ~1023u;  // [epilogue warp][32 x 32 fp16]
  static constexpr uint32_t total = ys + kEpiWarps * 2048;
  static constexpr size_t dyn_bytes = total + 1024;
  static_assert(uB % 1024 == 0 && pA % 1024 == 0, "operand stages keep the 1024-byte swizzle alignment");
};

struct PairCtx {
  volatile int* abort_flag;
  uint32_t peer_abort;   // cluster address of the peer CTA's abort flag
  int* status;           // device status word (code, site) or null
};

__device__ __forceinline__ void give_up(const PairCtx& c, int site) {
  if (c.status != nullptr && atomicCAS(c.status, 0, (int)SPINQ_ETIMEOUT) == 0) atomicExch(c.status + 1, site);
  *c.abort_flag = 1;
  st_shared_cluster_u32(c.peer_abort, 1u);
}

// Bounded wait.  Barriers that the peer CTA arrives on (or the pair's MMA
// commits) are waited on like local ones: an arrive from the peer orders the
// peer's earlier writes like a local arrive does.
__device__ __forceinline__ bool wait_local(uint64_t* bar, uint32_t parity, const PairCtx& c, int site) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (*c.abort_flag) return false;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      give_up(c, site);
      return false;
    }
  }
}

// Wait with sleeps between polls (32 ns doubling to max_ns), for waits off
// the critical path: they leave the issue slots and the barrier unit to the
// unpack warps sharing the SM sub-partition.
__device__ __forceinline__ bool wait_sleepy(uint64_t* bar, uint32_t parity, const PairCtx& c, int site,
                                            uint32_t max_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  uint32_t ns = 32;
  while (true) {
    __nanosleep(ns);
    if (mbar_try_wait(bar, parity)) return true;
    if (*c.abort_flag) return false;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      give_up(c, site);
      return false;
    }
    if (ns < max_ns) ns <<= 1;
  }
}

// bar.sync over the epilogue warps whose result is the OR of `pred` over
// them: one decision for all four, so that none is left at a later barrier
__device__ __forceinline__ bool epi_bar_any(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, %2, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)pred), "n"(kEpiWarps * 32)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ uint32_t swz_off(int r, int chunk) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((chunk ^ (r & 7)) << 4));
}

// 32 packed codes (16 bytes) -> 32 unsigned E4M3 bytes: nibble n -> byte
// (n ^ x) & 15; `lo` holds the even k of each byte group, `hi` the odd k
// (the same permutation of k for A and B, so the sums are unchanged).
__device__ __forceinline__ void unpack16(const uint4 w, uint32_t x, uint4& lo, uint4& hi) {
  uint32_t t;
  t = w.x ^ x; lo.x = t & 0x0F0F0F0Fu; hi.x = (t >> 4) & 0x0F0F0F0Fu;
  t = w.y ^ x; lo.y = t & 0x0F0F0F0Fu; hi.y = (t >> 4) & 0x0F0F0F0Fu;
  t = w.z ^ x; lo.z = t & 0x0F0F0F0Fu; hi.z = (t >> 4) & 0x0F0F0F0Fu;
  t = w.w ^ x; lo.w = t & 0x0F0F0F0Fu; hi.w = (t >> 4) & 0x0F0F0F0Fu;
}

template <int BN, bool ASYM, bool ACC_OUT>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                          const __grid_constant__ CUtensorMap tmY, GemmArgs args, int* status, int num_k,
                          int m_tiles, int num_tiles) {
  using L = PairCfg<BN>;
  constexpr int BNH = L::BNH, NP = L::NP, NU = L::NU, NACC = L::NACC;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-aligned base derived from the shared array itself (the same offset
  // in both CTAs: the MMA addresses the peer's operands by these offsets)
  uint8_t* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L::bars);
  uint64_t* full_p = bars;
  uint64_t* empty_p = full_p + NP;
  uint64_t* full_u = empty_p + NP;
  uint64_t* empty_u = full_u + NU;
  uint64_t* acc_full = empty_u + NU;
  uint64_t* acc_empty = acc_full + NACC;
  uint64_t* rs_full = acc_empty + NACC;
  uint64_t* rs_empty = rs_full + 2;
  uint64_t* drain = rs_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + L::misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + L::misc + 4);
  volatile uint32_t* scratch = reinterpret_cast<volatile uint32_t*>(base + L::misc + 8);   // see wait_loaded
  int* rs_a = reinterpret_cast<int*>(base + L::rs_a);
  float* col_s = reinterpret_cast<float*>(base + L::cols);
  float* col_r = col_s + BN;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_ctarank();
  const int cluster = (int)(blockIdx.x >> 1), nclusters = (int)(gridDim.x >> 1);
  const PairCtx ctx{abort_flag, mapa_shared(smem_u32((const void*)abort_flag), rank ^ 1u), status};

  if (tid == 0) {
    for (int i = 0; i < NP; ++i) {
      mbar_init(&full_p[i], 1);
      mbar_init(&empty_p[i], kUnpackWarps);
    }
    for (int i = 0; i < NU; ++i) {
      mbar_init(&full_u[i], 2 * kUnpackWarps);   // the unpack warps of both CTAs (leader's copy)
      mbar_init(&empty_u[i], 1);
    }
    for (int i = 0; i < NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 2 * kEpiWarps);   // the epilogues of both CTAs (leader's copy)
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&rs_full[i], kUnpackGroups * kUnpackWarps);
      mbar_init(&rs_empty[i], kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    // the first K steps of this CTA's half of the first tile's weights into
    // L2 before the wait on the previous kernel (L2 is coherent with its
    // stores; nothing reaches registers or shared memory before the wait)
    if (cluster < num_tiles)
      for (int kt = 0; kt < 4 && kt < num_k; ++kt)
        asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];\n" ::"l"(
                         reinterpret_cast<uint64_t>(&tmB)),
                     "r"(kt * 64), "r"((cluster / m_tiles) * BN + BNH * (int)rank)
                     : "memory");
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, 512);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  // barriers of both CTAs are initialised (and the tensor memory allocated)
  // before any CTA arrives on its peer's barriers
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  int prod_it = 0;   // copies the producer issued (for the drain after an abort)
  if (warp == 0) {
    // ------------------------------------------------ TMA producer (this CTA's halves)
    if (lane == 0) {
      int& it = prod_it;
      bool stop = false;
      for (int tile = cluster; tile < num_tiles && !stop; tile += nclusters) {
        const int32_t m0 = (tile % m_tiles) * 256 + 128 * (int)rank;
        const int32_t n0 = (tile / m_tiles) * BN + BNH * (int)rank;
        for (int kt = 0; kt < num_k; ++kt, ++it) {
          const int s = it % NP;
          if (!wait_sleepy(&empty_p[s], ((it / NP) & 1) ^ 1, ctx, 11, 256)) {
            stop = true;
            break;
          }
          mbar_arrive_expect_tx(&full_p[s], (128 + BNH) * 64);
          tma_load_2d(base + L::pA + s * 128 * 64, &tmA, &full_p[s], kt * 64, m0);
          tma_load_2d(base + L::pB + s * BNH * 64, &tmB, &full_p[s], kt * 64, n0);
        }
      }
      if (stop) {
        // let copies still in flight land before the CTA exits
        for (int j = it - NP < 0 ? 0 : it - NP; j < it; ++j) {
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(&full_p[j % NP], (j / NP) & 1) && globaltimer_ns() - t0 < kWaitLimitNs) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (leader CTA)
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = umma_idesc_e4m3_f32(256, BN);
      int it = 0, lt = 0;
      bool stop = false;
      for (int tile = cluster; tile < num_tiles && !stop; tile += nclusters, ++lt) {
        const int b = lt % NACC;
        if (!wait_local(&acc_empty[b], ((lt / NACC) & 1) ^ 1, ctx, 12)) break;
        tc_fence_after();
        for (int kt = 0; kt < num_k; ++kt, ++it) {
          const int su = it % NU;
          if (!wait_local(&full_u[su], (it / NU) & 1, ctx, 13)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(base + L::uA + su * 128 * 128);
          const uint32_t b0 = smem_u32(base + L::uB + su * BNH * 128);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_pair_f8f6f4(tmem + (uint32_t)(b * BN), umma_desc_sw128(a0 + kk * 32),
                               umma_desc_sw128(b0 + kk * 32), idesc, (kt | kk) != 0);
          tc_commit_pair_mc(&empty_u[su], kBothCtas);
        }
        if (stop) break;
        tc_commit_pair_mc(&acc_full[b], kBothCtas);
      }
      // every MMA of the pair has retired once `drain` fires in both CTAs
      tc_commit_pair_mc(drain, kBothCtas);
    }
    if (lane == 0) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(drain, 0) && globaltimer_ns() - t0 < kWaitLimitNs) __nanosleep(512);
    }
  } else if (warp >= kFirstUnpackWarp) {
    // ------------------------------------------------ unpack (group grp takes stages it % 2 == grp)
    const int grp = (warp - kFirstUnpackWarp) / kUnpackWarps;
    const int u = tid - (kFirstUnpackWarp + grp * kUnpackWarps) * 32;   // 0..255
    const uint32_t xa = ASYM ? 0u : 0x88888888u;
    uint32_t la[L::TA], sa[L::TA], ha[L::TA], lb[L::TB], sb[L::TB], hb[L::TB];
#pragma unroll
    for (int j = 0; j < L::TA; ++j) {
      const int i = u + 256 * j, r = i >> 2, ch = i & 3;
      la[j] = r * 64 + ch * 16;
      sa[j] = swz_off(r, 2 * ch);
      ha[j] = swz_off(r, 2 * ch + 1);
    }
#pragma unroll
    for (int j = 0; j < L::TB; ++j) {
      const int i = u + 256 * j, r = i >> 2, ch = i & 3;
      lb[j] = r * 64 + ch * 16;
      sb[j] = swz_off(r, 2 * ch);
      hb[j] = swz_off(r, 2 * ch + 1);
    }
    const uint32_t sbase = smem_u32(base);
    int it = 0, lt = 0;
    bool stop = false;
    for (int tile = cluster; tile < num_tiles && !stop; tile += nclusters, ++lt) {
      int rsum[L::TA];
#pragma unroll
      for (int j = 0; j < L::TA; ++j) rsum[j] = 0;
      for (int kt = 0; kt < num_k; ++kt, ++it) {
        if ((it & 1) != grp) continue;
        const int s = it % NP, su = it % NU;
        if (!wait_local(&full_p[s], (it / NP) & 1, ctx, 14) ||
            !wait_local(&empty_u[su], ((it / NU) & 1) ^ 1, ctx, 15)) {
          stop = true;
          break;
        }
        const uint32_t PA = sbase + L::pA + s * 128 * 64, PB = sbase + L::pB + s * BNH * 64;
        const uint32_t UA = sbase + L::uA + su * 128 * 128, UB = sbase + L::uB + su * BNH * 128;
        uint4 wa[L::TA], wb[L::TB];
#pragma unroll
        for (int j = 0; j < L::TA; ++j) wa[j] = lds128(PA + la[j]);
#pragma unroll
        for (int j = 0; j < L::TB; ++j) wb[j] = lds128(PB + lb[j]);
        // packed stage consumed, once every lane's loads have read it
        wait_loaded(wa, scratch);
        wait_loaded(wb, scratch);
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_p[s]);
#pragma unroll
        for (int j = 0; j < L::TA; ++j) {
          uint4 lo, hi;
          unpack16(wa[j], xa, lo, hi);
          rsum[j] = (int)__dp4a(lo.x + lo.y + lo.z + lo.w + hi.x + hi.y + hi.z + hi.w, 0x01010101u,
                                (unsigned)rsum[j]);
          sts128(UA + sa[j], lo);
          sts128(UA + ha[j], hi);
        }
#pragma unroll
        for (int j = 0; j < L::TB; ++j) {
          uint4 lo, hi;
          unpack16(wb[j], 0x88888888u, lo, hi);
          sts128(UB + sb[j], lo);
          sts128(UB + hb[j], hi);
        }
        // the operand tiles are read by the tensor cores (async proxy)
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(mapa_shared(smem_u32(&full_u[su]), 0));
      }
      if (stop) break;
      // row sums of the unsigned activation codes: 4 lanes share a row
#pragma unroll
      for (int j = 0; j < L::TA; ++j) {
        rsum[j] += __shfl_xor_sync(0xffffffffu, rsum[j], 1);
        rsum[j] += __shfl_xor_sync(0xffffffffu, rsum[j], 2);
      }
      const int b = lt & 1;
      if (!wait_local(&rs_empty[b], ((lt >> 1) & 1) ^ 1, ctx, 16)) break;
      if ((u & 3) == 0) {
#pragma unroll
        for (int j = 0; j < L::TA; ++j) rs_a[(b * kUnpackGroups + grp) * 128 + (u >> 2) + 64 * j] = rsum[j];
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&rs_full[b]);
    }
  } else if (warp >= kFirstEpiWarp && warp < kFirstEpiWarp + kEpiWarps) {
    // ------------------------------------------------ epilogue (this CTA's 128 rows)
    const int q = warp & 3;
    const int et = tid - kFirstEpiWarp * 32;   // 0..127
    uint8_t* ybuf = base + L::ys + (warp - kFirstEpiWarp) * 2048;
    if (lane == 0) prefetch_tmap(&tmY);
    const uint32_t acc_empty_leader0 = mapa_shared(smem_u32(&acc_empty[0]), 0);
    int lt = 0;
    for (int tile = cluster; tile < num_tiles; tile += nclusters, ++lt) {
      const int b = lt % NACC, rb = lt & 1;
      const int64_t n0 = (int64_t)(tile / m_tiles) * BN;
      const int64_t row0 = (int64_t)(tile % m_tiles) * 256 + 128 * (int64_t)rank + q * 32;   // of this warp
      // column constants of this tile (the previous tile's epilogue is done with them)
      named_bar_sync(1, kEpiWarps * 32);
      for (int j = et; j < BN; j += kEpiWarps * 32) {
        const int64_t n = n0 + j;
        col_s[j] = n < args.N ? __ldg(args.w_scale + n) : 0.f;
        col_r[j] = n < args.N ? (float)__ldg(args.w_rowsum + n) : 0.f;
      }
      bool ok = wait_sleepy(&acc_full[b], (lt / NACC) & 1, ctx, 17, 1024);
      ok = ok && wait_local(&rs_full[rb], (lt >> 1) & 1, ctx, 18);
      // (also publishes the column constants to the four warps)
      if (epi_bar_any(!ok)) break;
      tc_fence_after();
      const int64_t m = row0 + lane;
      const int rsa = rs_a[(rb * kUnpackGroups) * 128 + q * 32 + lane] +
                      rs_a[(rb * kUnpackGroups + 1) * 128 + q * 32 + lane];
      __syncwarp();
      if (lane == 0) mbar_arrive(&rs_empty[rb]);
      // y = s_n (alpha (S - 8 rs_a - 8 rw_n) + beta' rw_n), S = acc * 2^18, evaluated as
      // y = s_n * fma(alpha * 2^18, acc, c + d * rw_n), c = -8 alpha rs_a, d = beta' - 8 alpha,
      // on packed fp32 pairs (the same roundings as the scalar form)
      float alpha = 0.f, bp = 0.f;
      if (m < args.M) {
        alpha = __ldg(args.a_scale + m);
        if (ASYM) bp = __ldg(args.a_zero + m) + 8.f * alpha;
      }
      const float as = alpha * 262144.0f, cm = -8.f * alpha * (float)rsa, dm = bp - 8.f * alpha;
      const F2 as2 = f2_make(as, as), cm2 = f2_make(cm, cm), dm2 = f2_make(dm, dm);
      constexpr int NCH = BN / 16;
      const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * BN);
      uint32_t ra[16], rbuf[16];
      auto step = [&](int ci, uint32_t(&cur)[16], uint32_t(&nxt)[16]) {
        tmem_ld_wait(cur);
        if (ci + 1 < NCH) {
          tmem_ld_32x32b_x16(tbase + (uint32_t)((ci + 1) * 16), nxt);
        } else {
          // accumulator buffer b of this CTA is read out: tell the leader
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_remote(acc_empty_leader0 + (uint32_t)(b * 8));
        }
        if ((ci & 1) == 0) {
          // the previous block's store must have read the staging buffer
          if (lane == 0) bulk_wait_group_read<0>();
          __syncwarp();
        }
#pragma unroll
        for (int g8 = 0; g8 < 2; ++g8) {
          const int j0 = ci * 16 + g8 * 8;
          // (rows and columns outside y are dropped by the TMA store; their
          // column constants and alpha are zero)
          const ulonglong2 S0 = *reinterpret_cast<const ulonglong2*>(col_s + j0);
          const ulonglong2 S1 = *reinterpret_cast<const ulonglong2*>(col_s + j0 + 4);
          const ulonglong2 R0 = *reinterpret_cast<const ulonglong2*>(col_r + j0);
          const ulonglong2 R1 = *reinterpret_cast<const ulonglong2*>(col_r + j0 + 4);
          const unsigned long long scp[4] = {S0.x, S0.y, S1.x, S1.y};
          const unsigned long long rwp[4] = {R0.x, R0.y, R1.x, R1.y};
          uint32_t pw[4];
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            F2 sc2, rw2;
            sc2.u = scp[p];
            rw2.u = rwp[p];
            const F2 acc2 = f2_from_bits(cur[g8 * 8 + 2 * p], cur[g8 * 8 + 2 * p + 1]);
            const F2 y2 = f2_mul(sc2, f2_fma(as2, acc2, f2_fma(dm2, rw2, cm2)));
            float lo, hi;
            f2_split(y2, lo, hi);
            pw[p] = pack_half2_bits(lo, hi);
          }
          // row `lane`, 16-byte chunk c = 2 (ci & 1) + g8 of the 64-byte row, swizzled
          const int c = 2 * (ci & 1) + g8;
          sts128(smem_u32(ybuf + lane * 64 + ((c ^ ((lane >> 1) & 3)) << 4)), make_uint4(pw[0], pw[1], pw[2], pw[3]));
          if (ACC_OUT) {
            const int64_t n = n0 + j0;
            if (m < args.M && n < args.N) {
              const float rwf[8] = {__uint_as_float((uint32_t)R0.x), __uint_as_float((uint32_t)(R0.x >> 32)),
                                    __uint_as_float((uint32_t)R0.y), __uint_as_float((uint32_t)(R0.y >> 32)),
                                    __uint_as_float((uint32_t)R1.x), __uint_as_float((uint32_t)(R1.x >> 32)),
                                    __uint_as_float((uint32_t)R1.y), __uint_as_float((uint32_t)(R1.y >> 32))};
              int accs[8];
#pragma unroll
              for (int e = 0; e < 8; ++e)
                accs[e] = __float2int_rn(__uint_as_float(cur[g8 * 8 + e]) * 262144.0f) - 8 * rsa - 8 * (int)rwf[e];
              int4* ap = reinterpret_cast<int4*>(args.acc_out + m * args.N + n);
              ap[0] = make_int4(accs[0], accs[1], accs[2], accs[3]);
              ap[1] = make_int4(accs[4], accs[5], accs[6], accs[7]);
            }
          }
        }
        if ((ci & 1) == 1) {
          // the 32 x 32 block is complete: hand it to the TMA engine
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            const int64_t x = n0 + (ci - 1) * 16;   // a multiple of 32 elements: 16-byte aligned
            // a box that starts inside y is clipped to it by the TMA engine;
            // one wholly outside is not issued
            if (x < args.N && row0 < args.M) tma_store_2d(&tmY, ybuf, (int32_t)x, (int32_t)row0);
            bulk_commit_group();
          }
        }
      };
      tmem_ld_32x32b_x16(tbase, ra);
#pragma unroll 1
      for (int ci = 0; ci < NCH; ci += 2) {
        step(ci, ra, rbuf);
        step(ci + 1, rbuf, ra);
      }
    }
    // the staged blocks must be read (and written) before the CTA exits
    if (lane == 0) bulk_wait_group<0>();
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA leaves (or releases tensor memory) while its peer may still
  // arrive on its barriers or the pair's MMAs may still run
  cluster_sync_all();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair(tmem, 512);
  }
  // every role of both CTAs has stopped, so the abort flag is final here:
  // after an abort, let this CTA's last copies land before it goes away
  // (another role may have aborted after the producer issued them)
  if (warp == 0 && lane == 0 && *abort_flag)
    for (int j = prod_it - NP < 0 ? 0 : prod_it - NP; j < prod_it; ++j) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&full_p[j % NP], (j / NP) & 1) && globaltimer_ns() - t0 < kWaitLimitNs) {
      }
    }
}

// Co-resident clusters for this kernel (cached per device and kernel).
template <typename Kern>
cudaError_t max_pair_clusters(Kern kern, size_t smem, int* out) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, int> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  const auto key = std::make_pair(dev, reinterpret_cast<const void*>(kern));
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) {
    *out = it->second;
    return cudaSuccess;
  }
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.gridDim = dim3(2 * (unsigned)device_sm_count(), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  e = cudaOccupancyMaxActiveClusters(&n, kern, &cfg);
  if (e != cudaSuccess) return e;
  cache[key] = n;
  *out = n;
  return cudaSuccess;
}

template <int BN, bool ASYM, bool ACC_OUT>
cudaError_t launch_pair_t(const GemmArgs& a, cudaStream_t stream, bool* handled) {
  using L = PairCfg<BN>;
  auto kern = w4a4_gemm_pair_kernel<BN, ASYM, ACC_OUT>;
  int ncl = 0;
  cudaError_t e = max_pair_clusters(kern, L::dyn_bytes, &ncl);
  if (e != cudaSuccess) return e;
  if (ncl < 1) return cudaSuccess;   // not handled: no SM pair can host it
  CUtensorMap tmA, tmB, tmY;
  if (!encode_packed_map(&tmA, a.a_codes, a.M, a.K, 128)) return cudaErrorNotSupported;
  if (!encode_packed_map(&tmB, a.w_codes, a.N, a.K, L::BNH)) return cudaErrorNotSupported;
  if (!encode_y_map(&tmY, a.y, a.M, a.N)) return cudaErrorNotSupported;
  const int m_tiles = (int)((a.M + 255) / 256);
  const int n_tiles = (int)((a.N + BN - 1) / BN);
  const int tiles = m_tiles * n_tiles;
  const int clusters = tiles < ncl ? tiles : ncl;
  *handled = true;
  e = launch_pdl(kern, dim3(2 * (unsigned)clusters), dim3(kThreads), L::dyn_bytes, stream, 2, tmA, tmB, tmY, a,
                 device_status_word(), (int)(a.K / 128), m_tiles, tiles);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

int w4a4_gemm_pair_clusters() {
  int n = 0;
  if (max_pair_clusters(w4a4_gemm_pair_kernel<256, false, false>, PairCfg<256>::dyn_bytes, &n) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t launch_w4a4_gemm_pair(const GemmArgs& a, cudaStream_t stream, bool* handled) {
  *handled = false;
  if (a.M == 0 || a.N == 0) return cudaSuccess;
  // y rows must be 16-byte multiples for its TMA stores
  if ((a.N * 2) % 16 != 0) return cudaSuccess;
  const bool asym = a.a_zero != nullptr, acc = a.acc_out != nullptr;
  if (asym) return acc ? launch_pair_t<256, true, true>(a, stream, handled)
                       : launch_pair_t<256, true, false>(a, stream, handled);
  return acc ? launch_pair_t<256, false, true>(a, stream, handled)
             : launch_pair_t<256, false, false>(a, stream, handled);
}

}  // namespace spinq

