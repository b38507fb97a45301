// w4a4_gemm.cu -- W4A4 linear on the 5th-generation tensor core (sm_103a).
//
// y[m][n] = s_n (alpha_m acc[m][n] + beta'_m rowsum_n), acc = sum_k a_mk q_nk
// (the dequantized product of the two Eq. 1 operands; see spinq.h).
//
// sm_103a has no tcgen05 integer MMA, so the 4-bit codes travel as 8-bit
// floats.  Every code is first made unsigned, u = code + 8 for two's
// complement codes (nibble XOR 8) and u = code for asymmetric activations,
// and the byte holding u (0..15) is read as an E4M3 value: exponent field 0
// or 1 with a 3-bit mantissa is exactly u * 2^-9 (subnormals 0..7, the first
// normal binade 8..15).  Unpacking is therefore a mask and a shift per 8
// codes.  The tensor core accumulates S = sum_k u_a u_w * 2^-18 in fp32; S is
// an integer times 2^-18 below 2^24 * 2^-18, so every partial sum is exact and
// the epilogue recovers the integers
//   acc = S * 2^18 - 8 sum_k u_a[m][k] - 8 rowsum_n
// (sum_k u_w = rowsum_n + 8 K cancels the 64 K term).  sum_k u_a is counted
// by the unpack warps while they expand the activation tiles.
//
// Persistent kernel: one CTA per SM walks the output tiles (128 x 256 or
// 256 x 256, M fastest so that concurrently running CTAs share weight tiles
// in L2).  Warp
// roles (704 threads):
//   warp 0       TMA producer: packed A [128 x 64 B] and B [256 x 64 B] tiles
//                for one K step of 128, ring of NP stages.
//   warp 1       TMEM allocation (2 x 256 fp32 columns) and the single-thread
//                MMA issuer: 4 x tcgen05.mma.cta_group::1.kind::f8f6f4 (K = 32)
//                per stage into the accumulator buffer of the current tile.
//   warps 2..5   epilogue, one TMEM lane quadrant each (warp % 4): tcgen05.ld
//                of a finished accumulator, integer recovery, scales, fp16
//                stores.  128-row tiles: runs while the MMA fills the other
//                accumulator buffer.  256-row tiles (one accumulator): the
//                unpack warps share it (five warps per quadrant) and stage
//                y in the then idle operand ring, so that every store
//                instruction writes whole 128-byte row pieces.
//   warps 6..21  unpack the packed tiles into the 128-byte-swizzled K-major
//                E4M3 operand tiles (ring of NU stages) and count sum_k u_a;
//                two groups of 8 warps take alternate K stages so that one
//                group's barrier and fence latency overlaps the other's work.
// Every mbarrier wait is bounded in time; a wait that gives up records
// SPINQ_ETIMEOUT in the device status word and every role winds down.
#include <cuda.h>
#include <cuda_fp16.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>

#include "../../include/spinq.h"
#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"
#include "tensor_map.h"

namespace spinq {

// device status word: [0] = code (SPINQ_ETIMEOUT), [1] = the wait site that gave up
__device__ int g_status[2] = {0, 0};

namespace {

constexpr int BN = 256;
constexpr int kUnpackWarps = 8;   // per group; two groups take alternate K stages
constexpr int kUnpackGroups = 2;
constexpr int kEpiWarps = 4;
constexpr int kThreads = (6 + kUnpackGroups * kUnpackWarps) * 32;
constexpr int kFirstUnpackWarp = 6;
constexpr int kFirstEpiWarp = 2;
constexpr uint64_t kWaitLimitNs = 2000000000ull;
// limit of the ordinary waits (kWaitLimitNs unless a test lowers it); the
// drains of copies and MMAs in flight always use kWaitLimitNs
__device__ uint64_t g_wait_ns = kWaitLimitNs;

__device__ __forceinline__ void record_timeout(int site) {
  if (atomicCAS(&g_status[0], 0, (int)SPINQ_ETIMEOUT) == 0) atomicExch(&g_status[1], site);
}

// Bounded wait that also gives up as soon as another role has aborted.  The
// abort flag and the clock are read once every 64 polls: between them the
// loop touches only the barrier, which keeps polling warps from taking
// shared-memory bandwidth from the unpack and MMA traffic.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                              int site) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > g_wait_ns) {
      record_timeout(site);
      *abort_flag = 1;
      return false;
    }
  }
}

// bar.sync of the four epilogue warps (named barrier 1) whose result is the
// OR of `pred` over them: a decision every epilogue warp takes alike.
__device__ __forceinline__ bool epi_bar_or(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, %2, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(kEpiWarps * 32)
      : "memory");
  return r != 0;
}

// L2 prefetch of the box at (x, y) of a tensor map.  Issued before
// griddepcontrol.wait for the weights only: L2 is coherent with the previous
// kernel's stores and nothing reaches registers or shared memory.
__device__ __forceinline__ void tma_prefetch_2d(const void* tmap, int32_t x, int32_t y) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];\n" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(x), "r"(y)
               : "memory");
}
constexpr int kPrefetchSteps = 4;   // K steps of the first tile's weights prefetched into L2

__device__ __forceinline__ uint32_t swz_off(int r, int chunk) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((chunk ^ (r & 7)) << 4));
}

// 32 packed codes (16 bytes) -> 32 unsigned E4M3 bytes: nibble n -> byte
// (n ^ x) & 15; `lo` holds the even k of each byte group, `hi` the odd k.
__device__ __forceinline__ void unpack16(const uint4 w, uint32_t x, uint4& lo, uint4& hi) {
  uint32_t t;
  t = w.x ^ x; lo.x = t & 0x0F0F0F0Fu; hi.x = (t >> 4) & 0x0F0F0F0Fu;
  t = w.y ^ x; lo.y = t & 0x0F0F0F0Fu; hi.y = (t >> 4) & 0x0F0F0F0Fu;
  t = w.z ^ x; lo.z = t & 0x0F0F0F0Fu; hi.z = (t >> 4) & 0x0F0F0F0Fu;
  t = w.w ^ x; lo.w = t & 0x0F0F0F0Fu; hi.w = (t >> 4) & 0x0F0F0F0Fu;
}

// MT 128-row accumulators per output tile (tile = 128*MT x 256).  MT = 1
// double-buffers the accumulator so the epilogue overlaps the next tile; MT = 2
// uses all of tensor memory for the two accumulators of one tile and unpacks
// each weight tile once for both.
template <int MT>
struct Cfg {
  static constexpr int BMT = 128 * MT;
  static constexpr int NACC = MT == 1 ? 2 : 1;
  static constexpr int NP = MT == 1 ? 3 : 2;   // packed (TMA) stages
  static constexpr int NU = MT == 1 ? 3 : 2;   // unpacked (MMA operand) stages
  static constexpr int TA = BMT * 4 / (kUnpackWarps * 32);   // A chunks per unpack thread
  static constexpr int TB = BN * 4 / (kUnpackWarps * 32);    // B chunks per unpack thread
  static constexpr uint32_t uA = 0;
  static constexpr uint32_t uB = uA + NU * BMT * 128;
  static constexpr uint32_t pA = uB + NU * BN * 128;
  static constexpr uint32_t pB = pA + NP * BMT * 64;
  static constexpr uint32_t bars = pB + NP * BN * 64;
  // full_p[NP] empty_p[NP] full_u[NU] empty_u[NU] acc_full[NACC] acc_empty[NACC]
  // rs_full[2] rs_empty[2] drain cols_full[2] stg_free
  static constexpr int nbars = 2 * NP + 2 * NU + 2 * NACC + 8;
  static constexpr uint32_t misc = bars + nbars * 8;   // tmem slot, abort flag
  static constexpr uint32_t rs_a = (misc + 16 + 15) & ~15u;
  // [tile parity][s_n, (float) rowsum_n][BN]: the column constants of a tile
  static constexpr uint32_t cols = rs_a + 2 * kUnpackGroups * BMT * 4;
  // warps that share the epilogue of a 256-row tile per TMEM lane quadrant:
  // its epilogue warp and the four unpack warps of that quadrant.  Each
  // stages y in blocks of EPI_STAGE bytes: the epilogue warps in a region of
  // their own (estage), the unpack warps in the operand stage that the next
  // tile's first K step does not use (with two stages and two unpack groups,
  // group g always fills stage g: the group that owns the next tile's first
  // step unpacks it before its share, so that its MMA overlaps the stores).
  static constexpr int EPI_PARTS = MT == 2 ? 1 + kUnpackGroups * kUnpackWarps / 4 : 1;
  static constexpr uint32_t EPI_STAGE = 32 * 128;
  static constexpr uint32_t estage = (cols + 2 * 2 * BN * 4 + 1023) & ~1023u;
  static constexpr uint32_t total = MT == 2 ? estage + kEpiWarps * EPI_STAGE : cols + 2 * 2 * BN * 4;
  static constexpr size_t dyn_bytes = total + 1024;
  static_assert(MT == 1 || (NU == 2 && kUnpackGroups == 2 &&
                            kUnpackGroups * kUnpackWarps * EPI_STAGE == BMT * 128 + BN * 128),
                "the unpack warps' staging fills one operand stage");
};

// One warp's share of the epilogue of a 256 x 256 tile.  The tile's rows
// q * 32 + lane (accumulator 0) and 128 + q * 32 + lane (accumulator 1) of
// TMEM lane quadrant q form 8 blocks of 32 rows x 64 columns; this warp takes
// blocks g = part, part + nparts, ...  A block is read from tensor memory in
// four 16-column loads (a lane holds its row), turned into y with the
// epilogue formula on packed fp32 pairs and written as fp16 to the warp's
// 4 KB staging block in shared memory (row r at r * 128 bytes, 16-byte chunk
// c at (c ^ (r % 8)) * 16: conflict-free both ways); it is then read back
// with 8 lanes per row and stored with 16-byte stores, so that each store
// instruction writes 4 rows x 128 contiguous bytes of y instead of 32
// separate 16-byte pieces.  The accumulator is released (acc_empty) after
// the warp's last tensor-memory load, the staging block (stg_free, unless
// null) after its last read.
//   y = s_n (alpha (S - 8 rs_a - 8 rw_n) + beta' rw_n), S = acc * 2^18,
//   evaluated as y = s_n * fma(alpha * 2^18, acc, c + d * rw_n) with
//   c = -8 alpha rs_a and d = beta' - 8 alpha (the roundings of the other
//   kernels, so that every kernel gives the same bits).
template <bool ASYM, bool ACC_OUT>
__device__ __forceinline__ void epi256_share(const GemmArgs& args, uint32_t tq, int q, int lane, int part,
                                             int nparts, int64_t m_tile0, int64_t n0, const float* col_s,
                                             const float* col_r, int rsa0, int rsa1, uint32_t stage,
                                             uint64_t* acc_empty, uint64_t* stg_free) {
  constexpr int NBLK = 2 * (BN / 64);
  // per-row constants of the two accumulators, kept in scalars: the block
  // loop selects them with a runtime accumulator index
  F2 as2_0, cm2_0, dm2_0, as2_1, cm2_1, dm2_1;
  const int64_t m_0 = m_tile0 + q * 32 + lane, m_1 = m_0 + 128;
#pragma unroll
  for (int mt = 0; mt < 2; ++mt) {
    const int64_t m = mt ? m_1 : m_0;
    float alpha = 0.f, bp = 0.f;
    if (m < args.M) {
      alpha = __ldg(args.a_scale + m);
      if (ASYM) bp = __ldg(args.a_zero + m) + 8.f * alpha;
    }
    const float as = alpha * 262144.0f, cm = -8.f * alpha * (float)(mt ? rsa1 : rsa0), dm = bp - 8.f * alpha;
    (mt ? as2_1 : as2_0) = f2_make(as, as);
    (mt ? cm2_1 : cm2_0) = f2_make(cm, cm);
    (mt ? dm2_1 : dm2_0) = f2_make(dm, dm);
  }
  const uint32_t srow = stage + (uint32_t)lane * 128;
#pragma unroll 1
  for (int g = part; g < NBLK; g += nparts) {
    const int mt = g / (BN / 64), cb = g % (BN / 64);
    const int64_t m = mt ? m_1 : m_0;
    const F2 as2 = mt ? as2_1 : as2_0, cm2 = mt ? cm2_1 : cm2_0, dm2 = mt ? dm2_1 : dm2_0;
    const int rsam = mt ? rsa1 : rsa0;
#pragma unroll 1
    for (int c2 = 0; c2 < 2; ++c2) {
      // two 16-column loads in flight per wait
      uint32_t cur[32];
      tmem_ld_32x32b_x16(tq + (uint32_t)(mt * BN + cb * 64 + c2 * 32), cur);
      tmem_ld_32x32b_x16(tq + (uint32_t)(mt * BN + cb * 64 + c2 * 32 + 16), cur + 16);
      // (one wait covers both loads; each call ties its registers to the wait)
      tmem_ld_wait(cur);
      tmem_ld_wait(cur + 16);
#pragma unroll
      for (int g8 = 0; g8 < 4; ++g8) {
        const int j0 = cb * 64 + c2 * 32 + g8 * 8;
        const ulonglong2 S0 = *reinterpret_cast<const ulonglong2*>(col_s + j0);
        const ulonglong2 S1 = *reinterpret_cast<const ulonglong2*>(col_s + j0 + 4);
        const ulonglong2 R0 = *reinterpret_cast<const ulonglong2*>(col_r + j0);
        const ulonglong2 R1 = *reinterpret_cast<const ulonglong2*>(col_r + j0 + 4);
        uint32_t pw[4];
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          F2 sc2, rw2;
          sc2.u = p == 0 ? S0.x : p == 1 ? S0.y : p == 2 ? S1.x : S1.y;
          rw2.u = p == 0 ? R0.x : p == 1 ? R0.y : p == 2 ? R1.x : R1.y;
          const F2 acc2 = f2_from_bits(cur[g8 * 8 + 2 * p], cur[g8 * 8 + 2 * p + 1]);
          const F2 y2 = f2_mul(sc2, f2_fma(as2, acc2, f2_fma(dm2, rw2, cm2)));
          float lo, hi;
          f2_split(y2, lo, hi);
          pw[p] = pack_half2_bits(lo, hi);
        }
        const int c = c2 * 4 + g8;
        sts128(srow + (uint32_t)((c ^ (lane & 7)) << 4), make_uint4(pw[0], pw[1], pw[2], pw[3]));
        if (ACC_OUT) {
          // the integer accumulator (a debugging output): straight from the lane's row
          const int64_t n = n0 + j0;
          if (m < args.M && n < args.N) {
            int accs[8];
#pragma unroll
            for (int p = 0; p < 4; ++p) {
              const unsigned long long r2 = p == 0 ? R0.x : p == 1 ? R0.y : p == 2 ? R1.x : R1.y;
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                const float rwf = __uint_as_float((uint32_t)(r2 >> (32 * h)));
                accs[2 * p + h] =
                    __float2int_rn(__uint_as_float(cur[g8 * 8 + 2 * p + h]) * 262144.0f) - 8 * rsam - 8 * (int)rwf;
              }
            }
            int4* ap = reinterpret_cast<int4*>(args.acc_out + m * args.N + n);
            ap[0] = make_int4(accs[0], accs[1], accs[2], accs[3]);
            ap[1] = make_int4(accs[4], accs[5], accs[6], accs[7]);
          }
        }
      }
    }
    if (g + nparts >= NBLK) {
      // the warp's last tensor-memory load has completed
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty);
    }
    __syncwarp();   // the block's rows are in shared memory
    // lane l stores 16-byte chunk l % 8 of rows 4 i + l / 8 (N is a multiple
    // of 16: a chunk of 8 columns is wholly inside y or outside it)
    const int c = lane & 7;
    const int64_t n = n0 + cb * 64 + c * 8;
    const int64_t mrow0 = m_tile0 + mt * 128 + q * 32;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = 4 * i + (lane >> 3);
      const uint4 v = lds128(stage + (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)));
      if (mrow0 + r < args.M && n < args.N)
        *reinterpret_cast<uint4*>(reinterpret_cast<__half*>(args.y) + (mrow0 + r) * args.N + n) = v;
    }
    __syncwarp();   // every lane has read the block before it is overwritten
  }
  if (part >= NBLK) {
    // (no block for this warp: nothing to wait for)
    __syncwarp();
    if (lane == 0) mbar_arrive(acc_empty);
  }
  __syncwarp();
  if (stg_free != nullptr && lane == 0) mbar_arrive(stg_free);   // release: orders the block reads above before it
}

// An unpack warp's share of the epilogue of 256-row tile `plt` (local index;
// global tile index `ptile`): waits for the accumulator, the activation row
// sums and the column constants of that tile, then runs its share.  False
// when a wait gave up (the share is skipped; the accumulator and staging
// barriers are then left to the bounded waits of the other roles).
template <bool ASYM, bool ACC_OUT>
__device__ __forceinline__ bool unpack_epi_share(const GemmArgs& args, uint32_t tmem, int warp, int lane, int plt,
                                                 int ptile, int m_tiles, uint64_t* acc_full, uint64_t* acc_empty,
                                                 uint64_t* rs_full, uint64_t* cols_full, uint64_t* stg_free,
                                                 const int* rs_a, const float* cols, uint32_t stage,
                                                 volatile int* abort_flag) {
  constexpr int BMT = 256;
  const int rb = plt & 1;
  bool ok = wait_or_abort(&acc_full[0], plt & 1, abort_flag, 10);
  ok = ok && wait_or_abort(&rs_full[rb], (plt >> 1) & 1, abort_flag, 10);
  ok = ok && wait_or_abort(&cols_full[rb], (plt >> 1) & 1, abort_flag, 10);
  // warp-uniform: the tensor-memory loads are warp-collective
  if (!__all_sync(0xffffffffu, ok)) return false;
  tc_fence_after();
  const int q = warp & 3, part = 1 + (warp - kFirstUnpackWarp) / 4;
  const int r0 = q * 32 + lane, r1 = 128 + q * 32 + lane;
  const int rsa0 = rs_a[(rb * kUnpackGroups) * BMT + r0] + rs_a[(rb * kUnpackGroups + 1) * BMT + r0];
  const int rsa1 = rs_a[(rb * kUnpackGroups) * BMT + r1] + rs_a[(rb * kUnpackGroups + 1) * BMT + r1];
  const float* col_s = cols + rb * 2 * BN;
  constexpr int NPARTS = Cfg<2>::EPI_PARTS;
  epi256_share<ASYM, ACC_OUT>(args, tmem + ((uint32_t)(q * 32) << 16), q, lane, part, NPARTS,
                              (int64_t)(ptile % m_tiles) * BMT, (int64_t)(ptile / m_tiles) * BN, col_s, col_s + BN,
                              rsa0, rsa1, stage, &acc_empty[0], stg_free);
  return true;
}

template <int MT, bool ASYM, bool ACC_OUT>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     GemmArgs args, int num_k, int m_tiles, int num_tiles) {
  using L = Cfg<MT>;
  constexpr int BMT = L::BMT, NP = L::NP, NU = L::NU, NACC = L::NACC;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-aligned base derived from the shared array itself, so that the
  // accesses through it stay shared-memory accesses
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
  uint64_t* cols_full = drain + 1;   // [tile parity]: the tile's column constants are staged
  uint64_t* stg_free = cols_full + 2;   // 256-row tiles: the epilogue's staging blocks are read out
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + L::misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + L::misc + 4);
  volatile uint32_t* scratch = reinterpret_cast<volatile uint32_t*>(base + L::misc + 8);   // see wait_loaded
  int* rs_a = reinterpret_cast<int*>(base + L::rs_a);   // [2][groups][BMT]
  // column constants of tile lt at parity lt & 1: w_scale, then w_rowsum as float
  float* cols = reinterpret_cast<float*>(base + L::cols);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    for (int i = 0; i < NP; ++i) {
      mbar_init(&full_p[i], 1);
      mbar_init(&empty_p[i], kUnpackWarps);
    }
    for (int i = 0; i < NU; ++i) {
      mbar_init(&full_u[i], kUnpackWarps);
      mbar_init(&empty_u[i], 1);
    }
    for (int i = 0; i < NACC; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kEpiWarps * L::EPI_PARTS);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&rs_full[i], kUnpackGroups * kUnpackWarps);
      mbar_init(&rs_empty[i], kEpiWarps);
      mbar_init(&cols_full[i], kEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_init(stg_free, kUnpackGroups * kUnpackWarps);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    if ((int)blockIdx.x < num_tiles)
      for (int kt = 0; kt < kPrefetchSteps && kt < num_k; ++kt)
        tma_prefetch_2d(&tmB, kt * 64, (int)(blockIdx.x / m_tiles) * BN);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  int prod_it = 0;   // copies the producer issued (for the drain after an abort)
  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane == 0) {
      int& it = prod_it;
      bool stop = args.debug_stall != 0;   // a test of the time-outs issues no copies
      for (int tile = blockIdx.x; tile < num_tiles && !stop; tile += gridDim.x) {
        const int32_t m0 = (tile % m_tiles) * BMT, n0 = (tile / m_tiles) * BN;
        for (int kt = 0; kt < num_k; ++kt, ++it) {
          const int s = it % NP;
          if (!wait_or_abort(&empty_p[s], ((it / NP) & 1) ^ 1, abort_flag, 1)) {
            stop = true;
            break;
          }
          mbar_arrive_expect_tx(&full_p[s], (BMT + BN) * 64);
          tma_load_2d(base + L::pA + s * BMT * 64, &tmA, &full_p[s], kt * 64, m0);
          tma_load_2d(base + L::pB + s * BN * 64, &tmB, &full_p[s], kt * 64, n0);
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
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_e4m3_f32(128, BN);
      int it = 0, lt = 0;
      bool stop = false;
      for (int tile = blockIdx.x; tile < num_tiles && !stop; tile += gridDim.x, ++lt) {
        const int b = lt % NACC;
        if (!wait_or_abort(&acc_empty[b], ((lt / NACC) & 1) ^ 1, abort_flag, 2)) break;
        tc_fence_after();
        for (int kt = 0; kt < num_k; ++kt, ++it) {
          const int su = it % NU;
          if (!wait_or_abort(&full_u[su], (it / NU) & 1, abort_flag, 3)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(base + L::uA + su * BMT * 128);
          const uint32_t b0 = smem_u32(base + L::uB + su * BN * 128);
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            const uint32_t d = tmem + (uint32_t)((b * MT + mt) * BN);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_f8f6f4(d, umma_desc_sw128(a0 + mt * 128 * 128 + kk * 32), umma_desc_sw128(b0 + kk * 32),
                            idesc, (kt | kk) != 0);
          }
          tc_commit(&empty_u[su]);
        }
        tc_commit(&acc_full[b]);
      }
      // every MMA issued by this thread has retired once `drain` fires, so the
      // tensor memory can be released even when a role gave up early
      tc_commit(drain);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(drain, 0) && globaltimer_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else if (warp >= kFirstUnpackWarp) {
    // ------------------------------------------------ unpack (group grp takes stages it % 2 == grp)
    const int grp = (warp - kFirstUnpackWarp) / kUnpackWarps;
    const int u = tid - (kFirstUnpackWarp + grp * kUnpackWarps) * 32;   // 0..255
    const uint32_t xa = ASYM ? 0u : 0x88888888u;
    // chunk j of this thread: packed row r = u / 4 + 64 j, 16-byte chunk u % 4;
    // its two unpacked 16-byte chunks 2 (u % 4) and 2 (u % 4) + 1 of that row
    // (swizzled: they differ in address bit 4).  Rows 64 j further down are
    // 4096 bytes further in the packed tile and 8192 in the unpacked one,
    // for the activation and the weight tile alike.
    const uint32_t l0 = (uint32_t)((u >> 2) * 64 + (u & 3) * 16);
    const uint32_t s0 = swz_off(u >> 2, 2 * (u & 3));
    const uint32_t sbase = smem_u32(base);
    // One K step `it` into operand stage it % NU; false when a wait gave up.
    // The activation row sums of the step are added to rs[].
    auto unpack_step = [&](int it, int (&rs)[L::TA]) -> bool {
      const int s = it % NP, su = it % NU;
      if (!wait_or_abort(&full_p[s], (it / NP) & 1, abort_flag, 4) ||
          !wait_or_abort(&empty_u[su], ((it / NU) & 1) ^ 1, abort_flag, 5))
        return false;
      const uint32_t PA = sbase + L::pA + s * BMT * 64, PB = sbase + L::pB + s * BN * 64;
      const uint32_t UA = sbase + L::uA + su * BMT * 128, UB = sbase + L::uB + su * BN * 128;
      uint4 wa[L::TA], wb[L::TB];
#pragma unroll
      for (int j = 0; j < L::TA; ++j) wa[j] = lds128(PA + l0 + 4096 * j);
#pragma unroll
      for (int j = 0; j < L::TB; ++j) wb[j] = lds128(PB + l0 + 4096 * j);
      // packed stage consumed, once every lane's loads have read it
      wait_loaded(wa, scratch);
      wait_loaded(wb, scratch);
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_p[s]);
#pragma unroll
      for (int j = 0; j < L::TA; ++j) {
        uint4 lo, hi;
        unpack16(wa[j], xa, lo, hi);
        rs[j] = (int)__dp4a(lo.x + lo.y + lo.z + lo.w + hi.x + hi.y + hi.z + hi.w, 0x01010101u, (unsigned)rs[j]);
        sts128(UA + s0 + 8192 * j, lo);
        sts128(UA + (s0 ^ 16u) + 8192 * j, hi);
      }
#pragma unroll
      for (int j = 0; j < L::TB; ++j) {
        uint4 lo, hi;
        unpack16(wb[j], 0x88888888u, lo, hi);
        sts128(UB + s0 + 8192 * j, lo);
        sts128(UB + (s0 ^ 16u) + 8192 * j, hi);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&full_u[su]);
      return true;
    };
    // 256-row tiles: after unpacking a tile the warp takes its share of the
    // tile's epilogue, staging y in the operand stage that the next tile's
    // first K step does not use; the group that owns that first step unpacks
    // it before its share (`early`, its row sums in `carry`).  A group waits
    // for the staging blocks in its stage to be read out (stg_free of tile
    // `stg_due`) before it writes that stage again.
    int early = -1, stg_due = -1;
    int carry[L::TA];
#pragma unroll
    for (int j = 0; j < L::TA; ++j) carry[j] = 0;
    int it = 0, lt = 0;
    bool stop = false;
    for (int tile = blockIdx.x; tile < num_tiles && !stop; tile += gridDim.x, ++lt) {
      int rsum[L::TA];
#pragma unroll
      for (int j = 0; j < L::TA; ++j) {
        rsum[j] = carry[j];
        carry[j] = 0;
      }
      for (int kt = 0; kt < num_k; ++kt, ++it) {
        if ((it & 1) != grp) continue;
        if (it == early) continue;   // unpacked ahead, with the previous tile's epilogue
        if (MT == 2 && stg_due >= 0) {
          if (!wait_or_abort(stg_free, stg_due & 1, abort_flag, 11)) {
            stop = true;
            break;
          }
          stg_due = -1;
        }
        if (!unpack_step(it, rsum)) {
          stop = true;
          break;
        }
      }
      if (stop) break;
      // row sums of the unsigned activation codes: 4 lanes share a row
#pragma unroll
      for (int j = 0; j < L::TA; ++j) {
        rsum[j] += __shfl_xor_sync(0xffffffffu, rsum[j], 1);
        rsum[j] += __shfl_xor_sync(0xffffffffu, rsum[j], 2);
      }
      const int b = lt & 1;
      if (!wait_or_abort(&rs_empty[b], ((lt >> 1) & 1) ^ 1, abort_flag, 6)) break;
      if ((u & 3) == 0) {
#pragma unroll
        for (int j = 0; j < L::TA; ++j) rs_a[(b * kUnpackGroups + grp) * BMT + (u >> 2) + 64 * j] = rsum[j];
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&rs_full[b]);
      if constexpr (MT == 2) {
        // `it` is now the next tile's first K step, in stage it & 1
        const int first = it & 1;
        if (tile + (int)gridDim.x < num_tiles && first == grp) {
          if (stg_due >= 0) {
            if (!wait_or_abort(stg_free, stg_due & 1, abort_flag, 11)) break;
            stg_due = -1;
          }
          if (!unpack_step(it, carry)) break;
          early = it;
        }
        const int h = warp - kFirstUnpackWarp;   // 0..15
        const uint32_t stage = sbase + (h < 8 ? L::uA + (1 - first) * BMT * 128 : L::uB + (1 - first) * BN * 128) +
                               (uint32_t)(h & 7) * L::EPI_STAGE;
        if (!unpack_epi_share<ASYM, ACC_OUT>(args, tmem, warp, lane, lt, tile, m_tiles, acc_full, acc_empty, rs_full,
                                             cols_full, stg_free, rs_a, cols, stage, abort_flag))
          break;
        if (1 - first == grp) stg_due = lt;
      }
    }
  } else if (warp >= kFirstEpiWarp && warp < kFirstEpiWarp + kEpiWarps) {
    // ------------------------------------------------ epilogue
    const int q = warp & 3;
    const int et = tid - kFirstEpiWarp * 32;   // 0..127
    int lt = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++lt) {
      const int b = lt % NACC, rb = lt & 1;
      const int64_t n0 = (int64_t)(tile / m_tiles) * BN;
      const int64_t m_tile0 = (int64_t)(tile % m_tiles) * BMT;
      // column constants of this tile into the buffer of its parity.  Its
      // last readers worked on tile lt - 2: with 256-row tiles they all
      // finished before the accumulator of lt - 1 was released; with the
      // double-buffered 128-row accumulators a warp may run a tile ahead of
      // the others, so the four warps meet first
      if constexpr (MT == 1) named_bar_sync(1, kEpiWarps * 32);
      float* col_s = cols + rb * 2 * BN;
      float* col_r = col_s + BN;
      for (int j = et; j < BN; j += kEpiWarps * 32) {
        const int64_t n = n0 + j;
        col_s[j] = n < args.N ? __ldg(args.w_scale + n) : 0.f;
        col_r[j] = n < args.N ? (float)__ldg(args.w_rowsum + n) : 0.f;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&cols_full[rb]);   // release: the warp's stores are ordered before it
      bool ok = wait_or_abort(&acc_full[b], (lt / NACC) & 1, abort_flag, 7);
      ok = ok && wait_or_abort(&rs_full[rb], (lt >> 1) & 1, abort_flag, 8);
      ok = ok && wait_or_abort(&cols_full[rb], (lt >> 1) & 1, abort_flag, 9);
      // the tensor-memory loads below are warp-collective; with 128-row tiles
      // the four warps also meet at a barrier each tile, so they decide alike
      if (MT == 1 ? epi_bar_or(!ok) : !__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      int rsa[MT];
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        const int row = mt * 128 + q * 32 + lane;
        rsa[mt] = rs_a[(rb * kUnpackGroups) * BMT + row] + rs_a[(rb * kUnpackGroups + 1) * BMT + row];
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&rs_empty[rb]);
      const uint32_t tq = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * MT * BN);
      if constexpr (MT == 2) {
        epi256_share<ASYM, ACC_OUT>(args, tq, q, lane, 0, L::EPI_PARTS, m_tile0, n0, col_s, col_r, rsa[0],
                                    rsa[MT - 1], smem_u32(base + L::estage) + (uint32_t)(q * L::EPI_STAGE),
                                    &acc_empty[b], nullptr);
        continue;
      }
      // 128-row tiles: chunks of 16 accumulator columns, loads double-buffered
      // across chunks; the other accumulator buffer is meanwhile being filled
      constexpr int NCH = MT * (BN / 16);
      uint32_t ra[16], rbuf[16];
      auto step = [&](int ci, uint32_t(&cur)[16], uint32_t(&nxt)[16]) {
        tmem_ld_wait(cur);
        if (ci + 1 < NCH) {
          tmem_ld_32x32b_x16(tq + (uint32_t)((ci + 1) * 16), nxt);
        } else {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[b]);   // accumulator buffer free again
        }
        const int mt = ci / (BN / 16), cc = ci % (BN / 16);
        const int64_t m = m_tile0 + mt * 128 + q * 32 + lane;
        const bool mvalid = m < args.M;
        // y = s_n (alpha (S - 8 rs_a - 8 rw_n) + beta' rw_n), S = acc * 2^18, evaluated as
        // y = s_n * fma(alpha * 2^18, acc, c + d * rw_n), c = -8 alpha rs_a, d = beta' - 8 alpha
        float alpha = 0.f, bp = 0.f;
        if (mvalid) {
          alpha = __ldg(args.a_scale + m);
          if (ASYM) bp = __ldg(args.a_zero + m) + 8.f * alpha;
        }
        const float alpha_s = alpha * 262144.0f;
        const float cm = -8.f * alpha * (float)rsa[mt];
        const float dm = bp - 8.f * alpha;
        __half* yrow = reinterpret_cast<__half*>(args.y) + m * args.N;
#pragma unroll
        for (int g8 = 0; g8 < 2; ++g8) {
          const int j0 = cc * 16 + g8 * 8;
          const int64_t n = n0 + j0;
          if (!mvalid || n >= args.N) continue;
          const float4 s0 = *reinterpret_cast<const float4*>(col_s + j0);
          const float4 s1 = *reinterpret_cast<const float4*>(col_s + j0 + 4);
          const float4 q0 = *reinterpret_cast<const float4*>(col_r + j0);
          const float4 q1 = *reinterpret_cast<const float4*>(col_r + j0 + 4);
          const float sc[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
          const float rw[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
          float yv[8];
#pragma unroll
          for (int e = 0; e < 8; ++e)
            yv[e] = sc[e] * fmaf(alpha_s, __uint_as_float(cur[g8 * 8 + e]), fmaf(dm, rw[e], cm));
          *reinterpret_cast<uint4*>(yrow + n) =
              make_uint4(pack_half2_bits(yv[0], yv[1]), pack_half2_bits(yv[2], yv[3]),
                         pack_half2_bits(yv[4], yv[5]), pack_half2_bits(yv[6], yv[7]));
          if (ACC_OUT) {
            int accs[8];
#pragma unroll
            for (int e = 0; e < 8; ++e)
              accs[e] = __float2int_rn(__uint_as_float(cur[g8 * 8 + e]) * 262144.0f) - 8 * rsa[mt] -
                        8 * (int)rw[e];
            int4* ap = reinterpret_cast<int4*>(args.acc_out + m * args.N + n);
            ap[0] = make_int4(accs[0], accs[1], accs[2], accs[3]);
            ap[1] = make_int4(accs[4], accs[5], accs[6], accs[7]);
          }
        }
      };
      tmem_ld_32x32b_x16(tq, ra);
#pragma unroll 1
      for (int ci = 0; ci < NCH; ci += 2) {
        step(ci, ra, rbuf);
        step(ci + 1, rbuf, ra);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  // Every role has stopped, so the abort flag is final here.  After an abort
  // the unpack warps may not have consumed the last copies (another role can
  // abort after the producer issued them): let them land before the CTA and
  // its shared memory go away.
  if (warp == 0 && lane == 0 && *abort_flag)
    for (int j = prod_it - NP < 0 ? 0 : prod_it - NP; j < prod_it; ++j) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&full_p[j % NP], (j / NP) & 1) && globaltimer_ns() - t0 < kWaitLimitNs) {
      }
    }
}

// ---------------------------------------------------------------------------
// Decode / skinny GEMM (M <= 256): the weight tile is the MMA's M side
// (128 output channels per CTA), the tokens its N side (MN = M rounded up to
// 16), and K is split across CTAs so that every SM streams a disjoint slice of
// the weights.  Each split adds its exact integer partial
//   sum_k (u_a - 8)(u_w - 8) = S - 8 sum u_a - 8 sum u_w + 64 K_split
// into an fp32 workspace [M][N] (integer values below 2^24: the sums are exact
// and independent of the order of the adds); the last split of an output tile
// (per-tile counter) converts the tile to fp16 with the epilogue formula and
// clears its workspace rows and counter for the next call.
// ---------------------------------------------------------------------------
constexpr int kDecUnpackWarps = 4;
constexpr int kDecThreads = (6 + kDecUnpackWarps) * 32;   // TMA, MMA, 4 epilogue, 4 unpack warps
constexpr int kDecUnpackThreads = kDecUnpackWarps * 32;

template <int MN>
struct DecCfg {
  static constexpr int NP = MN <= 64 ? 4 : 3;
  static constexpr int NU = MN <= 64 ? 3 : 2;
  static constexpr int TW = 128 * 4 / kDecUnpackThreads;                        // W chunks per unpack thread
  static constexpr int TA = (MN * 4 + kDecUnpackThreads - 1) / kDecUnpackThreads;  // A chunks (last may idle)
  static constexpr uint32_t uW = 0;
  static constexpr uint32_t uA = uW + NU * 128 * 128;
  static constexpr uint32_t pW = uA + NU * MN * 128;
  static constexpr uint32_t pA = pW + NP * 128 * 64;
  static constexpr uint32_t bars = (pA + NP * MN * 64 + 7) & ~7u;
  // full_p[NP] empty_p[NP] full_u[NU] empty_u[NU] acc_full rs_full drain
  static constexpr int nbars = 2 * NP + 2 * NU + 3;
  static constexpr uint32_t misc = bars + nbars * 8;   // tmem slot, abort flag, last flag
  static constexpr uint32_t rsw = (misc + 16 + 15) & ~15u;   // [128] weight row sums of this split
  static constexpr uint32_t rsa = rsw + 128 * 4;               // [MN] token sums of this split
  static constexpr uint32_t tal = rsa + MN * 4;                // [MN] token scales alpha_m
  static constexpr uint32_t tbp = tal + MN * 4;                // [MN] beta'_m (asymmetric tokens)
  static constexpr uint32_t total = tbp + MN * 4;
  static constexpr size_t dyn_bytes = total + 1024;
  static constexpr uint32_t tmem_cols = MN <= 32 ? 32 : MN <= 64 ? 64 : MN <= 128 ? 128 : 256;
};

template <int MN, bool ASYM, bool ACC_OUT>
__global__ void __launch_bounds__(kDecThreads, 2)
    w4a4_decode_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmA,
                       GemmArgs args, float* ws_acc, int* ws_cnt, int ksteps, int nsplit) {
  using L = DecCfg<MN>;
  constexpr int NP = L::NP, NU = L::NU;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-aligned base derived from the shared array itself, so that the
  // accesses through it stay shared-memory accesses
  uint8_t* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L::bars);
  uint64_t* full_p = bars;
  uint64_t* empty_p = full_p + NP;
  uint64_t* full_u = empty_p + NP;
  uint64_t* empty_u = full_u + NU;
  uint64_t* acc_full = empty_u + NU;
  uint64_t* rs_full = acc_full + 1;
  uint64_t* drain = rs_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + L::misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + L::misc + 4);
  volatile int* last_flag = reinterpret_cast<volatile int*>(base + L::misc + 8);
  volatile uint32_t* scratch = reinterpret_cast<volatile uint32_t*>(base + L::misc + 12);   // see wait_loaded
  int* rsw = reinterpret_cast<int*>(base + L::rsw);
  int* rsa = reinterpret_cast<int*>(base + L::rsa);
  float* tal = reinterpret_cast<float*>(base + L::tal);
  float* tbp = reinterpret_cast<float*>(base + L::tbp);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int split = blockIdx.x, ntile = blockIdx.y;
  const int n0 = ntile * 128;
  const int k_begin = (int)((int64_t)split * ksteps / nsplit);
  const int k_end = (int)((int64_t)(split + 1) * ksteps / nsplit);
  const int nk = k_end - k_begin;

  if (tid == 0) {
    for (int i = 0; i < NP; ++i) {
      mbar_init(&full_p[i], 1);
      mbar_init(&empty_p[i], kDecUnpackWarps);
    }
    for (int i = 0; i < NU; ++i) {
      mbar_init(&full_u[i], kDecUnpackWarps);
      mbar_init(&empty_u[i], 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(rs_full, kDecUnpackWarps);
    mbar_init(drain, 1);
    *abort_flag = 0;
    *last_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmW);
    prefetch_tmap(&tmA);
    // this CTA's slice of the weights (up to 16 K steps) into L2
    for (int it = 0; it < nk && it < 16; ++it) tma_prefetch_2d(&tmW, (k_begin + it) * 64, n0);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, L::tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  int issued = 0;   // copies the producer issued (for the drain after an abort)
  if (warp == 0) {
    if (lane == 0) {
      for (int it = 0; it < nk; ++it) {
        const int s = it % NP;
        if (!wait_or_abort(&empty_p[s], ((it / NP) & 1) ^ 1, abort_flag, 11)) break;
        mbar_arrive_expect_tx(&full_p[s], (128 + MN) * 64);
        tma_load_2d(base + L::pW + s * 128 * 64, &tmW, &full_p[s], (k_begin + it) * 64, n0);
        tma_load_2d(base + L::pA + s * MN * 64, &tmA, &full_p[s], (k_begin + it) * 64, 0);
        issued = it + 1;
      }
      if (*abort_flag) {
        for (int j = issued - NP < 0 ? 0 : issued - NP; j < issued; ++j) {
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(&full_p[j % NP], (j / NP) & 1) && globaltimer_ns() - t0 < kWaitLimitNs) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_e4m3_f32(128, MN);
      for (int it = 0; it < nk; ++it) {
        const int su = it % NU;
        if (!wait_or_abort(&full_u[su], (it / NU) & 1, abort_flag, 12)) break;
        tc_fence_after();
        const uint32_t w0 = smem_u32(base + L::uW + su * 128 * 128);
        const uint32_t a0 = smem_u32(base + L::uA + su * MN * 128);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          tc_mma_f8f6f4(tmem, umma_desc_sw128(w0 + kk * 32), umma_desc_sw128(a0 + kk * 32), idesc, (it | kk) != 0);
        tc_commit(&empty_u[su]);
      }
      tc_commit(acc_full);
      tc_commit(drain);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(drain, 0) && globaltimer_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else if (warp >= kFirstUnpackWarp) {
    const int u = tid - kFirstUnpackWarp * 32;   // 0..127
    const uint32_t xa = ASYM ? 0u : 0x88888888u;
    const uint32_t sbase = smem_u32(base);
    int sw[L::TW], sa[L::TA];
#pragma unroll
    for (int j = 0; j < L::TW; ++j) sw[j] = 0;
#pragma unroll
    for (int j = 0; j < L::TA; ++j) sa[j] = 0;
    for (int it = 0; it < nk; ++it) {
      const int s = it % NP, su = it % NU;
      if (!wait_or_abort(&full_p[s], (it / NP) & 1, abort_flag, 13) ||
          !wait_or_abort(&empty_u[su], ((it / NU) & 1) ^ 1, abort_flag, 14))
        break;
      const uint32_t PW = sbase + L::pW + s * 128 * 64, PA = sbase + L::pA + s * MN * 64;
      const uint32_t UW = sbase + L::uW + su * 128 * 128, UA = sbase + L::uA + su * MN * 128;
      uint4 ww[L::TW], wa[L::TA];
#pragma unroll
      for (int j = 0; j < L::TW; ++j) {
        const int i = u + kDecUnpackThreads * j;
        ww[j] = lds128(PW + (i >> 2) * 64 + (i & 3) * 16);
      }
#pragma unroll
      for (int j = 0; j < L::TA; ++j) {
        const int i = u + kDecUnpackThreads * j;
        wa[j] = i < MN * 4 ? lds128(PA + (i >> 2) * 64 + (i & 3) * 16) : make_uint4(0, 0, 0, 0);
      }
      // packed stage consumed, once every lane's loads have read it
      wait_loaded(ww, scratch);
      wait_loaded(wa, scratch);
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_p[s]);
#pragma unroll
      for (int j = 0; j < L::TW; ++j) {
        const int i = u + kDecUnpackThreads * j, r = i >> 2, ch = i & 3;
        uint4 lo, hi;
        unpack16(ww[j], 0x88888888u, lo, hi);
        sw[j] = (int)__dp4a(lo.x + lo.y + lo.z + lo.w + hi.x + hi.y + hi.z + hi.w, 0x01010101u, (unsigned)sw[j]);
        sts128(UW + swz_off(r, 2 * ch), lo);
        sts128(UW + swz_off(r, 2 * ch + 1), hi);
      }
#pragma unroll
      for (int j = 0; j < L::TA; ++j) {
        const int i = u + kDecUnpackThreads * j, r = i >> 2, ch = i & 3;
        if (i < MN * 4) {
          uint4 lo, hi;
          unpack16(wa[j], xa, lo, hi);
          sa[j] = (int)__dp4a(lo.x + lo.y + lo.z + lo.w + hi.x + hi.y + hi.z + hi.w, 0x01010101u, (unsigned)sa[j]);
          sts128(UA + swz_off(r, 2 * ch), lo);
          sts128(UA + swz_off(r, 2 * ch + 1), hi);
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&full_u[su]);
    }
    // row sums over this split: 4 lanes share a row
#pragma unroll
    for (int j = 0; j < L::TW; ++j) {
      sw[j] += __shfl_xor_sync(0xffffffffu, sw[j], 1);
      sw[j] += __shfl_xor_sync(0xffffffffu, sw[j], 2);
      if ((u & 3) == 0) rsw[(u >> 2) + (kDecUnpackThreads / 4) * j] = sw[j];
    }
#pragma unroll
    for (int j = 0; j < L::TA; ++j) {
      sa[j] += __shfl_xor_sync(0xffffffffu, sa[j], 1);
      sa[j] += __shfl_xor_sync(0xffffffffu, sa[j], 2);
      const int r = (u >> 2) + (kDecUnpackThreads / 4) * j;
      if ((u & 3) == 0 && r < MN) rsa[r] = sa[j];
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(rs_full);
  } else if (warp >= kFirstEpiWarp && warp < kFirstEpiWarp + kEpiWarps) {
    const int q = warp & 3;
    const int nl = q * 32 + lane;                 // weight row of this lane (TMEM lane)
    const int64_t n = n0 + nl;
    const int et = tid - kFirstEpiWarp * 32;    // 0..127
    // the tokens' scales, staged while the main loop runs
    for (int m = et; m < MN; m += kEpiWarps * 32) {
      const float alpha = m < args.M ? __ldg(args.a_scale + m) : 0.f;
      tal[m] = alpha;
      tbp[m] = ASYM && m < args.M ? __ldg(args.a_zero + m) + 8.f * alpha : 0.f;
    }
    named_bar_sync(1, kEpiWarps * 32);
    bool ok = wait_or_abort(acc_full, 0, abort_flag, 15);
    ok = ok && wait_or_abort(rs_full, 0, abort_flag, 16);
    __syncwarp();
    tc_fence_after();
    const float kfix = 64.f * 128.f * (float)nk;
    const float wfix = kfix - 8.f * (float)(ok ? rsw[nl] : 0);
    const uint32_t taddr = tmem + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
    for (int c0 = 0; c0 < MN; c0 += 16) {
      uint32_t r[16];
      tmem_ld_32x32b_x16(taddr + (uint32_t)c0, r);
      tmem_ld_wait(r);
      if (!ok || n >= args.N) continue;
      if (nsplit == 1) {
        // the whole K range: this is the final sum, no workspace
        const float sn = __ldg(args.w_scale + n);
        const float rwf = (float)__ldg(args.w_rowsum + n);
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int m = c0 + e;
          if (m < args.M) {
            const float accf = fmaf(__uint_as_float(r[e]), 262144.0f, wfix - 8.f * (float)rsa[m]);
            reinterpret_cast<__half*>(args.y)[(int64_t)m * args.N + n] =
                __float2half_rn(sn * fmaf(tal[m], accf, tbp[m] * rwf));
            if (ACC_OUT) args.acc_out[(int64_t)m * args.N + n] = __float2int_rn(accf);
          }
        }
        continue;
      }
#pragma unroll
      for (int e = 0; e < 16; ++e) {
        const int m = c0 + e;
        if (m < args.M) {
          const float part = fmaf(__uint_as_float(r[e]), 262144.0f, wfix - 8.f * (float)rsa[m]);
          atomicAdd(ws_acc + (int64_t)m * args.N + n, part);
        }
      }
    }
    tc_fence_before();
    if (nsplit > 1) {
    // the last split of this output tile finishes it
    __threadfence();
    named_bar_sync(1, kEpiWarps * 32);
    if (et == 0) *last_flag = ok ? (atomicAdd(ws_cnt + ntile, 1) == nsplit - 1) : 0;
    named_bar_sync(1, kEpiWarps * 32);
    if (*last_flag) {
      __threadfence();
      // thread et owns channel n0 + et for every token; a batch of 32
      // independent loads per round trip to L2
      const int64_t nn = n0 + et;
      if (nn < args.N) {
        const float sn = args.w_scale[nn];
        const float rwf = (float)args.w_rowsum[nn];
        for (int mb = 0; mb < MN && mb < args.M; mb += 32) {
          float accf[32];
#pragma unroll
          for (int e = 0; e < 32; ++e)
            accf[e] = mb + e < args.M ? __ldcg(ws_acc + (int64_t)(mb + e) * args.N + nn) : 0.f;
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const int m = mb + e;
            if (m < args.M) {
              ws_acc[(int64_t)m * args.N + nn] = 0.f;
              reinterpret_cast<__half*>(args.y)[(int64_t)m * args.N + nn] =
                  __float2half_rn(sn * fmaf(tal[m], accf[e], tbp[m] * rwf));
              if (ACC_OUT) args.acc_out[(int64_t)m * args.N + nn] = __float2int_rn(accf[e]);
            }
          }
        }
      }
      if (et == 0) ws_cnt[ntile] = 0;
    }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, L::tmem_cols);
  }
  // the abort flag is final here: after an abort, let the producer's last
  // copies land before the CTA goes away (see the prefill kernel)
  if (warp == 0 && lane == 0 && *abort_flag)
    for (int j = issued - NP < 0 ? 0 : issued - NP; j < issued; ++j) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&full_p[j % NP], (j / NP) & 1) && globaltimer_ns() - t0 < kWaitLimitNs) {
      }
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
}  // namespace

bool encode_packed_map(CUtensorMap* map, const void* ptr, int64_t rows, int64_t K, int box_rows) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t gdim[2] = {(cuuint64_t)(K / 2), (cuuint64_t)rows};
  cuuint64_t gstride[1] = {(cuuint64_t)(K / 2)};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), gdim, gstride, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// y [M][N] fp16 for the epilogue's TMA stores: 32 x 32 boxes, 64-byte swizzle
bool encode_y_map(CUtensorMap* map, void* y, int64_t M, int64_t N) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t gdim[2] = {(cuuint64_t)N, (cuuint64_t)M};
  cuuint64_t gstride[1] = {(cuuint64_t)(N * 2)};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, y, gdim, gstride, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

namespace {

template <int MT, bool ASYM, bool ACC_OUT>
cudaError_t launch_t(const GemmArgs& a, cudaStream_t stream) {
  using L = Cfg<MT>;
  CUtensorMap tmA, tmB;
  if (!encode_packed_map(&tmA, a.a_codes, a.M, a.K, L::BMT)) return cudaErrorNotSupported;
  if (!encode_packed_map(&tmB, a.w_codes, a.N, a.K, BN)) return cudaErrorNotSupported;
  auto kern = w4a4_gemm_kernel<MT, ASYM, ACC_OUT>;
  const size_t smem = L::dyn_bytes;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, kThreads, smem, &per_sm);
  if (e != cudaSuccess) return e;
  const int sms = device_sm_count();
  const int m_tiles = (int)((a.M + L::BMT - 1) / L::BMT);
  const int n_tiles = (int)((a.N + BN - 1) / BN);
  const int tiles = m_tiles * n_tiles;
  const int grid = tiles < sms ? tiles : sms;
  GemmArgs la = a;
  la.debug_stall = take_debug_stall() ? 1 : 0;
  e = launch_pdl(kern, dim3(grid), dim3(kThreads), smem, stream, 1, tmA, tmB, la, (int)(a.K / 128), m_tiles,
                 tiles);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int MT>
cudaError_t launch_mt(const GemmArgs& a, cudaStream_t stream) {
  const bool asym = a.a_zero != nullptr, acc = a.acc_out != nullptr;
  if (asym) return acc ? launch_t<MT, true, true>(a, stream) : launch_t<MT, true, false>(a, stream);
  return acc ? launch_t<MT, false, true>(a, stream) : launch_t<MT, false, false>(a, stream);
}

template <int MN, bool ASYM, bool ACC_OUT>
cudaError_t launch_dec_t(const GemmArgs& a, float* ws_acc, int* ws_cnt, int nsplit, cudaStream_t stream) {
  using L = DecCfg<MN>;
  CUtensorMap tmW, tmA;
  if (!encode_packed_map(&tmW, a.w_codes, a.N, a.K, 128)) return cudaErrorNotSupported;
  if (!encode_packed_map(&tmA, a.a_codes, a.M, a.K, MN)) return cudaErrorNotSupported;
  auto kern = w4a4_decode_kernel<MN, ASYM, ACC_OUT>;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, kDecThreads, L::dyn_bytes, &per_sm);
  if (e != cudaSuccess) return e;
  const int ksteps = (int)(a.K / 128);
  const int ntiles = (int)((a.N + 127) / 128);
  // every slice owns at least one K step; slices need the workspace
  if (nsplit < 1 || nsplit > ksteps || (nsplit > 1 && (ws_acc == nullptr || ws_cnt == nullptr)))
    return cudaErrorInvalidValue;
  dim3 grid((unsigned)nsplit, (unsigned)ntiles);
  e = launch_pdl(kern, grid, dim3(kDecThreads), L::dyn_bytes, stream, 1, tmW, tmA, a, ws_acc, ws_cnt, ksteps, nsplit);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int MN>
cudaError_t launch_dec_mn(const GemmArgs& a, float* ws_acc, int* ws_cnt, int nsplit, cudaStream_t stream) {
  const bool asym = a.a_zero != nullptr, acc = a.acc_out != nullptr;
  if (asym) return acc ? launch_dec_t<MN, true, true>(a, ws_acc, ws_cnt, nsplit, stream)
                       : launch_dec_t<MN, true, false>(a, ws_acc, ws_cnt, nsplit, stream);
  return acc ? launch_dec_t<MN, false, true>(a, ws_acc, ws_cnt, nsplit, stream)
             : launch_dec_t<MN, false, false>(a, ws_acc, ws_cnt, nsplit, stream);
}

// Resident CTAs per SM of the split-K kernel for M tokens (the variants of one
// token bucket share their shared memory size).
template <int MN>
int dec_per_sm() {
  int p = 1;
  if (prepare_launch_tmem(w4a4_decode_kernel<MN, false, false>, kDecThreads, DecCfg<MN>::dyn_bytes,
                         (int)DecCfg<MN>::tmem_cols, &p) != cudaSuccess)
    return 1;
  return p;
}
int dec_per_sm_for(int64_t M, int* mn) {
  if (M <= 16) return *mn = 16, dec_per_sm<16>();
  if (M <= 32) return *mn = 32, dec_per_sm<32>();
  if (M <= 64) return *mn = 64, dec_per_sm<64>();
  if (M <= 128) return *mn = 128, dec_per_sm<128>();
  return *mn = 256, dec_per_sm<256>();
}

}  // namespace

std::atomic<int> g_gemm_kernel{SPINQ_GEMM_AUTO};

int w4a4_gemm_select(int kernel) {
  if (kernel < SPINQ_GEMM_AUTO || kernel > SPINQ_GEMM_TCGEMV) return -1;
  return g_gemm_kernel.exchange(kernel);
}

std::atomic<int> g_split_k{0};

int w4a4_gemm_split_k(int n) {
  if (n < 0 || n > 64) return -1;
  return g_split_k.exchange(n);
}

namespace {

// Kernel and tile height from a wave-quantised cost model (microseconds,
// constants measured on GB300 for these kernels; only their ratios matter).
// A persistent CTA (or SM pair) runs ceil(tiles / CTAs) tiles back to back:
//   128 x 256 tiles, one CTA:  0.485 us per 128-deep K step + 3 us (the
//     epilogue overlaps the next tile);
//   256 x 256 tiles, one CTA:  0.66 us per K step + 5.0 us per tile (the
//     single accumulator buffer serialises the epilogue, which all unpack
//     warps share) + 4.9 us once;
//   256 x 256 tiles, SM pair:  0.45 us per K step, epilogue overlapped,
//     + 3 us for the last tile's epilogue.
struct PrefillChoice {
  int kind;
  double us;
};

PrefillChoice choose_prefill(int64_t M, int64_t N, int64_t K, bool allow_pair) {
  const int64_t pairs = allow_pair && M > 128 ? w4a4_gemm_pair_clusters() : 0;
  const int64_t sms = device_sm_count(), ks = K / 128;
  const int64_t tiles256 = ((M + 255) / 256) * ((N + BN - 1) / BN);
  const int64_t tiles128 = ((M + 127) / 128) * ((N + BN - 1) / BN);
  const double est256 = (double)((tiles256 + sms - 1) / sms) * (0.66 * (double)ks + 5.0) + 4.9;
  const double est128 = (double)((tiles128 + sms - 1) / sms) * (0.485 * (double)ks + 3.0);
  PrefillChoice c = est256 < est128 ? PrefillChoice{SPINQ_GEMM_TILE256, est256} : PrefillChoice{SPINQ_GEMM_TILE128, est128};
  if (pairs > 0) {
    const double est_pair = (double)((tiles256 + pairs - 1) / pairs) * 0.45 * (double)ks + 3.0;
    if (est_pair < c.us) c = {SPINQ_GEMM_PAIR, est_pair};
  }
  return c;
}

// The tensor-core GEMV serves every entry point for the shapes it fits when
// it is selected.  Under the automatic choice it takes 3 to 16 tokens where
// its register-streamed form covers K, else 5 to 8 tokens.  Measured on GB300
// over K x N in {3072 x 8192, 8192 x 3072, 4096 x 14336, 14336 x 4096}
// (graphs of 40 calls over 8 weight sets), register-streamed form against
// the GEMV kernel / the split-K kernel:
//   3 tokens:  ~5.2 / 5.5 / 9.7 / 8.8 us against 5.8 / 6.6 / 9.1 / 10.9 (GEMV)
//   8 tokens:  5.4 / 6.1 / 9.9 / 9.2 us against 9.1 / 9.0 / 14.2 / 13.3 (split-K)
//   16 tokens: 7.9 / 8.2 / 13.9 / 12.8 us against 9.8 / 9.7 / 14.8 / 14.1 (split-K)
// and 1 or 2 tokens stay on the GEMV kernel (3.6 / 3.6 / 5.6 / 7.9 us at 1).
constexpr int64_t kGemvTcAutoLo = 5, kGemvTcAutoHi = 8;          // the shared-memory stage form
constexpr int64_t kGemvTcStreamLo = 3, kGemvTcStreamHi = 16;     // the register-streamed form
bool tcgemv_serves(int64_t M, int64_t N, int64_t K) {
  const int forced = g_gemm_kernel.load(std::memory_order_relaxed);
  if (!w4a4_gemv_tc_fits(M, N, K)) return false;
  if (forced == SPINQ_GEMM_TCGEMV) return true;
  if (forced != SPINQ_GEMM_AUTO) return false;
  if (w4a4_gemv_tc_streamed(K)) return M >= kGemvTcStreamLo && M <= kGemvTcStreamHi;
  return M >= kGemvTcAutoLo && M <= kGemvTcAutoHi;
}

}  // namespace

int plan_w4a4_gemm(int64_t M, int64_t N, int64_t K) {
  const int forced = g_gemm_kernel.load(std::memory_order_relaxed);
  if (tcgemv_serves(M, N, K)) return SPINQ_GEMM_TCGEMV;
  // a handful of tokens: the product streams the weights, no tile kernel fits
  // (the split-K selection concerns the other entry point only)
  if ((forced == SPINQ_GEMM_AUTO || forced == SPINQ_GEMM_GEMV || forced == SPINQ_GEMM_SPLITK) &&
      w4a4_gemv_fits(M, K))
    return SPINQ_GEMM_GEMV;
  if (forced == SPINQ_GEMM_TILE128 || forced == SPINQ_GEMM_TILE256) return forced;
  // (a forced GEMV that does not fit falls through to the cost model)
  if (forced == SPINQ_GEMM_PAIR && M > 128 && w4a4_gemm_pair_clusters() > 0) return SPINQ_GEMM_PAIR;
  return choose_prefill(M, N, K, true).kind;
}

cudaError_t launch_w4a4_gemm(const GemmArgs& a, cudaStream_t stream) {
  if (a.M == 0 || a.N == 0) return cudaSuccess;
  const int kind = plan_w4a4_gemm(a.M, a.N, a.K);
  if (kind == SPINQ_GEMM_TCGEMV) {
    bool handled = false;
    const cudaError_t e = launch_w4a4_gemv_tc(a, stream, &handled);
    if (e != cudaSuccess || handled) return e;
  }
  if (kind == SPINQ_GEMM_GEMV) {
    bool handled = false;
    const cudaError_t e = launch_w4a4_gemv(a, stream, &handled);
    if (e != cudaSuccess || handled) return e;
    return launch_mt<1>(a, stream);
  }
  if (kind == SPINQ_GEMM_PAIR) {
    bool handled = false;
    const cudaError_t e = launch_w4a4_gemm_pair(a, stream, &handled);
    if (e != cudaSuccess || handled) return e;
    return launch_mt<2>(a, stream);
  }
  if (kind == SPINQ_GEMM_TILE256) return launch_mt<2>(a, stream);
  return launch_mt<1>(a, stream);
}

// How spinq_w4a4_gemm_splitk serves 5..256 tokens, from a cost model fitted
// on GB300 over K x N in {3072 x 8192, 8192 x 3072, 4096 x 14336,
// 14336 x 4096}, 8..256 tokens and 1..32 slices (microseconds, within 5% on
// average): the split-K kernel with `nsplit` K slices per 128-channel tile,
// or the prefill kernels.  One CTA (a tile's K slice) takes
//   ceil(ks / nsplit) (0.322 + 0.0018 MN)    its 128-deep K steps (MN = tokens
//                                            rounded up to 16 .. 256: the
//                                            unpack and MMA of the tokens' tile)
//   + 3.92 + 0.0375 M                        start-up, epilogue
//   + (nsplit > 1) (1.83 + 0.089 M)          the partial sums' atomics, the
//                                            tile counter and the last
//                                            slice's pass over the workspace
// and the grid runs in ceil(tiles nsplit / resident CTAs) waves.  The
// prefill kernels take their own model + 3 (its constants were fitted on
// large shapes).
// The K slices range over [ns_lo, ns_hi] (both 1 when the caller has no room
// for the partial sums); `allow_prefill` false keeps the split-K kernel.
namespace {

struct DecodePlan {
  bool prefill;
  int nsplit;
};

DecodePlan plan_decode(int64_t M, int64_t N, int64_t K, int ns_lo, int ns_hi, bool allow_prefill) {
  int mn = 16;
  const int per_sm = dec_per_sm_for(M, &mn);
  const double slots = (double)device_sm_count() * per_sm;
  const int ks = (int)(K / 128), ntiles = (int)((N + 127) / 128);
  const double tk = 0.322 + 0.0018 * mn;
  double best = 1e30;
  int best_ns = 1;
  for (int ns = ns_lo; ns <= ns_hi; ++ns) {
    const double waves = std::ceil((double)ntiles * ns / slots);
    const double cta = std::ceil((double)ks / ns) * tk + 3.92 + 0.0375 * (double)M +
                       (ns > 1 ? 1.83 + 0.089 * (double)M : 0.0);
    const double t = waves * cta;
    if (t < best) {
      best = t;
      best_ns = ns;
    }
  }
  if (allow_prefill && choose_prefill(M, N, K, true).us + 3.0 < best) return {true, 0};
  return {false, best_ns};
}

constexpr int kMaxSplit = 64;

int64_t split_workspace_bytes(int64_t M, int64_t N) { return M * N * 4 + ((N + 127) / 128) * 4; }

// The plan of the split-K entry point for 1 <= M <= kDecodeMaxM under the
// current selection; `room`: the caller's workspace holds the partial sums.
DecodePlan plan_splitk_entry(int64_t M, int64_t N, int64_t K, bool room) {
  const int ks = (int)(K / 128);
  const int fixed = g_split_k.load(std::memory_order_relaxed);
  int lo = 1, hi = std::min(ks, kMaxSplit);
  if (fixed > 0) lo = hi = std::min(fixed, ks);
  if (!room) lo = hi = 1;
  // a forced split-K kernel runs whatever the model predicts for the others
  return plan_decode(M, N, K, lo, hi, g_gemm_kernel.load(std::memory_order_relaxed) != SPINQ_GEMM_SPLITK);
}

bool gemv_serves(int64_t M, int64_t K) {
  return g_gemm_kernel.load(std::memory_order_relaxed) != SPINQ_GEMM_SPLITK && w4a4_gemv_fits(M, K);
}

}  // namespace

int64_t w4a4_gemm_workspace_bytes(int64_t M, int64_t N, int64_t K) {
  // only split K slices sum through the workspace
  if (M <= 0 || N <= 0 || M > kDecodeMaxM || gemv_serves(M, K) || tcgemv_serves(M, N, K)) return 0;
  const DecodePlan p = plan_splitk_entry(M, N, K, true);
  if (p.prefill || p.nsplit <= 1) return 0;
  return split_workspace_bytes(M, N);
}

int plan_w4a4_gemm_splitk(int64_t M, int64_t N, int64_t K, int* nsplit) {
  *nsplit = 0;
  if (M > kDecodeMaxM) return plan_w4a4_gemm(M, N, K);
  if (tcgemv_serves(M, N, K)) return SPINQ_GEMM_TCGEMV;
  if (gemv_serves(M, K)) return SPINQ_GEMM_GEMV;
  const DecodePlan p = plan_splitk_entry(M, N, K, true);
  if (p.prefill) return plan_w4a4_gemm(M, N, K);
  *nsplit = p.nsplit;
  return SPINQ_GEMM_SPLITK;
}

cudaError_t launch_w4a4_gemm_splitk(const GemmArgs& a, void* workspace, int64_t workspace_bytes,
                                    cudaStream_t stream) {
  if (a.M == 0 || a.N == 0) return cudaSuccess;
  if (a.M > kDecodeMaxM) return launch_w4a4_gemm(a, stream);
  if (tcgemv_serves(a.M, a.N, a.K)) {
    bool handled = false;
    const cudaError_t et = launch_w4a4_gemv_tc(a, stream, &handled);
    if (et != cudaSuccess || handled) return et;
  }
  if (gemv_serves(a.M, a.K)) {
    bool handled = false;
    const cudaError_t eg = launch_w4a4_gemv(a, stream, &handled);
    if (eg != cudaSuccess || handled) return eg;
  }
  const bool room = workspace != nullptr && workspace_bytes >= split_workspace_bytes(a.M, a.N);
  const DecodePlan p = plan_splitk_entry(a.M, a.N, a.K, room);
  if (p.prefill) return launch_w4a4_gemm(a, stream);
  float* ws_acc = p.nsplit > 1 ? static_cast<float*>(workspace) : nullptr;
  int* ws_cnt = ws_acc == nullptr ? nullptr : reinterpret_cast<int*>(static_cast<char*>(workspace) + a.M * a.N * 4);
  if (a.M <= 16) return launch_dec_mn<16>(a, ws_acc, ws_cnt, p.nsplit, stream);
  if (a.M <= 32) return launch_dec_mn<32>(a, ws_acc, ws_cnt, p.nsplit, stream);
  if (a.M <= 64) return launch_dec_mn<64>(a, ws_acc, ws_cnt, p.nsplit, stream);
  if (a.M <= 128) return launch_dec_mn<128>(a, ws_acc, ws_cnt, p.nsplit, stream);
  return launch_dec_mn<256>(a, ws_acc, ws_cnt, p.nsplit, stream);
}

cudaError_t set_wait_limit_gemm(uint64_t ns) { return cudaMemcpyToSymbol(g_wait_ns, &ns, sizeof(ns)); }

int* device_status_word() {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess) return nullptr;
  return static_cast<int*>(p);
}

cudaError_t read_and_clear_device_status(int32_t* code, int32_t* detail) {
  int st[2] = {0, 0};
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(st, g_status, sizeof(st));
  if (e != cudaSuccess) return e;
  const int zero[2] = {0, 0};
  e = cudaMemcpyToSymbol(g_status, zero, sizeof(zero));
  *code = st[0];
  *detail = st[1];
  return e;
}

}  // namespace spinq
