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
// Persistent kernel: one CTA per SM walks the output tiles (128 x 256, M
// fastest so that concurrently running CTAs share weight tiles in L2).  Warp
// roles (704 threads):
//   warp 0       TMA producer: packed A [128 x 64 B] and B [256 x 64 B] tiles
//                for one K step of 128, ring of NP stages.
//   warp 1       TMEM allocation (2 x 256 fp32 columns) and the single-thread
//                MMA issuer: 4 x tcgen05.mma.cta_group::1.kind::f8f6f4 (K = 32)
//                per stage into the accumulator buffer of the current tile.
//   warps 2..5   epilogue, one TMEM lane quadrant each (warp % 4): tcgen05.ld
//                of a finished accumulator, integer recovery, scales, fp16
//                stores; runs while the MMA fills the other buffer.
//   warps 6..21  unpack the packed tiles into the 128-byte-swizzled K-major
//                E4M3 operand tiles (ring of NU stages) and count sum_k u_a;
//                two groups of 8 warps take alternate K stages so that one
//                group's barrier and fence latency overlaps the other's work.
// Every mbarrier wait is bounded in time; a wait that gives up records
// SPINQ_ETIMEOUT in the device status word and every role winds down.
#include <cuda.h>
#include <cuda_fp16.h>

#include <mutex>

#include "../../include/spinq.h"
#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {

__device__ int g_status_code = 0;
__device__ int g_status_detail = 0;

namespace {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int NP = 3;   // packed (TMA) stages
constexpr int NU = 3;   // unpacked (MMA operand) stages
constexpr int kUnpackWarps = 8;   // per group; two groups take alternate K stages
constexpr int kUnpackGroups = 2;
constexpr int kEpiWarps = 4;
constexpr int kThreads = (6 + kUnpackGroups * kUnpackWarps) * 32;
constexpr int kFirstUnpackWarp = 6;
constexpr int kFirstEpiWarp = 2;
constexpr uint64_t kWaitLimitNs = 2000000000ull;

__device__ __forceinline__ void record_timeout(int site) {
  if (atomicCAS(&g_status_code, 0, (int)SPINQ_ETIMEOUT) == 0) atomicExch(&g_status_detail, site);
}

// Bounded wait that also gives up as soon as another role has aborted.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                              int site) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      record_timeout(site);
      *abort_flag = 1;
      return false;
    }
  }
}

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

struct Layout {
  static constexpr uint32_t uA = 0;
  static constexpr uint32_t uB = uA + NU * BM * 128;
  static constexpr uint32_t pA = uB + NU * BN * 128;
  static constexpr uint32_t pB = pA + NP * BM * 64;
  static constexpr uint32_t bars = pB + NP * BN * 64;
  // full_p[NP] empty_p[NP] full_u[NU] empty_u[NU] acc_full[2] acc_empty[2] rs_full[2] rs_empty[2] drain
  static constexpr int nbars = 2 * NP + 2 * NU + 9;
  static constexpr uint32_t misc = bars + nbars * 8;   // tmem slot, abort flag
  static constexpr uint32_t rs_a = (misc + 16 + 15) & ~15u;
  static constexpr uint32_t total = rs_a + 2 * kUnpackGroups * BM * 4;
  static constexpr size_t dyn_bytes = total + 1024;
};

template <bool ASYM, bool ACC_OUT>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     GemmArgs args, int num_k, int m_tiles, int num_tiles) {
  using L = Layout;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L::bars);
  uint64_t* full_p = bars;
  uint64_t* empty_p = full_p + NP;
  uint64_t* full_u = empty_p + NP;
  uint64_t* empty_u = full_u + NU;
  uint64_t* acc_full = empty_u + NU;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* rs_full = acc_empty + 2;
  uint64_t* rs_empty = rs_full + 2;
  uint64_t* drain = rs_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + L::misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + L::misc + 4);
  int* rs_a = reinterpret_cast<int*>(base + L::rs_a);

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
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kEpiWarps);
      mbar_init(&rs_full[i], kUnpackGroups * kUnpackWarps);
      mbar_init(&rs_empty[i], kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 2 * BN);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane == 0) {
      int it = 0;
      bool stop = false;
      for (int tile = blockIdx.x; tile < num_tiles && !stop; tile += gridDim.x) {
        const int32_t m0 = (tile % m_tiles) * BM, n0 = (tile / m_tiles) * BN;
        for (int kt = 0; kt < num_k; ++kt, ++it) {
          const int s = it % NP;
          if (!wait_or_abort(&empty_p[s], ((it / NP) & 1) ^ 1, abort_flag, 1)) {
            stop = true;
            break;
          }
          mbar_arrive_expect_tx(&full_p[s], (BM + BN) * 64);
          tma_load_2d(base + L::pA + s * BM * 64, &tmA, &full_p[s], kt * 64, m0);
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
      constexpr uint32_t idesc = umma_idesc_e4m3_f32(BM, BN);
      int it = 0, lt = 0;
      bool stop = false;
      for (int tile = blockIdx.x; tile < num_tiles && !stop; tile += gridDim.x, ++lt) {
        const int b = lt & 1;
        if (!wait_or_abort(&acc_empty[b], ((lt >> 1) & 1) ^ 1, abort_flag, 2)) break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(b * BN);
        for (int kt = 0; kt < num_k; ++kt, ++it) {
          const int su = it % NU;
          if (!wait_or_abort(&full_u[su], (it / NU) & 1, abort_flag, 3)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(base + L::uA + su * BM * 128);
          const uint32_t b0 = smem_u32(base + L::uB + su * BN * 128);
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_f8f6f4(d, umma_desc_sw128(a0 + kk * 32), umma_desc_sw128(b0 + kk * 32), idesc,
                          (kt | kk) != 0);
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
    // fixed task assignment: 2 A chunks and 4 B chunks per thread per stage
    uint32_t la[2], sa[2], ha[2], lb[4], sb[4], hb[4];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int i = u + 256 * j, r = i >> 2, ch = i & 3;
      la[j] = r * 64 + ch * 16;
      sa[j] = swz_off(r, 2 * ch);
      ha[j] = swz_off(r, 2 * ch + 1);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int i = u + 256 * j, r = i >> 2, ch = i & 3;
      lb[j] = r * 64 + ch * 16;
      sb[j] = swz_off(r, 2 * ch);
      hb[j] = swz_off(r, 2 * ch + 1);
    }
    const uint32_t sbase = smem_u32(base);
    int it = 0, lt = 0;
    bool stop = false;
    for (int tile = blockIdx.x; tile < num_tiles && !stop; tile += gridDim.x, ++lt) {
      int rsum0 = 0, rsum1 = 0;
      for (int kt = 0; kt < num_k; ++kt, ++it) {
        if ((it & 1) != grp) continue;
        const int s = it % NP, su = it % NU;
        if (!wait_or_abort(&full_p[s], (it / NP) & 1, abort_flag, 4) ||
            !wait_or_abort(&empty_u[su], ((it / NU) & 1) ^ 1, abort_flag, 5)) {
          stop = true;
          break;
        }
        const uint32_t PA = sbase + L::pA + s * BM * 64, PB = sbase + L::pB + s * BN * 64;
        const uint32_t UA = sbase + L::uA + su * BM * 128, UB = sbase + L::uB + su * BN * 128;
        uint4 wa0 = lds128(PA + la[0]), wa1 = lds128(PA + la[1]);
        uint4 wb[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) wb[j] = lds128(PB + lb[j]);
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_p[s]);   // packed stage consumed
        uint4 lo, hi;
        unpack16(wa0, xa, lo, hi);
        rsum0 = (int)__dp4a(lo.x + lo.y + lo.z + lo.w + hi.x + hi.y + hi.z + hi.w, 0x01010101u, (unsigned)rsum0);
        sts128(UA + sa[0], lo);
        sts128(UA + ha[0], hi);
        unpack16(wa1, xa, lo, hi);
        rsum1 = (int)__dp4a(lo.x + lo.y + lo.z + lo.w + hi.x + hi.y + hi.z + hi.w, 0x01010101u, (unsigned)rsum1);
        sts128(UA + sa[1], lo);
        sts128(UA + ha[1], hi);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          unpack16(wb[j], 0x88888888u, lo, hi);
          sts128(UB + sb[j], lo);
          sts128(UB + hb[j], hi);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&full_u[su]);
      }
      if (stop) break;
      // row sums of the unsigned activation codes: 4 lanes share a row
      rsum0 += __shfl_xor_sync(0xffffffffu, rsum0, 1);
      rsum0 += __shfl_xor_sync(0xffffffffu, rsum0, 2);
      rsum1 += __shfl_xor_sync(0xffffffffu, rsum1, 1);
      rsum1 += __shfl_xor_sync(0xffffffffu, rsum1, 2);
      const int b = lt & 1;
      if (!wait_or_abort(&rs_empty[b], ((lt >> 1) & 1) ^ 1, abort_flag, 6)) break;
      if ((u & 3) == 0) {
        rs_a[(b * kUnpackGroups + grp) * BM + (u >> 2)] = rsum0;
        rs_a[(b * kUnpackGroups + grp) * BM + (u >> 2) + 64] = rsum1;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&rs_full[b]);
    }
  } else if (warp >= kFirstEpiWarp && warp < kFirstEpiWarp + kEpiWarps) {
    // ------------------------------------------------ epilogue
    const int q = warp & 3;
    const int row = q * 32 + lane;
    int lt = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++lt) {
      const int b = lt & 1;
      const int64_t m = (int64_t)(tile % m_tiles) * BM + row;
      const int64_t n0 = (int64_t)(tile / m_tiles) * BN;
      bool ok = wait_or_abort(&acc_full[b], (lt >> 1) & 1, abort_flag, 7);
      ok = ok && wait_or_abort(&rs_full[b], (lt >> 1) & 1, abort_flag, 8);
      __syncwarp();
      if (!ok) break;
      tc_fence_after();
      const int rsa = rs_a[(b * kUnpackGroups) * BM + row] + rs_a[(b * kUnpackGroups + 1) * BM + row];
      __syncwarp();
      if (lane == 0) mbar_arrive(&rs_empty[b]);
      const bool mvalid = m < args.M;
      // y = s_n (alpha (S - 8 rs_a - 8 rw_n) + beta' rw_n), S = acc * 2^18, evaluated as
      // y = s_n * fma(alpha * 2^18, acc, c + d * rw_n), c = -8 alpha rs_a, d = beta' - 8 alpha
      float alpha = 0.f, bp = 0.f;
      if (mvalid) {
        alpha = __ldg(args.a_scale + m);
        if (ASYM) bp = __ldg(args.a_zero + m) + 8.f * alpha;
      }
      const float alpha_s = alpha * 262144.0f;
      const float cm = -8.f * alpha * (float)rsa;
      const float dm = bp - 8.f * alpha;
      __half* yrow = reinterpret_cast<__half*>(args.y) + m * args.N;
#pragma unroll 1
      for (int cc = 0; cc < BN / 32; ++cc) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * BN + cc * 32), r);
        tmem_ld_wait();
        if (cc == BN / 32 - 1) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[b]);   // accumulator buffer free again
        }
#pragma unroll
        for (int g8 = 0; g8 < 4; ++g8) {
          const int64_t n = n0 + cc * 32 + g8 * 8;
          if (!mvalid || n >= args.N) continue;
          const float4 s0 = __ldg(reinterpret_cast<const float4*>(args.w_scale + n));
          const float4 s1 = __ldg(reinterpret_cast<const float4*>(args.w_scale + n) + 1);
          const int4 q0 = __ldg(reinterpret_cast<const int4*>(args.w_rowsum + n));
          const int4 q1 = __ldg(reinterpret_cast<const int4*>(args.w_rowsum + n) + 1);
          const float sc[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
          const int rw[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
          float yv[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float acc = __uint_as_float(r[g8 * 8 + e]);
            yv[e] = sc[e] * fmaf(alpha_s, acc, fmaf(dm, (float)rw[e], cm));
          }
          *reinterpret_cast<uint4*>(yrow + n) =
              make_uint4(pack_half2_bits(yv[0], yv[1]), pack_half2_bits(yv[2], yv[3]),
                         pack_half2_bits(yv[4], yv[5]), pack_half2_bits(yv[6], yv[7]));
          if (ACC_OUT) {
            int accs[8];
#pragma unroll
            for (int e = 0; e < 8; ++e)
              accs[e] = __float2int_rn(__uint_as_float(r[g8 * 8 + e]) * 262144.0f) - 8 * rsa - 8 * rw[e];
            int4* ap = reinterpret_cast<int4*>(args.acc_out + m * args.N + n);
            ap[0] = make_int4(accs[0], accs[1], accs[2], accs[3]);
            ap[1] = make_int4(accs[4], accs[5], accs[6], accs[7]);
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 2 * BN);
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

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

template <bool ASYM, bool ACC_OUT>
cudaError_t launch_t(const GemmArgs& a, cudaStream_t stream) {
  CUtensorMap tmA, tmB;
  if (!encode_packed_map(&tmA, a.a_codes, a.M, a.K, BM)) return cudaErrorNotSupported;
  if (!encode_packed_map(&tmB, a.w_codes, a.N, a.K, BN)) return cudaErrorNotSupported;
  auto kern = w4a4_gemm_kernel<ASYM, ACC_OUT>;
  const size_t smem = Layout::dyn_bytes;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, kThreads, smem, &per_sm);
  if (e != cudaSuccess) return e;
  const int sms = device_sm_count();
  const int m_tiles = (int)((a.M + BM - 1) / BM);
  const int n_tiles = (int)((a.N + BN - 1) / BN);
  const int tiles = m_tiles * n_tiles;
  const int grid = tiles < sms ? tiles : sms;
  kern<<<grid, kThreads, smem, stream>>>(tmA, tmB, a, (int)(a.K / 128), m_tiles, tiles);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_w4a4_gemm(const GemmArgs& a, cudaStream_t stream) {
  if (a.M == 0 || a.N == 0) return cudaSuccess;
  const bool asym = a.a_zero != nullptr, acc = a.acc_out != nullptr;
  if (asym) return acc ? launch_t<true, true>(a, stream) : launch_t<true, false>(a, stream);
  return acc ? launch_t<false, true>(a, stream) : launch_t<false, false>(a, stream);
}

cudaError_t read_and_clear_device_status(int32_t* code, int32_t* detail) {
  int c = 0, d = 0;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(&c, g_status_code, sizeof(int));
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(&d, g_status_detail, sizeof(int));
  if (e != cudaSuccess) return e;
  const int zero = 0;
  e = cudaMemcpyToSymbol(g_status_code, &zero, sizeof(int));
  if (e != cudaSuccess) return e;
  e = cudaMemcpyToSymbol(g_status_detail, &zero, sizeof(int));
  *code = c;
  *detail = d;
  return e;
}

}  // namespace spinq
