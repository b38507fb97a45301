// fp8_gemm.cu -- the 8-bit linears on the E4M3 tensor-core pipe (sm_103a):
// W-fp8-A-fp8 (appendix "Latency measurement on GPU": FP8 GEMM with the
// dequantization fused into the epilogue) and W4A8 (main results table,
// 4-8-x rows).
//
//   FP8:  y[m][n] = fp16(alpha_m s_n sum_k a_mk w_nk), a, w E4M3 codes, fp32
//         accumulation in tensor memory.
//   W4A8: the 8-bit activation code c (q, or u - 128) is split exactly as
//         c = 16 (c >> 4) + (c & 15); both parts are small integers that E4M3
//         holds exactly, and so are the 4-bit weight codes.  The activation
//         operand is [M][2K]: plane 0 (k < K) holds 16 (c >> 4), plane 1 holds
//         c & 15, and both planes meet the same weight column k mod K, so the
//         fp32 accumulator is sum_k c_mk q_nk exactly (every partial sum is an
//         integer below 1024 K <= 2^24 for K <= 16384).  Epilogue:
//         y = fp16(s_n (alpha_m acc + beta'_m rowsum_n)), beta' = beta + 128 alpha
//         (asymmetric) or 0.
//
// No unpacking: TMA lands the E4M3 tiles in shared memory with the 128-byte
// swizzle that the MMA reads.  Persistent CTAs (one per SM) walk 128 x 256
// output tiles, M fastest.  Warp roles (192 threads):
//   warp 0     TMA producer: A [128 x 128 B] and B [256 x 128 B] per K step of
//              128, ring of kStages stages;
//   warp 1     tensor-memory allocation (2 x 256 fp32 columns) and the
//              single-thread MMA issuer (4 x kind::f8f6f4, K = 32, per stage);
//   warps 2-5  epilogue, one tensor-memory lane quadrant each (warp % 4): it
//              drains one accumulator while the MMA fills the other.
// Every wait is bounded in time.  A wait that gives up records SPINQ_ETIMEOUT
// in the library's device status word and raises the CTA's abort flag; the
// producer then lets its copies in flight land, the MMA issuer drains its
// MMAs through a final commit, and the allocating warp frees tensor memory.
#include <cuda.h>
#include <cuda_fp16.h>

#include "../../include/spinq.h"
#include "launch_util.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"
#include "tensor_map.h"

namespace spinq {
namespace {

constexpr int BM = 128, BN = 256, BK = 128;
constexpr int kStages = 4;
constexpr int kStageA = BM * BK;            // 16 KB
constexpr int kStageB = BN * BK;            // 32 KB
constexpr int kStageBytes = kStageA + kStageB;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitLimitNs = 2000000000ull;
// limit of the ordinary waits (kWaitLimitNs unless a test lowers it); the
// drains of copies and MMAs in flight always use kWaitLimitNs
__device__ uint64_t g_wait_ns = kWaitLimitNs;
constexpr int OFF_BAR = kStages * kStageBytes;                  // full[S] empty[S] accf[2] acce[2] drain
constexpr int OFF_MISC = OFF_BAR + (2 * kStages + 5) * 8;       // tmem address, abort flag
constexpr int kSmemBytes = OFF_MISC + 16 + 1024;                // + alignment slack

struct Fp8GemmParams {
  const float* a_scale;
  const float* a_zero;     // W4A8 asymmetric only
  const float* w_scale;
  const int32_t* w_rowsum; // W4A8 only
  void* y;
  int32_t* acc_out;        // W4A8 only, optional
  int* status;
  int M, N, K;             // K: the weights' reduction length
  int ksteps;              // K steps of the activation operand (planes * K / 128)
  int debug_stall;         // issue no input copies, so the waits run out (tests)
};

__device__ __forceinline__ void set_timeout(int* status, int site) {
  if (status && atomicCAS(status, 0, (int)SPINQ_ETIMEOUT) == 0) atomicExch(status + 1, site);
}

// Bounded wait: polls the barrier, and every 64 polls the abort flag and the
// clock.  False when another role aborted or the limit expired (then it
// raises the flag and records the site).
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* status,
                                         int site) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > g_wait_ns) {
        *abort_flag = 1;
        set_timeout(status, site);
        return false;
      }
    }
  }
}

template <bool W4A8, bool ASYM>
__global__ void __launch_bounds__(kThreads, 1)
    fp8_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const Fp8GemmParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint64_t* empty = full + kStages;
  uint64_t* acc_full = empty + kStages;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + OFF_MISC + 4);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = (p.M + BM - 1) / BM, nt = (p.N + BN - 1) / BN;
  const int tiles = mt * nt;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();
  pdl_trigger();

  // the producer's last copy into each stage (for the drain after an abort)
  int last_issued[kStages];
  for (int s = 0; s < kStages; ++s) last_issued[s] = -1;
  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      uint32_t g = 0;
      bool ok = !p.debug_stall;   // a test of the time-outs issues no copies
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        const int m0 = (t % mt) * BM, n0 = (t / mt) * BN;
        for (int s = 0; s < p.ksteps; ++s, ++g) {
          const int st = g % kStages;
          if (!wait_bar(&empty[st], ((g / kStages) & 1u) ^ 1u, abort_flag, p.status, 1)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + st * kStageBytes;
          mbar_arrive_expect_tx(&full[st], kStageBytes);
          const int ka = s * BK;
          tma_load_2d(sa, &tmA, &full[st], ka, m0);
          tma_load_2d(sa + kStageA, &tmB, &full[st], W4A8 ? ka % p.K : ka, n0);
          last_issued[st] = (int)g;
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      constexpr uint32_t idesc = umma_idesc_e4m3_f32(BM, BN);
      uint32_t g = 0;
      int lt = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++lt) {
        const int b = lt & 1;
        if (!wait_bar(&acc_empty[b], ((uint32_t)(lt >> 1) & 1u) ^ 1u, abort_flag, p.status, 2)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)(b * BN);
        for (int s = 0; s < p.ksteps; ++s, ++g) {
          const int st = g % kStages;
          if (!wait_bar(&full[st], (g / kStages) & 1u, abort_flag, p.status, 3)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + st * kStageBytes);
#pragma unroll
          for (int kk = 0; kk < BK / 32; ++kk)
            tc_mma_f8f6f4(d, umma_desc_sw128(sa + kk * 32), umma_desc_sw128(sa + kStageA + kk * 32), idesc,
                          (s | kk) != 0);
          tc_commit(&empty[st]);   // the stage is free once these MMAs have read it
        }
        if (ok) tc_commit(&acc_full[b]);
      }
      // every MMA issued above has completed before tensor memory is freed
      tc_commit(drain);
      mbar_wait_bounded(drain, 0, kWaitLimitNs);
    }
  } else {
    // ---------------- epilogue: warp quadrant q = warp % 4 owns rows 32 q ..
    const int q = warp & 3;
    int lt = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++lt) {
      const int b = lt & 1;
      const bool ok = __all_sync(0xffffffffu, wait_bar(&acc_full[b], (uint32_t)(lt >> 1) & 1u, abort_flag,
                                                       p.status, 4));
      if (!ok) break;
      tc_fence_after();
      const int m0 = (t % mt) * BM, n0 = (t / mt) * BN;
      const int row = m0 + 32 * q + lane;
      const bool row_ok = row < p.M;
      const float al = row_ok ? p.a_scale[row] : 0.f;
      const float bp = (W4A8 && ASYM && row_ok) ? p.a_zero[row] + 128.f * al : 0.f;
      __half* yrow = reinterpret_cast<__half*>(p.y) + (size_t)(row_ok ? row : 0) * p.N;
#pragma unroll 1
      for (int cc = 0; cc < BN / 32; ++cc) {
        const int c0 = n0 + cc * 32;
        uint32_t r[32];
        const uint32_t taddr = tmem_base + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * BN + cc * 32);
        __syncwarp();   // the tensor-memory loads are warp-aligned
        tmem_ld_32x32b_x16(taddr, r);
        tmem_ld_32x32b_x16(taddr + 16, r + 16);
        tmem_ld_wait(r);
        tmem_ld_wait(r + 16);
        if (c0 < p.N && row_ok) {   // N is a multiple of 16: the chunk holds 16 or 32 columns
          const int ncol = p.N - c0 >= 32 ? 32 : 16;
          uint32_t h[16];
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float v0 = __uint_as_float(r[j]), v1 = __uint_as_float(r[j + 1]);
            const bool in = c0 + j < p.N;   // j even, N even: both columns or neither
            const float s0 = in ? p.w_scale[c0 + j] : 0.f;
            const float s1 = in ? p.w_scale[c0 + j + 1] : 0.f;
            if (W4A8) {
              const float rs0 = in ? (float)p.w_rowsum[c0 + j] : 0.f;
              const float rs1 = in ? (float)p.w_rowsum[c0 + j + 1] : 0.f;
              if (p.acc_out && in) {
                p.acc_out[(size_t)row * p.N + c0 + j] = (int32_t)v0;
                p.acc_out[(size_t)row * p.N + c0 + j + 1] = (int32_t)v1;
              }
              v0 = s0 * fmaf(al, v0, bp * rs0);
              v1 = s1 * fmaf(al, v1, bp * rs1);
            } else {
              v0 = s0 * (al * v0);
              v1 = s1 * (al * v1);
            }
            h[j >> 1] = pack_half2_bits(v0, v1);
          }
          uint4* dst = reinterpret_cast<uint4*>(yrow + c0);
          dst[0] = make_uint4(h[0], h[1], h[2], h[3]);
          dst[1] = make_uint4(h[4], h[5], h[6], h[7]);
          if (ncol == 32) {
            dst[2] = make_uint4(h[8], h[9], h[10], h[11]);
            dst[3] = make_uint4(h[12], h[13], h[14], h[15]);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[b]);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, kTmemCols);
  // Every role has stopped, so the abort flag is final here.  After an abort
  // the MMA may not have consumed the last copies: let them land before the
  // CTA (and its shared memory) can go away.  Without an abort every copy
  // was waited for by the MMA issuer.
  if (warp == 0 && lane == 0 && *abort_flag)
    for (int s = 0; s < kStages; ++s)
      if (last_issued[s] >= 0) mbar_wait_bounded(&full[s], ((uint32_t)last_issued[s] / kStages) & 1u, kWaitLimitNs);
}

// E4M3 bytes [rows][cols], boxes of 128 bytes x box_rows with the 128-byte
// swizzle the MMA descriptors expect.
bool encode_e4m3_map(CUtensorMap* map, const void* ptr, int64_t rows, int64_t cols, int box_rows) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t gdim[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t gstride[1] = {(cuuint64_t)cols};
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), gdim, gstride, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <bool W4A8, bool ASYM>
cudaError_t launch_t(const Fp8GemmArgs& a, cudaStream_t stream) {
  CUtensorMap tmA, tmB;
  const int planes = W4A8 ? 2 : 1;
  if (!encode_e4m3_map(&tmA, a.a_codes, a.M, planes * a.K, BM)) return cudaErrorNotSupported;
  if (!encode_e4m3_map(&tmB, a.w_codes, a.N, a.K, BN)) return cudaErrorNotSupported;
  auto kern = fp8_gemm_kernel<W4A8, ASYM>;
  int per_sm = 0;
  cudaError_t e = prepare_launch(kern, kThreads, kSmemBytes, &per_sm);
  if (e != cudaSuccess) return e;
  const int64_t tiles = ((a.M + BM - 1) / BM) * ((a.N + BN - 1) / BN);
  const int64_t cap = device_sm_count();
  const int grid = (int)(tiles < cap ? tiles : cap);
  Fp8GemmParams p{a.a_scale, a.a_zero, a.w_scale, a.w_rowsum, a.y, a.acc_out, device_status_word(),
                  (int)a.M, (int)a.N, (int)a.K, (int)(planes * a.K / BK), take_debug_stall() ? 1 : 0};
  e = launch_pdl(kern, dim3(grid), dim3(kThreads), kSmemBytes, stream, 1, tmA, tmB, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t set_wait_limit_fp8(uint64_t ns) { return cudaMemcpyToSymbol(g_wait_ns, &ns, sizeof(ns)); }

cudaError_t launch_fp8_gemm(const Fp8GemmArgs& a, cudaStream_t stream) {
  if (!a.w4a8) return launch_t<false, false>(a, stream);
  return a.a_zero ? launch_t<true, true>(a, stream) : launch_t<true, false>(a, stream);
}

}  // namespace spinq
