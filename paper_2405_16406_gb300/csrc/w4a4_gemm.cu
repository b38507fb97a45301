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
// CTA tile 128 x BN (BN = 128 or 256), K step 128.  Warp roles:
//   warp 0      TMA producer: packed A [128 x 64 B] and B [BN x 64 B] tiles,
//               4-stage ring.
//   warp 1      TMEM allocation and the single-thread MMA issuer
//               (tcgen05.mma.cta_group::1.kind::f8f6f4, 4 x K=32 per stage).
//   warps 4..7  unpack packed tiles into the 128-byte-swizzled K-major E4M3
//               operand tiles (2-stage ring), then the epilogue: tcgen05.ld of
//               the fp32 accumulator, integer recovery, scales, fp16 stores.
// Every mbarrier wait is bounded in time; a wait that gives up records
// SPINQ_ETIMEOUT in the device status word and the CTA winds down.
#include <cuda.h>
#include <cuda_fp16.h>

#include <mutex>

#include "../../include/spinq.h"
#include "spinq_device.cuh"
#include "spinq_internal.h"

namespace spinq {

__device__ int g_status_code = 0;
__device__ int g_status_detail = 0;

namespace {

constexpr int BM = 128;
constexpr int NP = 4;  // packed (TMA) stages
constexpr int NU = 2;  // unpacked (MMA operand) stages
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

__device__ __forceinline__ void unpack16(const uint4 w, uint32_t x, uint4& lo, uint4& hi) {
  uint32_t t;
  t = w.x ^ x; lo.x = t & 0x0F0F0F0Fu; hi.x = (t >> 4) & 0x0F0F0F0Fu;
  t = w.y ^ x; lo.y = t & 0x0F0F0F0Fu; hi.y = (t >> 4) & 0x0F0F0F0Fu;
  t = w.z ^ x; lo.z = t & 0x0F0F0F0Fu; hi.z = (t >> 4) & 0x0F0F0F0Fu;
  t = w.w ^ x; lo.w = t & 0x0F0F0F0Fu; hi.w = (t >> 4) & 0x0F0F0F0Fu;
}

template <int BN>
struct Layout {
  static constexpr uint32_t uA = 0;
  static constexpr uint32_t uB = uA + NU * BM * 128;
  static constexpr uint32_t pA = uB + NU * BN * 128;
  static constexpr uint32_t pB = pA + NP * BM * 64;
  static constexpr uint32_t bars = pB + NP * BN * 64;
  static constexpr int nbars = 2 * NP + 2 * NU + 1;
  static constexpr uint32_t misc = bars + nbars * 8;           // tmem slot, abort flag
  static constexpr uint32_t col_scale = (misc + 16 + 15) & ~15u;
  static constexpr uint32_t col_rowsum = col_scale + BN * 4;
  static constexpr uint32_t rs_a = col_rowsum + BN * 4;
  static constexpr uint32_t total = rs_a + BM * 4;
  static constexpr size_t dyn_bytes = total + 1024;              // alignment slack
};

template <int BN, bool ASYM, bool ACC_OUT>
__global__ void __launch_bounds__(256, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     GemmArgs args, int num_k) {
  using L = Layout<BN>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L::bars);
  uint64_t* full_p = bars;
  uint64_t* empty_p = bars + NP;
  uint64_t* full_u = bars + 2 * NP;
  uint64_t* empty_u = bars + 2 * NP + NU;
  uint64_t* acc_full = bars + 2 * NP + 2 * NU;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + L::misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + L::misc + 4);
  float* col_scale = reinterpret_cast<float*>(base + L::col_scale);
  int* col_rowsum = reinterpret_cast<int*>(base + L::col_rowsum);
  int* rs_a = reinterpret_cast<int*>(base + L::rs_a);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t m0 = (int64_t)blockIdx.y * BM, n0 = (int64_t)blockIdx.x * BN;

  if (tid == 0) {
    for (int i = 0; i < NP; ++i) {
      mbar_init(&full_p[i], 1);
      mbar_init(&empty_p[i], 4);
    }
    for (int i = 0; i < NU; ++i) {
      mbar_init(&full_u[i], 4);
      mbar_init(&empty_u[i], 1);
    }
    mbar_init(acc_full, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, BN);
    tmem_relinquish();
  }
  if (tid >= 128) {
    for (int j = tid - 128; j < BN; j += 128) {
      const int64_t n = n0 + j;
      col_scale[j] = n < args.N ? args.w_scale[n] : 0.f;
      col_rowsum[j] = n < args.N ? args.w_rowsum[n] : 0;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      int issued = 0;
      for (int kt = 0; kt < num_k; ++kt) {
        const int s = kt % NP;
        if (!wait_or_abort(&empty_p[s], ((kt / NP) & 1) ^ 1, abort_flag, 1)) break;
        mbar_arrive_expect_tx(&full_p[s], (BM + BN) * 64);
        tma_load_2d(base + L::pA + s * BM * 64, &tmA, &full_p[s], kt * 64, (int32_t)m0);
        tma_load_2d(base + L::pB + s * BN * 64, &tmB, &full_p[s], kt * 64, (int32_t)n0);
        issued = kt + 1;
      }
      if (*abort_flag) {
        // let the copies still in flight land before the CTA exits
        for (int kt = issued - NP < 0 ? 0 : issued - NP; kt < issued; ++kt) {
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(&full_p[kt % NP], (kt / NP) & 1) && globaltimer_ns() - t0 < kWaitLimitNs) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = umma_idesc_e4m3_f32(BM, BN);
      int kt = 0;
      for (; kt < num_k; ++kt) {
        const int su = kt % NU;
        if (!wait_or_abort(&full_u[su], (kt / NU) & 1, abort_flag, 2)) break;
        tc_fence_after();
        const uint32_t a0 = smem_u32(base + L::uA + su * BM * 128);
        const uint32_t b0 = smem_u32(base + L::uB + su * BN * 128);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          tc_mma_f8f6f4(tmem, umma_desc_sw128(a0 + kk * 32), umma_desc_sw128(b0 + kk * 32), idesc,
                        (kt | kk) != 0);
        tc_commit(&empty_u[su]);
      }
      tc_commit(acc_full);
      if (kt < num_k) {
        // aborted: wait (bounded) until the issued MMAs have retired
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(acc_full, 0) && globaltimer_ns() - t0 < kWaitLimitNs) {
        }
      }
    }
  } else if (warp >= 4) {
    const int u = tid - 128;
    const uint32_t xa = ASYM ? 0u : 0x88888888u;
    int rsum[4] = {0, 0, 0, 0};
    for (int kt = 0; kt < num_k; ++kt) {
      const int s = kt % NP, su = kt % NU;
      if (!wait_or_abort(&full_p[s], (kt / NP) & 1, abort_flag, 3)) break;
      if (!wait_or_abort(&empty_u[su], ((kt / NU) & 1) ^ 1, abort_flag, 4)) break;
      const uint8_t* PA = base + L::pA + s * BM * 64;
      const uint8_t* PB = base + L::pB + s * BN * 64;
      uint8_t* UA = base + L::uA + su * BM * 128;
      uint8_t* UB = base + L::uB + su * BN * 128;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int i = u + 128 * j, r = i >> 2, ch = i & 3;
        const uint4 w = *reinterpret_cast<const uint4*>(PA + r * 64 + ch * 16);
        uint4 lo, hi;
        unpack16(w, xa, lo, hi);
        const uint32_t t = lo.x + lo.y + lo.z + lo.w + hi.x + hi.y + hi.z + hi.w;
        rsum[j] = (int)__dp4a(t, 0x01010101u, (unsigned)rsum[j]);
        *reinterpret_cast<uint4*>(UA + swz_off(r, 2 * ch)) = lo;
        *reinterpret_cast<uint4*>(UA + swz_off(r, 2 * ch + 1)) = hi;
      }
#pragma unroll 4
      for (int j = 0; j < BN / 32; ++j) {
        const int i = u + 128 * j, r = i >> 2, ch = i & 3;
        const uint4 w = *reinterpret_cast<const uint4*>(PB + r * 64 + ch * 16);
        uint4 lo, hi;
        unpack16(w, 0x88888888u, lo, hi);
        *reinterpret_cast<uint4*>(UB + swz_off(r, 2 * ch)) = lo;
        *reinterpret_cast<uint4*>(UB + swz_off(r, 2 * ch + 1)) = hi;
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&full_u[su]);
        mbar_arrive(&empty_p[s]);
      }
    }
    // row sums of the unsigned activation codes: lanes u..u^3 share a row
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int v = rsum[j];
      v += __shfl_xor_sync(0xffffffffu, v, 1);
      v += __shfl_xor_sync(0xffffffffu, v, 2);
      if ((u & 3) == 0) rs_a[(u >> 2) + 32 * j] = v;
    }
    asm volatile("bar.sync 1, 128;\n" ::: "memory");

    // ---------------- epilogue ----------------
    const bool ok = wait_or_abort(acc_full, 0, abort_flag, 5);
    __syncwarp();
    tc_fence_after();
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const int64_t m = m0 + row;
    const bool mvalid = ok && !*abort_flag && m < args.M;
    float alpha = 0.f, bp = 0.f;
    if (mvalid) {
      alpha = args.a_scale[m];
      if (ASYM) bp = args.a_zero[m] + 8.f * alpha;
    }
    const int rsa8 = 8 * rs_a[row];
    __half* yrow = reinterpret_cast<__half*>(args.y) + m * args.N;
#pragma unroll 1
    for (int cc = 0; cc < BN / 32; ++cc) {
      uint32_t r[32];
      tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(cc * 32), r);
      tmem_ld_wait();
      if (!mvalid) continue;
#pragma unroll
      for (int g8 = 0; g8 < 4; ++g8) {
        const int64_t n = n0 + cc * 32 + g8 * 8;
        if (n >= args.N) break;
        uint32_t h[4];
        int accs[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int j = cc * 32 + g8 * 8 + e;
          const int S = __float2int_rn(__uint_as_float(r[g8 * 8 + e]) * 262144.0f);
          const int rsw = col_rowsum[j];
          const int acc = S - rsa8 - 8 * rsw;
          accs[e] = acc;
          const float yv = col_scale[j] * fmaf(alpha, (float)acc, bp * (float)rsw);
          if (e & 1) h[e >> 1] = pack_half2_bits(__uint_as_float(h[e >> 1]), yv);
          else h[e >> 1] = __float_as_uint(yv);
        }
        *reinterpret_cast<uint4*>(yrow + n) = make_uint4(h[0], h[1], h[2], h[3]);
        if (ACC_OUT) {
          int4* ap = reinterpret_cast<int4*>(args.acc_out + m * args.N + n);
          ap[0] = make_int4(accs[0], accs[1], accs[2], accs[3]);
          ap[1] = make_int4(accs[4], accs[5], accs[6], accs[7]);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, BN);
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

template <int BN, bool ASYM, bool ACC_OUT>
cudaError_t launch_t(const GemmArgs& a, cudaStream_t stream) {
  CUtensorMap tmA, tmB;
  if (!encode_packed_map(&tmA, a.a_codes, a.M, a.K, BM)) return cudaErrorNotSupported;
  if (!encode_packed_map(&tmB, a.w_codes, a.N, a.K, BN)) return cudaErrorNotSupported;
  auto kern = w4a4_gemm_kernel<BN, ASYM, ACC_OUT>;
  const size_t smem = Layout<BN>::dyn_bytes;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((a.N + BN - 1) / BN), (unsigned)((a.M + BM - 1) / BM));
  kern<<<grid, 256, smem, stream>>>(tmA, tmB, a, (int)(a.K / 128));
  return cudaGetLastError();
}

template <int BN>
cudaError_t launch_bn(const GemmArgs& a, cudaStream_t stream) {
  const bool asym = a.a_zero != nullptr, acc = a.acc_out != nullptr;
  if (asym) return acc ? launch_t<BN, true, true>(a, stream) : launch_t<BN, true, false>(a, stream);
  return acc ? launch_t<BN, false, true>(a, stream) : launch_t<BN, false, false>(a, stream);
}

}  // namespace

cudaError_t launch_w4a4_gemm(const GemmArgs& a, cudaStream_t stream) {
  if (a.M == 0 || a.N == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t tiles256 = ((a.N + 255) / 256) * ((a.M + BM - 1) / BM);
  if (tiles256 >= sms) return launch_bn<256>(a, stream);
  return launch_bn<128>(a, stream);
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
