// spinq_internal.h -- host-side launch interface between the C ABI layer
// (spinq_api.cu) and the kernels.  Every launcher enqueues on `stream`, does
// not synchronize and returns the launch status.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace spinq {

// Small Kronecker factor H_s of order n (n <= 32) as sign bits:
// bit i of neg[ip] is set when H_s[ip][i] == -1.
struct SmallHadamard {
  int n;
  uint32_t neg[32];
};

// Builds H_s for n in {1, 12, 20, 28} (Paley I for n > 1).  Returns false
// for an unsupported order.
bool build_small_hadamard(int n, SmallHadamard* out);

struct RotQuantArgs {
  const void* x;      // fp16 [rows][ldx]
  int64_t rows;
  int64_t K;
  int64_t ldx;
  int n_small;        // 0 = no rotation
  int n_pow2;
  SmallHadamard hs;
  bool symmetric;
  float clip;
  float norm;         // 1/sqrt(K) with a rotation, 1 without (applied to alpha and beta)
  uint8_t* codes;     // [rows][K/2]
  float* scale;       // [rows]
  float* zero;        // [rows] or nullptr
  int32_t* rowsum;    // [rows] or nullptr (weights)
  const uint8_t* signs;  // random signs S of R = S H: bit k set -> x_k negated; nullptr = none
  int* status;           // device status word (set by the launcher of kernels that record time-outs)
  int debug_stall;       // issue no input copies, so the waits run out (tests; 0 normally)
};

cudaError_t launch_rotate_quant_rows(const RotQuantArgs& a, cudaStream_t stream);

// Specialised activation kernels (no rotation, or a power-of-two rotation of
// 512..16384).  Sets *handled = false when the shape has no such kernel.
cudaError_t launch_rotate_quant_act_fast(const RotQuantArgs& a, cudaStream_t stream, bool* handled);

// Activation kernel for a Paley factor (n_small in {12, 20, 28}, n_pow2 in
// {128, 256, 512}).  Sets *handled = false for other shapes.
cudaError_t launch_rotate_quant_act_paley(const RotQuantArgs& a, cudaStream_t stream, bool* handled);

// Rotate+quant on the 5th-generation tensor core (rotate_quant_paley_tc.cu)
// for plain rotations H_s (x) H_P whose block count n_s P / 128 has an
// instance (H_28, H_20, H_12 with P = 512; H_12 with P = 256; Sylvester 8192
// and 16384) and a row count those rows-per-MMA divide into at least one MMA
// per SM; the Paley and power-of-two launchers try it first.  Sets
// *handled = false otherwise.
cudaError_t launch_rotate_quant_act_tc(const RotQuantArgs& a, cudaStream_t stream, bool* handled);
cudaError_t set_wait_limit_rq_tc(uint64_t ns);

struct KVArgs {
  const void* q_in;
  void* q_out;
  const void* k_in;
  const void* v_in;
  int64_t rows_q;     // B*S*Hq
  int64_t rows_kv;    // B*S*Hkv
  int D;
  float clip;
  float norm;         // 1/sqrt(D)
  uint8_t* k_codes;
  float* k_scale;
  float* k_zero;
  uint8_t* v_codes;
  float* v_scale;
  float* v_zero;
  // rotary embedding ahead of R3 (positions == nullptr: none)
  const int32_t* positions;  // [B*S] position of each token
  const float* cos_sin;      // [max_pos][D/2] (cos, sin) pairs
  int64_t max_pos;
  int64_t Hq, Hkv;
};

cudaError_t launch_rotate_quant_kv(const KVArgs& a, cudaStream_t stream);

struct AttnArgs {
  const void* q;            // fp16 [B][Hq][D]
  const uint8_t* k_codes;   // [B][S][Hkv][D/2]
  const float* k_scale;     // [B][S][Hkv]
  const float* k_zero;
  const uint8_t* v_codes;
  const float* v_scale;
  const float* v_zero;
  const int32_t* lens;      // [B] or nullptr (= S)
  int64_t B, S, Hq, Hkv;
  int D;
  float scale;
  void* out;                // fp16 [B][Hq][D]
  float* workspace;
};

// Chunks of the cache length that the decode attention splits over (the
// workspace holds B * Hq * chunks * (D + 2) floats).
int decode_attention_chunks(int64_t B, int64_t S, int64_t Hkv);
cudaError_t launch_decode_attention(const AttnArgs& a, int chunks, cudaStream_t stream);

struct GemmArgs {
  const uint8_t* a_codes;
  const float* a_scale;
  const float* a_zero;   // nullptr = symmetric activations
  const uint8_t* w_codes;
  const float* w_scale;
  const int32_t* w_rowsum;
  int64_t M, N, K;
  void* y;               // fp16 [M][N]
  int32_t* acc_out;      // optional
  int debug_stall;       // prefill kernels: issue no input copies (tests; 0 normally)
};

// Returns cudaErrorNotSupported when the TMA descriptor cannot be encoded.
cudaError_t launch_w4a4_gemm(const GemmArgs& a, cudaStream_t stream);

// Largest M served by the split-K decode kernel.
constexpr int64_t kDecodeMaxM = 256;

// Workspace bytes of launch_w4a4_gemm_splitk for (M, N, K); 0 unless its
// plan splits K (the GEMV kernel, the prefill kernels and unsplit tiles
// write y directly).
int64_t w4a4_gemm_workspace_bytes(int64_t M, int64_t N, int64_t K);
// GEMV kernel for M <= kGemvMaxM tokens (decode; beyond 4 tokens its integer
// dot products cost more than the split-K kernel's latency, measured on
// GB300): each warp owns whole output
// channels and streams their packed weights from global memory.  Sets
// *handled = false when M or the expanded tokens (M K bytes of shared
// memory) are out of its range.
constexpr int64_t kGemvMaxM = 4;
constexpr int64_t kGemvMaxSmem = 160 * 1024;
int64_t w4a4_gemv_smem_bytes(int64_t M, int64_t K);
inline bool w4a4_gemv_fits(int64_t M, int64_t K) {
  return M >= 1 && M <= kGemvMaxM && w4a4_gemv_smem_bytes(M, K) <= kGemvMaxSmem;
}
cudaError_t launch_w4a4_gemv(const GemmArgs& a, cudaStream_t stream, bool* handled);

// Tensor-core GEMV for M <= kGemvTcMaxM tokens: fp16 m16n8k16 MMAs on the
// exact codes, no workspace.  Where w4a4_gemv_tc_streamed(K) holds, warps
// split K and stream the weights straight into registers (one CTA per SM);
// else each CTA owns 16 channels and stages them through shared memory.
// Sets *handled = false when the shape is out of range.
constexpr int64_t kGemvTcMaxM = 16;
inline bool w4a4_gemv_tc_fits(int64_t M, int64_t N, int64_t K) {
  return M >= 1 && M <= kGemvTcMaxM && N >= 16 && N % 16 == 0 && K >= 128 && K % 128 == 0 && K <= 65536 &&
         N / 16 <= 0x7FFFFFFF;
}
cudaError_t launch_w4a4_gemv_tc(const GemmArgs& a, cudaStream_t stream, bool* handled);
// True when the register-streamed form takes K (K / 128 = NKW W with NKW in
// {1, 2, 4, 8} and W <= 16 warps).
bool w4a4_gemv_tc_streamed(int64_t K);

// Decode GEMM for M <= kDecodeMaxM (launch_w4a4_gemm above): the GEMV kernel,
// the split-K kernel or the prefill kernels, as a fitted cost model predicts
// fastest.  `workspace` holds `workspace_bytes` bytes that are zero before
// the call and zero again after it; K is split only when they hold the
// partial sums (M N 4 + 4 ceil(N / 128) bytes), else each tile keeps its
// whole K range.
cudaError_t launch_w4a4_gemm_splitk(const GemmArgs& a, void* workspace, int64_t workspace_bytes,
                                    cudaStream_t stream);

struct CayleyArgs {
  const float* R;     // [batch][n][n]
  const float* grad;  // [batch][n][n] loss gradient
  int64_t batch;
  int n;
  float alpha;
  int iters;
  float* R_out;       // [batch][n][n]
  float* Y_out;       // [batch][n][n] or nullptr
};

// One Cayley SGD step per rotation (n in {16, 32, 64, 128}); returns
// cudaErrorNotSupported for other n.
cudaError_t launch_cayley_step(const CayleyArgs& a, cudaStream_t stream);

// Code formats of the 8-bit quantizers (spinq_code_format in spinq.h).
constexpr int kFmtInt8Planes = 1;
constexpr int kFmtE4M3 = 2;
constexpr int kFmtInt4Bytes = 3;

struct Rq8Args {
  const void* x;      // fp16 [rows][ldx]
  int64_t rows, K, ldx;
  int n_small;        // 0 = no rotation
  int n_pow2;
  SmallHadamard hs;
  int format;         // kFmt*
  bool symmetric;
  float clip;
  float norm;         // 1/sqrt(K) with a rotation, else 1
  uint8_t* codes;     // [rows][2K] (int8 planes) or [rows][K]
  float* scale;       // [rows]
  float* zero;        // [rows] (asymmetric int8) or nullptr
  int32_t* rowsum;    // [rows] (int4 bytes) or nullptr
};

cudaError_t launch_rotate_quant_8bit(const Rq8Args& a, cudaStream_t stream);
// The 8-bit quantizers (int8 planes, E4M3; unclipped) on a Paley rotation,
// in the Paley rotate+quant kernel.  Sets *handled = false for other shapes.
cudaError_t launch_rotate_quant_8bit_paley(const Rq8Args& a, cudaStream_t stream, bool* handled);
// The FP8 quantizer (kFmtE4M3, symmetric, unclipped) on the tcgen05
// rotate+quant kernel, for H_28 (x) H_512 with at least one row per SM
// (rotate_quant_paley_tc.cu).  Sets *handled = false for other requests.
cudaError_t launch_rotate_quant_8bit_tc(const RotQuantArgs& a, int format, cudaStream_t stream, bool* handled);

struct Fp8GemmArgs {
  bool w4a8;              // false: FP8 x FP8; true: W4A8 (activation planes [M][2K])
  const uint8_t* a_codes; // E4M3 bytes [M][K] (FP8) or [M][2K] (W4A8 planes)
  const float* a_scale;   // [M]
  const float* a_zero;    // [M] (W4A8 asymmetric) or nullptr
  const uint8_t* w_codes; // E4M3 bytes [N][K]
  const float* w_scale;   // [N]
  const int32_t* w_rowsum;// [N] (W4A8) or nullptr
  int64_t M, N, K;
  void* y;                // fp16 [M][N]
  int32_t* acc_out;       // W4A8 only, optional
};

// 8-bit linears on the E4M3 pipe; cudaErrorNotSupported when a tensor map
// cannot be encoded.
cudaError_t launch_fp8_gemm(const Fp8GemmArgs& a, cudaStream_t stream);

// Launches of the Paley rotate+quant, W4A4 prefill and FP8 GEMM kernels still
// to issue no input copies (spinq_debug_stall_launches); take_debug_stall()
// consumes one.
bool take_debug_stall();

// Limit of the ordinary bounded waits of the Paley rotate+quant, W4A4 and
// FP8 GEMM kernels (2 s by default; lowered only by tests).
cudaError_t set_wait_limit_paley(uint64_t ns);
cudaError_t set_wait_limit_gemm(uint64_t ns);
cudaError_t set_wait_limit_fp8(uint64_t ns);

// Device status word written by bounded waits that gave up.
cudaError_t read_and_clear_device_status(int32_t* code, int32_t* detail);
// Its device address (two ints: code, wait site), for kernels in other
// translation units; null if it cannot be resolved.
int* device_status_word();
// Prefill GEMM on SM pairs (tcgen05 cta_group::2, 256 x 256 tiles).  Sets
// *handled = false when the shape or device cannot take it.
cudaError_t launch_w4a4_gemm_pair(const GemmArgs& a, cudaStream_t stream, bool* handled);
// SM pairs the pair kernel can keep resident at once (0 if none).
int w4a4_gemm_pair_clusters();
// Prefill kernel selection (spinq_gemm_kernel values); returns the previous one.
int w4a4_gemm_select(int kernel);
// Process-wide fixed count of the split-K kernel's K slices (0: the cost
// model picks).
int w4a4_gemm_split_k(int n);
// The prefill kernel (SPINQ_GEMM_TILE128 / TILE256 / PAIR) launch_w4a4_gemm
// runs for this shape on the current device.
int plan_w4a4_gemm(int64_t M, int64_t N, int64_t K);
// The kernel launch_w4a4_gemm_splitk runs with a full workspace:
// SPINQ_GEMM_SPLITK with its K slices in *nsplit, or another SPINQ_GEMM_*
// kernel (*nsplit = 0).
int plan_w4a4_gemm_splitk(int64_t M, int64_t N, int64_t K, int* nsplit);

}  // namespace spinq
