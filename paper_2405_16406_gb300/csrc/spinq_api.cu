// spinq_api.cu -- the extern "C" entry points declared in include/spinq.h:
// host-side argument validation, status codes and kernel dispatch.  No entry
// point allocates memory or synchronizes (except spinq_device_status, which
// documents that it does).
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>

#include "../../include/spinq.h"
#include "spinq_internal.h"

using namespace spinq;

namespace spinq {
std::atomic<int> g_fail_launches{0};
static std::atomic<int> g_debug_stall{0};
bool take_debug_stall() {
  return g_debug_stall.load(std::memory_order_relaxed) > 0 && g_debug_stall.fetch_sub(1) > 0;
}
}

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool is_pow2(int64_t v) { return v > 0 && (v & (v - 1)) == 0; }

spinq_status from_cuda(cudaError_t e) {
  if (e == cudaSuccess) return SPINQ_OK;
  if (e == cudaErrorNotSupported) return SPINQ_EUNSUPPORTED;
  return SPINQ_ECUDA;
}

bool clip_ok(float c) { return c > 0.f && c <= 1.f; }

// Validates a Hadamard spec for a rotated dimension of size `dim` and fills
// the small-factor table.  Returns SPINQ_OK, SPINQ_EINVAL or SPINQ_EUNSUPPORTED.
spinq_status check_had(const spinq_had_cfg* had, int64_t dim, SmallHadamard* hs) {
  if (had->n_small < 1 || had->n_pow2 < 1 || !is_pow2(had->n_pow2)) return SPINQ_EINVAL;
  if ((int64_t)had->n_small * had->n_pow2 != dim) return SPINQ_EINVAL;
  if (!build_small_hadamard(had->n_small, hs)) return SPINQ_EUNSUPPORTED;
  if (had->n_pow2 > 16384) return SPINQ_EUNSUPPORTED;
  return SPINQ_OK;
}

}  // namespace

extern "C" {

const char* spinq_status_string(spinq_status s) {
  switch (s) {
    case SPINQ_OK: return "SPINQ_OK";
    case SPINQ_EINVAL: return "SPINQ_EINVAL: invalid argument";
    case SPINQ_EUNSUPPORTED: return "SPINQ_EUNSUPPORTED: no kernel for this configuration";
    case SPINQ_ECUDA: return "SPINQ_ECUDA: CUDA launch or runtime error";
    case SPINQ_ETIMEOUT: return "SPINQ_ETIMEOUT: a bounded device wait gave up";
    case SPINQ_ESCRATCH:
      return "SPINQ_ESCRATCH: the request needs more workspace than the no-allocation entry point's "
             "fixed array holds";
  }
  return "SPINQ: unknown status";
}

const char* spinq_version(void) { return "spinq-gb300 sm_103a 0.1"; }

static spinq_status rqa(const void* x_f16, int64_t M, int64_t K, int64_t ldx, const spinq_had_cfg* had,
                        const uint8_t* signs, const spinq_quant_cfg* q, uint8_t* codes, float* scale, float* zero,
                        void* stream) {
  if (!q || M < 0 || K <= 0 || ldx < K) return SPINQ_EINVAL;
  if (signs && !had) return SPINQ_EINVAL;
  if (M > 0 && (!x_f16 || !codes || !scale)) return SPINQ_EINVAL;
  if (!clip_ok(q->clip_ratio)) return SPINQ_EINVAL;
  if (q->symmetric != 0 && q->symmetric != 1) return SPINQ_EINVAL;
  if (!q->symmetric && M > 0 && !zero) return SPINQ_EINVAL;
  if (K % 32 != 0 || ldx % 8 != 0 || !aligned16(x_f16) || !aligned16(codes)) return SPINQ_EINVAL;
  if (q->bits != 4 || q->granularity != SPINQ_PER_TOKEN) return SPINQ_EUNSUPPORTED;
  if (K > 32768) return SPINQ_EUNSUPPORTED;
  RotQuantArgs a{};
  if (had) {
    spinq_status st = check_had(had, K, &a.hs);
    if (st != SPINQ_OK) return st;
    a.n_small = had->n_small;
    a.n_pow2 = had->n_pow2;
    a.norm = (float)(1.0 / std::sqrt((double)K));
  } else {
    a.n_small = 0;
    a.n_pow2 = 1;
    a.norm = 1.f;
  }
  if (M == 0) return SPINQ_OK;
  a.x = x_f16;
  a.rows = M;
  a.K = K;
  a.ldx = ldx;
  a.symmetric = q->symmetric != 0;
  a.clip = q->clip_ratio;
  a.codes = codes;
  a.scale = scale;
  a.zero = q->symmetric ? nullptr : zero;
  a.rowsum = nullptr;
  a.signs = signs;
  return from_cuda(launch_rotate_quant_rows(a, static_cast<cudaStream_t>(stream)));
}

spinq_status spinq_rotate_quant_act(const void* x_f16, int64_t M, int64_t K, int64_t ldx,
                                    const spinq_had_cfg* had, const spinq_quant_cfg* q,
                                    uint8_t* codes, float* scale, float* zero, void* stream) {
  return rqa(x_f16, M, K, ldx, had, nullptr, q, codes, scale, zero, stream);
}

spinq_status spinq_rotate_quant_act_signed(const void* x_f16, int64_t M, int64_t K, int64_t ldx,
                                           const spinq_had_cfg* had, const uint8_t* signs,
                                           const spinq_quant_cfg* q, uint8_t* codes, float* scale, float* zero,
                                           void* stream) {
  if (!signs || !had) return SPINQ_EINVAL;
  return rqa(x_f16, M, K, ldx, had, signs, q, codes, scale, zero, stream);
}

static spinq_status qw(const void* w_f16, int64_t N, int64_t K, const spinq_had_cfg* had, const uint8_t* signs,
                       const spinq_quant_cfg* q, uint8_t* codes, float* scale, int32_t* rowsum, void* stream) {
  if (!q || N < 0 || K <= 0) return SPINQ_EINVAL;
  if (signs && !had) return SPINQ_EINVAL;
  if (N > 0 && (!w_f16 || !codes || !scale || !rowsum)) return SPINQ_EINVAL;
  if (!clip_ok(q->clip_ratio)) return SPINQ_EINVAL;
  if (K % 32 != 0 || !aligned16(w_f16) || !aligned16(codes)) return SPINQ_EINVAL;
  if (q->bits != 4 || q->symmetric != 1 || q->granularity != SPINQ_PER_CHANNEL) return SPINQ_EUNSUPPORTED;
  if (K > 32768) return SPINQ_EUNSUPPORTED;
  RotQuantArgs a{};
  if (had) {
    spinq_status st = check_had(had, K, &a.hs);
    if (st != SPINQ_OK) return st;
    a.n_small = had->n_small;
    a.n_pow2 = had->n_pow2;
    a.norm = (float)(1.0 / std::sqrt((double)K));
  } else {
    a.n_small = 0;
    a.n_pow2 = 1;
    a.norm = 1.f;
  }
  if (N == 0) return SPINQ_OK;
  a.x = w_f16;
  a.rows = N;
  a.K = K;
  a.ldx = K;
  a.symmetric = true;
  a.clip = q->clip_ratio;
  a.codes = codes;
  a.scale = scale;
  a.zero = nullptr;
  a.rowsum = rowsum;
  a.signs = signs;
  return from_cuda(launch_rotate_quant_rows(a, static_cast<cudaStream_t>(stream)));
}

spinq_status spinq_quant_weight(const void* w_f16, int64_t N, int64_t K, const spinq_had_cfg* had,
                                const spinq_quant_cfg* q, uint8_t* codes, float* scale,
                                int32_t* rowsum, void* stream) {
  return qw(w_f16, N, K, had, nullptr, q, codes, scale, rowsum, stream);
}

spinq_status spinq_quant_weight_signed(const void* w_f16, int64_t N, int64_t K, const spinq_had_cfg* had,
                                       const uint8_t* signs, const spinq_quant_cfg* q, uint8_t* codes,
                                       float* scale, int32_t* rowsum, void* stream) {
  if (!signs || !had) return SPINQ_EINVAL;
  return qw(w_f16, N, K, had, signs, q, codes, scale, rowsum, stream);
}

// bytes of the codes / alpha / beta hand-off of spinq_rotated_linear, each
// part 256-byte aligned
static int64_t align256(int64_t v) { return (v + 255) / 256 * 256; }

int64_t spinq_rotated_linear_workspace_bytes(int64_t M, int64_t K) {
  if (M <= 0 || K <= 0) return 0;
  return align256(M * (K / 2)) + 2 * align256(M * 4);
}

spinq_status spinq_rotated_linear(const void* x_f16, int64_t M, int64_t K, int64_t ldx, const spinq_had_cfg* had,
                                  const uint8_t* signs, const spinq_quant_cfg* q, const uint8_t* w_codes,
                                  const float* w_scale, const int32_t* w_rowsum, int64_t N, void* y_f16,
                                  void* workspace, int64_t workspace_bytes, void* stream) {
  if (!q || M < 0 || N < 0 || K <= 0) return SPINQ_EINVAL;
  const int64_t need = spinq_rotated_linear_workspace_bytes(M, K);
  if (M > 0 && (!workspace || !aligned16(workspace) || workspace_bytes < need)) return SPINQ_EINVAL;
  if (K % 128 != 0 || N % 16 != 0) return SPINQ_EINVAL;
  if (M > 0 && N > 0 && (!w_codes || !w_scale || !w_rowsum || !y_f16)) return SPINQ_EINVAL;
  if (M == 0 || N == 0) return SPINQ_OK;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  uint8_t* codes = ws;
  float* alpha = reinterpret_cast<float*>(ws + align256(M * (K / 2)));
  float* beta = reinterpret_cast<float*>(ws + align256(M * (K / 2)) + align256(M * 4));
  spinq_status st = rqa(x_f16, M, K, ldx, had, signs, q, codes, alpha, beta, stream);
  if (st != SPINQ_OK) return st;
  return spinq_w4a4_gemm(codes, alpha, q->symmetric ? nullptr : beta, w_codes, w_scale, w_rowsum, M, N, K, y_f16,
                         nullptr, stream);
}

spinq_status spinq_w4a4_gemm(const uint8_t* a_codes, const float* a_scale, const float* a_zero,
                             const uint8_t* w_codes, const float* w_scale,
                             const int32_t* w_rowsum, int64_t M, int64_t N, int64_t K,
                             void* y_f16, int32_t* acc_out, void* stream) {
  if (M < 0 || N < 0 || K <= 0) return SPINQ_EINVAL;
  if (M > 0 && N > 0 && (!a_codes || !a_scale || !w_codes || !w_scale || !w_rowsum || !y_f16))
    return SPINQ_EINVAL;
  if (K % 128 != 0 || N % 16 != 0) return SPINQ_EINVAL;
  if (!aligned16(a_codes) || !aligned16(w_codes) || !aligned16(y_f16) || !aligned16(w_scale) ||
      !aligned16(w_rowsum) || (acc_out && !aligned16(acc_out)))
    return SPINQ_EINVAL;
  if (K > 65536 || M > INT32_MAX || N > INT32_MAX) return SPINQ_EUNSUPPORTED;
  if (M == 0 || N == 0) return SPINQ_OK;
  GemmArgs g{a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y_f16, acc_out};
  return from_cuda(launch_w4a4_gemm(g, static_cast<cudaStream_t>(stream)));
}

int64_t spinq_w4a4_gemm_workspace_bytes(int64_t M, int64_t N, int64_t K) {
  return w4a4_gemm_workspace_bytes(M, N, K);
}

spinq_status spinq_w4a4_gemm_splitk(const uint8_t* a_codes, const float* a_scale, const float* a_zero,
                                    const uint8_t* w_codes, const float* w_scale,
                                    const int32_t* w_rowsum, int64_t M, int64_t N, int64_t K,
                                    void* y_f16, int32_t* acc_out, void* workspace,
                                    int64_t workspace_bytes, void* stream) {
  if (M < 0 || N < 0 || K <= 0) return SPINQ_EINVAL;
  if (M > 0 && N > 0 && (!a_codes || !a_scale || !w_codes || !w_scale || !w_rowsum || !y_f16))
    return SPINQ_EINVAL;
  if (K % 128 != 0 || N % 16 != 0) return SPINQ_EINVAL;
  if (!aligned16(a_codes) || !aligned16(w_codes) || !aligned16(y_f16) || !aligned16(w_scale) ||
      !aligned16(w_rowsum) || (acc_out && !aligned16(acc_out)))
    return SPINQ_EINVAL;
  const int64_t need = w4a4_gemm_workspace_bytes(M, N, K);
  if (need > 0 && (!workspace || !aligned16(workspace) || workspace_bytes < need)) return SPINQ_EINVAL;
  if (K > 65536 || M > INT32_MAX || N > INT32_MAX) return SPINQ_EUNSUPPORTED;
  if (M == 0 || N == 0) return SPINQ_OK;
  GemmArgs g{a_codes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y_f16, acc_out};
  return from_cuda(launch_w4a4_gemm_splitk(g, workspace, workspace_bytes, static_cast<cudaStream_t>(stream)));
}

spinq_status spinq_rotate_quant_kv(const void* q_in, void* q_out, const void* k_in,
                                   const void* v_in, int64_t B, int64_t S, int64_t Hq,
                                   int64_t Hkv, int64_t D, const spinq_had_cfg* had,
                                   const spinq_quant_cfg* kvq, uint8_t* k_codes, float* k_scale,
                                   float* k_zero, uint8_t* v_codes, float* v_scale,
                                   float* v_zero, void* stream) {
  if (!had || !kvq || B < 0 || S < 0 || Hq < 0 || Hkv < 0 || D <= 0) return SPINQ_EINVAL;
  const int64_t rows_q = B * S * Hq, rows_kv = B * S * Hkv;
  if (rows_q > 0 && (!q_in || !q_out)) return SPINQ_EINVAL;
  if (rows_kv > 0 && (!k_in || !v_in || !k_codes || !k_scale || !k_zero || !v_codes || !v_scale || !v_zero))
    return SPINQ_EINVAL;
  if (!clip_ok(kvq->clip_ratio)) return SPINQ_EINVAL;
  if (had->n_small != 1 || had->n_pow2 != D) return SPINQ_EINVAL;
  for (const void* p : {q_in, (const void*)q_out, k_in, v_in, (const void*)k_codes, (const void*)v_codes})
    if (p && !aligned16(p)) return SPINQ_EINVAL;
  if (kvq->bits != 4 || kvq->symmetric != 0 || kvq->granularity != SPINQ_PER_GROUP || kvq->group_size != D)
    return SPINQ_EUNSUPPORTED;
  if (D != 64 && D != 128) return SPINQ_EUNSUPPORTED;
  if (rows_q == 0 && rows_kv == 0) return SPINQ_OK;
  KVArgs a{q_in, q_out, k_in, v_in, rows_q, rows_kv, (int)D, kvq->clip_ratio,
           (float)(1.0 / std::sqrt((double)D)), k_codes, k_scale, k_zero, v_codes, v_scale, v_zero};
  return from_cuda(launch_rotate_quant_kv(a, static_cast<cudaStream_t>(stream)));
}

spinq_status spinq_cayley_step(const float* R, const float* grad, int64_t batch, int64_t n, float alpha,
                               int32_t iters, float* R_out, float* Y_out, void* stream) {
  if (batch < 0 || n <= 0 || iters < 0 || iters > 64 || !std::isfinite(alpha)) return SPINQ_EINVAL;
  if (batch > 0 && (!R || !grad || !R_out)) return SPINQ_EINVAL;
  for (const void* p : {(const void*)R, (const void*)grad, (const void*)R_out, (const void*)Y_out})
    if (p && !aligned16(p)) return SPINQ_EINVAL;
  if (n != 16 && n != 32 && n != 64 && n != 128) return SPINQ_EUNSUPPORTED;
  if (batch > INT32_MAX) return SPINQ_EUNSUPPORTED;
  if (batch == 0) return SPINQ_OK;
  CayleyArgs a{R, grad, batch, (int)n, alpha, (int)iters, R_out, Y_out};
  return from_cuda(launch_cayley_step(a, static_cast<cudaStream_t>(stream)));
}

static spinq_status rq8(const void* x, int64_t rows, int64_t K, int64_t ldx, const spinq_had_cfg* had,
                        const spinq_quant_cfg* q, int format, bool weights, uint8_t* codes, float* scale,
                        float* zero, int32_t* rowsum, void* stream) {
  if (!q || rows < 0 || K <= 0 || ldx < K) return SPINQ_EINVAL;
  if (rows > 0 && (!x || !codes || !scale)) return SPINQ_EINVAL;
  if (!clip_ok(q->clip_ratio)) return SPINQ_EINVAL;
  if (q->symmetric != 0 && q->symmetric != 1) return SPINQ_EINVAL;
  if (K % 128 != 0 || ldx % 8 != 0 || !aligned16(x) || !aligned16(codes)) return SPINQ_EINVAL;
  const bool act = !weights;
  if (act && format != SPINQ_FMT_INT8_PLANES && format != SPINQ_FMT_E4M3) return SPINQ_EINVAL;
  if (weights && format != SPINQ_FMT_E4M3 && format != SPINQ_FMT_INT4_BYTES) return SPINQ_EINVAL;
  if (act && !q->symmetric && format == SPINQ_FMT_INT8_PLANES && rows > 0 && !zero) return SPINQ_EINVAL;
  if (weights && format == SPINQ_FMT_INT4_BYTES && rows > 0 && !rowsum) return SPINQ_EINVAL;
  const int want_bits = format == SPINQ_FMT_INT4_BYTES ? 4 : 8;
  const int want_gran = weights ? SPINQ_PER_CHANNEL : SPINQ_PER_TOKEN;
  if (q->bits != want_bits || q->granularity != want_gran) return SPINQ_EUNSUPPORTED;
  if (format != SPINQ_FMT_INT8_PLANES && !q->symmetric) return SPINQ_EUNSUPPORTED;
  if (K > 32768) return SPINQ_EUNSUPPORTED;
  Rq8Args a{};
  if (had) {
    spinq_status st = check_had(had, K, &a.hs);
    if (st != SPINQ_OK) return st;
    a.n_small = had->n_small;
    a.n_pow2 = had->n_pow2;
    a.norm = (float)(1.0 / std::sqrt((double)K));
  } else {
    a.n_small = 0;
    a.n_pow2 = 1;
    a.norm = 1.f;
  }
  if (rows == 0) return SPINQ_OK;
  a.x = x;
  a.rows = rows;
  a.K = K;
  a.ldx = ldx;
  a.format = format;
  a.symmetric = q->symmetric != 0;
  a.clip = q->clip_ratio;
  a.codes = codes;
  a.scale = scale;
  a.zero = a.symmetric ? nullptr : zero;
  a.rowsum = rowsum;
  return from_cuda(launch_rotate_quant_8bit(a, static_cast<cudaStream_t>(stream)));
}

spinq_status spinq_rotate_quant_act8(const void* x_f16, int64_t M, int64_t K, int64_t ldx, const spinq_had_cfg* had,
                                     const spinq_quant_cfg* q, int32_t format, uint8_t* codes, float* scale,
                                     float* zero, void* stream) {
  return rq8(x_f16, M, K, ldx, had, q, format, false, codes, scale, zero, nullptr, stream);
}

spinq_status spinq_quant_weight8(const void* w_f16, int64_t N, int64_t K, const spinq_had_cfg* had,
                                 const spinq_quant_cfg* q, int32_t format, uint8_t* codes, float* scale,
                                 int32_t* rowsum, void* stream) {
  return rq8(w_f16, N, K, K, had, q, format, true, codes, scale, nullptr, rowsum, stream);
}

static spinq_status gemm8(bool w4a8, const uint8_t* a_codes, const float* a_scale, const float* a_zero,
                          const uint8_t* w_codes, const float* w_scale, const int32_t* w_rowsum, int64_t M,
                          int64_t N, int64_t K, void* y_f16, int32_t* acc_out, void* stream) {
  if (M < 0 || N < 0 || K <= 0) return SPINQ_EINVAL;
  if (M > 0 && N > 0 && (!a_codes || !a_scale || !w_codes || !w_scale || !y_f16 || (w4a8 && !w_rowsum)))
    return SPINQ_EINVAL;
  if (K % 128 != 0 || N % 16 != 0) return SPINQ_EINVAL;
  for (const void* p : {(const void*)a_codes, (const void*)w_codes, (const void*)y_f16, (const void*)acc_out})
    if (p && !aligned16(p)) return SPINQ_EINVAL;
  if (M > INT32_MAX || N > INT32_MAX || K > (w4a8 ? 16384 : 65536)) return SPINQ_EUNSUPPORTED;
  if (M == 0 || N == 0) return SPINQ_OK;
  Fp8GemmArgs g{w4a8, a_codes, a_scale, w4a8 ? a_zero : nullptr, w_codes, w_scale, w4a8 ? w_rowsum : nullptr,
                M, N, K, y_f16, w4a8 ? acc_out : nullptr};
  return from_cuda(launch_fp8_gemm(g, static_cast<cudaStream_t>(stream)));
}

spinq_status spinq_fp8_gemm(const uint8_t* a_codes, const float* a_scale, const uint8_t* w_codes,
                            const float* w_scale, int64_t M, int64_t N, int64_t K, void* y_f16, void* stream) {
  return gemm8(false, a_codes, a_scale, nullptr, w_codes, w_scale, nullptr, M, N, K, y_f16, nullptr, stream);
}

spinq_status spinq_w4a8_gemm(const uint8_t* a_planes, const float* a_scale, const float* a_zero,
                             const uint8_t* w_codes, const float* w_scale, const int32_t* w_rowsum, int64_t M,
                             int64_t N, int64_t K, void* y_f16, int32_t* acc_out, void* stream) {
  return gemm8(true, a_planes, a_scale, a_zero, w_codes, w_scale, w_rowsum, M, N, K, y_f16, acc_out, stream);
}

spinq_status spinq_rope_rotate_quant_kv(const void* q_in, void* q_out, const void* k_in, const void* v_in,
                                        const int32_t* positions, const float* cos_sin, int64_t max_pos, int64_t B,
                                        int64_t S, int64_t Hq, int64_t Hkv, int64_t D, const spinq_had_cfg* had,
                                        const spinq_quant_cfg* kvq, uint8_t* k_codes, float* k_scale,
                                        float* k_zero, uint8_t* v_codes, float* v_scale, float* v_zero,
                                        void* stream) {
  if (B * S > 0 && (!positions || !cos_sin || max_pos <= 0)) return SPINQ_EINVAL;
  if (cos_sin && !aligned16(cos_sin)) return SPINQ_EINVAL;
  if (!had || !kvq || B < 0 || S < 0 || Hq < 0 || Hkv < 0 || D <= 0) return SPINQ_EINVAL;
  const int64_t rows_q = B * S * Hq, rows_kv = B * S * Hkv;
  if (rows_q > 0 && (!q_in || !q_out)) return SPINQ_EINVAL;
  if (rows_kv > 0 && (!k_in || !v_in || !k_codes || !k_scale || !k_zero || !v_codes || !v_scale || !v_zero))
    return SPINQ_EINVAL;
  if (!clip_ok(kvq->clip_ratio)) return SPINQ_EINVAL;
  if (had->n_small != 1 || had->n_pow2 != D) return SPINQ_EINVAL;
  for (const void* p : {q_in, (const void*)q_out, k_in, v_in, (const void*)k_codes, (const void*)v_codes})
    if (p && !aligned16(p)) return SPINQ_EINVAL;
  if (kvq->bits != 4 || kvq->symmetric != 0 || kvq->granularity != SPINQ_PER_GROUP || kvq->group_size != D)
    return SPINQ_EUNSUPPORTED;
  if (D != 64 && D != 128) return SPINQ_EUNSUPPORTED;
  if (rows_q == 0 && rows_kv == 0) return SPINQ_OK;
  KVArgs a{q_in, q_out, k_in, v_in, rows_q, rows_kv, (int)D, kvq->clip_ratio,
           (float)(1.0 / std::sqrt((double)D)), k_codes, k_scale, k_zero, v_codes, v_scale, v_zero,
           positions, cos_sin, max_pos, Hq, Hkv};
  return from_cuda(launch_rotate_quant_kv(a, static_cast<cudaStream_t>(stream)));
}

int64_t spinq_decode_attention_workspace_bytes(int64_t B, int64_t S, int64_t Hq, int64_t Hkv, int64_t D) {
  if (B <= 0 || S <= 0 || Hq <= 0 || Hkv <= 0 || D <= 0) return 0;
  return B * Hq * (int64_t)decode_attention_chunks(B, S, Hkv) * (D + 2) * 4;
}

spinq_status spinq_decode_attention_kv4(const void* q, const uint8_t* k_codes, const float* k_scale,
                                        const float* k_zero, const uint8_t* v_codes, const float* v_scale,
                                        const float* v_zero, const int32_t* lens, int64_t B, int64_t S, int64_t Hq,
                                        int64_t Hkv, int64_t D, float softmax_scale, void* out, void* workspace,
                                        int64_t workspace_bytes, void* stream) {
  if (B < 0 || S <= 0 || Hq <= 0 || Hkv <= 0 || D <= 0 || !std::isfinite(softmax_scale)) return SPINQ_EINVAL;
  if (Hq % Hkv != 0) return SPINQ_EINVAL;
  if (B > 0 && (!q || !k_codes || !k_scale || !k_zero || !v_codes || !v_scale || !v_zero || !out)) return SPINQ_EINVAL;
  const int64_t need = spinq_decode_attention_workspace_bytes(B, S, Hq, Hkv, D);
  if (B > 0 && (!workspace || !aligned16(workspace) || workspace_bytes < need)) return SPINQ_EINVAL;
  for (const void* p : {q, (const void*)k_codes, (const void*)v_codes, (const void*)out})
    if (p && !aligned16(p)) return SPINQ_EINVAL;
  const int64_t G = Hq / Hkv;
  if ((D != 64 && D != 128) || (G != 1 && G != 2 && G != 4 && G != 8)) return SPINQ_EUNSUPPORTED;
  if (B > 65535 || Hkv > 65535 || S > INT32_MAX) return SPINQ_EUNSUPPORTED;
  if (S * Hkv * (D / 2) > INT32_MAX) return SPINQ_EUNSUPPORTED;   // one batch's cache within 2 GiB
  if (B == 0) return SPINQ_OK;
  AttnArgs a{q, k_codes, k_scale, k_zero, v_codes, v_scale, v_zero, lens, B, S, Hq, Hkv, (int)D, softmax_scale,
             out, static_cast<float*>(workspace)};
  return from_cuda(launch_decode_attention(a, decode_attention_chunks(B, S, Hkv), static_cast<cudaStream_t>(stream)));
}

spinq_status spinq_debug_set_wait_limit_ns(int64_t ns) {
  if (ns <= 0) return SPINQ_EINVAL;
  const uint64_t v = (uint64_t)ns;
  if (set_wait_limit_paley(v) != cudaSuccess || set_wait_limit_gemm(v) != cudaSuccess ||
      set_wait_limit_fp8(v) != cudaSuccess)
    return SPINQ_ECUDA;
  return SPINQ_OK;
}

int spinq_debug_stall_launches(int n) {
  if (n < 0) return -1;
  return g_debug_stall.exchange(n);
}

int spinq_debug_fail_launches(int n) {
  if (n < 0) return -1;
  return g_fail_launches.exchange(n);
}

int spinq_gemm_select_kernel(int kernel) { return w4a4_gemm_select(kernel); }

int spinq_gemm_split_k(int n) { return w4a4_gemm_split_k(n); }

int spinq_w4a4_gemm_plan(int64_t M, int64_t N, int64_t K) {
  if (M <= 0 || N <= 0 || K <= 0 || K % 128 != 0 || N % 16 != 0) return -1;
  return plan_w4a4_gemm(M, N, K);
}

int spinq_w4a4_gemm_splitk_plan(int64_t M, int64_t N, int64_t K, int* nsplit) {
  if (nsplit) *nsplit = 0;
  if (M <= 0 || N <= 0 || K <= 0 || K % 128 != 0 || N % 16 != 0 || K > 65536) return -1;
  int ns = 0;
  const int kind = plan_w4a4_gemm_splitk(M, N, K, &ns);
  if (nsplit) *nsplit = ns;
  return kind;
}

spinq_status spinq_device_status(int32_t* detail) {
  int32_t code = 0, d = 0;
  if (read_and_clear_device_status(&code, &d) != cudaSuccess) return SPINQ_ECUDA;
  if (detail) *detail = d;
  return static_cast<spinq_status>(code);
}

}  // extern "C"
