/*
 * spinq.h -- C ABI of the GB300 (sm_103a) rotated W4A4 hot path of SpinQuant
 * (arXiv 2405.16406).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * Pointers.  Every data pointer is a DEVICE pointer owned by the caller; the
 *   library never allocates, frees or keeps a pointer after the call returns.
 *   One exception: spinq_w4a4_gemm_noalloc keeps its workspace in a fixed
 *   device array of SPINQ_NOALLOC_SCRATCH_BYTES that the library owns (held
 *   by every GPU that loads the library until the process exits) and caches
 *   that array's device address per CUDA context.
 *   `stream` is a cudaStream_t (NULL = the legacy default stream).  Every
 *   call is asynchronous: it validates its arguments on the host, enqueues
 *   kernels on `stream` and returns; it never synchronizes.
 * Layouts.  Row-major, the reduction dimension K (or head_dim D) contiguous.
 *   4-bit codes are packed two per byte, the even index in the LOW nibble.
 *   Symmetric codes are two's complement nibbles in [-8, 7]; asymmetric codes
 *   are unsigned nibbles in [0, 15].  Scales and zeros are fp32.
 * Rotation.  A Hadamard spec {n_small, n_pow2} names R = (H_s (x) H_P)/sqrt(K)
 *   with K = n_small * n_pow2, H_P the natural-order Sylvester matrix of order
 *   n_pow2 and H_s the small factor of order n_small: [1] for n_small = 1, else
 *   the Paley I matrix of order n_small (n_small - 1 = q, a prime power with
 *   q = 3 mod 4; GF(q) = integers mod q for prime q, GF(27) =
 *   GF(3)[t]/(t^3 + 2t + 1) with element i = c0 + 3 c1 + 9 c2 <-> c0 + c1 t +
 *   c2 t^2; H_s = I + S, S = [[0, 1..1], [-1.., Q]], Q[i][j] = chi(a_i - a_j)).
 *   The small factor acts on the slow index (element k = i * n_pow2 + j) and
 *   activations are rotated as row vectors: x' = x R (Sec. 3.1, R3 and R4;
 *   Sec. 2.2 footnote for the Hadamard scaling).
 * Quantizer.  Eq. 1 (Sec. 2): symmetric alpha = clip * max|x| / (2^(N-1)-1),
 *   beta = 0, q = clamp(rint(x/alpha), -2^(N-1), 2^(N-1)-1); asymmetric
 *   alpha = clip * (max x - min x) / (2^N - 1), beta = clip * min x,
 *   u = clamp(rint((x - beta)/alpha), 0, 2^N - 1); a zero range stores
 *   alpha = 0 and codes 0.  rint is round-half-to-even.  The clipping ratio
 *   follows the appendix "Quantization choice".  Only N = 4 has kernels.
 * Errors.  Invalid arguments return SPINQ_EINVAL before any launch (NULL
 *   required pointer, non-positive or inconsistent size, K not even, a
 *   pointer not 16-byte aligned where noted, clip_ratio outside (0, 1]).
 *   A valid request with no compiled kernel (bits != 4, an unsupported
 *   Hadamard order or granularity) returns SPINQ_EUNSUPPORTED.  A failed
 *   launch returns SPINQ_ECUDA.  Device-side waits in the GEMM are bounded;
 *   a wait that gives up records SPINQ_ETIMEOUT in a device status word that
 *   spinq_device_status() reads back.
 */
#ifndef SPINQ_H_
#define SPINQ_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SPINQ_OK = 0,
  SPINQ_EINVAL = 1,
  SPINQ_EUNSUPPORTED = 2,
  SPINQ_ECUDA = 3,
  SPINQ_ETIMEOUT = 4,
  SPINQ_ESCRATCH = 5  /* spinq_w4a4_gemm_noalloc: the request needs more
                         workspace than its fixed array holds */
} spinq_status;

typedef enum {
  SPINQ_PER_TOKEN = 0,   /* one (alpha, beta) per row of activations      */
  SPINQ_PER_CHANNEL = 1, /* one scale per output channel (row) of weights */
  SPINQ_PER_GROUP = 2    /* one (alpha, beta) per group of group_size     */
} spinq_gran;

/* Quantizer of Eq. 1: bit width N, symmetric (1) or asymmetric (0),
 * granularity, group size (PER_GROUP only) and clipping ratio in (0, 1]. */
typedef struct {
  int32_t bits;
  int32_t symmetric;
  int32_t granularity;
  int32_t group_size;
  float clip_ratio;
} spinq_quant_cfg;

/* Online Hadamard of size n_small * n_pow2 (Sec. 3.1, R3/R4). */
typedef struct {
  int32_t n_small; /* 1, 12, 20 or 28 */
  int32_t n_pow2;  /* power of two, 1 .. 16384 */
} spinq_had_cfg;

/*
 * spinq_rotate_quant_act -- online rotation R4 fused with per-token 4-bit
 * activation quantization (Sec. 3.1 "Additional unabsorbed rotations" and
 * Eq. 1).  For each row m: x'_m = x_m R (skipped when had == NULL), then
 * Eq. 1 over the K values of x'_m with one (alpha_m, beta_m).  x' is kept in
 * fp32 and never stored.
 *   x_f16  [M][ldx] fp16, row m starts at x_f16 + m*ldx elements; 16-byte
 *          aligned rows (ldx % 8 == 0, pointer 16-byte aligned).
 *   had    NULL or a spec with n_small * n_pow2 == K.
 *   q      bits = 4, granularity = SPINQ_PER_TOKEN.
 *   codes  [M][K/2] packed codes (16-byte aligned).
 *   scale  [M] alpha_m.   zero [M] beta_m (asymmetric) or NULL (symmetric).
 * Supported K: 32 <= K <= 32768, K % 32 == 0 (with had: the spec's sizes).
 */
spinq_status spinq_rotate_quant_act(const void* x_f16, int64_t M, int64_t K, int64_t ldx,
                                    const spinq_had_cfg* had, const spinq_quant_cfg* q,
                                    uint8_t* codes, float* scale, float* zero, void* stream);

/*
 * spinq_quant_weight -- offline weight preparation: merge the rotation into
 * the weight (Sec. 3.1 rotational invariance: x' W'^T = x R R^T W^T = x W^T
 * with W' = W R, i.e. every output row rotated like an activation row), then
 * symmetric Eq. 1 per output channel (round-to-nearest, the RTN weight
 * quantizer of the appendix RTN-vs-GPTQ ablation), plus the integer row sum
 * of the codes that the GEMM epilogue needs.
 *   w_f16  [N][K] fp16 (16-byte aligned).   had NULL = no merge.
 *   q      bits = 4, symmetric = 1, granularity = SPINQ_PER_CHANNEL.
 *   codes  [N][K/2], scale [N] (s_n), rowsum [N] (sum_k q_nk).
 */
spinq_status spinq_quant_weight(const void* w_f16, int64_t N, int64_t K, const spinq_had_cfg* had,
                                const spinq_quant_cfg* q, uint8_t* codes, float* scale,
                                int32_t* rowsum, void* stream);

/*
 * Random-sign rotation (Sec. 2.2 footnote: a Hadamard matrix multiplied by a
 * random +-1 diagonal S is again a rotation, a "random Hadamard matrix"):
 * R = S (H_s (x) H_P) / sqrt(K), the signs acting on the input index k:
 * x' = (x S) (H_s (x) H_P) / sqrt(K), and W' = W S H / sqrt(K) for the merged
 * weights, so that x' W'^T = x W^T still holds.
 *   signs  device bit mask [K/8] bytes: bit (k % 8) of byte k / 8 set means
 *          s_k = -1.  Requires a Hadamard spec (had != NULL).
 * Other arguments as spinq_rotate_quant_act / spinq_quant_weight.
 */
spinq_status spinq_rotate_quant_act_signed(const void* x_f16, int64_t M, int64_t K, int64_t ldx,
                                           const spinq_had_cfg* had, const uint8_t* signs,
                                           const spinq_quant_cfg* q, uint8_t* codes, float* scale, float* zero,
                                           void* stream);
spinq_status spinq_quant_weight_signed(const void* w_f16, int64_t N, int64_t K, const spinq_had_cfg* had,
                                       const uint8_t* signs, const spinq_quant_cfg* q, uint8_t* codes,
                                       float* scale, int32_t* rowsum, void* stream);

/*
 * spinq_w4a4_gemm -- the W4A4 linear on Eq. 1 codes with an exact integer
 * accumulator and a fused per-token x per-channel dequantization epilogue.
 *   acc[m][n] = sum_k a_mk * q_nk, a = q (symmetric activations) or u - 8
 *               (asymmetric activations), exact in 32-bit integers;
 *   y[m][n]   = fp16( s_n * (alpha_m * acc[m][n] + beta'_m * rowsum_n) ),
 *               beta'_m = beta_m + 8 alpha_m (asymmetric) or 0 (symmetric),
 *   which equals sum_k (alpha_m c_mk + beta_m)(s_n q_nk), the product of the
 *   two dequantized operands of Eq. 1.
 *   a_codes [M][K/2], a_scale [M], a_zero [M] or NULL (symmetric);
 *   w_codes [N][K/2] symmetric, w_scale [N], w_rowsum [N];
 *   y_f16 [M][N] fp16; acc_out [M][N] int32 or NULL (debug output).
 *   Requirements: K % 128 == 0, N % 16 == 0, K <= 65536; code, output,
 *   w_scale and w_rowsum pointers 16-byte aligned.
 */
spinq_status spinq_w4a4_gemm(const uint8_t* a_codes, const float* a_scale, const float* a_zero,
                             const uint8_t* w_codes, const float* w_scale,
                             const int32_t* w_rowsum, int64_t M, int64_t N, int64_t K,
                             void* y_f16, int32_t* acc_out, void* stream);

/*
 * spinq_w4a4_gemm_workspace_bytes -- device workspace, in bytes, that
 * spinq_w4a4_gemm_splitk needs for an M x N x K call on the current CUDA
 * device: M*N*4 + 4*ceil(N/128) for the calls whose K range it splits across
 * CTAs (spinq_w4a4_gemm_splitk_plan), and 0 otherwise (those calls need no
 * workspace and may pass NULL).
 */
int64_t spinq_w4a4_gemm_workspace_bytes(int64_t M, int64_t N, int64_t K);

/*
 * spinq_w4a4_gemm_splitk -- the same operation and outputs as
 * spinq_w4a4_gemm, for small M (decode, M <= 256), where the GEMM is bound by
 * streaming the weights from HBM.  Up to 4 tokens (M * K <= 160 KiB) it runs
 * the GEMV kernel: each warp owns whole output channels, streams their packed
 * weights from global memory and takes exact integer dot products (no
 * workspace).  Otherwise a cost model fitted on GB300 picks between the
 * split-K kernel and the kernels of spinq_w4a4_gemm.  In the split-K kernel
 * each CTA owns 128 output channels and a slice of K, so every SM streams a
 * disjoint part of the weights; the slices' exact integer partial
 * accumulators are summed in `workspace` and the last slice of each
 * 128-channel tile applies the epilogue (with a single slice the CTA writes
 * the outputs itself and no workspace is used).  For M > 256 the call runs
 * the same kernel as spinq_w4a4_gemm and does not touch `workspace`.
 *   workspace       device buffer of spinq_w4a4_gemm_workspace_bytes(M, N, K)
 *                   bytes, 16-byte aligned, all zero before the first call;
 *                   each completed call leaves it zero again.  Calls that may
 *                   overlap on the GPU need distinct workspaces.  After a call
 *                   that recorded SPINQ_ETIMEOUT, clear it again.
 *   workspace_bytes its size (SPINQ_EINVAL if smaller than required).
 * Other arguments and requirements as spinq_w4a4_gemm.
 */
spinq_status spinq_w4a4_gemm_splitk(const uint8_t* a_codes, const float* a_scale, const float* a_zero,
                                    const uint8_t* w_codes, const float* w_scale,
                                    const int32_t* w_rowsum, int64_t M, int64_t N, int64_t K,
                                    void* y_f16, int32_t* acc_out, void* workspace,
                                    int64_t workspace_bytes, void* stream);

/* Size of the fixed device array spinq_w4a4_gemm_noalloc works in (8 MiB). */
#define SPINQ_NOALLOC_SCRATCH_BYTES (8ll << 20)

/*
 * spinq_w4a4_gemm_noalloc -- spinq_w4a4_gemm_splitk for callers that cannot
 * allocate device memory where they run the layer: a serving runtime that
 * reserves its whole memory budget at start-up and forbids later
 * allocations, a thread that must not call into an allocator while other
 * streams are being captured into CUDA graphs, an embedder with no device
 * allocator of its own to hand a workspace from.  The paper has no
 * counterpart: this is an interface convenience, not part of the method.
 *   Same arguments, outputs and requirements as spinq_w4a4_gemm; no workspace
 *   argument.  The workspace lives in a fixed device array of
 *   SPINQ_NOALLOC_SCRATCH_BYTES owned by the library, which every GPU that
 *   loads the library holds until the process exits.
 *   A request whose plan needs more workspace than that
 *   (spinq_w4a4_gemm_workspace_bytes(M, N, K) > SPINQ_NOALLOC_SCRATCH_BYTES,
 *   e.g. split-K decode plans with M * N * 4 above 8 MiB) is refused with
 *   SPINQ_ESCRATCH before anything is enqueued; split the tokens into smaller
 *   calls.  Requests whose plan needs no workspace (the GEMV, the prefill
 *   kernels, unsliced tiles) always run.
 *   The call itself allocates nothing: no cudaMalloc/cudaFree and no
 *   allocating library routine.  It clears the part of the array it uses
 *   (cudaMemsetAsync on `stream`) before the kernel, since the array keeps
 *   the previous call's contents.
 *   The first call in each CUDA context looks up the array's device address
 *   (cudaGetSymbolAddress, with that device current) and caches it for that
 *   context; make that first call outside any stream capture.
 *   Every call shares the one array per device: calls that may overlap on the
 *   GPU (different streams without ordering between them) race on it.
 */
spinq_status spinq_w4a4_gemm_noalloc(const uint8_t* a_codes, const float* a_scale, const float* a_zero,
                                     const uint8_t* w_codes, const float* w_scale,
                                     const int32_t* w_rowsum, int64_t M, int64_t N, int64_t K,
                                     void* y_f16, int32_t* acc_out, void* stream);

/*
 * spinq_rotated_linear -- the down_proj of Sec. 3.1 in one call: the online
 * rotation R4 (optionally with random signs, as spinq_rotate_quant_act_signed)
 * fused with the per-token Eq. 1 quantizer, then the W4A4 GEMM on those codes
 * against weights merged with the same rotation (spinq_quant_weight[_signed]).
 * The two kernels run back to back on `stream` (the GEMM's prologue overlaps
 * the quantizer's tail) and hand the codes over in `workspace`, which stays
 * in L2 between them (14.7 MB for 2048 tokens of K = 14336).
 *   x_f16 [M][ldx], had, signs (NULL = none), q (activation quantizer, 4
 *   bits, per token) as spinq_rotate_quant_act(_signed); w_codes [N][K/2],
 *   w_scale [N], w_rowsum [N], y_f16 [M][N] as spinq_w4a4_gemm.
 *   workspace  device buffer of spinq_rotated_linear_workspace_bytes(M, K)
 *              bytes, 16-byte aligned: the codes and scales in flight.
 */
int64_t spinq_rotated_linear_workspace_bytes(int64_t M, int64_t K);
spinq_status spinq_rotated_linear(const void* x_f16, int64_t M, int64_t K, int64_t ldx, const spinq_had_cfg* had,
                                  const uint8_t* signs, const spinq_quant_cfg* q, const uint8_t* w_codes,
                                  const float* w_scale, const int32_t* w_rowsum, int64_t N, void* y_f16,
                                  void* workspace, int64_t workspace_bytes, void* stream);

/*
 * spinq_rotate_quant_kv -- R3 on Q and K over head_dim, then the 4-bit
 * KV-cache quantizer (Sec. 3.1: R3 is an online Hadamard inserted for low-bit
 * KV-cache quantization; appendix "Quantization choice": asymmetric).
 * R2 is assumed merged into W_v / W_o, so V is quantized without rotation.
 *   q_in  [B][S][Hq][D] fp16 -> q_out (same layout; may equal q_in):
 *         q_out = fp16(q_in R).
 *   k_in, v_in [B][S][Hkv][D] fp16.
 *   K' = k_in R; K' and V quantized with kvq (bits = 4, symmetric = 0,
 *         granularity = SPINQ_PER_GROUP, group_size = D) into
 *   k_codes, v_codes [B][S][Hkv][D/2]; k_scale, k_zero, v_scale, v_zero
 *         [B][S][Hkv] fp32.
 *   had   {1, D}.  Supported D: 64 or 128.  All pointers 16-byte aligned.
 */
spinq_status spinq_rotate_quant_kv(const void* q_in, void* q_out, const void* k_in,
                                   const void* v_in, int64_t B, int64_t S, int64_t Hq,
                                   int64_t Hkv, int64_t D, const spinq_had_cfg* had,
                                   const spinq_quant_cfg* kvq, uint8_t* k_codes, float* k_scale,
                                   float* k_zero, uint8_t* v_codes, float* v_scale,
                                   float* v_zero, void* stream);

/*
 * spinq_gemm_select_kernel -- which kernel spinq_w4a4_gemm (and
 * spinq_w4a4_gemm_splitk / _noalloc for M > 256) runs, process-wide:
 *   SPINQ_GEMM_AUTO     the built-in cost model picks (the default);
 *   SPINQ_GEMM_TILE128  one CTA per 128 x 256 output tile;
 *   SPINQ_GEMM_TILE256  one CTA per 256 x 256 output tile;
 *   SPINQ_GEMM_PAIR     two CTAs (an SM pair) per 256 x 256 tile; calls it
 *                       cannot serve (M <= 128, no pair resident) use AUTO;
 *   SPINQ_GEMM_GEMV     (M <= 4 with M * K <= 160 KiB; AUTO picks it there
 *                       unless SPINQ_GEMM_TCGEMV takes the tokens, on the
 *                       _splitk / _noalloc entry points too) each warp
 *                       owns whole output channels and streams their packed
 *                       weights; calls it cannot serve use AUTO;
 *   SPINQ_GEMM_SPLITK   the split-K kernel on the _splitk / _noalloc entry
 *                       points for every M <= 256 (GEMV and prefill kernels
 *                       excluded); spinq_w4a4_gemm treats it as AUTO;
 *   SPINQ_GEMM_TCGEMV   (M <= 16, on every entry point; AUTO picks it for 3 to
 *                       16 tokens when K / 128 = NKW W with NKW in {1, 2, 4,
 *                       8} and W <= 16, else for 5 to 8 tokens) the products
 *                       on the tensor core (fp16 m16n8k16 on the exact codes),
 *                       no workspace: for such K, one CTA per SM whose W
 *                       warps split K and stream the packed weights straight
 *                       into registers; else a CTA per 16 output channels
 *                       that stages them through shared memory; calls it
 *                       cannot serve use AUTO.
 * All kernels compute bit-identical outputs; this is a tuning and testing
 * control.  Returns the previous selection, or -1 (and changes nothing) for
 * an unknown value.  Not synchronized with GEMM calls in other threads.
 */
typedef enum {
  SPINQ_GEMM_AUTO = 0,
  SPINQ_GEMM_TILE128 = 1,
  SPINQ_GEMM_TILE256 = 2,
  SPINQ_GEMM_PAIR = 3,
  SPINQ_GEMM_GEMV = 4,
  SPINQ_GEMM_SPLITK = 5,
  SPINQ_GEMM_TCGEMV = 6
} spinq_gemm_kernel;

int spinq_gemm_select_kernel(int kernel);

/*
 * spinq_gemm_split_k -- process-wide number of K slices per 128-channel tile
 * of the split-K kernel: 1..64 fixes it (at most K / 128), 0 lets the cost
 * model pick (the default).  A tuning and testing control like
 * spinq_gemm_select_kernel; spinq_w4a4_gemm_workspace_bytes and
 * spinq_w4a4_gemm_splitk_plan follow it.  Returns the previous value, or -1
 * (and changes nothing) for a value out of range.
 */
int spinq_gemm_split_k(int n);

/*
 * spinq_w4a4_gemm_plan -- the kernel (SPINQ_GEMM_TILE128, _TILE256, _PAIR,
 * _GEMV or _TCGEMV) that spinq_w4a4_gemm runs for an M x N x K call on the current CUDA
 * device under the current selection; -1 for shapes the call rejects.
 * Launches nothing.
 */
int spinq_w4a4_gemm_plan(int64_t M, int64_t N, int64_t K);

/*
 * spinq_w4a4_gemm_splitk_plan -- the kernel that spinq_w4a4_gemm_splitk runs
 * for an M x N x K call given a workspace of spinq_w4a4_gemm_workspace_bytes
 * bytes: SPINQ_GEMM_SPLITK, with *nsplit (may be NULL) set to its number of K
 * slices per 128-channel tile (1: no slicing, no workspace), or the kernel
 * spinq_w4a4_gemm would run (*nsplit = 0).  -1 for shapes the call rejects.
 * Launches nothing.
 */
int spinq_w4a4_gemm_splitk_plan(int64_t M, int64_t N, int64_t K, int* nsplit);

/*
 * spinq_rope_rotate_quant_kv -- spinq_rotate_quant_kv with the rotary
 * position embedding applied to Q and K first, in the same kernel: for each
 * token at position p and i < D/2, with (cos, sin) of angle p theta_i taken
 * from the caller's table,
 *   x_i <- x_i cos - x_{i+D/2} sin,   x_{i+D/2} <- x_i sin + x_{i+D/2} cos
 * (the rotate-half form), computed in fp32 and rounded to fp16 like the
 * model's activations; then R3 (Sec. 3.1, the online Hadamard that follows
 * RoPE on Q and K) and the KV quantizer exactly as spinq_rotate_quant_kv.
 *   positions [B][S] int32, each in [0, max_pos) (others are clamped).
 *   cos_sin   [max_pos][D/2] pairs (cos, sin) as fp32, 16-byte aligned; the
 *             caller computes angle p theta_i, theta_i = base^(-2i/D),
 *             accurately (e.g. in double) once.
 * Other arguments, layouts and requirements as spinq_rotate_quant_kv.
 */
spinq_status spinq_rope_rotate_quant_kv(const void* q_in, void* q_out, const void* k_in, const void* v_in,
                                        const int32_t* positions, const float* cos_sin, int64_t max_pos, int64_t B,
                                        int64_t S, int64_t Hq, int64_t Hkv, int64_t D, const spinq_had_cfg* had,
                                        const spinq_quant_cfg* kvq, uint8_t* k_codes, float* k_scale,
                                        float* k_zero, uint8_t* v_codes, float* v_scale, float* v_zero,
                                        void* stream);

/*
 * spinq_decode_attention_kv4 -- attention of one decode query per (batch,
 * query head) over the 4-bit KV cache written by spinq_rotate_quant_kv (or
 * its RoPE form), the consumer of R3 (Sec. 3.1: R3 rotates Q and K over
 * head_dim so that Q K^T is unchanged while K quantizes to 4 bits):
 *   s_t = softmax_scale * q . k_t,  k_t = k_scale * u_t + k_zero,
 *   o   = sum_t softmax_t(s) v_t,     v_t = v_scale * u'_t + v_zero,
 * over t < lens[b]; query head h reads kv head h / (Hq / Hkv).
 *   q        [B][Hq][D] fp16, already rotated by R3 (the q_out of the call
 *            above for the decode token).
 *   k_codes, v_codes [B][S][Hkv][D/2], 16-byte aligned; k_scale, k_zero,
 *            v_scale, v_zero [B][S][Hkv] fp32 (S is the cache capacity: the
 *            row stride).
 *   lens     [B] int32 in [1, S] (device), or NULL for S everywhere.
 *   out      [B][Hq][D] fp16.
 *   workspace device buffer of spinq_decode_attention_workspace_bytes(B, S,
 *            Hq, Hkv, D) bytes, 16-byte aligned (the per-chunk partial
 *            results; no zeroing needed).
 *   Supported: D = 64 or 128, Hq / Hkv in {1, 2, 4, 8}, S * Hkv * D / 2 <
 *   2^31 (one batch's codes within 2 GiB).  Both products run
 *   on the tensor core with fp32 accumulation: q . u on the fp16 query and
 *   the exact codes, the value sum on the codes and fp16 weights
 *   p * v_scale / max(v_scale) (relative rounding 2^-11 per weight); the
 *   softmax and the scales in fp32.  Two kernels on `stream` (the chunks,
 *   then their merge).
 */
int64_t spinq_decode_attention_workspace_bytes(int64_t B, int64_t S, int64_t Hq, int64_t Hkv, int64_t D);
spinq_status spinq_decode_attention_kv4(const void* q, const uint8_t* k_codes, const float* k_scale,
                                        const float* k_zero, const uint8_t* v_codes, const float* v_scale,
                                        const float* v_zero, const int32_t* lens, int64_t B, int64_t S, int64_t Hq,
                                        int64_t Hkv, int64_t D, float softmax_scale, void* out, void* workspace,
                                        int64_t workspace_bytes, void* stream);

/*
 * 8-bit variants (main results table, W4A8 rows "4-8-x"; appendix "Latency
 * measurement on GPU": W-fp8-A-fp8 with the dequantization fused into the
 * GEMM epilogue).  They share the rotation convention above and run on the
 * E4M3 tensor-core pipe without unpacking.
 *
 * Code formats:
 *   SPINQ_FMT_INT8_PLANES  Eq. 1 with N = 8 per token: the code c = q
 *       (symmetric, [-128, 127]) or u - 128 (asymmetric, u in [0, 255]) is
 *       stored as two E4M3 planes, row [2K] bytes: byte k = E4M3(16 (c >> 4)),
 *       byte K + k = E4M3(c & 15) (both exact), so c = dec(k) + dec(K + k).
 *   SPINQ_FMT_E4M3         per-row FP8: alpha = clip max|x'| / 448, code =
 *       E4M3(x' / alpha), round to nearest even, saturating at +-448
 *       (E4M3: 1 sign, 4 exponent bits with bias 7, 3 mantissa bits, no
 *       infinities), [K] bytes per row.
 *   SPINQ_FMT_INT4_BYTES   (weights of the W4A8 linear) Eq. 1 with N = 4,
 *       symmetric per output channel, each code q in [-8, 7] stored as the
 *       E4M3 byte of q, [K] bytes per row, plus rowsum = sum_k q.
 */
typedef enum {
  SPINQ_FMT_INT8_PLANES = 1,
  SPINQ_FMT_E4M3 = 2,
  SPINQ_FMT_INT4_BYTES = 3
} spinq_code_format;

/*
 * spinq_rotate_quant_act8 -- online rotation (as spinq_rotate_quant_act)
 * then the 8-bit per-token quantizer `format`:
 *   SPINQ_FMT_INT8_PLANES  q: bits = 8, symmetric or asymmetric; codes
 *                          [M][2K]; scale [M]; zero [M] (asymmetric) or NULL.
 *   SPINQ_FMT_E4M3         q: bits = 8, symmetric = 1; codes [M][K]; scale [M].
 *   q->granularity = SPINQ_PER_TOKEN.  K % 128 == 0, K <= 32768, x rows and
 *   codes 16-byte aligned.  Other formats return SPINQ_EINVAL.
 */
spinq_status spinq_rotate_quant_act8(const void* x_f16, int64_t M, int64_t K, int64_t ldx,
                                     const spinq_had_cfg* had, const spinq_quant_cfg* q, int32_t format,
                                     uint8_t* codes, float* scale, float* zero, void* stream);

/*
 * spinq_quant_weight8 -- offline weight preparation of the 8-bit linears:
 * W' = W R (when had != NULL), then per output channel
 *   SPINQ_FMT_E4M3        q: bits = 8, symmetric; codes [N][K]; scale [N];
 *                         rowsum unused (may be NULL);
 *   SPINQ_FMT_INT4_BYTES  q: bits = 4, symmetric; codes [N][K]; scale [N];
 *                         rowsum [N].
 *   q->granularity = SPINQ_PER_CHANNEL; sizes as spinq_rotate_quant_act8.
 */
spinq_status spinq_quant_weight8(const void* w_f16, int64_t N, int64_t K, const spinq_had_cfg* had,
                                 const spinq_quant_cfg* q, int32_t format, uint8_t* codes, float* scale,
                                 int32_t* rowsum, void* stream);

/*
 * spinq_fp8_gemm -- W-fp8-A-fp8 linear:
 *   y[m][n] = fp16(alpha_m s_n sum_k a_mk w_nk), a, w decoded E4M3 codes,
 * products exact and summed in fp32 on the tensor core.
 *   a_codes [M][K] (SPINQ_FMT_E4M3), a_scale [M]; w_codes [N][K], w_scale [N].
 *   K % 128 == 0, K <= 65536, N % 16 == 0; code and output pointers 16-byte
 *   aligned.
 */
spinq_status spinq_fp8_gemm(const uint8_t* a_codes, const float* a_scale, const uint8_t* w_codes,
                            const float* w_scale, int64_t M, int64_t N, int64_t K, void* y_f16, void* stream);

/*
 * spinq_w4a8_gemm -- W4A8 linear on Eq. 1 codes, exact integer accumulator:
 *   acc[m][n] = sum_k c_mk q_nk (c = q or u - 128, exact in fp32: every
 *               partial sum is an integer of magnitude <= 1024 K <= 2^24);
 *   y[m][n]   = fp16(s_n (alpha_m acc + beta'_m rowsum_n)),
 *               beta'_m = beta_m + 128 alpha_m (asymmetric) or 0,
 *   the dequantized product of the two Eq. 1 operands.
 *   a_planes [M][2K] (SPINQ_FMT_INT8_PLANES), a_scale [M], a_zero [M] or NULL;
 *   w_codes [N][K] (SPINQ_FMT_INT4_BYTES), w_scale [N], w_rowsum [N];
 *   acc_out [M][N] int32 or NULL (debug).
 *   K % 128 == 0, K <= 16384, N % 16 == 0; code and output pointers 16-byte
 *   aligned.
 */
spinq_status spinq_w4a8_gemm(const uint8_t* a_planes, const float* a_scale, const float* a_zero,
                             const uint8_t* w_codes, const float* w_scale, const int32_t* w_rowsum, int64_t M,
                             int64_t N, int64_t K, void* y_f16, int32_t* acc_out, void* stream);

/*
 * spinq_cayley_step -- one Cayley SGD update of a batch of rotations
 * (Sec. 3.2, the R' update and its Y / G_hat definitions), for learning R2
 * (head_dim x head_dim, one per layer) with the weights frozen:
 *   G_hat = G R^T - 1/2 R R^T G R^T,   Y = G_hat - G_hat^T,
 *   R'    = (I - alpha/2 Y)^-1 (I + alpha/2 Y) R,
 * computed, as the paper does, by the fixed-point iteration of Cayley SGD:
 *   R'_0 = R + alpha Y R,   R'_{k+1} = R + (alpha/2) Y (R + R'_k),
 *   k = 0 .. iters-1 (it converges to R' when |alpha Y / 2| < 1).
 * G is the NEGATIVE of the loss gradient `grad` passed here: the objective
 * is an argmin and the cited Cayley SGD forms G_hat from the negative
 * gradient (with G = +grad the printed update would climb the loss).
 *   R      [batch][n][n] fp32 row-major, each orthonormal (device).
 *   grad   [batch][n][n] fp32, dL/dR (device).
 *   alpha  learning rate (finite); iters in 0 .. 64.
 *   R_out  [batch][n][n] fp32; may be R itself (in-place update), must not
 *          overlap R or grad otherwise.
 *   Y_out  [batch][n][n] fp32 or NULL: the skew-symmetric Y of each update.
 *   Supported n: 16, 32, 64, 128.  Pointers 16-byte aligned.  Arithmetic in
 *   fp32 (the oracle works in double).
 */
spinq_status spinq_cayley_step(const float* R, const float* grad, int64_t batch, int64_t n, float alpha,
                               int32_t iters, float* R_out, float* Y_out, void* stream);

/*
 * Testing controls of the failure paths (the paper has no counterpart).
 * spinq_debug_set_wait_limit_ns -- time limit of the ordinary bounded waits
 *   of the Paley rotate+quant, W4A4 and FP8 GEMM kernels on the current
 *   device (2e9 ns by default; the drains of copies and MMAs in flight keep
 *   their full limit).  A test lowers it so that those waits give up, checks
 *   SPINQ_ETIMEOUT through spinq_device_status and sets it back.  Outputs of
 *   a call that gave up are undefined.  SPINQ_EINVAL for ns <= 0.
 * spinq_debug_stall_launches -- the next n launches of the Paley rotate+quant,
 *   the W4A4 prefill (128- and 256-row tiles) and the FP8 GEMM kernels issue
 *   no input copies, so the waits of their consumers run out of time (a
 *   barrier that nothing completes): SPINQ_ETIMEOUT is recorded, every role
 *   leaves its loop, MMAs in flight are drained and tensor memory is freed.
 *   Lower the wait limit first so that this takes a millisecond, not 2 s.
 *   Outputs of such a call are undefined.  Returns the previous count, or -1
 *   for n < 0.
 * spinq_debug_fail_launches -- the next n kernel launches of the library are
 *   refused on the host (the call returns SPINQ_ECUDA; nothing reaches the
 *   GPU).  Returns the previous count, or -1 for n < 0.
 */
spinq_status spinq_debug_set_wait_limit_ns(int64_t ns);
int spinq_debug_stall_launches(int n);
int spinq_debug_fail_launches(int n);

/* Human-readable name of a status code (static storage). */
const char* spinq_status_string(spinq_status s);

/*
 * spinq_device_status -- read and clear the device status word that bounded
 * waits in the kernels write when they give up (SPINQ_ETIMEOUT), for the
 * current CUDA device.  Synchronizes the device.  Returns SPINQ_OK when no
 * kernel recorded an error since the last call, SPINQ_ECUDA if the read
 * itself failed.  `detail` (may be NULL) receives the recorded site code.
 */
spinq_status spinq_device_status(int32_t* detail);

/* Library build identifier (static storage). */
const char* spinq_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SPINQ_H_ */
