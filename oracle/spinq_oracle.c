/*
 * spinq_oracle.c -- plain, slow, double-precision CPU oracle for the rotated
 * W4A4 hot path of SpinQuant (arXiv 2405.16406).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference leg of bench.py may load this library.  It shares
 * no code, header, table or constant with the CUDA library under
 * paper_2405_16406_gb300/csrc, and the CUDA library never calls it.
 *
 * Every function computes the plain definition of what it names, in double,
 * with no blocking, fusion or reordering beyond what that definition states.
 * Rows are independent; OpenMP only splits independent rows across cores.
 *
 * Paper passages followed (section / equation of the paper):
 *   - Eq. 1 (Sec. 2): min-max round-to-nearest quantizer, symmetric and
 *     asymmetric forms, N bits.
 *   - Sec. 2.2 footnote: a Hadamard matrix is a rotation whose entries all
 *     share one magnitude; read here as R = H / sqrt(n) with H in {+1,-1}.
 *   - Sec. 3.1 ("Additional unabsorbed rotations"): R4 is an online Hadamard
 *     on the down_proj input, R3 an online Hadamard on Q/K over head_dim,
 *     both computed with a fast Hadamard transform.
 *   - Sec. 3.1 ("Rotating activations in residual"): rotational invariance,
 *     x R (W R)^T = x W^T for orthonormal R, which fixes how a rotated weight
 *     is merged (W' = W R).
 *   - Appendix "Quantization choice": clipping ratio of the min-max range;
 *     asymmetric quantization for activations and the KV cache.
 *
 * Readings where the paper is silent:
 *   - Sylvester H_{2^k}[i][j] = (-1)^popcount(i & j) (natural order).
 *   - Paley I for a prime power q = 3 mod 4, order q + 1: H = I + S with
 *     S = [[0, 1^T], [-1, Q]], Q[i][j] = chi(a_i - a_j), chi the quadratic
 *     character.  GF(p) for prime q (a_i = i); GF(27) = GF(3)[t]/(t^3+2t+1)
 *     with a_i = c0 + c1 t + c2 t^2 for i = c0 + 3 c1 + 9 c2.
 *   - Non-power-of-two sizes K = n_s * P use H_s (x) H_P with the small
 *     factor on the slow index: k = i * P + j.  The rotation is the row-vector
 *     product y = x (H_s (x) H_P) / sqrt(K).
 *   - Rounding is round-half-to-even (nearbyint in the default mode).
 *   - Symmetric codes clamp to [-2^(N-1), 2^(N-1)-1]; asymmetric to
 *     [0, 2^N - 1]; a zero range gives alpha = 0 and all codes 0.
 *   - Clipping scales max|x| (symmetric) or both min and max (asymmetric).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_EINVAL 1

/* ------------------------------------------------------------------ */
/* threads                                                             */
/* ------------------------------------------------------------------ */
int oracle_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
  return omp_get_max_threads();
#else
  (void)n;
  return 1;
#endif
}

/* ------------------------------------------------------------------ */
/* IEEE 754 binary16 <-> double, written from the format definition    */
/* ------------------------------------------------------------------ */
double oracle_f16_to_double(uint16_t h) {
  int s = (h >> 15) & 1, e = (h >> 10) & 0x1f, m = h & 0x3ff;
  double v;
  if (e == 0)
    v = ldexp((double)m, -24); /* subnormal: m * 2^-24 */
  else if (e == 31)
    v = m ? NAN : INFINITY;
  else
    v = ldexp((double)(m + 1024), e - 25); /* (1 + m/1024) 2^(e-15) */
  return s ? -v : v;
}

/* Round-to-nearest-even from double. */
uint16_t oracle_double_to_f16(double d) {
  uint16_t sign = signbit(d) ? 0x8000 : 0;
  double a = fabs(d);
  if (isnan(d)) return 0x7e00;
  if (a >= 65520.0) return sign | 0x7c00; /* halfway to 2^16 and above -> inf */
  if (a < ldexp(1.0, -14)) {
    double q = nearbyint(ldexp(a, 24)); /* subnormal quantum 2^-24; q <= 1024 */
    return sign | (uint16_t)q;
  }
  int e;
  double f = frexp(a, &e);          /* a = f 2^e, f in [0.5, 1) */
  double q = nearbyint(ldexp(f, 11)); /* significand with hidden bit, [1024, 2048] */
  int E = e + 14;                   /* biased exponent */
  if (q == 2048.0) {
    q = 1024.0;
    E += 1;
  }
  if (E >= 31) return sign | 0x7c00;
  return (uint16_t)(sign | (E << 10) | ((int)q - 1024));
}

void oracle_f16_array_to_double(const uint16_t* h, double* d, int64_t n) {
  for (int64_t i = 0; i < n; ++i) d[i] = oracle_f16_to_double(h[i]);
}

void oracle_double_array_to_f16(const double* d, uint16_t* h, int64_t n) {
  for (int64_t i = 0; i < n; ++i) h[i] = oracle_double_to_f16(d[i]);
}

/* ------------------------------------------------------------------ */
/* Hadamard constructions (Sec. 2.2 footnote; Sec. 3.1 R3/R4)           */
/* ------------------------------------------------------------------ */
static int is_pow2(int64_t n) { return n > 0 && (n & (n - 1)) == 0; }

static int popcount_u64(uint64_t x) {
  int c = 0;
  while (x) {
    c += (int)(x & 1u);
    x >>= 1;
  }
  return c;
}

/* Sylvester: H_1 = [1], H_2n = [[H, H], [H, -H]], i.e. (-1)^popcount(i&j). */
int oracle_sylvester(int64_t n, int8_t* H) {
  if (!is_pow2(n)) return OR_EINVAL;
  for (int64_t i = 0; i < n; ++i)
    for (int64_t j = 0; j < n; ++j)
      H[i * n + j] = (popcount_u64((uint64_t)(i & j)) & 1) ? -1 : 1;
  return OR_OK;
}

/* GF(q) arithmetic for the Paley construction.  q prime: integers mod q.
 * q = 27: polynomials over GF(3) modulo t^3 + 2t + 1, element index
 * c0 + 3 c1 + 9 c2 for c0 + c1 t + c2 t^2.                              */
static int gf_sub(int q, int a, int b) {
  if (q != 27) return ((a - b) % q + q) % q;
  int r = 0, p = 1;
  for (int d = 0; d < 3; ++d) {
    int da = a % 3, db = b % 3;
    r += (((da - db) % 3 + 3) % 3) * p;
    a /= 3;
    b /= 3;
    p *= 3;
  }
  return r;
}

static int gf_mul(int q, int a, int b) {
  if (q != 27) return (a * b) % q;
  int ca[3], cb[3], prod[5] = {0, 0, 0, 0, 0};
  for (int d = 0; d < 3; ++d) {
    ca[d] = a % 3;
    cb[d] = b % 3;
    a /= 3;
    b /= 3;
  }
  for (int i = 0; i < 3; ++i)
    for (int j = 0; j < 3; ++j) prod[i + j] += ca[i] * cb[j];
  /* reduce degrees 4 and 3 with t^3 = -2t - 1 = t + 2 (mod 3) */
  for (int d = 4; d >= 3; --d) {
    int c = prod[d] % 3;
    prod[d] = 0;
    prod[d - 3 + 1] += c;     /* c * t^(d-3) * t   */
    prod[d - 3] += 2 * c;     /* c * t^(d-3) * 2   */
  }
  return (prod[0] % 3) + 3 * (prod[1] % 3) + 9 * (prod[2] % 3);
}

/* quadratic character: a^((q-1)/2) is 1 for a nonzero square, -1 otherwise */
static int gf_chi(int q, int a) {
  if (a == 0) return 0;
  int r = 1;
  for (int e = 0; e < (q - 1) / 2; ++e) r = gf_mul(q, r, a);
  if (r == 1) return 1;
  /* -1 is q-1 for prime q and the constant 2 (index 2) in GF(27) */
  if ((q != 27 && r == q - 1) || (q == 27 && r == 2)) return -1;
  return -2; /* not a field: caller treats as error */
}

static int paley_q_supported(int q) {
  if (q == 27) return 1;
  if (q < 3 || q % 4 != 3) return 0;
  for (int d = 2; d * d <= q; ++d)
    if (q % d == 0) return 0;
  return 1;
}

/* Paley I of order q + 1 (q = 3 mod 4 a prime power): H = I + S. */
int oracle_paley1(int q, int8_t* H) {
  if (!paley_q_supported(q)) return OR_EINVAL;
  int n = q + 1;
  for (int r = 0; r < n; ++r)
    for (int c = 0; c < n; ++c) {
      int s;
      if (r == 0 && c == 0)
        s = 0;
      else if (r == 0)
        s = 1;
      else if (c == 0)
        s = -1;
      else {
        s = gf_chi(q, gf_sub(q, r - 1, c - 1));
        if (s == -2) return OR_EINVAL;
      }
      H[r * n + c] = (int8_t)((r == c ? 1 : 0) + s);
    }
  return OR_OK;
}

/* The small Kronecker factor H_s of order n_s: [1] for n_s = 1, Paley I of
 * order n_s otherwise (n_s - 1 a supported prime power).                 */
int oracle_small_hadamard(int n_s, int8_t* H) {
  if (n_s == 1) {
    H[0] = 1;
    return OR_OK;
  }
  return oracle_paley1(n_s - 1, H);
}

/* ------------------------------------------------------------------ */
/* Rotation y = x (H_s (x) H_P) / sqrt(K)   (Sec. 3.1, R3 and R4)      */
/* ------------------------------------------------------------------ */

/* In-place fast Walsh-Hadamard transform, natural order: v <- H_n v.  H_n
 * (Sylvester) is symmetric, so this is also the row-vector product v H_n. */
void oracle_fwht(double* v, int64_t n) {
  for (int64_t h = 1; h < n; h <<= 1)
    for (int64_t i = 0; i < n; i += 2 * h)
      for (int64_t j = i; j < i + h; ++j) {
        double a = v[j], b = v[j + h];
        v[j] = a + b;
        v[j + h] = a - b;
      }
}

/* rows x K, K = n_s * n_pow2. */
int oracle_rotate(const double* x, double* y, int64_t rows, int n_s, int64_t n_pow2) {
  if (!is_pow2(n_pow2) || n_s < 1) return OR_EINVAL;
  int8_t* Hs = (int8_t*)malloc((size_t)n_s * n_s);
  if (!Hs) return OR_EINVAL;
  if (oracle_small_hadamard(n_s, Hs) != OR_OK) {
    free(Hs);
    return OR_EINVAL;
  }
  const int64_t P = n_pow2, K = (int64_t)n_s * P;
  const double inv = 1.0 / sqrt((double)K);
  int err = 0;
#pragma omp parallel
  {
    double* t = (double*)malloc(sizeof(double) * (size_t)K);
    if (!t) {
#pragma omp atomic write
      err = 1;
    }
#pragma omp for schedule(static)
    for (int64_t r = 0; r < rows; ++r) {
      if (!t) continue;
      const double* xr = x + r * K;
      double* yr = y + r * K;
      memcpy(t, xr, sizeof(double) * (size_t)K);
      /* X[i][:] <- X[i][:] H_P for every slow index i */
      for (int i = 0; i < n_s; ++i) oracle_fwht(t + (int64_t)i * P, P);
      /* Y[i][j] = sum_i' X[i'][j] H_s[i'][i]  (row vector times H_s) */
      for (int64_t j = 0; j < P; ++j)
        for (int i = 0; i < n_s; ++i) {
          double acc = 0.0;
          for (int ip = 0; ip < n_s; ++ip) acc += t[(int64_t)ip * P + j] * (double)Hs[ip * n_s + i];
          yr[(int64_t)i * P + j] = acc * inv;
        }
    }
    free(t);
  }
  free(Hs);
  return err ? OR_EINVAL : OR_OK;
}

/* ------------------------------------------------------------------ */
/* Eq. 1 quantizer, per row (token / output channel / group)           */
/* ------------------------------------------------------------------ */
/* x: rows x K; each row is quantized with its own (alpha, beta).
 * symmetric : alpha = clip max|x| / (2^(N-1) - 1), beta = 0,
 *             q = clamp(rint(x / alpha), -2^(N-1), 2^(N-1) - 1)
 * asymmetric: alpha = clip (max x - min x) / (2^N - 1), beta = clip min x,
 *             u = clamp(rint((x - beta) / alpha), 0, 2^N - 1)
 * Dequantized value is alpha * code + beta (Eq. 1).                     */
int oracle_quantize_rows(const double* x, int64_t rows, int64_t K, int bits, int symmetric,
                         double clip, int32_t* codes, double* alpha, double* beta) {
  if (bits < 2 || bits > 8 || K <= 0 || !(clip > 0.0 && clip <= 1.0)) return OR_EINVAL;
  const double smax = (double)((1 << (bits - 1)) - 1), smin = -(double)(1 << (bits - 1));
  const double amax = (double)((1 << bits) - 1);
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r) {
    const double* xr = x + r * K;
    int32_t* cr = codes + r * K;
    double a, b;
    if (symmetric) {
      double m = 0.0;
      for (int64_t k = 0; k < K; ++k) m = fmax(m, fabs(xr[k]));
      a = clip * m / smax;
      b = 0.0;
      for (int64_t k = 0; k < K; ++k) {
        double q = a > 0.0 ? nearbyint(xr[k] / a) : 0.0;
        cr[k] = (int32_t)fmin(fmax(q, smin), smax);
      }
    } else {
      double hi = xr[0], lo = xr[0];
      for (int64_t k = 1; k < K; ++k) {
        hi = fmax(hi, xr[k]);
        lo = fmin(lo, xr[k]);
      }
      hi *= clip;
      lo *= clip;
      a = (hi - lo) / amax;
      b = lo;
      for (int64_t k = 0; k < K; ++k) {
        double u = a > 0.0 ? nearbyint((xr[k] - b) / a) : 0.0;
        cr[k] = (int32_t)fmin(fmax(u, 0.0), amax);
      }
    }
    alpha[r] = a;
    beta[r] = b;
  }
  return OR_OK;
}

/* Dequantize codes back to reals: x_Q = alpha * code + beta (Eq. 1). */
void oracle_dequantize_rows(const int32_t* codes, const double* alpha, const double* beta,
                            int64_t rows, int64_t K, double* xq) {
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t k = 0; k < K; ++k)
      xq[r * K + k] = alpha[r] * (double)codes[r * K + k] + (beta ? beta[r] : 0.0);
}

/* ------------------------------------------------------------------ */
/* 4-bit packing: two codes per byte, even index in the low nibble.     */
/* Signed codes are stored as two's complement nibbles.                 */
/* ------------------------------------------------------------------ */
void oracle_pack4(const int32_t* codes, int64_t n, uint8_t* packed) {
  for (int64_t i = 0; i < n / 2; ++i)
    packed[i] = (uint8_t)((codes[2 * i] & 0xF) | ((codes[2 * i + 1] & 0xF) << 4));
}

void oracle_unpack4(const uint8_t* packed, int64_t n, int is_signed, int32_t* codes) {
  for (int64_t i = 0; i < n; ++i) {
    int v = (packed[i / 2] >> (4 * (i & 1))) & 0xF;
    if (is_signed && v >= 8) v -= 16;
    codes[i] = v;
  }
}

/* ------------------------------------------------------------------ */
/* W4A4 linear: integer accumulator and dequantized output              */
/* ------------------------------------------------------------------ */
/* a_codes: M x K stored activation codes (q for symmetric, u for asymmetric)
 * w_codes: N x K symmetric weight codes q_w.
 * acc[m][n] = sum_k a_int * q_w with a_int = q (symmetric) or u - 2^(N-1)
 *             (asymmetric, the zero-centred code); checked to fit int32.
 * y[m][n]   = sum_k (alpha_m c_mk + beta_m) (s_n q_w,nk), the plain
 *             dequantized product (Eq. 1 applied to both operands).       */
static int gemm_one(const int32_t* a, const int32_t* w, int64_t K, int sym, double am, double bm,
                    double sn, int32_t* acc_out, double* y_out) {
  int64_t acc = 0;
  double y = 0.0;
  for (int64_t k = 0; k < K; ++k) {
    const int64_t ai = sym ? a[k] : (int64_t)a[k] - 8;
    acc += ai * (int64_t)w[k];
    y += (am * (double)a[k] + bm) * (sn * (double)w[k]);
  }
  if (acc > INT32_MAX || acc < INT32_MIN) return OR_EINVAL;
  *acc_out = (int32_t)acc;
  *y_out = y;
  return OR_OK;
}

int oracle_w4a4_gemm(const int32_t* a_codes, const double* a_scale, const double* a_zero,
                     const int32_t* w_codes, const double* w_scale, int64_t M, int64_t N, int64_t K,
                     int32_t* acc, double* y) {
  const int sym = a_zero == NULL;
  int err = 0;
#pragma omp parallel for schedule(static) collapse(2)
  for (int64_t m = 0; m < M; ++m)
    for (int64_t n = 0; n < N; ++n) {
      int e = gemm_one(a_codes + m * K, w_codes + n * K, K, sym, a_scale[m], sym ? 0.0 : a_zero[m],
                       w_scale[n], acc + m * N + n, y + m * N + n);
      if (e) {
#pragma omp atomic write
        err = 1;
      }
    }
  return err ? OR_EINVAL : OR_OK;
}

/* Same definition at an explicit list of (m, n) output coordinates. */
int oracle_w4a4_gemm_sampled(const int32_t* a_codes, const double* a_scale, const double* a_zero,
                             const int32_t* w_codes, const double* w_scale, int64_t K,
                             const int64_t* ms, const int64_t* ns, int64_t count, int32_t* acc,
                             double* y) {
  const int sym = a_zero == NULL;
  int err = 0;
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < count; ++i) {
    const int64_t m = ms[i], n = ns[i];
    int e = gemm_one(a_codes + m * K, w_codes + n * K, K, sym, a_scale[m], sym ? 0.0 : a_zero[m],
                     w_scale[n], acc + i, y + i);
    if (e) {
#pragma omp atomic write
      err = 1;
    }
  }
  return err ? OR_EINVAL : OR_OK;
}

/* Integer row sums of codes: rowsum[r] = sum_k codes[r][k]. */
void oracle_rowsum(const int32_t* codes, int64_t rows, int64_t K, int32_t* rowsum) {
  for (int64_t r = 0; r < rows; ++r) {
    int64_t s = 0;
    for (int64_t k = 0; k < K; ++k) s += codes[r * K + k];
    rowsum[r] = (int32_t)s;
  }
}

/* ------------------------------------------------------------------ */
/* Cayley SGD step (Sec. 3.2)                                          */
/* ------------------------------------------------------------------ */
/* C = op(A) op(B) for n x n row-major matrices, op = transpose when the
 * flag is set; the plain triple loop in double. */
static void mat_mul(const double* A, int ta, const double* B, int tb, int64_t n, double* C) {
  for (int64_t i = 0; i < n; ++i)
    for (int64_t j = 0; j < n; ++j) {
      double s = 0.0;
      for (int64_t k = 0; k < n; ++k) {
        const double a = ta ? A[k * n + i] : A[i * n + k];
        const double b = tb ? B[j * n + k] : B[k * n + j];
        s += a * b;
      }
      C[i * n + j] = s;
    }
}

/* Y of Sec. 3.2 for one rotation R and the loss gradient G:
 *   G_hat = G R^T - 1/2 R R^T G R^T,   Y = G_hat - G_hat^T. */
int oracle_cayley_y(const double* R, const double* G, int64_t n, double* Y) {
  if (n <= 0) return OR_EINVAL;
  double* GRt = (double*)malloc(sizeof(double) * n * n);
  double* RtGRt = (double*)malloc(sizeof(double) * n * n);
  double* RRtGRt = (double*)malloc(sizeof(double) * n * n);
  double* Gh = (double*)malloc(sizeof(double) * n * n);
  if (!GRt || !RtGRt || !RRtGRt || !Gh) {
    free(GRt), free(RtGRt), free(RRtGRt), free(Gh);
    return OR_EINVAL;
  }
  mat_mul(G, 0, R, 1, n, GRt);         /* G R^T           */
  mat_mul(R, 1, GRt, 0, n, RtGRt);     /* R^T G R^T       */
  mat_mul(R, 0, RtGRt, 0, n, RRtGRt);  /* R R^T G R^T     */
  for (int64_t e = 0; e < n * n; ++e) Gh[e] = GRt[e] - 0.5 * RRtGRt[e];
  for (int64_t i = 0; i < n; ++i)
    for (int64_t j = 0; j < n; ++j) Y[i * n + j] = Gh[i * n + j] - Gh[j * n + i];
  free(GRt), free(RtGRt), free(RRtGRt), free(Gh);
  return OR_OK;
}

/* R' of Sec. 3.2, R' = (I - a/2 Y)^-1 (I + a/2 Y) R, by the fixed-point
 * iteration the paper cites for it (Cayley SGD):
 *   R'_0 = R + a Y R,   R'_{k+1} = R + (a/2) Y (R + R'_k),  k = 0 .. iters-1,
 * whose fixed point solves (I - a/2 Y) R' = (I + a/2 Y) R.
 * Reading of the sign: the objective is an argmin, and the cited Cayley SGD
 * forms G_hat from the negative gradient (its momentum buffer accumulates
 * -grad); with G = +grad the printed update would climb the loss.  So `grad`
 * here is the loss gradient and Y is built from G = -grad.
 * A batch of independent (R, grad) pairs; Y_out (may be NULL) receives each Y. */
int oracle_cayley_step(const double* R, const double* grad, int64_t batch, int64_t n, double alpha, int iters,
                       double* R_out, double* Y_out) {
  if (n <= 0 || batch < 0 || iters < 0) return OR_EINVAL;
  int err = 0;
#pragma omp parallel for schedule(dynamic)
  for (int64_t b = 0; b < batch; ++b) {
    const double* Rb = R + b * n * n;
    double* Y = (double*)malloc(sizeof(double) * n * n);
    double* T = (double*)malloc(sizeof(double) * n * n);
    double* P = (double*)malloc(sizeof(double) * n * n);
    if (!Y || !T || !P) {
#pragma omp atomic write
      err = 1;
      free(Y), free(T), free(P);
      continue;
    }
    for (int64_t e = 0; e < n * n; ++e) T[e] = -grad[b * n * n + e]; /* G = -grad */
    if (oracle_cayley_y(Rb, T, n, Y) != OR_OK) {
#pragma omp atomic write
      err = 1;
      free(Y), free(T), free(P);
      continue;
    }
    mat_mul(Y, 0, Rb, 0, n, T); /* Y R */
    for (int64_t e = 0; e < n * n; ++e) P[e] = Rb[e] + alpha * T[e];
    for (int k = 0; k < iters; ++k) {
      for (int64_t e = 0; e < n * n; ++e) P[e] = Rb[e] + P[e]; /* R + R'_k */
      mat_mul(Y, 0, P, 0, n, T);                               /* Y (R + R'_k) */
      for (int64_t e = 0; e < n * n; ++e) P[e] = Rb[e] + 0.5 * alpha * T[e];
    }
    memcpy(R_out + b * n * n, P, sizeof(double) * n * n);
    if (Y_out) memcpy(Y_out + b * n * n, Y, sizeof(double) * n * n);
    free(Y), free(T), free(P);
  }
  return err ? OR_EINVAL : OR_OK;
}

/* ------------------------------------------------------------------ */
/* 8-bit variants: W4A8 and W-fp8-A-fp8 (main results table, 4-8-x    */
/* rows; appendix "Latency measurement on GPU", FP8 GEMM setting)      */
/* ------------------------------------------------------------------ */
/* E4M3 (the FP8 format of the FP8 setting, in its finite-only form):
 * 1 sign, 4 exponent (bias 7) and 3 mantissa bits; exponent field 0 holds
 * the subnormals m 2^-9; no infinities; 448 is the largest finite value and
 * S.1111.111 is NaN. */
double oracle_e4m3_to_double(uint8_t b) {
  const int s = b >> 7, e = (b >> 3) & 15, m = b & 7;
  if (e == 15 && m == 7) return NAN;
  const double v = e == 0 ? ldexp((double)m, -9) : ldexp(1.0 + m / 8.0, e - 7);
  return s ? -v : v;
}

/* Round to the nearest E4M3 value (ties to the even mantissa), saturating at
 * +-448; the sign of a value that rounds to zero is kept. */
uint8_t oracle_double_to_e4m3(double v) {
  const uint8_t sign = (v < 0 || (v == 0 && signbit(v))) ? 0x80 : 0;
  double a = fabs(v);
  if (a >= 448.0) return sign | 0x7E;
  int e2;
  frexp(a, &e2);                 /* a = f 2^e2, f in [0.5, 1) */
  int E = e2 - 1;                /* exponent of the leading bit */
  if (E < -6) E = -6;            /* the subnormal quantum 2^-9 */
  const double q = ldexp(1.0, E - 3);
  double r = nearbyint(a / q) * q;
  if (r > 448.0) r = 448.0;
  if (r == 0.0) return sign;
  if (r < ldexp(1.0, -6)) return sign | (uint8_t)(r / ldexp(1.0, -9));
  int e3;
  frexp(r, &e3);
  const int Er = e3 - 1;
  const int mant = (int)((r / ldexp(1.0, Er) - 1.0) * 8.0);
  return sign | (uint8_t)(((Er + 7) << 3) | mant);
}

void oracle_e4m3_array_to_double(const uint8_t* b, double* d, int64_t n) {
  for (int64_t i = 0; i < n; ++i) d[i] = oracle_e4m3_to_double(b[i]);
}

/* Per-row FP8 quantization (the FP8 setting's per-token / per-channel
 * scaling): alpha = clip * max|x| / 448, code = E4M3(x / alpha); a zero row
 * stores alpha = 0 and zero codes. */
int oracle_quantize_rows_e4m3(const double* x, int64_t rows, int64_t K, double clip, uint8_t* codes,
                              double* alpha) {
  if (rows < 0 || K <= 0 || !(clip > 0.0 && clip <= 1.0)) return OR_EINVAL;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < rows; ++r) {
    const double* xr = x + r * K;
    double mx = 0.0;
    for (int64_t k = 0; k < K; ++k) mx = fmax(mx, fabs(xr[k]));
    const double a = clip * mx / 448.0;
    alpha[r] = a;
    for (int64_t k = 0; k < K; ++k) codes[r * K + k] = a > 0.0 ? oracle_double_to_e4m3(xr[k] / a) : 0;
  }
  return OR_OK;
}

/* W4A8 linear: acc[m][n] = sum_k a_int * q_w with a_int = q (symmetric
 * 8-bit codes) or u - 128 (asymmetric), exact in int64 and checked to fit
 * int32; y = sum_k (alpha_m c_mk + beta_m)(s_n q_w,nk), the dequantized
 * product of the two Eq. 1 operands. */
int oracle_w4a8_gemm(const int32_t* a_codes, const double* a_scale, const double* a_zero,
                     const int32_t* w_codes, const double* w_scale, int64_t M, int64_t N, int64_t K,
                     int32_t* acc, double* y) {
  const int sym = a_zero == NULL;
  int err = 0;
#pragma omp parallel for schedule(static) collapse(2)
  for (int64_t m = 0; m < M; ++m)
    for (int64_t n = 0; n < N; ++n) {
      int64_t s = 0;
      double yy = 0.0;
      const int32_t* a = a_codes + m * K;
      const int32_t* w = w_codes + n * K;
      const double am = a_scale[m], bm = sym ? 0.0 : a_zero[m], sn = w_scale[n];
      for (int64_t k = 0; k < K; ++k) {
        s += (int64_t)(sym ? a[k] : a[k] - 128) * w[k];
        yy += (am * (double)a[k] + bm) * (sn * (double)w[k]);
      }
      if (s > INT32_MAX || s < INT32_MIN) {
#pragma omp atomic write
        err = 1;
      }
      acc[m * N + n] = (int32_t)s;
      y[m * N + n] = yy;
    }
  return err ? OR_EINVAL : OR_OK;
}

/* W-fp8-A-fp8 linear: y = sum_k (alpha_m a_mk)(s_n w_nk) with a, w the
 * decoded E4M3 codes. */
int oracle_fp8_gemm(const uint8_t* a_codes, const double* a_scale, const uint8_t* w_codes,
                    const double* w_scale, int64_t M, int64_t N, int64_t K, double* y) {
#pragma omp parallel for schedule(static) collapse(2)
  for (int64_t m = 0; m < M; ++m)
    for (int64_t n = 0; n < N; ++n) {
      double s = 0.0;
      for (int64_t k = 0; k < K; ++k)
        s += (a_scale[m] * oracle_e4m3_to_double(a_codes[m * K + k])) *
             (w_scale[n] * oracle_e4m3_to_double(w_codes[n * K + k]));
      y[m * N + n] = s;
    }
  return OR_OK;
}

/* ------------------------------------------------------------------ */
/* Decode attention over the 4-bit KV cache, and RoPE in front of R3   */
/* (Sec. 3.1: R3 rotates Q and K over head_dim so that the KV cache    */
/* quantizes to 4 bits; appendix "Latency measurement on GPU": decode  */
/* time per token)                                                     */
/* ------------------------------------------------------------------ */
/* Rotary position embedding of one head vector (the rotate-half form of
 * LLaMA): for i < D/2 with theta_i = base^(-2i/D) and angle p theta_i,
 *   y_i = x_i cos - x_{i+D/2} sin,   y_{i+D/2} = x_i sin + x_{i+D/2} cos.
 * rows x D values; pos[r] is the position of row r. */
int oracle_rope(const double* x, const int64_t* pos, int64_t rows, int64_t D, double base, double* y) {
  if (D <= 0 || D % 2 || rows < 0) return OR_EINVAL;
  const int64_t h = D / 2;
  for (int64_t r = 0; r < rows; ++r)
    for (int64_t i = 0; i < h; ++i) {
      const double th = pow(base, -2.0 * (double)i / (double)D);
      const double ang = (double)pos[r] * th;
      const double c = cos(ang), s = sin(ang);
      const double a = x[r * D + i], b = x[r * D + i + h];
      y[r * D + i] = a * c - b * s;
      y[r * D + i + h] = a * s + b * c;
    }
  return OR_OK;
}

/* Attention of one decode query per (batch, query head) over a cache of
 * dequantized keys and values:
 *   s_t = scale * q . k_t,  p = softmax_t(s) over t < len_b,  o = sum_t p_t v_t,
 * q [B][Hq][D], k, v [B][S][Hkv][D]; query head h reads kv head h / (Hq/Hkv). */
int oracle_decode_attention(const double* q, const double* k, const double* v, const int64_t* lens, int64_t B,
                            int64_t S, int64_t Hq, int64_t Hkv, int64_t D, double scale, double* o) {
  if (B < 0 || S <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv || D <= 0) return OR_EINVAL;
  int err = 0;
#pragma omp parallel for schedule(static) collapse(2)
  for (int64_t b = 0; b < B; ++b)
    for (int64_t h = 0; h < Hq; ++h) {
      const int64_t L = lens ? lens[b] : S;
      const int64_t hk = h / (Hq / Hkv);
      double* out = o + (b * Hq + h) * D;
      if (L <= 0 || L > S) {
#pragma omp atomic write
        err = 1;
        continue;
      }
      double* s = (double*)malloc(sizeof(double) * L);
      if (!s) {
#pragma omp atomic write
        err = 1;
        continue;
      }
      const double* qh = q + (b * Hq + h) * D;
      double mx = -INFINITY;
      for (int64_t t = 0; t < L; ++t) {
        const double* kt = k + ((b * S + t) * Hkv + hk) * D;
        double acc = 0.0;
        for (int64_t d = 0; d < D; ++d) acc += qh[d] * kt[d];
        s[t] = scale * acc;
        if (s[t] > mx) mx = s[t];
      }
      double den = 0.0;
      for (int64_t t = 0; t < L; ++t) den += exp(s[t] - mx);
      for (int64_t d = 0; d < D; ++d) out[d] = 0.0;
      for (int64_t t = 0; t < L; ++t) {
        const double p = exp(s[t] - mx) / den;
        const double* vt = v + ((b * S + t) * Hkv + hk) * D;
        for (int64_t d = 0; d < D; ++d) out[d] += p * vt[d];
      }
      free(s);
    }
  return err ? OR_EINVAL : OR_OK;
}
