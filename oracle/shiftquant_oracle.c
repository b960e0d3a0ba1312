/*
 * ShiftQuant CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously-correct restatement of the definitions of
 * "Towards Accurate and Efficient Sub-8-Bit Integer Training" (arXiv 2411.10948):
 *   - per-channel range and the power-of-two grouping        (Sec. 3.1, Eq. 1-3)
 *   - per-group quantization with step (tau_0 / B) * 2^-g     (App. D, first equation)
 *   - stochastic rounding SR(x)                              (App. B, Eq. "SR")
 *   - per-channel weight quantization by role                (Sec. 5.1 setup)
 *   - the integer contraction with a per-group shift         (Eq. 4 and the left-shift
 *     form of App. D)
 *
 * Only the test suite, the smoke check and the CPU-baseline leg of the benchmark may
 * load this library.  It shares no code, header or constant with the CUDA path.
 *
 * Arithmetic is IEEE binary32 where the method rounds (the build passes
 * -ffp-contract=off so no multiply-add is fused), int64 where it accumulates, and
 * binary64 only for the final dequantising multiply.
 *
 * Readings of the paper that this file takes (each is listed with its reason in the
 * design notes of the repository):
 *   R1  r_max (tau_0) is the MAXIMUM of the channel ranges.
 *   R2  The thresholds are tau_g = tau_0 * 2^-g; a channel goes to the 0-indexed group
 *       e = min(G-1, floor(log2(tau_0 / r))), i.e. tau_0 2^-(e+1) < r <= tau_0 2^-e,
 *       and the last group also takes everything below, zero channels included.
 *   R3  Group e quantizes with step s * 2^-e, s = tau_0 / Q, Q = 2^(b-1) - 1
 *       (symmetric signed codes; -2^(b-1) is never produced).
 *   R4  The range is max|x| (symmetric, zero point Z = 0).
 *   R5  Both round-to-nearest-even and stochastic rounding are provided.
 *   R6  SR draws u = (H(seed, idx) >> 40) * 2^-24 with H the SplitMix64 output
 *       function (Steele, Lea, Flood, OOPSLA 2014) applied to seed + (idx+1)*golden;
 *       idx = r*C + c in the logical [R, C] tensor.
 *   R7  Weight-gradient GEMM: both channel axes are outer dimensions, so the shifts
 *       of both operands apply to the whole inner sum.
 *   R8  tau_0 == 0, or Q/tau_0 not finite: every code is 0 and the scale is 0.
 *       A NaN or Inf in the input sets the non-finite status; exponents are then 0.
 *
 * The fully-quantized L1 batch normalization (Sec. 4, App. C) takes these readings:
 *   R12 sigma_1 of a channel is its mean absolute deviation (1/R) sum_r |x - mu| over the
 *       channel's R elements (App. C writes the L1 norm |x - mu|_1; as a batch statistic it
 *       is divided by the element count, as the L2 form is by its own).
 *   R13 "all input features, statistics and parameters are quantized" (Sec. 4; 8 bits in
 *       the paper's experiments): the input by ShiftQuant (round to nearest) to codes q with
 *       per-channel steps s_c; the mean onto the channel's own code grid,
 *       m_c = round-half-even(sum_r q / R), mu^q = m_c s_c, so that x^q - mu^q = (q - m) s_c
 *       is an integer code difference; sigma to 8-bit codes on one per-tensor grid,
 *       sigma^q = k_c (sigma_max / 127); gamma and beta to 8-bit symmetric per-tensor codes.
 *   R14 a channel whose sigma^q is 0 outputs beta^q (x-hat = 0) and passes no gradient.
 *   R15 backward: the incoming gradient by ShiftQuant with stochastic rounding, every
 *       quantizer passed straight through, and the chain rule of L1 normalization
 *       (sigma' = mean(sign(x - mu)) terms in place of L2's x-hat):
 *       dx = (gamma / sigma)(g - mean g - mean(g xhat) (sign(d) - mean sign(d))),
 *       dgamma = sum g xhat, dbeta = sum g.
 *   R16 the binary32 order of every per-channel and per-element step, written out in
 *       sqo_l1bn_forward / sqo_l1bn_backward; the sums over a channel are exact integers.
 *
 * Packed sub-byte storage (Sec. 5.2: with N_G = 4 the grouping map takes exactly 2 bits):
 *   R17 codes of at most 4 bits are stored two per byte as 4-bit two's complement: element c
 *       of a row in byte c / 2, the low nibble for even c and the high nibble for odd c; a
 *       row of C codes takes ceil(C / 2) bytes, an odd row's last high nibble is 0.
 *   R18 the grouping map stores each channel's exponent in w = 1, 2 or 4 bits (N_G <= 2,
 *       <= 4, <= 8: the smallest power-of-two field that holds N_G - 1, so that no field
 *       straddles a byte), 8 / w channels per byte, channel c at bit (c mod (8 / w)) w of
 *       byte c / (8 / w).
 */
#include <math.h>
#ifdef _OPENMP
#include <omp.h>
#endif
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define SQO_OK 0
#define SQO_NONFINITE 1

/* threads the OpenMP loops of this file use (reported beside oracle timings) */
int sqo_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ---------------------------------------------------------------- R6: hash */
/* SplitMix64 output function applied to the (idx+1)-th state of a generator seeded
 * with `seed`: the value equals the (idx+1)-th output of Vigna's splitmix64.c. */
uint64_t sqo_hash(uint64_t seed, uint64_t idx) {
    uint64_t z = seed + (idx + 1u) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* uniform draw on the 2^-24 grid in [0, 1) */
static float sqo_uniform24(uint64_t seed, uint64_t idx) {
    return (float)(sqo_hash(seed, idx) >> 40) * 0x1p-24f;
}

static int sqo_finite(float v) { return isfinite(v) != 0; }

/* ------------------------------------------------------- Sec. 3.1: ranges */
/* r_c = max_r |x[r, c]| for every column c (the channel axis of an activation or a
 * gradient, or the out-channel axis of a forward weight).  Returns SQO_NONFINITE if any
 * element is NaN or Inf (the range of that channel is then NaN or Inf too). */
int sqo_range_cols(const float *x, int64_t R, int64_t C, int64_t ld, float *range) {
    int bad = 0;
    for (int64_t c = 0; c < C; ++c) range[c] = 0.0f;
    for (int64_t r = 0; r < R; ++r) {
        for (int64_t c = 0; c < C; ++c) {
            float a = fabsf(x[r * ld + c]);
            if (!sqo_finite(a)) {
                bad = 1;
                if (isnan(a) || !isnan(range[c])) range[c] = a;
            } else if (!isnan(range[c]) && a > range[c]) {
                range[c] = a;
            }
        }
    }
    return bad ? SQO_NONFINITE : SQO_OK;
}

/* r_r = max_c |x[r, c]| for every row r (the in-channel axis of a weight used in the
 * loss-propagation GEMM). */
int sqo_range_rows(const float *x, int64_t R, int64_t C, int64_t ld, float *range) {
    int bad = 0;
    for (int64_t r = 0; r < R; ++r) {
        float m = 0.0f;
        for (int64_t c = 0; c < C; ++c) {
            float a = fabsf(x[r * ld + c]);
            if (!sqo_finite(a)) {
                bad = 1;
                if (isnan(a) || !isnan(m)) m = a;
            } else if (!isnan(m) && a > m) {
                m = a;
            }
        }
        range[r] = m;
    }
    return bad ? SQO_NONFINITE : SQO_OK;
}

/* ------------------------------------------- Eq. 3 (R1, R2): the grouping */
/* tau_0 = max_c r_c; e_c = min(G-1, floor(log2(tau_0 / r_c))), evaluated exactly from
 * the frexp decomposition tau_0 = m0 2^E0, r = m 2^E with m, m0 in [0.5, 1):
 * tau_0 / r = (m0 / m) 2^(E0-E) with m0/m in (1/2, 2), so the floor of its log2 is
 * E0 - E when m <= m0 and E0 - E - 1 when m > m0. */
int sqo_group(const float *range, int64_t C, int G, float *tau0_out, uint8_t *exp_out) {
    float tau0 = 0.0f;
    int bad = 0, has_nan = 0;
    for (int64_t c = 0; c < C; ++c) {
        float r = range[c];
        if (!sqo_finite(r)) {
            bad = 1;
            if (isnan(r)) has_nan = 1;
        } else if (r > tau0) {
            tau0 = r;
        }
    }
    if (bad) {
        *tau0_out = has_nan ? NAN : INFINITY;
        for (int64_t c = 0; c < C; ++c) exp_out[c] = 0;
        return SQO_NONFINITE;
    }
    *tau0_out = tau0;
    int E0 = 0;
    float m0 = frexpf(tau0, &E0);
    for (int64_t c = 0; c < C; ++c) {
        float r = range[c];
        int e;
        if (r == 0.0f) {
            e = G - 1; /* R2: the last group holds the zero channels */
        } else {
            int E = 0;
            float m = frexpf(r, &E);
            int k = E0 - E - (m > m0 ? 1 : 0);
            e = k < G - 1 ? k : G - 1;
        }
        exp_out[c] = (uint8_t)e;
    }
    return SQO_OK;
}

/* ---------------------------------------------- rounding (App. B, R5, R6) */
static int32_t sqo_round(float v, int mode, uint64_t seed, uint64_t idx, int32_t Q) {
    float q;
    if (mode == 0) {
        q = rintf(v); /* round half to even (default rounding mode) */
    } else {
        /* SR: lower level l = floor(v), upper l+1, up with probability v - l */
        float l = floorf(v);
        float frac = v - l; /* exact: v and l share the binade grid below 2^24 */
        q = (sqo_uniform24(seed, idx) < frac) ? l + 1.0f : l;
    }
    if (q > (float)Q) q = (float)Q;
    if (q < (float)-Q) q = (float)-Q;
    return (int32_t)q;
}

/* ------------------------------------------- App. D (R3): group quantizer */
/* code[r, c] = round(x[r, c] / ((tau_0 / Q) 2^-e_c)), computed as
 * fl(fl(x * 2^e_c) * fl(Q / tau_0)) then rounded; the first product is exact.
 * The R rows of x are rows row0 .. row0+R-1 of the logical tensor (a row shard of it):
 * stochastic rounding draws with the logical index (row0 + r) * C + c (R6). */
int sqo_quantize_shift(const float *x, int64_t R, int64_t C, int64_t ld, int bits, int G,
                       float tau0, const uint8_t *exp, int mode, uint64_t seed, int64_t row0,
                       int8_t *q, float *scale_out) {
    (void)G;
    const int32_t Q = (1 << (bits - 1)) - 1;
    float invS = (float)Q / tau0;
    int zero_mode = !(tau0 > 0.0f) || !sqo_finite(tau0) || !sqo_finite(invS);
    *scale_out = zero_mode ? 0.0f : tau0 / (float)Q;
    for (int64_t r = 0; r < R; ++r) {
        for (int64_t c = 0; c < C; ++c) {
            int32_t code = 0;
            if (!zero_mode) {
                float xs = ldexpf(x[r * ld + c], (int)exp[c]);
                float v = xs * invS;
                code = sqo_round(v, mode, seed, (uint64_t)((row0 + r) * C + c), Q);
            }
            q[r * C + c] = (int8_t)code;
        }
    }
    return SQO_OK;
}

/* ------------------------------------- Sec. 5.1: per-channel weights (R4) */
/* axis 0: one scale per column (per-out-channel, forward GEMM);
 * axis 1: one scale per row (per-in-channel, loss-propagation GEMM).
 * code = round(w * fl(Q / range)), scale = range / Q; a zero range gives zero codes. */
int sqo_quantize_channel(const float *x, int64_t R, int64_t C, int64_t ld, int bits,
                         int axis, const float *range, int mode, uint64_t seed, int8_t *q,
                         float *scale_out) {
    const int32_t Q = (1 << (bits - 1)) - 1;
    int64_t nch = axis == 0 ? C : R;
    for (int64_t i = 0; i < nch; ++i) {
        float inv = (float)Q / range[i];
        int zero = !(range[i] > 0.0f) || !sqo_finite(range[i]) || !sqo_finite(inv);
        scale_out[i] = zero ? 0.0f : range[i] / (float)Q;
    }
    for (int64_t r = 0; r < R; ++r) {
        for (int64_t c = 0; c < C; ++c) {
            int64_t ch = axis == 0 ? c : r;
            float rg = range[ch];
            float inv = (float)Q / rg;
            int32_t code = 0;
            if (rg > 0.0f && sqo_finite(rg) && sqo_finite(inv)) {
                float v = x[r * ld + c] * inv;
                code = sqo_round(v, mode, seed, (uint64_t)(r * C + c), Q);
            }
            q[r * C + c] = (int8_t)code;
        }
    }
    return SQO_OK;
}

/* ---------------------------------------- Eq. 4 / App. D: the contraction */
/* Forward, Y = X W.  X codes qA [M, K] (ShiftQuant over K), weight codes qW [K, N]
 * (per-out-channel).  The sum is split by group exactly as Eq. 4 writes it: for each
 * group g the integer partial product over the inner indices of P^g, then the partials
 * are combined with the left-shift of App. D, T = sum_g partial_g << (G-1-g), which is
 * 2^(G-1) times the right-shift form of Eq. 4.  Rows listed in `rows` (or all M when
 * rows == NULL) are written to T [n_rows, N]. */
void sqo_gemm_fwd(const int8_t *qA, const uint8_t *eA, const int8_t *qW, int64_t M,
                  int64_t N, int64_t K, int G, const int64_t *rows, int64_t n_rows,
                  int64_t *T) {
    if (rows == NULL) n_rows = M;
#pragma omp parallel
    {
        int64_t *part = (int64_t *)malloc(sizeof(int64_t) * (size_t)(N > 0 ? N : 1));
#pragma omp for schedule(dynamic, 4)
        for (int64_t i = 0; i < n_rows; ++i) {
            int64_t m = rows ? rows[i] : i;
            int64_t *out = T + i * N;
            for (int64_t n = 0; n < N; ++n) out[n] = 0;
            for (int g = 0; g < G; ++g) {
                for (int64_t n = 0; n < N; ++n) part[n] = 0;
                for (int64_t k = 0; k < K; ++k) {
                    if ((int)eA[k] != g) continue;
                    int64_t a = qA[m * K + k];
                    if (a == 0) continue;
                    const int8_t *wrow = qW + k * N;
                    for (int64_t n = 0; n < N; ++n) part[n] += a * (int64_t)wrow[n];
                }
                for (int64_t n = 0; n < N; ++n) out[n] += part[n] * ((int64_t)1 << (G - 1 - g));
            }
        }
        free(part);
    }
}

/* Loss propagation, G_A = G_B W^T (Eq. 4 as printed).  Gradient codes qY [M, N]
 * (ShiftQuant over N, the inner dimension here), weight codes qW [K, N]
 * (per-in-channel, one scale per row k).  T [n_rows, K]. */
void sqo_gemm_dgrad(const int8_t *qY, const uint8_t *eY, const int8_t *qW, int64_t M,
                    int64_t N, int64_t K, int G, const int64_t *rows, int64_t n_rows,
                    int64_t *T) {
    if (rows == NULL) n_rows = M;
#pragma omp parallel for schedule(dynamic, 4)
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t m = rows ? rows[i] : i;
        for (int64_t k = 0; k < K; ++k) {
            int64_t total = 0;
            for (int g = 0; g < G; ++g) {
                int64_t part = 0;
                for (int64_t j = 0; j < N; ++j) {
                    if ((int)eY[j] != g) continue;
                    part += (int64_t)qY[m * N + j] * (int64_t)qW[k * N + j];
                }
                total += part * ((int64_t)1 << (G - 1 - g));
            }
            T[i * K + k] = total;
        }
    }
}

/* Weight gradient, dW = X^T G_B (R7).  qX [M, K] (ShiftQuant over K), qY [M, N]
 * (ShiftQuant over N); the inner dimension is the token axis M, so channel i of X and
 * channel j of the gradient stay in one group each for the whole sum:
 * T[i, j] = (sum_m qX[m, i] qY[m, j]) << ((G-1-eX_i) + (G-1-eY_j)).
 * Channels listed in `rows` (or all K) are written to T [n_rows, N]. */
void sqo_gemm_wgrad(const int8_t *qX, const uint8_t *eX, const int8_t *qY,
                    const uint8_t *eY, int64_t M, int64_t K, int64_t N, int G,
                    const int64_t *rows, int64_t n_rows, int64_t *T) {
    if (rows == NULL) n_rows = K;
#pragma omp parallel
    {
        int64_t *acc = (int64_t *)malloc(sizeof(int64_t) * (size_t)(N > 0 ? N : 1));
#pragma omp for schedule(dynamic, 4)
        for (int64_t t = 0; t < n_rows; ++t) {
            int64_t i = rows ? rows[t] : t;
            for (int64_t j = 0; j < N; ++j) acc[j] = 0;
            for (int64_t m = 0; m < M; ++m) {
                int64_t a = qX[m * K + i];
                if (a == 0) continue;
                const int8_t *yrow = qY + m * N;
                for (int64_t j = 0; j < N; ++j) acc[j] += a * (int64_t)yrow[j];
            }
            for (int64_t j = 0; j < N; ++j) {
                int sh = (G - 1 - (int)eX[i]) + (G - 1 - (int)eY[j]);
                T[t * N + j] = acc[j] * ((int64_t)1 << sh);
            }
        }
        free(acc);
    }
}

/* --------------------------------------------------- Eq. 4: dequantization */
/* Y[i, j] = (float)( (double)T[i, j] * s_a * s_b * 2^-shift * col_scale[j] ), in binary64
 * up to the final rounding.  shift is G-1 for the forward and loss-propagation GEMMs
 * (one shifted operand, s_b = 1, col_scale = the weight's per-channel scales) and
 * 2(G-1) for the weight-gradient GEMM (s_a = s_X, s_b = s_G, col_scale == NULL). */
void sqo_dequant(const int64_t *T, int64_t rows, int64_t cols, float s_a, float s_b,
                 int shift, const float *col_scale, float *Y) {
    double base = (double)s_a * (double)s_b * ldexp(1.0, -shift);
    for (int64_t i = 0; i < rows; ++i)
        for (int64_t j = 0; j < cols; ++j) {
            double f = col_scale ? (double)col_scale[j] : 1.0;
            Y[i * cols + j] = (float)((double)T[i * cols + j] * base * f);
        }
}

/* ---------------------------------- Sec. 4, App. C: fully-quantized L1 BatchNorm */
/* round-half-even of the rational a / b (b > 0), in integers */
static int64_t sqo_rne_div(int64_t a, int64_t b) {
    int64_t q = a / b, r = a % b;
    if (r < 0) { q -= 1; r += b; }          /* floor division: 0 <= r < b */
    if (2 * r > b || (2 * r == b && (q & 1))) q += 1;
    return q;
}

/* symmetric 8-bit per-tensor quantization of a vector v[n] (R13): returns each v^q */
static void sqo_quant8_tensor(const float *v, int64_t n, float *vq) {
    float vmax = 0.0f;
    for (int64_t i = 0; i < n; ++i) if (fabsf(v[i]) > vmax) vmax = fabsf(v[i]);
    float inv = 127.0f / vmax, step = vmax / 127.0f;
    int zero = !(vmax > 0.0f) || !sqo_finite(inv);
    for (int64_t i = 0; i < n; ++i) {
        float k = zero ? 0.0f : rintf(v[i] * inv);
        if (k > 127.0f) k = 127.0f;
        if (k < -127.0f) k = -127.0f;
        vq[i] = k * step;
    }
}

/* Forward of the fully-quantized L1 BatchNorm over x [R, C] (channels = columns, the R rows
 * are the batch and spatial positions).  Outputs: q [R, C] the input's ShiftQuant codes,
 * y [R, C], stats [3, C] = (sum q, sum |q - m|, sum sign(q - m)) and chan [6, C] =
 * (s_c, m_c, sigma_c, sigma^q_c, gamma^q_c, beta^q_c).  Returns the input's status. */
int sqo_l1bn_forward(const float *x, int64_t R, int64_t C, int bits, int G, const float *gamma,
                     const float *beta, int8_t *q, float *y, int64_t *stats, float *chan) {
    float *rng = (float *)malloc(sizeof(float) * (size_t)(C > 0 ? C : 1));
    uint8_t *e = (uint8_t *)malloc((size_t)(C > 0 ? C : 1));
    float tau0 = 0.0f, scale = 0.0f;
    int st = sqo_range_cols(x, R, C, C, rng);
    st |= sqo_group(rng, C, G, &tau0, e);
    sqo_quantize_shift(x, R, C, C, bits, G, tau0, e, 0, 0, 0, q, &scale);
    float *s_c = chan, *m_c = chan + C, *sig = chan + 2 * C, *sq = chan + 3 * C;
    float *gq = chan + 4 * C, *bq = chan + 5 * C;
    const float Rf = (float)R;
    for (int64_t c = 0; c < C; ++c) {
        int64_t S1 = 0, S = 0, Z = 0;
        for (int64_t r = 0; r < R; ++r) S1 += q[r * C + c];
        const int64_t m = R > 0 ? sqo_rne_div(S1, R) : 0;            /* mu^q = m s_c */
        for (int64_t r = 0; r < R; ++r) {
            const int64_t d = q[r * C + c] - m;
            S += d < 0 ? -d : d;
            Z += (d > 0) - (d < 0);
        }
        stats[c] = S1;
        stats[C + c] = S;
        stats[2 * C + c] = Z;
        s_c[c] = ldexpf(scale, -(int)e[c]);                             /* step of channel c */
        m_c[c] = (float)m;
        sig[c] = ((float)S / Rf) * s_c[c];                              /* sigma_1 (R12) */
    }
    /* sigma^q on one 8-bit grid over the channels (sigma >= 0) */
    sqo_quant8_tensor(sig, C, sq);
    sqo_quant8_tensor(gamma, C, gq);
    sqo_quant8_tensor(beta, C, bq);
    for (int64_t r = 0; r < R; ++r) {
        for (int64_t c = 0; c < C; ++c) {
            const float xq = (float)q[r * C + c] * s_c[c];              /* x^q, exact */
            const float mq = m_c[c] * s_c[c];                           /* mu^q, exact */
            const float xhat = sq[c] > 0.0f ? (xq - mq) / sq[c] : 0.0f; /* R14 */
            y[r * C + c] = gq[c] * xhat + bq[c];
        }
    }
    free(rng);
    free(e);
    return st;
}

/* Backward (R15) from the incoming gradient gy [R, C], the forward's codes q, stats and
 * chan.  Outputs: p [R, C] the gradient's ShiftQuant codes (stochastic rounding under
 * `seed`), dx [R, C], dgamma [C], dbeta [C].  Returns the gradient's status. */
int sqo_l1bn_backward(const float *gy, int64_t R, int64_t C, int bits, int G, uint64_t seed,
                      const int8_t *q, const int64_t *stats, const float *chan, int8_t *p,
                      float *dx, float *dgamma, float *dbeta) {
    float *rng = (float *)malloc(sizeof(float) * (size_t)(C > 0 ? C : 1));
    uint8_t *e = (uint8_t *)malloc((size_t)(C > 0 ? C : 1));
    float tau0 = 0.0f, scale = 0.0f;
    int st = sqo_range_cols(gy, R, C, C, rng);
    st |= sqo_group(rng, C, G, &tau0, e);
    sqo_quantize_shift(gy, R, C, C, bits, G, tau0, e, 1, seed, 0, p, &scale);
    const float *s_c = chan, *m_c = chan + C, *sq = chan + 3 * C, *gq = chan + 4 * C;
    const float Rf = (float)R;
    for (int64_t c = 0; c < C; ++c) {
        const int64_t m = (int64_t)m_c[c];
        int64_t P = 0, D = 0;
        for (int64_t r = 0; r < R; ++r) {
            P += p[r * C + c];
            D += (int64_t)p[r * C + c] * (q[r * C + c] - m);
        }
        const float t = ldexpf(scale, -(int)e[c]);                      /* step of g's channel */
        const float u = sq[c] > 0.0f ? gq[c] / sq[c] : 0.0f;            /* gamma / sigma */
        const float mg = ((float)P * t) / Rf;                           /* mean g */
        const float dg = sq[c] > 0.0f ? (((float)D * t) * s_c[c]) / sq[c] : 0.0f;
        const float mgx = dg / Rf;                                      /* mean(g xhat) */
        const float zs = (float)stats[2 * C + c] / Rf;                  /* mean sign(d) */
        dgamma[c] = dg;
        dbeta[c] = (float)P * t;
        for (int64_t r = 0; r < R; ++r) {
            const int64_t d = q[r * C + c] - m;
            const float g = (float)p[r * C + c] * t;
            const float sg = (float)((d > 0) - (d < 0));
            dx[r * C + c] = u * ((g - mg) - mgx * (sg - zs));
        }
    }
    free(rng);
    free(e);
    return st;
}

/* ------------------------------- Sec. 5.2 (R17, R18): packed sub-byte storage */
void sqo_pack4(const int8_t *q, int64_t R, int64_t C, uint8_t *out) {
    const int64_t W = (C + 1) / 2;
    for (int64_t r = 0; r < R; ++r)
        for (int64_t b = 0; b < W; ++b) {
            const int lo = q[r * C + 2 * b];
            const int hi = 2 * b + 1 < C ? q[r * C + 2 * b + 1] : 0;
            out[r * W + b] = (uint8_t)((lo & 0xF) | ((hi & 0xF) << 4));
        }
}

void sqo_unpack4(const uint8_t *in, int64_t R, int64_t C, int8_t *q) {
    const int64_t W = (C + 1) / 2;
    for (int64_t r = 0; r < R; ++r)
        for (int64_t c = 0; c < C; ++c) {
            const int nib = (in[r * W + c / 2] >> (4 * (c & 1))) & 0xF;
            q[r * C + c] = (int8_t)(nib >= 8 ? nib - 16 : nib);     /* two's complement */
        }
}

static int sqo_group_bits(int G) { return G <= 2 ? 1 : (G <= 4 ? 2 : 4); }

void sqo_pack_groups(const uint8_t *e, int64_t C, int G, uint8_t *out) {
    const int w = sqo_group_bits(G), per = 8 / w;
    const int64_t W = (C + per - 1) / per;
    for (int64_t b = 0; b < W; ++b) out[b] = 0;
    for (int64_t c = 0; c < C; ++c)
        out[c / per] |= (uint8_t)((e[c] & ((1 << w) - 1)) << ((c % per) * w));
}

void sqo_unpack_groups(const uint8_t *in, int64_t C, int G, uint8_t *e) {
    const int w = sqo_group_bits(G), per = 8 / w;
    for (int64_t c = 0; c < C; ++c)
        e[c] = (uint8_t)((in[c / per] >> ((c % per) * w)) & ((1 << w) - 1));
}
