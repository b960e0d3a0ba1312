/*
 * shiftquant.h -- C ABI of the GB300 (sm_103a) ShiftQuant library, libshiftquant.so.
 *
 * ShiftQuant is the quantizer of "Towards Accurate and Efficient Sub-8-Bit Integer
 * Training" (arXiv 2411.10948).  One quantized linear layer Y = X W runs as
 *
 *   forward          Y  = X  W      X: ShiftQuant over its channels (the inner dim),
 *                                   W: per-out-channel                     (Sec. 5.1)
 *   loss propagation dX = dY W^T    dY: ShiftQuant over its channels (the inner dim),
 *                                   W: per-in-channel                       (Eq. 4)
 *   weight gradient  dW = X^T dY    both operands reuse their ShiftQuant codes; the
 *                                   inner dim is the token axis
 *
 * and each ShiftQuant tensor goes through: a range pass (per-channel max|x|, Sec. 3.1),
 * the power-of-two grouping (Eq. 3: channel c gets exponent e_c, its group, with
 * tau_0 2^-(e_c+1) < r_c <= tau_0 2^-e_c), and quantization with step
 * s 2^-e_c, s = tau_0 / Q, Q = 2^(b-1) - 1 (App. D).  The contraction applies the
 * group shift to every product before accumulation (ShiftMM, Sec. 3.2 and the
 * left-shift form of App. D), then one dequantizing multiply.
 *
 * Conventions for every entry point
 *   - Every pointer is a DEVICE pointer unless the argument says otherwise.  The caller
 *     owns every buffer; the library never allocates device memory and never
 *     synchronises.  Calls are asynchronous and ordered on `stream` (a cudaStream_t
 *     passed as void*; NULL is the legacy default stream).
 *   - Matrices are row-major with an explicit leading dimension `ld*` in ELEMENTS.
 *   - Host-detectable errors (bad sizes, NULL pointers, alignment, unsupported
 *     bit/group combinations) return a negative sq_status before anything is launched;
 *     shiftquant_last_error() then holds a message (per host thread).
 *   - Device-detected conditions are OR-ed into the caller's int32 `dev_status` word
 *     (SQ_DEV_* bits), which the caller zeroes and reads after synchronising.
 *   - Codes are the signed integers q, |q| <= Q, stored in the operand format of the
 *     float tensor-core MMA that multiplies them exactly (sm_103a has no integer MMA):
 *     one byte FP8 E4M3 or two bytes BF16, see shiftquant_code_type().  Every stored
 *     value is an integer (times a power of two for weight codes) and is exact.
 */
#ifndef SHIFTQUANT_H
#define SHIFTQUANT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int sq_status;
#define SQ_OK 0
#define SQ_EINVAL (-1)        /* bad size, NULL pointer, bad enum value */
#define SQ_EALIGN (-2)        /* pointer or leading dimension breaks a 16-byte rule */
#define SQ_EUNSUPPORTED (-3)  /* bit/group/size combination outside the exact range */
#define SQ_ECUDA (-4)         /* a CUDA runtime call failed (message has the name) */

/* bits OR-ed into *dev_status by the kernels */
#define SQ_DEV_NONFINITE 1    /* a NaN or Inf was met in the range pass */
#define SQ_DEV_TIMEOUT 2      /* a pipeline wait gave up (about 1 s); outputs invalid */
#define SQ_DEV_INTERNAL 4     /* a kernel precondition failed (shared-memory alignment) */

typedef enum { SQ_ROUND_NEAREST_EVEN = 0, SQ_ROUND_STOCHASTIC = 1 } sq_round;

/* Granularity of a quantizer call.
 *   SQ_GRAN_SHIFT   ShiftQuant over the columns (the channel axis) of an activation or
 *                   gradient [rows = tokens, cols = channels].
 *   SQ_GRAN_PER_COL one scale per column: a weight W [K, N] in the forward GEMM
 *                   (per-out-channel, Sec. 5.1).
 *   SQ_GRAN_PER_ROW one scale per row: a weight W [K, N] in the loss-propagation GEMM
 *                   (per-in-channel, Sec. 5.1). */
typedef enum { SQ_GRAN_SHIFT = 0, SQ_GRAN_PER_COL = 1, SQ_GRAN_PER_ROW = 2 } sq_gran;

typedef enum { SQ_CODE_E4M3 = 0, SQ_CODE_BF16 = 1 } sq_code_type;

/* Storage type of the codes for `bits` in [2, 8] and `n_groups` (N_G) in [1, 8]:
 * FP8 E4M3 when Q <= 15 and the largest shifted weight code Q 2^(N_G-1) <= 448 (the
 * exactly representable integers of E4M3), else BF16.  Returns a negative sq_status
 * for out-of-range arguments. */
int shiftquant_code_type(int bits, int n_groups);

/* Bytes per stored code (1 or 2), or a negative sq_status. */
int shiftquant_code_bytes(int bits, int n_groups);

/* Range pass and grouping (Sec. 3.1, Eq. 3).
 *   x [rows, ld] fp32.
 *   gran == SQ_GRAN_SHIFT: range_out[cols] = max_r |x[r, c]|, *tau0_out = max_c of it
 *     (r_max of Eq. 1), exp_out[cols] = e_c = min(n_groups-1, floor(log2(tau0/r_c)))
 *     computed exactly (a zero channel gets n_groups-1).
 *   gran == SQ_GRAN_PER_COL: range_out[cols] only; tau0_out and exp_out may be NULL.
 *   gran == SQ_GRAN_PER_ROW: range_out[rows] = max_c |x[r, c]|; the others may be NULL.
 *   A NaN/Inf anywhere sets SQ_DEV_NONFINITE; tau0 is then NaN or Inf and every e_c 0.
 *   rows or cols == 0 is allowed (tau0 = 0). */
sq_status shiftquant_calibrate(const float *x, int64_t rows, int64_t cols, int64_t ld,
                               int gran, int n_groups, float *range_out, float *tau0_out,
                               uint8_t *exp_out, int32_t *dev_status, void *stream);

/* Grouping alone (Eq. 3) from a given per-channel range vector:
 *   range[channels] fp32 (device, non-negative: max |x| per channel), *tau0_out = its
 *   maximum, exp_out[channels] = e_c exactly as shiftquant_calibrate with SQ_GRAN_SHIFT.
 *   A NaN/Inf range sets SQ_DEV_NONFINITE (tau0 NaN or Inf, every e_c 0).  channels == 0
 *   gives tau0 = 0.
 * Use: a tensor split by rows (tokens) across devices quantizes bit for bit as the whole
 *   would when every shard
 *   1. takes its per-column ranges (shiftquant_calibrate, SQ_GRAN_PER_COL),
 *   2. replaces them by their element-wise maximum over the shards (an all-reduce(max):
 *      exact, as a maximum of floats is),
 *   3. calls shiftquant_group on the result, and
 *   4. quantizes with SQ_GRAN_SHIFT, passing the shard's first row as row0 to
 *      shiftquant_quantize, so that stochastic rounding draws the whole tensor's numbers. */
sq_status shiftquant_group(const float *range, int64_t channels, int n_groups,
                           float *tau0_out, uint8_t *exp_out, int32_t *dev_status,
                           void *stream);

/* Quantization (App. D; stochastic rounding of App. B).
 *   x [rows, ld] fp32, bits in [2, 8], Q = 2^(bits-1) - 1.
 *   gran == SQ_GRAN_SHIFT: range_or_tau0 -> the device scalar tau_0 and exp[cols] from
 *     shiftquant_calibrate; q[r, c] = round(x 2^e_c Q / tau_0); *scale_out = tau_0 / Q.
 *     fold_exp must be NULL.
 *   gran == SQ_GRAN_PER_COL: range_or_tau0 -> range[cols]; q = round(x Q / range[c]);
 *     scale_out[cols] = range[c] / Q.  fold_exp, if not NULL, is indexed by ROW.
 *   gran == SQ_GRAN_PER_ROW: range_or_tau0 -> range[rows]; scale_out[rows].
 *     fold_exp, if not NULL, is indexed by COLUMN.
 *   fold_exp: the group exponents of the OTHER operand along this weight's GEMM inner
 *     index; the stored value becomes q 2^(n_groups-1-fold_exp[i]), which is how the
 *     ShiftMM shift of Eq. 4 enters the contraction at no cost.
 *   mode: SQ_ROUND_NEAREST_EVEN (ties to even) or SQ_ROUND_STOCHASTIC: up with
 *     probability frac(v) using u = (SplitMix64(seed + (idx+1) 0x9E3779B97F4A7C15) >> 40)
 *     2^-24, idx = (row0 + r) * cols + c.
 *   row0 (>= 0): the index of x's first row within the logical tensor.  0 for a whole
 *     tensor; a row (token) shard starting at row r0 passes r0 and draws exactly the
 *     numbers the whole tensor draws for those rows (see shiftquant_group).
 *   Outputs (codes in the type of shiftquant_code_type(bits, n_groups)):
 *     codes [rows, ld_codes] (may be NULL), codes_t [cols, ld_t], the transpose (may be
 *     NULL); at least one must be given.  tau_0 == 0 (or Q/tau_0 overflowing) gives
 *     all-zero codes and a zero scale; likewise per channel. */
sq_status shiftquant_quantize(const float *x, int64_t rows, int64_t cols, int64_t ld,
                              int gran, int bits, int n_groups, const float *range_or_tau0,
                              const uint8_t *exp, const uint8_t *fold_exp, int mode,
                              uint64_t seed, int64_t row0, void *codes, int64_t ld_codes,
                              void *codes_t, int64_t ld_t, float *scale_out, void *stream);

/* Both weight roles of a layer (Sec. 5.1) in two passes over W instead of four: the
 * range pass of the forward GEMM's per-out-channel scales and of loss propagation's
 * per-in-channel scales (Sec. 3.1 channel ranges) from one read of W.
 *   w [rows = K, ld] fp32 (rows: in-channels, cols: out-channels).
 *   range_out_ch[cols] = max_r |w[r, c]|, range_in_ch[rows] = max_c |w[r, c]|: bit for bit
 *     shiftquant_calibrate with SQ_GRAN_PER_COL and with SQ_GRAN_PER_ROW.
 *   A NaN/Inf sets SQ_DEV_NONFINITE.  rows or cols == 0 gives zero ranges. */
sq_status shiftquant_calibrate_weight(const float *w, int64_t rows, int64_t cols, int64_t ld,
                                      float *range_out_ch, float *range_in_ch,
                                      int32_t *dev_status, void *stream);

/* Both weight roles quantized from one read of W (App. D quantizer, round to nearest even;
 * Sec. 5.1 roles), with the ranges of shiftquant_calibrate_weight:
 *   codes_fwd [cols, ld_fwd], scale_fwd[cols]: the forward GEMM's per-out-channel codes,
 *     TRANSPOSED, with fold_fwd[rows] (the activation's exponents, or NULL) folded in --
 *     bit for bit shiftquant_quantize(w, SQ_GRAN_PER_COL, ..., fold_exp = fold_fwd,
 *     codes = NULL, codes_t = codes_fwd, ...).
 *   codes_dgrad [rows, ld_dgrad], scale_dgrad[rows]: loss propagation's per-in-channel
 *     codes with fold_dgrad[cols] (the gradient's exponents, or NULL) folded in -- bit for
 *     bit shiftquant_quantize(w, SQ_GRAN_PER_ROW, ..., fold_exp = fold_dgrad,
 *     codes = codes_dgrad, codes_t = NULL, ...).
 *   rows or cols == 0 gives zero scales and writes no code. */
sq_status shiftquant_quantize_weight(const float *w, int64_t rows, int64_t cols, int64_t ld,
                                     int bits, int n_groups, const float *range_out_ch,
                                     const float *range_in_ch, const uint8_t *fold_fwd,
                                     const uint8_t *fold_dgrad, void *codes_fwd, int64_t ld_fwd,
                                     float *scale_fwd, void *codes_dgrad, int64_t ld_dgrad,
                                     float *scale_dgrad, void *stream);

/* Group order of a GEMM inner index (Sec. 3.2's per-group GEMMs, done as one launch):
 * from exp[channels] (the exponents of shiftquant_calibrate / shiftquant_group), a stable
 * order with every group's channels contiguous and each group's segment starting on a
 * K-block boundary (128 bytes of codes: 64 BF16 or 128 E4M3 codes).
 *   pos_out[channels]: the position of each channel (int32, device);
 *   seg_out[2 n_groups + 1]: the segment starts seg[0..n_groups] in elements (seg[n_groups]
 *     = the padded width used) then the channel count of each group (int32, device).
 * In this layout each group of the contraction accumulates without a shift and its exact
 * sum is shifted once (shiftquant_gemm_layer with x_seg / g_seg): the per-chunk exact range
 * is that of unshifted products, so 8-bit codes work with any n_groups <= 8. */
sq_status shiftquant_group_order(const uint8_t *exp, int64_t channels, int bits, int n_groups,
                                 int32_t *pos_out, int32_t *seg_out, void *stream);

/* The largest padded width of a group order of `channels` channels (elements): the code
 * buffers of a group-ordered operand need at least this leading dimension.  -1 for
 * invalid arguments. */
int64_t shiftquant_group_order_width(int64_t channels, int bits, int n_groups);

/* shiftquant_quantize writing the codes of the GEMM inner index in a group order
 * (pos, seg of shiftquant_group_order over that index), the padding between segments set to
 * zero, and no folded shift (fold_exp is not taken):
 *   SQ_GRAN_SHIFT   codes [rows, ld_codes]: column c at pos[c] (the channels are the inner
 *                   index of the forward / loss-propagation GEMM); codes_t unchanged
 *   SQ_GRAN_PER_COL codes_t [cols, ld_t]: its column r (x's row) at pos[r] (W [K, N] in the
 *                   forward role, ordered by X's channels k); codes unchanged
 *   SQ_GRAN_PER_ROW codes [rows, ld_codes]: column n at pos[n] (W in the loss-propagation
 *                   role, ordered by dY's channels n); codes_t unchanged
 * The ordered output is required, with a leading dimension of at least
 * shiftquant_group_order_width(); every other argument is shiftquant_quantize's. */
sq_status shiftquant_quantize_ordered(const float *x, int64_t rows, int64_t cols, int64_t ld,
                                      int gran, int bits, int n_groups, const float *range_or_tau0,
                                      const uint8_t *exp, int mode, uint64_t seed, int64_t row0,
                                      const int32_t *pos, const int32_t *seg, void *codes,
                                      int64_t ld_codes, void *codes_t, int64_t ld_t,
                                      float *scale_out, void *stream);

/* Forward GEMM Y[M, N] = X[M, K] W[K, N] on quantized operands (Eq. 4 with the roles of
 * Sec. 5.1):
 *   a_codes [M, lda]: ShiftQuant codes of X (SQ_GRAN_SHIFT, unshifted), a_scale: device
 *     scalar s_X.
 *   b_codes [N, ldb]: per-out-channel codes of W stored TRANSPOSED (codes_t of a
 *     SQ_GRAN_PER_COL call with fold_exp = X's exponents), b_scale[N] = s_W.
 *   Result: T[m, n] = sum_k q_X[m, k] q_W[k, n] 2^(G-1-e_k) exactly (int32, see the
 *     limits below), Y = float(T) * (s_X 2^-(G-1) * s_W[n]).
 *   acc_out [M, ld_acc] int64 (may be NULL): T itself, for exactness checks.
 *   workspace: optional scratch of shiftquant_gemm_workspace_bytes() bytes (16-byte
 *     aligned); with it, a GEMM with too few output tiles splits K across SMs; NULL never
 *     splits.
 *   Alignment: lda * code_bytes and ldb * code_bytes multiples of 16, code pointers
 *     16-byte aligned (the operands are read by TMA).
 *   Exact range: T is exact for every K.  While max|q_X| max|q_W| 2^(G-1) K < 2^31 it is
 *     summed in int32.  Beyond that (8 bits, N_G = 4: K > 16642) the K loop is split into
 *     parts that each stay within int32 and the parts are added in int64 in the workspace,
 *     which is then required (its size, M N 8 bytes rounded up, is what
 *     shiftquant_gemm_workspace_bytes reports); without it the call returns
 *     SQ_EUNSUPPORTED.  One K block (64 or 128 inner elements) of worst-case products must
 *     stay within 2^24, the exact FP32 range of the tensor cores' sums (8 bits allows
 *     N_G <= 5); otherwise SQ_EUNSUPPORTED.  M, N or K == 0 is allowed. */
sq_status shiftquant_gemm_fwd(const void *a_codes, int64_t lda, const float *a_scale,
                              const void *b_codes, int64_t ldb, const float *b_scale,
                              int64_t M, int64_t N, int64_t K, int bits, int n_groups,
                              float *y, int64_t ldy, int64_t *acc_out, int64_t ld_acc,
                              void *workspace, size_t workspace_bytes, int32_t *dev_status,
                              void *stream);

/* Loss-propagation GEMM dX[M, K] = dY[M, N] W^T (Eq. 4 as printed):
 *   a_codes [M, lda]: ShiftQuant codes of dY (inner dim N), a_scale: s_dY.
 *   b_codes [K, ldb]: per-in-channel codes of W [K, N] in their natural layout (codes of
 *     a SQ_GRAN_PER_ROW call with fold_exp = dY's exponents), b_scale[K].
 *   In the argument list below the GEMM is written as out[M, N_out] = a [M, K_in] b^T with
 *   N_out = K (W's in-channels) and K_in = N (dY's channels); everything else is as for
 *   shiftquant_gemm_fwd. */
sq_status shiftquant_gemm_dgrad(const void *a_codes, int64_t lda, const float *a_scale,
                                const void *b_codes, int64_t ldb, const float *b_scale,
                                int64_t M, int64_t N_out, int64_t K_in, int bits,
                                int n_groups, float *dx, int64_t ldx, int64_t *acc_out,
                                int64_t ld_acc, void *workspace, size_t workspace_bytes,
                                int32_t *dev_status, void *stream);

/* Weight-gradient GEMM dW[Ci, Co] = X^T dY over T tokens:
 *   xt_codes [Ci, ldx]: the transposed ShiftQuant codes of X (codes_t), x_scale s_X,
 *     x_exp[Ci] its group exponents.
 *   gt_codes [Co, ldg]: the transposed ShiftQuant codes of dY, g_scale, g_exp[Co].
 *   Both channel axes are outer dims here, so each group shift applies to the whole
 *   inner sum: T[i, j] = (sum_t q_X[t, i] q_dY[t, j]) 2^((G-1-eX_i) + (G-1-eY_j)) and
 *   dW = float(sum) * (s_X s_dY) 2^-(eX_i + eY_j).  acc_out receives T (int64).
 *   Exact range as for shiftquant_gemm_fwd with max|q_X| max|q_dY| T in place of the
 *   forward bound (8 bits: int64 sums, with a workspace, beyond 133144 tokens). */
sq_status shiftquant_gemm_wgrad(const void *xt_codes, int64_t ldx, const float *x_scale,
                                const uint8_t *x_exp, const void *gt_codes, int64_t ldg,
                                const float *g_scale, const uint8_t *g_exp, int64_t Ci,
                                int64_t Co, int64_t T, int bits, int n_groups, float *dw,
                                int64_t ld_dw, int64_t *acc_out, int64_t ld_acc,
                                void *workspace, size_t workspace_bytes,
                                int32_t *dev_status, void *stream);

/* The weight gradient over tokens split across ranks, exact: each rank sums its own tokens
 * and the ranks add the integer sums before the one dequantizing multiply, so the result
 * is bit for bit shiftquant_gemm_wgrad's over all tokens.
 * shiftquant_gemm_wgrad_partial: the shard's raw sums
 *   t_out[i, j] = sum over the shard's T tokens of q_X[t, i] q_dY[t, j]
 *   (int32, dense [Ci, Co], 16-byte aligned, Co a multiple of 4), with the operands of
 *   shiftquant_gemm_wgrad (xt_codes [Ci, ldx], gt_codes [Co, ldg], unshifted codes; the
 *   scales and exponents are required as there, although the sums do not use them).  The
 *   exact range is checked for total_tokens, the tokens of all shards together, so that
 *   the all-reduce(sum) of the shards' t_out (int32) stays exact.
 * shiftquant_gemm_wgrad_finish: dw[i, j] = float(T[i, j]) 2^-(eX_i + eY_j) (s_X s_dY) from
 *   the summed T, and acc_out (may be NULL) = T << (2(G-1) - eX_i - eY_j) as int64. */
sq_status shiftquant_gemm_wgrad_partial(const void *xt_codes, int64_t ldx, const float *x_scale,
                                        const uint8_t *x_exp, const void *gt_codes, int64_t ldg,
                                        const float *g_scale, const uint8_t *g_exp, int64_t Ci,
                                        int64_t Co, int64_t T, int64_t total_tokens, int bits,
                                        int n_groups, int32_t *t_out, int32_t *dev_status,
                                        void *stream);
sq_status shiftquant_gemm_wgrad_finish(const int32_t *t, int64_t Ci, int64_t Co, int bits,
                                       int n_groups, const float *x_scale, const uint8_t *x_exp,
                                       const float *g_scale, const uint8_t *g_exp, float *dw,
                                       int64_t ld_dw, int64_t *acc_out, int64_t ld_acc,
                                       int32_t *dev_status, void *stream);

/* The three GEMMs of one quantized linear layer in ONE persistent launch.  They are
 * independent (each reads only codes produced before the call), so their output tiles share
 * the SMs: the work units of all three form one list, the GEMM with the longest K loop per
 * unit first.  Semantics, layouts and limits of every part are those of
 * shiftquant_gemm_fwd / _dgrad / _wgrad with these operands (X [M, K], W [K, N],
 * dY [M, N]; all codes with the same bits and n_groups):
 *   forward            y [M, N]  from x_codes [M, K] and wf_codes [N, K] (per-out-channel W
 *                      codes, transposed, X's shifts folded in), scales x_scale, wf_scale[N]
 *   loss propagation   dx [M, K] from g_codes [M, N] and wd_codes [K, N] (per-in-channel W
 *                      codes, dY's shifts folded in), scales g_scale, wd_scale[K]
 *   weight gradient    dw [K, N] from xt_codes [K, M] and gt_codes [N, M] with the exponents
 *                      x_exp[K], g_exp[N] and the scales x_scale, g_scale.  xt_codes NULL:
 *                      it reads x_codes [M, ld_x] in place (the tensor core takes the
 *                      operand MN-major), so X needs no transposed copy; gt_codes NULL
 *                      likewise reads g_codes.  Not with x_seg (g_seg): a group-ordered
 *                      operand's channels are permuted, and the call returns SQ_EINVAL.
 * acc_* are the optional int64 exactness-check outputs.  The struct lives in host memory and
 * is read during the call only.
 * The launch sizes the exact FP32 accumulation chunks of the forward and loss-propagation
 * GEMMs from x_exp and g_exp (a K block's products are bounded by max|q|^2 times its
 * channels' shifts): wf_codes and wd_codes must carry exactly the shifts 2^(G-1-e) of those
 * exponents, as shiftquant_quantize with fold_exp = x_exp / g_exp writes them, and every
 * code magnitude must be at most Q = 2^(bits-1) - 1. */
typedef struct {
  const void *x_codes;  int64_t ld_x;
  const void *xt_codes; int64_t ld_xt;
  const float *x_scale; const uint8_t *x_exp;
  const void *g_codes;  int64_t ld_g;
  const void *gt_codes; int64_t ld_gt;
  const float *g_scale; const uint8_t *g_exp;
  const void *wf_codes; int64_t ld_wf; const float *wf_scale;
  const void *wd_codes; int64_t ld_wd; const float *wd_scale;
  int64_t M, K, N;
  int bits, n_groups;
  float *y;  int64_t ld_y;
  float *dx; int64_t ld_dx;
  float *dw; int64_t ld_dw;
  int64_t *acc_y;  int64_t ld_acc_y;
  int64_t *acc_dx; int64_t ld_acc_dx;
  int64_t *acc_dw; int64_t ld_acc_dw;
  /* Which GEMMs to run: bit 0 forward, bit 1 loss propagation, bit 2 weight gradient; 0 runs
   * all three.  Fields of GEMMs left out are not read. */
  int gemm_mask;
  /* At most this many CTAs (0: one per SM), for a launch that shares the GPU with work
   * running beside it on other streams. */
  int max_ctas;
  /* Optional (NULL: not formed): the range pass of the next consumer of an output, formed in
   * the GEMM's epilogue instead of a separate pass over the output (Sec. 3.1's channel
   * ranges): y_range[N] = max_m |y[m, n]|, dx_range[K] = max_m |dx[m, k]|, equal bit for bit
   * to shiftquant_calibrate(y or dx, SQ_GRAN_PER_COL).  The call zeroes them first.  When Y
   * is the next layer's activation (or dX the previous layer's gradient), shiftquant_group
   * on the range gives its tau_0 and exponents, and shiftquant_quantize follows without a
   * range pass. */
  float *y_range;
  float *dx_range;
  /* Optional (NULL: the folded layout above): the group order of the forward GEMM's inner
   * index (X's channels, x_seg) and of the loss-propagation GEMM's (dY's channels, g_seg):
   * the seg tables of shiftquant_group_order.  With x_seg, x_codes [M, ld_x] and wf_codes
   * [N, ld_wf] hold their K channels in that order over the padded width
   * shiftquant_group_order_width(K, bits, n_groups) (ld_x, ld_wf at least that), as
   * shiftquant_quantize_ordered writes them, and wf_codes carry NO folded shifts; each
   * group accumulates unshifted and its exact sum is shifted once.  g_seg likewise for
   * g_codes [M, ld_g] and wd_codes [K, ld_wd] over dY's N channels. */
  const int32_t *x_seg;
  const int32_t *g_seg;
} sq_layer_gemms;

/* workspace: optional int32 scratch of shiftquant_gemm_layer_workspace_bytes() bytes,
 * 16-byte aligned.  Its first 256 bytes hold the counter through which the CTAs take their
 * work units as they free up (the units of the three GEMMs differ in length); without a
 * workspace each CTA strides over the unit list.  After it, each GEMM with too few output
 * tiles for the SMs splits its K loop into its own region -- into fewer parts than alone,
 * as the other GEMMs of the launch keep the SMs busy. */
sq_status shiftquant_gemm_layer(const sq_layer_gemms *args, void *workspace,
                                size_t workspace_bytes, int32_t *dev_status, void *stream);

/* Bytes of workspace that let shiftquant_gemm_layer schedule its units dynamically and
 * split every GEMM that would benefit on the current device (at least 256), and hold the
 * int64 sums of a GEMM past the int32 range.  The _grouped form sizes a launch whose
 * forward and loss-propagation inner indices are both group-ordered (x_seg and g_seg;
 * K and N are the channel counts). */
size_t shiftquant_gemm_layer_workspace_bytes(int64_t M, int64_t K, int64_t N, int bits,
                                             int n_groups);
size_t shiftquant_gemm_layer_workspace_bytes_grouped(int64_t M, int64_t K, int64_t N, int bits,
                                                     int n_groups);

/* Number of kernels one shiftquant_gemm_layer call with this shape, workspace size and
 * gemm_mask launches on the current device: the GEMM launch, plus one output pass per GEMM
 * that splits its K loop (0 when every GEMM is empty; memsets are not counted).  -1 for
 * invalid arguments, a shape beyond the exact range, or no device. */
int shiftquant_gemm_layer_kernel_launches(int64_t M, int64_t K, int64_t N, int bits,
                                          int n_groups, size_t workspace_bytes, int gemm_mask);

/* Tile mode of one shiftquant_gemm_layer call with this shape and gemm_mask on the current
 * device: 1 when it runs on 2-CTA clusters with 256 x 256 tiles (cta_group::2 MMAs; chosen
 * when the launch's units average at least 26 K blocks), 0 when each CTA runs 128 x 256
 * tiles, -1 for invalid arguments, an empty launch, a shape beyond the exact range, or no
 * device.  Results do not depend on the mode. */
int shiftquant_gemm_layer_cta_pairs(int64_t M, int64_t K, int64_t N, int bits, int n_groups,
                                    int gemm_mask);

/* Layout advice for a layer's X and dY codes on the current device: 1 when the weight
 * gradient of shiftquant_gemm_layer (all three GEMMs, this shape) is expected to run as fast
 * on the codes in place (xt_codes / gt_codes NULL) as on transposed copies -- so the
 * quantizer can skip writing the copies; 0 when transposed copies are faster (an MN-major
 * operand slows the tensor core where it sets the launch's pace: CTA pairs, unsplit units
 * filling at least half the pairs, K loops of 64 blocks or more); -1 for invalid arguments,
 * a shape beyond the exact range, or no device.  Results do not depend on the choice. */
int shiftquant_gemm_layer_wgrad_in_place(int64_t M, int64_t K, int64_t N, int bits,
                                         int n_groups);

/* One training step of one quantized linear layer X [M, K], W [K, N], dY [M, N], with the
 * operand roles of the paper's setup (Sec. 5.1): every quantizer pass and the three GEMMs
 * (Eq. 4 with the left-shift form of App. D), in stream order:
 *   1. X:  range pass + grouping (Sec. 3.1, Eq. 3), codes and transposed codes, round to
 *          nearest even (App. D); xt_codes NULL writes no transposed copy, and the weight
 *          gradient reads x_codes in place (see sq_layer_gemms);
 *   2. dY: the same with stochastic rounding (App. B) drawn under `seed` (gt_codes NULL:
 *          likewise);
 *   3. W per out-channel (forward role): codes written transposed [N, K] with X's group
 *      shifts folded in; W per in-channel (loss-propagation role): codes [K, N] with dY's
 *      shifts folded in -- both roles by shiftquant_calibrate_weight and
 *      shiftquant_quantize_weight;
 *   4. the forward, loss-propagation and weight-gradient GEMMs as one launch
 *      (shiftquant_gemm_layer).
 * Every buffer is a caller-owned DEVICE buffer; the layouts are those of the calls above:
 *   x [M, K], w [K, N], dy [M, N], y [M, N], dx [M, K], dw [K, N]: fp32, dense row-major
 *     (leading dimension = row length).  x, w and dy are written only by the host variant.
 *   x_codes [M, ld_x], xt_codes [K, ld_xt] (or NULL), x_range[K], x_exp[K], x_tau0,
 *     x_scale (one float each); g_codes [M, ld_g], gt_codes [N, ld_gt] (or NULL), g_range[N],
 *     g_exp[N], g_tau0,
 *     g_scale; wf_codes [N, ld_wf], wf_range[N], wf_scale[N]; wd_codes [K, ld_wd],
 *     wd_range[K], wd_scale[K].  Codes in the type of shiftquant_code_type(bits, n_groups),
 *     rows 16-byte aligned (ld * code bytes a multiple of 16, pointers 16-byte aligned).
 *   workspace: optional, as for shiftquant_gemm_layer (shiftquant_gemm_layer_workspace_bytes).
 *   dev_status: the device status word (see the conventions above).
 * The struct lives in host memory and is read during the call only.  The quantizer and GEMM
 * launches run one after the other on `stream`; M, K or N == 0 does nothing. */
typedef struct {
  int64_t M, K, N;
  int bits, n_groups;
  float *x, *w, *dy;
  void *x_codes;  int64_t ld_x;
  void *xt_codes; int64_t ld_xt;
  float *x_range, *x_tau0, *x_scale; uint8_t *x_exp;
  void *g_codes;  int64_t ld_g;
  void *gt_codes; int64_t ld_gt;
  float *g_range, *g_tau0, *g_scale; uint8_t *g_exp;
  void *wf_codes; int64_t ld_wf; float *wf_range, *wf_scale;
  void *wd_codes; int64_t ld_wd; float *wd_range, *wd_scale;
  float *y, *dx, *dw;
  void *workspace; size_t workspace_bytes;
  int32_t *dev_status;
} sq_layer_step;

sq_status shiftquant_layer_step(const sq_layer_step *args, uint64_t seed, void *stream);

/* The same step fed from HOST memory and returned to it, all in the order of `stream`:
 * copies x_host [M, K], w_host [K, N] and dy_host [M, N] (fp32, dense) into args->x, w, dy,
 * runs shiftquant_layer_step, and copies y, dx, dw back into y_host [M, N], dx_host [M, K]
 * and dw_host [K, N].  A NULL host pointer skips that copy (an input already on the device,
 * an output left there).  The copies are cudaMemcpyAsync calls: with page-locked host memory
 * (cudaHostAlloc / cudaHostRegister) they overlap work on other streams, so a caller that
 * alternates two sets of device buffers on two streams overlaps one step's copies with the
 * other's compute; with pageable memory they still give the right result but block the
 * host.  The host outputs hold the results once the stream reaches the end of the call.
 * inputs_queued (may be NULL): a cudaEvent_t the caller created; it is recorded on `stream`
 * right after the input copies, so that the caller can queue the next call's copies behind
 * this call's (another stream waiting on the event) while this call computes and copies
 * back -- which keeps both directions of the host link busy. */
sq_status shiftquant_layer_step_host(const sq_layer_step *args, const float *x_host,
                                     const float *w_host, const float *dy_host, float *y_host,
                                     float *dx_host, float *dw_host, uint64_t seed,
                                     void *inputs_queued, void *stream);

/* The same step with its copies on their own streams: the input copies on copy_in_stream,
 * the step (shiftquant_layer_step) on `stream`, the copies back on copy_out_stream, joined
 * by caller-created cudaEvent_t handles:
 *   buffers_free (may be NULL): copy_in_stream waits for it before copying in -- the event
 *     of the previous call's copies back from these device buffers;
 *   inputs_in:   recorded on copy_in_stream after the input copies; `stream` waits for it;
 *   step_done:   recorded on `stream` after the step; copy_out_stream waits for it;
 *   outputs_out: recorded on copy_out_stream after the copies back (the host outputs hold
 *     the results, and the device buffers are free, once it completes).
 * A copy engine serves its copies in the order they were queued, so copies in queued on
 * one stream behind another call's copies back wait for them; with one stream for all
 * copies in and one for all copies back, a caller that alternates device buffer sets keeps
 * both directions of the host link busy while earlier steps compute.  Host pointers as in
 * shiftquant_layer_step_host (page-locked memory for overlap; NULL skips a copy); the three
 * streams may be the same stream. */
sq_status shiftquant_layer_step_host_split(const sq_layer_step *args, const float *x_host,
                                           const float *w_host, const float *dy_host,
                                           float *y_host, float *dx_host, float *dw_host,
                                           uint64_t seed, void *copy_in_stream, void *stream,
                                           void *copy_out_stream, void *buffers_free,
                                           void *inputs_in, void *step_done,
                                           void *outputs_out);

/* Weight-gradient GEMM for callers that cannot allocate device memory -- for instance a
 * plug-in running inside a host framework that owns every device allocation, or a
 * deployment whose device memory is fixed when the library is loaded.  The paper has no
 * counterpart: this is an allocation strategy, not part of the method.
 *   Arguments, results and limits are those of shiftquant_gemm_wgrad, minus the workspace.
 *   Scratch: instead of a caller workspace, the split-K int32 partial sums live in a 4 MiB
 *     array inside the library (`static __device__`, held by every GPU that loads the
 *     library until the process exits).  Ci * Co must not exceed 1048576; larger outputs
 *     return SQ_EUNSUPPORTED before anything is launched.  Past the int32 range (8 bits:
 *     more than 133144 tokens) the sums are int64 and Ci * Co may not exceed 524288.
 *   Nothing is allocated: no cudaMalloc, no cudaFree, no allocating library routine.
 *   Each call made outside stream capture looks up the array's device address
 *     (cudaGetSymbolAddress) with the call's device current, so a device reset between
 *     calls is harmless; a call made while its stream is being captured reuses the address
 *     of the device's last such lookup.  The first call on each device must therefore come
 *     before any stream capture begins (a first call during capture returns SQ_EINVAL).
 *   All calls on a device share the one array, and it keeps the last call's contents
 *     (each call clears the part it uses before use).  Two calls whose work overlaps on
 *     the GPU -- on different streams, or from different host threads -- race on it and
 *     give wrong results: order them on one stream. */
sq_status shiftquant_gemm_wgrad_static(const void *xt_codes, int64_t ldx, const float *x_scale,
                                       const uint8_t *x_exp, const void *gt_codes, int64_t ldg,
                                       const float *g_scale, const uint8_t *g_exp, int64_t Ci,
                                       int64_t Co, int64_t T, int bits, int n_groups,
                                       float *dw, int64_t ld_dw, int64_t *acc_out,
                                       int64_t ld_acc, int32_t *dev_status, void *stream);

/* Bytes of int32 scratch that lets a GEMM of this shape split its inner dimension across
 * SMs on the current device (0 when it would not split).  which: 0 fwd, 1 dgrad,
 * 2 wgrad; M, N are the output dims and K the inner dim. */
size_t shiftquant_gemm_workspace_bytes(int which, int64_t M, int64_t N, int64_t K,
                                       int bits, int n_groups);

/* Fully-quantized L1 batch normalization (Sec. 4; App. C), training mode, over x [rows,
 * channels] fp32 (row-major with leading dimension ld_x; the rows are a channel's batch
 * and spatial positions, N H W).  With the readings this library takes of the paper:
 *   - x quantized by ShiftQuant (bits, n_groups; round to nearest even) to int8 codes q,
 *     step s_c = s 2^-e_c per channel;
 *   - the mean onto the channel's code grid: m_c = round-half-even(sum_r q / rows),
 *     mu^q = m_c s_c, so that x^q - mu^q = (q - m_c) s_c exactly;
 *   - the L1 deviation sigma_c = (sum_r |q - m_c| / rows) s_c (mean absolute deviation);
 *   - sigma, gamma[channels] and beta[channels] each quantized to 8-bit symmetric codes on
 *     one per-tensor grid (step max / 127);
 *   - y = gamma^q ((x^q - mu^q) / sigma^q) + beta^q, and beta^q where sigma^q is 0.
 * Every channel sum is an exact integer and every other step one IEEE binary32 operation
 * in a fixed order, so results do not depend on the launch configuration.
 * state: a caller-owned device buffer of shiftquant_l1bn_state_bytes(rows, channels) bytes
 *   (16-byte aligned) that the forward fills and the backward reads and extends: the int8
 *   codes of x, row-major [rows, channels], at its start (kept for the backward, as a
 *   quantized activation is), then the gradient's codes, the channel sums and values.
 * rows >= 1 when channels >= 1; channels == 0 does nothing.  A NaN/Inf in x sets
 * SQ_DEV_NONFINITE. */
size_t shiftquant_l1bn_state_bytes(int64_t rows, int64_t channels);

sq_status shiftquant_l1bn_forward(const float *x, int64_t rows, int64_t channels, int64_t ld_x,
                                  const float *gamma, const float *beta, int bits,
                                  int n_groups, float *y, int64_t ld_y, void *state,
                                  size_t state_bytes, int32_t *dev_status, void *stream);

/* Backward of the layer above from dy [rows, channels] (leading dimension ld_dy) and the
 * state its forward left: dy quantized by ShiftQuant (bits, n_groups) with stochastic
 * rounding drawn under `seed` (element index r * channels + c) to int8 codes p, g = p t_c;
 * every quantizer passed straight through, the L1 normalization's chain rule
 *   dx = (gamma^q / sigma^q) (g - mean g - mean(g xhat) (sign(q - m) - mean sign(q - m)))
 * with xhat = (q - m) s_c / sigma^q, and dgamma[c] = sum_r g xhat, dbeta[c] = sum_r g (a
 * channel with sigma^q = 0 passes dx = 0 and dgamma = 0).  dx [rows, ld_dx]. */
sq_status shiftquant_l1bn_backward(const float *dy, int64_t rows, int64_t channels,
                                   int64_t ld_dy, int bits, int n_groups, uint64_t seed,
                                   void *state, size_t state_bytes, float *dx, int64_t ld_dx,
                                   float *dgamma, float *dbeta, int32_t *dev_status,
                                   void *stream);

/* Kernels one shiftquant_l1bn_forward (backward = 0) or _backward (1) call launches on the
 * current device: 1 for at most 1024 channels on a device that runs cooperative launches
 * (the passes then run as phases of one launch, separated by bounded grid barriers, after
 * one memset of the state's counter and range slots), else the chain of 9 (forward) or 7
 * (backward) kernels; 0 for no channels, -1 for a negative count or no device.  Results do
 * not depend on the form. */
int shiftquant_l1bn_kernel_launches(int64_t channels, int backward);

/* Self-test of the single-launch L1 batch normalization's grid barrier (failure path):
 * a cooperative launch of 8 blocks in which one block never arrives, so every block's
 * bounded wait runs out after about 1 s, ORs SQ_DEV_TIMEOUT into dev_status and returns;
 * the context stays usable.  scratch: 256 bytes of device memory (16-byte aligned), zeroed
 * here.  For tests of the failure path only. */
sq_status shiftquant_selftest_grid_barrier_timeout(void *scratch, int32_t *dev_status,
                                                   void *stream);

/* Packed sub-byte storage (Sec. 5.2: with N_G = 4 the grouping map takes exactly 2 bits).
 * The tensor cores read codes as E4M3 / BF16 (there is no integer MMA on sm_103a, and the
 * 4-bit float E2M1 lacks the integers 5 and 7), so the packed form is the storage of a
 * quantized tensor between its quantization and its use -- for instance the activation
 * codes kept for the backward pass, at half the bytes -- expanded before the GEMM.
 * shiftquant_pack_codes: codes [rows, ld] of bits <= 4 (the library's storage type for
 *   bits / n_groups; unshifted ShiftQuant codes, |q| <= 7) -> packed [rows, ld_packed]
 *   bytes, ld_packed >= ceil(cols / 2): element c of a row in byte c / 2, the low nibble
 *   for even c, as a 4-bit two's complement; an odd row's last high nibble is 0.  A code
 *   outside [-8, 7] (a shifted weight code) sets SQ_DEV_INTERNAL.
 * shiftquant_unpack_codes: the inverse, into codes [rows, ld] of the storage type. */
sq_status shiftquant_pack_codes(const void *codes, int64_t rows, int64_t cols, int64_t ld,
                                int bits, int n_groups, uint8_t *packed, int64_t ld_packed,
                                int32_t *dev_status, void *stream);
sq_status shiftquant_unpack_codes(const uint8_t *packed, int64_t ld_packed, int64_t rows,
                                  int64_t cols, int bits, int n_groups, void *codes, int64_t ld,
                                  void *stream);

/* The grouping map (each channel's exponent) in w-bit fields, w = 1, 2 or 4 for n_groups
 * <= 2, <= 4, <= 8 (2 bits at the default N_G = 4): channel c at bit (c mod (8 / w)) w of byte
 * c / (8 / w).  shiftquant_packed_groups_bytes gives the packed size (-1 for bad
 * arguments). */
int64_t shiftquant_packed_groups_bytes(int64_t channels, int n_groups);
sq_status shiftquant_pack_groups(const uint8_t *exp, int64_t channels, int n_groups,
                                 uint8_t *packed, void *stream);
sq_status shiftquant_unpack_groups(const uint8_t *packed, int64_t channels, int n_groups,
                                   uint8_t *exp, void *stream);

/* Failure-path self-test (for tests of the device-side timeout; the paper has no
 * counterpart).  One GEMM launch with the operands and layout of shiftquant_gemm_fwd whose
 * TMA producer arms every pipeline stage but issues no operand copy, so nothing is ever in
 * flight and the tensor-core issuer's bounded wait on the first stage runs out after about
 * 1 s.  The launch then records SQ_DEV_TIMEOUT in *dev_status, every role of every CTA
 * leaves through the abort path (no copy or MMA outstanding, tensor memory freed) and the
 * kernel returns; the CUDA context stays usable.  y is not written.  M, N and K must be in
 * [1, 4096]; the checks and limits of shiftquant_gemm_fwd apply otherwise. */
sq_status shiftquant_selftest_wait_timeout(const void *a_codes, int64_t lda, const float *a_scale,
                                           const void *b_codes, int64_t ldb, const float *b_scale,
                                           int64_t M, int64_t N, int64_t K, int bits,
                                           int n_groups, float *y, int64_t ldy,
                                           int32_t *dev_status, void *stream);

/* Static description of a status code. */
const char *shiftquant_status_string(sq_status status);

/* Message of the last host-side error on this thread ("" if none). */
const char *shiftquant_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SHIFTQUANT_H */
