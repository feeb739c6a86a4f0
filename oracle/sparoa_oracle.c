/*
 * SparOA oracle: a plain, slow, obviously correct CPU statement of what the
 * sparsity/intensity-dispatched operator path computes.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, includes or
 * calls this file; only the tests, the smoke check and the CPU-baseline leg of
 * the benchmark load it.  It shares no header, table or helper with the CUDA
 * path.
 *
 * Conventions
 *   - Activations and weights are bfloat16 bit patterns (uint16_t).  A
 *     bfloat16 is the upper half of an IEEE-754 binary32: 1 sign bit, 8
 *     exponent bits (bias 127), 7 fraction bits.
 *   - Every product and sum is taken in IEEE double (fp64); the library
 *     rounds to bf16 only where a caller asks for it (orc_f64_to_bf16).
 *   - Activations are NHWC; a conv/FC input is viewed as a matrix [R, C] with
 *     R = N*H*W (or M for a fully connected layer) and C = channels (or K).
 *   - Loops run in a fixed order (k_h, k_w, c_in) and are never blocked,
 *     fused or reordered.
 *
 * What each function follows (section / equation of the SparOA paper,
 * arXiv 2511.19457):
 *   orc_stats            Eq. 1 (sparsity = 1 - nonzeros / elements), Sec. 3.1
 *                        plus the occupancy bitmaps the zero-skipping kernels
 *                        consume (no paper counterpart; layout documented below)
 *   orc_conv_work/fc     Eq. 2 (computational intensity), Sec. 3.1, restated as
 *                        FLOPs per input byte (Sec. 1 and Sec. 4.1 describe the
 *                        intensity as FLOPs per unit of input data)
 *   orc_decide           the threshold rule of Sec. 2.2 / Sec. 3 with the
 *                        sparsity and intensity thresholds as plain parameters
 *   orc_conv2d / orc_fc  the operators themselves (Sec. 5.1 executes them);
 *                        skip_zeros = 1 drops every product whose activation is
 *                        an exact zero, which is what Sec. 2.1 means by skipping
 *                        zero-value operations "without affecting the output"
 *   orc_maxpool / orc_avgpool_global / orc_bn_act   textbook definitions of
 *                        the memory-bound operators the paper places in its
 *                        low-intensity quadrant (Sec. 2.2)
 *
 * Parity pins (tests/test_oracle_*.py) check this file against brute force on
 * tiny inputs, library routines (torch float64 conv2d/matmul, numpy), closed
 * forms of the FLOP counts, Table 2's ResNet-18 figure, and the invariant that
 * skip_zeros = 1 returns exactly the same doubles as skip_zeros = 0.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------ */
/* bfloat16 <-> double                                                      */
/* ------------------------------------------------------------------------ */

/* Exact value of a bfloat16 bit pattern. */
double orc_bf16_to_f64(uint16_t b)
{
    int sign = (b >> 15) & 1;
    int e = (b >> 7) & 0xFF;
    int f = b & 0x7F;
    double v;
    if (e == 0xFF)
        v = f ? NAN : INFINITY;
    else if (e == 0)
        v = ldexp((double)f, -126 - 7);            /* subnormal: f * 2^-133 */
    else
        v = ldexp((double)(128 + f), e - 127 - 7); /* 1.f * 2^(e-127)       */
    return sign ? -v : v;
}

/* Round a double to the nearest bfloat16, ties to even (IEEE-754 roundTiesToEven),
 * directly from the double (no intermediate binary32, so no double rounding).
 * Overflow rounds to infinity; NaN maps to the canonical quiet NaN 0x7FC0. */
uint16_t orc_f64_to_bf16(double v)
{
    if (isnan(v))
        return 0x7FC0;
    uint16_t sign = signbit(v) ? 0x8000 : 0;
    double a = fabs(v);
    if (isinf(a))
        return sign | 0x7F80;
    if (a == 0.0)
        return sign;
    int e;
    (void)frexp(a, &e);             /* a = m * 2^e, m in [0.5, 1) */
    int E = e - 1;                  /* a in [2^E, 2^(E+1))        */
    /* spacing of bf16 values around a: 2^(E-7) for normals, 2^-133 below 2^-126 */
    int qexp = (E < -126) ? -133 : E - 7;
    double q = ldexp(a, -qexp);     /* exact: power-of-two scaling */
    double fl = floor(q);
    double frac = q - fl;           /* exact */
    double r = fl;
    if (frac > 0.5 || (frac == 0.5 && fmod(fl, 2.0) != 0.0))
        r = fl + 1.0;
    double rv = ldexp(r, qexp);
    if (rv >= 0x1p128)
        return sign | 0x7F80;
    if (rv < 0x1p-126)              /* subnormal (or zero): fraction = r */
        return sign | (uint16_t)r;
    int e2;
    (void)frexp(rv, &e2);
    int E2 = e2 - 1;
    double mant = ldexp(rv, -(E2 - 7));      /* in [128, 256) */
    uint16_t frac7 = (uint16_t)(mant - 128.0);
    return sign | (uint16_t)((E2 + 127) << 7) | frac7;
}

void orc_f64_to_bf16_array(const double *in, uint16_t *out, int64_t n)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = orc_f64_to_bf16(in[i]);
}

void orc_bf16_to_f64_array(const uint16_t *in, double *out, int64_t n)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = orc_bf16_to_f64(in[i]);
}

/* c(O) of Eq. 1 counts non-zero elements.  Both signed zeros are zero; every
 * other pattern (subnormals, infinities, NaN) is non-zero. */
static int is_nonzero(uint16_t b) { return orc_bf16_to_f64(b) != 0.0 || isnan(orc_bf16_to_f64(b)); }

/* ------------------------------------------------------------------------ */
/* Eq. 1 statistics and occupancy bitmaps of a tensor viewed as [R, C]       */
/* ------------------------------------------------------------------------ */
/*
 * Outputs (all zero-initialised here):
 *   nnz                 c(O) of Eq. 1
 *   col_nnz[C]          non-zeros of each column
 *   tile_nnz[T]         non-zeros of each 64-column tile, T = ceil(C/64)
 *   row_bm[R*W64]       bit (t % 64) of word t/64 of row r is set iff row r has a
 *                       non-zero in columns [64t, min(64t+64, C)); W64 = ceil(T/64)
 *   blk_mask[RB*C32]    bit (c % 32) of word c/32 of block b is set iff column c has
 *                       a non-zero in rows [128b, min(128b+128, R));
 *                       RB = ceil(R/128), C32 = ceil(C/32)
 * Bits past the last column or row are zero; words are little-endian in bits.
 */
void orc_stats(const uint16_t *x, int64_t R, int64_t C, uint64_t *nnz,
               uint32_t *col_nnz, uint32_t *tile_nnz, uint64_t *row_bm,
               uint32_t *blk_mask)
{
    int64_t T = (C + 63) / 64;
    int64_t W64 = (T + 63) / 64;
    int64_t RB = (R + 127) / 128;
    int64_t C32 = (C + 31) / 32;
    uint64_t total = 0;
    memset(col_nnz, 0, sizeof(uint32_t) * (size_t)C);
    memset(tile_nnz, 0, sizeof(uint32_t) * (size_t)T);
    memset(row_bm, 0, sizeof(uint64_t) * (size_t)(R * W64));
    memset(blk_mask, 0, sizeof(uint32_t) * (size_t)(RB * C32));
    for (int64_t r = 0; r < R; ++r) {
        for (int64_t c = 0; c < C; ++c) {
            if (!is_nonzero(x[r * C + c]))
                continue;
            int64_t t = c / 64;
            total += 1;
            col_nnz[c] += 1;
            tile_nnz[t] += 1;
            row_bm[r * W64 + t / 64] |= (uint64_t)1 << (t % 64);
            blk_mask[(r / 128) * C32 + c / 32] |= (uint32_t)1 << (c % 32);
        }
    }
    *nnz = total;
}

/* ------------------------------------------------------------------------ */
/* Eq. 2: work of a convolution / fully connected operator                   */
/* ------------------------------------------------------------------------ */
/*
 * Eq. 2 writes I = K_h * K_w * C_in * C_out * H * W (a multiply-accumulate count
 * of one image).  The dispatch rule uses the intensity as FLOPs per byte of
 * input activation:
 *   flops       = 2 * N * H_out * W_out * C_out * (C_in / groups) * K_h * K_w
 *   input_bytes = N * H * W * C_in * sizeof(bf16)
 *   macs_eq2    = K_h * K_w * C_in * C_out * H_out * W_out   (Eq. 2 literally)
 */
void orc_conv_work(int64_t N, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                   int64_t kh, int64_t kw, int64_t stride, int64_t pad,
                   int64_t groups, uint64_t *flops, uint64_t *macs_eq2,
                   uint64_t *input_bytes, int64_t *Ho, int64_t *Wo)
{
    int64_t ho = (H + 2 * pad - kh) / stride + 1;
    int64_t wo = (W + 2 * pad - kw) / stride + 1;
    *Ho = ho;
    *Wo = wo;
    *flops = (uint64_t)2 * N * ho * wo * Cout * (Cin / groups) * kh * kw;
    *macs_eq2 = (uint64_t)kh * kw * Cin * Cout * ho * wo;
    *input_bytes = (uint64_t)N * H * W * Cin * 2;
}

/* A fully connected layer y[M,N] = x[M,K] W[N,K]^T is a 1x1 convolution of a
 * 1x1 image with M images: flops = 2*M*K*N, Eq. 2 gives K*N. */
void orc_fc_work(int64_t M, int64_t K, int64_t N, uint64_t *flops,
                 uint64_t *macs_eq2, uint64_t *input_bytes)
{
    *flops = (uint64_t)2 * M * K * N;
    *macs_eq2 = (uint64_t)K * N;
    *input_bytes = (uint64_t)M * K * 2;
}

/* ------------------------------------------------------------------------ */
/* Threshold rule                                                            */
/* ------------------------------------------------------------------------ */
/*
 * Path codes: 1 = dense tensor-core kernel, 2 = zero-skipping kernel.
 * force_path: 0 = rule, 1 = always dense, 2 = always zero-skip.
 * intensity_mode: 0 = compare FLOPs per input byte (fpb) with c_thr,
 *                 1 = compare the Eq. 2 count (macs_eq2) with c_thr.
 * Rule: the operator is zero-skipped when its zero fraction reaches s_thr,
 *   (double)(numel - nnz) >= s_thr * (double)numel;
 * otherwise it runs dense when its intensity reaches c_thr, else zero-skip.
 * Ties go to zero-skip on sparsity (>=) and to dense on intensity (>=).
 */
int orc_decide(uint64_t numel, uint64_t nnz, double fpb, uint64_t macs_eq2,
               double s_thr, double c_thr, int intensity_mode, int force_path)
{
    if (force_path == 1)
        return 1;
    if (force_path == 2)
        return 2;
    double zeros = (double)(numel - nnz);
    if (zeros >= s_thr * (double)numel)
        return 2;
    double intensity = intensity_mode == 1 ? (double)macs_eq2 : fpb;
    if (intensity >= c_thr)
        return 1;
    return 2;
}

/* ------------------------------------------------------------------------ */
/* Epilogue: + bias, batch norm, + residual, activation (all in fp64)        */
/* ------------------------------------------------------------------------ */
/* act: 0 = identity, 1 = ReLU, 2 = ReLU6, 3 = GELU (exact: v * Phi(v), Phi the
 * standard normal CDF, Phi(v) = (1 + erf(v / sqrt 2)) / 2).
 * bn (nullable) holds 4 rows of C values: gamma, beta, running mean, running var;
 * BN(v) = (v - mean) * gamma / sqrt(var + eps) + beta. */
static double epilogue(double acc, int64_t c, int64_t C, const float *bias,
                       const float *bn, double eps, const uint16_t *res_elem,
                       int act)
{
    double v = acc;
    if (bias)
        v += (double)bias[c];
    if (bn) {
        double gamma = bn[c], beta = bn[C + c], mean = bn[2 * C + c], var = bn[3 * C + c];
        v = (v - mean) * (gamma / sqrt(var + eps)) + beta;
    }
    if (res_elem)
        v += orc_bf16_to_f64(*res_elem);
    if (act == 1)
        v = v > 0.0 ? v : 0.0;
    else if (act == 2)
        v = v > 0.0 ? (v < 6.0 ? v : 6.0) : 0.0;
    else if (act == 3)
        v = 0.5 * v * (1.0 + erf(v / sqrt(2.0)));
    return v;
}

/* ------------------------------------------------------------------------ */
/* Convolution (NHWC), direct loops, fp64 accumulation                       */
/* ------------------------------------------------------------------------ */
/*
 * x  : [N, H, W, Cin] bf16
 * w  : [Cout, kh, kw, Cin/groups] bf16
 * res: [N, Ho, Wo, Cout] bf16 or NULL
 * y  : [N, Ho, Wo, Cout] double (before any bf16 rounding)
 * Padding positions contribute nothing (zero padding).  skip_zeros = 1 leaves
 * out every product whose activation is +0 or -0.
 */
void orc_conv2d(const uint16_t *x, int64_t N, int64_t H, int64_t W, int64_t Cin,
                const uint16_t *w, int64_t Cout, int64_t kh, int64_t kw,
                int64_t stride, int64_t pad, int64_t groups, const float *bias,
                const float *bn, double eps, const uint16_t *res, int act,
                int skip_zeros, double *y)
{
    int64_t Ho = (H + 2 * pad - kh) / stride + 1;
    int64_t Wo = (W + 2 * pad - kw) / stride + 1;
    int64_t cin_g = Cin / groups, cout_g = Cout / groups;
    int64_t P = N * Ho * Wo;
    /* exact values of the operands, converted once */
    int64_t nx = N * H * W * Cin, nw = Cout * kh * kw * cin_g;
    double *xd = (double *)malloc(sizeof(double) * (size_t)(nx > 0 ? nx : 1));
    double *wd = (double *)malloc(sizeof(double) * (size_t)(nw > 0 ? nw : 1));
    orc_bf16_to_f64_array(x, xd, nx);
    orc_bf16_to_f64_array(w, wd, nw);
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < P; ++p) {
        int64_t n = p / (Ho * Wo);
        int64_t oh = (p / Wo) % Ho;
        int64_t ow = p % Wo;
        for (int64_t co = 0; co < Cout; ++co) {
            int64_t g = co / cout_g;
            double acc = 0.0;
            for (int64_t r = 0; r < kh; ++r) {
                int64_t ih = oh * stride - pad + r;
                if (ih < 0 || ih >= H)
                    continue;
                for (int64_t s = 0; s < kw; ++s) {
                    int64_t iw = ow * stride - pad + s;
                    if (iw < 0 || iw >= W)
                        continue;
                    const double *xp = xd + ((n * H + ih) * W + iw) * Cin + g * cin_g;
                    const double *wp = wd + ((co * kh + r) * kw + s) * cin_g;
                    for (int64_t ci = 0; ci < cin_g; ++ci) {
                        if (skip_zeros && xp[ci] == 0.0)
                            continue;
                        acc += xp[ci] * wp[ci];
                    }
                }
            }
            y[p * Cout + co] = epilogue(acc, co, Cout, bias, bn, eps,
                                        res ? res + p * Cout + co : NULL, act);
        }
    }
    free(xd);
    free(wd);
}

/* Fully connected: y[M, Nout] = x[M, K] * W[Nout, K]^T, then the epilogue. */
void orc_fc(const uint16_t *x, int64_t M, int64_t K, const uint16_t *w,
            int64_t Nout, const float *bias, const float *bn, double eps,
            const uint16_t *res, int act, int skip_zeros, double *y)
{
    double *xd = (double *)malloc(sizeof(double) * (size_t)(M * K > 0 ? M * K : 1));
    double *wd = (double *)malloc(sizeof(double) * (size_t)(Nout * K > 0 ? Nout * K : 1));
    orc_bf16_to_f64_array(x, xd, M * K);
    orc_bf16_to_f64_array(w, wd, Nout * K);
#pragma omp parallel for schedule(static)
    for (int64_t m = 0; m < M; ++m) {
        for (int64_t n = 0; n < Nout; ++n) {
            double acc = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                double xv = xd[m * K + k];
                if (skip_zeros && xv == 0.0)
                    continue;
                acc += xv * wd[n * K + k];
            }
            y[m * Nout + n] = epilogue(acc, n, Nout, bias, bn, eps,
                                       res ? res + m * Nout + n : NULL, act);
        }
    }
    free(xd);
    free(wd);
}

/* ------------------------------------------------------------------------ */
/* Pooling and the standalone batch-norm/activation                          */
/* ------------------------------------------------------------------------ */
/* Max pooling, NHWC; padded positions are ignored (as if -infinity). */
void orc_maxpool(const uint16_t *x, int64_t N, int64_t H, int64_t W, int64_t C,
                 int64_t k, int64_t stride, int64_t pad, double *y)
{
    int64_t Ho = (H + 2 * pad - k) / stride + 1;
    int64_t Wo = (W + 2 * pad - k) / stride + 1;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < N * Ho * Wo; ++p) {
        int64_t n = p / (Ho * Wo), oh = (p / Wo) % Ho, ow = p % Wo;
        for (int64_t c = 0; c < C; ++c) {
            double m = -INFINITY;
            for (int64_t r = 0; r < k; ++r) {
                int64_t ih = oh * stride - pad + r;
                if (ih < 0 || ih >= H)
                    continue;
                for (int64_t s = 0; s < k; ++s) {
                    int64_t iw = ow * stride - pad + s;
                    if (iw < 0 || iw >= W)
                        continue;
                    double v = orc_bf16_to_f64(x[((n * H + ih) * W + iw) * C + c]);
                    if (v > m)
                        m = v;
                }
            }
            y[p * C + c] = m;
        }
    }
}

/* Global average pooling: y[n, c] = (sum over h, w of x[n, h, w, c]) / (H * W). */
void orc_avgpool_global(const uint16_t *x, int64_t N, int64_t H, int64_t W,
                        int64_t C, double *y)
{
    for (int64_t n = 0; n < N; ++n)
        for (int64_t c = 0; c < C; ++c) {
            double s = 0.0;
            for (int64_t h = 0; h < H; ++h)
                for (int64_t w = 0; w < W; ++w)
                    s += orc_bf16_to_f64(x[((n * H + h) * W + w) * C + c]);
            y[n * C + c] = s / (double)(H * W);
        }
}

/* Element-wise batch norm and activation over a [R, C] view. */
void orc_bn_act(const uint16_t *x, int64_t R, int64_t C, const float *bias,
                const float *bn, double eps, const uint16_t *res, int act,
                double *y)
{
    for (int64_t r = 0; r < R; ++r)
        for (int64_t c = 0; c < C; ++c)
            y[r * C + c] = epilogue(orc_bf16_to_f64(x[r * C + c]), c, C, bias, bn,
                                    eps, res ? res + r * C + c : NULL, act);
}

/* Threads the OpenMP loops above use (1 without OpenMP). */
int orc_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void orc_set_num_threads(int n)
{
#ifdef _OPENMP
    if (n > 0)
        omp_set_num_threads(n);
#else
    (void)n;
#endif
}
