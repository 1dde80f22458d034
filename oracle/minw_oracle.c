/*
 * minw_oracle.c -- plain CPU oracle for the MINW-Net inference path, the
 * AQE quantizer and the fp32 pieces of Algorithm 1's training step (arXiv
 * 2003.04296, "Propagating Asymptotic-Estimated Gradients for Low Bitwidth
 * Quantized Neural Networks").
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * definition the CUDA path is checked against.  Only tests/, the smoke()
 * entry of __graft_entry__ and the cpu_baseline leg of bench.py may load it.
 * It shares no code, header or table with the CUDA library and never calls it.
 *
 * Every routine is single-threaded, uses no SIMD and no blocking, and follows
 * the paper's definitions in the paper's order.  Floating point is fp64 except
 * where the value decides an integer (a quantized level) or is compared
 * bit-for-bit (the fp32 epilogue): there the fp32 operation is written out
 * (one IEEE multiply, one fmaf) because the kernel takes the same decision in
 * fp32.
 *
 * Readings of the paper used here (the paper is silent or garbled there):
 *   sign(0) = -1                      (Sec. II-A2, Eq. sign: "-1 otherwise")
 *   QNN bins: |u| <= D_q -> 0, D_{p+1} < |u| <= D_p -> +-2^-p, |u| > D_1 -> +-1
 *                                     (Eq. qnn, whose two branches both read "<=")
 *   zero padding is applied to the dequantized level tensor (paper silent)
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Level functions h(.)                                                      */
/* ------------------------------------------------------------------------ */

/* Eq. sign (Sec. II-A2): +1 if the input is positive, -1 otherwise. */
static double orc_sign(double u) { return (u > 0.0) ? 1.0 : -1.0; }

/* Eq. tnn (Sec. III-C): 0 if |u| <= delta, sign(u) otherwise. */
static double orc_tnn(double u, double delta)
{
    if (fabs(u) <= delta) return 0.0;
    return orc_sign(u);
}

/* Eq. qnn (Sec. III-C) for an n-bit QNN: q = 2^(n-1) - 1 descending thresholds
 * thr[0] = D_1 > thr[1] = D_2 > ... > thr[q-1] = D_q.  Levels are
 * sign(u) * 2^-p with p running from q-1 (just above D_q) down to 0 (above D_1),
 * and 0 at or below D_q.  n = 1 has no threshold and reduces to Eq. sign. */
double orc_qnn(double u, int n, const double *thr)
{
    int q = (1 << (n - 1)) - 1;
    if (q == 0) return orc_sign(u);
    double m = fabs(u);
    if (m <= thr[q - 1]) return 0.0;
    /* find the smallest p such that |u| > D_{p+1}: walk p = q-1 .. 0 */
    for (int p = q - 1; p >= 1; --p) {
        /* bin (D_{p+1}, D_p] -> 2^-p ; D_{p+1} = thr[p], D_p = thr[p-1] */
        if (m > thr[p] && m <= thr[p - 1]) return orc_sign(u) * ldexp(1.0, -p);
    }
    return orc_sign(u);                         /* |u| > D_1 -> 2^0 */
}

/* h for the three bit widths MINW-Net uses (Sec. IV-A: 1 bit -> Eq. sign,
 * 2 bit -> Eq. tnn, 3 bit -> Eq. qnn).  The input first goes through one fp32
 * multiply u = x * scale (scale = 1 reproduces the paper; a per-channel scale
 * maps latent weights onto [-1, 1], the range the paper clips weights to in
 * Algorithm 1).  Returns the dequantized level. */
double orc_h(float x, int bits, const float *thr, float scale)
{
    float u = x * scale;                        /* fp32, decides the level */
    double dthr[3] = {0.0, 0.0, 0.0};
    if (bits == 1) return orc_sign((double)u);
    if (bits == 2) return orc_tnn((double)u, (double)thr[0]);
    for (int j = 0; j < 3; ++j) dthr[j] = (double)thr[j];
    return orc_qnn((double)u, 3, dthr);
}

/* Quantize a tensor laid out as n_outer blocks of n_inner values; block i uses
 * scale[i] (scale == NULL -> 1).  Eq. inference: W^ = h(W), a^ = h(a). */
void orc_quantize(const float *x, int64_t n_outer, int64_t n_inner, int bits,
                  const float *thr, const float *scale, double *levels)
{
    for (int64_t i = 0; i < n_outer; ++i) {
        float s = scale ? scale[i] : 1.0f;
        for (int64_t j = 0; j < n_inner; ++j)
            levels[i * n_inner + j] = orc_h(x[i * n_inner + j], bits, thr, s);
    }
}

/* ------------------------------------------------------------------------ */
/* AQE forward / backward (Eq. ours, Eq. activation, Eq. weight)             */
/* ------------------------------------------------------------------------ */

/* Eq. ours / Eq. activation forward: h^ = alpha * h(a) + (1 - alpha) * a. */
void orc_aqe_forward(const float *x, int64_t n, double alpha, int bits,
                     const float *thr, float scale, double *y)
{
    for (int64_t i = 0; i < n; ++i) {
        double h = orc_h(x[i], bits, thr, scale);
        y[i] = alpha * h + (1.0 - alpha) * (double)x[i];
    }
}

/* Eq. activation / Eq. weight backward: dL/da = 2 alpha dL/dh 1[|a| <= 1]. */
void orc_aqe_backward(const float *x, const float *g, int64_t n, double alpha,
                      double *gx)
{
    for (int64_t i = 0; i < n; ++i) {
        double mask = (fabs((double)x[i]) <= 1.0) ? 1.0 : 0.0;
        gx[i] = 2.0 * alpha * (double)g[i] * mask;
    }
}

/* ------------------------------------------------------------------------ */
/* Training step pieces in the fp32 operations the step is defined with      */
/* (Algorithm 1): each is one IEEE operation per element, written out        */
/* ------------------------------------------------------------------------ */

/* Eq. activation / Eq. weight forward in fp32: fmaf(alpha, h(x), (1 - alpha) x)
 * with 1 - alpha and (1 - alpha) x each rounded to fp32. */
void orc_aqe_forward_f32(const float *x, int64_t n, float alpha, int bits, const float *thr, float scale, float *y)
{
    const float oma = 1.0f - alpha;
    for (int64_t i = 0; i < n; ++i) {
        const float h = (float)orc_h(x[i], bits, thr, scale);
        const float t = oma * x[i];
        y[i] = fmaf(alpha, h, t);
    }
}

/* Eq. activation / Eq. weight backward in fp32: (|x| <= 1) ? g (2 alpha) : 0. */
void orc_aqe_backward_f32(const float *x, const float *g, int64_t n, float alpha, float *gx)
{
    const float two_alpha = 2.0f * alpha;
    for (int64_t i = 0; i < n; ++i) gx[i] = (fabsf(x[i]) <= 1.0f) ? g[i] * two_alpha : 0.0f;
}

/* The update of Algorithm 1 with a plain gradient step and the clip:
 * w = min(1, max(-1, fmaf(-lr, g, w))). */
void orc_sgd_clip(float *w, const float *g, int64_t n, float lr)
{
    for (int64_t i = 0; i < n; ++i) w[i] = fminf(1.0f, fmaxf(-1.0f, fmaf(-lr, g[i], w[i])));
}

/* ------------------------------------------------------------------------ */
/* Stochastic AQE (Eq. our): h = alpha sign(a - z) + (1 - alpha) a, z ~ U[-1,1] */
/* ------------------------------------------------------------------------ */

/* Philox4x64-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as
 * easy as 1, 2, 3", SC 2011): ten rounds of two 64 x 64 -> 128-bit products
 * on the counter, the key bumped by the Weyl constants between rounds. */
void orc_philox4x64_10(const uint64_t ctr[4], const uint64_t key[2], uint64_t out[4])
{
    const uint64_t M0 = 0xD2E7470EE14C6C93ull, M1 = 0xCA5A826395121157ull;
    const uint64_t W0 = 0x9E3779B97F4A7C15ull, W1 = 0xBB67AE8584CAA73Bull;
    uint64_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    uint64_t k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; ++r) {
        const unsigned __int128 p0 = (unsigned __int128)M0 * c0;
        const unsigned __int128 p1 = (unsigned __int128)M1 * c2;
        const uint64_t hi0 = (uint64_t)(p0 >> 64), lo0 = (uint64_t)p0;
        const uint64_t hi1 = (uint64_t)(p1 >> 64), lo1 = (uint64_t)p1;
        c0 = hi1 ^ c1 ^ k0;
        c1 = lo1;
        c2 = hi0 ^ c3 ^ k1;
        c3 = lo0;
        k0 += W0;
        k1 += W1;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* The noise of element i: 32-bit word (i mod 8) of philox4x64_10(counter =
 * (offset + i / 8, 0, 0, 0), key = (seed, 0)) (words in order, low half of each
 * 64-bit output first), u -> z = (u >> 8) 2^-23 - 1, a point of the 2^-23 grid
 * on [-1, 1) (exact in fp32). */
float orc_noise(uint64_t i, uint64_t seed, uint64_t offset)
{
    const uint64_t ctr[4] = {offset + (i >> 3), 0, 0, 0};
    const uint64_t key[2] = {seed, 0};
    uint64_t r[4];
    orc_philox4x64_10(ctr, key, r);
    const uint64_t w = r[(i & 7) >> 1];
    const uint32_t u = (i & 1) ? (uint32_t)(w >> 32) : (uint32_t)w;
    return (float)((double)(u >> 8) * (1.0 / 8388608.0) - 1.0);
}

/* Eq. our with the sign of Eq. sign (sign(0) = -1): y in fp64, the noise and
 * the decision s = [a > z] exactly as drawn. */
void orc_aqe_forward_stochastic(const float *x, int64_t n, double alpha, uint64_t seed, uint64_t offset,
                                double *y, float *z)
{
    for (int64_t i = 0; i < n; ++i) {
        const float zi = orc_noise((uint64_t)i, seed, offset);
        const double s = ((double)x[i] - (double)zi > 0.0) ? 1.0 : -1.0;
        y[i] = alpha * s + (1.0 - alpha) * (double)x[i];
        if (z) z[i] = zi;
    }
}

/* ------------------------------------------------------------------------ */
/* Bit-plane packing of quantized levels                                     */
/* ------------------------------------------------------------------------ */

/* Number of bit-planes per value. */
int orc_planes(int bits) { return bits; }

/* Pack dequantized levels given in [N][C][H][W] order into planes laid out as
 * uint32 [N][H][W][P][ceil(C/32)], bit c%32 of word c/32 holding channel c.
 *   plane 0       : 1 iff the level is negative (1-bit: 1 iff level == -1)
 *   2-bit plane 1 : 1 iff the level is non-zero
 *   3-bit planes 1,2 : bits 0,1 of code k, |level| = 2^(k-3) for k > 0
 * Bits of channels >= C are 0.  The same routine packs weights [O][C][kh][kw]
 * into [O][kh][kw][P][ceil(C/32)]. */
void orc_pack(const double *lv, int N, int C, int H, int W, int bits,
              uint32_t *planes)
{
    int P = orc_planes(bits);
    int NW = (C + 31) / 32;
    memset(planes, 0, sizeof(uint32_t) * (size_t)N * H * W * P * NW);
    for (int n = 0; n < N; ++n)
        for (int c = 0; c < C; ++c)
            for (int y = 0; y < H; ++y)
                for (int x = 0; x < W; ++x) {
                    double v = lv[(((size_t)n * C + c) * H + y) * W + x];
                    uint32_t bit = 1u << (c % 32);
                    size_t pix = ((size_t)n * H + y) * W + x;
                    uint32_t *base = planes + pix * P * NW + c / 32;
                    if (v < 0.0) base[0] |= bit;
                    if (bits == 2 && v != 0.0) base[NW] |= bit;
                    if (bits == 3 && v != 0.0) {
                        double m = fabs(v);
                        int k = (m == 1.0) ? 3 : (m == 0.5) ? 2 : 1;
                        if (k & 1) base[NW] |= bit;
                        if (k & 2) base[2 * NW] |= bit;
                    }
                }
}

/* ------------------------------------------------------------------------ */
/* Convolution of dequantized levels (Algorithm 1, inference branch:        */
/* a~_l = a^q_{l-1} W^q_l)                                                   */
/* ------------------------------------------------------------------------ */

/* Direct convolution in fp64 of activation levels a [B][C][H][W] with weight
 * levels w [O][C][kh][kw], zero padding, then scaled by 2^units_shift to the
 * integer accumulator.  Returns 0 when every accumulator is an integer, -1
 * otherwise. */
int orc_conv2d(const double *a, int B, int C, int H, int W,
               const double *w, int O, int kh, int kw, int stride, int pad,
               int units_shift, int32_t *acc)
{
    int Ho = (H + 2 * pad - kh) / stride + 1;
    int Wo = (W + 2 * pad - kw) / stride + 1;
    int ok = 0;
    for (int b = 0; b < B; ++b)
        for (int o = 0; o < O; ++o)
            for (int yo = 0; yo < Ho; ++yo)
                for (int xo = 0; xo < Wo; ++xo) {
                    double s = 0.0;
                    for (int c = 0; c < C; ++c)
                        for (int ky = 0; ky < kh; ++ky)
                            for (int kx = 0; kx < kw; ++kx) {
                                int yi = yo * stride - pad + ky;
                                int xi = xo * stride - pad + kx;
                                if (yi < 0 || yi >= H || xi < 0 || xi >= W) continue;
                                s += a[(((size_t)b * C + c) * H + yi) * W + xi] *
                                     w[(((size_t)o * C + c) * kh + ky) * kw + kx];
                            }
                    double u = ldexp(s, units_shift);
                    if (u != floor(u)) ok = -1;
                    acc[(((size_t)b * O + o) * Ho + yo) * Wo + xo] = (int32_t)u;
                }
    return ok;
}

/* ------------------------------------------------------------------------ */
/* Weight-only quantized layers (Sec. IV: full-precision activations times  */
/* 1-3-bit weights, the XNOR / SHIFT ADDER rows of Tables II-IV)             */
/* ------------------------------------------------------------------------ */

/* bf16 of an fp32 value, round to nearest, ties to even (the 8 most
 * significant bits of the significand are kept): the fp32 value of it.
 * NaN stays NaN. */
float orc_bf16_round(float x)
{
    uint32_t u;
    memcpy(&u, &x, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return x;
    const uint32_t lsb = (u >> 16) & 1u;
    u = (u + 0x7FFFu + lsb) & 0xFFFF0000u;
    float r;
    memcpy(&r, &u, 4);
    return r;
}

/* orc_bf16_round over n values. */
void orc_bf16_round_array(const float *x, int64_t n, float *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = orc_bf16_round(x[i]);
}

/* Direct convolution in fp64 of real activations a [B][C][H][W] with weights
 * w [O][C][kh][kw], zero padding: the exact real-valued accumulator (every
 * product of a bf16 value and a level is exact, and so is the fp64 sum at
 * these sizes up to its own rounding). */
void orc_conv2d_real(const double *a, int B, int C, int H, int W,
                     const double *w, int O, int kh, int kw, int stride, int pad, double *out)
{
    int Ho = (H + 2 * pad - kh) / stride + 1;
    int Wo = (W + 2 * pad - kw) / stride + 1;
    for (int b = 0; b < B; ++b)
        for (int o = 0; o < O; ++o)
            for (int yo = 0; yo < Ho; ++yo)
                for (int xo = 0; xo < Wo; ++xo) {
                    double s = 0.0;
                    for (int c = 0; c < C; ++c)
                        for (int ky = 0; ky < kh; ++ky)
                            for (int kx = 0; kx < kw; ++kx) {
                                int yi = yo * stride - pad + ky;
                                int xi = xo * stride - pad + kx;
                                if (yi < 0 || yi >= H || xi < 0 || xi >= W) continue;
                                s += a[(((size_t)b * C + c) * H + yi) * W + xi] *
                                     w[(((size_t)o * C + c) * kh + ky) * kw + kx];
                            }
                    out[(((size_t)b * O + o) * Ho + yo) * Wo + xo] = s;
                }
}

/* The two backward products of Algorithm 1 for a convolutional layer whose
 * forward is orc_conv2d_real (a~ = a * W, zero padding), in fp64:
 *   input gradient  g_a[b][c][y][x]   = sum over (o, yo, xo, ky, kx) with
 *                   y = yo stride - pad + ky, x = xo stride - pad + kx of
 *                   g[b][o][yo][xo] w[o][c][ky][kx]
 *   weight gradient g_w[o][c][ky][kx] = sum over (b, yo, xo) of
 *                   g[b][o][yo][xo] a[b][c][yo stride - pad + ky][xo stride - pad + kx]
 *                   (taps outside the image contribute 0).
 * Both walk the forward's index map directly: every (output, tap) pair of the
 * forward adds its product to the input or weight it came from. */
void orc_conv2d_input_grad(const double *g, int B, int O, int Ho, int Wo,
                           const double *w, int C, int kh, int kw, int stride, int pad,
                           int H, int W, double *ga)
{
    for (size_t i = 0; i < (size_t)B * C * H * W; ++i) ga[i] = 0.0;
    for (int b = 0; b < B; ++b)
        for (int o = 0; o < O; ++o)
            for (int yo = 0; yo < Ho; ++yo)
                for (int xo = 0; xo < Wo; ++xo) {
                    const double gv = g[(((size_t)b * O + o) * Ho + yo) * Wo + xo];
                    for (int c = 0; c < C; ++c)
                        for (int ky = 0; ky < kh; ++ky)
                            for (int kx = 0; kx < kw; ++kx) {
                                int yi = yo * stride - pad + ky;
                                int xi = xo * stride - pad + kx;
                                if (yi < 0 || yi >= H || xi < 0 || xi >= W) continue;
                                ga[(((size_t)b * C + c) * H + yi) * W + xi] +=
                                    gv * w[(((size_t)o * C + c) * kh + ky) * kw + kx];
                            }
                }
}

void orc_conv2d_weight_grad(const double *g, int B, int O, int Ho, int Wo,
                            const double *a, int C, int H, int W, int kh, int kw, int stride, int pad,
                            double *gw)
{
    for (size_t i = 0; i < (size_t)O * C * kh * kw; ++i) gw[i] = 0.0;
    for (int b = 0; b < B; ++b)
        for (int o = 0; o < O; ++o)
            for (int yo = 0; yo < Ho; ++yo)
                for (int xo = 0; xo < Wo; ++xo) {
                    const double gv = g[(((size_t)b * O + o) * Ho + yo) * Wo + xo];
                    for (int c = 0; c < C; ++c)
                        for (int ky = 0; ky < kh; ++ky)
                            for (int kx = 0; kx < kw; ++kx) {
                                int yi = yo * stride - pad + ky;
                                int xi = xo * stride - pad + kx;
                                if (yi < 0 || yi >= H || xi < 0 || xi >= W) continue;
                                gw[(((size_t)o * C + c) * kh + ky) * kw + kx] +=
                                    gv * a[(((size_t)b * C + c) * H + yi) * W + xi];
                            }
                }
}

/* ------------------------------------------------------------------------ */
/* Layer pieces around the convolution (Sec. III-E)                          */
/* ------------------------------------------------------------------------ */

/* k x k max pooling with stride s over int32 [B][C][H][W]. */
void orc_maxpool_i32(const int32_t *in, int B, int C, int H, int W, int k, int s,
                     int32_t *out)
{
    int Ho = (H - k) / s + 1, Wo = (W - k) / s + 1;
    for (int b = 0; b < B; ++b)
        for (int c = 0; c < C; ++c)
            for (int y = 0; y < Ho; ++y)
                for (int x = 0; x < Wo; ++x) {
                    int32_t m = INT32_MIN;
                    for (int i = 0; i < k; ++i)
                        for (int j = 0; j < k; ++j) {
                            int32_t v = in[(((size_t)b * C + c) * H + y * s + i) * W + x * s + j];
                            if (v > m) m = v;
                        }
                    out[(((size_t)b * C + c) * Ho + y) * Wo + x] = m;
                }
}

/* k x k max pooling with stride s and padding p over fp32 [B][C][H][W]
 * (padded taps are skipped). */
void orc_maxpool_f32(const float *in, int B, int C, int H, int W, int k, int s,
                     int p, float *out)
{
    int Ho = (H + 2 * p - k) / s + 1, Wo = (W + 2 * p - k) / s + 1;
    for (int b = 0; b < B; ++b)
        for (int c = 0; c < C; ++c)
            for (int y = 0; y < Ho; ++y)
                for (int x = 0; x < Wo; ++x) {
                    float m = -INFINITY;
                    for (int i = 0; i < k; ++i)
                        for (int j = 0; j < k; ++j) {
                            int yi = y * s - p + i, xi = x * s - p + j;
                            if (yi < 0 || yi >= H || xi < 0 || xi >= W) continue;
                            float v = in[(((size_t)b * C + c) * H + yi) * W + xi];
                            if (v > m) m = v;
                        }
                    out[(((size_t)b * C + c) * Ho + y) * Wo + x] = m;
                }
}

/* Batch normalisation at inference as a per-channel affine map on the integer
 * accumulator: y = fmaf((float)acc, scale[c], shift[c]) over [B][C][HW]. */
void orc_affine_i32(const int32_t *acc, int B, int C, int HW, const float *scale,
                    const float *shift, float *y)
{
    for (int b = 0; b < B; ++b)
        for (int c = 0; c < C; ++c)
            for (int i = 0; i < HW; ++i) {
                size_t k = ((size_t)b * C + c) * HW + i;
                y[k] = fmaf((float)acc[k], scale[c], shift[c]);
            }
}

/* The same affine map on an fp32 input. */
void orc_affine_f32(const float *x, int B, int C, int HW, const float *scale,
                    const float *shift, float *y)
{
    for (int b = 0; b < B; ++b)
        for (int c = 0; c < C; ++c)
            for (int i = 0; i < HW; ++i) {
                size_t k = ((size_t)b * C + c) * HW + i;
                y[k] = fmaf(x[k], scale[c], shift[c]);
            }
}

/* HardTanh (Sec. III-E): max(-1, min(1, x)), in place. */
void orc_hardtanh(float *y, int64_t n)
{
    for (int64_t i = 0; i < n; ++i) {
        float v = y[i];
        if (v > 1.0f) v = 1.0f;
        if (v < -1.0f) v = -1.0f;
        y[i] = v;
    }
}

/* fp32 convolution whose input is not quantized (the first layer, Sec. III-E)
 * with fp32 weights (already quantized levels, or latent fp32 weights where a
 * layer keeps them).  Each output is one fmaf chain over (ci, ky, kx) in that
 * order, starting from 0, padded taps skipped. */
void orc_conv2d_f32_seq(const float *x, int B, int C, int H, int W, const float *w,
                        int O, int kh, int kw, int stride, int pad, float *out)
{
    int Ho = (H + 2 * pad - kh) / stride + 1;
    int Wo = (W + 2 * pad - kw) / stride + 1;
    for (int b = 0; b < B; ++b)
        for (int o = 0; o < O; ++o)
            for (int yo = 0; yo < Ho; ++yo)
                for (int xo = 0; xo < Wo; ++xo) {
                    float s = 0.0f;
                    for (int c = 0; c < C; ++c)
                        for (int ky = 0; ky < kh; ++ky)
                            for (int kx = 0; kx < kw; ++kx) {
                                int yi = yo * stride - pad + ky;
                                int xi = xo * stride - pad + kx;
                                if (yi < 0 || yi >= H || xi < 0 || xi >= W) continue;
                                s = fmaf(x[(((size_t)b * C + c) * H + yi) * W + xi],
                                         w[(((size_t)o * C + c) * kh + ky) * kw + kx], s);
                            }
                    out[(((size_t)b * O + o) * Ho + yo) * Wo + xo] = s;
                }
}

/* Global average pooling over [B][C][HW]: sequential fp32 sum, then one
 * division by HW. */
void orc_avgpool_f32(const float *x, int B, int C, int HW, float *out)
{
    for (int b = 0; b < B; ++b)
        for (int c = 0; c < C; ++c) {
            float s = 0.0f;
            for (int i = 0; i < HW; ++i) s += x[((size_t)b * C + c) * HW + i];
            out[(size_t)b * C + c] = s / (float)HW;
        }
}

/* Fully connected fp32 layer y[b][o] = sum_k x[b][k] w[o][k] + bias[o]: one
 * fmaf chain over k in order, bias added last. */
void orc_linear_f32_seq(const float *x, int B, int K, const float *w, int O,
                        const float *bias, float *y)
{
    for (int b = 0; b < B; ++b)
        for (int o = 0; o < O; ++o) {
            float s = 0.0f;
            for (int k = 0; k < K; ++k)
                s = fmaf(x[(size_t)b * K + k], w[(size_t)o * K + k], s);
            y[(size_t)b * O + o] = s + (bias ? bias[o] : 0.0f);
        }
}
