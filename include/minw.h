/*
 * minw.h -- C ABI of libminw.so: the MINW-Net low-bit inference hot path and
 * the AQE quantizer of "Propagating Asymptotic-Estimated Gradients for Low
 * Bitwidth Quantized Neural Networks" (arXiv 2003.04296), on one GB300
 * (sm_103a).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every pointer argument is a DEVICE pointer unless its comment says host.
 *   The caller allocates and frees all tensors; only a minw_net owns memory.
 * - Calls are asynchronous on the given CUDA stream (`stream` is a
 *   cudaStream_t passed as void*; NULL = legacy default stream).  The return
 *   value reports argument validation and launch errors only.
 * - Device-side failures (a bounded wait that ran out) are latched in a
 *   device flag and read with minw_get_last_device_error().
 * - No call allocates device memory except minw_net_create.
 * - Tensors are dense and row-major in the order written; device pointers
 *   must be 16-byte aligned.
 *
 * Packed bit-plane layout ("planes")
 * ----------------------------------
 * A quantized tensor with `bits` in {1,2,3} is stored as uint32 words
 *     [N][H][W][P][NW],  P = bits, NW = ceil(C/32),
 * bit (c % 32) of word (c / 32) holding channel c; bits of channels >= C are 0.
 *   plane 0           : 1 iff the level is negative (1-bit: 1 iff level = -1)
 *   2-bit plane 1     : 1 iff the level is non-zero
 *   3-bit planes 1, 2 : bits 0 and 1 of the magnitude code k,
 *                       |level| = 2^(k-3) for k in {1,2,3}, 0 for k = 0
 * Levels (Sec. IV-A): 1 bit {-1, 1} (Eq. sign), 2 bit {-1, 0, 1} (Eq. tnn),
 * 3 bit {0, +-1/4, +-1/2, +-1} (Eq. qnn).  Weights [O][C][kh][kw] pack to
 * [O][kh][kw][P][NW] (the same layout with N = O, H = kh, W = kw).
 *
 * Integer accumulators
 * --------------------
 * A convolution of quantized operands returns the exact integer
 *     acc = (sum over valid taps of a_level * w_level) * 2^(f_a + f_w),
 * f = 2 for a 3-bit operand, 0 otherwise (3-bit levels are multiples of 1/4).
 * Zero padding contributes nothing (padding of the dequantized tensor).
 */
#ifndef MINW_H
#define MINW_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define MINW_API __attribute__((visibility("default")))
#else
#define MINW_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MINW_OK = 0,
    MINW_EINVAL = 1,          /* bad argument: null pointer, size, alignment, bits */
    MINW_EUNSUPPORTED = 2,    /* valid request outside what the kernels cover */
    MINW_ECUDA = 3,           /* a CUDA runtime call or launch failed */
    MINW_ETIMEOUT = 4,        /* a bounded device-side wait ran out */
    MINW_EDEVICE = 5          /* no usable sm_103a device */
} minw_status;

/* Quantizer h of Eq. sign / Eq. tnn / Eq. qnn applied to u = x * scale
 * (one fp32 multiply; scale = 1 is the paper's quantizer).
 *   bits 1: level = +1 if u > 0, -1 otherwise (sign(0) = -1).
 *   bits 2: level = 0 if |u| <= thr[0], sign(u) otherwise.
 *   bits 3: |u| <= thr[2] -> 0; thr[2] < |u| <= thr[1] -> +-1/4;
 *           thr[1] < |u| <= thr[0] -> +-1/2; |u| > thr[0] -> +-1.
 * thr must be descending; unused entries are ignored.  Host struct. */
typedef struct {
    int32_t bits;
    float thr[3];
    float scale;
} minw_quant;

/* Human-readable name of a status code (static string). */
MINW_API const char *minw_status_string(minw_status s);

/* Version of the library as MAJOR*10000 + MINOR*100 + PATCH. */
MINW_API int32_t minw_version(void);

/* ---------------------------------------------------------------------- */
/* AQE elementwise (Sec. III-C, Eq. activation / Eq. weight, Eq. ours)     */
/* ---------------------------------------------------------------------- */

/* AQE forward, Eq. ours: y = alpha * h(x) + (1 - alpha) * x, evaluated in
 * fp32 as fmaf(alpha, h(x * q->scale), (1 - alpha) * x).
 * x, y: n floats (may alias).  alpha in [0, 1].  q: host pointer.
 * Errors: MINW_EINVAL for n < 0, null pointers, misalignment, bad q. */
MINW_API minw_status aqe_forward(const float *x, float *y, int64_t n, float alpha,
                        const minw_quant *q, void *stream);

/* Stochastic AQE forward, Eq. our (Sec. III-A): y = alpha * sign(x - z) +
 * (1 - alpha) * x with z ~ U[-1, 1) and sign(0) = -1, evaluated in fp32 as
 * fmaf(alpha, x > z ? 1 : -1, (1 - alpha) * x).  The noise of element i is a
 * pure function of (seed, offset, i): 32-bit word i mod 8 of
 * Philox4x64-10(counter = (offset + i / 8, 0, 0, 0), key = (seed, 0))
 * (Salmon et al., SC 2011; the low half of each 64-bit output first), mapped
 * to z = (u >> 8) * 2^-23 - 1.  Successive calls advance offset by
 * ceil(n / 8) for fresh noise.  x, y: n floats (may alias), 16-byte aligned.
 * Errors: MINW_EINVAL for n < 0, null pointers, misalignment, alpha outside
 * [0, 1].  The backward is aqe_backward (Eq. activation). */
MINW_API minw_status aqe_forward_stochastic(const float *x, float *y, int64_t n, float alpha,
                                            uint64_t seed, uint64_t offset, void *stream);

/* AQE backward, Eq. activation / Eq. weight:
 * gx = (|x| <= 1) ? gy * (2 * alpha) : 0   (fp32, one rounding).
 * x, gy, gx: n floats (gx may alias gy). */
MINW_API minw_status aqe_backward(const float *x, const float *gy, float *gx,
                         int64_t n, float alpha, void *stream);

/* Quantize + pack (Eq. inference: a^ = h(a)) with the AQE forward and the
 * backward mask of Eq. activation fused into the same pass over x.
 * x: fp32 NCHW [B][C][H][W].  planes: packed layout above (q->bits planes).
 * y (nullable): AQE forward output at `alpha`, NCHW fp32, as aqe_forward.
 * mask (nullable): 1 bit per element of x in flat NCHW order,
 *   bit (i % 32) of word (i / 32) = 1[|x_i| <= 1]; ceil(B*C*H*W/32) words.
 * Errors: MINW_EINVAL for non-positive sizes, null x/planes, bad q. */
MINW_API minw_status aqe_quantize_pack(const float *x, int32_t B, int32_t C, int32_t H,
                              int32_t W, const minw_quant *q, uint32_t *planes,
                              float alpha, float *y, uint32_t *mask,
                              void *stream);

/* AQE backward from the packed mask written by aqe_quantize_pack:
 * gx_i = bit_i(mask) ? gy_i * (2 * alpha) : 0, n elements. */
MINW_API minw_status aqe_backward_masked(const uint32_t *mask, const float *gy,
                                float *gx, int64_t n, float alpha,
                                void *stream);

/* Quantize + pack latent weights w [O][C][kh][kw] (Eq. inference:
 * W^ = h(W)) into planes [O][kh][kw][q->bits][ceil(C/32)].
 * channel_scale (nullable): per-output-channel multiplier replacing
 * q->scale, u = w * channel_scale[o]. */
MINW_API minw_status minw_pack_weights(const float *w, int32_t O, int32_t C, int32_t kh,
                              int32_t kw, const minw_quant *q,
                              const float *channel_scale, uint32_t *planes,
                              void *stream);

/* ---------------------------------------------------------------------- */
/* Quantized convolution (Algorithm 1, inference: a~ = a^q W^q)            */
/* ---------------------------------------------------------------------- */

enum {
    MINW_VARIANT_AUTO = 0,    /* per-shape choice from measurements: at creation a network times each
                                 layer the tensor cores cover with E4M3 operands, with E2M1 operands,
                                 with E2M1 operands as CTA pairs of 128-channel tiles or as single-CTA
                                 128-channel tiles, and on the popcount path (bit-planes), and keeps
                                 the fastest (the times stay
                                 readable through minw_net_layer_candidates); the popcount path
                                 where the tensor cores do not apply */
    MINW_VARIANT_POPC = 1,    /* bit-serial XNOR/AND + popcount on the integer pipe */
    MINW_VARIANT_TC = 2,      /* tcgen05 tensor cores on exact level values: E2M1 operands where
                                 the shape allows (C % 128 == 0), else E4M3 */
    MINW_VARIANT_TC_E4M3 = 3, /* tensor cores on E4M3 operands only (a network request) */
    MINW_VARIANT_TC_E2M1 = 4, /* tensor cores on E2M1 operands where the shape allows (a network
                                 request, as MINW_VARIANT_TC); reported for a layer on E2M1 operands */
    MINW_VARIANT_TC_E2M1_PAIRS = 5, /* E2M1 operands as CTA pairs of 256 pixels x 128 channels where the
                                 shape allows (output channels a multiple of 128, no K split): two
                                 accumulators per CTA, so each tile's epilogue overlaps the next
                                 tile's MMAs (a network request; reported for such a layer) */
    MINW_VARIANT_TC_E2M1_N128 = 6  /* E2M1 operands on single CTAs with 128-channel tiles (layers with
                                 more than 128 output channels and pixel-major tiles): two accumulators
                                 per CTA at half the MMA width (a network request; reported for such a
                                 layer) */
};

/* Convolution of packed activations act [B][H][W][bits_a][C/32] with packed
 * weights wgt [O][kh][kw][bits_w][C/32]; C must be a multiple of 32.
 * Output size Ho = (H + 2 pad - kh)/stride + 1, Wo likewise.
 * acc_out (nullable): int32 NCHW [B][O][Ho][Wo], the exact accumulator.
 * y_out (nullable): fp32 NCHW, y = fmaf((float)acc, scale[o], shift[o]);
 *   scale/shift (length O) are required when y_out is given.
 * variant: MINW_VARIANT_*.  At least one output must be non-null.
 * Errors: MINW_EINVAL (sizes, pointers, bits), MINW_EUNSUPPORTED (C % 32,
 * a variant that does not cover the shape). */
MINW_API minw_status minw_conv2d(const uint32_t *act, int32_t B, int32_t C, int32_t H,
                        int32_t W, int32_t bits_a, const uint32_t *wgt,
                        int32_t O, int32_t kh, int32_t kw, int32_t bits_w,
                        int32_t stride, int32_t pad, int32_t *acc_out,
                        const float *scale, const float *shift, float *y_out,
                        int32_t variant, void *stream);

/* One MINW-Net block (Sec. III-E): QuantizedConv - [2x2/2 max pool] - BN -
 * HardTanh - quantize, the quantize + pack of the next layer's input fused
 * into the epilogue.  Pooling acts on the integer accumulator (the order the
 * paper's block prescribes); BN is y = fmaf((float)acc, scale[o], shift[o]).
 * pool: 0 or 1 (requires even Ho, Wo).
 * q_out (nullable, host): quantizer of the output; when given, the output is
 *   HardTanh'ed and packed into planes_out [B][Hp][Wp][q_out->bits][ceil(O/32)]
 *   (Hp, Wp = pooled size).  When NULL the block is a last layer: no
 *   HardTanh, no quantization.
 * y_out (nullable): fp32 NCHW output after BN (and HardTanh when q_out).
 * At least one of planes_out / y_out must be given. */
MINW_API minw_status minw_conv_block(const uint32_t *act, int32_t B, int32_t C,
                            int32_t H, int32_t W, int32_t bits_a,
                            const uint32_t *wgt, int32_t O, int32_t kh,
                            int32_t kw, int32_t bits_w, int32_t stride,
                            int32_t pad, int32_t pool, const float *scale,
                            const float *shift, const minw_quant *q_out,
                            uint32_t *planes_out, float *y_out,
                            int32_t variant, void *stream);

/* ---------------------------------------------------------------------- */
/* Level-code layout and the tensor-core convolution                       */
/* ---------------------------------------------------------------------- */

/* "Codes" layout: one byte per value, the level in integer units (3-bit:
 * quarters) written as an FP8 E4M3 number -- 0 -> 0x00, +-1 -> 0x38/0xB8,
 * +-2 -> 0x40/0xC0, +-4 -> 0x48/0xC8.  Activations [N][H][W][C] (channels
 * innermost), weights [O][kh][kw][C].  Products of two codes are exact, so a
 * tensor-core FP8 contraction with fp32 accumulation returns the same integer
 * accumulator as the popcount path.  C must be a multiple of 16 (128 for the
 * convolution). */

/* Quantize (Eq. inference) NCHW fp32 activations into NHWC codes. */
MINW_API minw_status aqe_quantize_codes(const float *x, int32_t B, int32_t C, int32_t H,
                                        int32_t W, const minw_quant *q, uint8_t *codes,
                                        void *stream);

/* Quantize latent weights [O][C][kh][kw] into codes [O][kh][kw][C];
 * channel_scale as in minw_pack_weights. */
MINW_API minw_status minw_pack_weight_codes(const float *w, int32_t O, int32_t C, int32_t kh,
                                            int32_t kw, const minw_quant *q,
                                            const float *channel_scale, uint8_t *codes,
                                            void *stream);

/* "E2M1 codes" layout: the same levels as 4-bit FP4 E2M1 numbers, two
 * channels per byte (channel 2j in the low nibble of byte j) -- 0 -> 0x0,
 * +-1 -> 0x2/0xA, +-2 -> 0x4/0xC, +-4 -> 0x6/0xE.  Activations
 * [N][H][W][C / 2] bytes, weights [O][kh][kw][C / 2].  The products are as
 * exact as E4M3's; the tensor cores take them with unit block scales
 * (tcgen05 kind::mxf4), at twice the K per instruction and half the bytes. */
enum { MINW_CODES_E4M3 = 0, MINW_CODES_E2M1 = 1 };

/* aqe_quantize_codes into E2M1 codes (C % 32 == 0). */
MINW_API minw_status aqe_quantize_codes_e2m1(const float *x, int32_t B, int32_t C, int32_t H,
                                             int32_t W, const minw_quant *q, uint8_t *codes,
                                             void *stream);

/* minw_pack_weight_codes into E2M1 codes [O][kh][kw][C / 2] (C % 16 == 0). */
MINW_API minw_status minw_pack_weight_codes_e2m1(const float *w, int32_t O, int32_t C, int32_t kh,
                                                 int32_t kw, const minw_quant *q,
                                                 const float *channel_scale, uint8_t *codes,
                                                 void *stream);

/* minw_conv2d on codes operands, run on the tcgen05 tensor cores.
 * Supported: stride 1 or 2, C % 64 == 0, pad < kh, kw; otherwise
 * MINW_EUNSUPPORTED.  bits_a / bits_w document the operands (1..3). */
MINW_API minw_status minw_conv2d_codes(const uint8_t *act, int32_t B, int32_t C, int32_t H,
                                       int32_t W, int32_t bits_a, const uint8_t *wgt,
                                       int32_t O, int32_t kh, int32_t kw, int32_t bits_w,
                                       int32_t stride, int32_t pad, int32_t *acc_out,
                                       const float *scale, const float *shift, float *y_out,
                                       void *stream);

/* minw_conv_block on codes operands (tensor cores).  With q_out the quantized
 * output goes to codes_out [B][Hp][Wp][O] (O % 16 == 0) and/or planes_out. */
MINW_API minw_status minw_conv_block_codes(const uint8_t *act, int32_t B, int32_t C,
                                           int32_t H, int32_t W, int32_t bits_a,
                                           const uint8_t *wgt, int32_t O, int32_t kh,
                                           int32_t kw, int32_t bits_w, int32_t stride,
                                           int32_t pad, int32_t pool, const float *scale,
                                           const float *shift, const minw_quant *q_out,
                                           uint8_t *codes_out, uint32_t *planes_out,
                                           float *y_out, void *stream);

/* ---------------------------------------------------------------------- */
/* Weight-only quantized convolution (Sec. IV, the XNOR / SHIFT ADDER       */
/* layers of Tables II-IV: full-precision activations, 1-3-bit weights)    */
/* ---------------------------------------------------------------------- */

/* fp32 NCHW [B][C][H][W] -> bf16 NHWC [B][H][W][C], round to nearest even. */
MINW_API minw_status minw_to_bf16_nhwc(const float *x, int32_t B, int32_t C, int32_t H, int32_t W,
                                       uint16_t *out, void *stream);

/* Quantize latent weights [O][C][kh][kw] (Eq. sign / tnn / qnn at x *
 * channel_scale[o], or q->scale when channel_scale is null) into bf16 level
 * values in integer units [O][kh][kw][C]: +-1 (1-bit), {-1, 0, 1} (2-bit),
 * {0, +-1, +-2, +-4} (3-bit, quarters), all exact in bf16.  out 16-byte
 * aligned, C % 8 == 0 (else MINW_EUNSUPPORTED). */
MINW_API minw_status minw_pack_weight_bf16(const float *w, int32_t O, int32_t C, int32_t kh, int32_t kw,
                                           const minw_quant *q, const float *channel_scale, uint16_t *out,
                                           void *stream);

/* Narrow layers (channel counts that are not a multiple of 64, as in the
 * 16- and 32-channel stages of ResNet-110 or the 12-channel growth of
 * DenseNet-100, Table III): the same conversions with the channels padded to
 * Cp >= C (the row length of the output), channels C .. Cp written as 0.  A
 * zero activation or weight adds exactly 0 to every product, so
 * minw_conv2d_bf16 run with C = Cp (a multiple of 64) on both padded
 * operands gives the product of the unpadded ones.  Cp % 8 == 0 for the
 * weights (MINW_EUNSUPPORTED otherwise); MINW_EINVAL for Cp < C. */
MINW_API minw_status minw_to_bf16_nhwc_pad(const float *x, int32_t B, int32_t C, int32_t H, int32_t W, int32_t Cp,
                                           uint16_t *out, void *stream);
MINW_API minw_status minw_pack_weight_bf16_pad(const float *w, int32_t O, int32_t C, int32_t kh, int32_t kw,
                                               int32_t Cp, const minw_quant *q, const float *channel_scale,
                                               uint16_t *out, void *stream);

/* Weight-only quantized convolution on the tcgen05 tensor cores (kind::f16,
 * bf16 x bf16 -> fp32 in TMEM): acc[b][o][y][x] = sum over (ky, kx, c) of
 * act * wgt with the accumulation order of the tensor core (not the oracle's),
 * then [2x2 / 2 max pool] and y_out = fmaf(acc, scale[o], shift[o]) fp32 NCHW
 * (no HardTanh, no quantizer: the next layer's activations stay full
 * precision).  act: bf16 NHWC [B][H][W][C]; wgt: bf16 [O][kh][kw][C] from
 * minw_pack_weight_bf16 (bits_w documents it).  Supported: stride 1 or 2,
 * C % 64 == 0, pad < kh, kw, even output size when pooling.  Errors:
 * MINW_EINVAL (arguments), MINW_EUNSUPPORTED (shape). */
MINW_API minw_status minw_conv2d_bf16(const uint16_t *act, int32_t B, int32_t C, int32_t H, int32_t W,
                                      const uint16_t *wgt, int32_t O, int32_t kh, int32_t kw, int32_t bits_w,
                                      int32_t stride, int32_t pad, int32_t pool, const float *scale,
                                      const float *shift, float *y_out, void *stream);

/* The same convolution (no pool) with the next layer's input as its output:
 * v = fmaf(acc, scale[o], shift[o]) [+ residual[b][o][y][x], one fp32 add:
 * a residual block's shortcut, fp32 NCHW, nullable], clamped to [-1, 1]
 * (HardTanh); out[pixel][out_off + o] = bf16(v) (round to nearest even),
 * bf16 NHWC rows of out_ld elements per output pixel, and y_out (nullable)
 * v as fp32 NCHW [B][O][Ho][Wo]; the other elements of each out row are not
 * written (a DenseNet block appends its new channels to its feature buffer
 * this way).  act: bf16 NHWC rows of ldc elements per pixel (0: C), of which
 * the first C are read (ldc a multiple of 64, at least C).  The accumulators
 * are those minw_conv2d_bf16 forms for the same operands, so out equals the
 * bf16 rounding of HardTanh of its y_out.  Errors: MINW_EINVAL (arguments,
 * out_ld < out_off + O), MINW_EUNSUPPORTED (shape, as minw_conv2d_bf16). */
MINW_API minw_status minw_conv2d_bf16_hardtanh(const uint16_t *act, int32_t B, int32_t C, int32_t H, int32_t W,
                                               int32_t ldc, const uint16_t *wgt, int32_t O, int32_t kh, int32_t kw,
                                               int32_t bits_w, int32_t stride, int32_t pad, const float *scale,
                                               const float *shift, uint16_t *out, int32_t out_ld, int32_t out_off,
                                               const float *residual, float *y_out, void *stream);

/* ---------------------------------------------------------------------- */
/* Training step of a fully connected layer (Algorithm 1)                  */
/* ---------------------------------------------------------------------- */

/* The bf16 operands of Algorithm 1's training products (bf16 roundings of
 * the fp32 operands, fp32 sums: a precision departure from the paper's fp32
 * training, with the error bound stated at minw_fc_train_step's products).
 * out (bf16, round to nearest even, row-major (transpose ? cols : rows) x
 * out_cols) = in (fp32 row-major rows x cols),
 * transposed when transpose != 0, zero in the columns past the source's.
 * Caller-owned device buffers; asynchronous on stream.  MINW_EINVAL for null
 * pointers, non-positive sizes or out_cols below the source's columns;
 * MINW_EUNSUPPORTED past 65535 x 32 output rows. */
MINW_API minw_status minw_bf16_matrix(const float *in, int32_t rows, int32_t cols, int32_t transpose,
                                      int32_t out_cols, uint16_t *out, void *stream);

/* The update of Algorithm 1 with a plain gradient step (update(W, g, eta)
 * then the clip to [-1, 1]): w = min(1, max(-1, fmaf(-lr, g, w))), n fp32
 * values of device memory in place (g is the already masked gradient).
 * Asynchronous on stream; n == 0 does nothing; MINW_EINVAL for n < 0 or null
 * pointers. */
MINW_API minw_status minw_sgd_clip(float *w, const float *g, int64_t n, float lr, void *stream);

/* Bytes of device workspace minw_fc_train_step needs (0 for bad sizes). */
MINW_API size_t minw_fc_train_workspace_bytes(int32_t B, int32_t K, int32_t O);

/* One step of Algorithm 1 for a fully connected layer with input A [B][K]
 * (fp32, the previous layer's AQE output or the network input), latent
 * weights W [O][K] (fp32, updated in place) and the upstream gradient g_out
 * [B][O] = dL/d(a_out):
 *   W^ = fmaf(alpha, h_w(W), (1 - alpha) W)        (Eq. weight, q_w)
 *   a~ = bf16(A) bf16(W^)^T                         (tensor cores, fp32 sums)
 *   a_out = fmaf(alpha, h_a(a~), (1 - alpha) a~)    (Eq. activation, q_a; a_out = a~ when q_a is null: last layer)
 *   g_a~ = 2 alpha g_out 1[|a~| <= 1]               (Eq. activation; g_out itself when q_a is null)
 *   g_in = bf16(g_a~) bf16(W^)                      ([B][K], skipped when g_in is null)
 *   g_W^ = bf16(g_a~)^T bf16(A)                     ([O][K])
 *   W = min(1, max(-1, W - lr 2 alpha g_W^ 1[|W| <= 1]))   (Eq. weight, update and clip)
 * a_pre (nullable, [B][O]) receives a~ when q_a is set (ignored without q_a,
 * where a_out is a~ itself).
 * Each product P Q of K terms takes bf16 roundings of its fp32 operands (the
 * paper trains on fp32 ones: a precision departure) and differs from the
 * exact product of the fp32 operands by at most
 * (2^-7 + 2^-16 + K 2^-23 (1 + 2^-8)^2) (|P| |Q|): the two operand roundings
 * and the fp32 accumulation in any order.
 * A product with few output tiles and a long reduction adds its fp32 sums in K
 * slices, slice by slice in a fixed order (deterministic, same bound).
 * Requirements: K % 64 == 0 and B % 64 == 0 (else MINW_EUNSUPPORTED), alpha in
 * [0, 1], 16-byte aligned pointers, workspace of minw_fc_train_workspace_bytes
 * (scratch: nothing in it survives the call).  All buffers are caller-owned
 * device memory; the call is asynchronous on stream and launches five to eight kernels.
 * MINW_EINVAL: null A, W, g_out, a_out, q_w or workspace, an invalid quantizer,
 * alpha outside [0, 1], a misaligned pointer or a short workspace;
 * MINW_EUNSUPPORTED: the shapes above, or sizes past the kernels' 32-bit
 * index and grid limits. */
MINW_API minw_status minw_fc_train_step(const float *A, float *W, const float *g_out, int32_t B, int32_t K,
                                        int32_t O, float alpha, float lr, const minw_quant *q_w,
                                        const minw_quant *q_a, float *a_out, float *g_in, float *a_pre,
                                        void *workspace, size_t workspace_bytes, void *stream);

/* Bytes of device workspace minw_conv_train_step needs for this shape (0
 * for bad or unsupported sizes). */
MINW_API size_t minw_conv_train_workspace_bytes(int32_t B, int32_t C, int32_t H, int32_t W, int32_t O, int32_t kh,
                                                int32_t kw, int32_t stride, int32_t pad);

/* One step of Algorithm 1 for a convolutional layer (the training branch
 * treats convolutional and fully connected layers alike) with input A
 * [B][C][H][W] (fp32 NCHW, the previous layer's AQE output or the network
 * input), latent weights W [O][C][kh][kw] (fp32, updated in place) and the
 * upstream gradient g_out [B][O][Ho][Wo] = dL/d(a_out), zero padding pad and
 * stride stride:
 *   W^ = fmaf(alpha, h_w(W), (1 - alpha) W)             (Eq. weight, q_w)
 *   a~ = conv(bf16(A), bf16(W^))                         (tensor cores, fp32 sums)
 *   a_out = fmaf(alpha, h_a(a~), (1 - alpha) a~)         (Eq. activation, q_a; a_out = a~ when q_a is null)
 *   g_a~ = 2 alpha g_out 1[|a~| <= 1]                    (Eq. activation; g_out itself when q_a is null)
 *   g_in = conv^T(bf16(g_a~), bf16(W^))                  ([B][C][H][W], skipped when g_in is null)
 *   g_W^ = sum over b, y, x of bf16(g_a~) x bf16(A patch) ([O][C][kh][kw])
 *   W = min(1, max(-1, W - lr 2 alpha g_W^ 1[|W| <= 1]))  (Eq. weight, update and clip)
 * a_pre (nullable, [B][O][Ho][Wo]) receives a~ when q_a is set (ignored
 * without q_a).  The three products take bf16 roundings of their fp32
 * operands (the paper's operands are fp32: this is a precision departure
 * with the per-product error bound of minw_fc_train_step), and the weight
 * gradient's reduction over the pixels is split across the SMs and summed
 * slice by slice in a fixed order (the same bits on every call).
 * Requirements: C % 64 == 0, B Ho Wo % 64 == 0, stride 1 or 2, pad < kh and
 * pad < kw (else MINW_EUNSUPPORTED); alpha in [0, 1]; 16-byte aligned
 * pointers; workspace of minw_conv_train_workspace_bytes (scratch: nothing
 * in it survives the call).  All buffers are caller-owned device memory; the
 * call is asynchronous on stream and launches eight to eleven kernels (and a
 * memset of the input gradient's spread image for stride 2 or O % 64 != 0).
 * MINW_EINVAL: null A, W, g_out, a_out, q_w or workspace, an invalid
 * quantizer, alpha outside [0, 1], a misaligned pointer or a short workspace;
 * MINW_EUNSUPPORTED: the shapes above, or sizes past the kernels' index and
 * grid limits. */
MINW_API minw_status minw_conv_train_step(const float *A, float *W, const float *g_out, int32_t B, int32_t C,
                                          int32_t H, int32_t Wd, int32_t O, int32_t kh, int32_t kw, int32_t stride,
                                          int32_t pad, float alpha, float lr, const minw_quant *q_w,
                                          const minw_quant *q_a, float *a_out, float *g_in, float *a_pre,
                                          void *workspace, size_t workspace_bytes, void *stream);

/* Extra inputs and outputs of a residual block (ResNet-style MINW-Net,
 * where the paper leaves the block wiring open).  Host struct.
 * res_codes (nullable): shortcut as level codes [B][Hp][Wp][O] of bit width
 *   res_bits (its levels are added as values: 3-bit codes count quarters).
 * res_f32 (nullable): shortcut as fp32 NHWC [B][Hp][Wp][O].
 * y_nhwc (nullable, output): the BN output before the shortcut, fp32 NHWC.
 * With a shortcut the block computes y = fmaf(acc, scale, shift) + shortcut
 * (one fp32 add), then HardTanh and the output quantizer.
 * in_format (MINW_CODES_E4M3 or MINW_CODES_E2M1): layout of act and wgt; E2M1
 *   operands need C % 128 == 0 (else MINW_EUNSUPPORTED).
 * out_format, res_format: layouts of codes_out and res_codes.
 * acc_out (nullable, output): the exact int32 accumulators, NCHW, for a block
 *   without pooling.
 * e2m1_pairs: with E2M1 operands, run CTA pairs of 256 pixels x 128 channels
 *   (two accumulators per CTA, so each tile's epilogue overlaps the next
 *   tile's MMAs) where the shape allows it (O % 128 == 0); elsewhere, and for
 *   E4M3 operands, the default tiling.  The results are the same integers
 *   either way; only the speed differs, which is why callers measure both.
 * A zero-initialised struct is the E4M3 block without extras. */
typedef struct {
    const uint8_t *res_codes;
    int32_t res_bits;
    const float *res_f32;
    float *y_nhwc;
    int32_t in_format;
    int32_t out_format;
    int32_t res_format;
    int32_t *acc_out;
    int32_t e2m1_pairs;
} minw_block_extra;

/* minw_conv_block_codes with the residual inputs / outputs of extra
 * (nullable).  At most one shortcut. */
MINW_API minw_status minw_conv_block_codes_ex(const uint8_t *act, int32_t B, int32_t C,
                                              int32_t H, int32_t W, int32_t bits_a,
                                              const uint8_t *wgt, int32_t O, int32_t kh,
                                              int32_t kw, int32_t bits_w, int32_t stride,
                                              int32_t pad, int32_t pool, const float *scale,
                                              const float *shift, const minw_quant *q_out,
                                              uint8_t *codes_out, uint32_t *planes_out,
                                              float *y_out, const minw_block_extra *extra,
                                              void *stream);

/* Fully connected layer a~ = a^q W^q (Algorithm 1, inference) on the tensor
 * cores, with the reduction over K split across CTAs when the output alone
 * would leave most SMs idle (split-K).  act: codes [B][K]; wgt: codes [O][K];
 * K % 128 == 0.  Outputs as minw_conv_block_codes with H = W = 1: codes_out
 * [B][O] (O % 16 == 0), planes_out [B][bits][ceil(O/32)], y_out fp32 [B][O];
 * acc_out (nullable) int32 [B][O] exact accumulators.  q_out NULL = last layer.
 * workspace: device scratch of minw_fc_workspace_bytes(B, K, O) bytes for
 * the full split (a smaller one splits K into fewer slices; 0 bytes or NULL
 * runs without the split).  Its contents need no initialisation and are
 * meaningless after the call.  Calls that share a workspace must not run
 * concurrently.  With a split the call launches a second kernel that sums
 * the K slices and runs the epilogue. */
MINW_API size_t minw_fc_workspace_bytes(int32_t B, int32_t K, int32_t O);
/* K slices minw_fc_codes uses for this shape with a workspace of
 * workspace_bytes (1: no split; 0: shape not supported).  Host-only query. */
MINW_API int32_t minw_fc_ksplit(int32_t B, int32_t K, int32_t O, size_t workspace_bytes);
MINW_API minw_status minw_fc_codes(const uint8_t *act, int32_t B, int32_t K, int32_t bits_a,
                                   const uint8_t *wgt, int32_t O, int32_t bits_w,
                                   const float *scale, const float *shift,
                                   const minw_quant *q_out, uint8_t *codes_out,
                                   uint32_t *planes_out, float *y_out, int32_t *acc_out,
                                   void *workspace, size_t workspace_bytes, void *stream);

/* minw_fc_codes for callers that cannot allocate device memory (no
 * counterpart in the paper; an interface addition).  Such callers include a
 * plugin run by a host framework that owns all device memory and passes in
 * only the tensors of the call, and a service that reserves its memory at
 * start-up and forbids allocations afterwards.  The split-K scratch lives
 * in a fixed array of MINW_FC_NOALLOC_SCRATCH_BYTES inside the library, held
 * on every GPU that loads the library until the process exits.  The call
 * allocates nothing (no cudaMalloc/cudaFree, no allocating library routine).
 * - The first call on each device looks up the array's device address
 *   (cudaGetSymbolAddress, with that device current); make that first call
 *   before any stream capture.  The address is kept for the life of the
 *   process: after cudaDeviceReset (or anything else that ends the device's
 *   primary context) it is stale, so a process that resets a device must not
 *   call this entry point again on that device.
 * - Every call shares the one array.  Nothing in it needs to start at zero
 *   (each call overwrites what it reads) and it keeps the last call's
 *   contents; calls that overlap on the GPU (other streams, other threads)
 *   race on it and must be serialised by the caller.
 * - K is split into as many slices as the array holds; a shape whose
 *   smallest split (two slices of int32 partial sums plus the breakpoints)
 *   needs more than the array returns MINW_EUNSUPPORTED before any launch.
 * Arguments and outputs as minw_fc_codes. */
#define MINW_FC_NOALLOC_SCRATCH_BYTES (8u << 20)
MINW_API minw_status minw_fc_codes_noalloc(const uint8_t *act, int32_t B, int32_t K,
                                           int32_t bits_a, const uint8_t *wgt, int32_t O,
                                           int32_t bits_w, const float *scale,
                                           const float *shift, const minw_quant *q_out,
                                           uint8_t *codes_out, uint32_t *planes_out,
                                           float *y_out, int32_t *acc_out, void *stream);

/* First layer (Sec. III-E): the fp32 image x [B][C][H][W] is NOT quantized;
 * the weights are.  w: latent fp32 weights [O][C][kh][kw]; q_w (host) and
 * channel_scale (nullable) quantize them as minw_pack_weights does; q_w NULL
 * keeps the fp32 weights as they are.  Each output is one fp32 fmaf chain over
 * (c, ky, kx) in that order, padded taps skipped.  Then [pool 2x2/2 on fp32],
 * BN (fmaf), and, with q_out, HardTanh + quantize + pack as minw_conv_block. */
MINW_API minw_status minw_conv_first(const float *x, int32_t B, int32_t C, int32_t H,
                            int32_t W, const float *w, int32_t O, int32_t kh,
                            int32_t kw, int32_t stride, int32_t pad,
                            const minw_quant *q_w, const float *channel_scale,
                            int32_t pool, const float *scale,
                            const float *shift, const minw_quant *q_out,
                            uint32_t *planes_out, float *y_out, void *stream);

/* ---------------------------------------------------------------------- */
/* Whole-network forward (Algorithm 1, inference branch)                   */
/* ---------------------------------------------------------------------- */

enum { MINW_LAYER_CONV = 0, MINW_LAYER_FC = 1 };

/* One layer of a sequential MINW-Net.  Pointers are device pointers read
 * during minw_net_create only (the net keeps its own packed copy).
 * - CONV: input [C][H][W], kernel kh x kw, stride, pad, optional pool.
 * - FC: input is the previous output flattened in (c, h, w) order; C, H, W
 *   describe that input (K = C*H*W); w is [O][K].
 * bits_in 0 marks the first layer (fp32 input, minw_conv_first);
 * bits_out 0 marks the last layer (fp32 logits, no HardTanh). */
typedef struct {
    int32_t kind;
    int32_t C, H, W, O;
    int32_t kh, kw, stride, pad, pool;
    int32_t bits_in, bits_w, bits_out;
    float thr_w[3];           /* weight quantizer thresholds */
    float thr_out[3];         /* output quantizer thresholds */
    const float *w;           /* latent weights */
    const float *w_scale;     /* per-output-channel prescale, nullable */
    const float *scale;       /* BN scale (length O) */
    const float *shift;       /* BN shift (length O) */
    int32_t variant;          /* this layer's kernel request, in the values
                                 minw_net_layer_variants reports; 0 follows the network's
                                 request.  A non-zero request skips the layer's creation-time
                                 measurement and runs: MINW_VARIANT_POPC the popcount path,
                                 MINW_VARIANT_TC or _TC_E4M3 E4M3 operands, _TC_E2M1 E2M1
                                 operands, _TC_E2M1_PAIRS E2M1 CTA pairs, each where the shape
                                 allows it (a replay of a measured plan, e.g. under a profiler
                                 whose overhead would distort the measurement) */
} minw_layer_desc;

typedef struct minw_net minw_net;

/* Build a network: validates the layer chain, packs every weight tensor,
 * plans a kernel per layer (variant: MINW_VARIANT_*) and allocates activation
 * buffers for up to max_batch images.  layers: host array.  Synchronous. */
MINW_API minw_status minw_net_create(const minw_layer_desc *layers, int32_t n_layers,
                            int32_t max_batch, int32_t variant, void *stream,
                            minw_net **out);

/* Forward pass of B <= max_batch images x [B][C][H][W] (fp32) to logits
 * [B][O_last] (fp32).  All work is enqueued on `stream`. */
MINW_API minw_status minw_forward(minw_net *net, const float *x, int32_t B,
                         float *logits, void *stream);

/* Forward pass from HOST buffers: copies x_host [B][C][H][W] (fp32; pinned
 * memory gives asynchronous copies) into a device staging buffer the net owns,
 * runs minw_forward and copies the logits back into logits_host [B][O_last];
 * returns after the stream has finished (the logits are ready). */
MINW_API minw_status minw_forward_host(minw_net *net, const float *x_host, int32_t B,
                              float *logits_host, void *stream);

/* Per-layer timing: with on != 0 every later minw_forward records a CUDA
 * event after each layer's kernel; minw_net_layer_times then writes the
 * elapsed milliseconds of each layer of the most recent forward into ms
 * (host array of minw_net_launches() floats), synchronising on the events. */
MINW_API minw_status minw_net_enable_timing(minw_net *net, int32_t on);
MINW_API minw_status minw_net_layer_times(minw_net *net, float *ms);

/* Kernel chosen for each layer (host array of minw_net_launches() ints):
 * 0 for the fp32 first layer, else MINW_VARIANT_POPC, MINW_VARIANT_TC (E4M3
 * operands), MINW_VARIANT_TC_E2M1, MINW_VARIANT_TC_E2M1_PAIRS or
 * MINW_VARIANT_TC_E2M1_N128. */
MINW_API minw_status minw_net_layer_variants(const minw_net *net, int32_t *variants);

/* The creation-time measurement behind layer `layer`'s kernel choice under
 * MINW_VARIANT_AUTO (runtime introspection; the paper has no counterpart):
 * ms (host array of 4 floats) receives the least of three timed launches of
 * each candidate at the net's max_batch, in milliseconds, in the order E4M3
 * operands, E2M1 operands, E2M1 CTA pairs of 128-channel tiles, popcount on
 * bit-planes, E2M1 single-CTA 128-channel tiles (ms: host array of 5
 * floats); -1 for a candidate the layer's shape does not allow, and -1 in
 * every entry for the first layer and for nets not created with
 * MINW_VARIANT_AUTO.  The kernel minw_net_layer_variants reports is the
 * fastest entry.  MINW_EINVAL for a null argument or a layer out of range,
 * MINW_EUNSUPPORTED for a residual network (its formats follow a fixed
 * rule). */
MINW_API minw_status minw_net_layer_candidates(const minw_net *net, int32_t layer, float *ms);

/* ResNet-18-shaped MINW-Net (Table V's network).  The paper leaves the
 * residual wiring open; the reading implemented here:
 *   stem: fp32 7x7/2 conv (fp32 weights, pad 3) -> 3x3/2 max pool (pad 1) ->
 *         BN -> HardTanh -> quantize (the block order of Sec. III-E);
 *   block (widths 64-128-256-512, two per stage, stride 2 entering stages
 *         2-4): u = quantized input; v = h(HardTanh(BN1(conv1(u))));
 *         y = BN2(conv2(v)) + s with s = u, or s = BN_d(conv_d(u)) for the
 *         1x1 / 2 shortcut of the first block of stages 2-4 (fp32 sum);
 *         output h(HardTanh(y));
 *   head: global average pool of the last levels -> fp32 fully connected
 *         layer [classes][512] -> BN -> fp32 logits.
 * Every convolution weight of the blocks is quantized with (bits_w, thr_w)
 * and its per-output-channel prescale (nullable); activations with
 * (bits_a, thr_a).  conv_w[2b], conv_w[2b+1]: block b's two convolutions
 * [O][C][3][3]; down_*[i]: the shortcut of stage i+2 [O][C][1][1].
 * image_hw: multiple of 32 (224 for ImageNet crops).  Device pointers, read
 * during creation only.  minw_forward then takes x [B][3][hw][hw] and writes
 * logits [B][num_classes]. */
typedef struct {
    int32_t bits_a, bits_w;
    float thr_a[3], thr_w[3];
    int32_t image_hw, num_classes;
    const float *stem_w, *stem_scale, *stem_shift;
    const float *conv_w[16], *conv_wscale[16], *conv_scale[16], *conv_shift[16];
    const float *down_w[3], *down_wscale[3], *down_scale[3], *down_shift[3];
    const float *fc_w, *fc_scale, *fc_shift;
} minw_resnet18_desc;

MINW_API minw_status minw_resnet18_create(const minw_resnet18_desc *desc, int32_t max_batch,
                                          void *stream, minw_net **out);

/* The weight-only MINW-Net residual network of Table III (3-bit weights,
 * full-precision activations; ResNet-110 for n = 18): a CIFAR ResNet-(6n+2)
 * whose block convolutions multiply bf16 activations by N-bit weight levels
 * on the tensor cores (the SHIFT ADDER layers of Sec. IV, as
 * minw_conv2d_bf16), with fp32 first and last layers (Sec. III-E).  The
 * paper leaves the block wiring open; the reading implemented here:
 *   stem: fp32 3x3 conv 3 -> 16 (fp32 weights, pad 1; one fmaf chain per
 *         output over (c, ky, kx)) -> BN -> HardTanh;
 *   block (3 stages of n blocks, 16, 32 and 64 channels, stride 2 entering
 *         stages 2 and 3): h = HardTanh(BN1(conv1(x))),
 *         out = HardTanh(BN2(conv2(h)) + s) with s = x, or s = BN_d(conv_d(x))
 *         for the 1x1 / 2 shortcut entering stages 2 and 3 (one fp32 add);
 *         each convolution reads the bf16 rounding of its fp32 input;
 *   head: global average pool (one fp32 sum in pixel order, one division) ->
 *         fp32 fully connected layer [classes][64] -> BN -> fp32 logits.
 * Block b (0 .. 3n - 1, stage b / n) has c1_*[b] [O][C][3][3] and
 * c2_*[b] [O][O][3][3]; down_*[i] is the shortcut entering stage i + 2
 * [O][C][1][1]; *_wscale: per-output-channel weight prescale (nullable);
 * every block weight is quantized with (bits_w, thr_w) to levels in integer
 * units.  The 16- and 32-channel layers run on operands padded to 64
 * channels.  image_hw: a multiple of 4 (32 for CIFAR).  Device pointers, read
 * during creation only.  minw_forward takes x [B][3][hw][hw] and writes
 * logits [B][num_classes].  Errors: MINW_EINVAL (arguments, n outside
 * 1 .. MINW_WRESNET_MAX_N), MINW_EUNSUPPORTED (sizes past the 32-bit index
 * range), MINW_ECUDA. */
#define MINW_WRESNET_MAX_N 18
typedef struct {
    int32_t n;
    int32_t bits_w;
    float thr_w[3];
    int32_t image_hw, num_classes;
    const float *stem_w, *stem_scale, *stem_shift;
    const float *c1_w[3 * MINW_WRESNET_MAX_N], *c1_wscale[3 * MINW_WRESNET_MAX_N];
    const float *c1_scale[3 * MINW_WRESNET_MAX_N], *c1_shift[3 * MINW_WRESNET_MAX_N];
    const float *c2_w[3 * MINW_WRESNET_MAX_N], *c2_wscale[3 * MINW_WRESNET_MAX_N];
    const float *c2_scale[3 * MINW_WRESNET_MAX_N], *c2_shift[3 * MINW_WRESNET_MAX_N];
    const float *down_w[2], *down_wscale[2], *down_scale[2], *down_shift[2];
    const float *fc_w, *fc_scale, *fc_shift;
    int32_t keep_activations;   /* nonzero: keep every block's fp32 output for minw_wresnet_activation */
} minw_wresnet_desc;

MINW_API minw_status minw_wresnet_create(const minw_wresnet_desc *desc, int32_t max_batch, void *stream,
                                         minw_net **out);

/* Introspection of a net created with keep_activations (no counterpart in
 * the paper): copies the fp32 NCHW output of stage-step `index` of the most
 * recent forward -- 0 the stem's HardTanh output [B][16][hw][hw], b + 1 block
 * b's output -- into dst (device memory of at least count floats), on stream.
 * MINW_EINVAL for a net without kept activations, an index out of range or a
 * short dst. */
MINW_API minw_status minw_wresnet_activation(const minw_net *net, int32_t index, float *dst, size_t count,
                                             void *stream);

/* The weight-only MINW-Net DenseNet-BC of Table III (DenseNet-100 for
 * layers = 16, growth k = 12, 3-bit weights): N-bit weights times
 * full-precision (bf16) activations on the tensor cores for every layer
 * inside the network, fp32 first and last layers (Sec. III-E).  The paper
 * gives no wiring beyond DenseNet's; the reading implemented here keeps the
 * block order conv -> BN -> HardTanh of Sec. III-E:
 *   stem : fp32 3x3 conv 3 -> 2k (fp32 weights, pad 1, one fmaf chain per
 *          output over (c, ky, kx)) -> BN -> HardTanh; the block's features
 *          F start as its bf16 rounding;
 *   layer: h = HardTanh(BN(conv 1x1 (F) to 4k channels)),
 *          n = HardTanh(BN(conv 3x3 pad 1 (bf16(h)) to k channels)),
 *          F <- concat(F, bf16(n)) along channels;
 *   trans: between blocks, F <- bf16(avgpool 2x2(HardTanh(BN(conv 1x1 (F)
 *          to floor(c / 2) channels)))), the pool ((v00 + v01) + v10) + v11
 *          in fp32, times 1/4;
 *   head : global average pool of the last F (one fp32 sum in pixel order,
 *          one division) -> fp32 fully connected layer -> BN -> logits.
 * Three blocks of `layers` layers; block b starts with c_b channels (c_0 =
 * 2k) and its layer i reads c_b + i k.  Layer j = b * layers + i has b_*[j]
 * [4k][c_b + i k][1][1] and c_*[j] [k][4k][3][3]; t_*[b] [c / 2][c][1][1] is
 * the transition after block b (c its final channels); fc_w [classes][c]
 * for the last block's c.  *_wscale: per-output-channel weight prescale
 * (nullable); every convolution after the stem is quantized with (bits_w,
 * thr_w) to levels in integer units.  Each block's features live in one bf16
 * NHWC buffer of pad64(final c) channels per pixel that the layers append
 * to in place (no concatenation copies); each 1x1 convolution reads the
 * first pad64(c) channels of its rows (zero weights past c).  image_hw: a
 * multiple of 4, at least 8.  Device pointers, read during creation only.
 * minw_forward takes x [B][3][hw][hw] and writes logits [B][num_classes].
 * Errors: MINW_EINVAL (arguments; layers outside 1 .. MINW_WDENSE_MAX_LAYERS,
 * growth outside 1 .. 64), MINW_EUNSUPPORTED (sizes past the 32-bit index
 * range, more than 1536 final channels), MINW_ECUDA. */
#define MINW_WDENSE_MAX_LAYERS 32
typedef struct {
    int32_t layers, growth;
    int32_t bits_w;
    float thr_w[3];
    int32_t image_hw, num_classes;
    const float *stem_w, *stem_scale, *stem_shift;
    const float *b_w[3 * MINW_WDENSE_MAX_LAYERS], *b_wscale[3 * MINW_WDENSE_MAX_LAYERS];
    const float *b_scale[3 * MINW_WDENSE_MAX_LAYERS], *b_shift[3 * MINW_WDENSE_MAX_LAYERS];
    const float *c_w[3 * MINW_WDENSE_MAX_LAYERS], *c_wscale[3 * MINW_WDENSE_MAX_LAYERS];
    const float *c_scale[3 * MINW_WDENSE_MAX_LAYERS], *c_shift[3 * MINW_WDENSE_MAX_LAYERS];
    const float *t_w[2], *t_wscale[2], *t_scale[2], *t_shift[2];
    const float *fc_w, *fc_scale, *fc_shift;
} minw_wdense_desc;

MINW_API minw_status minw_wdense_create(const minw_wdense_desc *desc, int32_t max_batch, void *stream,
                                        minw_net **out);

/* Introspection (no counterpart in the paper): copies block `block`'s
 * features after the most recent forward -- bf16 bit patterns, NHWC
 * [B][h][h][*row] with *row = pad64(the block's final channels) elements per
 * pixel, channels past the final count unspecified; h = image_hw >> block --
 * into dst (device memory of at least count uint16), on stream, and stores
 * the block's final channel count in *channels and the row length in *row
 * (host pointers, nullable).  Block b's first c_b channels are the stem's
 * or the previous transition's output, and channels c_b + i k .. + k the
 * output of its layer i.  MINW_EINVAL for a net of another kind, a block
 * outside 0 .. 2, no forward yet, or a short dst. */
MINW_API minw_status minw_wdense_features(const minw_net *net, int32_t block, uint16_t *dst, size_t count,
                                          int32_t *channels, int32_t *row, void *stream);

/* Number of layers (and of entries minw_net_layer_times fills). */
MINW_API int32_t minw_net_launches(const minw_net *net);

/* Number of kernels one minw_forward launches (a layer whose K reduction is
 * split across CTAs launches two). */
MINW_API int32_t minw_net_kernels(const minw_net *net);

/* Release a network (synchronises its device memory frees). */
MINW_API void minw_net_destroy(minw_net *net);

/* ---------------------------------------------------------------------- */
/* Errors                                                                  */
/* ---------------------------------------------------------------------- */

/* Reads and clears the device error flag after synchronising `stream`:
 * MINW_OK, or MINW_ETIMEOUT when a bounded wait inside a kernel gave up. */
MINW_API minw_status minw_get_last_device_error(void *stream);

/* ---------------------------------------------------------------------- */
/* Plan options (process-wide; no counterpart in the paper)                 */
/* ---------------------------------------------------------------------- */

/* Choices between kernel variants that compute the same results, and the
 * limit of the kernels' bounded waits.  The defaults (1, 1, 2, 1, 2, 1, 1, 1,
 * 1, 0, 2^31) are the measured fastest variants.  The options are read when a
 * launch is planned: a change applies to standalone calls made after it and
 * to networks created after it (a network keeps the plan it was created
 * with, except pdl and graph, read at every forward).
 * - cta_pairs: 256-channel layers with long K loops as CTA pairs (cta_group::2).
 * - channel_major: 64- and 128-channel layers as 128-channel x 256-pixel tiles
 *   when at least channel_major_min_tiles_per_sm such tiles per SM exist.
 * - dup_weights: a 64-channel channel-major tile loads its weight rows twice
 *   (else pads with zero rows).
 * - kblocks_per_stage: K blocks per pipeline stage of the tensor-core kernel (1 or 2).
 * - first_tma: first-layer input patches by TMA boxes (else per-word copies).
 * - pdl: programmatic dependent launch between the kernels of a forward.
 * - graph: minw_forward replays a captured CUDA graph.
 * - tma_lanes: lanes of each TMA warp of the tensor-core kernel that issue
 *   loads (1 to 8; each load keeps its issuing thread busy for about an L2
 *   round trip, so more issuers keep more bytes in flight).
 * - resident_weights: a tensor-core layer not split along K whose weights fit
 *   in shared memory keeps them there for all of its tiles (each CTA then
 *   works on one channel tile) instead of loading them per tile.  Off by
 *   default: it halves the loads per K block, but the shared memory the
 *   weights take shortens the activation ring, and on GB300 the CIFAR layers
 *   measured 0-6 % slower with it.
 * - first_tensor_cores: a first layer whose output is the next layer's
 *   levels (O a multiple of 64 up to 256) runs on the tensor cores with fp16
 *   split operands and an error bound, recomputing exactly the outputs whose
 *   level the bound leaves open (the levels are those of the fp32 chain
 *   either way); else the fp32 chain runs on the CUDA cores for every output.
 * - wait_cycles: SM clocks after which a bounded wait (TMA load, MMA, TMEM
 *   hand-off) gives up; the kernel then finishes without its outputs and
 *   minw_get_last_device_error reports MINW_ETIMEOUT. */
typedef struct {
    int32_t cta_pairs;
    int32_t channel_major;
    int32_t channel_major_min_tiles_per_sm;
    int32_t dup_weights;
    int32_t kblocks_per_stage;
    int32_t first_tma;
    int32_t pdl;
    int32_t graph;
    int32_t tma_lanes;
    int32_t resident_weights;
    int32_t first_tensor_cores;
    int64_t wait_cycles;
} minw_plan_options;

/* Current options (host struct). */
MINW_API minw_status minw_get_plan_options(minw_plan_options *out);
/* Replace the options; NULL restores the defaults.  MINW_EINVAL on a
 * kblocks_per_stage other than 1 or 2, tma_lanes outside 1..8 or a
 * non-positive wait_cycles. */
MINW_API minw_status minw_set_plan_options(const minw_plan_options *opt);

/* Test hook of the timeout path (no counterpart in the paper): the next launch
 * of the named kernel -- MINW_STALL_CONV_TC, the single-CTA tensor-core
 * convolution, or MINW_STALL_CONV_FIRST, the first layer with TMA patches --
 * first waits on a barrier that nothing completes.  That wait runs out after
 * wait_cycles, the kernel skips its work, drains its own loads and frees its
 * tensor memory, and minw_get_last_device_error reports MINW_ETIMEOUT once.
 * One launch only; 0 cancels a pending request.  No GPU fault is involved. */
enum { MINW_STALL_CONV_TC = 1, MINW_STALL_CONV_FIRST = 2 };
MINW_API minw_status minw_test_stall_next_launch(int32_t kernel);

/* ---------------------------------------------------------------------- */
/* Pipe rates (no counterpart in the paper: the measurement behind the      */
/* per-shape choice of path)                                                */
/* ---------------------------------------------------------------------- */

/* Throughput of the pipes the quantized convolution can run on, measured on
 * the current device with all SMs busy (host struct, filled by the call):
 * - sm_clock_mhz: SM clock during the tensor-core probes (clock64 / events);
 * - popc_per_s: 32-bit XOR + POPC + add per second, the inner loop of the
 *   bit-serial path (x 32 binary MACs);
 * - bmma_b1_mac_per_s, imma_s8_mac_per_s: the legacy warp MMAs the toolchain
 *   exposes for sm_103a (mma.sync m16n8k256 b1 xor.popc, m16n8k32 s8);
 * - tc_e4m3 / tc_e2m1 / tc_bf16_flop_per_s[j]: tcgen05.mma kind::f8f6f4,
 *   kind::mxf4 (unit scales) and kind::f16 at M = 128 and N = 128 (j = 0) or
 *   256 (j = 1), issued warp-uniformly with a commit every four MMAs;
 * - tma_box_cycles: SM clocks one issuing thread spends per 32 KB 4D TMA
 *   box (128-byte rows) from L2 with three boxes in flight.
 * Allocates about 10 MB of device memory for the call and runs about a second
 * of kernels on stream; MINW_ETIMEOUT if a bounded wait ran out. */
typedef struct {
    double sm_clock_mhz;
    double popc_per_s;
    double bmma_b1_mac_per_s;
    double imma_s8_mac_per_s;
    double tc_e4m3_flop_per_s[2];
    double tc_e2m1_flop_per_s[2];
    double tc_bf16_flop_per_s[2];
    double tma_box_cycles;
} minw_pipe_rates;
MINW_API minw_status minw_measure_pipe_rates(minw_pipe_rates *out, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* MINW_H */
