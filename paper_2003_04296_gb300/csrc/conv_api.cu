// conv_api.cu -- host entry points of the quantized convolution: argument
// checks, output-shape arithmetic and the per-shape choice between the
// popcount path and the tensor-core path.
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

using namespace minw;
using namespace minw_host;

namespace minw {

// Fill a ConvArgs from the ABI arguments; returns MINW_OK or the error.
minw_status make_conv_args(ConvArgs &a, const uint32_t *act, int B, int C, int H, int W,
                           int bits_a, const uint32_t *wgt, int O, int kh, int kw, int bits_w,
                           int stride, int pad) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || O <= 0 || kh <= 0 || kw <= 0 || stride <= 0 ||
        pad < 0)
        return MINW_EINVAL;
    if (bits_a < 1 || bits_a > 3 || bits_w < 1 || bits_w > 3) return MINW_EINVAL;
    if (!act || !wgt || !aligned16(act) || !aligned16(wgt)) return MINW_EINVAL;
    if (C % 32 != 0) return MINW_EUNSUPPORTED;
    if (pad >= kh || pad >= kw) return MINW_EUNSUPPORTED;
    const int Ho = (H + 2 * pad - kh) / stride + 1;
    const int Wo = (W + 2 * pad - kw) / stride + 1;
    if (Ho <= 0 || Wo <= 0) return MINW_EINVAL;
    if ((long long)B * H * W >= (1ll << 31) / 4) return MINW_EUNSUPPORTED;
    a = ConvArgs{};
    a.act = act; a.wgt = wgt;
    a.B = B; a.C = C; a.H = H; a.W = W; a.O = O; a.kh = kh; a.kw = kw;
    a.stride = stride; a.pad = pad; a.Ho = Ho; a.Wo = Wo; a.NW = C / 32;
    a.bits_a = bits_a; a.bits_w = bits_w;
    a.M = (long long)B * Ho * Wo;
    return MINW_OK;
}

// Per-shape choice for a layer whose input layout is still free (the network
// planner): the tensor-core path wherever it covers the shape, the popcount
// path elsewhere.
int choose_variant(const ConvArgs &a, int requested) {
    if (requested == MINW_VARIANT_POPC) return MINW_VARIANT_POPC;
    if (requested == MINW_VARIANT_TC) return MINW_VARIANT_TC;
    return conv_tc_supported(a) ? MINW_VARIANT_TC : MINW_VARIANT_POPC;
}

// Packed-plane operands run on the popcount path; the tensor-core path takes
// its operands in the codes layout (minw_conv2d_codes / minw_conv_block_codes).
minw_status run_conv(const ConvArgs &a, int variant, cudaStream_t s) {
    if (variant == MINW_VARIANT_TC) return MINW_EUNSUPPORTED;
    return launch_conv_popc(a, s);
}

}  // namespace minw

extern "C" {

minw_status minw_conv2d(const uint32_t *act, int32_t B, int32_t C, int32_t H, int32_t W,
                        int32_t bits_a, const uint32_t *wgt, int32_t O, int32_t kh, int32_t kw,
                        int32_t bits_w, int32_t stride, int32_t pad, int32_t *acc_out,
                        const float *scale, const float *shift, float *y_out, int32_t variant,
                        void *stream) {
    ConvArgs a;
    minw_status st = make_conv_args(a, act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad);
    if (st != MINW_OK) return st;
    if (!acc_out && !y_out) return MINW_EINVAL;
    if (y_out && (!scale || !shift)) return MINW_EINVAL;
    if (variant < 0 || variant > 2) return MINW_EINVAL;
    a.acc_out = acc_out;
    a.y_out = y_out;
    a.scale = scale;
    a.shift = shift;
    return run_conv(a, variant, (cudaStream_t)stream);
}

minw_status minw_conv_block(const uint32_t *act, int32_t B, int32_t C, int32_t H, int32_t W,
                            int32_t bits_a, const uint32_t *wgt, int32_t O, int32_t kh, int32_t kw,
                            int32_t bits_w, int32_t stride, int32_t pad, int32_t pool,
                            const float *scale, const float *shift, const minw_quant *q_out,
                            uint32_t *planes_out, float *y_out, int32_t variant, void *stream) {
    ConvArgs a;
    minw_status st = make_conv_args(a, act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad);
    if (st != MINW_OK) return st;
    if (!scale || !shift) return MINW_EINVAL;
    if (q_out && (!valid_quant(q_out) || !planes_out)) return MINW_EINVAL;
    if (!q_out && !y_out) return MINW_EINVAL;
    if (pool != 0 && pool != 1) return MINW_EINVAL;
    if (pool && ((a.Ho & 1) || (a.Wo & 1))) return MINW_EUNSUPPORTED;
    if (variant < 0 || variant > 2) return MINW_EINVAL;
    a.scale = scale;
    a.shift = shift;
    a.pool = pool;
    a.quant_out = q_out != nullptr;
    if (q_out) a.qo = to_qparams(q_out);
    a.planes_out = planes_out;
    a.y_out = y_out;
    return run_conv(a, variant, (cudaStream_t)stream);
}

static minw_status make_codes_args(ConvArgs &a, const uint8_t *act, int B, int C, int H, int W, int bits_a,
                                   const uint8_t *wgt, int O, int kh, int kw, int bits_w, int stride, int pad,
                                   bool check_ptrs = true) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || O <= 0 || kh <= 0 || kw <= 0 || stride <= 0 || pad < 0)
        return MINW_EINVAL;
    if (bits_a < 1 || bits_a > 3 || bits_w < 1 || bits_w > 3) return MINW_EINVAL;
    if (check_ptrs && (!act || !wgt || !aligned16(act) || !aligned16(wgt))) return MINW_EINVAL;
    if (C % 64 != 0 || (stride != 1 && stride != 2) || pad >= kh || pad >= kw) return MINW_EUNSUPPORTED;
    const int Ho = (H + 2 * pad - kh) / stride + 1;
    const int Wo = (W + 2 * pad - kw) / stride + 1;
    if (Ho <= 0 || Wo <= 0) return MINW_EINVAL;
    if ((long long)B * H * W * C >= (1ll << 40)) return MINW_EUNSUPPORTED;
    a = ConvArgs{};
    a.act8 = act; a.wgt8 = wgt;
    a.B = B; a.C = C; a.H = H; a.W = W; a.O = O; a.kh = kh; a.kw = kw;
    a.stride = stride; a.pad = pad; a.Ho = Ho; a.Wo = Wo; a.NW = C / 32;
    a.bits_a = bits_a; a.bits_w = bits_w;
    a.M = (long long)B * Ho * Wo;
    return MINW_OK;
}

}  // extern "C"

namespace minw {

minw_status conv2d_bf16(const uint16_t *act, int B, int C, int H, int W, const uint16_t *wgt, int O, int kh, int kw,
                        int bits_w, int stride, int pad, int pool, const float *scale, const float *shift,
                        float *y_out, void *workspace, size_t workspace_bytes, size_t *workspace_need,
                        cudaStream_t s, int upd, float upd_lr, float upd_2a, int ldc) {
    ConvArgs a;
    if (ldc != 0 && (ldc < C || ldc % 64 != 0)) return MINW_EINVAL;
    const bool query = workspace_need != nullptr;      // shape only: no pointer is used
    minw_status st = make_codes_args(a, reinterpret_cast<const uint8_t *>(act), B, C, H, W, 1,
                                     reinterpret_cast<const uint8_t *>(wgt), O, kh, kw, bits_w, stride, pad, !query);
    if (st != MINW_OK) return st;
    if (!query && (!scale || !shift || !y_out)) return MINW_EINVAL;
    if (pool != 0 && pool != 1) return MINW_EINVAL;
    if (pool && ((a.Ho & 1) || (a.Wo & 1))) return MINW_EUNSUPPORTED;
    if ((long long)B * H * W * (ldc ? ldc : C) >= (1ll << 39)) return MINW_EUNSUPPORTED;
    a.bf16 = 1;
    a.ldc = ldc;
    a.bits_a = 0;
    a.scale = scale;
    a.shift = shift;
    a.pool = pool;
    a.y_out = y_out;
    if (query) {
        *workspace_need = conv_tc_workspace_bytes(a);
        return MINW_OK;
    }
    if (workspace != nullptr && !aligned16(workspace)) return MINW_EINVAL;
    a.workspace = workspace;
    a.workspace_bytes = workspace_bytes;
    a.upd = upd;
    a.upd_lr = upd_lr;
    a.upd_2a = upd_2a;
    return launch_conv_tc(a, s);
}

minw_status conv2d_bf16_hardtanh(const uint16_t *act, int B, int C, int H, int W, int ldc, const uint16_t *wgt,
                                 int O, int kh, int kw, int bits_w, int stride, int pad, const float *scale,
                                 const float *shift, uint16_t *hb_out, int hb_ld, int hb_off, cudaStream_t s,
                                 const float *res, float *z) {
    ConvArgs a;
    if (ldc != 0 && (ldc < C || ldc % 64 != 0)) return MINW_EINVAL;
    if (!scale || !shift || !hb_out || hb_off < 0 || hb_ld < hb_off + O) return MINW_EINVAL;
    minw_status st = make_codes_args(a, reinterpret_cast<const uint8_t *>(act), B, C, H, W, 1,
                                     reinterpret_cast<const uint8_t *>(wgt), O, kh, kw, bits_w, stride, pad);
    if (st != MINW_OK) return st;
    if ((long long)B * H * W * (ldc ? ldc : C) >= (1ll << 39) || a.M * hb_ld >= (1ll << 39)) return MINW_EUNSUPPORTED;
    a.bf16 = 1;
    a.bits_a = 0;
    a.ldc = ldc;
    a.scale = scale;
    a.shift = shift;
    a.hb_out = hb_out;
    a.hb_ld = hb_ld;
    a.hb_off = hb_off;
    a.hb_res = res;
    a.hb_z = z;
    return launch_conv_tc(a, s);
}

}  // namespace minw

extern "C" {

minw_status minw_conv2d_codes(const uint8_t *act, int32_t B, int32_t C, int32_t H, int32_t W, int32_t bits_a,
                              const uint8_t *wgt, int32_t O, int32_t kh, int32_t kw, int32_t bits_w,
                              int32_t stride, int32_t pad, int32_t *acc_out, const float *scale,
                              const float *shift, float *y_out, void *stream) {
    ConvArgs a;
    minw_status st = make_codes_args(a, act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad);
    if (st != MINW_OK) return st;
    if (!acc_out && !y_out) return MINW_EINVAL;
    if (y_out && (!scale || !shift)) return MINW_EINVAL;
    a.acc_out = acc_out;
    a.y_out = y_out;
    a.scale = scale;
    a.shift = shift;
    return launch_conv_tc(a, (cudaStream_t)stream);
}

minw_status minw_conv2d_bf16_hardtanh(const uint16_t *act, int32_t B, int32_t C, int32_t H, int32_t W, int32_t ldc,
                                      const uint16_t *wgt, int32_t O, int32_t kh, int32_t kw, int32_t bits_w,
                                      int32_t stride, int32_t pad, const float *scale, const float *shift,
                                      uint16_t *out, int32_t out_ld, int32_t out_off, const float *residual,
                                      float *y_out, void *stream) {
    return minw::conv2d_bf16_hardtanh(act, B, C, H, W, ldc, wgt, O, kh, kw, bits_w, stride, pad, scale, shift, out,
                                      out_ld, out_off, (cudaStream_t)stream, residual, y_out);
}

minw_status minw_conv2d_bf16(const uint16_t *act, int32_t B, int32_t C, int32_t H, int32_t W, const uint16_t *wgt,
                             int32_t O, int32_t kh, int32_t kw, int32_t bits_w, int32_t stride, int32_t pad,
                             int32_t pool, const float *scale, const float *shift, float *y_out, void *stream) {
    return minw::conv2d_bf16(act, B, C, H, W, wgt, O, kh, kw, bits_w, stride, pad, pool, scale, shift, y_out,
                             nullptr, 0, nullptr, (cudaStream_t)stream);
}

minw_status minw_conv_block_codes(const uint8_t *act, int32_t B, int32_t C, int32_t H, int32_t W,
                                  int32_t bits_a, const uint8_t *wgt, int32_t O, int32_t kh, int32_t kw,
                                  int32_t bits_w, int32_t stride, int32_t pad, int32_t pool, const float *scale,
                                  const float *shift, const minw_quant *q_out, uint8_t *codes_out,
                                  uint32_t *planes_out, float *y_out, void *stream) {
    ConvArgs a;
    minw_status st = make_codes_args(a, act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad);
    if (st != MINW_OK) return st;
    if (!scale || !shift) return MINW_EINVAL;
    if (q_out && (!valid_quant(q_out) || (!planes_out && !codes_out))) return MINW_EINVAL;
    if (codes_out && (O % 16 != 0 || !aligned16(codes_out))) return MINW_EUNSUPPORTED;
    if (!q_out && !y_out) return MINW_EINVAL;
    if (pool != 0 && pool != 1) return MINW_EINVAL;
    if (pool && ((a.Ho & 1) || (a.Wo & 1))) return MINW_EUNSUPPORTED;
    a.scale = scale;
    a.shift = shift;
    a.pool = pool;
    a.quant_out = q_out != nullptr;
    if (q_out) a.qo = to_qparams(q_out);
    a.planes_out = planes_out;
    a.codes_out = q_out ? codes_out : nullptr;
    a.y_out = y_out;
    return launch_conv_tc(a, (cudaStream_t)stream);
}

minw_status minw_conv_block_codes_ex(const uint8_t *act, int32_t B, int32_t C, int32_t H, int32_t W,
                                     int32_t bits_a, const uint8_t *wgt, int32_t O, int32_t kh, int32_t kw,
                                     int32_t bits_w, int32_t stride, int32_t pad, int32_t pool,
                                     const float *scale, const float *shift, const minw_quant *q_out,
                                     uint8_t *codes_out, uint32_t *planes_out, float *y_out,
                                     const minw_block_extra *extra, void *stream) {
    ConvArgs a;
    minw_status st = make_codes_args(a, act, B, C, H, W, bits_a, wgt, O, kh, kw, bits_w, stride, pad);
    if (st != MINW_OK) return st;
    if (q_out && (!valid_quant(q_out) || (!planes_out && !codes_out))) return MINW_EINVAL;
    if (codes_out && (O % 16 != 0 || !aligned16(codes_out))) return MINW_EUNSUPPORTED;
    if (pool != 0 && pool != 1) return MINW_EINVAL;
    if (pool && ((a.Ho & 1) || (a.Wo & 1))) return MINW_EUNSUPPORTED;
    if (extra && extra->res_codes && extra->res_f32) return MINW_EINVAL;
    if (extra && extra->res_codes && (extra->res_bits < 1 || extra->res_bits > 3)) return MINW_EINVAL;
    if (extra && ((unsigned)extra->in_format > 1u || (unsigned)extra->out_format > 1u ||
                  (unsigned)extra->res_format > 1u))
        return MINW_EINVAL;
    if (extra && extra->acc_out && pool) return MINW_EUNSUPPORTED;
    const bool any_out = q_out || y_out || (extra && (extra->y_nhwc || extra->acc_out));
    if (!any_out) return MINW_EINVAL;
    if ((q_out || y_out || (extra && extra->y_nhwc)) && (!scale || !shift)) return MINW_EINVAL;
    a.scale = scale;
    a.shift = shift;
    a.pool = pool;
    a.quant_out = q_out != nullptr;
    if (q_out) a.qo = to_qparams(q_out);
    a.planes_out = planes_out;
    a.codes_out = q_out ? codes_out : nullptr;
    a.y_out = y_out;
    if (extra) {
        a.res_codes = extra->res_codes;
        a.res_unit = extra->res_bits == 3 ? 0.25f : 1.0f;
        a.res_f32 = extra->res_f32;
        a.y_nhwc = extra->y_nhwc;
        a.fp4 = extra->in_format == MINW_CODES_E2M1;
        a.codes_out4 = extra->out_format == MINW_CODES_E2M1;
        a.res_codes4 = extra->res_format == MINW_CODES_E2M1;
        a.acc_out = extra->acc_out;
        a.pair_n128 = (extra->e2m1_pairs != 0 && a.fp4) ? 1 : 0;
    }
    return launch_conv_tc(a, (cudaStream_t)stream);
}

size_t minw_fc_workspace_bytes(int32_t B, int32_t K, int32_t O) {
    if (B <= 0 || K <= 0 || O <= 0 || K % 128 != 0) return 0;
    ConvArgs a{};
    a.B = B; a.C = K; a.H = 1; a.W = 1; a.O = O; a.kh = 1; a.kw = 1; a.stride = 1; a.pad = 0;
    a.Ho = 1; a.Wo = 1; a.NW = K / 32; a.M = B;
    return conv_tc_workspace_bytes(a);
}

int32_t minw_fc_ksplit(int32_t B, int32_t K, int32_t O, size_t workspace_bytes) {
    if (B <= 0 || K <= 0 || O <= 0 || K % 128 != 0) return 0;
    ConvArgs a{};
    a.B = B; a.C = K; a.H = 1; a.W = 1; a.O = O; a.kh = 1; a.kw = 1; a.stride = 1; a.pad = 0;
    a.Ho = 1; a.Wo = 1; a.NW = K / 32; a.M = B;
    a.y_out = reinterpret_cast<float *>(256);           // shape planning only: never dereferenced
    a.workspace = workspace_bytes ? reinterpret_cast<void *>(256) : nullptr;
    a.workspace_bytes = workspace_bytes;
    return conv_tc_ksplit(a);
}

minw_status minw_fc_codes(const uint8_t *act, int32_t B, int32_t K, int32_t bits_a, const uint8_t *wgt, int32_t O,
                          int32_t bits_w, const float *scale, const float *shift, const minw_quant *q_out,
                          uint8_t *codes_out, uint32_t *planes_out, float *y_out, int32_t *acc_out,
                          void *workspace, size_t workspace_bytes, void *stream) {
    ConvArgs a;
    minw_status st = make_codes_args(a, act, B, K, 1, 1, bits_a, wgt, O, 1, 1, bits_w, 1, 0);
    if (st != MINW_OK) return st;
    if (q_out && (!valid_quant(q_out) || (!planes_out && !codes_out))) return MINW_EINVAL;
    if ((q_out || y_out) && (!scale || !shift)) return MINW_EINVAL;
    if (codes_out && (O % 16 != 0 || !aligned16(codes_out))) return MINW_EUNSUPPORTED;
    if (!q_out && !y_out && !acc_out) return MINW_EINVAL;
    if (workspace && !aligned16(workspace)) return MINW_EINVAL;
    a.scale = scale;
    a.shift = shift;
    a.quant_out = q_out != nullptr;
    if (q_out) a.qo = to_qparams(q_out);
    a.planes_out = planes_out;
    a.codes_out = q_out ? codes_out : nullptr;
    a.y_out = y_out;
    a.acc_out = acc_out;
    a.workspace = workspace_bytes ? workspace : nullptr;
    a.workspace_bytes = workspace_bytes;
    return launch_conv_tc(a, (cudaStream_t)stream);
}

}  // extern "C"
