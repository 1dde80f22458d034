// kernels.cuh -- argument blocks and launchers shared by the translation units.
#pragma once

#include "common.cuh"

namespace minw {

// Everything one quantized-convolution launch needs (passed by value).
struct ConvArgs {
    const uint32_t *act;   // [B][H][W][PA][NW]
    const uint32_t *wgt;   // [O][kh][kw][PW][NW]
    int B, C, H, W, O, kh, kw, stride, pad;
    int Ho, Wo, NW;
    int bits_a, bits_w;
    long long M;           // B * Ho * Wo output pixels
    // epilogue
    int32_t *acc_out;      // int32 NCHW, unpooled (nullable)
    float *y_out;          // fp32 NCHW after BN [+HardTanh] (nullable)
    // weight update in place of the fp32 output (fully connected bf16 products):
    // y_out holds latent weights w, and each BN output g replaces its w by
    // min(1, max(-1, w - lr 2 alpha g 1[|w| <= 1]))
    int upd;
    float upd_lr, upd_2a;
    const float *scale;    // BN scale [O]
    const float *shift;    // BN shift [O]
    int pool;              // 2x2/2 max pool on the accumulator before BN
    int quant_out;         // HardTanh + quantize + pack into planes_out
    QParams qo;            // quantizer of the output
    uint32_t *planes_out;  // [B][Hp][Wp][qo.bits][ceil(O/32)] (nullable)
    uint8_t *codes_out;    // [B][Hp][Wp][O] E4M3 level codes (nullable; O % 16 == 0)
    // tensor-core operands: E4M3 level codes, or bf16 values when bf16 is set
    const uint8_t *act8;   // [B][H][W][C]
    const uint8_t *wgt8;   // [O][kh][kw][C]
    int bf16;              // operands are bf16 (weight-only quantized layers): fp32 outputs only
    int fp4;               // operands are E2M1 level codes, two channels per byte (C % 128 == 0)
    int codes_out4;        // codes_out receives E2M1 codes [B][Hp][Wp][O / 2]
    int res_codes4;        // res_codes holds E2M1 codes
    const float *thr;      // output-quantizer breakpoints [O][levels] (nullable: computed in-kernel)
    // residual blocks (tensor-core path): y = BN(acc) + shortcut before HardTanh + quantize
    const uint8_t *res_codes;  // shortcut as level codes [B][Hp][Wp][O] (nullable)
    float res_unit;            // value of one level unit of res_codes
    const float *res_f32;      // shortcut as fp32 NHWC (nullable)
    float *y_nhwc;             // BN output before the shortcut, fp32 NHWC (nullable)
    const float *ythr;         // breakpoints of the output quantizer on y [8] (nullable: computed in-kernel)
    // split-K (tensor-core path): zero-initialised workspace, left zero by every call
    void *workspace;       // nullable: no split
    size_t workspace_bytes;
    int ksplit;            // 0: chosen from the shape
    int n128;              // E2M1: single-CTA tiles of 128 pixels x 128 channels (two accumulators fit the
                           // tensor memory beside the scale factors)
    int pair_n128;         // E2M1: CTA pairs of 256 pixels x 128 channels (two accumulators fit the tensor
                           // memory beside the scale factors, so the epilogue overlaps the next MMAs)
    int ldc;               // bf16 operands: elements between pixel rows of act8 (0: C); the product reads
                           // channels 0 .. C of each row (the first C of a wider feature buffer)
    // bf16 operands, in place of y_out: HardTanh(BN(acc)) rounded to bf16 into NHWC rows of hb_ld
    // elements, channels hb_off .. hb_off + O of each (the next weight-only layer's input)
    uint16_t *hb_out;
    int hb_ld, hb_off;
    const float *hb_res;   // ... with a shortcut added before the HardTanh: fp32 NCHW [B][O][Ho][Wo] (nullable)
    float *hb_z;           // ... and the HardTanh output also as fp32 NCHW (nullable)
};

// First-layer convolution on the fp32 image (see conv_first.cu).
struct FirstArgs {
    const float *x;            // [B][C][H][W]
    const float *w;            // latent [O][C][kh][kw]
    const float *cscale;       // per-output-channel weight prescale (nullable)
    int quant_w;               // quantize weights with qw
    QParams qw;
    int B, C, H, W, O, kh, kw, stride, pad, Ho, Wo;
    const float *scale, *shift;
    int quant_out;
    QParams qo;
    uint32_t *planes_out;      // [B][Ho][Wo][qo.bits][ceil(O/32)] (nullable)
    uint8_t *codes_out;        // [B][Ho][Wo][O] E4M3 level codes (nullable)
    int codes4;                // codes_out receives E2M1 codes [B][Ho][Wo][O / 2] instead
    float *y_out;              // [B][O][Ho][Wo] (nullable)
    const float *thr;          // fp32 breakpoints [O][8] (nullable: computed in-kernel)
    const float *wt;           // prepared weights [K][O] (levels when quantized; nullable: from w)
    long long wait_cycles;     // limit of the bounded patch waits (set by the launcher)
    int stall;                 // timeout-path test: first wait on a barrier nothing completes (set by the launcher)
};

// Launchers (host).  Return MINW_OK or an error status.
minw_status launch_conv_first(const FirstArgs &a, cudaStream_t s);
// The tensor-core first layer (conv_first_tc.cu): whether it applies, its
// launch, and its timeout flag (as take_first_error).
bool first_tc_supported(const FirstArgs &a);
minw_status launch_first_tc(const FirstArgs &a, cudaStream_t s);
int take_first_tc_error();
// The first-layer kernels' timeout flag: 1 if set (and clears it), 0, or -1 on a CUDA error.
int take_first_error();
minw_status launch_ythresholds(const QParams &q, float *out, cudaStream_t s);
minw_status launch_first_weights(const float *w, int O, int K, int quant_w, const QParams &qw, const float *cscale,
                                 float *wt, cudaStream_t s);
minw_status launch_thresholds_f32(const float *scale, const float *shift, int O, const QParams &q, float *out,
                                  cudaStream_t s);
minw_status launch_conv_popc(const ConvArgs &a, cudaStream_t s);
minw_status make_conv_args(ConvArgs &a, const uint32_t *act, int B, int C, int H, int W,
                           int bits_a, const uint32_t *wgt, int O, int kh, int kw, int bits_w,
                           int stride, int pad);
int choose_variant(const ConvArgs &a, int requested);
minw_status run_conv(const ConvArgs &a, int variant, cudaStream_t s);
minw_status launch_conv_tc(const ConvArgs &a, cudaStream_t s);
// bf16 convolution (minw_conv2d_bf16) with an optional split-K workspace;
// with workspace_need set, only stores the workspace bytes the shape can use.
minw_status conv2d_bf16(const uint16_t *act, int B, int C, int H, int W, const uint16_t *wgt, int O, int kh, int kw,
                        int bits_w, int stride, int pad, int pool, const float *scale, const float *shift,
                        float *y_out, void *workspace, size_t workspace_bytes, size_t *workspace_need,
                        cudaStream_t s, int upd = 0, float upd_lr = 0.0f, float upd_2a = 0.0f, int ldc = 0);
// The same convolution with the HardTanh + bf16 NHWC epilogue (ConvArgs::hb_out): input rows of
// ldc elements (0: C), output rows of hb_ld elements at channel offset hb_off.
minw_status conv2d_bf16_hardtanh(const uint16_t *act, int B, int C, int H, int W, int ldc, const uint16_t *wgt,
                                 int O, int kh, int kw, int bits_w, int stride, int pad, const float *scale,
                                 const float *shift, uint16_t *hb_out, int hb_ld, int hb_off, cudaStream_t s,
                                 const float *res = nullptr, float *z = nullptr);
bool conv_tc_supported(const ConvArgs &a);
// Workspace the tensor-core path needs to split K for this shape (0: it does not split).
size_t conv_tc_workspace_bytes(const ConvArgs &a);
// Smallest workspace with which this shape still splits K (two slices); 0 when it does not split.
size_t conv_tc_min_split_bytes(const ConvArgs &a);
// K slices of the tensor-core plan for this shape and workspace (1: no split; 0: not supported).
int conv_tc_ksplit(const ConvArgs &a);
// Whether the plan of this shape runs as CTA pairs of 128-channel E2M1 tiles (a.pair_n128 honoured).
bool conv_tc_pairs128(const ConvArgs &a);
// Whether a.n128 changes this shape's plan to single-CTA 128-channel E2M1 tiles.
bool conv_tc_n128(const ConvArgs &a);
// Kernels one tensor-core launch issues for this shape and workspace (2 with a split).
int conv_tc_launches(const ConvArgs &a);
minw_status launch_thresholds(const float *scale, const float *shift, int O, const QParams &q, float *out,
                              cudaStream_t s);

}  // namespace minw
