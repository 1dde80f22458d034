// resnet.cu -- a ResNet-18-shaped MINW-Net (Table V's network) on the
// tensor-core path.
//
// The paper fixes the layer block (QuantizedConv - [pool] - BN - HardTanh,
// Sec. III-E), that the input of the first convolution stays fp32, and (for
// ResNet-18, Table V's first footnote) that the first layer is not quantized.
// It leaves the residual wiring open; the reading implemented here:
//   u = h(x)                       (block input, quantized levels)
//   v = h(HardTanh(BN1(conv1(u))))
//   y = BN2(conv2(v)) + s,  s = u (identity) or BN_d(conv_d(u)) (1x1 / 2)
//   out = h(HardTanh(y))           (the next block's quantized input)
// with the sum in fp32.  Stem: fp32 7x7/2 convolution -> 3x3/2 max pool ->
// BN -> HardTanh -> quantize (the block order); head: global average pool of
// the last block's levels -> fp32 fully connected layer -> BN -> logits.
//
// The stem's pool runs on quantized levels: BN + HardTanh + h is monotone in
// the convolution output (non-decreasing for a BN scale >= 0, non-increasing
// for < 0), so the level of the max-pooled output equals the max (resp. min)
// over the window of the levels -- the same result as pooling first, without
// an fp32 copy of the 112x112 stem output.
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <vector>

#include "net.cuh"

using namespace minw;
using namespace minw_host;

namespace {

// Integer units of an E4M3 level code (0, +-1, +-2, +-4).
__device__ __forceinline__ int code_to_units(uint32_t c) {
    if ((c & 0x7Fu) == 0u) return 0;
    const int m = 1 << (((c >> 3) & 0xFu) - 7u);
    return (c & 0x80u) ? -m : m;
}

// E4M3 level codes (0x00, +-0x38, +-0x40, +-0x48), four per word, mapped to
// bytes whose unsigned order is the order of the levels (positive c -> c ^ 0x80,
// negative c -> c ^ 0xFF), and back.
__device__ __forceinline__ uint32_t codes_to_ordered(uint32_t w) {
    return w ^ 0x80808080u ^ (((w >> 7) & 0x01010101u) * 0x7Fu);
}
__device__ __forceinline__ uint32_t ordered_to_codes(uint32_t o) {
    return o ^ 0x80808080u ^ (((~o >> 7) & 0x01010101u) * 0x7Fu);
}

// 3x3 / stride 2 / pad 1 pooling of level codes [B][H][W][C] -> [B][Ho][Wo][C]:
// per channel the max of the levels when the stem's BN scale is >= 0, the min
// otherwise (padded taps skipped).  Thread = one output pixel x 16 channels;
// the codes are compared as order-preserving bytes, four per word.  Index
// arithmetic in 32 bits (the host keeps B Ho Wo C / 16 below 2^31); the
// max/min byte selectors of each channel group sit in shared memory.
__global__ void __launch_bounds__(256) pool_levels_kernel(const uint8_t *__restrict__ in, int B, int H, int W, int C,
                                                          const float *__restrict__ scale, uint8_t *__restrict__ out,
                                                          int Ho, int Wo) {
    __shared__ uint32_t sup[64];                     // C / 4 words: 0xFF bytes where the scale is >= 0
    for (int i = threadIdx.x; i < (C >> 2); i += blockDim.x) {
        uint32_t m = 0u;
        for (int j = 0; j < 4; ++j) m |= (__ldg(scale + 4 * i + j) >= 0.0f ? 0xFFu : 0u) << (8 * j);
        sup[i] = m;
    }
    __syncthreads();
    pdl_wait();
    pdl_trigger();
    const unsigned groups = (unsigned)C >> 4;
    const unsigned total = (unsigned)B * (unsigned)Ho * (unsigned)Wo * groups;
    for (unsigned t = blockIdx.x * blockDim.x + threadIdx.x; t < total; t += gridDim.x * blockDim.x) {
        const unsigned g = t % groups, pix = t / groups;
        const unsigned xo = pix % (unsigned)Wo, r = pix / (unsigned)Wo;
        const unsigned yo = r % (unsigned)Ho, b = r / (unsigned)Ho;
        uint32_t mx[4], mn[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            mx[q] = 0x00000000u;
            mn[q] = 0xFFFFFFFFu;
        }
        const uint8_t *base = in + ((size_t)b * H * W) * C + g * 16;
#pragma unroll
        for (int ky = 0; ky < 3; ++ky) {
            const int yi = 2 * (int)yo - 1 + ky;
            if (yi < 0 || yi >= H) continue;
#pragma unroll
            for (int kx = 0; kx < 3; ++kx) {
                const int xi = 2 * (int)xo - 1 + kx;
                if (xi < 0 || xi >= W) continue;
                const uint4 v = __ldg(reinterpret_cast<const uint4 *>(base + ((size_t)yi * W + xi) * C));
                const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint32_t o = codes_to_ordered(w[q]);
                    mx[q] = __vmaxu4(mx[q], o);
                    mn[q] = __vminu4(mn[q], o);
                }
            }
        }
        uint32_t res[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t up = sup[4 * g + q];
            res[q] = ordered_to_codes((mx[q] & up) | (mn[q] & ~up));
        }
        *reinterpret_cast<uint4 *>(out + (size_t)pix * C + g * 16) = make_uint4(res[0], res[1], res[2], res[3]);
    }
}

// Head, first part: global average pool of level codes [B][HW][C] (E4M3
// bytes, or E2M1 nibbles with fp4) -> fp32 [B][C]; thread = (image, channel),
// one fp32 sum over the pixels in order, then one division.
__global__ void __launch_bounds__(256) avgpool_levels_kernel(const uint8_t *__restrict__ X, int B, int HW, int C,
                                                             float unit, int fp4, float *__restrict__ pooled) {
    pdl_wait();
    pdl_trigger();
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= B * C) return;
    const int b = i / C, c = i - b * C;
    float s = 0.0f;
    if (fp4) {
        const uint8_t *src = X + ((long long)b * HW * C + c) / 2;
        const int sh = 4 * (c & 1);
        for (int p = 0; p < HW; ++p) s += code_units_e2m1(__ldg(src + (long long)p * (C / 2)) >> sh) * unit;
    } else {
        const uint8_t *src = X + (long long)b * HW * C + c;
        for (int p = 0; p < HW; ++p) s += (float)code_to_units(__ldg(src + (long long)p * C)) * unit;
    }
    pooled[i] = s / (float)HW;
}

// Head, second part: fp32 fully connected layer (one fmaf chain over the
// features in order; weights transposed to [C][classes]) and BN (fmaf).
// CTA = 8 images x 32 classes, one output per thread (many small chains keep
// the SMs busy); the pooled features of its images sit in shared memory.
constexpr int HEAD_IMGS = 8, HEAD_CLS = 32;
__global__ void __launch_bounds__(HEAD_IMGS * HEAD_CLS) fc_head_kernel(const float *__restrict__ pooled, int B, int C,
                                                                       const float *__restrict__ wt, int classes,
                                                                       const float *__restrict__ scale,
                                                                       const float *__restrict__ shift,
                                                                       float *__restrict__ logits) {
    extern __shared__ float sp[];                    // [HEAD_IMGS][C]
    pdl_wait();
    pdl_trigger();
    const int b0 = blockIdx.y * HEAD_IMGS;
    const int nimg = min(HEAD_IMGS, B - b0);
    const int tid = threadIdx.y * HEAD_CLS + threadIdx.x;
    for (int i = tid; i < HEAD_IMGS * C; i += HEAD_IMGS * HEAD_CLS)
        sp[i] = i < nimg * C ? pooled[(long long)b0 * C + i] : 0.0f;
    __syncthreads();
    const int o = blockIdx.x * HEAD_CLS + threadIdx.x, im = threadIdx.y;
    if (o >= classes || im >= nimg) return;
    const float *x = sp + im * C;
    float acc = 0.0f;
#pragma unroll 8
    for (int k = 0; k < C; ++k) acc = fmaf(x[k], __ldg(wt + (long long)k * classes + o), acc);
    logits[(long long)(b0 + im) * classes + o] = fmaf(acc, __ldg(scale + o), __ldg(shift + o));
}

__global__ void transpose_kernel(const float *__restrict__ in, int rows, int cols, float *__restrict__ out) {
    const long long n = (long long)rows * cols;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const int r = (int)(i / cols), c = (int)(i - (long long)r * cols);
        out[(long long)c * rows + r] = in[i];
    }
}

}  // namespace

// Tensors of 128 channels or more are held as E2M1 codes (two channels per
// byte), the 64-channel ones as E4M3 codes: a convolution's input and weights
// follow its C, its quantized output (and a residual shortcut) its O.
static int e2m1_channels(int c) { return c % 128 == 0 ? 1 : 0; }

// One quantized convolution of a block.
struct ResConv {
    int C, H, W, O, k, stride, pad, Ho, Wo;
    uint8_t *wcodes = nullptr;
    float *scale = nullptr, *shift = nullptr, *thr = nullptr;
};

struct ResBlock {
    ResConv c1, c2, d;
    bool down = false;
};

struct ResNetPlan {
    int hw = 0, classes = 0, bits_a = 0, bits_w = 0;
    minw_quant qa{};
    float *stem_w = nullptr, *stem_scale = nullptr, *stem_shift = nullptr, *stem_thr = nullptr;
    float *stem_wt = nullptr;              // stem weights as [147][64]
    int Hs = 0, Hp = 0;                    // stem output, pooled size
    ResBlock blocks[8];
    float *fc_wt = nullptr, *fc_scale = nullptr, *fc_shift = nullptr;
    float *pooled = nullptr;               // head: average-pooled features [max_batch][512]
    float *ythr = nullptr;                 // breakpoints of the activation quantizer on y [8]
    uint8_t *S = nullptr, *X = nullptr, *Y = nullptr, *V = nullptr;
    float *D = nullptr;
};

template <typename T>
static minw_status alloc_owned(minw_net *n, T **p, size_t count) {
    void *q = nullptr;
    if (cudaMalloc(&q, count * sizeof(T) + 16) != cudaSuccess) return MINW_ECUDA;
    n->owned.push_back(q);
    *p = reinterpret_cast<T *>(q);
    return MINW_OK;
}

static minw_status copy_owned(minw_net *n, float **dst, const float *src, size_t count, cudaStream_t s) {
    minw_status st = alloc_owned(n, dst, count);
    if (st != MINW_OK) return st;
    return cudaMemcpyAsync(*dst, src, count * sizeof(float), cudaMemcpyDeviceToDevice, s) == cudaSuccess ? MINW_OK
                                                                                                         : MINW_ECUDA;
}

static ConvArgs conv_args(const ResConv &c, int B) {
    ConvArgs a{};
    a.B = B; a.C = c.C; a.H = c.H; a.W = c.W; a.O = c.O; a.kh = c.k; a.kw = c.k;
    a.stride = c.stride; a.pad = c.pad; a.Ho = c.Ho; a.Wo = c.Wo; a.NW = c.C / 32;
    a.M = (long long)B * c.Ho * c.Wo;
    a.scale = c.scale; a.shift = c.shift;
    a.wgt8 = c.wcodes;
    a.fp4 = e2m1_channels(c.C);
    return a;
}

void resnet_free(minw_net *net) {
    delete net->res;
    net->res = nullptr;
}

int32_t resnet_ops(const minw_net *net) {
    int ops = 3;                           // stem, pool, head
    for (const ResBlock &bk : net->res->blocks) ops += bk.down ? 3 : 2;
    return ops;
}

// Variant of each op in forward order: 0 for the stem, its pool and the head,
// MINW_VARIANT_TC or MINW_VARIANT_TC_E2M1 for the block convolutions.
void resnet_variants(const minw_net *net, int32_t *variants) {
    int k = 0;
    variants[k++] = 0;
    variants[k++] = 0;
    for (const ResBlock &bk : net->res->blocks) {
        variants[k++] = e2m1_channels(bk.c1.C) ? MINW_VARIANT_TC_E2M1 : MINW_VARIANT_TC;
        if (bk.down) variants[k++] = e2m1_channels(bk.d.C) ? MINW_VARIANT_TC_E2M1 : MINW_VARIANT_TC;
        variants[k++] = e2m1_channels(bk.c2.C) ? MINW_VARIANT_TC_E2M1 : MINW_VARIANT_TC;
    }
    variants[k++] = 0;
}

// Arguments of one block convolution: which = 0 conv1 (X -> V, quantized),
// 1 the 1x1 / 2 shortcut (X -> D, fp32 BN output), 2 conv2 (V -> Y with the
// shortcut added, quantized).
static ConvArgs block_conv(const minw_net *net, const ResBlock &bk, int which, int B, const uint8_t *X, uint8_t *Y) {
    const ResNetPlan *R = net->res;
    ConvArgs a = conv_args(which == 0 ? bk.c1 : which == 1 ? bk.d : bk.c2, B);
    a.workspace = net->ws;
    a.workspace_bytes = net->ws_bytes;
    if (which == 0) {
        a.act8 = X;
        a.quant_out = 1; a.qo = to_qparams(&R->qa); a.thr = bk.c1.thr;
        a.codes_out = R->V;
        a.codes_out4 = e2m1_channels(bk.c1.O);
    } else if (which == 1) {
        a.act8 = X;
        a.y_nhwc = R->D;
    } else {
        a.act8 = R->V;
        a.quant_out = 1; a.qo = to_qparams(&R->qa);
        a.codes_out = Y;
        a.codes_out4 = e2m1_channels(bk.c2.O);
        a.ythr = R->ythr;
        if (bk.down) {
            a.res_f32 = R->D;
        } else {
            a.res_codes = X;
            a.res_codes4 = e2m1_channels(bk.c2.O);
            a.res_unit = R->bits_a == 3 ? 0.25f : 1.0f;
        }
    }
    return a;
}

int32_t resnet_kernels(const minw_net *net) {
    int k = 4;                             // stem, pool, average pool + classifier
    const ResNetPlan *R = net->res;
    for (const ResBlock &bk : R->blocks)
        for (int which = 0; which < 3; ++which)
            if (which != 1 || bk.down) k += conv_tc_launches(block_conv(net, bk, which, net->max_batch, R->X, R->Y));
    return k;
}

extern "C" minw_status minw_resnet18_create(const minw_resnet18_desc *d, int32_t max_batch, void *stream,
                                            minw_net **out) {
    if (!d || !out || max_batch <= 0) return MINW_EINVAL;
    *out = nullptr;
    if (d->bits_a < 1 || d->bits_a > 3 || d->bits_w < 1 || d->bits_w > 3 || d->num_classes <= 0 ||
        d->image_hw < 32 || d->image_hw % 32 != 0)
        return MINW_EINVAL;
    if (!d->stem_w || !d->stem_scale || !d->stem_shift || !d->fc_w || !d->fc_scale || !d->fc_shift)
        return MINW_EINVAL;
    for (int i = 0; i < 16; ++i)
        if (!d->conv_w[i] || !d->conv_scale[i] || !d->conv_shift[i]) return MINW_EINVAL;
    for (int i = 0; i < 3; ++i)
        if (!d->down_w[i] || !d->down_scale[i] || !d->down_shift[i]) return MINW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    minw_net *n = new minw_net();
    n->kind = 1;
    n->max_batch = max_batch;
    ResNetPlan *R = new ResNetPlan();
    n->res = R;
    auto fail = [&](minw_status st) {
        cudaStreamSynchronize(s);
        for (void *p : n->owned) cudaFree(p);
        delete R;
        delete n;
        return st;
    };
    R->hw = d->image_hw;
    R->classes = d->num_classes;
    R->bits_a = d->bits_a;
    R->bits_w = d->bits_w;
    R->qa.bits = d->bits_a;
    R->qa.scale = 1.0f;
    for (int i = 0; i < 3; ++i) R->qa.thr[i] = d->thr_a[i];
    minw_quant qw{};
    qw.bits = d->bits_w;
    qw.scale = 1.0f;
    for (int i = 0; i < 3; ++i) qw.thr[i] = d->thr_w[i];
    if (!valid_quant(&R->qa) || !valid_quant(&qw)) return fail(MINW_EINVAL);
    minw_status st;

    // stem: fp32 7x7 / 2 convolution on the fp32 image, fp32 weights
    R->Hs = d->image_hw / 2;
    R->Hp = R->Hs / 2;
    if ((st = copy_owned(n, &R->stem_w, d->stem_w, 64 * 3 * 49, s)) != MINW_OK) return fail(st);
    if ((st = copy_owned(n, &R->stem_scale, d->stem_scale, 64, s)) != MINW_OK) return fail(st);
    if ((st = copy_owned(n, &R->stem_shift, d->stem_shift, 64, s)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &R->stem_thr, 64 * 8)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &R->stem_wt, 64 * 3 * 49)) != MINW_OK) return fail(st);
    if ((st = launch_first_weights(R->stem_w, 64, 3 * 49, 0, QParams{}, nullptr, R->stem_wt, s)) != MINW_OK)
        return fail(st);
    if ((st = launch_thresholds_f32(R->stem_scale, R->stem_shift, 64, to_qparams(&R->qa), R->stem_thr, s)) != MINW_OK)
        return fail(st);

    // residual stages: widths 64-128-256-512, two blocks each, stride 2 + 1x1 / 2 shortcut entering stages 2-4
    const int widths[4] = {64, 128, 256, 512};
    int c_in = 64, hcur = R->Hp;
    size_t ws = 0;
    for (int b = 0; b < 8; ++b) {
        const int stage = b / 2, first = (b % 2) == 0;
        ResBlock &bk = R->blocks[b];
        const int O = widths[stage];
        const int stride = (stage > 0 && first) ? 2 : 1;
        const int hout = (hcur + 2 - 3) / stride + 1;
        bk.c1 = ResConv{c_in, hcur, hcur, O, 3, stride, 1, hout, hout};
        bk.c2 = ResConv{O, hout, hout, O, 3, 1, 1, hout, hout};
        bk.down = stage > 0 && first;
        if (bk.down) bk.d = ResConv{c_in, hcur, hcur, O, 1, 2, 0, hout, hout};
        struct Src { ResConv *c; const float *w, *wsc, *sc, *sh; bool thr; };
        Src srcs[3] = {{&bk.c1, d->conv_w[2 * b], d->conv_wscale[2 * b], d->conv_scale[2 * b], d->conv_shift[2 * b], true},
                       {&bk.c2, d->conv_w[2 * b + 1], d->conv_wscale[2 * b + 1], d->conv_scale[2 * b + 1],
                        d->conv_shift[2 * b + 1], false},
                       {bk.down ? &bk.d : nullptr, bk.down ? d->down_w[stage - 1] : nullptr,
                        bk.down ? d->down_wscale[stage - 1] : nullptr, bk.down ? d->down_scale[stage - 1] : nullptr,
                        bk.down ? d->down_shift[stage - 1] : nullptr, false}};
        for (Src &x : srcs) {
            if (!x.c) continue;
            ResConv &c = *x.c;
            if ((st = alloc_owned(n, &c.wcodes, (size_t)c.O * c.k * c.k * c.C)) != MINW_OK) return fail(st);
            st = e2m1_channels(c.C) ? minw_pack_weight_codes_e2m1(x.w, c.O, c.C, c.k, c.k, &qw, x.wsc, c.wcodes, stream)
                                    : minw_pack_weight_codes(x.w, c.O, c.C, c.k, c.k, &qw, x.wsc, c.wcodes, stream);
            if (st != MINW_OK) return fail(st);
            if ((st = copy_owned(n, &c.scale, x.sc, c.O, s)) != MINW_OK) return fail(st);
            if ((st = copy_owned(n, &c.shift, x.sh, c.O, s)) != MINW_OK) return fail(st);
            if (x.thr) {
                if ((st = alloc_owned(n, &c.thr, (size_t)c.O * num_levels(d->bits_a))) != MINW_OK) return fail(st);
                if ((st = launch_thresholds(c.scale, c.shift, c.O, to_qparams(&R->qa), c.thr, s)) != MINW_OK)
                    return fail(st);
            }
            ConvArgs a = conv_args(c, max_batch);
            a.act8 = c.wcodes;                       // shape check only
            a.quant_out = x.thr;
            if (x.thr) a.qo = to_qparams(&R->qa);
            if (!conv_tc_supported(a)) return fail(MINW_EUNSUPPORTED);
            const size_t w = conv_tc_workspace_bytes(a);
            if (w > ws) ws = w;
        }
        c_in = O;
        hcur = hout;
    }
    if (c_in != 512) return fail(MINW_EINVAL);
    // head: transposed fp32 classifier weights
    if ((st = alloc_owned(n, &R->fc_wt, (size_t)512 * d->num_classes)) != MINW_OK) return fail(st);
    transpose_kernel<<<256, 256, 0, s>>>(d->fc_w, d->num_classes, 512, R->fc_wt);
    if ((st = copy_owned(n, &R->fc_scale, d->fc_scale, d->num_classes, s)) != MINW_OK) return fail(st);
    if ((st = copy_owned(n, &R->fc_shift, d->fc_shift, d->num_classes, s)) != MINW_OK) return fail(st);

    // activation buffers: stem codes, block input / output / middle codes, fp32 shortcut
    const size_t Bm = (size_t)max_batch;
    const size_t stem_codes = Bm * R->Hs * R->Hs * 64;
    size_t act_codes = 0, down_f32 = 0;
    for (const ResBlock &bk : R->blocks) {
        act_codes = std::max(act_codes, Bm * bk.c1.H * bk.c1.W * bk.c1.C);
        act_codes = std::max(act_codes, Bm * bk.c1.Ho * bk.c1.Wo * bk.c1.O);
        if (bk.down) down_f32 = std::max(down_f32, Bm * bk.d.Ho * bk.d.Wo * bk.d.O);
    }
    if ((st = alloc_owned(n, &R->S, stem_codes)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &R->X, act_codes)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &R->Y, act_codes)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &R->V, act_codes)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &R->D, down_f32)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &R->pooled, Bm * 512)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &R->ythr, 8)) != MINW_OK) return fail(st);
    if ((st = launch_ythresholds(to_qparams(&R->qa), R->ythr, s)) != MINW_OK) return fail(st);
    if (ws) {
        uint8_t *w = nullptr;
        if ((st = alloc_owned(n, &w, ws)) != MINW_OK) return fail(st);
        n->ws = w;
        n->ws_bytes = ws;
    }
    n->x_elems = Bm * 3 * d->image_hw * d->image_hw;
    n->logit_elems = Bm * d->num_classes;
    if ((st = alloc_owned(n, &n->x_stage, n->x_elems)) != MINW_OK) return fail(st);
    if ((st = alloc_owned(n, &n->logits_stage, n->logit_elems)) != MINW_OK) return fail(st);
    if (cudaStreamSynchronize(s) != cudaSuccess || cudaGetLastError() != cudaSuccess) return fail(MINW_ECUDA);
    *out = n;
    return MINW_OK;
}

minw_status resnet_forward(minw_net *net, const float *x, int B, float *logits, cudaStream_t s) {
    ResNetPlan *R = net->res;
    int ev = 0;
    auto mark = [&]() -> minw_status {
        ++ev;
        if (net->timing && cudaEventRecord(net->events[ev], s) != cudaSuccess) return MINW_ECUDA;
        return MINW_OK;
    };
    if (net->timing && cudaEventRecord(net->events[0], s) != cudaSuccess) return MINW_ECUDA;
    minw_status st;
    // stem convolution -> level codes [B][Hs][Hs][64]
    {
        FirstArgs a{};
        a.x = x; a.w = R->stem_w; a.quant_w = 0;
        a.B = B; a.C = 3; a.H = R->hw; a.W = R->hw; a.O = 64; a.kh = 7; a.kw = 7; a.stride = 2; a.pad = 3;
        a.Ho = R->Hs; a.Wo = R->Hs;
        a.scale = R->stem_scale; a.shift = R->stem_shift;
        a.quant_out = 1; a.qo = to_qparams(&R->qa);
        a.codes_out = R->S;
        a.thr = R->stem_thr;
        a.wt = R->stem_wt;
        if ((st = launch_conv_first(a, s)) != MINW_OK) return st;
        if ((st = mark()) != MINW_OK) return st;
    }
    // stem pool on levels -> X [B][Hp][Hp][64]
    {
        const long long items = (long long)B * R->Hp * R->Hp * 4;
        if (items >= (1ll << 31)) return MINW_EUNSUPPORTED;
        const int sms = num_sms() > 0 ? num_sms() : 152;
        long long g = (items + 255) / 256;
        if (g > sms * 8LL) g = sms * 8LL;
        launch_pdl(pool_levels_kernel, dim3((unsigned)g), dim3(256), 0, s, (const uint8_t *)R->S, B, R->Hs, R->Hs, 64,
                   (const float *)R->stem_scale, R->X, R->Hp, R->Hp);
        if (cudaGetLastError() != cudaSuccess) return MINW_ECUDA;
        if ((st = mark()) != MINW_OK) return st;
    }
    uint8_t *X = R->X, *Y = R->Y;
    const float unit = R->bits_a == 3 ? 0.25f : 1.0f;
    for (const ResBlock &bk : R->blocks) {
        for (int which = 0; which < 3; ++which) {
            if (which == 1 && !bk.down) continue;
            if ((st = launch_conv_tc(block_conv(net, bk, which, B, X, Y), s)) != MINW_OK) return st;
            if ((st = mark()) != MINW_OK) return st;
        }
        uint8_t *t = X; X = Y; Y = t;
    }
    // head
    {
        const ResConv &last = R->blocks[7].c2;
        const int HW = last.Ho * last.Wo;
        launch_pdl(avgpool_levels_kernel, dim3((unsigned)((B * 512 + 255) / 256)), dim3(256), 0, s, (const uint8_t *)X,
                   B, HW, 512, unit, e2m1_channels(512), R->pooled);
        const size_t smem = sizeof(float) * HEAD_IMGS * 512;
        const dim3 grid((unsigned)((R->classes + HEAD_CLS - 1) / HEAD_CLS), (unsigned)((B + HEAD_IMGS - 1) / HEAD_IMGS));
        launch_pdl(fc_head_kernel, grid, dim3(HEAD_CLS, HEAD_IMGS), smem, s, (const float *)R->pooled, B, 512,
                   (const float *)R->fc_wt, R->classes, (const float *)R->fc_scale, (const float *)R->fc_shift, logits);
        if (cudaGetLastError() != cudaSuccess) return MINW_ECUDA;
        if ((st = mark()) != MINW_OK) return st;
    }
    return MINW_OK;
}
