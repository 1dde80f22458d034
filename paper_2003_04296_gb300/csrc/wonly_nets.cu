// wonly_nets.cu -- the weight-only MINW-Net networks of Table III: the residual
// network below, and the DenseNet-BC (DenseNet-100) after it.
//
// The residual network is a CIFAR
// ResNet-(6n+2) (ResNet-110 for n = 18) whose block convolutions use N-bit
// weights (the SHIFT ADDER rows: full-precision activations times level
// weights, Sec. IV) and whose first and last layers keep fp32 weights
// (Sec. III-E).  The paper leaves the block wiring open; the reading built:
//   stem : fp32 3x3 conv 3 -> 16 (one fmaf chain per output, as the first
//          layer of the ConvNet) -> BN -> HardTanh
//   block: y1 = BN1(conv1(x)); h = HardTanh(y1); y2 = BN2(conv2(h));
//          out = HardTanh(y2 + s), s = x, or s = BN_d(conv_d(x)) for the
//          1x1 / 2 shortcut entering stages 2 and 3 (one fp32 add)
//   head : global average pool (one fp32 sum in pixel order, one division)
//          -> fp32 fully connected layer -> BN -> logits
// Stages of n blocks each, 16, 32 and 64 channels, stride 2 entering stages 2
// and 3.  Every block convolution runs on the bf16 tensor cores
// (conv2d_bf16): its input is the bf16 rounding of the fp32 activation, its
// weights the exact levels as bf16, both held with their channels padded to
// a multiple of 64 (zeros add nothing to a product), and its output, the fp32
// BN map, goes through the epilogue of conv2d_bf16_hardtanh: for conv1,
// HardTanh of it rounded to bf16 straight into conv2's padded NHWC input; for
// conv2, the shortcut added (one fp32 add), HardTanh, and the result written
// both as the next block's padded bf16 NHWC input and as the fp32 NCHW copy a
// later shortcut reads.  The 1x1 / 2 shortcut convolution writes its fp32
// BN map (NCHW).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <vector>

#include "net.cuh"

using namespace minw;
using namespace minw_host;

namespace {

// v = HardTanh(y + s) (s nullable: v = HardTanh(y)) over NCHW fp32 [B][C][HW]
// (the fp32 operations of the oracle: one add, then the two clamps), written
// as fp32 NCHW to z (nullable) and as bf16 NHWC rows of Cp channels to zb,
// channels zo .. zo + C (the rest of each row is not written).
// Block (32, 8): 32 channels x 32 pixels of one image through shared memory;
// each thread's loads issue before its first store.
__global__ void __launch_bounds__(256) wres_post_kernel(const float *__restrict__ y, const float *__restrict__ s,
                                                        int C, int Cp, int zo, int HW, float *__restrict__ z,
                                                        uint16_t *__restrict__ zb) {
    __shared__ float tile[32][33];
    const int b = blockIdx.z, c0 = blockIdx.y * 32, p0 = blockIdx.x * 32;
    float yv[4], sv[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int c = c0 + threadIdx.y + 8 * k, p = p0 + threadIdx.x;
        yv[k] = sv[k] = 0.0f;
        if (c < C && p < HW) {
            const int64_t idx = ((int64_t)b * C + c) * HW + p;
            yv[k] = __ldg(y + idx);
            if (s != nullptr) sv[k] = __ldg(s + idx);
        }
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int c = c0 + threadIdx.y + 8 * k, p = p0 + threadIdx.x;
        float v = 0.0f;
        if (c < C && p < HW) {
            v = s != nullptr ? yv[k] + sv[k] : yv[k];
            if (v > 1.0f) v = 1.0f;
            if (v < -1.0f) v = -1.0f;
            if (z != nullptr) z[((int64_t)b * C + c) * HW + p] = v;
        }
        tile[threadIdx.y + 8 * k][threadIdx.x] = v;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int p = p0 + threadIdx.y + 8 * k, c = c0 + threadIdx.x;
        if (c < C && p < HW)
            zb[((int64_t)b * HW + p) * Cp + zo + c] =
                __bfloat16_as_ushort(__float2bfloat16_rn(tile[threadIdx.x][threadIdx.y + 8 * k]));
    }
}

// Head, first part: global average pool of fp32 NCHW [B][C][HW] (one fp32 sum
// over the pixels in order, one division); thread = (image, channel).
__global__ void wres_avgpool_kernel(const float *__restrict__ x, int B, int C, int HW, float *__restrict__ pooled) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= B * C) return;
    const float *src = x + (int64_t)i * HW;
    float s = 0.0f;
    for (int p = 0; p < HW; ++p) s += __ldg(src + p);
    pooled[i] = s / (float)HW;
}

// Head, second part: the fp32 fully connected layer (one fmaf chain over the
// features in order, weights transposed to [C][classes]) and BN (fmaf); one
// output per thread, the CTA's images' features in shared memory.
constexpr int WHEAD_IMGS = 8, WHEAD_CLS = 32;
__global__ void __launch_bounds__(WHEAD_IMGS * WHEAD_CLS) wres_fc_kernel(const float *__restrict__ pooled, int B,
                                                                        int C, const float *__restrict__ wt,
                                                                        int classes, const float *__restrict__ scale,
                                                                        const float *__restrict__ shift,
                                                                        float *__restrict__ logits) {
    extern __shared__ float sp[];                    // [WHEAD_IMGS][C]
    const int b0 = blockIdx.y * WHEAD_IMGS;
    const int nimg = min(WHEAD_IMGS, B - b0);
    const int tid = threadIdx.y * WHEAD_CLS + threadIdx.x;
    for (int i = tid; i < WHEAD_IMGS * C; i += WHEAD_IMGS * WHEAD_CLS)
        sp[i] = i < nimg * C ? pooled[(int64_t)b0 * C + i] : 0.0f;
    __syncthreads();
    const int o = blockIdx.x * WHEAD_CLS + threadIdx.x, im = threadIdx.y;
    if (o >= classes || im >= nimg) return;
    const float *xs = sp + im * C;
    float acc = 0.0f;
    for (int k = 0; k < C; ++k) acc = fmaf(xs[k], __ldg(wt + (int64_t)k * classes + o), acc);
    acc = acc + 0.0f;                                 // the oracle's sum without bias
    logits[(int64_t)(b0 + im) * classes + o] = fmaf(acc, __ldg(scale + o), __ldg(shift + o));
}

__global__ void wres_transpose_kernel(const float *__restrict__ in, int rows, int cols, float *__restrict__ out) {
    const int64_t n = (int64_t)rows * cols;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int r = (int)(i / cols), c = (int)(i - (int64_t)r * cols);
        out[(int64_t)c * rows + r] = in[i];
    }
}

// DenseNet transition pool: out = bf16(((v00 + v01) + v10) + v11) * 1/4) with
// v = HardTanh(y) over 2x2 windows of NCHW fp32 [B][C][H][W], written as rows
// of zs channels of bf16 NHWC [B][H/2][W/2] (channels 0 .. C).  Block (32, 8):
// 32 channels x 32 pooled pixels of one image through shared memory.
__global__ void __launch_bounds__(256) wdense_pool_kernel(const float *__restrict__ y, int C, int H, int W, int zs,
                                                          uint16_t *__restrict__ zb) {
    __shared__ float tile[32][33];
    const int Ho = H / 2, Wo = W / 2, HWo = Ho * Wo;
    const int b = blockIdx.z, c0 = blockIdx.y * 32, p0 = blockIdx.x * 32;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int c = c0 + threadIdx.y + 8 * k, p = p0 + threadIdx.x;
        float o = 0.0f;
        if (c < C && p < HWo) {
            const int yo = p / Wo, xo = p - yo * Wo;
            const float *src = y + (((int64_t)b * C + c) * H + 2 * yo) * W + 2 * xo;
            float v[4] = {__ldg(src), __ldg(src + 1), __ldg(src + W), __ldg(src + W + 1)};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if (v[j] > 1.0f) v[j] = 1.0f;
                if (v[j] < -1.0f) v[j] = -1.0f;
            }
            o = ((v[0] + v[1]) + v[2]) + v[3];
            o = o * 0.25f;
        }
        tile[threadIdx.y + 8 * k][threadIdx.x] = o;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int p = p0 + threadIdx.y + 8 * k, c = c0 + threadIdx.x;
        if (c < C && p < HWo)
            zb[((int64_t)b * HWo + p) * zs + c] =
                __bfloat16_as_ushort(__float2bfloat16_rn(tile[threadIdx.x][threadIdx.y + 8 * k]));
    }
}

// DenseNet head, first part: global average pool of bf16 NHWC features (rows
// of zs channels, channels 0 .. C): one fp32 sum over the pixels in order, one
// division; thread = (image, channel).
__global__ void wdense_avgpool_kernel(const uint16_t *__restrict__ F, int B, int C, int HW, int zs,
                                      float *__restrict__ pooled) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= B * C) return;
    const int b = i / C, c = i - b * C;
    const uint16_t *src = F + (int64_t)b * HW * zs + c;
    float s = 0.0f;
    for (int p = 0; p < HW; ++p) s += __uint_as_float((uint32_t)__ldg(src + (int64_t)p * zs) << 16);
    pooled[i] = s / (float)HW;
}

struct WConv {
    int C = 0, Cp = 0, O = 0, k = 0, stride = 1, pad = 0, H = 0, W = 0, Ho = 0, Wo = 0;
    uint16_t *wb = nullptr;                // bf16 levels [O][k][k][Cp]
    float *scale = nullptr, *shift = nullptr;
};

struct WBlock {
    WConv c1, c2, d;
    bool down = false;
};

int pad64(int c) { return (c + 63) / 64 * 64; }

}  // namespace

struct WResPlan {
    int n = 0, hw = 0, classes = 0, bits_w = 0;
    float *stem_w = nullptr, *stem_wt = nullptr, *stem_scale = nullptr, *stem_shift = nullptr;
    std::vector<WBlock> blocks;
    float *fc_wt = nullptr, *fc_scale = nullptr, *fc_shift = nullptr;
    float *A[2] = {nullptr, nullptr};      // fp32 NCHW block activations (ping-pong)
    // padded bf16 NHWC inputs of the convolutions, per stage (the channels past a stage's
    // count stay zero from creation on): block outputs (ping-pong) and HardTanh(BN1(conv1))
    uint16_t *AB[3][2] = {{nullptr, nullptr}, {nullptr, nullptr}, {nullptr, nullptr}};
    uint16_t *HB[3] = {nullptr, nullptr, nullptr};
    float *Y1 = nullptr, *S = nullptr;     // fp32 NCHW outputs of the stem and of the shortcut convolutions
    float *pooled = nullptr;
    std::vector<float *> keep;             // with keep_activations: the stem's and every block's fp32 output
    std::vector<size_t> keep_elems;        // ... their sizes at max_batch
    int keep_B = 0;                        // batch of the most recent forward
};

template <typename T>
static minw_status walloc(minw_net *n, T **p, size_t count) {
    void *q = nullptr;
    if (cudaMalloc(&q, count * sizeof(T) + 256) != cudaSuccess) return MINW_ECUDA;
    n->owned.push_back(q);
    *p = reinterpret_cast<T *>(q);
    return MINW_OK;
}

static minw_status wcopy(minw_net *n, float **dst, const float *src, size_t count, cudaStream_t s) {
    minw_status st = walloc(n, dst, count);
    if (st != MINW_OK) return st;
    return cudaMemcpyAsync(*dst, src, count * sizeof(float), cudaMemcpyDeviceToDevice, s) == cudaSuccess ? MINW_OK
                                                                                                         : MINW_ECUDA;
}

// The fused pass into rows of zs channels at offset zo (zs = the padded channel
// count by default: the block networks' own buffers).
static minw_status post(const float *y, const float *s, int B, int C, int HW, float *z, uint16_t *zb, cudaStream_t st,
                        int zs = 0, int zo = 0) {
    if (zs == 0) zs = pad64(C);
    const dim3 grid((unsigned)((HW + 31) / 32), (unsigned)((C + 31) / 32), (unsigned)B);
    wres_post_kernel<<<grid, dim3(32, 8), 0, st>>>(y, s, C, zs, zo, HW, z, zb);
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

// A weight-only convolution's plan: channels C (padded to Cp = pad64(C)), O
// outputs, k x k, stride, square H; weights quantized with qw into padded bf16
// levels [O][k][k][Cp], BN maps copied.
static minw_status make_wconv(minw_net *n, const minw_quant &qw, WConv &c, int C, int O, int k, int stride, int H,
                              const float *w, const float *ws, const float *sc, const float *sh, cudaStream_t s) {
    c.C = C; c.Cp = pad64(C); c.O = O; c.k = k; c.stride = stride; c.pad = k / 2; c.H = H; c.W = H;
    c.Ho = (H + 2 * c.pad - k) / stride + 1;
    c.Wo = c.Ho;
    minw_status e;
    if ((e = walloc(n, &c.wb, (size_t)O * k * k * c.Cp)) != MINW_OK) return e;
    if ((e = minw_pack_weight_bf16_pad(w, O, C, k, k, c.Cp, &qw, ws, c.wb, s)) != MINW_OK) return e;
    if ((e = wcopy(n, &c.scale, sc, O, s)) != MINW_OK) return e;
    return wcopy(n, &c.shift, sh, O, s);
}

// ... with the fused HardTanh + bf16 NHWC epilogue: input rows of ldc
// elements (0: the padded channels), output rows of ld elements at off.
static minw_status wconv_ht(const WConv &c, const uint16_t *in, int ldc, int B, uint16_t *out, int ld, int off,
                            cudaStream_t s, int bits_w) {
    return conv2d_bf16_hardtanh(in, B, c.Cp, c.H, c.W, ldc, c.wb, c.O, c.k, c.k, bits_w, c.stride, c.pad, c.scale,
                                c.shift, out, ld, off, s);
}

static minw_status wconv(const WConv &c, const uint16_t *in, int B, float *y, cudaStream_t s, int bits_w) {
    return conv2d_bf16(in, B, c.Cp, c.H, c.W, c.wb, c.O, c.k, c.k, bits_w, c.stride, c.pad, 0, c.scale, c.shift, y,
                       nullptr, 0, nullptr, s);
}

void wresnet_free(minw_net *net) {
    delete net->wres;
    net->wres = nullptr;
}

// Ops timed by minw_net_layer_times, in forward order: the stem, its HardTanh
// pass, per block conv1 (its HardTanh fused), [the shortcut], conv2 (the
// shortcut add and HardTanh fused), the head.
int32_t wresnet_ops(const minw_net *net) {
    int ops = 3;
    for (const WBlock &bk : net->wres->blocks) ops += bk.down ? 3 : 2;
    return ops;
}

void wresnet_variants(const minw_net *net, int32_t *v) {
    const int n = wresnet_ops(net);
    int k = 0;
    v[k++] = 0;
    v[k++] = 0;
    for (const WBlock &bk : net->wres->blocks) {
        v[k++] = MINW_VARIANT_TC;
        if (bk.down) v[k++] = MINW_VARIANT_TC;
        v[k++] = MINW_VARIANT_TC;
    }
    while (k < n) v[k++] = 0;
}

int32_t wresnet_kernels(const minw_net *net) {
    return wresnet_ops(net) + 1;                       // the head is two kernels
}

minw_status wresnet_forward(minw_net *net, const float *x, int B, float *logits, cudaStream_t s) {
    WResPlan *R = net->wres;
    int ev = 0;
    auto mark = [&]() -> minw_status {
        ++ev;
        if (net->timing && cudaEventRecord(net->events[ev], s) != cudaSuccess) return MINW_ECUDA;
        return MINW_OK;
    };
    if (net->timing && cudaEventRecord(net->events[0], s) != cudaSuccess) return MINW_ECUDA;
    minw_status st;
    const int hw = R->hw;
    {
        FirstArgs a{};
        a.x = x; a.w = R->stem_w; a.quant_w = 0;
        a.B = B; a.C = 3; a.H = hw; a.W = hw; a.O = 16; a.kh = 3; a.kw = 3; a.stride = 1; a.pad = 1;
        a.Ho = hw; a.Wo = hw;
        a.scale = R->stem_scale; a.shift = R->stem_shift;
        a.quant_out = 0;
        a.y_out = R->Y1;
        a.wt = R->stem_wt;
        if ((st = launch_conv_first(a, s)) != MINW_OK) return st;
        if ((st = mark()) != MINW_OK) return st;
        float *a0 = R->keep.empty() ? R->A[0] : R->keep[0];
        if ((st = post(R->Y1, nullptr, B, 16, hw * hw, a0, R->AB[0][1], s)) != MINW_OK) return st;
        if ((st = mark()) != MINW_OK) return st;
    }
    int cur = 0, bi = 0;
    const float *acur = R->keep.empty() ? R->A[0] : R->keep[0];    // this block's fp32 input (its identity shortcut)
    const uint16_t *xin = R->AB[0][1];                               // ... and its bf16 input
    for (const WBlock &bk : R->blocks) {
        float *anext = R->keep.empty() ? R->A[cur ^ 1] : R->keep[bi + 1];
        const int stg = bi / R->n, j = bi - stg * R->n;
        uint16_t *xout = R->AB[stg][j & 1];
        if ((st = wconv_ht(bk.c1, xin, 0, B, R->HB[stg], pad64(bk.c1.O), 0, s, R->bits_w)) != MINW_OK) return st;
        if ((st = mark()) != MINW_OK) return st;
        const float *sc = acur;
        if (bk.down) {
            if ((st = wconv(bk.d, xin, B, R->S, s, R->bits_w)) != MINW_OK) return st;
            if ((st = mark()) != MINW_OK) return st;
            sc = R->S;
        }
        if ((st = conv2d_bf16_hardtanh(R->HB[stg], B, bk.c2.Cp, bk.c2.H, bk.c2.W, 0, bk.c2.wb, bk.c2.O, 3, 3,
                                       R->bits_w, 1, 1, bk.c2.scale, bk.c2.shift, xout, pad64(bk.c2.O), 0, s, sc,
                                       anext)) != MINW_OK)
            return st;
        if ((st = mark()) != MINW_OK) return st;
        cur ^= 1;
        ++bi;
        acur = anext;
        xin = xout;
    }
    R->keep_B = B;
    {
        const WConv &last = R->blocks.back().c2;
        const int HW = last.Ho * last.Wo, C = last.O;
        wres_avgpool_kernel<<<(unsigned)((B * C + 255) / 256), 256, 0, s>>>(acur, B, C, HW, R->pooled);
        const dim3 grid((unsigned)((R->classes + WHEAD_CLS - 1) / WHEAD_CLS),
                        (unsigned)((B + WHEAD_IMGS - 1) / WHEAD_IMGS));
        wres_fc_kernel<<<grid, dim3(WHEAD_CLS, WHEAD_IMGS), sizeof(float) * WHEAD_IMGS * C, s>>>(
            R->pooled, B, C, R->fc_wt, R->classes, R->fc_scale, R->fc_shift, logits);
        if (cudaGetLastError() != cudaSuccess) return MINW_ECUDA;
        if ((st = mark()) != MINW_OK) return st;
    }
    return MINW_OK;
}

extern "C" minw_status minw_wresnet_create(const minw_wresnet_desc *d, int32_t max_batch, void *stream,
                                           minw_net **out) {
    if (!d || !out || max_batch <= 0) return MINW_EINVAL;
    *out = nullptr;
    if (d->n < 1 || d->n > MINW_WRESNET_MAX_N || d->bits_w < 1 || d->bits_w > 3 || d->num_classes <= 0 ||
        d->image_hw < 8 || d->image_hw % 4 != 0)
        return MINW_EINVAL;
    if (!d->stem_w || !d->stem_scale || !d->stem_shift || !d->fc_w || !d->fc_scale || !d->fc_shift)
        return MINW_EINVAL;
    minw_quant qw{};
    qw.bits = d->bits_w;
    qw.scale = 1.0f;
    for (int i = 0; i < 3; ++i) qw.thr[i] = d->thr_w[i];
    if (!valid_quant(&qw)) return MINW_EINVAL;
    const int nb = 3 * d->n;
    for (int b = 0; b < nb; ++b)
        if (!d->c1_w[b] || !d->c1_scale[b] || !d->c1_shift[b] || !d->c2_w[b] || !d->c2_scale[b] || !d->c2_shift[b])
            return MINW_EINVAL;
    for (int i = 0; i < 2; ++i)
        if (!d->down_w[i] || !d->down_scale[i] || !d->down_shift[i]) return MINW_EINVAL;
    if ((long long)max_batch * 64 * d->image_hw * d->image_hw >= (1ll << 31)) return MINW_EUNSUPPORTED;
    cudaStream_t s = (cudaStream_t)stream;
    minw_net *n = new minw_net();
    n->kind = 2;
    n->max_batch = max_batch;
    n->wres = new WResPlan();
    WResPlan *R = n->wres;
    R->n = d->n; R->hw = d->image_hw; R->classes = d->num_classes; R->bits_w = d->bits_w;
    auto fail = [&](minw_status st) {
        cudaStreamSynchronize(s);
        minw_net_destroy(n);
        return st;
    };
    minw_status st;
    // stem: fp32 weights [16][3][3][3], prepared as [27][16]
    if ((st = wcopy(n, &R->stem_w, d->stem_w, 16 * 27, s)) != MINW_OK) return fail(st);
    if ((st = wcopy(n, &R->stem_scale, d->stem_scale, 16, s)) != MINW_OK) return fail(st);
    if ((st = wcopy(n, &R->stem_shift, d->stem_shift, 16, s)) != MINW_OK) return fail(st);
    if ((st = walloc(n, &R->stem_wt, 16 * 27)) != MINW_OK) return fail(st);
    if ((st = launch_first_weights(R->stem_w, 16, 27, 0, QParams{}, nullptr, R->stem_wt, s)) != MINW_OK)
        return fail(st);
    // blocks
    auto make_conv = [&](WConv &c, int C, int O, int k, int stride, int H, const float *w, const float *ws,
                         const float *sc, const float *sh) -> minw_status {
        return make_wconv(n, qw, c, C, O, k, stride, H, w, ws, sc, sh, s);
    };
    int c_in = 16, size = d->image_hw, bi = 0;
    const int widths[3] = {16, 32, 64};
    for (int stage = 0; stage < 3; ++stage) {
        for (int j = 0; j < d->n; ++j, ++bi) {
            WBlock bk;
            const int width = widths[stage];
            const int stride = (stage > 0 && j == 0) ? 2 : 1;
            if ((st = make_conv(bk.c1, c_in, width, 3, stride, size, d->c1_w[bi], d->c1_wscale[bi], d->c1_scale[bi],
                                d->c1_shift[bi])) != MINW_OK)
                return fail(st);
            const int so = bk.c1.Ho;
            if ((st = make_conv(bk.c2, width, width, 3, 1, so, d->c2_w[bi], d->c2_wscale[bi], d->c2_scale[bi],
                                d->c2_shift[bi])) != MINW_OK)
                return fail(st);
            if (stride == 2) {
                bk.down = true;
                if ((st = make_conv(bk.d, c_in, width, 1, 2, size, d->down_w[stage - 1], d->down_wscale[stage - 1],
                                    d->down_scale[stage - 1], d->down_shift[stage - 1])) != MINW_OK)
                    return fail(st);
            }
            R->blocks.push_back(bk);
            c_in = width;
            size = so;
        }
    }
    // head: fp32 weights [classes][64] transposed to [64][classes]
    {
        float *fc_w = nullptr;
        if ((st = wcopy(n, &fc_w, d->fc_w, (size_t)d->num_classes * 64, s)) != MINW_OK) return fail(st);
        if ((st = walloc(n, &R->fc_wt, (size_t)d->num_classes * 64)) != MINW_OK) return fail(st);
        wres_transpose_kernel<<<64, 256, 0, s>>>(fc_w, d->num_classes, 64, R->fc_wt);
        if ((st = wcopy(n, &R->fc_scale, d->fc_scale, d->num_classes, s)) != MINW_OK) return fail(st);
        if ((st = wcopy(n, &R->fc_shift, d->fc_shift, d->num_classes, s)) != MINW_OK) return fail(st);
        if ((st = walloc(n, &R->pooled, (size_t)max_batch * 64)) != MINW_OK) return fail(st);
    }
    // activations: the stage-1 sizes are the largest (16 channels, 64 padded, at hw x hw)
    const size_t px = (size_t)max_batch * d->image_hw * d->image_hw;
    for (int i = 0; i < 2; ++i)
        if ((st = walloc(n, &R->A[i], px * 16)) != MINW_OK) return fail(st);
    for (int stg = 0; stg < 3; ++stg) {
        const size_t e = px / ((size_t)1 << (2 * stg)) * 64;      // the stage's pixels x 64 padded channels
        for (int i = 0; i < 3; ++i) {
            uint16_t *b = nullptr;
            if ((st = walloc(n, &b, e)) != MINW_OK) return fail(st);
            if (cudaMemsetAsync(b, 0, e * sizeof(uint16_t), s) != cudaSuccess) return fail(MINW_ECUDA);
            if (i < 2) R->AB[stg][i] = b; else R->HB[stg] = b;
        }
    }
    if ((st = walloc(n, &R->Y1, px * 16)) != MINW_OK ||
        (st = walloc(n, &R->S, px * 16)) != MINW_OK)
        return fail(st);
    if (d->keep_activations) {
        size_t e = px * 16;                               // the stem's output
        R->keep_elems.push_back(e);
        for (const WBlock &bk : R->blocks) R->keep_elems.push_back((size_t)max_batch * bk.c2.O * bk.c2.Ho * bk.c2.Wo);
        for (size_t k : R->keep_elems) {
            float *q = nullptr;
            if ((st = walloc(n, &q, k)) != MINW_OK) return fail(st);
            R->keep.push_back(q);
        }
    }
    n->x_elems = px * 3;
    n->logit_elems = (size_t)max_batch * d->num_classes;
    if ((st = walloc(n, &n->x_stage, n->x_elems)) != MINW_OK ||
        (st = walloc(n, &n->logits_stage, n->logit_elems)) != MINW_OK)
        return fail(st);
    if (cudaStreamSynchronize(s) != cudaSuccess || cudaGetLastError() != cudaSuccess) return fail(MINW_ECUDA);
    *out = n;
    return MINW_OK;
}

extern "C" minw_status minw_wresnet_activation(const minw_net *net, int32_t index, float *dst, size_t count,
                                               void *stream) {
    if (!net || net->kind != 2 || !net->wres || !dst) return MINW_EINVAL;
    const WResPlan *R = net->wres;
    if (R->keep.empty() || index < 0 || index >= (int32_t)R->keep.size() || R->keep_B <= 0) return MINW_EINVAL;
    const size_t elems = R->keep_elems[(size_t)index] / (size_t)net->max_batch * (size_t)R->keep_B;
    if (count < elems) return MINW_EINVAL;
    return cudaMemcpyAsync(dst, R->keep[(size_t)index], elems * sizeof(float), cudaMemcpyDeviceToDevice,
                           (cudaStream_t)stream) == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

// ---------------------------------------------------------------------------
// The weight-only DenseNet-BC of Table III (DenseNet-100: 16 bottleneck
// layers per block, growth 12).  Each block's features live in one bf16 NHWC
// buffer F of pad64(final channels) elements per pixel: the stem (or the
// transition before the block) writes channels 0 .. c_b, layer i appends
// channels c_b + i k .. + k in place, and layer i's 1x1 convolution reads the
// first pad64(c_b + i k) channels of each row through a tensor map whose row
// stride is the buffer's (its weights are zero past c_b + i k, and every
// stale value there is a finite HardTanh output, or the zero the buffer held
// at creation).  No concatenation is ever copied.
// ---------------------------------------------------------------------------

struct WDenseLayer {
    WConv b, c;          // 1x1 to 4k channels, 3x3 to k channels
    int cin = 0;         // channels the layer reads (its output lands there)
};

struct WDensePlan {
    int layers = 0, growth = 0, hw = 0, classes = 0, bits_w = 0;
    float *stem_w = nullptr, *stem_wt = nullptr, *stem_scale = nullptr, *stem_shift = nullptr;
    std::vector<WDenseLayer> lay[3];
    WConv trans[2];
    int cfin[3] = {0, 0, 0};             // each block's final channels
    int row[3] = {0, 0, 0};              // ... and its buffer's elements per pixel, pad64(cfin)
    uint16_t *F[3] = {nullptr, nullptr, nullptr};
    uint16_t *HB = nullptr;              // bf16 NHWC HardTanh(BN(conv 1x1)), pad64(4k) per pixel
    float *Y = nullptr;                  // fp32 NCHW convolution outputs
    float *fc_wt = nullptr, *fc_scale = nullptr, *fc_shift = nullptr, *pooled = nullptr;
    int last_B = 0;                      // batch of the most recent forward
};

void wdense_free(minw_net *net) {
    delete net->wdense;
    net->wdense = nullptr;
}

// Ops timed by minw_net_layer_times, in forward order: the stem, its pass;
// per layer the 1x1 convolution and the 3x3 convolution (each with its
// HardTanh and bf16 output fused); per transition its convolution and its
// pool; the head.
int32_t wdense_ops(const minw_net *net) {
    const WDensePlan *D = net->wdense;
    return 2 + 2 * 3 * D->layers + 2 * 2 + 1;
}

void wdense_variants(const minw_net *net, int32_t *v) {
    const WDensePlan *D = net->wdense;
    int k = 0;
    v[k++] = 0;
    v[k++] = 0;
    for (int b = 0; b < 3; ++b) {
        for (int i = 0; i < D->layers; ++i) {
            v[k++] = MINW_VARIANT_TC;
            v[k++] = MINW_VARIANT_TC;
        }
        if (b < 2) {
            v[k++] = MINW_VARIANT_TC;
            v[k++] = 0;
        }
    }
    v[k++] = 0;
}

int32_t wdense_kernels(const minw_net *net) {
    return wdense_ops(net) + 1;                        // the head is two kernels
}

minw_status wdense_forward(minw_net *net, const float *x, int B, float *logits, cudaStream_t s) {
    WDensePlan *D = net->wdense;
    int ev = 0;
    auto mark = [&]() -> minw_status {
        ++ev;
        if (net->timing && cudaEventRecord(net->events[ev], s) != cudaSuccess) return MINW_ECUDA;
        return MINW_OK;
    };
    if (net->timing && cudaEventRecord(net->events[0], s) != cudaSuccess) return MINW_ECUDA;
    minw_status st;
    const int c0 = 2 * D->growth, k4 = 4 * D->growth;
    {
        FirstArgs a{};
        a.x = x; a.w = D->stem_w; a.quant_w = 0;
        a.B = B; a.C = 3; a.H = D->hw; a.W = D->hw; a.O = c0; a.kh = 3; a.kw = 3; a.stride = 1; a.pad = 1;
        a.Ho = D->hw; a.Wo = D->hw;
        a.scale = D->stem_scale; a.shift = D->stem_shift;
        a.quant_out = 0;
        a.y_out = D->Y;
        a.wt = D->stem_wt;
        if ((st = launch_conv_first(a, s)) != MINW_OK) return st;
        if ((st = mark()) != MINW_OK) return st;
        if ((st = post(D->Y, nullptr, B, c0, D->hw * D->hw, nullptr, D->F[0], s, D->row[0], 0)) != MINW_OK)
            return st;
        if ((st = mark()) != MINW_OK) return st;
    }
    for (int b = 0; b < 3; ++b) {
        const int h = D->hw >> b, HW = h * h;
        for (const WDenseLayer &L : D->lay[b]) {
            if ((st = wconv_ht(L.b, D->F[b], D->row[b], B, D->HB, pad64(k4), 0, s, D->bits_w)) != MINW_OK) return st;
            if ((st = mark()) != MINW_OK) return st;
            if ((st = wconv_ht(L.c, D->HB, 0, B, D->F[b], D->row[b], L.cin, s, D->bits_w)) != MINW_OK) return st;
            if ((st = mark()) != MINW_OK) return st;
        }
        if (b < 2) {
            const WConv &T = D->trans[b];
            if ((st = conv2d_bf16(D->F[b], B, T.Cp, h, h, T.wb, T.O, 1, 1, D->bits_w, 1, 0, 0, T.scale, T.shift,
                                  D->Y, nullptr, 0, nullptr, s, 0, 0.0f, 0.0f, D->row[b])) != MINW_OK)
                return st;
            if ((st = mark()) != MINW_OK) return st;
            const dim3 grid((unsigned)((HW / 4 + 31) / 32), (unsigned)((T.O + 31) / 32), (unsigned)B);
            wdense_pool_kernel<<<grid, dim3(32, 8), 0, s>>>(D->Y, T.O, h, h, D->row[b + 1], D->F[b + 1]);
            if (cudaGetLastError() != cudaSuccess) return MINW_ECUDA;
            if ((st = mark()) != MINW_OK) return st;
        }
    }
    D->last_B = B;
    {
        const int h = D->hw >> 2, C = D->cfin[2];
        wdense_avgpool_kernel<<<(unsigned)((B * C + 255) / 256), 256, 0, s>>>(D->F[2], B, C, h * h, D->row[2],
                                                                              D->pooled);
        const dim3 grid((unsigned)((D->classes + WHEAD_CLS - 1) / WHEAD_CLS),
                        (unsigned)((B + WHEAD_IMGS - 1) / WHEAD_IMGS));
        wres_fc_kernel<<<grid, dim3(WHEAD_CLS, WHEAD_IMGS), sizeof(float) * WHEAD_IMGS * C, s>>>(
            D->pooled, B, C, D->fc_wt, D->classes, D->fc_scale, D->fc_shift, logits);
        if (cudaGetLastError() != cudaSuccess) return MINW_ECUDA;
        if ((st = mark()) != MINW_OK) return st;
    }
    return MINW_OK;
}

extern "C" minw_status minw_wdense_create(const minw_wdense_desc *d, int32_t max_batch, void *stream,
                                          minw_net **out) {
    if (!d || !out || max_batch <= 0) return MINW_EINVAL;
    *out = nullptr;
    if (d->layers < 1 || d->layers > MINW_WDENSE_MAX_LAYERS || d->growth < 1 || d->growth > 64 || d->bits_w < 1 ||
        d->bits_w > 3 || d->num_classes <= 0 || d->image_hw < 8 || d->image_hw % 4 != 0)
        return MINW_EINVAL;
    if (!d->stem_w || !d->stem_scale || !d->stem_shift || !d->fc_w || !d->fc_scale || !d->fc_shift)
        return MINW_EINVAL;
    minw_quant qw{};
    qw.bits = d->bits_w;
    qw.scale = 1.0f;
    for (int i = 0; i < 3; ++i) qw.thr[i] = d->thr_w[i];
    if (!valid_quant(&qw)) return MINW_EINVAL;
    for (int j = 0; j < 3 * d->layers; ++j)
        if (!d->b_w[j] || !d->b_scale[j] || !d->b_shift[j] || !d->c_w[j] || !d->c_scale[j] || !d->c_shift[j])
            return MINW_EINVAL;
    for (int i = 0; i < 2; ++i)
        if (!d->t_w[i] || !d->t_scale[i] || !d->t_shift[i]) return MINW_EINVAL;
    const int k = d->growth, hw = d->image_hw;
    int cfin[3], cstart[3];
    {
        int c = 2 * k;
        for (int b = 0; b < 3; ++b) {
            cstart[b] = c;
            cfin[b] = c + d->layers * k;
            c = cfin[b] / 2;
        }
    }
    // the widest fp32 output (the stem's 2k channels, or a transition's) and bf16 buffer, at max_batch
    size_t y_px = (size_t)2 * k * hw * hw;
    for (int b = 0; b < 2; ++b) y_px = std::max(y_px, (size_t)(cfin[b] / 2) * (hw >> b) * (hw >> b));
    const size_t row_px = (size_t)std::max(pad64(cfin[0]), pad64(4 * k)) * hw * hw;   // block 1's buffer, HB
    if ((long long)max_batch * (long long)std::max(row_px, y_px) >= (1ll << 31)) return MINW_EUNSUPPORTED;
    if (sizeof(float) * WHEAD_IMGS * cfin[2] > 48 * 1024) return MINW_EUNSUPPORTED;   // the head's staged features
    cudaStream_t s = (cudaStream_t)stream;
    minw_net *n = new minw_net();
    n->kind = 3;
    n->max_batch = max_batch;
    n->wdense = new WDensePlan();
    WDensePlan *D = n->wdense;
    D->layers = d->layers; D->growth = k; D->hw = hw; D->classes = d->num_classes; D->bits_w = d->bits_w;
    auto fail = [&](minw_status st) {
        cudaStreamSynchronize(s);
        minw_net_destroy(n);
        return st;
    };
    minw_status st;
    // stem: fp32 weights [2k][3][3][3], prepared as [27][2k]
    const int c0 = 2 * k;
    if ((st = wcopy(n, &D->stem_w, d->stem_w, (size_t)c0 * 27, s)) != MINW_OK) return fail(st);
    if ((st = wcopy(n, &D->stem_scale, d->stem_scale, c0, s)) != MINW_OK) return fail(st);
    if ((st = wcopy(n, &D->stem_shift, d->stem_shift, c0, s)) != MINW_OK) return fail(st);
    if ((st = walloc(n, &D->stem_wt, (size_t)c0 * 27)) != MINW_OK) return fail(st);
    if ((st = launch_first_weights(D->stem_w, c0, 27, 0, QParams{}, nullptr, D->stem_wt, s)) != MINW_OK)
        return fail(st);
    for (int b = 0; b < 3; ++b) {
        const int h = hw >> b;
        for (int i = 0; i < d->layers; ++i) {
            const int j = b * d->layers + i;
            WDenseLayer L;
            L.cin = cstart[b] + i * k;
            if ((st = make_wconv(n, qw, L.b, L.cin, 4 * k, 1, 1, h, d->b_w[j], d->b_wscale[j], d->b_scale[j],
                                 d->b_shift[j], s)) != MINW_OK)
                return fail(st);
            if ((st = make_wconv(n, qw, L.c, 4 * k, k, 3, 1, h, d->c_w[j], d->c_wscale[j], d->c_scale[j],
                                 d->c_shift[j], s)) != MINW_OK)
                return fail(st);
            D->lay[b].push_back(L);
        }
        D->cfin[b] = cfin[b];
        D->row[b] = pad64(cfin[b]);
        if (b < 2 && (st = make_wconv(n, qw, D->trans[b], cfin[b], cfin[b] / 2, 1, 1, h, d->t_w[b], d->t_wscale[b],
                                      d->t_scale[b], d->t_shift[b], s)) != MINW_OK)
            return fail(st);
    }
    // head: fp32 weights [classes][c] transposed to [c][classes]
    {
        const int C = cfin[2];
        float *fc_w = nullptr;
        if ((st = wcopy(n, &fc_w, d->fc_w, (size_t)d->num_classes * C, s)) != MINW_OK) return fail(st);
        if ((st = walloc(n, &D->fc_wt, (size_t)d->num_classes * C)) != MINW_OK) return fail(st);
        wres_transpose_kernel<<<64, 256, 0, s>>>(fc_w, d->num_classes, C, D->fc_wt);
        if ((st = wcopy(n, &D->fc_scale, d->fc_scale, d->num_classes, s)) != MINW_OK) return fail(st);
        if ((st = wcopy(n, &D->fc_shift, d->fc_shift, d->num_classes, s)) != MINW_OK) return fail(st);
        if ((st = walloc(n, &D->pooled, (size_t)max_batch * C)) != MINW_OK) return fail(st);
    }
    // activations; the bf16 buffers start at zero (what their padding channels are read as
    // before any layer has written them)
    for (int b = 0; b < 4; ++b) {
        const int h = hw >> (b < 3 ? b : 0);
        const size_t e = (size_t)max_batch * h * h * (b < 3 ? D->row[b] : pad64(4 * k));
        uint16_t *q = nullptr;
        if ((st = walloc(n, &q, e)) != MINW_OK) return fail(st);
        if (cudaMemsetAsync(q, 0, e * sizeof(uint16_t), s) != cudaSuccess) return fail(MINW_ECUDA);
        if (b < 3) D->F[b] = q; else D->HB = q;
    }
    if ((st = walloc(n, &D->Y, (size_t)max_batch * y_px)) != MINW_OK) return fail(st);
    n->x_elems = (size_t)max_batch * 3 * hw * hw;
    n->logit_elems = (size_t)max_batch * d->num_classes;
    if ((st = walloc(n, &n->x_stage, n->x_elems)) != MINW_OK ||
        (st = walloc(n, &n->logits_stage, n->logit_elems)) != MINW_OK)
        return fail(st);
    if (cudaStreamSynchronize(s) != cudaSuccess || cudaGetLastError() != cudaSuccess) return fail(MINW_ECUDA);
    *out = n;
    return MINW_OK;
}

extern "C" minw_status minw_wdense_features(const minw_net *net, int32_t block, uint16_t *dst, size_t count,
                                            int32_t *channels, int32_t *row, void *stream) {
    if (!net || net->kind != 3 || !net->wdense || !dst || block < 0 || block > 2) return MINW_EINVAL;
    const WDensePlan *D = net->wdense;
    if (D->last_B <= 0) return MINW_EINVAL;
    const int h = D->hw >> block;
    const size_t elems = (size_t)D->last_B * h * h * D->row[block];
    if (count < elems) return MINW_EINVAL;
    if (channels) *channels = D->cfin[block];
    if (row) *row = D->row[block];
    return cudaMemcpyAsync(dst, D->F[block], elems * sizeof(uint16_t), cudaMemcpyDeviceToDevice,
                           (cudaStream_t)stream) == cudaSuccess ? MINW_OK : MINW_ECUDA;
}
