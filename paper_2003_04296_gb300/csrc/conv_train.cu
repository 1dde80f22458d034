// conv_train.cu -- one training step of a convolutional MINW-Net layer
// (Algorithm 1, training branch, which treats convolutional and fully
// connected layers alike): the weight AQE forward (Eq. weight), the forward
// convolution a~ = a W^, the activation AQE and the backward mask of Eq.
// activation, the input gradient (the convolution's transpose applied to
// g~), the weight gradient (the correlation of g~ with the input over the
// batch and the image), the mask of Eq. weight and the clipped update.
//
// The three products run on the tensor cores (conv_tc_kernel on bf16
// operands, kind::f16, fp32 accumulation):
//   forward         implicit GEMM over (ky, kx, c) of the NHWC input and the
//                   weights [O][kh][kw][C]
//   input gradient  the same kernel, stride 1, on g~ spread over an image of
//                   the input's size class (rows and columns y s, x s; zero
//                   between them and in the padded channels) against the
//                   flipped, transposed weights [C][kh][kw][Op] with padding
//                   kh - 1 - pad: the transposed convolution, no scatter
//   weight gradient a GEMM over the B Ho Wo output pixels of g~ [O][n] and
//                   the input's patches [(c, ky, kx)][n] (im2col, K-major),
//                   split along the pixels across the SMs; its output rows are
//                   W's own (c, ky, kx) order, so the update reads W in place.
// Every operand is written once by a pass over its fp32 source.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>

#include "kernels.cuh"

namespace minw {

__device__ __forceinline__ uint16_t bf16_bits(float v) { return __bfloat16_as_ushort(__float2bfloat16_rn(v)); }

// W^ = alpha h(W) + (1 - alpha) W of the latent weights W [O][C][kh][kw]
// (Eq. weight, the fp32 operations of aqe_forward), as bf16 in two layouts:
//   wf [O][kh][kw][C]   the forward product's weights
//   wd [C][kh][kw][Op]  wd[c][ky][kx][o] = W^[o][c][kh-1-ky][kw-1-kx], zero
//                       for o >= O: the input gradient's weights
// Also fills ones[0..M) = 1 and zeros[0..M) = 0 (the unit BN of the products).
__global__ void __launch_bounds__(256) train_weights_kernel(const float *__restrict__ W, int O, int C, int kh, int kw,
                                                            int Op, float alpha, QParams q, uint16_t *__restrict__ wf,
                                                            uint16_t *__restrict__ wd, float *__restrict__ ones,
                                                            float *__restrict__ zeros, int M) {
    // element counts below 2^31 (checked by the host): 32-bit index arithmetic
    const float oma = 1.0f - alpha;
    const int khw = kh * kw;
    const int nf = O * khw * C, nd = C * khw * Op;
    const int stride = gridDim.x * blockDim.x;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nf; i += stride) {
        // i = ((o kh + ky) kw + kx) C + c
        const int c = i % C, r = i / C;
        const int t = r % khw, o = r / khw;
        const float x = W[(o * C + c) * khw + t];
        wf[i] = bf16_bits(fmaf(alpha, level_value(x * q.scale, q), oma * x));
    }
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nd; i += stride) {
        // i = ((c kh + ky) kw + kx) Op + o, source tap (kh - 1 - ky, kw - 1 - kx)
        const int o = i % Op, r = i / Op;
        const int t = r % khw, c = r / khw;
        float v = 0.0f;
        if (o < O) {
            const int ky = t / kw, kx = t - ky * kw;
            const float x = W[(o * C + c) * khw + (kh - 1 - ky) * kw + (kw - 1 - kx)];
            v = fmaf(alpha, level_value(x * q.scale, q), oma * x);
        }
        wd[i] = bf16_bits(v);
    }
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < M; i += stride) {
        ones[i] = 1.0f;
        zeros[i] = 0.0f;
    }
}

// The input's patches, transposed: colT[(c kh + ky) kw + kx][n] =
// bf16(A[b][c][y s - pad + ky][x s - pad + kx]) for output pixel n = (b Ho +
// y) Wo + x, zero outside the image.  A thread takes eight consecutive pixels
// n0 .. n0 + 7 of one channel c (blockIdx.y) and writes them for every tap:
// kh kw 16-byte stores, each warp's store of a tap 512 contiguous bytes of
// that tap's row.  The pixels' (b, y, x) come from one division and carries;
// the taps' overlapping input reads hit L1, so each input value crosses from
// L2 about once instead of once per tap.
__global__ void __launch_bounds__(256) train_patches_kernel(const float *__restrict__ A, int B, int C, int H, int W,
                                                            int kh, int kw, int stride, int pad, int Ho, int Wo,
                                                            uint16_t *__restrict__ colT) {
    const int HoWo = Ho * Wo;
    const int npix = B * HoWo;                            // < 2^31 and a multiple of 8 (checked by the host)
    const int c = blockIdx.y;
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= npix / 8) return;
    const int n0 = 8 * g;
    // the eight pixels: image offset, first input row and column
    int64_t base[8];
    int iy0[8], ix0[8];
    {
        int b = n0 / HoWo;
        const int r = n0 - b * HoWo;
        int y = r / Wo, x = r - (r / Wo) * Wo;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            base[e] = ((int64_t)b * C + c) * H * W;
            iy0[e] = y * stride - pad;
            ix0[e] = x * stride - pad;
            if (++x == Wo) {
                x = 0;
                if (++y == Ho) {
                    y = 0;
                    ++b;
                }
            }
        }
    }
    for (int ky = 0; ky < kh; ++ky) {
        for (int kx = 0; kx < kw; ++kx) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int iy = iy0[e] + ky, ix = ix0[e] + kx;
                const float v = (iy >= 0 && iy < H && ix >= 0 && ix < W) ? __ldg(A + base[e] + (int64_t)iy * W + ix)
                                                                          : 0.0f;
                if (e & 1)
                    w[e >> 1] |= (uint32_t)bf16_bits(v) << 16;
                else
                    w[e >> 1] = (uint32_t)bf16_bits(v);
            }
            const int64_t row = ((int64_t)c * kh + ky) * kw + kx;
            *reinterpret_cast<uint4 *>(colT + row * npix + n0) = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

// The pass over the forward output a~ and the upstream gradient g (both
// [B][O][Ho][Wo]):
//   a_out = alpha h(a~) + (1 - alpha) a~            (Eq. activation; with q_a)
//   g~    = 2 alpha g 1[|a~| <= 1]                 (its backward; g itself without q_a)
//   gT[o][n] = bf16(g~)                            the weight gradient's operand, n = (b Ho + y) Wo + x
//   gd[b][y s][x s][o] = bf16(g~)                  the input gradient's operand (NHWC [B][Hd][Wd][Op],
//                                                  zero elsewhere: the buffer is cleared beforehand)
// A block takes 32 channels x 32 pixels of one image through shared memory,
// so that the NCHW reads and the gT writes run along pixels and the gd writes
// along channels.
__global__ void __launch_bounds__(256) train_grad_kernel(const float *__restrict__ at, const float *__restrict__ G,
                                                         int O, int HoWo, int Wo, int stride, int Hd, int Wd, int Op,
                                                         float alpha, int quant_a, QParams qa,
                                                         float *__restrict__ a_out, uint16_t *__restrict__ gT,
                                                         uint16_t *__restrict__ gd, int64_t npix) {
    __shared__ float tile[32][33];
    const int b = blockIdx.z;
    const int o0 = blockIdx.y * 32, p0 = blockIdx.x * 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;      // 8 rows of 32
    const float oma = 1.0f - alpha, two_alpha = 2.0f * alpha;
    // the four rows' loads first, then the arithmetic and the stores
    float gl[4], xl[4];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
        const int o = o0 + ty + 8 * kk, p = p0 + tx;
        gl[kk] = xl[kk] = 0.0f;
        if (o < O && p < HoWo) {
            const int64_t idx = ((int64_t)b * O + o) * HoWo + p;
            gl[kk] = __ldg(G + idx);
            if (quant_a) xl[kk] = __ldg(at + idx);
        }
    }
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
        const int k = ty + 8 * kk;
        const int o = o0 + k, p = p0 + tx;
        float gv = 0.0f;
        if (o < O && p < HoWo) {
            const int64_t idx = ((int64_t)b * O + o) * HoWo + p;
            if (quant_a) {
                const float x = xl[kk];
                a_out[idx] = fmaf(alpha, level_value(x * qa.scale, qa), oma * x);
                gv = (fabsf(x) <= 1.0f) ? gl[kk] * two_alpha : 0.0f;
            } else {
                gv = gl[kk];
            }
            gT[(int64_t)o * npix + (int64_t)b * HoWo + p] = bf16_bits(gv);
        }
        tile[k][tx] = gv;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
        const int k = ty + 8 * kk;
        const int p = p0 + k, o = o0 + tx;
        if (p < HoWo && o < O) {
            const int y = p / Wo, x = p - y * Wo;
            gd[(((int64_t)b * Hd + (int64_t)y * stride) * Wd + (int64_t)x * stride) * Op + o] = bf16_bits(tile[tx][k]);
        }
    }
}

// Eq. weight's mask and the update with the clip, in the fp32 operations of
// aqe_backward and minw_sgd_clip: w = min(1, max(-1, fmaf(-lr, g', w))) with
// g' = g 2 alpha where |w| <= 1, else 0.
__global__ void train_update_kernel(float *__restrict__ w, const float *__restrict__ g, int64_t n, float lr,
                                    float two_alpha) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const float wi = w[i];
        const float gm = (fabsf(wi) <= 1.0f) ? g[i] * two_alpha : 0.0f;
        w[i] = fminf(1.0f, fmaxf(-1.0f, fmaf(-lr, gm, wi)));
    }
}

static unsigned grid_for(int64_t n) {
    const int sms = minw_host::num_sms() > 0 ? minw_host::num_sms() : 152;
    int64_t g = (n + 255) / 256;
    if (g > (int64_t)sms * 16) g = (int64_t)sms * 16;
    return (unsigned)(g < 1 ? 1 : g);
}

// Shape of one step: the input gradient's spread image is the output image
// with stride - 1 zero rows and columns between samples, plus the rows and
// columns the forward convolution's stride left unread at the bottom and the
// right, so that its stride-1 convolution with padding kh - 1 - pad gives H x W.
struct ConvTrainShape {
    int Ho, Wo, Hd, Wd, Op, Kw;
    int64_t npix;
};

static bool conv_train_shape(int B, int C, int H, int W, int O, int kh, int kw, int stride, int pad,
                             ConvTrainShape &s) {
    s.Ho = (H + 2 * pad - kh) / stride + 1;
    s.Wo = (W + 2 * pad - kw) / stride + 1;
    if (s.Ho <= 0 || s.Wo <= 0) return false;
    s.Hd = (s.Ho - 1) * stride + 1 + (H + 2 * pad - kh) % stride;
    s.Wd = (s.Wo - 1) * stride + 1 + (W + 2 * pad - kw) % stride;
    s.Op = (O + 63) / 64 * 64;
    s.Kw = C * kh * kw;
    s.npix = (int64_t)B * s.Ho * s.Wo;
    return true;
}

// Workspace of minw_conv_train_step: regions 256-byte aligned, in this order.
struct ConvTrainLayout {
    size_t wf, wd, ab, colT, at, gT, gd, gW, ones, zeros, split, split_bytes, total;
};

static size_t al256c(size_t x) { return (x + 255) & ~(size_t)255; }

static minw_status conv_train_layout(int B, int C, int H, int W, int O, int kh, int kw, int stride, int pad,
                                     ConvTrainLayout &L) {
    ConvTrainShape s;
    if (!conv_train_shape(B, C, H, W, O, kh, kw, stride, pad, s)) return MINW_EINVAL;
    size_t need = 0;
    minw_status st;
    auto want = [&](const uint16_t *, int nb, int c, int h, int w, int o, int k1, int k2, int str, int pd) {
        size_t q = 0;
        const minw_status r = conv2d_bf16(nullptr, nb, c, h, w, nullptr, o, k1, k2, 1, str, pd, 0, nullptr, nullptr,
                                          nullptr, nullptr, 0, &q, nullptr);
        if (r == MINW_OK && q > need) need = q;
        return r;
    };
    if ((st = want(nullptr, B, C, H, W, O, kh, kw, stride, pad)) != MINW_OK) return st;                 // forward
    if ((st = want(nullptr, B, s.Op, s.Hd, s.Wd, C, kh, kw, 1, kh - 1 - pad)) != MINW_OK) return st;    // input gradient
    if (s.npix > INT32_MAX) return MINW_EUNSUPPORTED;
    if ((st = want(nullptr, O, (int)s.npix, 1, 1, s.Kw, 1, 1, 1, 0)) != MINW_OK) return st;            // weight gradient
    size_t off = 0;
    auto take = [&](size_t bytes) { const size_t r = off; off += al256c(bytes); return r; };
    const int khw = kh * kw;
    L.wf = take(2 * (size_t)O * khw * C);
    L.wd = take(2 * (size_t)C * khw * s.Op);
    L.ab = take(2 * (size_t)B * H * W * C);
    L.colT = take(2 * (size_t)s.Kw * s.npix);
    L.at = take(4 * (size_t)O * s.npix);
    L.gT = take(2 * (size_t)O * s.npix);
    L.gd = take(2 * (size_t)B * s.Hd * s.Wd * s.Op);
    L.gW = take(4 * (size_t)O * s.Kw);
    const size_t M = (size_t)std::max(std::max(O, C), s.Kw);
    L.ones = take(4 * M);
    L.zeros = take(4 * M);
    L.split_bytes = need;
    L.split = take(need);
    L.total = off;
    return MINW_OK;
}

}  // namespace minw

using namespace minw;
using namespace minw_host;

extern "C" {

size_t minw_conv_train_workspace_bytes(int32_t B, int32_t C, int32_t H, int32_t W, int32_t O, int32_t kh, int32_t kw,
                                       int32_t stride, int32_t pad) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || O <= 0 || kh <= 0 || kw <= 0 || stride <= 0 || pad < 0) return 0;
    ConvTrainLayout L;
    if (conv_train_layout(B, C, H, W, O, kh, kw, stride, pad, L) != MINW_OK) return 0;
    return L.total;
}

minw_status minw_conv_train_step(const float *A, float *Wt, const float *g_out, int32_t B, int32_t C, int32_t H,
                                 int32_t W, int32_t O, int32_t kh, int32_t kw, int32_t stride, int32_t pad,
                                 float alpha, float lr, const minw_quant *q_w, const minw_quant *q_a, float *a_out,
                                 float *g_in, float *a_pre, void *workspace, size_t workspace_bytes, void *stream) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || O <= 0 || kh <= 0 || kw <= 0 || stride <= 0 || pad < 0)
        return MINW_EINVAL;
    if (!A || !Wt || !g_out || !a_out || !q_w || !workspace) return MINW_EINVAL;
    if (!(alpha >= 0.0f && alpha <= 1.0f)) return MINW_EINVAL;
    if (!valid_quant(q_w) || (q_a && !valid_quant(q_a))) return MINW_EINVAL;
    if (!aligned16(A) || !aligned16(Wt) || !aligned16(g_out) || !aligned16(a_out) || (g_in && !aligned16(g_in)) ||
        (a_pre && !aligned16(a_pre)) || !aligned16(workspace))
        return MINW_EINVAL;
    if (stride > 2 || pad >= kh || pad >= kw || C % 64 != 0) return MINW_EUNSUPPORTED;
    ConvTrainShape sh;
    if (!conv_train_shape(B, C, H, W, O, kh, kw, stride, pad, sh)) return MINW_EINVAL;
    if (sh.npix % 64 != 0 || sh.npix > INT32_MAX) return MINW_EUNSUPPORTED;
    // 32-bit grid limits of the gradient pass; 64-bit element indices everywhere else
    if ((O + 31) / 32 > 65535 || B > 65535 || C > 65535) return MINW_EUNSUPPORTED;

    if ((int64_t)sh.Kw * (O > sh.Op ? O : sh.Op) >= (1ll << 31)) return MINW_EUNSUPPORTED;     // weight pass indices
    ConvTrainLayout L;
    minw_status st = conv_train_layout(B, C, H, W, O, kh, kw, stride, pad, L);
    if (st != MINW_OK) return st;
    if (workspace_bytes < L.total) return MINW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    uint16_t *wf = reinterpret_cast<uint16_t *>(ws + L.wf), *wd = reinterpret_cast<uint16_t *>(ws + L.wd);
    uint16_t *ab = reinterpret_cast<uint16_t *>(ws + L.ab), *colT = reinterpret_cast<uint16_t *>(ws + L.colT);
    uint16_t *gT = reinterpret_cast<uint16_t *>(ws + L.gT), *gd = reinterpret_cast<uint16_t *>(ws + L.gd);
    float *at = a_pre ? a_pre : reinterpret_cast<float *>(ws + L.at);
    float *gW = reinterpret_cast<float *>(ws + L.gW);
    float *ones = reinterpret_cast<float *>(ws + L.ones), *zeros = reinterpret_cast<float *>(ws + L.zeros);
    void *split = L.split_bytes ? ws + L.split : nullptr;
    const QParams qw = to_qparams(q_w), qa = q_a ? to_qparams(q_a) : QParams{};
    const int M = std::max(std::max(O, C), sh.Kw);
#define TRY(x) do { if ((st = (x)) != MINW_OK) return st; } while (0)
    // W^ (Eq. weight) in both layouts; the input as bf16 NHWC and as transposed patches
    train_weights_kernel<<<grid_for((int64_t)O * kh * kw * C), 256, 0, s>>>(Wt, O, C, kh, kw, sh.Op, alpha, qw, wf,
                                                                             wd, ones, zeros, M);
    TRY(launch_status());
    TRY(minw_to_bf16_nhwc(A, B, C, H, W, ab, stream));
    {
        const dim3 grid((unsigned)((sh.npix / 8 + 255) / 256), (unsigned)C);
        train_patches_kernel<<<grid, 256, 0, s>>>(A, B, C, H, W, kh, kw, stride, pad, sh.Ho, sh.Wo, colT);
    }
    TRY(launch_status());
    // a~ = a * W^ (fp32 NCHW [B][O][Ho][Wo]); the last layer emits a~ itself
    float *fwd_out = q_a ? at : a_out;
    TRY(conv2d_bf16(ab, B, C, H, W, wf, O, kh, kw, q_w->bits, stride, pad, 0, ones, zeros, fwd_out, split,
                    L.split_bytes, nullptr, s));
    // g~ (Eq. activation's backward) and a_out; the spread image is cleared first where it has gaps
    if (g_in && (stride > 1 || sh.Op > O || sh.Hd > (sh.Ho - 1) * stride + 1 || sh.Wd > (sh.Wo - 1) * stride + 1))
        if (cudaMemsetAsync(gd, 0, (size_t)B * sh.Hd * sh.Wd * sh.Op * 2, s) != cudaSuccess) return MINW_ECUDA;
    {
        const dim3 grid((unsigned)((sh.Ho * sh.Wo + 31) / 32), (unsigned)((O + 31) / 32), (unsigned)B);
        train_grad_kernel<<<grid, 256, 0, s>>>(q_a ? at : g_out, g_out, O, sh.Ho * sh.Wo, sh.Wo, stride, sh.Hd, sh.Wd,
                                               sh.Op, alpha, q_a ? 1 : 0, qa, a_out, gT, gd, sh.npix);
        TRY(launch_status());
    }
    // the input gradient: the stride-1 convolution of the spread g~ with the flipped weights (NCHW [B][C][H][W])
    if (g_in)
        TRY(conv2d_bf16(gd, B, sh.Op, sh.Hd, sh.Wd, wd, C, kh, kw, q_w->bits, 1, kh - 1 - pad, 0, ones, zeros, g_in,
                        split, L.split_bytes, nullptr, s));
    // the weight gradient [O][(c, ky, kx)] = g~^T patches, reduced over the B Ho Wo pixels
    TRY(conv2d_bf16(gT, O, (int)sh.npix, 1, 1, colT, sh.Kw, 1, 1, q_w->bits, 1, 0, 0, ones, zeros, gW, split,
                    L.split_bytes, nullptr, s));
    // Eq. weight's mask, the update and the clip, on W in place
    const int64_t nw = (int64_t)O * sh.Kw;
    train_update_kernel<<<grid_for(nw), 256, 0, s>>>(Wt, gW, nw, lr, 2.0f * alpha);
    TRY(launch_status());
#undef TRY
    return MINW_OK;
}

}  // extern "C"
