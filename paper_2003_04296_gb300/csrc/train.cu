// train.cu -- one training step of a fully connected MINW-Net layer
// (Algorithm 1, which applies to convolutional and fully connected layers
// alike): the weight AQE forward (Eq. weight, alpha < 1), the forward product
// a~ = a^q W^q, the activation AQE forward (Eq. activation), the backward mask
// of Eq. activation, the input gradient g_a = g_a~ W^q, the weight gradient
// g_W^q = g_a~^T a^q, the mask of Eq. weight, and the update with the clip to
// [-1, 1].  The three products run on the tensor cores as 1 x 1 convolutions
// of bf16 operands (conv_tc_kernel, kind::f16); each operand is made in one
// pass over its fp32 source (AQE, bf16 rounding, the transposed copy), and the
// weight-gradient product applies the mask of Eq. weight and the update in its
// epilogue, so that the weight gradient never reaches memory.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace minw {

// out[i][j] (out_rows x out_cols, bf16, round to nearest even) = in[i][j], or
// in[j][i] when trans, zero outside the source; through 32 x 32 shared tiles,
// so that both the reads and the writes coalesce.
__global__ void bf16_matrix_kernel(const float *__restrict__ in, int rows, int cols, int trans, int out_rows,
                                   int out_cols, uint16_t *__restrict__ out) {
    __shared__ float tile[32][33];
    const int i0 = blockIdx.y * 32, j0 = blockIdx.x * 32;          // output tile origin
    // source tile: rows [i0, i0 + 32) x cols [j0, j0 + 32) of the output, read from in
    for (int k = threadIdx.y; k < 32; k += blockDim.y) {
        if (trans) {        // out[i][j] = in[j][i]: read in[j0 + k][i0 + x]
            const int r = j0 + k, c = i0 + threadIdx.x;
            tile[threadIdx.x][k] = (r < rows && c < cols) ? in[(int64_t)r * cols + c] : 0.0f;
        } else {
            const int r = i0 + k, c = j0 + threadIdx.x;
            tile[k][threadIdx.x] = (r < rows && c < cols) ? in[(int64_t)r * cols + c] : 0.0f;
        }
    }
    __syncthreads();
    for (int k = threadIdx.y; k < 32; k += blockDim.y) {
        const int i = i0 + k, j = j0 + threadIdx.x;
        if (i < out_rows && j < out_cols)
            out[(int64_t)i * out_cols + j] = __bfloat16_as_ushort(__float2bfloat16_rn(tile[k][threadIdx.x]));
    }
}

// w <- min(1, max(-1, w - lr g)), the fp32 update of Algorithm 1 (plain
// gradient step, then the clip to [-1, 1]).
__global__ void sgd_clip_kernel(float *__restrict__ w, const float *__restrict__ g, int64_t n, float lr) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        w[i] = fminf(1.0f, fmaxf(-1.0f, fmaf(-lr, g[i], w[i])));
}

static int64_t grid_of(int64_t n) {
    const int sms = minw_host::num_sms() > 0 ? minw_host::num_sms() : 152;
    int64_t g = (n + 255) / 256;
    if (g > sms * 8) g = sms * 8;
    return g < 1 ? 1 : g;
}

__device__ __forceinline__ uint32_t bf16x2(float lo, float hi) {
    return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(lo)) |
           ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(hi)) << 16);
}

// The operand preparation of one product pair, in one pass over a row-major
// fp32 matrix X [R][C]: v = f(X) as bf16 both row-major (vb [R][Cp], columns
// C..Cp zero) and transposed (vtb [C][Rp], columns R..Rp zero), through a
// 32 x 64 shared tile.
//   MODE 0  weights: v = alpha h(W) + (1 - alpha) W (Eq. weight); also fills
//           ones[0..M) = 1 and zeros[0..M) = 0 (the unit BN of the products)
//   MODE 1  activations: v = a
//   MODE 2  output gradients: with a_out, v = 2 alpha g 1[|a~| <= 1] (the
//           backward of Eq. activation, X = a~, G = g) and a_out = alpha h(a~)
//           + (1 - alpha) a~; without it (a layer without an activation
//           quantizer), v = g
// Every value takes the same fp32 operations as aqe_forward / aqe_backward.
template <int MODE>
__global__ void __launch_bounds__(256) prep_kernel(const float *__restrict__ X, const float *__restrict__ G, int R,
                                                   int C, int Cp, int Rp, float alpha, QParams q,
                                                   uint16_t *__restrict__ vb, uint16_t *__restrict__ vtb,
                                                   float *__restrict__ a_out, float *__restrict__ ones,
                                                   float *__restrict__ zeros, int M) {
    __shared__ float tile[32][65];
    const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 64;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;     // columns 4 tx .. 4 tx + 3 of rows ty, ty + 16
    const float oma = 1.0f - alpha, two_alpha = 2.0f * alpha;
    const int c = c0 + 4 * tx;
    const bool vec = (C & 3) == 0 && c < C;                       // four columns inside, 16-byte aligned
    // all loads first (two rows x four columns of X, and of G)
    float x[2][4], g[2][4];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int r = r0 + ty + 16 * h;
        const int64_t at = (int64_t)r * C + c;
#pragma unroll
        for (int e = 0; e < 4; ++e) x[h][e] = g[h][e] = 0.0f;
        if (r >= R) continue;
        if (vec) {
            const float4 x4 = *reinterpret_cast<const float4 *>(X + at);
            x[h][0] = x4.x; x[h][1] = x4.y; x[h][2] = x4.z; x[h][3] = x4.w;
            if (MODE == 2) {
                const float4 g4 = *reinterpret_cast<const float4 *>(G + at);
                g[h][0] = g4.x; g[h][1] = g4.y; g[h][2] = g4.z; g[h][3] = g4.w;
            }
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e)
                if (c + e < C) {
                    x[h][e] = X[at + e];
                    if (MODE == 2) g[h][e] = G[at + e];
                }
        }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int k = ty + 16 * h, r = r0 + k;
        const int64_t at = (int64_t)r * C + c;
        float v[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        if (r < R) {
            float ao[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                if (c + e >= C) continue;
                if (MODE == 0) {
                    v[e] = fmaf(alpha, level_value(x[h][e] * q.scale, q), oma * x[h][e]);
                } else if (MODE == 1) {
                    v[e] = x[h][e];
                } else if (a_out != nullptr) {
                    ao[e] = fmaf(alpha, level_value(x[h][e] * q.scale, q), oma * x[h][e]);
                    v[e] = (fabsf(x[h][e]) <= 1.0f) ? g[h][e] * two_alpha : 0.0f;
                } else {
                    v[e] = g[h][e];
                }
            }
            if (MODE == 2 && a_out != nullptr) {
                if (vec) {
                    *reinterpret_cast<float4 *>(a_out + at) = make_float4(ao[0], ao[1], ao[2], ao[3]);
                } else {
                    for (int e = 0; e < 4; ++e)
                        if (c + e < C) a_out[at + e] = ao[e];
                }
            }
            uint16_t *dst = vb + (int64_t)r * Cp + c;
            if (c + 3 < Cp && (Cp & 3) == 0)
                *reinterpret_cast<uint2 *>(dst) = make_uint2(bf16x2(v[0], v[1]), bf16x2(v[2], v[3]));
            else
                for (int e = 0; e < 4; ++e)
                    if (c + e < Cp) dst[e] = __bfloat16_as_ushort(__float2bfloat16_rn(v[e]));
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) tile[k][4 * tx + e] = v[e];
    }
    if (MODE == 0) {
        const int64_t nthr = (int64_t)gridDim.x * gridDim.y * blockDim.x;
        for (int64_t i = ((int64_t)blockIdx.y * gridDim.x + blockIdx.x) * blockDim.x + threadIdx.x; i < M; i += nthr) {
            ones[i] = 1.0f;
            zeros[i] = 0.0f;
        }
    }
    __syncthreads();
    // transposed: row c0 + cc of vtb, its 32 values r0 .. r0 + 31 as four 8-value runs
    const int cc = threadIdx.x >> 2, part = threadIdx.x & 3;
    const int ct = c0 + cc, rt = r0 + part * 8;
    if (ct < C && rt < Rp) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) w[e] = bf16x2(tile[part * 8 + 2 * e][cc], tile[part * 8 + 2 * e + 1][cc]);
        uint16_t *dst = vtb + (int64_t)ct * Rp + rt;
        if (rt + 8 <= Rp && (Rp & 7) == 0) {
            *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
        } else {
            for (int e = 0; e < 8 && rt + e < Rp; ++e) dst[e] = (uint16_t)(w[e >> 1] >> (16 * (e & 1)));
        }
    }
}

// Workspace of minw_fc_train_step: regions 256-byte aligned, in this order;
// split holds the K-sliced partial sums of the products.
struct TrainLayout {
    size_t wb, wtb, ab, atb, at, gb, gtb, ones, zeros, split, split_bytes, total;
};

static size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

static TrainLayout train_layout(int B, int K, int O) {
    const int Op = (O + 63) / 64 * 64;
    const size_t M = (size_t)(K > O ? K : O);
    // split-K partial sums: the largest need of the three products
    size_t need = 0;
    auto want = [&](int nb, int c, int o) {
        size_t w = 0;
        if (conv2d_bf16(nullptr, nb, c, 1, 1, nullptr, o, 1, 1, 1, 1, 0, 0, nullptr, nullptr, nullptr, nullptr, 0, &w,
                        nullptr) == MINW_OK &&
            w > need)
            need = w;
    };
    want(B, K, O);        // forward
    want(B, Op, K);       // input gradient (the weight gradient never splits: it updates W in its epilogue)
    TrainLayout L;
    size_t off = 0;
    auto take = [&](size_t bytes) { const size_t r = off; off += al256(bytes); return r; };
    L.wb = take(2 * (size_t)O * K);
    L.wtb = take(2 * (size_t)K * Op);
    L.ab = take(2 * (size_t)B * K);
    L.atb = take(2 * (size_t)K * B);
    L.at = take(4 * (size_t)B * O);
    L.gb = take(2 * (size_t)B * Op);
    L.gtb = take(2 * (size_t)O * B);
    L.ones = take(4 * M);
    L.zeros = take(4 * M);
    L.split_bytes = need;
    L.split = take(need);
    L.total = off;
    return L;
}

}  // namespace minw

using namespace minw;
using namespace minw_host;

extern "C" {

minw_status minw_bf16_matrix(const float *in, int32_t rows, int32_t cols, int32_t transpose, int32_t out_cols,
                             uint16_t *out, void *stream) {
    if (rows <= 0 || cols <= 0 || !in || !out) return MINW_EINVAL;
    const int out_rows = transpose ? cols : rows;
    if (out_cols < (transpose ? rows : cols)) return MINW_EINVAL;
    if (out_rows > 65535 * 32) return MINW_EUNSUPPORTED;
    const dim3 grid((unsigned)((out_cols + 31) / 32), (unsigned)((out_rows + 31) / 32));
    bf16_matrix_kernel<<<grid, dim3(32, 8), 0, (cudaStream_t)stream>>>(in, rows, cols, transpose ? 1 : 0, out_rows,
                                                                       out_cols, out);
    return launch_status();
}

minw_status minw_sgd_clip(float *w, const float *g, int64_t n, float lr, void *stream) {
    if (n < 0 || !w || !g) return MINW_EINVAL;
    if (n == 0) return MINW_OK;
    sgd_clip_kernel<<<(unsigned)grid_of(n), 256, 0, (cudaStream_t)stream>>>(w, g, n, lr);
    return launch_status();
}

size_t minw_fc_train_workspace_bytes(int32_t B, int32_t K, int32_t O) {
    if (B <= 0 || K <= 0 || O <= 0) return 0;
    return train_layout(B, K, O).total;
}

minw_status minw_fc_train_step(const float *A, float *W, const float *g_out, int32_t B, int32_t K, int32_t O,
                               float alpha, float lr, const minw_quant *q_w, const minw_quant *q_a, float *a_out,
                               float *g_in, float *a_pre, void *workspace, size_t workspace_bytes, void *stream) {
    if (B <= 0 || K <= 0 || O <= 0 || !A || !W || !g_out || !a_out || !q_w || !workspace) return MINW_EINVAL;
    if (!(alpha >= 0.0f && alpha <= 1.0f)) return MINW_EINVAL;
    if (!valid_quant(q_w) || (q_a && !valid_quant(q_a))) return MINW_EINVAL;
    if (K % 64 != 0 || B % 64 != 0) return MINW_EUNSUPPORTED;
    if (!aligned16(A) || !aligned16(W) || !aligned16(g_out) || !aligned16(a_out) || (g_in && !aligned16(g_in)) ||
        (a_pre && !aligned16(a_pre)) ||
        !aligned16(workspace))
        return MINW_EINVAL;
    const TrainLayout L = train_layout(B, K, O);
    if (workspace_bytes < L.total) return MINW_EINVAL;
    if ((int64_t)K * (O + 63) >= (1ll << 31) || (int64_t)B * K >= (1ll << 31)) return MINW_EUNSUPPORTED;
    if ((O + 63) / 32 > 65535 || B / 32 > 65535) return MINW_EUNSUPPORTED;       // grid rows of the passes
    cudaStream_t s = (cudaStream_t)stream;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    float *at = a_pre ? a_pre : reinterpret_cast<float *>(ws + L.at);
    float *ones = reinterpret_cast<float *>(ws + L.ones), *zeros = reinterpret_cast<float *>(ws + L.zeros);
    uint16_t *wb = reinterpret_cast<uint16_t *>(ws + L.wb), *wtb = reinterpret_cast<uint16_t *>(ws + L.wtb);
    uint16_t *ab = reinterpret_cast<uint16_t *>(ws + L.ab), *atb = reinterpret_cast<uint16_t *>(ws + L.atb);
    uint16_t *gb = reinterpret_cast<uint16_t *>(ws + L.gb), *gtb = reinterpret_cast<uint16_t *>(ws + L.gtb);
    void *split = L.split_bytes ? ws + L.split : nullptr;
    const int Op = (O + 63) / 64 * 64, M = K > O ? K : O;
    const QParams qw = to_qparams(q_w), qa = q_a ? to_qparams(q_a) : QParams{};
    minw_status st;
#define TRY(x) do { if ((st = (x)) != MINW_OK) return st; } while (0)
    // 1.1 forward: W^ = alpha h(W) + (1 - alpha) W as bf16 [O][K] and [K][Op]; a as bf16 [B][K] and [K][B]
    prep_kernel<0><<<dim3((unsigned)(K / 64), (unsigned)(Op / 32)), 256, 0, s>>>(
        W, nullptr, O, K, K, Op, alpha, qw, wb, wtb, nullptr, ones, zeros, M);
    prep_kernel<1><<<dim3((unsigned)(K / 64), (unsigned)(B / 32)), 256, 0, s>>>(
        A, nullptr, B, K, K, B, 0.0f, qw, ab, atb, nullptr, nullptr, nullptr, 0);
    TRY(launch_status());
    // a~ = a W^T  ([B][O], reduction over K); the last layer emits a~ itself
    float *fwd_out = q_a ? at : a_out;
    TRY(conv2d_bf16(ab, B, K, 1, 1, wb, O, 1, 1, q_w->bits, 1, 0, 0, ones, zeros, fwd_out, split, L.split_bytes,
                    nullptr, s));
    // 1.2 backward through the activation AQE (Eq. activation): g_a~ = 2 alpha g 1[|a~| <= 1], as bf16
    // [B][Op] and [O][B]; a_l = alpha h(a~) + (1 - alpha) a~
    prep_kernel<2><<<dim3((unsigned)(Op / 64), (unsigned)(B / 32)), 256, 0, s>>>(
        q_a ? at : g_out, g_out, B, O, Op, B, alpha, qa, gb, gtb, q_a ? a_out : nullptr, nullptr, nullptr, 0);
    TRY(launch_status());
    if (g_in)                                          // g_a = g_a~ W^  ([B][K], reduction over O)
        TRY(conv2d_bf16(gb, B, Op, 1, 1, wtb, K, 1, 1, q_w->bits, 1, 0, 0, ones, zeros, g_in, split, L.split_bytes,
                        nullptr, s));
    // g_W^ = g_a~^T a  ([O][K], reduction over the batch), and in the same epilogue
    // 2. the mask of Eq. weight on the latent weights, the update and the clip:
    // W = min(1, max(-1, W - lr 2 alpha g_W^ 1[|W| <= 1])), element by element
    TRY(conv2d_bf16(gtb, O, B, 1, 1, atb, K, 1, 1, q_w->bits, 1, 0, 0, ones, zeros, W, nullptr, 0, nullptr, s, 1, lr,
                    2.0f * alpha));
#undef TRY
    return MINW_OK;
}

}  // extern "C"
