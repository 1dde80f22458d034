// train.cu -- one training step of a fully connected MINW-Net layer
// (Algorithm 1, which applies to convolutional and fully connected layers
// alike): the weight AQE forward (Eq. weight, alpha < 1), the forward product
// a~ = a^q W^q, the activation AQE forward (Eq. activation), the backward mask
// of Eq. activation, the input gradient g_a = g_a~ W^q, the weight gradient
// g_W^q = g_a~^T a^q, the mask of Eq. weight, and the update with the clip to
// [-1, 1].  The three products run on the tensor cores as 1 x 1 convolutions
// of bf16 operands (conv_tc_kernel, kind::f16); the rest are elementwise
// kernels here and in aqe.cu.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

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

__global__ void fill_kernel(float *__restrict__ p, int64_t n, float v) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        p[i] = v;
}

static int64_t grid_of(int64_t n) {
    const int sms = minw_host::num_sms() > 0 ? minw_host::num_sms() : 152;
    int64_t g = (n + 255) / 256;
    if (g > sms * 8) g = sms * 8;
    return g < 1 ? 1 : g;
}

// Workspace of minw_fc_train_step: regions 256-byte aligned, in this order.
struct TrainLayout {
    size_t what, wb, wtb, ab, atb, at, gat, gb, gtb, gwhat, gw, ones, zeros, total;
};

static size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

static TrainLayout train_layout(int B, int K, int O) {
    const size_t Op = (size_t)((O + 63) / 64 * 64), M = (size_t)(K > O ? K : O);
    TrainLayout L;
    size_t off = 0;
    auto take = [&](size_t bytes) { const size_t r = off; off += al256(bytes); return r; };
    L.what = take(4 * (size_t)O * K);
    L.wb = take(2 * (size_t)O * K);
    L.wtb = take(2 * (size_t)K * Op);
    L.ab = take(2 * (size_t)B * K);
    L.atb = take(2 * (size_t)K * B);
    L.at = take(4 * (size_t)B * O);
    L.gat = take(4 * (size_t)B * O);
    L.gb = take(2 * (size_t)B * Op);
    L.gtb = take(2 * (size_t)O * B);
    L.gwhat = take(4 * (size_t)O * K);
    L.gw = take(4 * (size_t)O * K);
    L.ones = take(4 * M);
    L.zeros = take(4 * M);
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
                               float *g_in, void *workspace, size_t workspace_bytes, void *stream) {
    if (B <= 0 || K <= 0 || O <= 0 || !A || !W || !g_out || !a_out || !q_w || !workspace) return MINW_EINVAL;
    if (!(alpha >= 0.0f && alpha <= 1.0f)) return MINW_EINVAL;
    if (!valid_quant(q_w) || (q_a && !valid_quant(q_a))) return MINW_EINVAL;
    if (K % 64 != 0 || B % 64 != 0) return MINW_EUNSUPPORTED;
    if (!aligned16(A) || !aligned16(W) || !aligned16(g_out) || !aligned16(a_out) || (g_in && !aligned16(g_in)) ||
        !aligned16(workspace))
        return MINW_EINVAL;
    const TrainLayout L = train_layout(B, K, O);
    if (workspace_bytes < L.total) return MINW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    float *what = reinterpret_cast<float *>(ws + L.what), *at = reinterpret_cast<float *>(ws + L.at);
    float *gat = reinterpret_cast<float *>(ws + L.gat), *gwhat = reinterpret_cast<float *>(ws + L.gwhat);
    float *gw = reinterpret_cast<float *>(ws + L.gw);
    float *ones = reinterpret_cast<float *>(ws + L.ones), *zeros = reinterpret_cast<float *>(ws + L.zeros);
    uint16_t *wb = reinterpret_cast<uint16_t *>(ws + L.wb), *wtb = reinterpret_cast<uint16_t *>(ws + L.wtb);
    uint16_t *ab = reinterpret_cast<uint16_t *>(ws + L.ab), *atb = reinterpret_cast<uint16_t *>(ws + L.atb);
    uint16_t *gb = reinterpret_cast<uint16_t *>(ws + L.gb), *gtb = reinterpret_cast<uint16_t *>(ws + L.gtb);
    const int Op = (O + 63) / 64 * 64, M = K > O ? K : O;
    minw_status st;
#define TRY(x) do { if ((st = (x)) != MINW_OK) return st; } while (0)
    fill_kernel<<<(unsigned)grid_of(M), 256, 0, s>>>(ones, M, 1.0f);
    fill_kernel<<<(unsigned)grid_of(M), 256, 0, s>>>(zeros, M, 0.0f);
    TRY(launch_status());
    // 1.1 forward: W^ = alpha h(W) + (1 - alpha) W, a~ = a W^T, a_l = alpha h(a~) + (1 - alpha) a~
    TRY(aqe_forward(W, what, (int64_t)O * K, alpha, q_w, stream));
    TRY(minw_bf16_matrix(what, O, K, 0, K, wb, stream));
    TRY(minw_bf16_matrix(what, O, K, 1, Op, wtb, stream));
    TRY(minw_bf16_matrix(A, B, K, 0, K, ab, stream));
    TRY(minw_bf16_matrix(A, B, K, 1, B, atb, stream));
    float *fwd_out = q_a ? at : a_out;                 // the last layer emits a~ itself
    TRY(minw_conv2d_bf16(ab, B, K, 1, 1, wb, O, 1, 1, q_w->bits, 1, 0, 0, ones, zeros, fwd_out, stream));
    const float *g_at = g_out;
    if (q_a) {
        TRY(aqe_forward(at, a_out, (int64_t)B * O, alpha, q_a, stream));
        // 1.2 backward through the activation AQE (Eq. activation): 2 alpha g 1[|a~| <= 1]
        TRY(aqe_backward(at, g_out, gat, (int64_t)B * O, alpha, stream));
        g_at = gat;
    }
    TRY(minw_bf16_matrix(g_at, B, O, 0, Op, gb, stream));
    TRY(minw_bf16_matrix(g_at, B, O, 1, B, gtb, stream));
    if (g_in)                                          // g_a = g_a~ W^  ([B][K], reduction over O)
        TRY(minw_conv2d_bf16(gb, B, Op, 1, 1, wtb, K, 1, 1, q_w->bits, 1, 0, 0, ones, zeros, g_in, stream));
    // g_W^ = g_a~^T a  ([O][K], reduction over the batch)
    TRY(minw_conv2d_bf16(gtb, O, B, 1, 1, atb, K, 1, 1, q_w->bits, 1, 0, 0, ones, zeros, gwhat, stream));
    // 2. the mask of Eq. weight on the latent weights, then the update and the clip
    TRY(aqe_backward(W, gwhat, gw, (int64_t)O * K, alpha, stream));
    TRY(minw_sgd_clip(W, gw, (int64_t)O * K, lr, stream));
#undef TRY
    return MINW_OK;
}

}  // extern "C"
