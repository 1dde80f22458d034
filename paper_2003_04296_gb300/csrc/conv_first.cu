// conv_first.cu -- the first layer of a MINW-Net (Sec. III-E): the fp32 image
// is not quantized, its weights are.  Each output is one fp32 fmaf chain over
// (c, ky, kx) in that order with padded taps skipped, so the result does not
// depend on the launch shape.  BN (fmaf), HardTanh and quantize + pack of the
// next layer's input are fused into the epilogue.
//
// A CTA owns 256 consecutive output pixels and one group of 32 output
// channels (one packed word per plane per pixel); the group's quantized
// weights sit in shared memory and are read as broadcasts.
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace minw {


constexpr int FIRST_NT = 256;

__global__ void __launch_bounds__(FIRST_NT) conv_first_kernel(const FirstArgs a) {
    extern __shared__ float sW[];                 // [32][K]
    const int K = a.C * a.kh * a.kw;
    const int g = blockIdx.y;
    const int ochan = min(32, a.O - g * 32);
    for (int i = threadIdx.x; i < 32 * K; i += FIRST_NT) {
        const int oc = i / K, k = i - (i / K) * K;
        float v = 0.0f;
        if (oc < ochan) {
            const int o = g * 32 + oc;
            v = a.w[(long long)o * K + k];
            if (a.quant_w) {
                const float s = a.cscale ? a.cscale[o] : a.qw.scale;
                v = level_value(v * s, a.qw);
            }
        }
        sW[i] = v;
    }
    __syncthreads();

    const long long HoWo = (long long)a.Ho * a.Wo;
    const long long m = (long long)blockIdx.x * FIRST_NT + threadIdx.x;
    if (m >= (long long)a.B * HoWo) return;
    const int b = (int)(m / HoWo);
    const int pix = (int)(m - (long long)b * HoWo);
    const int yo = pix / a.Wo, xo = pix - (pix / a.Wo) * a.Wo;
    const int yb = yo * a.stride - a.pad, xb = xo * a.stride - a.pad;

    float acc[32];
#pragma unroll
    for (int o = 0; o < 32; ++o) acc[o] = 0.0f;
    int k = 0;
    for (int c = 0; c < a.C; ++c) {
        const float *xc = a.x + ((long long)b * a.C + c) * a.H * a.W;
        for (int ky = 0; ky < a.kh; ++ky) {
            const int yi = yb + ky;
            for (int kx = 0; kx < a.kw; ++kx, ++k) {
                const int xi = xb + kx;
                if (yi < 0 || yi >= a.H || xi < 0 || xi >= a.W) continue;
                const float xv = __ldg(xc + (long long)yi * a.W + xi);
#pragma unroll
                for (int o = 0; o < 32; ++o) acc[o] = fmaf(xv, sW[o * K + k], acc[o]);
            }
        }
    }

    uint32_t words[3] = {0u, 0u, 0u};
    uint32_t cw[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
#pragma unroll
    for (int oc = 0; oc < 32; ++oc) {
        if (oc < ochan) {
            const int o = g * 32 + oc;
            float y = fmaf(acc[oc], __ldg(a.scale + o), __ldg(a.shift + o));
            if (a.quant_out) {
                y = fminf(fmaxf(y, -1.0f), 1.0f);
                const int lv = level_units(y * a.qo.scale, a.qo);
                const uint32_t pb = level_plane_bits(lv, a.qo.bits);
                cw[oc >> 2] |= (uint32_t)level_code_e4m3(lv) << ((oc & 3) * 8);
                words[0] |= (pb & 1u) << oc;
                words[1] |= ((pb >> 1) & 1u) << oc;
                words[2] |= ((pb >> 2) & 1u) << oc;
            }
            if (a.y_out) a.y_out[((long long)b * a.O + o) * HoWo + pix] = y;
        }
    }
    if (a.quant_out && a.codes_out != nullptr) {
        uint4 *dst = reinterpret_cast<uint4 *>(a.codes_out + m * a.O + g * 32);
        dst[0] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
        if (ochan > 16) dst[1] = make_uint4(cw[4], cw[5], cw[6], cw[7]);
    }
    if (a.quant_out && a.planes_out != nullptr) {
        const int NWo = (a.O + 31) >> 5;
        uint32_t *dst = a.planes_out + (m * a.qo.bits) * NWo + g;
        for (int p = 0; p < a.qo.bits; ++p) dst[p * NWo] = words[p];
    }
}

minw_status launch_conv_first(const FirstArgs &a, cudaStream_t s) {
    const int K = a.C * a.kh * a.kw;
    const size_t smem = sizeof(float) * 32 * (size_t)K;
    if (smem > 200 * 1024) return MINW_EUNSUPPORTED;
    static int configured_bytes = 0;
    if ((int)smem > configured_bytes) {
        if (cudaFuncSetAttribute(conv_first_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem) != cudaSuccess)
            return MINW_ECUDA;
        configured_bytes = (int)smem;
    }
    const long long M = (long long)a.B * a.Ho * a.Wo;
    const dim3 grid((unsigned)((M + FIRST_NT - 1) / FIRST_NT), (unsigned)((a.O + 31) / 32));
    conv_first_kernel<<<grid, FIRST_NT, smem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

}  // namespace minw

using namespace minw;
using namespace minw_host;

extern "C" minw_status minw_conv_first(const float *x, int32_t B, int32_t C, int32_t H, int32_t W,
                                       const float *w, int32_t O, int32_t kh, int32_t kw,
                                       int32_t stride, int32_t pad, const minw_quant *q_w,
                                       const float *channel_scale, int32_t pool,
                                       const float *scale, const float *shift,
                                       const minw_quant *q_out, uint32_t *planes_out,
                                       float *y_out, void *stream) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || O <= 0 || kh <= 0 || kw <= 0 || stride <= 0 ||
        pad < 0)
        return MINW_EINVAL;
    if (!x || !w || !scale || !shift) return MINW_EINVAL;
    if (q_w && !valid_quant(q_w)) return MINW_EINVAL;
    if (q_out && (!valid_quant(q_out) || !planes_out)) return MINW_EINVAL;
    if (!q_out && !y_out) return MINW_EINVAL;
    if (pool) return MINW_EUNSUPPORTED;
    const int Ho = (H + 2 * pad - kh) / stride + 1;
    const int Wo = (W + 2 * pad - kw) / stride + 1;
    if (Ho <= 0 || Wo <= 0) return MINW_EINVAL;
    FirstArgs a{};
    a.x = x; a.w = w; a.cscale = channel_scale;
    a.quant_w = q_w != nullptr;
    if (q_w) a.qw = to_qparams(q_w);
    a.B = B; a.C = C; a.H = H; a.W = W; a.O = O; a.kh = kh; a.kw = kw;
    a.stride = stride; a.pad = pad; a.Ho = Ho; a.Wo = Wo;
    a.scale = scale; a.shift = shift;
    a.quant_out = q_out != nullptr;
    if (q_out) a.qo = to_qparams(q_out);
    a.planes_out = planes_out; a.y_out = y_out;
    return launch_conv_first(a, (cudaStream_t)stream);
}
