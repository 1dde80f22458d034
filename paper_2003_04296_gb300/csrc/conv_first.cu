// conv_first.cu -- the first layer of a MINW-Net (Sec. III-E): the fp32 image
// is not quantized, its weights are.  Each output is one fp32 fmaf chain over
// (c, ky, kx) in that order with padded taps skipped, so the result does not
// depend on the launch shape.  BN (fmaf), HardTanh and quantize + pack of the
// next layer's input are fused into the epilogue.
//
// See conv_first_kernel for the tiling.
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace minw {


constexpr int FIRST_NT = 128;
constexpr int FIRST_PPT = 4;                    // output pixels per thread
constexpr int FIRST_MAXPIX = FIRST_PPT * FIRST_NT;

template <int OUTB>
__device__ __forceinline__ uint32_t first_code(int k) {
    if constexpr (OUTB == 1) return k ? 0x38u : 0xB8u;
    else if constexpr (OUTB == 2) return (uint32_t)((0x3800B8u >> (8 * k)) & 0xFFu);
    else return (uint32_t)((0x0048403800B8C0C8ull >> (8 * k)) & 0xFFull);
}
template <int OUTB>
__device__ __forceinline__ uint32_t first_planes(int k) {
    if constexpr (OUTB == 1) return k ? 0u : 1u;
    else if constexpr (OUTB == 2) return (0x203u >> (4 * k)) & 0x3u;
    else return (uint32_t)((06420357ull >> (3 * k)) & 7ull);
}

struct FirstTile {
    int R;            // output rows per CTA
    int Rin, Win;     // input patch rows / columns (zero padded)
    size_t smem;      // bytes of dynamic shared memory
};

static FirstTile first_tile(const FirstArgs &a) {
    FirstTile t;
    t.R = FIRST_MAXPIX / a.Wo;
    if (t.R > a.Ho) t.R = a.Ho;
    if (t.R < 1) t.R = 1;
    t.Rin = (t.R - 1) * a.stride + a.kh;
    t.Win = (a.Wo - 1) * a.stride + a.kw;
    const int K = a.C * a.kh * a.kw;
    t.smem = sizeof(float) * (32 * (size_t)K + (size_t)a.C * t.Rin * t.Win + 32 * 8) + sizeof(int) * K;
    return t;
}

// A CTA owns R full output rows of one image (R * Wo <= 512 pixels) and one
// group of 32 output channels.  Its zero-padded input patch, the group's
// weights ([K][32]) and the tap offsets sit in shared memory; a thread holds
// four output pixels x 32 channels and per tap does four patch loads, eight
// 128-bit broadcast weight loads and 128 fmaf.  Zero padding: the accumulator
// starts at +0, a sum that rounds to zero is +0 in round-to-nearest, so it
// never becomes -0 and fmaf(0, w, acc) == acc exactly -- the same value as
// skipping the tap.  BN + HardTanh + quantize use exact fp32 breakpoints.
template <int OUTB>
__global__ void __launch_bounds__(FIRST_NT) conv_first_kernel(const FirstArgs a, const FirstTile tl) {
    extern __shared__ float4 smem4[];
    float *sW = reinterpret_cast<float *>(smem4);                 // [K][32]
    const int K = a.C * a.kh * a.kw;
    float *sX = sW + 32 * K;                                      // [C][Rin][Win]
    float *sT = sX + (size_t)a.C * tl.Rin * tl.Win;               // [32][8] breakpoints
    int *sOff = reinterpret_cast<int *>(sT + 32 * 8);             // [K] patch offsets

    const int g = blockIdx.y;
    const int ochan = min(32, a.O - g * 32);
    const int rblocks = (a.Ho + tl.R - 1) / tl.R;
    const int b = blockIdx.x / rblocks;
    const int oy0 = (blockIdx.x - b * rblocks) * tl.R;
    const int iy0 = oy0 * a.stride - a.pad, ix0 = -a.pad;

    for (int i = threadIdx.x; i < 32 * K; i += FIRST_NT) {
        const int k = i >> 5, oc = i & 31;
        float v = 0.0f;
        if (oc < ochan) {
            const int o = g * 32 + oc;
            v = a.w[(long long)o * K + k];
            if (a.quant_w) {
                const float sc = a.cscale ? a.cscale[o] : a.qw.scale;
                v = level_value(v * sc, a.qw);
            }
        }
        sW[i] = v;
    }
    const int plane = tl.Rin * tl.Win;
    for (int i = threadIdx.x; i < a.C * plane; i += FIRST_NT) {
        const int c = i / plane, rem = i - c * plane;
        const int ry = rem / tl.Win, rx = rem - ry * tl.Win;
        const int yi = iy0 + ry, xi = ix0 + rx;
        float v = 0.0f;
        if (yi >= 0 && yi < a.H && xi >= 0 && xi < a.W) v = __ldg(a.x + (((long long)b * a.C + c) * a.H + yi) * a.W + xi);
        sX[i] = v;
    }
    for (int k = threadIdx.x; k < K; k += FIRST_NT) {
        const int c = k / (a.kh * a.kw), r = k - c * a.kh * a.kw;
        const int ky = r / a.kw, kx = r - ky * a.kw;
        sOff[k] = c * plane + ky * tl.Win + kx;
    }
    if (a.quant_out && threadIdx.x < ochan) {
        const int o = g * 32 + threadIdx.x;
        if (a.thr != nullptr) {
#pragma unroll
            for (int u = 0; u < 8; ++u) sT[threadIdx.x * 8 + u] = __ldg(a.thr + o * 8 + u);
        } else {
            channel_thresholds_f32(__ldg(a.scale + o), __ldg(a.shift + o), a.qo, sT + threadIdx.x * 8);
        }
    }
    __syncthreads();

    const int npix = min(tl.R, a.Ho - oy0) * a.Wo;
    int base[FIRST_PPT];
    bool live[FIRST_PPT];
#pragma unroll
    for (int i = 0; i < FIRST_PPT; ++i) {
        const int pidx = threadIdx.x + i * FIRST_NT;
        live[i] = pidx < npix;
        const int ly = live[i] ? pidx / a.Wo : 0, lx = live[i] ? pidx - (pidx / a.Wo) * a.Wo : 0;
        base[i] = ly * a.stride * tl.Win + lx * a.stride;
    }
    if (!live[0]) return;

    float acc[FIRST_PPT][32];
#pragma unroll
    for (int i = 0; i < FIRST_PPT; ++i)
#pragma unroll
        for (int o = 0; o < 32; ++o) acc[i][o] = 0.0f;
    for (int k = 0; k < K; ++k) {
        const int off = sOff[k];
        float xv[FIRST_PPT];
#pragma unroll
        for (int i = 0; i < FIRST_PPT; ++i) xv[i] = sX[base[i] + off];
#pragma unroll
        for (int o4 = 0; o4 < 8; ++o4) {
            const float4 w = smem4[k * 8 + o4];
#pragma unroll
            for (int i = 0; i < FIRST_PPT; ++i) {
                acc[i][4 * o4 + 0] = fmaf(xv[i], w.x, acc[i][4 * o4 + 0]);
                acc[i][4 * o4 + 1] = fmaf(xv[i], w.y, acc[i][4 * o4 + 1]);
                acc[i][4 * o4 + 2] = fmaf(xv[i], w.z, acc[i][4 * o4 + 2]);
                acc[i][4 * o4 + 3] = fmaf(xv[i], w.w, acc[i][4 * o4 + 3]);
            }
        }
    }

    const long long HoWo = (long long)a.Ho * a.Wo;
    const int NWo = (a.O + 31) >> 5;
    constexpr int NL = OUTB == 0 ? 1 : (OUTB == 1 ? 2 : (OUTB == 2 ? 3 : 7));
#pragma unroll
    for (int i = 0; i < FIRST_PPT; ++i) {
        if (!live[i]) continue;
        const int pix = oy0 * a.Wo + threadIdx.x + i * FIRST_NT;
        const long long m = (long long)b * HoWo + pix;
        if (a.y_out) {
#pragma unroll
            for (int oc = 0; oc < 32; ++oc) {
                if (oc < ochan) {
                    const int o = g * 32 + oc;
                    float y = fmaf(acc[i][oc], __ldg(a.scale + o), __ldg(a.shift + o));
                    if (OUTB > 0) y = fminf(fmaxf(y, -1.0f), 1.0f);
                    a.y_out[((long long)b * a.O + o) * HoWo + pix] = y;
                }
            }
        }
        if constexpr (OUTB > 0) {
            int kq[32];
#pragma unroll
            for (int oc = 0; oc < 32; ++oc) {
                const float *th = sT + oc * 8;
                const float v = acc[i][oc] * th[NL - 1];
                int k = 0;
#pragma unroll
                for (int u = 0; u < NL - 1; ++u) k += (v >= th[u]) ? 1 : 0;
                kq[oc] = k;
            }
            if (a.codes_out != nullptr) {
                uint32_t cw[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
#pragma unroll
                for (int oc = 0; oc < 32; ++oc) cw[oc >> 2] |= first_code<OUTB>(kq[oc]) << ((oc & 3) * 8);
                uint4 *dst = reinterpret_cast<uint4 *>(a.codes_out + m * a.O + g * 32);
                dst[0] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
                if (ochan > 16) dst[1] = make_uint4(cw[4], cw[5], cw[6], cw[7]);
            }
            if (a.planes_out != nullptr) {
                uint32_t words[OUTB];
#pragma unroll
                for (int u = 0; u < OUTB; ++u) words[u] = 0u;
#pragma unroll
                for (int oc = 0; oc < 32; ++oc) {
                    const uint32_t pb = (oc < ochan) ? first_planes<OUTB>(kq[oc]) : 0u;
#pragma unroll
                    for (int u = 0; u < OUTB; ++u) words[u] |= ((pb >> u) & 1u) << oc;
                }
                uint32_t *dst = a.planes_out + (m * OUTB) * NWo + g;
#pragma unroll
                for (int u = 0; u < OUTB; ++u) dst[u * NWo] = words[u];
            }
        }
    }
}

// fp32 breakpoints of every channel, [O][8]: one thread per channel.
__global__ void thresholds_f32_kernel(const float *__restrict__ scale, const float *__restrict__ shift, int O,
                                      QParams q, float *__restrict__ out) {
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o < O) channel_thresholds_f32(scale[o], shift[o], q, out + o * 8);
}

minw_status launch_thresholds_f32(const float *scale, const float *shift, int O, const QParams &q, float *out,
                                  cudaStream_t s) {
    thresholds_f32_kernel<<<(O + 63) / 64, 64, 0, s>>>(scale, shift, O, q, out);
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

minw_status launch_conv_first(const FirstArgs &a, cudaStream_t s) {
    if (a.Wo > FIRST_MAXPIX) return MINW_EUNSUPPORTED;
    const FirstTile tl = first_tile(a);
    if (tl.smem > 200 * 1024) return MINW_EUNSUPPORTED;
    const int outb = a.quant_out ? a.qo.bits : 0;
    void (*kern)(const FirstArgs, const FirstTile) =
        outb == 1 ? conv_first_kernel<1> : outb == 2 ? conv_first_kernel<2> : outb == 3 ? conv_first_kernel<3>
                                                                                       : conv_first_kernel<0>;
    static size_t configured_bytes[4] = {0, 0, 0, 0};
    if (tl.smem > configured_bytes[outb]) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tl.smem) != cudaSuccess)
            return MINW_ECUDA;
        configured_bytes[outb] = tl.smem;
    }
    const int rblocks = (a.Ho + tl.R - 1) / tl.R;
    const dim3 grid((unsigned)(a.B * rblocks), (unsigned)((a.O + 31) / 32));
    kern<<<grid, FIRST_NT, tl.smem, s>>>(a, tl);
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
