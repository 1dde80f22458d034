// conv_first.cu -- the first layer of a MINW-Net (Sec. III-E): the fp32 image
// is not quantized, its weights are.  Each output is one fp32 fmaf chain over
// (c, ky, kx) in that order with padded taps skipped, so the result does not
// depend on the launch shape.  BN (fmaf), HardTanh and quantize + pack of the
// next layer's input are fused into the epilogue.  The same kernel runs the
// ResNet stem (7x7 / 2, fp32 weights).
//
// See conv_first_kernel for the tiling.
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace minw {


constexpr int FIRST_NT = 256;                   // 8 warps
constexpr int FIRST_PX = 4;                     // output pixels per thread (16 apart)

// Two fp32 lanes in one 64-bit register for the packed fma.rn.f32x2: each
// lane is an IEEE fmaf of its own, so a chain of them is bit-identical to
// the scalar chain.
__device__ __forceinline__ unsigned long long dup2(float x) {
    unsigned long long r;
    asm("mov.b64 %0, {%1, %1};" : "=l"(r) : "f"(x));
    return r;
}
__device__ __forceinline__ void ffma2(unsigned long long &acc, unsigned long long a, unsigned long long b) {
    asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(acc) : "l"(a), "l"(b));
}
__device__ __forceinline__ float lane2(unsigned long long v, int hi) {
    float lo_, hi_;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo_), "=f"(hi_) : "l"(v));
    return hi ? hi_ : lo_;
}

struct FirstTile {
    int OCB;          // output channels per CTA (32 or 64)
    int groups;       // 32-channel groups per CTA
    int PB;           // output pixels per CTA (64 per pixel block, 8 / groups blocks)
    int tiles;        // CTAs along the pixels of one image
    int Rmax;         // input patch rows
    int Ws;           // patch columns per stride phase
    int RP;           // patch row pitch (stride x Ws)
    int K;            // C x kh x kw
    int nb;           // input patch buffers (2 or 3: the patch of tile t + (nb - 1) G is in flight)
    size_t smem;      // bytes of dynamic shared memory
};

static FirstTile first_tile(const FirstArgs &a) {
    FirstTile t;
    t.OCB = a.O > 32 ? 64 : 32;
    t.groups = t.OCB / 32;
    t.PB = 64 * (8 / t.groups);
    const int npix = a.Ho * a.Wo;
    t.tiles = (npix + t.PB - 1) / t.PB;
    const int rows = min(a.Ho, (t.PB + a.Wo - 2) / a.Wo + 1);      // rows PB consecutive pixels can touch
    t.Rmax = (rows - 1) * a.stride + a.kh;
    const int Win = (a.Wo - 1) * a.stride + a.kw;
    t.Ws = (Win + a.stride - 1) / a.stride;
    t.RP = t.Ws * a.stride;
    t.K = a.C * a.kh * a.kw;
    // three patch buffers (two tiles of look-ahead) where two CTAs still fit on an SM
    const size_t fixed = sizeof(float) * ((size_t)t.K * t.OCB + (size_t)t.OCB * 8);
    const size_t pbytes = sizeof(float) * (size_t)a.C * t.Rmax * t.RP;
    t.nb = fixed + 3 * pbytes <= 112 * 1024 ? 3 : 2;
    t.smem = fixed + t.nb * pbytes;
    return t;
}

// 4-byte asynchronous global -> shared copy; src_bytes = 0 writes a zero.
__device__ __forceinline__ void cp_async4(float *dst, const float *src, int src_bytes) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"((uint32_t)__cvta_generic_to_shared(dst)),
                 "l"(src), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// Persistent CTAs own 32 or 64 output channels and walk pixel tiles of PB
// consecutive output pixels (row-major within one image).  Shared memory
// holds the weights [K][OCB] and breakpoints, loaded once, and two input
// patches [C][rows][columns] (zero padded; columns split by stride phase, column
// rx at (rx % S) * Ws + rx / S, so that threads reading neighbouring output
// pixels read neighbouring words for any stride): the next tile's patch
// arrives by cp.async while the current one is computed (and, where shared
// memory allows, the one after it: a small patch takes about as long to
// arrive as a tile takes to compute).  Warp = 32 output
// channels x 64 pixels; a thread holds four pixels (16 apart) x 16 channels
// as 8 channel pairs and per tap does four patch loads, four 128-bit weight
// loads (one address per half warp) and 32 packed fma.rn.f32x2, one fmaf
// chain per output over (c, ky, kx) in that order.  Zero padding: the accumulator starts at +0 and
// a sum that rounds to zero is +0, so it is never -0 and fmaf(0, w, acc) ==
// acc: the padded taps change nothing, exactly as skipping them.  The
// epilogue turns each pixel's 32 channels into level masks (the sign bits of
// fmaf(acc, sigma, -T)) and stores planes or codes from them.  KH, KW, S = 0:
// runtime shape.
template <int OUTB, int KH, int KW, int S>
__global__ void __launch_bounds__(FIRST_NT, 2) conv_first_kernel(const FirstArgs a, const FirstTile tl) {
    extern __shared__ float4 smem4[];
    const int kh = KH ? KH : a.kh, kw = KW ? KW : a.kw, st = S ? S : a.stride;
    const int OCB = tl.OCB, K = tl.K, RP = tl.RP, Ws = tl.Ws;
    const size_t patch = (size_t)a.C * tl.Rmax * RP;
    float *sW = reinterpret_cast<float *>(smem4);                 // [K][OCB]
    float *sT = sW + (size_t)K * OCB;                             // [OCB][8] -breakpoints, sigma
    float *sX0 = sT + OCB * 8;                                    // [nb][C][Rmax][RP]

    const int o0 = blockIdx.y * OCB;
    const int ochan = min(OCB, a.O - o0);
    const int npix = a.Ho * a.Wo;
    const int Win = (a.Wo - 1) * st + kw;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int total = a.B * tl.tiles;

    // asynchronous load of tile t's input patch into buffer buf
    auto load_patch = [&](int t, int buf) {
        const int b = t / tl.tiles;
        const int p0 = (t - b * tl.tiles) * tl.PB;
        const int pend = min(p0 + tl.PB, npix);
        const int y_first = p0 / a.Wo, y_last = (pend - 1) / a.Wo;
        const int rows_in = (y_last - y_first) * st + kh;
        const int iy0 = y_first * st - a.pad, ix0 = -a.pad;
        float *sX = sX0 + buf * patch;
        for (int cr = warp; cr < a.C * rows_in; cr += FIRST_NT / 32) {
            const int c = cr / rows_in, r = cr - c * rows_in;
            const int yi = iy0 + r;
            const bool row_ok = yi >= 0 && yi < a.H;
            const float *src = a.x + (((long long)b * a.C + c) * a.H + (row_ok ? yi : 0)) * a.W;
            float *dst = sX + ((size_t)c * tl.Rmax + r) * RP;
            for (int rx = lane; rx < Win; rx += 32) {
                const int xi = ix0 + rx;
                const bool ok = row_ok && xi >= 0 && xi < a.W;
                cp_async4(dst + (rx % st) * Ws + rx / st, ok ? src + xi : src, ok ? 4 : 0);
            }
        }
        cp_async_commit();
    };

    int t = blockIdx.x;

    // weights: prepared [K][O] levels (coalesced), else the latent [O][K] array
    const int osh = OCB == 64 ? 6 : 5;
    for (int i = threadIdx.x; i < K * OCB; i += FIRST_NT) {
        const int k = i >> osh, oc = i & (OCB - 1);
        float v = 0.0f;
        if (oc < ochan) {
            const int o = o0 + oc;
            if (a.wt != nullptr) {
                v = __ldg(a.wt + (long long)k * a.O + o);
            } else {
                v = __ldg(a.w + (long long)o * K + k);
                if (a.quant_w) v = level_value(v * (a.cscale ? __ldg(a.cscale + o) : a.qw.scale), a.qw);
            }
        }
        sW[i] = v;
    }
    // breakpoints held for the mask test: (-T_1 .. -T_{n-1}, sigma); padding channels never reached
    if (a.quant_out && threadIdx.x < OCB) {
        float *th = sT + threadIdx.x * 8;
        const int o = o0 + threadIdx.x;
        const int nl = num_levels(a.qo.bits);
        if (threadIdx.x >= ochan) {
            for (int u = 0; u < 8; ++u) th[u] = u == nl - 1 ? 1.0f : -INFINITY;
        } else {
            if (a.thr != nullptr) {
#pragma unroll
                for (int u = 0; u < 8; ++u) th[u] = __ldg(a.thr + o * 8 + u);
            } else {
                channel_thresholds_f32(__ldg(a.scale + o), __ldg(a.shift + o), a.qo, th);
            }
            for (int u = 0; u < nl - 1; ++u) th[u] = mask_breakpoint(th[u]);
        }
    }

    // warp = 32 channels x 64 pixels; lane = (channel half h, pixel l16):
    // 4 pixels (16 apart) x 16 channels per thread
    pdl_trigger();                                               // set-up done
    pdl_wait();                                                  // the image and the output buffer are shared
    // one cp.async group per tile slot (empty past the end), so that the wait count is fixed
    const int nb = tl.nb;
    for (int j = 0; j < nb - 1; ++j) {
        if (t + j * (int)gridDim.x < total)
            load_patch(t + j * (int)gridDim.x, j);
        else
            cp_async_commit();
    }
    const int g = warp % tl.groups, pb = warp / tl.groups;
    const int h = lane >> 4, l16 = lane & 15;
    const int NWo = (a.O + 31) >> 5;
    const int gch = min(32, ochan - g * 32);                     // live channels of this warp (may be <= 0)
    const int hch = gch - 16 * h;                                // live channels of this half (may be <= 0)
    const int ob = o0 + g * 32;
    const float *wg = sW + g * 32 + h * 16;
    constexpr int NL = OUTB == 0 ? 1 : (OUTB == 1 ? 2 : (OUTB == 2 ? 3 : 7));
    for (int buf = 0; t < total; t += gridDim.x, buf = buf + 1 == nb ? 0 : buf + 1) {
        const int tn = t + (nb - 1) * (int)gridDim.x;
        const int bn = buf == 0 ? nb - 1 : buf - 1;              // the slot tile t - G used
        if (tn < total)
            load_patch(tn, bn);
        else
            cp_async_commit();
        if (nb == 3)
            cp_async_wait<2>();
        else
            cp_async_wait<1>();
        __syncthreads();                                         // patch t (and the weights) visible

        const int b = t / tl.tiles;
        const int p0 = (t - b * tl.tiles) * tl.PB;
        const int pend = min(p0 + tl.PB, npix);
        const int y_first = p0 / a.Wo;
        const float *sX = sX0 + buf * patch;
        int pofs[FIRST_PX], pix[FIRST_PX];
        bool live[FIRST_PX];
#pragma unroll
        for (int i = 0; i < FIRST_PX; ++i) {
            const int p = p0 + pb * 64 + l16 + 16 * i;
            live[i] = p < pend;
            pix[i] = live[i] ? p : p0;
            const int yy = pix[i] / a.Wo, xx = pix[i] - yy * a.Wo;
            pofs[i] = (yy - y_first) * st * RP + xx;
        }
        if (p0 + pb * 64 < pend && gch > 0) {                   // warp-uniform: the epilogue shuffles
            // accumulators of channel pairs (2j, 2j + 1), packed for fma.rn.f32x2
            unsigned long long acc[FIRST_PX][8];
#pragma unroll
            for (int i = 0; i < FIRST_PX; ++i)
#pragma unroll
                for (int o = 0; o < 8; ++o) acc[i][o] = 0ull;
            for (int c = 0; c < a.C; ++c) {
#pragma unroll (KH ? KH : 1)
                for (int ky = 0; ky < kh; ++ky) {
                    const float *xrow = sX + ((size_t)c * tl.Rmax + ky) * RP;
                    const float *wrow = wg + (size_t)((c * kh + ky) * kw) * OCB;
                    const float *xp[FIRST_PX];
#pragma unroll
                    for (int i = 0; i < FIRST_PX; ++i) xp[i] = xrow + pofs[i];
#pragma unroll (KW ? KW : 1)
                    for (int kx = 0; kx < kw; ++kx) {
                        // tap column kx: stride phase kx % S, offset kx / S within the phase
                        const int ph = kx % st, xo = kx / st;
                        unsigned long long xv[FIRST_PX];
#pragma unroll
                        for (int i = 0; i < FIRST_PX; ++i) xv[i] = dup2((ph == 0 ? xp[i] : xp[i] + ph * Ws)[xo]);
                        const ulonglong2 *w2 = reinterpret_cast<const ulonglong2 *>(wrow + kx * OCB);
#pragma unroll
                        for (int o4 = 0; o4 < 4; ++o4) {
                            const ulonglong2 w = w2[o4];
#pragma unroll
                            for (int i = 0; i < FIRST_PX; ++i) {
                                ffma2(acc[i][2 * o4], xv[i], w.x);
                                ffma2(acc[i][2 * o4 + 1], xv[i], w.y);
                            }
                        }
                    }
                }
            }

            if (a.y_out) {
#pragma unroll
                for (int i = 0; i < FIRST_PX; ++i) {
                    if (!live[i]) continue;
#pragma unroll
                    for (int oc = 0; oc < 16; ++oc) {
                        if (oc < hch) {
                            const int o = ob + 16 * h + oc;
                            float y = fmaf(lane2(acc[i][oc >> 1], oc & 1), __ldg(a.scale + o), __ldg(a.shift + o));
                            if (OUTB > 0) y = fminf(fmaxf(y, -1.0f), 1.0f);
                            a.y_out[((long long)b * a.O + o) * npix + pix[i]] = y;
                        }
                    }
                }
            }
            if constexpr (OUTB > 0) {
                // level masks of this half's 16 channels: bit oc of M = [sigma * acc < T_u], from the
                // sign of fmaf(acc, sigma, -T_u); then the two halves make the 32-channel word
                const float *thb = sT + (g * 32 + 16 * h) * 8;
                uint32_t MM[FIRST_PX][NL - 1];
#pragma unroll
                for (int i = 0; i < FIRST_PX; ++i)
#pragma unroll
                    for (int u = 0; u < NL - 1; ++u) MM[i][u] = 0u;
#pragma unroll
                for (int oc = 15; oc >= 0; --oc) {
                    const float *th = thb + oc * 8;
                    const float sg = th[NL - 1];
#pragma unroll
                    for (int u = 0; u < NL - 1; ++u) {
                        const float nt = th[u];
#pragma unroll
                        for (int i = 0; i < FIRST_PX; ++i)
                            MM[i][u] = __funnelshift_l(__float_as_uint(fmaf(lane2(acc[i][oc >> 1], oc & 1), sg, nt)),
                                                       MM[i][u], 1);
                    }
                }
#pragma unroll
                for (int i = 0; i < FIRST_PX; ++i) {
                    uint32_t *M = MM[i];
#pragma unroll
                    for (int u = 0; u < NL - 1; ++u) {
                        const uint32_t other = __shfl_xor_sync(0xffffffffu, M[u], 16);
                        M[u] = h ? (other | (M[u] << 16)) : (M[u] | (other << 16));
                    }
                    if (!live[i]) continue;
                    const long long m = (long long)b * npix + pix[i];
                    uint32_t P[3];
                    level_planes<OUTB>(M, P);
                    if (a.planes_out != nullptr && h == 0) {
                        const uint32_t vm = gch >= 32 ? 0xffffffffu : ((1u << gch) - 1u);
                        uint32_t *dst = a.planes_out + (m * OUTB) * NWo + (ob >> 5);
#pragma unroll
                        for (int u = 0; u < OUTB; ++u) dst[u * NWo] = P[u] & vm;
                    }
                    if (a.codes_out != nullptr && hch > 0)
                        *reinterpret_cast<uint4 *>(a.codes_out + m * a.O + ob + 16 * h) =
                            make_uint4(level_code_word<OUTB>(P, 4 * h), level_code_word<OUTB>(P, 4 * h + 1),
                                       level_code_word<OUTB>(P, 4 * h + 2), level_code_word<OUTB>(P, 4 * h + 3));
                }
            }
        }
        __syncthreads();                                         // buffer buf is free for tile t + nb G
    }
}

// Weights of a first layer prepared once: [K][O] (output channel fastest),
// quantized to their levels with the per-channel prescale when quant_w.
__global__ void first_weights_kernel(const float *__restrict__ w, int O, int K, int quant_w, QParams qw,
                                     const float *__restrict__ cscale, float *__restrict__ wt) {
    const long long n = (long long)O * K;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const int o = (int)(i / K), k = (int)(i - (long long)o * K);
        float v = w[i];
        if (quant_w) v = level_value(v * (cscale ? cscale[o] : qw.scale), qw);
        wt[(long long)k * O + o] = v;
    }
}

minw_status launch_first_weights(const float *w, int O, int K, int quant_w, const QParams &qw, const float *cscale,
                                 float *wt, cudaStream_t s) {
    first_weights_kernel<<<256, 256, 0, s>>>(w, O, K, quant_w, qw, cscale, wt);
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

// fp32 breakpoints of every channel, [O][8]: one thread per channel.
__global__ void thresholds_f32_kernel(const float *__restrict__ scale, const float *__restrict__ shift, int O,
                                      QParams q, float *__restrict__ out) {
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o < O) channel_thresholds_f32(scale[o], shift[o], q, out + o * 8);
}

// Breakpoints of a quantizer on its input y itself (HardTanh included): the
// level index of y is #{u : y >= out[u]}.
__global__ void ythresholds_kernel(QParams q, float *__restrict__ out) {
    if (threadIdx.x == 0 && blockIdx.x == 0) channel_thresholds_f32(1.0f, 0.0f, q, out);
}

minw_status launch_ythresholds(const QParams &q, float *out, cudaStream_t s) {
    ythresholds_kernel<<<1, 32, 0, s>>>(q, out);
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

minw_status launch_thresholds_f32(const float *scale, const float *shift, int O, const QParams &q, float *out,
                                  cudaStream_t s) {
    thresholds_f32_kernel<<<(O + 63) / 64, 64, 0, s>>>(scale, shift, O, q, out);
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

template <int OUTB, int KH, int KW, int S>
static minw_status launch_first_shape(const FirstArgs &a, const FirstTile &tl, cudaStream_t s) {
    static size_t configured = 0;
    void (*kern)(const FirstArgs, const FirstTile) = conv_first_kernel<OUTB, KH, KW, S>;
    if (tl.smem > configured) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tl.smem) != cudaSuccess)
            return MINW_ECUDA;
        configured = tl.smem;
    }
    // persistent: two CTAs per SM over all channel tiles
    const int octiles = (a.O + tl.OCB - 1) / tl.OCB;
    const int sms = minw_host::num_sms() > 0 ? minw_host::num_sms() : 152;
    const int total = a.B * tl.tiles;
    int gx = (2 * sms + octiles - 1) / octiles;
    if (gx > total) gx = total;
    const dim3 grid((unsigned)gx, (unsigned)octiles);
    if (minw_host::launch_pdl(kern, grid, dim3(FIRST_NT), tl.smem, s, a, tl) != cudaSuccess) return MINW_ECUDA;
    return MINW_OK;
}

template <int OUTB>
static minw_status launch_first_bits(const FirstArgs &a, const FirstTile &tl, cudaStream_t s) {
    if (a.kh == 3 && a.kw == 3 && a.stride == 1) return launch_first_shape<OUTB, 3, 3, 1>(a, tl, s);
    if (a.kh == 7 && a.kw == 7 && a.stride == 2) return launch_first_shape<OUTB, 7, 7, 2>(a, tl, s);
    return launch_first_shape<OUTB, 0, 0, 0>(a, tl, s);
}

minw_status launch_conv_first(const FirstArgs &a, cudaStream_t s) {
    const FirstTile tl = first_tile(a);
    if (tl.smem > 200 * 1024) return MINW_EUNSUPPORTED;
    if (a.codes_out != nullptr && a.O % 16 != 0) return MINW_EUNSUPPORTED;
    const int outb = a.quant_out ? a.qo.bits : 0;
    switch (outb) {
        case 1: return launch_first_bits<1>(a, tl, s);
        case 2: return launch_first_bits<2>(a, tl, s);
        case 3: return launch_first_bits<3>(a, tl, s);
        default: return launch_first_bits<0>(a, tl, s);
    }
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
