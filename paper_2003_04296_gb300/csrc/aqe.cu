// aqe.cu -- AQE elementwise kernels (Eq. ours, Eq. activation, Eq. weight),
// the fused quantize + bit-plane pack of activations (Eq. inference) and the
// packing of latent weights.  All of them stream HBM: 128-bit loads where the
// layout allows, grids sized from the SM count.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdlib.h>

#include "common.cuh"

namespace minw {

// ---------------------------------------------------------------------------
// AQE forward / backward, flat fp32 arrays.
// ---------------------------------------------------------------------------

__device__ __forceinline__ float aqe_fwd1(float x, float alpha, float oma, const QParams &q) {
    const float h = level_value(x * q.scale, q);
    return fmaf(alpha, h, oma * x);
}

__global__ void __launch_bounds__(256) aqe_forward_kernel(const float *__restrict__ x,
                                                          float *__restrict__ y, int64_t n,
                                                          float alpha, float oma, QParams q) {
    const int64_t n4 = n >> 2;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const float4 *x4 = reinterpret_cast<const float4 *>(x);
    float4 *y4 = reinterpret_cast<float4 *>(y);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
        float4 v = __ldcs(x4 + i);
        float4 r;
        r.x = aqe_fwd1(v.x, alpha, oma, q);
        r.y = aqe_fwd1(v.y, alpha, oma, q);
        r.z = aqe_fwd1(v.z, alpha, oma, q);
        r.w = aqe_fwd1(v.w, alpha, oma, q);
        __stcs(y4 + i, r);
    }
    for (int64_t i = (n4 << 2) + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        y[i] = aqe_fwd1(x[i], alpha, oma, q);
}

// ---------------------------------------------------------------------------
// Stochastic AQE (Eq. our): alpha sign(a - z) + (1 - alpha) a with z ~ U[-1, 1)
// from a counter-based generator, so that any element's noise is a pure
// function of (seed, offset, index).
// ---------------------------------------------------------------------------

// Philox4x64-10 (Salmon, Moraes, Dror, Shaw, SC 2011): ten rounds of two
// 64 x 64 -> 128-bit products on the counter, the key bumped by the Weyl
// constants between rounds.
__device__ __forceinline__ void philox4x64_10(uint64_t c[4], uint64_t k0, uint64_t k1) {
    const uint64_t M0 = 0xD2E7470EE14C6C93ull, M1 = 0xCA5A826395121157ull;
    const uint64_t W0 = 0x9E3779B97F4A7C15ull, W1 = 0xBB67AE8584CAA73Bull;
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint64_t hi0 = __umul64hi(M0, c[0]), lo0 = M0 * c[0];
        const uint64_t hi1 = __umul64hi(M1, c[2]), lo1 = M1 * c[2];
        const uint64_t n0 = hi1 ^ c[1] ^ k0, n2 = hi0 ^ c[3] ^ k1;
        c[0] = n0;
        c[1] = lo1;
        c[2] = n2;
        c[3] = lo0;
        k0 += W0;
        k1 += W1;
    }
}

// z = (u >> 8) 2^-23 - 1: a point of the 2^-23 grid on [-1, 1), exact in fp32.
__device__ __forceinline__ float noise_of(uint32_t u) { return (float)(u >> 8) * 1.1920928955078125e-7f - 1.0f; }

__device__ __forceinline__ float aqe_sto1(float x, float z, float alpha, float oma) {
    return fmaf(alpha, x > z ? 1.0f : -1.0f, oma * x);      // sign(x - z), sign(0) = -1
}

// Thread = one block of eight elements: one Philox4x64-10 call (counter
// offset + block, key (seed, 0)) gives the eight 32-bit noise words, low half
// of each 64-bit output first; two 128-bit loads and stores.
__global__ void __launch_bounds__(256) aqe_forward_stochastic_kernel(const float *__restrict__ x,
                                                                     float *__restrict__ y, int64_t n,
                                                                     float alpha, float oma, uint64_t seed,
                                                                     uint64_t offset) {
    const int64_t nb = (n + 7) >> 3;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < nb; b += stride) {
        const int64_t i0 = b << 3;
        const bool whole = i0 + 8 <= n;
        // the loads first, so that they are in flight during the generator's rounds
        float v[8];
        if (whole) {
            const float4 *x4 = reinterpret_cast<const float4 *>(x + i0);
            const float4 v0 = __ldcs(x4), v1 = __ldcs(x4 + 1);
            v[0] = v0.x; v[1] = v0.y; v[2] = v0.z; v[3] = v0.w;
            v[4] = v1.x; v[5] = v1.y; v[6] = v1.z; v[7] = v1.w;
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = i0 + j < n ? x[i0 + j] : 0.0f;
        }
        uint64_t c[4] = {offset + (uint64_t)b, 0ull, 0ull, 0ull};
        philox4x64_10(c, seed, 0ull);
        float r[8];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            r[2 * j] = aqe_sto1(v[2 * j], noise_of((uint32_t)c[j]), alpha, oma);
            r[2 * j + 1] = aqe_sto1(v[2 * j + 1], noise_of((uint32_t)(c[j] >> 32)), alpha, oma);
        }
        if (whole) {
            float4 *y4 = reinterpret_cast<float4 *>(y + i0);
            __stcs(y4, make_float4(r[0], r[1], r[2], r[3]));
            __stcs(y4 + 1, make_float4(r[4], r[5], r[6], r[7]));
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (i0 + j < n) y[i0 + j] = r[j];
        }
    }
}

__device__ __forceinline__ float aqe_bwd1(float x, float g, float two_alpha) {
    return (fabsf(x) <= 1.0f) ? g * two_alpha : 0.0f;
}

__global__ void __launch_bounds__(256) aqe_backward_kernel(const float *__restrict__ x,
                                                           const float *gy, float *gx,
                                                           int64_t n, float two_alpha) {
    const int64_t n4 = n >> 2;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const float4 *x4 = reinterpret_cast<const float4 *>(x);
    const float4 *g4 = reinterpret_cast<const float4 *>(gy);
    float4 *o4 = reinterpret_cast<float4 *>(gx);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
        float4 v = __ldcs(x4 + i);
        float4 g = __ldcs(g4 + i);
        float4 r;
        r.x = aqe_bwd1(v.x, g.x, two_alpha);
        r.y = aqe_bwd1(v.y, g.y, two_alpha);
        r.z = aqe_bwd1(v.z, g.z, two_alpha);
        r.w = aqe_bwd1(v.w, g.w, two_alpha);
        __stcs(o4 + i, r);
    }
    for (int64_t i = (n4 << 2) + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        gx[i] = aqe_bwd1(x[i], gy[i], two_alpha);
}

__global__ void __launch_bounds__(256) aqe_backward_masked_kernel(const uint32_t *__restrict__ mask,
                                                                  const float *gy, float *gx,
                                                                  int64_t n, float two_alpha) {
    const int64_t n4 = n >> 2;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const float4 *g4 = reinterpret_cast<const float4 *>(gy);
    float4 *o4 = reinterpret_cast<float4 *>(gx);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
        const uint32_t m = __ldg(mask + (i >> 3)) >> ((i & 7) * 4);
        float4 g = __ldcs(g4 + i);
        float4 r;
        r.x = (m & 1u) ? g.x * two_alpha : 0.0f;
        r.y = (m & 2u) ? g.y * two_alpha : 0.0f;
        r.z = (m & 4u) ? g.z * two_alpha : 0.0f;
        r.w = (m & 8u) ? g.w * two_alpha : 0.0f;
        __stcs(o4 + i, r);
    }
    for (int64_t i = (n4 << 2) + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const uint32_t m = (mask[i >> 5] >> (i & 31)) & 1u;
        gx[i] = m ? gy[i] * two_alpha : 0.0f;
    }
}

// ---------------------------------------------------------------------------
// Quantize + pack of NCHW activations into [B][H][W][P][NW] planes, with the
// AQE forward output and the |x| <= 1 mask of the backward produced from the
// same load of x.
//
// One warp owns 32 channels x 128 pixels of one image: lane l holds pixels
// p0 + 4l .. p0 + 4l + 3 and reads them with one 128-bit load per channel, so
// every load instruction of the warp covers 512 contiguous bytes.  A lane
// owns whole output words (32 channels of one pixel), so no transpose is
// needed.  Requires HW % 4 == 0 (16-byte aligned channel rows).
// ---------------------------------------------------------------------------

template <int P>
__global__ void __launch_bounds__(256) quantize_pack_vec_kernel(
    const float *__restrict__ x, int B, int C, int HW, QParams q, uint32_t *__restrict__ planes,
    float alpha, float oma, float *__restrict__ y, uint32_t *__restrict__ mask, int mask_atomic) {
    const int NW = (C + 31) >> 5;
    const int chunks = (HW + 127) >> 7;               // 128-pixel chunks per image
    const int lane = threadIdx.x & 31;
    const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t total = (int64_t)B * NW * chunks;
    for (int64_t t = warp; t < total; t += nwarps) {
        const int chunk = (int)(t % chunks);
        const int cw = (int)((t / chunks) % NW);
        const int b = (int)(t / ((int64_t)chunks * NW));
        const int p = chunk * 128 + lane * 4;          // first pixel of this lane
        const bool live = p < HW;                      // HW % 4 == 0: all 4 or none
        uint32_t w[4][P];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int k = 0; k < P; ++k) w[i][k] = 0u;
        const int cmax = min(32, C - cw * 32);
        for (int c = 0; c < cmax; ++c) {
            const int ch = cw * 32 + c;
            const int64_t off = ((int64_t)b * C + ch) * HW + p;
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (live) v = __ldcs(reinterpret_cast<const float4 *>(x + off));
            const float vv[4] = {v.x, v.y, v.z, v.w};
            uint32_t mbits = 0u;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int lv = level_units(vv[i] * q.scale, q);
                const uint32_t pb = level_plane_bits(lv, P);
#pragma unroll
                for (int k = 0; k < P; ++k) w[i][k] |= ((pb >> k) & 1u) << c;
                mbits |= (fabsf(vv[i]) <= 1.0f ? 1u : 0u) << i;
            }
            if (y != nullptr && live) {
                const float hs = (P == 3) ? 0.25f : 1.0f;
                float4 r;
                r.x = fmaf(alpha, hs * (float)level_units(v.x * q.scale, q), oma * v.x);
                r.y = fmaf(alpha, hs * (float)level_units(v.y * q.scale, q), oma * v.y);
                r.z = fmaf(alpha, hs * (float)level_units(v.z * q.scale, q), oma * v.z);
                r.w = fmaf(alpha, hs * (float)level_units(v.w * q.scale, q), oma * v.w);
                __stcs(reinterpret_cast<float4 *>(y + off), r);
            }
            if (mask != nullptr) {
                if (!mask_atomic) {
                    // HW % 32 == 0: 8 lanes cover one 32-bit mask word
                    uint32_t mw = mbits << ((lane & 7) * 4);
                    mw |= __shfl_xor_sync(0xffffffffu, mw, 1);
                    mw |= __shfl_xor_sync(0xffffffffu, mw, 2);
                    mw |= __shfl_xor_sync(0xffffffffu, mw, 4);
                    if (live && (lane & 7) == 0) mask[off >> 5] = mw;
                } else if (live && mbits) {
                    atomicOr(mask + (off >> 5), mbits << (off & 31));
                }
            }
        }
        if (live) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                uint32_t *dst = planes + ((int64_t)b * HW + p + i) * (P * NW) + cw;
#pragma unroll
                for (int k = 0; k < P; ++k) dst[k * NW] = w[i][k];
            }
        }
    }
}

// Scalar variant for HW % 4 != 0: lane l owns pixel p0 + l.
template <int P>
__global__ void __launch_bounds__(256) quantize_pack_scalar_kernel(
    const float *__restrict__ x, int B, int C, int HW, QParams q, uint32_t *__restrict__ planes,
    float alpha, float oma, float *__restrict__ y, uint32_t *__restrict__ mask) {
    const int NW = (C + 31) >> 5;
    const int chunks = (HW + 31) >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t total = (int64_t)B * NW * chunks;
    for (int64_t t = warp; t < total; t += nwarps) {
        const int chunk = (int)(t % chunks);
        const int cw = (int)((t / chunks) % NW);
        const int b = (int)(t / ((int64_t)chunks * NW));
        const int p = chunk * 32 + lane;
        const bool live = p < HW;
        uint32_t w[P];
#pragma unroll
        for (int k = 0; k < P; ++k) w[k] = 0u;
        const int cmax = min(32, C - cw * 32);
        for (int c = 0; c < cmax; ++c) {
            const int64_t off = ((int64_t)b * C + cw * 32 + c) * HW + p;
            if (!live) continue;
            const float v = __ldcs(x + off);
            const int lv = level_units(v * q.scale, q);
            const uint32_t pb = level_plane_bits(lv, P);
#pragma unroll
            for (int k = 0; k < P; ++k) w[k] |= ((pb >> k) & 1u) << c;
            if (y != nullptr) {
                const float hs = (P == 3) ? 0.25f : 1.0f;
                y[off] = fmaf(alpha, hs * (float)lv, oma * v);
            }
            if (mask != nullptr && fabsf(v) <= 1.0f) atomicOr(mask + (off >> 5), 1u << (off & 31));
        }
        if (live) {
            uint32_t *dst = planes + ((int64_t)b * HW + p) * (P * NW) + cw;
#pragma unroll
            for (int k = 0; k < P; ++k) dst[k * NW] = w[k];
        }
    }
}

// ---------------------------------------------------------------------------
// Weight packing: [O][C][kh][kw] -> [O][kh][kw][P][NW]; one thread per output
// word (the tensor is small and read once).
// ---------------------------------------------------------------------------

template <int P>
__global__ void pack_weights_kernel(const float *__restrict__ w, int O, int C, int kh, int kw,
                                    QParams q, const float *__restrict__ cscale,
                                    uint32_t *__restrict__ planes) {
    const int NW = (C + 31) >> 5;
    const int64_t total = (int64_t)O * kh * kw * NW;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int cw = (int)(t % NW);
        const int tap = (int)((t / NW) % (kh * kw));
        const int o = (int)(t / ((int64_t)NW * kh * kw));
        const float s = cscale ? cscale[o] : q.scale;
        uint32_t wd[P];
#pragma unroll
        for (int k = 0; k < P; ++k) wd[k] = 0u;
        const int cmax = min(32, C - cw * 32);
        for (int c = 0; c < cmax; ++c) {
            const float v = w[((int64_t)o * C + cw * 32 + c) * (kh * kw) + tap];
            const uint32_t pb = level_plane_bits(level_units(v * s, q), P);
#pragma unroll
            for (int k = 0; k < P; ++k) wd[k] |= ((pb >> k) & 1u) << c;
        }
        uint32_t *dst = planes + ((int64_t)o * kh * kw + tap) * (P * NW) + cw;
#pragma unroll
        for (int k = 0; k < P; ++k) dst[k * NW] = wd[k];
    }
}

// ---------------------------------------------------------------------------
// Level codes: NCHW fp32 -> NHWC bytes (E4M3 levels), the tensor-core operand.
// One warp owns 32 pixels x 32 channels of an image: lane l reads pixel p0+l of
// each channel (coalesced along the row) and writes its 32 channel bytes with
// two 16-byte stores.  C % 16 == 0.  With FP4 the codes are E2M1 nibbles, two
// channels per byte (16 bytes per lane; C % 32 == 0).
// ---------------------------------------------------------------------------

template <bool FP4>
__global__ void __launch_bounds__(256) quantize_codes_kernel(const float *__restrict__ x, int B, int C,
                                                             int HW, QParams q, uint8_t *__restrict__ codes) {
    const int groups = (C + 31) >> 5;
    const int chunks = (HW + 31) >> 5;
    const int lane = threadIdx.x & 31;
    const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t total = (int64_t)B * groups * chunks;
    for (int64_t t = warp; t < total; t += nwarps) {
        const int chunk = (int)(t % chunks);
        const int g = (int)((t / chunks) % groups);
        const int b = (int)(t / ((int64_t)chunks * groups));
        const int p = chunk * 32 + lane;
        if (p >= HW) continue;
        const int c0 = g * 32;
        const int cmax = min(32, C - c0);
        uint32_t w[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
#pragma unroll 8
        for (int c = 0; c < cmax; ++c) {
            const float v = __ldcs(x + ((int64_t)b * C + c0 + c) * HW + p);
            const int u = level_units(v * q.scale, q);
            if (FP4)
                w[c >> 3] |= level_code_e2m1(u) << ((c & 7) * 4);
            else
                w[c >> 2] |= (uint32_t)level_code_e4m3(u) << ((c & 3) * 8);
        }
        if (FP4) {
            uint8_t *dst = codes + ((((int64_t)b * HW + p) * C + c0) >> 1);
            if (cmax > 16)
                *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
            else
                *reinterpret_cast<uint2 *>(dst) = make_uint2(w[0], w[1]);
        } else {
            uint4 *dst = reinterpret_cast<uint4 *>(codes + ((int64_t)b * HW + p) * C + c0);
            dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
            if (cmax > 16) dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
        }
    }
}

// Weights [O][C][kh][kw] -> codes [O][kh][kw][C]: one thread per 16 channels
// (E4M3 bytes, or E2M1 nibbles with FP4).
template <bool FP4>
__global__ void weight_codes_kernel(const float *__restrict__ w, int O, int C, int kh, int kw, QParams q,
                                    const float *__restrict__ cscale, uint8_t *__restrict__ codes) {
    const int G = C >> 4;
    const int taps = kh * kw;
    const int64_t total = (int64_t)O * taps * G;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int g = (int)(t % G);
        const int tap = (int)((t / G) % taps);
        const int o = (int)(t / ((int64_t)G * taps));
        const float s = cscale ? cscale[o] : q.scale;
        uint32_t wd[4] = {0u, 0u, 0u, 0u};
        for (int c = 0; c < 16; ++c) {
            const float v = w[((int64_t)o * C + g * 16 + c) * taps + tap];
            const int u = level_units(v * s, q);
            if (FP4)
                wd[c >> 3] |= level_code_e2m1(u) << ((c & 7) * 4);
            else
                wd[c >> 2] |= (uint32_t)level_code_e4m3(u) << ((c & 3) * 8);
        }
        if (FP4)
            *reinterpret_cast<uint2 *>(codes + ((((int64_t)o * taps + tap) * C + g * 16) >> 1)) = make_uint2(wd[0], wd[1]);
        else
            *reinterpret_cast<uint4 *>(codes + ((int64_t)o * taps + tap) * C + g * 16) =
                make_uint4(wd[0], wd[1], wd[2], wd[3]);
    }
}

// Weights [O][C][kh][kw] -> bf16 level values in integer units [O][kh][kw][C]
// (1, 2 or 4 for the 3-bit magnitudes, all exact in bf16): one thread per
// 8 channels, one 128-bit store.
// out [O][kh][kw][Cp]: channels C .. Cp hold 0 (Cp >= C, a multiple of 8).
__global__ void weight_bf16_kernel(const float *__restrict__ w, int O, int C, int Cp, int kh, int kw, QParams q,
                                   const float *__restrict__ cscale, uint16_t *__restrict__ out) {
    const int G = Cp >> 3;
    const int taps = kh * kw;
    const int64_t total = (int64_t)O * taps * G;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int g = (int)(t % G);
        const int tap = (int)((t / G) % taps);
        const int o = (int)(t / ((int64_t)G * taps));
        const float s = cscale ? cscale[o] : q.scale;
        uint32_t wd[4];
        for (int j = 0; j < 4; ++j) {
            const int c = g * 8 + 2 * j;
            const float lo = c < C ? (float)level_units(w[((int64_t)o * C + c) * taps + tap] * s, q) : 0.0f;
            const float hi = c + 1 < C ? (float)level_units(w[((int64_t)o * C + c + 1) * taps + tap] * s, q) : 0.0f;
            wd[j] = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(lo)) |
                    ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(hi)) << 16);
        }
        *reinterpret_cast<uint4 *>(out + ((int64_t)o * taps + tap) * Cp + g * 8) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
    }
}

// fp32 NCHW -> bf16 NHWC, round to nearest even: one thread per output element
// of a 32 x 32 (channel, pixel) tile transposed through shared memory.
// Block (32, 8): a 32-channel x 32-pixel tile of one image through shared
// memory; each thread's four loads issue before its first shared-memory store.
// out [B][HW][Cp]: channels C .. Cp hold 0 (Cp >= C).
__global__ void __launch_bounds__(256) to_bf16_nhwc_kernel(const float *__restrict__ x, int C, int Cp, int HW,
                                                           uint16_t *__restrict__ out) {
    __shared__ float tile[32][33];
    const int b = blockIdx.z, c0 = blockIdx.y * 32, p0 = blockIdx.x * 32;
    float v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int i = threadIdx.y + 8 * k;
        const int c = c0 + i, p = p0 + threadIdx.x;
        v[k] = (c < C && p < HW) ? __ldg(x + ((int64_t)b * C + c) * HW + p) : 0.0f;
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) tile[threadIdx.y + 8 * k][threadIdx.x] = v[k];
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int i = threadIdx.y + 8 * k;
        const int p = p0 + i, c = c0 + threadIdx.x;
        if (c < Cp && p < HW)
            out[((int64_t)b * HW + p) * Cp + c] = __bfloat16_as_ushort(__float2bfloat16_rn(tile[threadIdx.x][i]));
    }
}

}  // namespace minw

// ===========================================================================
// Host side
// ===========================================================================

namespace minw_host {

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool valid_quant(const minw_quant *q) {
    if (q == nullptr) return false;
    if (q->bits < 1 || q->bits > 3) return false;
    if (!(q->scale == q->scale)) return false;            // NaN
    if (q->bits == 2 && !(q->thr[0] >= 0.0f)) return false;
    if (q->bits == 3 && !(q->thr[0] >= q->thr[1] && q->thr[1] >= q->thr[2] && q->thr[2] >= 0.0f))
        return false;
    return true;
}

int num_sms() {
    static int sms = 0;
    if (sms == 0) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess) return 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) sms = 0;
    }
    return sms;
}

minw_status launch_status() {
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

static int64_t grid_for(int64_t work_items, int threads) {
    const int sms = num_sms() > 0 ? num_sms() : 152;
    int64_t g = (work_items + threads - 1) / threads;
    const int64_t cap = (int64_t)sms * 8;   // 8 resident 256-thread CTAs per SM
    if (g > cap) g = cap;
    if (g < 1) g = 1;
    return g;
}

}  // namespace minw_host

using namespace minw;
using namespace minw_host;

extern "C" {

const char *minw_status_string(minw_status s) {
    switch (s) {
        case MINW_OK: return "ok";
        case MINW_EINVAL: return "invalid argument";
        case MINW_EUNSUPPORTED: return "unsupported shape or variant";
        case MINW_ECUDA: return "CUDA error";
        case MINW_ETIMEOUT: return "device-side wait timed out";
        case MINW_EDEVICE: return "no usable sm_103a device";
    }
    return "unknown status";
}

int32_t minw_version(void) { return 100; }

minw_status aqe_forward(const float *x, float *y, int64_t n, float alpha, const minw_quant *q,
                        void *stream) {
    if (n < 0 || !valid_quant(q) || !(alpha >= 0.0f && alpha <= 1.0f)) return MINW_EINVAL;
    if (n == 0) return MINW_OK;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return MINW_EINVAL;
    const QParams qp = to_qparams(q);
    const int64_t g = grid_for(n / 4 + 1, 256);
    aqe_forward_kernel<<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(x, y, n, alpha, 1.0f - alpha, qp);
    return launch_status();
}

minw_status aqe_forward_stochastic(const float *x, float *y, int64_t n, float alpha, uint64_t seed,
                                   uint64_t offset, void *stream) {
    if (n < 0 || !(alpha >= 0.0f && alpha <= 1.0f)) return MINW_EINVAL;
    if (n == 0) return MINW_OK;
    if (!x || !y || !aligned16(x) || !aligned16(y)) return MINW_EINVAL;
    const int64_t g = grid_for((n + 7) / 8, 256);
    aqe_forward_stochastic_kernel<<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(x, y, n, alpha, 1.0f - alpha, seed,
                                                                                offset);
    return launch_status();
}

minw_status aqe_backward(const float *x, const float *gy, float *gx, int64_t n, float alpha,
                         void *stream) {
    if (n < 0 || !(alpha >= 0.0f && alpha <= 1.0f)) return MINW_EINVAL;
    if (n == 0) return MINW_OK;
    if (!x || !gy || !gx || !aligned16(x) || !aligned16(gy) || !aligned16(gx)) return MINW_EINVAL;
    const int64_t g = grid_for(n / 4 + 1, 256);
    aqe_backward_kernel<<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(x, gy, gx, n, 2.0f * alpha);
    return launch_status();
}

minw_status aqe_backward_masked(const uint32_t *mask, const float *gy, float *gx, int64_t n,
                                float alpha, void *stream) {
    if (n < 0 || !(alpha >= 0.0f && alpha <= 1.0f)) return MINW_EINVAL;
    if (n == 0) return MINW_OK;
    if (!mask || !gy || !gx || !aligned16(gy) || !aligned16(gx)) return MINW_EINVAL;
    const int64_t g = grid_for(n / 4 + 1, 256);
    aqe_backward_masked_kernel<<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(mask, gy, gx, n,
                                                                            2.0f * alpha);
    return launch_status();
}

minw_status aqe_quantize_pack(const float *x, int32_t B, int32_t C, int32_t H, int32_t W,
                              const minw_quant *q, uint32_t *planes, float alpha, float *y,
                              uint32_t *mask, void *stream) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || !valid_quant(q)) return MINW_EINVAL;
    if (!x || !planes) return MINW_EINVAL;
    if (y && !(alpha >= 0.0f && alpha <= 1.0f)) return MINW_EINVAL;
    const int64_t HW = (int64_t)H * W;
    if (HW > (1ll << 30) || (int64_t)B * C * HW > (1ll << 40)) return MINW_EUNSUPPORTED;
    const QParams qp = to_qparams(q);
    cudaStream_t s = (cudaStream_t)stream;
    const int64_t n = (int64_t)B * C * HW;
    const bool vec = (HW % 4 == 0) && aligned16(x) && (!y || aligned16(y));
    const bool mask_atomic = mask && !(vec && HW % 32 == 0);
    if (mask_atomic) {
        if (cudaMemsetAsync(mask, 0, sizeof(uint32_t) * ((n + 31) / 32), s) != cudaSuccess)
            return MINW_ECUDA;
    }
    const int NW = (C + 31) / 32;
    if (vec) {
        const int64_t warps = (int64_t)B * NW * ((HW + 127) / 128);
        const int64_t g = grid_for(warps * 32, 256);
        switch (q->bits) {
            case 1: quantize_pack_vec_kernel<1><<<(unsigned)g, 256, 0, s>>>(x, B, C, (int)HW, qp, planes, alpha, 1.0f - alpha, y, mask, mask_atomic); break;
            case 2: quantize_pack_vec_kernel<2><<<(unsigned)g, 256, 0, s>>>(x, B, C, (int)HW, qp, planes, alpha, 1.0f - alpha, y, mask, mask_atomic); break;
            default: quantize_pack_vec_kernel<3><<<(unsigned)g, 256, 0, s>>>(x, B, C, (int)HW, qp, planes, alpha, 1.0f - alpha, y, mask, mask_atomic); break;
        }
    } else {
        const int64_t warps = (int64_t)B * NW * ((HW + 31) / 32);
        const int64_t g = grid_for(warps * 32, 256);
        switch (q->bits) {
            case 1: quantize_pack_scalar_kernel<1><<<(unsigned)g, 256, 0, s>>>(x, B, C, (int)HW, qp, planes, alpha, 1.0f - alpha, y, mask); break;
            case 2: quantize_pack_scalar_kernel<2><<<(unsigned)g, 256, 0, s>>>(x, B, C, (int)HW, qp, planes, alpha, 1.0f - alpha, y, mask); break;
            default: quantize_pack_scalar_kernel<3><<<(unsigned)g, 256, 0, s>>>(x, B, C, (int)HW, qp, planes, alpha, 1.0f - alpha, y, mask); break;
        }
    }
    return launch_status();
}

minw_status minw_pack_weights(const float *w, int32_t O, int32_t C, int32_t kh, int32_t kw,
                              const minw_quant *q, const float *channel_scale, uint32_t *planes,
                              void *stream) {
    if (O <= 0 || C <= 0 || kh <= 0 || kw <= 0 || !valid_quant(q) || !w || !planes)
        return MINW_EINVAL;
    const QParams qp = to_qparams(q);
    const int64_t words = (int64_t)O * kh * kw * ((C + 31) / 32);
    const int64_t g = grid_for(words, 256);
    cudaStream_t s = (cudaStream_t)stream;
    switch (q->bits) {
        case 1: pack_weights_kernel<1><<<(unsigned)g, 256, 0, s>>>(w, O, C, kh, kw, qp, channel_scale, planes); break;
        case 2: pack_weights_kernel<2><<<(unsigned)g, 256, 0, s>>>(w, O, C, kh, kw, qp, channel_scale, planes); break;
        default: pack_weights_kernel<3><<<(unsigned)g, 256, 0, s>>>(w, O, C, kh, kw, qp, channel_scale, planes); break;
    }
    return launch_status();
}

minw_status aqe_quantize_codes(const float *x, int32_t B, int32_t C, int32_t H, int32_t W,
                               const minw_quant *q, uint8_t *codes, void *stream) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || !valid_quant(q) || !x || !codes) return MINW_EINVAL;
    if (C % 16 != 0 || !aligned16(codes)) return MINW_EUNSUPPORTED;
    const int64_t HW = (int64_t)H * W;
    if (HW > (1ll << 30)) return MINW_EUNSUPPORTED;
    const int64_t warps = (int64_t)B * ((C + 31) / 32) * ((HW + 31) / 32);
    const int64_t g = grid_for(warps * 32, 256);
    quantize_codes_kernel<false><<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(x, B, C, (int)HW, to_qparams(q), codes);
    return launch_status();
}

minw_status aqe_quantize_codes_e2m1(const float *x, int32_t B, int32_t C, int32_t H, int32_t W,
                                    const minw_quant *q, uint8_t *codes, void *stream) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || !valid_quant(q) || !x || !codes) return MINW_EINVAL;
    if (C % 32 != 0 || !aligned16(codes)) return MINW_EUNSUPPORTED;
    const int64_t HW = (int64_t)H * W;
    if (HW > (1ll << 30)) return MINW_EUNSUPPORTED;
    const int64_t warps = (int64_t)B * ((C + 31) / 32) * ((HW + 31) / 32);
    const int64_t g = grid_for(warps * 32, 256);
    quantize_codes_kernel<true><<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(x, B, C, (int)HW, to_qparams(q), codes);
    return launch_status();
}

minw_status minw_pack_weight_codes(const float *w, int32_t O, int32_t C, int32_t kh, int32_t kw,
                                   const minw_quant *q, const float *channel_scale, uint8_t *codes,
                                   void *stream) {
    if (O <= 0 || C <= 0 || kh <= 0 || kw <= 0 || !valid_quant(q) || !w || !codes) return MINW_EINVAL;
    if (C % 16 != 0 || !aligned16(codes)) return MINW_EUNSUPPORTED;
    const int64_t items = (int64_t)O * kh * kw * (C / 16);
    const int64_t g = grid_for(items, 256);
    weight_codes_kernel<false><<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(w, O, C, kh, kw, to_qparams(q),
                                                                             channel_scale, codes);
    return launch_status();
}

minw_status minw_pack_weight_codes_e2m1(const float *w, int32_t O, int32_t C, int32_t kh, int32_t kw,
                                        const minw_quant *q, const float *channel_scale, uint8_t *codes,
                                        void *stream) {
    if (O <= 0 || C <= 0 || kh <= 0 || kw <= 0 || !valid_quant(q) || !w || !codes) return MINW_EINVAL;
    if (C % 16 != 0 || !aligned16(codes)) return MINW_EUNSUPPORTED;
    const int64_t items = (int64_t)O * kh * kw * (C / 16);
    const int64_t g = grid_for(items, 256);
    weight_codes_kernel<true><<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(w, O, C, kh, kw, to_qparams(q),
                                                                            channel_scale, codes);
    return launch_status();
}

minw_status minw_pack_weight_bf16_pad(const float *w, int32_t O, int32_t C, int32_t kh, int32_t kw, int32_t Cp,
                                      const minw_quant *q, const float *channel_scale, uint16_t *out, void *stream) {
    if (O <= 0 || C <= 0 || kh <= 0 || kw <= 0 || Cp < C || !valid_quant(q) || !w || !out) return MINW_EINVAL;
    if (Cp % 8 != 0 || !aligned16(out)) return MINW_EUNSUPPORTED;
    const int64_t items = (int64_t)O * kh * kw * (Cp / 8);
    const int64_t g = grid_for(items, 256);
    weight_bf16_kernel<<<(unsigned)g, 256, 0, (cudaStream_t)stream>>>(w, O, C, Cp, kh, kw, to_qparams(q),
                                                                     channel_scale, out);
    return launch_status();
}

minw_status minw_pack_weight_bf16(const float *w, int32_t O, int32_t C, int32_t kh, int32_t kw,
                                  const minw_quant *q, const float *channel_scale, uint16_t *out, void *stream) {
    if (C > 0 && C % 8 != 0) return MINW_EUNSUPPORTED;
    return minw_pack_weight_bf16_pad(w, O, C, kh, kw, C, q, channel_scale, out, stream);
}

minw_status minw_to_bf16_nhwc_pad(const float *x, int32_t B, int32_t C, int32_t H, int32_t W, int32_t Cp,
                                  uint16_t *out, void *stream) {
    if (B <= 0 || C <= 0 || H <= 0 || W <= 0 || Cp < C || !x || !out) return MINW_EINVAL;
    const int64_t HW = (int64_t)H * W;
    if (HW > (1ll << 30) || B > 65535 || (Cp + 31) / 32 > 65535) return MINW_EUNSUPPORTED;
    const dim3 grid((unsigned)((HW + 31) / 32), (unsigned)((Cp + 31) / 32), (unsigned)B);
    to_bf16_nhwc_kernel<<<grid, dim3(32, 8), 0, (cudaStream_t)stream>>>(x, C, Cp, (int)HW, out);
    return launch_status();
}

minw_status minw_to_bf16_nhwc(const float *x, int32_t B, int32_t C, int32_t H, int32_t W, uint16_t *out,
                              void *stream) {
    return minw_to_bf16_nhwc_pad(x, B, C, H, W, C, out, stream);
}

}  // extern "C"
