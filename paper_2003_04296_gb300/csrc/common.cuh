// common.cuh -- shared device helpers of libminw.so (sm_103a only).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/minw.h"

#if defined(__CUDA_ARCH__) && (__CUDA_ARCH__ != 1030)
#error "libminw is built for sm_103a only"
#endif

namespace minw {

// Quantizer parameters as passed to kernels (by value).
struct QParams {
    int bits;
    float thr0, thr1, thr2;   // D_1 > D_2 > D_3
    float scale;
};

inline QParams to_qparams(const minw_quant *q) {
    QParams p;
    p.bits = q->bits;
    p.thr0 = q->thr[0];
    p.thr1 = q->thr[1];
    p.thr2 = q->thr[2];
    p.scale = q->scale;
    return p;
}

// Level of u (already scaled) in integer units: 1-bit and 2-bit levels are
// the values themselves, 3-bit levels count quarters (Eq. sign / tnn / qnn).
__device__ __forceinline__ int level_units(float u, const QParams &q) {
    const int s = (u > 0.0f) ? 1 : -1;
    if (q.bits == 1) return s;
    const float m = fabsf(u);
    if (q.bits == 2) return (m <= q.thr0) ? 0 : s;
    if (m <= q.thr2) return 0;
    if (m <= q.thr1) return s;
    if (m <= q.thr0) return 2 * s;
    return 4 * s;
}

// Dequantized level as fp32 (exact: +-1, +-1/2, +-1/4, 0).
__device__ __forceinline__ float level_value(float u, const QParams &q) {
    const int v = level_units(u, q);
    return (q.bits == 3) ? 0.25f * (float)v : (float)v;
}

// Plane bits of one level (units) for the packed layout:
// bit 0 sign, then (2-bit) non-zero mask or (3-bit) code bits 0, 1.
__device__ __forceinline__ uint32_t level_plane_bits(int v, int bits) {
    uint32_t r = (v < 0) ? 1u : 0u;
    if (bits == 2) r |= (v != 0) ? 2u : 0u;
    if (bits == 3) {
        const int m = v < 0 ? -v : v;
        const uint32_t k = (m == 4) ? 3u : (m == 2) ? 2u : (m == 1) ? 1u : 0u;
        r |= k << 1;
    }
    return r;
}

// FP8 E4M3 encoding of a level in integer units {0, +-1, +-2, +-4}: the
// tensor-core operand of the "codes" layout (exact: powers of two).
__host__ __device__ __forceinline__ uint8_t level_code_e4m3(int v) {
    if (v == 0) return 0u;
    const int m = v < 0 ? -v : v;
    const uint32_t e = (m == 4) ? 9u : (m == 2) ? 8u : 7u;     // biased exponent, bias 7
    return (uint8_t)(((v < 0) ? 0x80u : 0u) | (e << 3));
}

}  // namespace minw

// Host-side helpers shared by the translation units.
namespace minw_host {

bool aligned16(const void *p);
bool valid_quant(const minw_quant *q);
int num_sms();
minw_status launch_status();

}  // namespace minw_host
