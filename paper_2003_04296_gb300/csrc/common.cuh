// common.cuh -- shared device helpers of libminw.so (sm_103a only).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

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

// FP4 E2M1 encoding of a level in integer units (sign bit 3, exponent bits
// 2-1 with bias 1, mantissa bit 0): 0 -> 0x0, +-1 -> 0x2/0xA, +-2 -> 0x4/0xC,
// +-4 -> 0x6/0xE.  Every level is exact, so E2M1 products are exact too.  The
// packed "E2M1 codes" layout holds two channels per byte, channel 2j in the
// low nibble of byte j.
__host__ __device__ __forceinline__ uint32_t level_code_e2m1(int v) {
    if (v == 0) return 0u;
    const int m = v < 0 ? -v : v;
    const uint32_t c = (m == 4) ? 3u : (m == 2) ? 2u : 1u;
    return ((v < 0) ? 8u : 0u) | (c << 1);
}

// Value in integer units of an E2M1 level code (low nibble of c).
__host__ __device__ __forceinline__ float code_units_e2m1(uint32_t c) {
    const uint32_t e = (c >> 1) & 3u;
    if (e == 0u) return 0.0f;
    const float m = (float)(1u << (e - 1u));
    return (c & 8u) ? -m : m;
}

// ---------------------------------------------------------------------------
// Output quantization as integer thresholds.
//
// A hidden layer's output level is L(acc) = h(HardTanh(fmaf(acc, s, t))).
// fmaf is monotone in acc, HardTanh and h are monotone, so L is a monotone
// step function of the integer accumulator: with sigma = sign(s) (+1 for
// s = 0), level index k(acc) = #{j : sigma * acc >= T_j} for per-channel
// integer breakpoints T_1 <= ... <= T_{n-1} (n levels).  The breakpoints are
// found by binary search on the very same fp32 operations, so the decision is
// bit-identical to evaluating the chain element by element.
// ---------------------------------------------------------------------------

// Number of levels of a quantizer and the level index of a BN output y.
__host__ __device__ __forceinline__ int num_levels(int bits) { return bits == 1 ? 2 : bits == 2 ? 3 : 7; }

__device__ __forceinline__ int level_index_of_y(float y, const QParams &q) {
    y = fminf(fmaxf(y, -1.0f), 1.0f);
    const int u = level_units(y * q.scale, q);
    if (q.bits == 1) return u > 0 ? 1 : 0;
    if (q.bits == 2) return u + 1;
    const int m = u < 0 ? -u : u;
    const int e = (m == 4) ? 3 : m;                    // 0,1,2,4 -> 0,1,2,3
    return 3 + (u < 0 ? -e : e);
}

// E4M3 code and plane bits (sign | code << 1) of level index k, packed tables.
__device__ __forceinline__ uint32_t code_of_index(int k, int bits) {
    if (bits == 1) return k ? 0x38u : 0xB8u;
    if (bits == 2) return (uint32_t)((0x3800B8ull >> (8 * k)) & 0xFF);
    return (uint32_t)((0x0048403800B8C0C8ull >> (8 * k)) & 0xFF);
}
__device__ __forceinline__ uint32_t planes_of_index(int k, int bits) {
    if (bits == 1) return k ? 0u : 1u;
    if (bits == 2) return (0x0203u >> (4 * k)) & 0x3u;     // idx 0: 3, 1: 0, 2: 2
    return (uint32_t)((06420357ull >> (3 * k)) & 7ull);     // octal digits, idx 0 = low
}

// Breakpoints of channel o: T[0 .. n-2] and sigma, written to out[0 .. n-1].
__device__ __forceinline__ void channel_thresholds(float s, float t, const QParams &q, float *out) {
    const float sigma = (s < 0.0f) ? -1.0f : 1.0f;
    const int n = num_levels(q.bits);
    const int V = (1 << 24) - 1;                       // |acc| < 2^24 always
    for (int j = 1; j < n; ++j) {
        auto idx = [&](int v) { return level_index_of_y(fmaf((float)v * sigma, s, t), q); };
        float T;
        if (idx(-V) >= j) {
            T = -INFINITY;
        } else if (idx(V) < j) {
            T = INFINITY;
        } else {
            int lo = -V, hi = V;                       // idx(lo) < j <= idx(hi)
            while (hi - lo > 1) {
                const int mid = lo + ((hi - lo) >> 1);
                if (idx(mid) >= j) hi = mid; else lo = mid;
            }
            T = (float)hi;
        }
        out[j - 1] = T;
    }
    out[n - 1] = sigma;
}

// The same breakpoints for an fp32 accumulator (the first layer, whose input
// is not quantized): T_j is the smallest fp32 v with level index >= j when
// evaluated at acc = sigma * v, found by binary search over the ordered fp32
// bit patterns (finite values only).
__device__ __forceinline__ int f32_order(float v) {
    const int i = __float_as_int(v);
    return i >= 0 ? i : (int)(0x80000000u - (uint32_t)i);   // monotone in v; -0 -> 0
}
__device__ __forceinline__ float f32_from_order(int k) {
    return k >= 0 ? __int_as_float(k) : __int_as_float((int)(0x80000000u - (uint32_t)k));
}
__device__ __forceinline__ void channel_thresholds_f32(float s, float t, const QParams &q, float *out) {
    const float sigma = (s < 0.0f) ? -1.0f : 1.0f;
    const int n = num_levels(q.bits);
    const int V = 0x7F7FFFFF;                          // order of FLT_MAX
    for (int j = 1; j < n; ++j) {
        auto idx = [&](int k) { return level_index_of_y(fmaf(f32_from_order(k) * sigma, s, t), q); };
        float T;
        if (idx(-V) >= j) {
            T = -INFINITY;
        } else if (idx(V) < j) {
            T = INFINITY;
        } else {
            int lo = -V, hi = V;
            while ((long long)hi - lo > 1) {                  // 2V overflows int
                const int mid = (int)(((long long)lo + hi) >> 1);
                if (idx(mid) >= j) hi = mid; else lo = mid;
            }
            T = f32_from_order(hi);
        }
        out[j - 1] = T;
    }
    out[n - 1] = sigma;
}

// Level index of an accumulator (exact integer held in fp32) from the
// breakpoints of its channel (n - 1 thresholds then sigma).
__device__ __forceinline__ int level_index_of_acc(float acc, const float *thr, int n) {
    const float v = acc * thr[n - 1];
    int k = 0;
    for (int j = 0; j < n - 1; ++j) k += (v >= thr[j]) ? 1 : 0;
    return k;
}

// ---------------------------------------------------------------------------
// Level masks.  For 32 channels of one output pixel and each breakpoint u,
// M_u has bit j set when channel j stays below breakpoint u (sigma * acc <
// T_u), i.e. its level index k <= u; the breakpoints ascend, so the masks are
// nested.  Bit planes and E4M3 codes of the levels follow by bitwise logic.
// ---------------------------------------------------------------------------

// Four channels' bits (nibble g of m) spread to the low bit of four bytes.
__device__ __forceinline__ uint32_t spread4(uint32_t m, int g) {
    return (((m >> (4 * g)) & 0xFu) * 0x00204081u) & 0x01010101u;
}

// Planes of OUTB-bit levels from their masks: sign, then the non-zero mask
// (2 bits) or the magnitude code |k - 3| (3 bits), one bit per channel.
template <int OUTB>
__device__ __forceinline__ void level_planes(const uint32_t *M, uint32_t *P) {
    if constexpr (OUTB == 1) {
        P[0] = M[0];
    } else if constexpr (OUTB == 2) {
        P[0] = M[0];
        P[1] = M[0] | ~M[1];
    } else {
        P[0] = M[2];
        P[1] = M[0] | (M[2] & ~M[1]) | (M[4] & ~M[3]) | ~M[5];     // |k - 3| in {1, 3}
        P[2] = M[1] | ~M[4];                                        // |k - 3| in {2, 3}
    }
}

// E4M3 codes of channels 4g .. 4g + 3 (one byte each) from the planes.
template <int OUTB>
__device__ __forceinline__ uint32_t level_code_word(const uint32_t *P, int g) {
    if constexpr (OUTB == 1) {
        return (spread4(P[0], g) * 0x80u) | 0x38383838u;
    } else if constexpr (OUTB == 2) {
        return spread4(P[1], g) * 0x38u + spread4(P[0], g) * 0x80u;
    } else {
        const uint32_t c0 = P[1], c1 = P[2];
        return spread4(c0, g) * 0x08u + spread4(c0 & ~c1, g) * 0x30u + spread4(c1, g) * 0x40u +
               spread4(P[0] & (c0 | c1), g) * 0x80u;
    }
}

// Eight channels' bits (byte g of m) spread to the low bit of eight nibbles.
__device__ __forceinline__ uint32_t spread8n(uint32_t m, int g) {
    uint32_t x = (m >> (8 * g)) & 0xFFu;
    x = (x | (x << 12)) & 0x000F000Fu;
    x = (x | (x << 6)) & 0x03030303u;
    x = (x | (x << 3)) & 0x11111111u;
    return x;
}

// E2M1 codes of channels 8g .. 8g + 7 (one nibble each, channel 8g lowest)
// from the planes: the nibble is sign * 8 + magnitude code * 2.
template <int OUTB>
__device__ __forceinline__ uint32_t level_code_word4(const uint32_t *P, int g) {
    if constexpr (OUTB == 1) {
        return (spread8n(P[0], g) * 8u) | 0x22222222u;
    } else if constexpr (OUTB == 2) {
        return spread8n(P[1], g) * 2u + spread8n(P[0], g) * 8u;
    } else {
        return spread8n(P[1], g) * 2u + spread8n(P[2], g) * 4u + spread8n(P[0] & (P[1] | P[2]), g) * 8u;
    }
}

// E2M1 code of level index k of an OUTB-bit quantizer (packed nibble tables).
template <int OUTB>
__device__ __forceinline__ uint32_t code4_k(int k) {
    if constexpr (OUTB == 1) return (0x2Au >> (4 * k)) & 0xFu;
    else if constexpr (OUTB == 2) return (0x20Au >> (4 * k)) & 0xFu;
    else return (0x6420ACEu >> (4 * k)) & 0xFu;
}

// Stores the planes (bits of channels >= nvalid cleared) and the E4M3 codes
// (ncodes = 16 or 32 bytes; the second 16 only when nvalid > 16) of OUTB-bit
// levels given by their masks M[0 .. levels - 2].
// With codes4 the codes are E2M1 nibbles instead (codes then points at the
// byte of the first channel: 16 bytes for 32 channels, 8 for 16).
template <int OUTB>
__device__ __forceinline__ void store_level_masks(const uint32_t *M, int nvalid, int ncodes, uint32_t *planes, int NWo,
                                                  uint8_t *codes, bool codes4 = false) {
    uint32_t P[3];
    level_planes<OUTB>(M, P);
    if (planes != nullptr) {
        const uint32_t vm = nvalid >= 32 ? 0xffffffffu : ((1u << nvalid) - 1u);
#pragma unroll
        for (int u = 0; u < OUTB; ++u) planes[u * NWo] = P[u] & vm;
    }
    if (codes != nullptr && codes4) {
        if (nvalid > 16 && ncodes > 16)
            *reinterpret_cast<uint4 *>(codes) = make_uint4(level_code_word4<OUTB>(P, 0), level_code_word4<OUTB>(P, 1),
                                                           level_code_word4<OUTB>(P, 2), level_code_word4<OUTB>(P, 3));
        else
            *reinterpret_cast<uint2 *>(codes) = make_uint2(level_code_word4<OUTB>(P, 0), level_code_word4<OUTB>(P, 1));
    } else if (codes != nullptr) {
        uint4 *dst = reinterpret_cast<uint4 *>(codes);
        dst[0] = make_uint4(level_code_word<OUTB>(P, 0), level_code_word<OUTB>(P, 1), level_code_word<OUTB>(P, 2),
                            level_code_word<OUTB>(P, 3));
        if (nvalid > 16 && ncodes > 16)
            dst[1] = make_uint4(level_code_word<OUTB>(P, 4), level_code_word<OUTB>(P, 5), level_code_word<OUTB>(P, 6),
                                level_code_word<OUTB>(P, 7));
    }
}

// Programmatic dependent launch: the kernels of a forward are launched so
// that the next one may start (its set-up: barriers, TMEM, breakpoints,
// weights) while the previous one finishes.  Each waits here before it reads
// what an earlier kernel wrote or writes what an earlier kernel reads, and
// lets its own dependents launch once its CTAs run.  Both are no-ops when
// the launch did not ask for it.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

// A breakpoint held for the mask test: -T, with -0 replaced by +0, so that
// fmaf(acc, sigma, -T) is never -0 and its sign bit is exactly [sigma * acc < T].
__host__ __device__ __forceinline__ float mask_breakpoint(float T) { return T == 0.0f ? 0.0f : -T; }

}  // namespace minw

// Host-side helpers shared by the translation units.
namespace minw_host {

bool aligned16(const void *p);
bool valid_quant(const minw_quant *q);
int num_sms();
minw_status launch_status();
bool pdl_enabled();                 // plan option pdl
minw_plan_options plan_options();   // the process-wide plan options (runtime.cu)
int take_stall(int which);          // 1 once after minw_test_stall_next_launch(which)
// Every kernel of the library asks for the largest shared-memory carve-out
// of the SM (set once per kernel): consecutive kernels of a forward then need
// no L1 / shared-memory reconfiguration of the SM between them, so the next
// kernel's CTAs start as soon as an SM frees up.
void max_shared_carveout(const void *kern);

// cuTensorMapEncodeTiled from the driver (nullptr when it is unavailable).
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();

// Kernel launch on stream s that may overlap the previous kernel in the
// stream (programmatic stream serialization); the kernel calls pdl_wait()
// before its dependent accesses.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 1 : 0;
    max_shared_carveout(reinterpret_cast<const void *>(kern));
    return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

}  // namespace minw_host
