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
#include <stdlib.h>
#include <string.h>

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
__device__ __forceinline__ unsigned long long fma2(unsigned long long a, unsigned long long b, unsigned long long c) {
    unsigned long long d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ float lane2(unsigned long long v, int hi) {
    float lo_, hi_;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo_), "=f"(hi_) : "l"(v));
    return hi ? hi_ : lo_;
}

// Shared-memory loads by 32-bit shared address (the address arithmetic of
// the tap loop stays in 32-bit registers with immediate offsets).
__device__ __forceinline__ float lds_f32(uint32_t a) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1];\n" : "=f"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ unsigned long long lds_u64(uint32_t a) {
    unsigned long long v;
    asm volatile("ld.shared.u64 %0, [%1];\n" : "=l"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ void lds_2x64(uint32_t a, unsigned long long &x, unsigned long long &y) {
    asm volatile("ld.shared.v2.u64 {%0, %1}, [%2];\n" : "=l"(x), "=l"(y) : "r"(a));
}

// Error flag of this file's bounded waits (read with the tensor-core
// kernels' flag by minw_get_last_device_error).
__device__ int g_first_error = 0;

__device__ __forceinline__ uint32_t saddr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void fbar_init(uint64_t *bar) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(saddr(bar)));
}

__device__ __forceinline__ bool fbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, 100000;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(saddr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait for a patch: false (and the error flag set) after limit SM
// clocks (about a second by default).
__device__ __forceinline__ bool fbar_wait(uint64_t *bar, uint32_t parity, long long limit) {
    if (fbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!fbar_try_wait(bar, parity)) {
        if (clock64() - t0 > limit) {
            atomicExch(&g_first_error, 1);
            return false;
        }
    }
    return true;
}

// One box of the image [B][C][H][W] (x, y, c, b from the origin given) into
// shared memory, completing its bytes on bar.  Zero outside the image.
__device__ __forceinline__ void patch_tma(void *dst, const CUtensorMap *map, uint64_t *bar, uint32_t bytes, int x,
                                          int y, int b) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(saddr(bar)), "r"(bytes)
                 : "memory");
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];\n" ::"r"(saddr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(0), "r"(b), "r"(saddr(bar))
        : "memory");
}

struct FirstTile {
    int OCB;          // output channels per CTA (32 or 64)
    int groups;       // 32-channel groups per CTA
    int PB;           // output pixels per CTA (64 per pixel block, 8 / groups blocks)
    int tiles;        // CTAs along the pixels of one image
    int Rmax;         // input patch rows
    int Ws;           // patch columns per stride phase (cp.async patches)
    int RP;           // patch row pitch: stride x Ws, or the box width (TMA patches)
    int K;            // C x kh x kw
    int nb;           // input patch buffers (2 or 3: the patch of tile t + (nb - 1) G is in flight)
    int tma;          // patches as one TMA box each (row-major columns from x0, zero padded)
    int x0;           // TMA patches: first image column of the box (a multiple of 4, <= -pad)
    int xsh;          // TMA patches: box column of image column -pad (-pad - x0)
    int xoff;         // float offset of the first patch buffer (a multiple of 32: 128-byte aligned)
    int pstride;      // floats per patch buffer (a multiple of 32)
    size_t smem;      // bytes of dynamic shared memory
};

static FirstTile first_tile(const FirstArgs &a, bool tma) {
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
    // TMA box: image columns x0 .. x0 + RP - 1 with x0 rounded down to 16 bytes
    t.x0 = -((a.pad + 3) / 4) * 4;
    t.xsh = -a.pad - t.x0;
    t.tma = tma && (Win + t.xsh + 3) / 4 * 4 <= 256 && t.Rmax <= 256 && a.C <= 256;
    if (t.tma) t.RP = (Win + t.xsh + 3) / 4 * 4;
    t.xoff = (t.K * t.OCB + t.OCB * 8 + 31) / 32 * 32;
    t.pstride = (a.C * t.Rmax * t.RP + 31) / 32 * 32;
    // three patch buffers (two tiles of look-ahead) where two CTAs still fit on an SM
    const size_t fixed = sizeof(float) * (size_t)t.xoff + 4 * sizeof(uint64_t);   // nb patch barriers + the stall test's
    const size_t pbytes = sizeof(float) * (size_t)t.pstride;
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
// runtime shape.  TM: each patch is one TMA box of the image (rows of RP
// columns from x0, zero outside the image, completion on an mbarrier per
// buffer), not per-word cp.async copies split by stride phase; a thread then
// reads its pixels' words S apart (16 lanes on 16 distinct banks for S <= 2).
template <int OUTB, int KH, int KW, int S, bool TM>
__global__ void __launch_bounds__(FIRST_NT, 2)
    conv_first_kernel(const FirstArgs a, const FirstTile tl, const __grid_constant__ CUtensorMap tmX) {
    extern __shared__ float4 smem4[];
    const int kh = KH ? KH : a.kh, kw = KW ? KW : a.kw, st = S ? S : a.stride;
    const int OCB = tl.OCB, K = tl.K, RP = tl.RP, Ws = tl.Ws;
    const size_t patch = (size_t)tl.pstride;
    float *sW = reinterpret_cast<float *>(smem4);                 // [K][OCB]
    float *sT = sW + (size_t)K * OCB;                             // [8][OCB] -breakpoints, sigma (row 7)
    float *sX0 = sW + tl.xoff;                                    // [nb][C][Rmax][RP]
    uint64_t *fullb = reinterpret_cast<uint64_t *>(sX0 + (size_t)tl.nb * patch);   // [nb] TMA patch arrivals, then
                                                                                  // the timeout test's barrier
    int issued[3] = {0, 0, 0}, landed[3] = {0, 0, 0};       // TMA patches per buffer (thread 0 issues them all)

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
        if constexpr (TM) {       // one thread: the whole patch as one box
            patch_tma(sX0 + buf * patch, &tmX, &fullb[buf], (uint32_t)(sizeof(float) * a.C * tl.Rmax * RP), tl.x0,
                      (p0 / a.Wo) * st - a.pad, b);
            ++issued[buf];
            return;
        }
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
        float th[8];
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
        // channel-fastest rows (a channel pair is one 64-bit word); sigma in row 7
        for (int u = 0; u < nl - 1; ++u) sT[u * OCB + threadIdx.x] = th[u];
        sT[7 * OCB + threadIdx.x] = th[nl - 1];
    }

    if (TM && threadIdx.x == 0) {
        for (int j = 0; j <= tl.nb; ++j) fbar_init(&fullb[j]);
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    __syncthreads();                                             // barriers initialised

    // warp = 32 channels x 64 pixels; lane = (channel half h, pixel l16):
    // 4 pixels (16 apart) x 16 channels per thread
    pdl_trigger();                                               // set-up done
    pdl_wait();                                                  // the image and the output buffer are shared
    // TMA: thread 0 issues; cp.async: one group per tile slot (empty past the
    // end), so that the wait count is fixed
    const int nb = tl.nb;
    for (int j = 0; j < nb - 1; ++j) {
        if (t + j * (int)gridDim.x < total) {
            if (!TM || threadIdx.x == 0) load_patch(t + j * (int)gridDim.x, j);
        } else if (!TM) {
            cp_async_commit();
        }
    }
    bool dead = false;                                           // a patch wait ran out: skip the work
    // timeout-path test: a wait on a barrier that nothing completes runs out
    if (TM && a.stall && !fbar_wait(&fullb[tl.nb], 0u, a.wait_cycles)) dead = true;
    const int g = warp % tl.groups, pb = warp / tl.groups;
    const int h = lane >> 4, l16 = lane & 15;
    const int NWo = (a.O + 31) >> 5;
    const int gch = min(32, ochan - g * 32);                     // live channels of this warp (may be <= 0)
    const int hch = gch - 16 * h;                                // live channels of this half (may be <= 0)
    const int ob = o0 + g * 32;
    const float *wg = sW + g * 32 + h * 16;
    constexpr int NL = OUTB == 0 ? 1 : (OUTB == 1 ? 2 : (OUTB == 2 ? 3 : 7));
    for (int buf = 0, it = 0; t < total; t += gridDim.x, buf = buf + 1 == nb ? 0 : buf + 1, ++it) {
        const int tn = t + (nb - 1) * (int)gridDim.x;
        const int bn = buf == 0 ? nb - 1 : buf - 1;              // the slot tile t - G used
        if constexpr (TM) {
            if (tn < total && threadIdx.x == 0 && !dead) load_patch(tn, bn);
            if (!dead) {
                if (fbar_wait(&fullb[buf], (uint32_t)(it / nb) & 1u, a.wait_cycles))
                    ++landed[buf];
                else
                    dead = true;
            }
        } else {
            if (tn < total)
                load_patch(tn, bn);
            else
                cp_async_commit();
            if (nb == 3)
                cp_async_wait<2>();
            else
                cp_async_wait<1>();
        }
        dead = __syncthreads_or(dead);                           // patch t (and the weights) visible

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
            pofs[i] = (yy - y_first) * st * RP + (TM ? xx * st + tl.xsh : xx);
        }
        if (p0 + pb * 64 < pend && gch > 0 && !dead) {          // warp-uniform: the epilogue shuffles
            // accumulators of channel pairs (2j, 2j + 1), packed for fma.rn.f32x2
            unsigned long long acc[FIRST_PX][8];
#pragma unroll
            for (int i = 0; i < FIRST_PX; ++i)
#pragma unroll
                for (int o = 0; o < 8; ++o) acc[i][o] = 0ull;
            const uint32_t xs = (uint32_t)__cvta_generic_to_shared(sX);
            const uint32_t ws = (uint32_t)__cvta_generic_to_shared(wg);
            uint32_t xa[FIRST_PX];
#pragma unroll
            for (int i = 0; i < FIRST_PX; ++i) xa[i] = xs + 4u * (uint32_t)pofs[i];
            for (int c = 0; c < a.C; ++c) {
#pragma unroll (KH ? KH : 1)
                for (int ky = 0; ky < kh; ++ky) {
                    const uint32_t ro = 4u * (uint32_t)((c * tl.Rmax + ky) * RP);
                    const uint32_t wr = ws + 4u * (uint32_t)((c * kh + ky) * kw * OCB);
#pragma unroll (KW ? KW : 1)
                    for (int kx = 0; kx < kw; ++kx) {
                        // tap column kx: stride phase kx % S, offset kx / S within the phase
                        const uint32_t xo = ro + 4u * (uint32_t)(TM ? kx : (kx % st) * Ws + kx / st);
                        unsigned long long xv[FIRST_PX];
#pragma unroll
                        for (int i = 0; i < FIRST_PX; ++i) xv[i] = dup2(lds_f32(xa[i] + xo));
                        const uint32_t wk = wr + 4u * (uint32_t)(kx * OCB);
#pragma unroll
                        for (int o4 = 0; o4 < 4; ++o4) {
                            unsigned long long wx, wy;
                            lds_2x64(wk + 16u * o4, wx, wy);
#pragma unroll
                            for (int i = 0; i < FIRST_PX; ++i) {
                                ffma2(acc[i][2 * o4], xv[i], wx);
                                ffma2(acc[i][2 * o4 + 1], xv[i], wy);
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
                // sign of fmaf(acc, sigma, -T_u) (one packed fma.rn.f32x2 per channel pair); then the
                // two halves make the 32-channel word
                const uint32_t tb = (uint32_t)__cvta_generic_to_shared(sT + g * 32 + 16 * h);
                uint32_t MM[FIRST_PX][NL - 1];
#pragma unroll
                for (int i = 0; i < FIRST_PX; ++i)
#pragma unroll
                    for (int u = 0; u < NL - 1; ++u) MM[i][u] = 0u;
#pragma unroll
                for (int j = 7; j >= 0; --j) {                   // channels 2j + 1, 2j (high bit first)
                    const unsigned long long sg = lds_u64(tb + 4u * (uint32_t)(7 * OCB + 2 * j));
#pragma unroll
                    for (int u = 0; u < NL - 1; ++u) {
                        const unsigned long long nt = lds_u64(tb + 4u * (uint32_t)(u * OCB + 2 * j));
#pragma unroll
                        for (int i = 0; i < FIRST_PX; ++i) {
                            const unsigned long long r = fma2(acc[i][j], sg, nt);
                            MM[i][u] = __funnelshift_l(__float_as_uint(lane2(r, 1)), MM[i][u], 1);
                            MM[i][u] = __funnelshift_l(__float_as_uint(lane2(r, 0)), MM[i][u], 1);
                        }
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
                    if (a.codes_out != nullptr && hch > 0 && a.codes4)
                        *reinterpret_cast<uint2 *>(a.codes_out + ((m * a.O + ob + 16 * h) >> 1)) =
                            make_uint2(level_code_word4<OUTB>(P, 2 * h), level_code_word4<OUTB>(P, 2 * h + 1));
                    else if (a.codes_out != nullptr && hch > 0)
                        *reinterpret_cast<uint4 *>(a.codes_out + m * a.O + ob + 16 * h) =
                            make_uint4(level_code_word<OUTB>(P, 4 * h), level_code_word<OUTB>(P, 4 * h + 1),
                                       level_code_word<OUTB>(P, 4 * h + 2), level_code_word<OUTB>(P, 4 * h + 3));
                }
            }
        }
        __syncthreads();                                         // buffer buf is free for tile t + nb G
    }
    // a run that gave up leaves patches in flight: every one lands before the CTA exits
    if (TM && threadIdx.x == 0)
        for (int j = 0; j < tl.nb; ++j)
            while (landed[j] < issued[j]) {
                if (!fbar_wait(&fullb[j], (uint32_t)landed[j] & 1u, a.wait_cycles)) break;
                ++landed[j];
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

template <int OUTB, int KH, int KW, int S, bool TM>
static minw_status launch_first_shape(const FirstArgs &a, const FirstTile &tl, const CUtensorMap &tm,
                                      cudaStream_t s) {
    static size_t configured = 0;
    void (*kern)(const FirstArgs, const FirstTile, const CUtensorMap) = conv_first_kernel<OUTB, KH, KW, S, TM>;
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
    FirstArgs ar = a;
    ar.wait_cycles = (long long)minw_host::plan_options().wait_cycles;
    ar.stall = TM ? minw_host::take_stall(MINW_STALL_CONV_FIRST) : 0;
    if (minw_host::launch_pdl(kern, grid, dim3(FIRST_NT), tl.smem, s, ar, tl, tm) != cudaSuccess) return MINW_ECUDA;
    return MINW_OK;
}

static bool tma_shape(const FirstArgs &a) {
    return (a.kh == 3 && a.kw == 3 && a.stride == 1) || (a.kh == 7 && a.kw == 7 && a.stride == 2);
}

template <int OUTB>
static minw_status launch_first_bits(const FirstArgs &a, const FirstTile &tl, const CUtensorMap &tm, cudaStream_t s) {
    if (a.kh == 3 && a.kw == 3 && a.stride == 1)
        return tl.tma ? launch_first_shape<OUTB, 3, 3, 1, true>(a, tl, tm, s)
                      : launch_first_shape<OUTB, 3, 3, 1, false>(a, tl, tm, s);
    if (a.kh == 7 && a.kw == 7 && a.stride == 2)
        return tl.tma ? launch_first_shape<OUTB, 7, 7, 2, true>(a, tl, tm, s)
                      : launch_first_shape<OUTB, 7, 7, 2, false>(a, tl, tm, s);
    return launch_first_shape<OUTB, 0, 0, 0, false>(a, tl, tm, s);
}

// Patches by TMA (plan option first_tma; else per-word cp.async) where the
// image rows are 16-byte multiples at a 16-byte aligned base and the box fits
// the limits.
static bool first_tma_pref() { return minw_host::plan_options().first_tma != 0; }

int take_first_error() {
    int flag = 0;
    if (cudaMemcpyFromSymbol(&flag, g_first_error, sizeof(int)) != cudaSuccess) return -1;
    if (flag) {
        const int zero = 0;
        if (cudaMemcpyToSymbol(g_first_error, &zero, sizeof(int)) != cudaSuccess) return -1;
    }
    return flag;
}

minw_status launch_conv_first(const FirstArgs &a, cudaStream_t s) {
    if (minw_host::plan_options().first_tensor_cores != 0 && first_tc_supported(a)) return launch_first_tc(a, s);
    const bool tma_ok = first_tma_pref() && tma_shape(a) && a.W % 4 == 0 && minw_host::aligned16(a.x) &&
                        minw_host::tensor_map_encoder() != nullptr;
    FirstTile tl = first_tile(a, tma_ok);
    CUtensorMap tm;
    memset(&tm, 0, sizeof(tm));
    if (tl.tma) {
        const cuuint64_t dims[4] = {(cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.C, (cuuint64_t)a.B};
        const cuuint64_t strides[3] = {(cuuint64_t)a.W * 4, (cuuint64_t)a.H * a.W * 4,
                                       (cuuint64_t)a.C * a.H * a.W * 4};
        const cuuint32_t box[4] = {(cuuint32_t)tl.RP, (cuuint32_t)tl.Rmax, (cuuint32_t)a.C, 1u};
        const cuuint32_t es[4] = {1u, 1u, 1u, 1u};
        if (minw_host::tensor_map_encoder()(&tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float *>(a.x), dims,
                                            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                                            CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            tl = first_tile(a, false);
    }
    if (tl.smem > 200 * 1024) return MINW_EUNSUPPORTED;
    if (a.codes_out != nullptr && a.O % 16 != 0) return MINW_EUNSUPPORTED;
    const int outb = a.quant_out ? a.qo.bits : 0;
    switch (outb) {
        case 1: return launch_first_bits<1>(a, tl, tm, s);
        case 2: return launch_first_bits<2>(a, tl, tm, s);
        case 3: return launch_first_bits<3>(a, tl, tm, s);
        default: return launch_first_bits<0>(a, tl, tm, s);
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
