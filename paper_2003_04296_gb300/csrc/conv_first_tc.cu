// conv_first_tc.cu -- the first layer of a MINW-Net (Sec. III-E) on the tensor
// cores, with the same output levels as the fp32 fmaf chain of conv_first.cu.
//
// The first layer keeps its fp32 input (and, for the ResNet stem, fp32
// weights), so its product is not an exact integer contraction.  Its output
// is only the next layer's levels, though: the level of an output is a step
// function of the fp32 chain value acc (one fmaf per tap over (c, ky, kx),
// padded taps skipped) with per-channel breakpoints T_u, decided as
// [sigma acc < T_u].  This kernel computes an approximation D of acc on the
// tensor cores together with a rigorous bound E >= |D - acc|, takes every
// decision with |sigma D - T_u| > E from D, and recomputes acc exactly (the
// same fmaf chain) for the few outputs whose decision the bound leaves open.
// The levels written are therefore those of the fp32 chain, bit for bit.
//
// D: every input x is split into two fp16 pieces, x1 = fp16(x) and
// x2 = fp16(x - x1) (|x - x1 - x2| <= max(2^-22 |x|, 2^-25)); every weight,
// scaled per channel by a power of two 2^e (so that its largest magnitude
// lies in [2^13, 2^14)), into w1 = fp16(w 2^e) and w2 = fp16(w 2^e - w1)
// (w2 = 0 for quantized weights: the levels are exact in fp16).  Products
// of fp16 pieces are exact in fp32; kind::f16 MMAs sum x1 w1 + x2 w1
// (+ x1 w2) with fp32 accumulators in TMEM, so D = 2^e acc up to the
// dropped piece products, the accumulation and the chain's own rounding.
// The bound per output (pixel p, channel o), in units of the scaled sum:
//   E = W1s_o (c1 maxabs_p + 2^-25) + K 2^-25 maxabs_p,
// with W1s_o = sum_k |w 2^e| and maxabs_p = max |x| over the pixel's taps
// (so sum |x w 2^e| <= maxabs_p W1s_o), and
//   c1 = 1.02 ((4 + 1.002 m + 2^-10 m') 2^-22 + 1.01 K 2^-24):
// the representation errors of x and w and the dropped x2 w2 (2^-22 each),
// at most 2^-22 per product for the tensor core's fp32 accumulation (twice
// one fp32 rounding per product) over the m products summed with x1 w1 and
// the m' small products (at most 2^-10 of the main ones) summed apart, the
// fp32 add of the two accumulators, and gamma_K for the chain's K roundings.
// Where 4 O TMEM columns fit, x1 w1 has an accumulator of its own (m = K,
// m' = 2K or K); else all products share one (m = 2K or 3K, m' = 0).  A
// pixel with max |x| >= 2^15 (or a non-finite x) has maxabs = inf: all of
// its outputs are recomputed.
//
// Tiling: persistent CTAs, one per SM; tile = 128 consecutive output pixels
// of one image (MMA M) x all O channels (MMA N = O <= 256); K blocks of 32
// taps.  Shared memory holds the weight pieces of every K block and the fp32
// weights of the exact recompute (both built once per CTA), a ring of input
// patches (one TMA box each, zero outside the image, as in conv_first.cu) and
// a ring of A blocks (128 rows of [x1 | x2] pieces, 64 bytes each, in
// 128-byte swizzled rows, built by four warps from the patch).
// Warp roles (448 threads): warp 0 issues the patch boxes, warp 1 owns TMEM
// and issues the MMAs (two accumulators: the epilogue of one tile overlaps
// the MMAs of the next), warps 2-5 build the A blocks (one pixel row per
// thread) and warps 6-13 run the epilogue (two per TMEM lane quarter, each
// half of the channels): decisions, the exact recompute of open decisions
// (one per lane, spread over the warp), and stores of the next layer's codes
// or bit-planes.  Every wait is bounded; a wait that runs out sets the
// kernel's error flag and the CTA winds down.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>

#include "kernels.cuh"

namespace minw {

__device__ int g_first_tc_error = 0;

namespace ftc {

constexpr int NT = 448;
constexpr int BUILD0 = 2, NBUILD = 4, EPI0 = 6, NEPI = 8;

struct Params {
    int B, C, H, W, O, kh, kw, S, pad, Ho, Wo, npix;
    int K;                 // C kh kw
    int nkb;               // K blocks of 32 taps
    int nsets;             // 2 (x1 w1 + x2 w1) or 3 (+ x1 w2)
    int split;             // x1 w1 in one accumulator, the small products in another (4 O <= 512 columns)
    int tiles_img, tiles;  // 128-pixel tiles per image, in all
    int Rmax, RP, x0, xsh; // patch rows, row pitch (floats), first box column, box column of image column -pad
    uint32_t patch_floats; // per patch slot (a multiple of 32)
    int NP, SA;            // patch slots, A block slots
    uint32_t b_block;      // bytes of one weight K block (O rows of 128 bytes)
    uint32_t idesc, tmem_cols;
    uint32_t off_a, off_patch, off_w32, off_chan, off_koff, off_max, off_scr, off_bar;
    float c1;
    int nl;                // levels of the output quantizer
    const float *x;
    const float *w;        // latent [O][K] (when wt is null)
    const float *wt;       // prepared [K][O] (nullable)
    const float *cscale;
    int quant_w;
    QParams qw;
    const float *thr;      // fp32 breakpoints [O][8] (nullable)
    const float *scale, *shift;
    QParams qo;
    uint32_t *planes_out;
    uint8_t *codes_out;
    int codes4;
    long long wait_cycles;
    int stall;
};

__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void bar_init(uint64_t *b, uint32_t n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(su32(b)), "r"(n));
}
__device__ __forceinline__ void bar_arrive(uint64_t *b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(su32(b)) : "memory");
}
__device__ __forceinline__ bool bar_try(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, 100000;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(su32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait: false (and the error flag set) after limit SM clocks.
__device__ __forceinline__ bool bar_wait(uint64_t *b, uint32_t parity, long long limit) {
    if (bar_try(b, parity)) return true;
    const long long t0 = clock64();
    while (!bar_try(b, parity)) {
        if (clock64() - t0 > limit) {
            atomicExch(&g_first_tc_error, 1);
            return false;
        }
    }
    return true;
}

__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }
// Generic-proxy writes to shared memory made visible to the tensor core.
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }

// K-major operand rows of 128 bytes with the 128-byte swizzle (8-row groups 1024 bytes apart).
__device__ __forceinline__ uint64_t desc128(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// fp16 x fp16 -> fp32, issued by one elected lane of the converged MMA warp.
__device__ __forceinline__ void mma_f16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                        uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p, e;\n .reg .b32 r;\n setp.ne.b32 p, %4, 0;\n elect.sync r|e, 0xffffffff;\n"
        " @e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}
__device__ __forceinline__ void mma_commit(uint64_t *b) {
    asm volatile("{\n .reg .pred e;\n .reg .b32 r;\n elect.sync r|e, 0xffffffff;\n"
                 " @e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}\n" ::"r"(su32(b))
                 : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
          "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
          "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

// The fp32 weight of tap k, channel o, as the chain uses it.
__device__ __forceinline__ float weight(const Params &p, int k, int o) {
    if (p.wt != nullptr) return __ldg(p.wt + (long long)k * p.O + o);
    float v = __ldg(p.w + (long long)o * p.K + k);
    if (p.quant_w) v = level_value(v * (p.cscale ? __ldg(p.cscale + o) : p.qw.scale), p.qw);
    return v;
}

__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
    const __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// Per-channel record of the epilogue (16 floats, one 64-byte row per channel):
// sigma, the bound's coefficients A and B (E = A maxabs + B), the scaled
// breakpoints -T_u 2^e, the unscaled -T_u of the exact recompute, and 2^e.
constexpr int CREC = 16, R_SG = 0, R_A = 1, R_B = 2, R_NTS = 3, R_NT = 9, R_SC = 15;

// Compile-time first-layer shapes (the taps and their patch offsets unroll):
// 1 = 3 channels 3 x 3 stride 1 (CIFAR), 2 = 3 channels 7 x 7 stride 2 (ResNet stem), 0 = any.
template <int SHAPE> struct Shape { static constexpr int C = 0, KH = 0, KW = 0, S = 0, K = 0; };
template <> struct Shape<1> { static constexpr int C = 3, KH = 3, KW = 3, S = 1, K = 27; };
template <> struct Shape<2> { static constexpr int C = 3, KH = 7, KW = 7, S = 2, K = 147; };

// Input of tap k of the pixel whose patch origin is pat (0 past the last tap).
template <int SHAPE>
__device__ __forceinline__ float tap(const float *pat, const int *sK, int k, int K, int Rmax, int RP) {
    if constexpr (SHAPE == 0) {
        return k < K ? pat[sK[min(k, K - 1)]] : 0.0f;
    } else {
        constexpr int KH = Shape<SHAPE>::KH, KW = Shape<SHAPE>::KW;
        if (k >= Shape<SHAPE>::K) return 0.0f;
        const int c = k / (KH * KW), rr = k - c * (KH * KW), ky = rr / KW, kx = rr - ky * KW;
        return pat[(c * Rmax + ky) * RP + kx];
    }
}

template <int OUTB, int SHAPE>
__global__ void __launch_bounds__(NT, 1)
    first_tc_kernel(const __grid_constant__ Params p, const __grid_constant__ CUtensorMap tmX) {
    constexpr int NL = OUTB == 1 ? 2 : (OUTB == 2 ? 3 : 7);
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *smem = smem_raw + ((1024u - (su32(smem_raw) & 1023u)) & 1023u);
    uint8_t *sB = smem;                                             // [nkb] weight K blocks
    uint8_t *sA = smem + p.off_a;                                   // [SA] A blocks
    float *sP = reinterpret_cast<float *>(smem + p.off_patch);      // [NP] patches
    float *sW = reinterpret_cast<float *>(smem + p.off_w32);        // [O][Ks] fp32 weights of the chain
    float *sC = reinterpret_cast<float *>(smem + p.off_chan);       // [O][CREC] channel records
    uint32_t *sOpen = reinterpret_cast<uint32_t *>(sC + (size_t)p.O * CREC);   // [O / 32] always-open channels
    int *sK = reinterpret_cast<int *>(smem + p.off_koff);           // [K] patch offset of each tap
    float *sM = reinterpret_cast<float *>(smem + p.off_max);        // [NP][128] maxabs per pixel row
    uint32_t *sS = reinterpret_cast<uint32_t *>(smem + p.off_scr);  // [NEPI][32] recompute lists
    uint64_t *pfull = reinterpret_cast<uint64_t *>(smem + p.off_bar);
    uint64_t *pempty = pfull + p.NP;
    uint64_t *mfull = pempty + p.NP;
    uint64_t *afull = mfull + p.NP;
    uint64_t *aempty = afull + p.SA;
    uint64_t *tfull = aempty + p.SA;     // [2]
    uint64_t *tempty = tfull + 2;        // [2]
    uint64_t *tstall = tempty + 2;       // timeout-path test: a barrier nothing completes
    uint64_t *wready = tstall + 1;       // weight pieces and channel records in place
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(wready + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int O = p.O;
    constexpr int KC = Shape<SHAPE>::K;
    const int K = SHAPE ? KC : p.K;
    const int nkb = SHAPE ? (KC + 31) / 32 : p.nkb;
    const int S = SHAPE ? Shape<SHAPE>::S : p.S;
    const int Rmax = p.Rmax, RP = p.RP;
    const int Ks = K | 1;                 // odd row stride of the fp32 weights: lanes on distinct channels,
                                          // same tap, hit distinct banks

    if (threadIdx.x == 0) {
        for (int i = 0; i < p.NP; ++i) {
            bar_init(&pfull[i], 1);
            bar_init(&pempty[i], NBUILD + NEPI);
            bar_init(&mfull[i], NBUILD);
        }
        for (int i = 0; i < p.SA; ++i) {
            bar_init(&afull[i], NBUILD);
            bar_init(&aempty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            bar_init(&tfull[i], 1);
            bar_init(&tempty[i], NEPI);
        }
        bar_init(tstall, 1);
        bar_init(wready, NEPI);
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(su32(tmem_slot)),
                     "r"(p.tmem_cols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n");
    }
    if (SHAPE == 0) {
        const int khw = p.kh * p.kw;
        for (int k = threadIdx.x; k < K; k += NT) {
            const int c = k / khw, rr = k - c * khw, ky = rr / p.kw, kx = rr - (rr / p.kw) * p.kw;
            sK[k] = (c * Rmax + ky) * RP + kx;
        }
    }
    for (int g = threadIdx.x; g < O / 32; g += NT) sOpen[g] = 0u;
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem_base = *tmem_slot;
    pdl_trigger();

    const int npix = p.npix;
    if (warp == 0) {
        // ---------------- patch producer ----------------
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];\n" ::"l"(reinterpret_cast<uint64_t>(&tmX)) : "memory");
            pdl_wait();                       // the image may come from an earlier kernel
            int n = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x, ++n) {
                const int slot = n % p.NP, lap = n / p.NP;
                if (lap > 0 && !bar_wait(&pempty[slot], (uint32_t)(lap - 1) & 1u, p.wait_cycles)) { ok = false; break; }
                const int b = t / p.tiles_img, p0 = (t - b * p.tiles_img) * 128;
                const uint32_t bytes = (uint32_t)sizeof(float) * (uint32_t)(p.C * Rmax * RP);
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(su32(&pfull[slot])),
                             "r"(bytes)
                             : "memory");
                asm volatile(
                    "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
                    " [%0], [%1, {%2, %3, %4, %5}], [%6];\n" ::"r"(su32(sP + (size_t)slot * p.patch_floats)),
                    "l"(reinterpret_cast<uint64_t>(&tmX)), "r"(p.x0), "r"((p0 / p.Wo) * S - p.pad), "r"(0), "r"(b),
                    "r"(su32(&pfull[slot]))
                    : "memory");
            }
            // every box this thread issued has landed before the CTA exits
            for (int j = n > p.NP ? n - p.NP : 0; j < n; ++j)
                if (!bar_wait(&pfull[j % p.NP], (uint32_t)(j / p.NP) & 1u, p.wait_cycles)) break;
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        bool alive = __all_sync(0xffffffffu, bar_wait(wready, 0u, p.wait_cycles));
        if (alive && p.stall && !__all_sync(0xffffffffu, bar_wait(tstall, 0u, p.wait_cycles))) alive = false;
        fence_after();
        const uint32_t sa0 = su32(sA), sb0 = su32(sB);
        const uint32_t acols = p.split ? 2u * (uint32_t)O : (uint32_t)O;   // columns of one buffer
        int n = 0;
        for (int t = blockIdx.x; t < p.tiles && alive; t += gridDim.x, ++n) {
            const int ab = n & 1, use = n >> 1;
            if (use > 0 && !__all_sync(0xffffffffu, bar_wait(&tempty[ab], (uint32_t)(use - 1) & 1u, p.wait_cycles)))
                break;
            fence_after();
            const uint32_t dmain = tmem_base + (uint32_t)ab * acols;
            const uint32_t dsmall = p.split ? dmain + (uint32_t)O : dmain;
            uint32_t acc1 = 0u, acc2 = p.split ? 0u : 1u;
            for (int kbi = 0; kbi < nkb; ++kbi) {
                const int g = n * nkb + kbi, slot = g % p.SA;
                if (!__all_sync(0xffffffffu, bar_wait(&afull[slot], (uint32_t)(g / p.SA) & 1u, p.wait_cycles))) {
                    alive = false;
                    break;
                }
                fence_after();
                const uint32_t a = sa0 + (uint32_t)slot * 16384u;
                const uint32_t b = sb0 + (uint32_t)kbi * p.b_block;
                // A rows [x1 | x2], B rows [w1 | w2] (64 bytes each); two K = 16 steps per piece.
                // x1 w1 into the main accumulator; x2 w1 (+ x1 w2) into the small one (split) or the same
#pragma unroll
                for (int s = 0; s < 2; ++s) {
                    mma_f16(dmain, desc128(a + 32u * s), desc128(b + 32u * s), p.idesc, acc1);
                    acc1 = 1u;
                    if (!p.split && acc2 == 0u) acc2 = 1u;
                    mma_f16(dsmall, desc128(a + 64u + 32u * s), desc128(b + 32u * s), p.idesc, acc2);
                    acc2 = 1u;
                    if (p.nsets == 3) mma_f16(dsmall, desc128(a + 32u * s), desc128(b + 64u + 32u * s), p.idesc, 1u);
                }
                mma_commit(&aempty[slot]);
            }
            if (!alive) break;
            mma_commit(&tfull[ab]);
        }
    } else if (warp < EPI0) {
        // ---------------- A builders: one pixel row per thread ----------------
        const int r = (warp - BUILD0) * 32 + lane;
        int n = 0;
        bool alive = true;
        for (int t = blockIdx.x; t < p.tiles && alive; t += gridDim.x, ++n) {
            const int pslot = n % p.NP;
            if (!__all_sync(0xffffffffu, bar_wait(&pfull[pslot], (uint32_t)(n / p.NP) & 1u, p.wait_cycles))) break;
            const int b = t / p.tiles_img, p0 = (t - b * p.tiles_img) * 128;
            const int px = p0 + r;
            const bool valid = px < npix;
            const int pc = valid ? px : p0;
            const int oy = pc / p.Wo, ox = pc - oy * p.Wo;
            const float *pat = sP + (size_t)pslot * p.patch_floats + (oy - p0 / p.Wo) * S * RP + ox * S + p.xsh;
            uint32_t mb = 0u;          // max |x| as a bit pattern (NaN patterns exceed infinity's)
            auto build = [&](int kbi, uint8_t *row) {
#pragma unroll
                for (int gi = 0; gi < 4; ++gi) {
                    float x1[8], x2[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        float x = tap<SHAPE>(pat, sK, kbi * 32 + 8 * gi + j, K, Rmax, RP);
                        x = valid ? x : 0.0f;
                        mb = max(mb, __float_as_uint(x) & 0x7FFFFFFFu);
                        const float h1 = __half2float(__float2half_rn(x));
                        x1[j] = h1;
                        x2[j] = x - h1;
                    }
                    const uint4 v1 = make_uint4(pack_h2(x1[0], x1[1]), pack_h2(x1[2], x1[3]), pack_h2(x1[4], x1[5]),
                                                pack_h2(x1[6], x1[7]));
                    const uint4 v2 = make_uint4(pack_h2(x2[0], x2[1]), pack_h2(x2[2], x2[3]), pack_h2(x2[4], x2[5]),
                                                pack_h2(x2[6], x2[7]));
                    *reinterpret_cast<uint4 *>(row + ((gi ^ (r & 7)) << 4)) = v1;
                    *reinterpret_cast<uint4 *>(row + (((4 + gi) ^ (r & 7)) << 4)) = v2;
                }
            };
            auto block = [&](int kbi) -> bool {
                const int g = n * nkb + kbi, slot = g % p.SA, lap = g / p.SA;
                if (lap > 0 &&
                    !__all_sync(0xffffffffu, bar_wait(&aempty[slot], (uint32_t)(lap - 1) & 1u, p.wait_cycles)))
                    return false;
                build(kbi, sA + (size_t)slot * 16384u + (size_t)r * 128);
                fence_async_smem();
                __syncwarp();
                if (lane == 0) bar_arrive(&afull[slot]);
                return true;
            };
            if constexpr (SHAPE > 0) {
#pragma unroll
                for (int kbi = 0; kbi < (KC + 31) / 32; ++kbi)
                    if (alive && !block(kbi)) alive = false;
            } else {
                for (int kbi = 0; kbi < nkb && alive; ++kbi)
                    if (!block(kbi)) alive = false;
            }
            // the pixel's bound input for the epilogue: inf where the fp16 pieces do not hold x
            sM[pslot * 128 + r] = mb >= 0x47000000u ? __int_as_float(0x7F800000) : __uint_as_float(mb);
            __syncwarp();
            if (lane == 0) {
                bar_arrive(&mfull[pslot]);
                bar_arrive(&pempty[pslot]);
            }
        }
    } else {
        // ---------------- epilogue warps: weight preparation, then the epilogue ----------------
        const int et = threadIdx.x - EPI0 * 32;   // 0 .. 255
        // the chain's fp32 weights, [O][Ks]
        for (int i = et; i < K * O; i += NEPI * 32) {
            const int k = i / O, o = i - k * O;
            sW[o * Ks + k] = weight(p, k, o);
        }
        asm volatile("bar.sync 1, %0;\n" ::"n"(NEPI * 32) : "memory");
        // channel records (one thread per channel, over the weights in shared memory)
        for (int o = et; o < O; o += NEPI * 32) {
            float wmax = 0.0f, wsum = 0.0f;
            for (int k = 0; k < K; ++k) {
                const float a = fabsf(sW[o * Ks + k]);
                wmax = fmaxf(wmax, a);
                wsum += a;
            }
            int e = 0;
            if (wmax > 0.0f) e = min(40, max(-40, 13 - ilogbf(wmax)));
            const float sc = ldexpf(1.0f, e);
            // sum_k |w 2^e|, rounded upward for the K roundings of the fp32 sum
            const float w1 = wsum * sc * (1.0f + (float)K * 0x1p-23f);
            float th[8];
            if (p.thr != nullptr) {
#pragma unroll
                for (int u = 0; u < 8; ++u) th[u] = __ldg(p.thr + o * 8 + u);
            } else {
                channel_thresholds_f32(__ldg(p.scale + o), __ldg(p.shift + o), p.qo, th);
            }
            // every decision of the channel stays open where its bound or the scaling of a
            // breakpoint by 2^e is not exact (non-finite weights, breakpoints near underflow)
            bool open = !(w1 < __int_as_float(0x7F800000));
            for (int u = 0; u < NL - 1; ++u)
                if (th[u] != 0.0f && fabsf(th[u]) < 0x1p-80f && isfinite(th[u])) open = true;
            float *rec = sC + (size_t)o * CREC;
            rec[R_SG] = th[NL - 1];
            rec[R_A] = fmaf(w1, p.c1, (float)K * 0x1p-25f);
            rec[R_B] = w1 * 0x1p-25f;
            rec[R_SC] = sc;
            for (int u = 0; u < 6; ++u) {
                rec[R_NTS + u] = u < NL - 1 ? mask_breakpoint(th[u] * sc) : 0.0f;
                rec[R_NT + u] = u < NL - 1 ? mask_breakpoint(th[u]) : 0.0f;
            }
            if (open) atomicOr(&sOpen[o >> 5], 1u << (o & 31));
        }
        asm volatile("bar.sync 1, %0;\n" ::"n"(NEPI * 32) : "memory");
        // weight pieces of every K block: rows = channels, 128 bytes = [w1 (32 taps) | w2 (32 taps)]
        // as 8 units of 8 fp16, unit u of row o at (u ^ (o & 7))
        for (int i = et; i < nkb * O * 8; i += NEPI * 32) {
            const int u = i & 7, o = (i >> 3) % O, kbi = (i >> 3) / O;
            const bool second = u >= 4;
            const int k0 = kbi * 32 + 8 * (u & 3);
            const float sc = sC[(size_t)o * CREC + R_SC];
            float v[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int k = k0 + j;
                const float wsc = k < K ? sW[o * Ks + k] * sc : 0.0f;
                const float w1 = __half2float(__float2half_rn(wsc));
                v[j] = second ? wsc - w1 : wsc;      // w2 is rounded by pack_h2 below
            }
            uint8_t *row = sB + (size_t)kbi * p.b_block + (size_t)o * 128;
            *reinterpret_cast<uint4 *>(row + ((u ^ (o & 7)) << 4)) =
                make_uint4(pack_h2(v[0], v[1]), pack_h2(v[2], v[3]), pack_h2(v[4], v[5]), pack_h2(v[6], v[7]));
        }
        fence_async_smem();
        asm volatile("bar.sync 1, %0;\n" ::"n"(NEPI * 32) : "memory");
        if (lane == 0) bar_arrive(wready);

        pdl_wait();                               // the output buffer may be read by an earlier kernel
        const int q = warp & 3, h = (warp - EPI0) >> 2;
        const int r = q * 32 + lane;
        const int NWo = (O + 31) >> 5;
        uint32_t *scr = sS + (warp - EPI0) * 32;
        const int cpw = O / 64;                   // 32-channel chunks per warp (O / 2 channels per half)
        const uint32_t acols = p.split ? 2u * (uint32_t)O : (uint32_t)O;
        int n = 0;
        bool dead = false;
        for (int t = blockIdx.x; t < p.tiles; t += gridDim.x, ++n) {
            const int ab = n & 1, use = n >> 1, pslot = n % p.NP;
            const uint32_t pph = (uint32_t)(n / p.NP) & 1u;
            if (!dead && !bar_wait(&tfull[ab], (uint32_t)use & 1u, p.wait_cycles)) dead = true;
            if (!dead && !bar_wait(&mfull[pslot], pph, p.wait_cycles)) dead = true;
            if (!dead && !bar_wait(&pfull[pslot], pph, p.wait_cycles)) dead = true;
            dead = !__all_sync(0xffffffffu, !dead);
            fence_after();
            const int b = t / p.tiles_img, p0 = (t - b * p.tiles_img) * 128;
            const int oyf = p0 / p.Wo;
            const float *pat0 = sP + (size_t)pslot * p.patch_floats;
            const float mx = sM[pslot * 128 + r];
            const int px = p0 + r;
            const bool valid = px < npix;
            for (int c = 0; c < cpw && !dead; ++c) {
                const int ch0 = h * (O / 2) + 32 * c;
                const uint32_t ta = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)ab * acols + (uint32_t)ch0;
                uint32_t v[32];
                __syncwarp();
                tmem_ld32(ta, v);
                if (p.split) {
                    uint32_t w[32];
                    tmem_ld32(ta + (uint32_t)O, w);
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = __float_as_uint(__uint_as_float(v[j]) + __uint_as_float(w[j]));
                }
                uint32_t M[NL - 1], fl = 0u;
#pragma unroll
                for (int u = 0; u < NL - 1; ++u) M[u] = 0u;
#pragma unroll
                for (int j = 31; j >= 0; --j) {
                    const float *rec = sC + (size_t)(ch0 + j) * CREC;
                    const float4 r0 = *reinterpret_cast<const float4 *>(rec);    // sigma, A, B, -T_1 2^e
                    const float E = fmaf(mx, r0.y, r0.z);
                    const float D = __uint_as_float(v[j]);
                    float d = fmaf(D, r0.x, r0.w);
                    M[0] = __funnelshift_l(__float_as_uint(d), M[0], 1);
                    float dm = fabsf(d);
#pragma unroll
                    for (int u = 1; u < NL - 1; ++u) {
                        d = fmaf(D, r0.x, rec[R_NTS + u]);
                        M[u] = __funnelshift_l(__float_as_uint(d), M[u], 1);
                        dm = fminf(dm, fabsf(d));
                    }
                    // open where min_u |sigma D - T_u 2^e| < E (a NaN D has inf maxabs: opened below)
                    fl = __funnelshift_l(__float_as_uint(dm - E), fl, 1);
                }
                fl |= sOpen[ch0 >> 5];
                if (!(mx < __int_as_float(0x7F800000))) fl = 0xFFFFFFFFu;
                if (!valid) fl = 0u;
                // open decisions: the exact fmaf chain, one output per lane, spread over the warp
                if (__any_sync(0xffffffffu, fl != 0u)) {
                    const uint32_t cnt = __popc(fl);
                    uint32_t excl = cnt;
#pragma unroll
                    for (int dd = 1; dd < 32; dd <<= 1) {
                        const uint32_t y = __shfl_up_sync(0xffffffffu, excl, dd);
                        if (lane >= dd) excl += y;
                    }
                    const uint32_t total = __shfl_sync(0xffffffffu, excl, 31);
                    excl -= cnt;
                    for (uint32_t base = 0; base < total; base += 32) {
                        uint32_t f = fl, idx = excl;
                        while (f) {
                            const int j = __ffs(f) - 1;
                            f &= f - 1u;
                            if (idx >= base && idx < base + 32) scr[idx - base] = ((uint32_t)lane << 8) | (uint32_t)j;
                            ++idx;
                        }
                        __syncwarp();
                        if ((uint32_t)lane < total - base) {
                            const uint32_t e = scr[lane];
                            const int sl = (int)(e >> 8), j = (int)(e & 255u);
                            const int o = ch0 + j;
                            const int ps = p0 + q * 32 + sl;
                            const int oy = ps / p.Wo, ox = ps - oy * p.Wo;
                            const float *pat = pat0 + (oy - oyf) * S * RP + ox * S + p.xsh;
                            const float *wo = sW + o * Ks;
                            // the chain in batches of 16 taps: loads first, then the fmafs in tap order
                            // (a padded tap past K adds fmaf(0, 0, acc) = acc: acc is never -0)
                            float acc = 0.0f;
                            if constexpr (SHAPE > 0) {
#pragma unroll
                                for (int k0 = 0; k0 < KC; k0 += 16) {
                                    float xs[16], ws[16];
#pragma unroll
                                    for (int i = 0; i < 16; ++i) {
                                        xs[i] = tap<SHAPE>(pat, sK, k0 + i, K, Rmax, RP);
                                        ws[i] = k0 + i < KC ? wo[k0 + i] : 0.0f;
                                    }
#pragma unroll
                                    for (int i = 0; i < 16; ++i)
                                        if (k0 + i < KC) acc = fmaf(xs[i], ws[i], acc);
                                }
                            } else {
                                for (int k0 = 0; k0 < K; k0 += 16) {
                                    float xs[16], ws[16];
#pragma unroll
                                    for (int i = 0; i < 16; ++i) {
                                        const int k = min(k0 + i, K - 1);
                                        xs[i] = k0 + i < K ? pat[sK[k]] : 0.0f;
                                        ws[i] = k0 + i < K ? wo[k] : 0.0f;
                                    }
#pragma unroll
                                    for (int i = 0; i < 16; ++i) acc = fmaf(xs[i], ws[i], acc);
                                }
                            }
                            const float *rec = sC + (size_t)o * CREC;
                            uint32_t bits = 0u;
#pragma unroll
                            for (int u = 0; u < NL - 1; ++u)
                                bits |= (__float_as_uint(fmaf(acc, rec[R_SG], rec[R_NT + u])) >> 31) << u;
                            scr[lane] = e | (bits << 16);
                        }
                        __syncwarp();
                        f = fl;
                        idx = excl;
                        while (f) {
                            const int j = __ffs(f) - 1;
                            f &= f - 1u;
                            if (idx >= base && idx < base + 32) {
                                const uint32_t bits = scr[idx - base] >> 16;
#pragma unroll
                                for (int u = 0; u < NL - 1; ++u)
                                    M[u] = (M[u] & ~(1u << j)) | (((bits >> u) & 1u) << j);
                            }
                            ++idx;
                        }
                        __syncwarp();
                    }
                }
                if (valid) {
                    const long long m = (long long)b * npix + px;
                    store_level_masks<OUTB>(M, 32, 32, p.planes_out ? p.planes_out + (m * OUTB) * NWo + (ch0 >> 5) : nullptr,
                                            NWo, p.codes_out ? p.codes_out + ((m * O + ch0) >> p.codes4) : nullptr,
                                            p.codes4 != 0);
                }
            }
            fence_before();
            __syncwarp();
            if (lane == 0 && !dead) {
                bar_arrive(&tempty[ab]);
                bar_arrive(&pempty[pslot]);
            }
        }
    }
    __syncthreads();
    if (warp == 1) {
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(p.tmem_cols));
    }
}

}  // namespace ftc

// ---------------------------------------------------------------- host

int take_first_tc_error() {
    int flag = 0;
    if (cudaMemcpyFromSymbol(&flag, g_first_tc_error, sizeof(int)) != cudaSuccess) return -1;
    if (flag) {
        const int zero = 0;
        if (cudaMemcpyToSymbol(g_first_tc_error, &zero, sizeof(int)) != cudaSuccess) return -1;
    }
    return flag;
}

static size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// The plan of a first layer on the tensor cores, or false where this path
// does not apply (the caller then runs conv_first_kernel): level outputs
// only, O a multiple of 64 up to 256, the image rows 16-byte multiples at a
// 16-byte aligned base, and a patch box and shared memory within limits.
static bool first_tc_plan(const FirstArgs &a, ftc::Params &p) {
    if (!a.quant_out || a.y_out != nullptr || a.O % 64 != 0 || a.O > 256) return false;
    if (a.planes_out == nullptr && a.codes_out == nullptr) return false;
    if (a.W % 4 != 0 || !minw_host::aligned16(a.x) || minw_host::tensor_map_encoder() == nullptr) return false;
    p = ftc::Params{};
    p.B = a.B; p.C = a.C; p.H = a.H; p.W = a.W; p.O = a.O; p.kh = a.kh; p.kw = a.kw; p.S = a.stride;
    p.pad = a.pad; p.Ho = a.Ho; p.Wo = a.Wo; p.npix = a.Ho * a.Wo;
    p.K = a.C * a.kh * a.kw;
    p.nkb = (p.K + 31) / 32;
    if (p.nkb > 8) return false;
    p.nsets = a.quant_w ? 2 : 3;
    p.tiles_img = (p.npix + 127) / 128;
    p.tiles = a.B * p.tiles_img;
    const int rows = std::min(a.Ho, (128 + a.Wo - 2) / a.Wo + 1);   // output rows 128 consecutive pixels touch
    p.Rmax = (rows - 1) * a.stride + a.kh;
    const int Win = (a.Wo - 1) * a.stride + a.kw;
    p.x0 = -((a.pad + 3) / 4) * 4;
    p.xsh = -a.pad - p.x0;
    p.RP = (Win + p.xsh + 3) / 4 * 4;
    if (p.RP > 256 || p.Rmax > 256 || a.C > 256) return false;
    p.patch_floats = (uint32_t)align_up((size_t)a.C * p.Rmax * p.RP, 32);
    p.b_block = (uint32_t)a.O * 128u;
    const int nl = num_levels(a.qo.bits);
    p.nl = nl;
    // the bound's coefficient: representation errors (3 x 2^-22), 2^-22 per product accumulated with
    // the main products (the small ones, 2^-11 of them, count 2^-10 each), one fp32 add of the two
    // accumulators, and the chain's K roundings
    p.split = 4 * a.O <= 512 ? 1 : 0;
    const double m_main = p.split ? (double)p.K : (double)p.nsets * p.K;
    const double m_small = p.split ? (double)(p.nsets - 1) * p.K : 0.0;
    p.c1 = (float)(1.02 * ((4.0 + 1.002 * m_main + 0x1p-10 * m_small) * 0x1p-22 + 1.01 * p.K * 0x1p-24));
    // shared memory: weight pieces, A ring, patch ring, fp32 weights, channel table, taps, maxabs,
    // recompute lists, barriers (three patches and three A blocks in flight where they fit)
    const size_t limit = 227 * 1024 - 1024;
    static const int np_[6] = {4, 3, 3, 2, 2, 1}, sa_[6] = {4, 4, 3, 3, 2, 2};
    for (int cfg = 0; cfg < 6; ++cfg) {
        p.NP = np_[cfg];
        p.SA = sa_[cfg];
        size_t off = (size_t)p.nkb * p.b_block;
        p.off_a = (uint32_t)off;
        off += (size_t)p.SA * 16384u;
        p.off_patch = (uint32_t)off;
        off += (size_t)p.NP * p.patch_floats * sizeof(float);
        p.off_w32 = (uint32_t)off;
        off += align_up((size_t)(p.K | 1) * a.O * sizeof(float), 16);
        p.off_chan = (uint32_t)off;
        off += (size_t)a.O * ftc::CREC * sizeof(float) + align_up((size_t)(a.O / 32) * sizeof(uint32_t), 16);
        p.off_koff = (uint32_t)off;
        off += align_up((size_t)p.K * sizeof(int), 16);
        p.off_max = (uint32_t)off;
        off += (size_t)p.NP * 128 * sizeof(float);
        p.off_scr = (uint32_t)off;
        off += (size_t)ftc::NEPI * 32 * sizeof(uint32_t);
        off = align_up(off, 8);
        p.off_bar = (uint32_t)off;
        off += (size_t)(3 * p.NP + 2 * p.SA + 6) * sizeof(uint64_t) + 16;
        if (off <= limit) {
            p.tmem_cols = 32;
            while (p.tmem_cols < (p.split ? 4u : 2u) * (uint32_t)a.O) p.tmem_cols <<= 1;
            // D fp32, A and B fp16 (kind::f16), K-major, N = O, M = 128
            p.idesc = (1u << 4) | ((uint32_t)(a.O >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
            return true;
        }
    }
    return false;
}

static size_t first_tc_smem(const ftc::Params &p) {
    return (size_t)p.off_bar + (size_t)(3 * p.NP + 2 * p.SA + 6) * sizeof(uint64_t) + 16 + 1024;
}

bool first_tc_supported(const FirstArgs &a) {
    ftc::Params p;
    return first_tc_plan(a, p);
}

template <int OUTB, int SHAPE>
static minw_status launch_first_tc_shape(const ftc::Params &p, const CUtensorMap &tm, cudaStream_t s) {
    static size_t configured = 0;
    const size_t smem = first_tc_smem(p);
    if (smem > configured) {
        if (cudaFuncSetAttribute(ftc::first_tc_kernel<OUTB, SHAPE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem) != cudaSuccess)
            return MINW_ECUDA;
        configured = smem;
    }
    const int sms = minw_host::num_sms() > 0 ? minw_host::num_sms() : 152;
    const int grid = std::min(p.tiles, sms);
    if (minw_host::launch_pdl(ftc::first_tc_kernel<OUTB, SHAPE>, dim3((unsigned)grid), dim3(ftc::NT), smem, s, p,
                              tm) != cudaSuccess)
        return MINW_ECUDA;
    return MINW_OK;
}

// The CIFAR (3 channels, 3 x 3 / 1) and ResNet-stem (3 channels, 7 x 7 / 2) shapes with their
// taps unrolled at compile time, any other shape with a tap table.
template <int OUTB>
static minw_status launch_first_tc_bits(const ftc::Params &p, const CUtensorMap &tm, cudaStream_t s) {
    if (p.C == 3 && p.kh == 3 && p.kw == 3 && p.S == 1) return launch_first_tc_shape<OUTB, 1>(p, tm, s);
    if (p.C == 3 && p.kh == 7 && p.kw == 7 && p.S == 2) return launch_first_tc_shape<OUTB, 2>(p, tm, s);
    return launch_first_tc_shape<OUTB, 0>(p, tm, s);
}

minw_status launch_first_tc(const FirstArgs &a, cudaStream_t s) {
    ftc::Params p;
    if (!first_tc_plan(a, p)) return MINW_EUNSUPPORTED;
    p.x = a.x; p.w = a.w; p.wt = a.wt; p.cscale = a.cscale; p.quant_w = a.quant_w; p.qw = a.qw;
    p.thr = a.thr; p.scale = a.scale; p.shift = a.shift; p.qo = a.qo;
    p.planes_out = a.planes_out; p.codes_out = a.codes_out; p.codes4 = a.codes4;
    p.wait_cycles = (long long)minw_host::plan_options().wait_cycles;
    p.stall = minw_host::take_stall(MINW_STALL_CONV_FIRST);
    CUtensorMap tm;
    memset(&tm, 0, sizeof(tm));
    const cuuint64_t dims[4] = {(cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.C, (cuuint64_t)a.B};
    const cuuint64_t strides[3] = {(cuuint64_t)a.W * 4, (cuuint64_t)a.H * a.W * 4, (cuuint64_t)a.C * a.H * a.W * 4};
    const cuuint32_t box[4] = {(cuuint32_t)p.RP, (cuuint32_t)p.Rmax, (cuuint32_t)a.C, 1u};
    const cuuint32_t es[4] = {1u, 1u, 1u, 1u};
    if (minw_host::tensor_map_encoder()(&tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float *>(a.x), dims,
                                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                                        CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return MINW_EUNSUPPORTED;
    switch (a.qo.bits) {
        case 1: return launch_first_tc_bits<1>(p, tm, s);
        case 2: return launch_first_tc_bits<2>(p, tm, s);
        default: return launch_first_tc_bits<3>(p, tm, s);
    }
}

}  // namespace minw
