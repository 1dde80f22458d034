// conv_tc.cu -- tensor-core path of the quantized convolution (tcgen05).
//
// The levels of Sec. IV-A are exact powers of two in integer units
// ({0, +-1, +-2, +-4}), so their FP8 E4M3 encodings multiply exactly and
// every partial sum is an integer of magnitude <= 16 * K < 2^24: an fp32
// accumulator holds the convolution exactly.  The kernel therefore runs the
// XNOR/SHIFT products of Table I as a dense FP8 contraction on the 5th-gen
// tensor cores (tcgen05.mma kind::f8f6f4, fp32 accumulators in TMEM).
//
// Implicit GEMM: M = 128 output pixels per CTA tile (a bb x bh x bw block of
// images x rows x columns), N = BN output channels, K = taps x C taken as one
// 128-channel chunk of one tap per pipeline stage.  Per stage:
//   - one TMA 4D box {128 ch, bw, bh, bb} of the NHWC activation codes at the
//     tap's shifted coordinates (out-of-range rows and columns arrive as zero
//     bytes = level 0: the zero padding of the dequantized tensor), and
//   - one TMA 2D box {128, BN} of the [O][kh][kw][C] weight codes,
// both with 128-byte swizzle, i.e. the canonical K-major layout the MMA reads.
// Persistent CTAs (one per SM) walk the tiles; the stage ring runs across tile
// boundaries, and two TMEM accumulators let the epilogue of one tile overlap
// the MMAs of the next.  Warp roles (352 threads): warp 0 issues the
// activation TMA boxes and warp 10 the weight boxes, warp 1 owns TMEM and
// issues MMAs (4 x K=32 per stage), warps 2-9 drain TMEM (two per lane
// quarter, each half of the accumulator columns) and run the fused epilogue: 2x2 max pool via warp
// shuffles on the exact accumulators, then BN + HardTanh + quantize as
// per-channel integer thresholds (bit-identical to the fp32 chain, see
// common.cuh), and stores of the next layer's codes or bit-planes; raw int32
// or fp32 NCHW outputs go through fmaf as in the paper's block.
//
// Every mbarrier wait is bounded (about one second of clock64); a wait that
// runs out sets the device error flag read by minw_get_last_device_error, the
// CTA stops issuing work, drains its own TMA loads and frees its TMEM.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdlib.h>

#include <mutex>

#include "kernels.cuh"

namespace minw {

__device__ int g_device_error = 0;

namespace tc {

constexpr int NT = 352;                 // 11 warps: TMA (A), MMA, 8 epilogue, TMA (B)
constexpr int EPI_WARPS = 8;            // two per TMEM lane quarter, each half of the columns
constexpr int B_WARP = 2 + EPI_WARPS;   // the weight-box TMA warp


struct Params {
    int B, C, H, W, O, kh, kw, pad, Ho, Wo;
    int stride;                // 1 or 2 (TMA element strides)
    int ck;                    // channels per K chunk
    int esize;                 // operand bytes: 1 (E4M3 level codes) or 2 (bf16)
    int cb;                    // bytes of one row of a K chunk: 128 (128-byte swizzle) or 64 (64-byte swizzle);
                               // = ck for E4M3 level codes, 2 ck for bf16 operands
    uint32_t a_bytes;          // activation box bytes of one K block: 128 rows x cb
    uint32_t b_bytes;          // weight box bytes of one K block: BN rows x cb
    int trans;                 // 1: tile = 128 output channels (MMA M) x 256 pixels (MMA N)
    int mrows;                 // output pixels per tile: 128, or 256 when trans
    int acc_cols;              // TMEM columns of one accumulator: BN, or 256 when trans
    int kps;                   // K blocks per pipeline stage (1 or 2): a stage holds kps activation
                               // boxes, then kps weight boxes, and is released by one commit
    int bw, bh, bb, nbx, nby, nbb, ntn;
    int BN, nck, nk, S;
    uint32_t stage_bytes, idesc, tmem_cols;
    const float *thr;          // precomputed breakpoints [O][nlev] (nullable)
    int nlev;                  // levels of the output quantizer
    int ksplit;                // K slices per output tile (1: no split)
    int cl;                    // CTAs per cluster: 2 for CTA pairs, else 1
    int dup;                   // channel-major 64-channel layer: the weight rows loaded twice (MMA rows
                               // 64 .. 127 repeat 0 .. 63), so that all eight epilogue warps hold channels
    int pair;                  // CTA pairs (cl = 2): one cta_group::2 MMA of M = 256 pixels per pair, each
                               // CTA holding its 128 pixels and half of the weight rows
    int tiles_mp;              // pixel tiles per channel tile, padded to a multiple of cl (even for pairs)
    int32_t *part;             // split-K: int32 partial sums [ksplit][tiles][128][BN]
    // residual blocks: y = BN(acc) + shortcut, then HardTanh + quantize
    const uint8_t *res_codes;  // shortcut as level codes [B][Hp][Wp][O] (nullable)
    float res_unit;            // value of one level unit of res_codes (1 or 1/4)
    const float *res_f32;      // shortcut as fp32 NHWC [B][Hp][Wp][O] (nullable)
    float *y_nhwc;             // BN output (before the shortcut) as fp32 NHWC (nullable)
    const float *ythr;         // breakpoints of the output quantizer on y (nullable: computed here)
    uint16_t *hb_out;          // bf16 operands: HardTanh(BN(acc) [+ hb_res]) as bf16 NHWC rows of hb_ld, at hb_off
    int hb_ld, hb_off;
    const float *hb_res;       // fp32 NCHW shortcut (nullable)
    float *hb_z;               // fp32 NCHW copy of the HardTanh output (nullable)
    int32_t *acc_out;
    float *y_out;
    const float *scale, *shift;
    int pool, quant_out;
    QParams qo;
    uint32_t *planes_out;
    uint8_t *codes_out;
    int rowst;                 // row-contiguous stores through a per-warp staging tile: the split-K
                               // partial sums, and fp32 outputs of 1 x 1 images (fully connected)
    int ystage;                // 32-bit words of the staging tiles (8 warps x 32 x 16, or 0)
    int upd;                   // fully connected output: y_out holds latent weights, updated in place
    float upd_lr, upd_2a;      // (Algorithm 1: learning rate and 2 alpha of the mask of Eq. weight)
    int fp4;                   // operands are E2M1 codes, two channels per byte (kind::mxf4, unit scales)
    int out4;                  // codes_out receives E2M1 codes
    int res4;                  // res_codes holds E2M1 codes
    int nacc;                  // TMEM accumulators: 2 (the epilogue of one tile overlaps the MMAs of the
                               // next) or 1 (E2M1 tiles of 256 columns: the scale factors take the rest)
    uint32_t sf_col;           // E2M1 operands: TMEM column of A's unit scale factors (B's at + 32)
    long long wait_cycles;     // limit of every bounded wait (SM clocks)
    int tlanes;                // lanes of each TMA warp that issue loads (stage g belongs to lane g % tlanes)
    int wres;                  // resident weights: each CTA (pair) keeps one channel tile and holds all of its
                               // weight K blocks in shared memory, loaded once; the ring carries activations
                               // only, issued by both TMA warps in turn (no K split)
    uint32_t wres_off;         // byte offset of the resident weights from the shared-memory base
    int stall;                 // timeout-path test: the MMA issuer first waits on a barrier nothing completes
};

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, 100000;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait for the phase with the given parity; false (and the device
// error flag set) when it does not complete within limit SM clocks.  Each
// try_wait may suspend the thread up to 100 us (the hint) until the phase
// completes, so waiting warps do not take issue slots from the MMA thread.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, long long limit) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > limit) {
            atomicExch(&g_device_error, 1);
            return false;
        }
    }
    return true;
}

__device__ __forceinline__ void tma_load_4d(void *dst, const CUtensorMap *map, uint64_t *bar, int c0, int c1,
                                            int c2, int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];\n" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release;\nbarrier.cluster.wait.acquire;\n" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
    return r;
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];\n" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
        : "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile stored as rows of
// ck bytes with the ck-byte swizzle (ck = 128 or 64): 8-row groups 8*ck bytes
// apart.
__device__ __forceinline__ uint64_t sw_desc(uint32_t saddr, int ck) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);   // start address
    d |= (uint64_t)1 << 16;                             // leading byte offset (unused here)
    d |= (uint64_t)((8 * ck) >> 4) << 32;               // stride byte offset: next 8 rows
    d |= (uint64_t)1 << 46;                             // descriptor version
    d |= (uint64_t)(ck == 128 ? 2 : 4) << 61;           // 128- or 64-byte swizzle
    return d;
}

// Value of an E4M3 level code in integer units (0, +-1, +-2, +-4).
__device__ __forceinline__ float code_units(uint32_t c) {
    if ((c & 0x7Fu) == 0u) return 0.0f;
    const float m = (float)(1u << (((c >> 3) & 0xFu) - 7u));
    return (c & 0x80u) ? -m : m;
}

// MMA issue.  The whole issuing warp executes these wrappers with warp-uniform
// operands and one lane, chosen by elect.sync, issues the instruction: the
// descriptors then stay in uniform registers.  Issued from a single divergent
// thread instead, each tcgen05.mma costs that thread about 108 cycles (M = 128,
// N <= 128) and a commit every four MMAs about 40 more; warp-uniform issue
// runs at the tensor pipe's rate (64 cycles at N = 128, 128 at N = 256, with
// the commit hidden).  The elected lane is the same for every call of a
// converged warp, so its commits track the MMAs it issued.
#define MINW_ELECT_PROLOGUE "{\n .reg .pred p, e;\n .reg .b32 r;\n setp.ne.b32 p, %4, 0;\n elect.sync r|e, 0xffffffff;\n"

__device__ __forceinline__ void mma_f8(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
    asm volatile(MINW_ELECT_PROLOGUE
                 " @e tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
                 "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("{\n .reg .pred e;\n .reg .b32 r;\n elect.sync r|e, 0xffffffff;\n"
                 " @e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}\n" ::"r"(
                     smem_u32(bar))
                 : "memory");
}

// bf16 x bf16 -> fp32 (weight-only quantized layers: full-precision bf16
// activations, weights at their exact level values).
__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(MINW_ELECT_PROLOGUE
                 " @e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
                 "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

// CTA pairs (cta_group::2).  The even CTA of a cluster of two issues each MMA
// for both: A = the pair's 256 pixel rows (128 in each CTA's shared memory),
// B = the 256 weight rows (128 in each), D = 128 accumulator lanes in each
// CTA's tensor memory.  Loads of both CTAs complete on the even CTA's barrier.
__device__ __forceinline__ void mma_f8_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
    asm volatile(MINW_ELECT_PROLOGUE
                 " @e tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
                 "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

__device__ __forceinline__ void mma_bf16_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                              uint32_t accumulate) {
    asm volatile(MINW_ELECT_PROLOGUE
                 " @e tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
                 "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

// E2M1 x E2M1 -> fp32 with block scaling (kind::mxf4, 32 elements per
// UE8M0 scale, K = 64 per instruction): every scale factor in tensor memory
// is 2^0, so the products are the plain level products, exact like E4M3's.
// The packed operands halve the bytes per K step, and the instruction covers
// twice the K of an E4M3 one at the same issue cost.
__device__ __forceinline__ void mma_f4(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate, uint32_t sfa, uint32_t sfb) {
    asm volatile(MINW_ELECT_PROLOGUE
                 " @e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%0], %1, %2, %3, [%5], [%6], p;\n}\n"
                 ::"r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate), "r"(sfa), "r"(sfb));
}

__device__ __forceinline__ void mma_f4_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate, uint32_t sfa, uint32_t sfb) {
    asm volatile(MINW_ELECT_PROLOGUE
                 " @e tcgen05.mma.cta_group::2.kind::mxf4.block_scale.scale_vec::2X [%0], %1, %2, %3, [%5], [%6], p;\n}\n"
                 ::"r"(tmem_d), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate), "r"(sfa), "r"(sfb));
}

// Arrive on the barrier at this offset in both CTAs of the pair once the
// pair's MMAs issued so far have completed (an mbarrier signal to each CTA).
__device__ __forceinline__ void mma_commit_pair(uint64_t *bar) {
    asm volatile("{\n .reg .pred e;\n .reg .b32 r;\n elect.sync r|e, 0xffffffff;\n"
                 " @e tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;\n}\n"
                 ::"r"(smem_u32(bar)), "h"((uint16_t)3)
                 : "memory");
}

// Shared::cluster address of the object at this offset in CTA 0 of the cluster.
__device__ __forceinline__ uint32_t cta0_addr(const void *p) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, 0;\n" : "=r"(r) : "r"(smem_u32(p)));
    return r;
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];\n" ::"r"(cluster_addr) : "memory");
}

// Tile loads of a pair: into this CTA's shared memory, completing on the
// barrier at a shared::cluster address (the even CTA's).
__device__ __forceinline__ void tma_load_4d_pair(void *dst, const CUtensorMap *map, uint32_t bar, int c0, int c1,
                                                 int c2, int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];\n" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void tma_load_2d_pair(void *dst, const CUtensorMap *map, uint32_t bar, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];\n" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

// Bounded wait with cluster-scope acquire (arrivals from the other CTA of a pair).
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t *bar, uint32_t parity, long long limit) {
    const long long t0 = clock64();
    while (true) {
        uint32_t ok;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, 100000;\n"
            " selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(ok)
            : "r"(smem_u32(bar)), "r"(parity)
            : "memory");
        if (ok) return true;
        if (clock64() - t0 > limit) {
            atomicExch(&g_device_error, 1);
            return false;
        }
    }
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15}, [%16];\n"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

// 32 columns of this warp's 32 TMEM lanes, without waiting: tmem_wait_ld()
// before the first use of v (it waits for every load this thread issued).
__device__ __forceinline__ void tmem_ld32_nw(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
          "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
          "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory"); }

// Sign bits of 32 values as one word (bit j = sign of x[j]), built as four
// independent 8-bit chains so that the funnel shifts overlap.
__device__ __forceinline__ uint32_t sign_word(const float (&x)[32]) {
    uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int j = 7; j >= 0; --j)
#pragma unroll
        for (int k = 0; k < 4; ++k) w[k] = __funnelshift_l(__float_as_uint(x[8 * k + j]), w[k], 1);
    return w[0] | (w[1] << 8) | (w[2] << 16) | (w[3] << 24);
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

__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(smem_u32(bar)) : "memory");
}

// Compile-time tables of the OUTB-bit output quantizer (see common.cuh).
template <int OUTB>
__device__ __forceinline__ uint32_t code_k(int k) {
    if constexpr (OUTB == 1) return k ? 0x38u : 0xB8u;
    else if constexpr (OUTB == 2) return (uint32_t)((0x3800B8u >> (8 * k)) & 0xFFu);
    else return (uint32_t)((0x0048403800B8C0C8ull >> (8 * k)) & 0xFFull);
}
template <int OUTB>
__device__ __forceinline__ uint32_t planes_k(int k) {
    if constexpr (OUTB == 1) return k ? 0u : 1u;
    else if constexpr (OUTB == 2) return (0x203u >> (4 * k)) & 0x3u;
    else return (uint32_t)((06420357ull >> (3 * k)) & 7ull);
}

// 32 x 32 bit transpose across a warp: lane l holds row l; on return lane j
// holds column j (bit c of lane j's word = bit j of lane c's word).
__device__ __forceinline__ uint32_t transpose32(uint32_t a, int lane) {
    const uint32_t ms[5] = {0xFFFF0000u, 0xFF00FF00u, 0xF0F0F0F0u, 0xCCCCCCCCu, 0xAAAAAAAAu};
#pragma unroll
    for (int k = 0; k < 5; ++k) {
        const int j = 16 >> k;
        const uint32_t m = ms[k];
        const uint32_t q = __shfl_xor_sync(0xffffffffu, a, j);
        a = (lane & j) ? (((q >> j) & ~m) | (a & m)) : ((a & ~m) | ((q << j) & m));
    }
    return a;
}

// Epilogue of one 32-column chunk (16 when tail16 is false) of exact
// accumulators, one tile row per lane, when the only output is the next
// layer's levels.  For each breakpoint u the chunk becomes one 32-bit mask
// M_u (bit j set when channel j's sigma * acc stays below T_u, taken from the
// sign of fmaf(acc, sigma, -T_u): exact, as acc and T_u are integers, and
// never -0, as -T_u = 0 is held as +0), so the
// level index is k = #{u : bit clear}.  A 2x2 max pool of the accumulators
// maps to the masks: for sigma = +1 the pooled level is the window's largest
// (M pooled = AND over the window), for sigma = -1 its smallest (OR).  Bit
// planes and E4M3 codes follow from the masks with bitwise logic.  th: the
// chunk's first channel in rows of tstride floats (-T_1 .. -T_{n-1}, sigma).
template <int OUTB>
__device__ __forceinline__ void mask_chunk_regs(const uint32_t (&v)[32], bool full32, const float *th, int tstride,
                                                uint32_t sig, int pool, int bw, bool writer, int nvalid,
                                                uint32_t *planes, int NWo, uint8_t *codes, bool codes4) {
    constexpr int NL = OUTB == 1 ? 2 : (OUTB == 2 ? 3 : 7);
    uint32_t M[NL - 1];
#pragma unroll
    for (int u = 0; u < NL - 1; ++u) M[u] = 0u;
    if constexpr (NL == 2) {
        // one breakpoint: the 32 sign bits as four independent chains
        float d[32];
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4) {
            const float4 sg4 = *reinterpret_cast<const float4 *>(th + tstride + 4 * j4);
            const float4 nt4 = *reinterpret_cast<const float4 *>(th + 4 * j4);
            d[4 * j4] = fmaf(__uint_as_float(v[4 * j4]), sg4.x, nt4.x);
            d[4 * j4 + 1] = fmaf(__uint_as_float(v[4 * j4 + 1]), sg4.y, nt4.y);
            d[4 * j4 + 2] = fmaf(__uint_as_float(v[4 * j4 + 2]), sg4.z, nt4.z);
            d[4 * j4 + 3] = fmaf(__uint_as_float(v[4 * j4 + 3]), sg4.w, nt4.w);
        }
        M[0] = sign_word(d);
    } else
    // breakpoints of four channels per 128-bit load (rows of tstride floats, channel fastest)
#pragma unroll
    for (int j4 = 7; j4 >= 0; --j4) {
        const float4 sg4 = *reinterpret_cast<const float4 *>(th + (NL - 1) * tstride + 4 * j4);
        float4 nt4[NL - 1];
#pragma unroll
        for (int u = 0; u < NL - 1; ++u) nt4[u] = *reinterpret_cast<const float4 *>(th + u * tstride + 4 * j4);
        const float sg[4] = {sg4.x, sg4.y, sg4.z, sg4.w};
#pragma unroll
        for (int jj = 3; jj >= 0; --jj) {
            const float a = __uint_as_float(v[4 * j4 + jj]);
#pragma unroll
            for (int u = 0; u < NL - 1; ++u) {
                const float nt = jj == 0 ? nt4[u].x : jj == 1 ? nt4[u].y : jj == 2 ? nt4[u].z : nt4[u].w;
                M[u] = __funnelshift_l(__float_as_uint(fmaf(a, sg[jj], nt)), M[u], 1);
            }
        }
    }
    if (pool) {
#pragma unroll
        for (int u = 0; u < NL - 1; ++u) {
            const uint32_t m = M[u];
            const uint32_t n1 = __shfl_xor_sync(0xffffffffu, m, 1);
            const uint32_t a1 = m & n1, o1 = m | n1;
            const uint32_t a2 = a1 & __shfl_xor_sync(0xffffffffu, a1, bw);
            const uint32_t o2 = o1 | __shfl_xor_sync(0xffffffffu, o1, bw);
            M[u] = (sig & a2) | (~sig & o2);
        }
    }
    if (!writer) return;
    store_level_masks<OUTB>(M, nvalid, full32 ? 32 : 16, planes, NWo, codes, codes4);
}

template <int OUTB>
__device__ __forceinline__ void mask_chunk(uint32_t taddr, bool full32, const float *th, int tstride, uint32_t sig,
                                           int pool, int bw, bool writer, int nvalid, uint32_t *planes, int NWo,
                                           uint8_t *codes, bool codes4) {
    uint32_t v[32];
    if (full32) {
        tmem_ld32(taddr, v);
    } else {
        uint32_t v16[16];
        tmem_ld16(taddr, v16);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            v[j] = v16[j];
            v[j + 16] = 0u;
        }
    }
    mask_chunk_regs<OUTB>(v, full32, th, tstride, sig, pool, bw, writer, nvalid, planes, NWo, codes, codes4);
}

// Epilogue of one 32-column chunk (16 when full32 is false) of a residual
// block, one output pixel per lane: y = fmaf(acc, scale, shift), stored as
// fp32 NHWC when asked (the BN output before the shortcut), then y + shortcut
// (one fp32 add) and the next layer's levels from the sign bits of
// y + (-T_u) against the quantizer's own breakpoints on y (HardTanh included),
// through the same level masks as the plain epilogue.
template <int OUTB>
__device__ __forceinline__ void resid_chunk(uint32_t taddr, bool full32, const Params &p, int ob, long long opix,
                                            bool writer, const float *syt, int NWo) {
    uint32_t v[32];
    if (full32) {
        tmem_ld32(taddr, v);
    } else {
        uint32_t v16[16];
        tmem_ld16(taddr, v16);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            v[j] = v16[j];
            v[j + 16] = 0u;
        }
    }
    if (!writer) return;
    const int nvalid = min(32, p.O - ob);                 // a multiple of 16
    const int ncol = full32 ? 32 : 16;
    float y[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        const int o = min(ob + j, p.O - 1);
        y[j] = fmaf(__uint_as_float(v[j]), __ldg(p.scale + o), __ldg(p.shift + o));
    }
    const long long base = opix * p.O + ob;
    if (p.y_nhwc != nullptr) {
        float4 *dst = reinterpret_cast<float4 *>(p.y_nhwc + base);
#pragma unroll
        for (int q4 = 0; q4 < 8; ++q4)
            if (q4 * 4 < nvalid && q4 * 4 < ncol) dst[q4] = make_float4(y[4 * q4], y[4 * q4 + 1], y[4 * q4 + 2], y[4 * q4 + 3]);
    }
    if constexpr (OUTB > 0) {
        if (p.res_codes != nullptr && p.res4) {
            const uint2 *src = reinterpret_cast<const uint2 *>(p.res_codes + base / 2);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                if (h * 16 >= nvalid || h * 16 >= ncol) break;
                const uint2 cv = __ldg(src + h);
                const uint32_t cw[2] = {cv.x, cv.y};
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    y[h * 16 + j] += code_units_e2m1(cw[j >> 3] >> (4 * (j & 7))) * p.res_unit;
            }
        } else if (p.res_codes != nullptr) {
            const uint4 *src = reinterpret_cast<const uint4 *>(p.res_codes + base);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                if (h * 16 >= nvalid || h * 16 >= ncol) break;
                const uint4 cv = __ldg(src + h);
                const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    y[h * 16 + j] += code_units((cw[j >> 2] >> (8 * (j & 3))) & 0xFFu) * p.res_unit;
            }
        } else if (p.res_f32 != nullptr) {
            const float4 *src = reinterpret_cast<const float4 *>(p.res_f32 + base);
#pragma unroll
            for (int q4 = 0; q4 < 8; ++q4) {
                if (q4 * 4 >= nvalid || q4 * 4 >= ncol) break;
                const float4 r = __ldg(src + q4);
                y[4 * q4] += r.x;
                y[4 * q4 + 1] += r.y;
                y[4 * q4 + 2] += r.z;
                y[4 * q4 + 3] += r.w;
            }
        }
        constexpr int NL = OUTB == 1 ? 2 : (OUTB == 2 ? 3 : 7);
        float nt[NL - 1];
#pragma unroll
        for (int u = 0; u < NL - 1; ++u) nt[u] = syt[u];
        uint32_t M[NL - 1];
#pragma unroll
        for (int u = 0; u < NL - 1; ++u) M[u] = 0u;
#pragma unroll
        for (int j = 31; j >= 0; --j)
#pragma unroll
            for (int u = 0; u < NL - 1; ++u) M[u] = __funnelshift_l(__float_as_uint(y[j] + nt[u]), M[u], 1);
        store_level_masks<OUTB>(M, nvalid, ncol, p.planes_out ? p.planes_out + (opix * OUTB) * NWo + (ob >> 5) : nullptr,
                                NWo, p.codes_out ? p.codes_out + (p.out4 ? base / 2 : base) : nullptr, p.out4 != 0);
    }
}

// Work item n (0, 1, ...) of this CTA, or -1 past its last: an (output tile,
// K slice) index w (tile t = w / ksplit, tile t = tn * tiles_m + tm).  By
// default CTA b takes w = b, b + grid, ...; with resident weights, unit u
// (a CTA, or a pair) keeps channel tile tn = u % ntn and walks its pixel
// tiles (the pair's two CTAs on adjacent ones).
__device__ __forceinline__ int cta_item(const Params &p, int n, int items, int tiles_m, int crank) {
    if (!p.wres) {
        const int w = (int)blockIdx.x + n * (int)gridDim.x;
        return w < items ? w : -1;
    }
    const int units = (int)gridDim.x / p.cl, upt = units / p.ntn, u = (int)blockIdx.x / p.cl;
    const int tm = (u / p.ntn + n * upt) * p.cl + crank;
    return tm < tiles_m ? (u % p.ntn) * tiles_m + tm : -1;
}

// OUTB: bits of the quantized output (0 when the launch writes none).
// PAIR: CTA pairs with cta_group::2 MMAs (a kernel uses one CTA group only).
// FMT: operand format -- 0 E4M3 level codes (kind::f8f6f4), 1 bf16 (kind::f16),
// 2 E2M1 level codes (kind::mxf4); all three consume 32 bytes of K per MMA
// step (32, 16 and 64 elements).
// Stores the 16 words u[] of each lane's tile row (row = lane) row-contiguously:
// row rr goes to dst0 + rr * rstride + [0, 16), rows < nrows, columns < ncols.
// The warp transposes through its 32 x 16-word shared tile in 16-byte chunks,
// chunk m of row rr at rr * 4 + (m ^ ((rr >> 1) & 3)) (no bank conflict on the
// writes nor on the reads), so that each 16-byte store instruction covers eight
// 64-byte row segments.  With scale and shift, the words are fp32 accumulators
// and column c stores fmaf(u, scale[c], shift[c]): after the transpose a lane
// holds four fixed columns c = 4 (lane & 3) .. + 3, whose BN values the caller
// passes in sc[] and sh[].  With upd, dst0 holds latent weights w and each
// value g replaces its w by the clipped masked step of sgd_masked.
__device__ __forceinline__ float sgd_masked(float w, float g, float lr, float two_alpha) {
    const float gw = (fabsf(w) <= 1.0f) ? g * two_alpha : 0.0f;
    return fminf(1.0f, fmaxf(-1.0f, fmaf(-lr, gw, w)));
}

__device__ __forceinline__ void rows_store16(uint32_t *sw, const uint32_t (&u)[16], int lane, uint32_t *dst0,
                                             long long rstride, int nrows, int ncols,
                                             const float *sc = nullptr, const float *sh = nullptr,
                                             bool upd = false, float lr = 0.0f, float two_alpha = 0.0f) {
    uint4 *sw4 = reinterpret_cast<uint4 *>(sw);
    __syncwarp();
#pragma unroll
    for (int m = 0; m < 4; ++m)
        sw4[lane * 4 + (m ^ ((lane >> 1) & 3))] = make_uint4(u[4 * m], u[4 * m + 1], u[4 * m + 2], u[4 * m + 3]);
    __syncwarp();
    const int k = lane & 3, c = 4 * k;
    // the update's latent weights: all four loads in flight before any store
    float4 wv[4];
    if (upd) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int rr = 8 * i + (lane >> 2);
            wv[i] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (rr < nrows) {
                const float *wd = reinterpret_cast<const float *>(dst0 + (long long)rr * rstride + c);
                if (c + 4 <= ncols && (reinterpret_cast<uintptr_t>(wd) & 15) == 0) {
                    wv[i] = *reinterpret_cast<const float4 *>(wd);
                } else {
                    if (c < ncols) wv[i].x = wd[0];
                    if (c + 1 < ncols) wv[i].y = wd[1];
                    if (c + 2 < ncols) wv[i].z = wd[2];
                    if (c + 3 < ncols) wv[i].w = wd[3];
                }
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int rr = 8 * i + (lane >> 2);
        uint4 x = sw4[rr * 4 + (k ^ ((rr >> 1) & 3))];
        if (sc != nullptr) {
            x.x = __float_as_uint(fmaf(__uint_as_float(x.x), sc[0], sh[0]));
            x.y = __float_as_uint(fmaf(__uint_as_float(x.y), sc[1], sh[1]));
            x.z = __float_as_uint(fmaf(__uint_as_float(x.z), sc[2], sh[2]));
            x.w = __float_as_uint(fmaf(__uint_as_float(x.w), sc[3], sh[3]));
        }
        if (rr < nrows) {
            uint32_t *d = dst0 + (long long)rr * rstride + c;
            const bool v4 = c + 4 <= ncols && (reinterpret_cast<uintptr_t>(d) & 15) == 0;
            if (upd) {
                float *wd = reinterpret_cast<float *>(d);
                float4 w = wv[i];
                w.x = sgd_masked(w.x, __uint_as_float(x.x), lr, two_alpha);
                w.y = sgd_masked(w.y, __uint_as_float(x.y), lr, two_alpha);
                w.z = sgd_masked(w.z, __uint_as_float(x.z), lr, two_alpha);
                w.w = sgd_masked(w.w, __uint_as_float(x.w), lr, two_alpha);
                if (v4) {
                    *reinterpret_cast<float4 *>(wd) = w;
                } else {
                    if (c < ncols) wd[0] = w.x;
                    if (c + 1 < ncols) wd[1] = w.y;
                    if (c + 2 < ncols) wd[2] = w.z;
                    if (c + 3 < ncols) wd[3] = w.w;
                }
            } else if (v4) {
                *reinterpret_cast<uint4 *>(d) = x;
            } else {
                if (c < ncols) d[0] = x.x;
                if (c + 1 < ncols) d[1] = x.y;
                if (c + 2 < ncols) d[2] = x.z;
                if (c + 3 < ncols) d[3] = x.w;
            }
        }
    }
}

template <int OUTB, bool PAIR, int FMT>
__global__ void __launch_bounds__(NT, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const Params p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // 1024-byte aligned base (the 128-byte swizzle repeats every 1024 bytes);
    // pointer arithmetic on the shared array keeps the shared address space
    uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    constexpr int NL = OUTB == 0 ? 1 : (OUTB == 1 ? 2 : (OUTB == 2 ? 3 : 7));
    // breakpoints [NL][O32] (channels padded to a multiple of 32, channel
    // fastest), then the per-32-channel masks of channels with sigma = +1
    const int O32 = (p.O + 31) & ~31;
    float *sthr = reinterpret_cast<float *>(smem + (size_t)p.S * p.stage_bytes +
                                            (p.wres ? (size_t)p.nk * p.b_bytes : 0));   // after the resident weights
    const int thr_floats = OUTB ? O32 * NL : 0;
    uint32_t *ssig = reinterpret_cast<uint32_t *>(sthr + thr_floats);              // [O32 / 32]
    const int sig_words = OUTB ? O32 / 32 : 0;
    // breakpoints of the output quantizer on y itself (residual blocks), held as -T
    float *syt = reinterpret_cast<float *>(ssig + ((sig_words + 1) & ~1));
    // staging tiles of the row-contiguous stores, one 32 x 16-word tile per epilogue warp
    uint32_t *sy = reinterpret_cast<uint32_t *>(syt + (OUTB ? 8 : 0));
    sy += (4u - ((smem_u32(sy) >> 2) & 3u)) & 3u;            // 16-byte aligned
    uint64_t *full = reinterpret_cast<uint64_t *>(sy + p.ystage);
    uint64_t *empty = full + p.S;
    uint64_t *tfull = empty + p.S;            // [2] accumulator ready
    uint64_t *tempty = tfull + 2;             // [2] accumulator drained
    uint64_t *tstall = tempty + 2;            // timeout-path test: a barrier nothing completes
    uint64_t *wfull = tstall + 1;             // resident weights landed
    uint64_t *sfready = wfull + 1;            // E2M1: the unit scale factors are in tensor memory
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(sfready + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // pixel tiles padded to a multiple of the cluster size: the CTAs of a
    // cluster walk tiles of the same channel tile in lock step (a padded tile
    // reads zero boxes and writes nothing)
    const int tiles_m = p.tiles_mp;
    const int tiles = tiles_m * p.ntn;
    const int items = tiles * p.ksplit;       // (output tile, K slice) work items
    const int crank = PAIR ? (int)cluster_ctarank() : 0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < p.S; ++s) {
            mbar_init(&full[s], p.wres ? 1 : 2);  // one arrival per TMA warp loading the stage (pairs: CTA 0's)
            mbar_init(&empty[s], 1);              // one release per slot (pairs: CTA 0 commits to both CTAs)
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], PAIR ? 2 * EPI_WARPS : EPI_WARPS);   // pairs: both CTAs' epilogues
        }
        mbar_init(tstall, 1);
        mbar_init(wfull, 1);
        mbar_init(sfready, PAIR ? 8 : 4);     // one arrival per filling warp (pairs: both CTAs' on CTA 0)
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 1) {
        if constexpr (PAIR) {      // one warp of each CTA of the pair allocates the same columns in both
            asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                             smem_u32(tmem_slot)),
                         "r"(p.tmem_cols));
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;\n");
        } else {
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(
                             smem_u32(tmem_slot)),
                         "r"(p.tmem_cols));
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n");
        }
    }
    fence_before();
    __syncthreads();
    if constexpr (PAIR) cluster_sync_all();   // every barrier of the pair is initialised
    fence_after();
    const uint32_t tmem_base = *tmem_slot;
    // set-up done: the next kernel may start its own.  The TMA producers start
    // at once; the epilogue warps first write the E2M1 unit scale factors
    // (the MMA issuer waits for them on sfready) and load the breakpoints.
    pdl_trigger();

    if (warp == 0 || warp == B_WARP) {
        if (lane < p.tlanes) {
            // ---------------- TMA producers: warp 0 activations, warp 10 weights ----------------
            // Lane l of a warp owns the pipeline stages g with g % tlanes == l
            // (own slot waits, own arrival on the stage's barrier).  With resident
            // weights, warp 10 first loads every weight K block of its channel
            // tile once, then both warps issue activation stages in turn.
            const bool wwarp = warp == B_WARP;
            const bool act = !wwarp || p.wres;     // this warp issues activation boxes
            const CUtensorMap *map = act ? &tmA : &tmB;
            if (lane == 0) asm volatile("prefetch.tensormap [%0];\n" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
            const uint32_t bytes = act ? p.a_bytes : p.b_bytes;   // per K block
            const int bslice = PAIR ? p.BN / 2 : p.BN;   // weight rows this CTA loads
            // pairs: this operand's loads of both CTAs complete on CTA 0's barrier, whose
            // producers alone arrive (expecting both CTAs' bytes)
            const bool arrive = !PAIR || crank == 0;
            const int nissue = p.wres ? 2 * p.tlanes : p.tlanes;          // issuers of this operand
            const int myid = (p.wres && wwarp) ? p.tlanes + lane : lane;
            if (p.wres && wwarp && lane == 0) {
                // the channel tile's weights, all K blocks, once
                const int o0 = (((int)blockIdx.x / p.cl) % p.ntn) * p.BN;
                uint8_t *wres = smem + p.wres_off;
                if (arrive) mbar_expect_tx(wfull, (uint32_t)p.nk * p.b_bytes * (PAIR ? 2u : 1u));
                const uint32_t fb = PAIR ? cta0_addr(wfull) : 0u;
                for (int kb = 0; kb < p.nk; ++kb) {
                    const int kx_ = FMT == 2 ? (kb * p.ck) >> 1 : kb * p.ck;
                    uint8_t *sb = wres + (size_t)kb * p.b_bytes;
                    if constexpr (PAIR) {
                        tma_load_2d_pair(sb, &tmB, fb, kx_, o0 + crank * bslice);
                    } else {
                        tma_load_2d(sb, &tmB, wfull, kx_, o0);
                        if (p.dup) tma_load_2d(sb + (size_t)64 * p.cb, &tmB, wfull, kx_, o0);
                    }
                }
            }
            if (act) pdl_wait();                  // activations come from the previous kernel
                                                  // (the weights above do not: they load before)
            int g = 0, s = 0, lap = 0;             // stages walked, ring slot, ring lap
            bool alive = true;
            for (int n = 0, w; alive && (w = cta_item(p, n, items, tiles_m, crank)) >= 0; ++n) {
                const int t = w / p.ksplit, kp = w - t * p.ksplit;
                const int kb = (int)((long long)kp * p.nk / p.ksplit), ke = (int)((long long)(kp + 1) * p.nk / p.ksplit);
                const int tn = t / tiles_m, tm = t - tn * tiles_m;
                const int xb = tm % p.nbx, yb = (tm / p.nbx) % p.nby, bbk = tm / (p.nbx * p.nby);
                const int x0 = xb * p.bw * p.stride - p.pad, y0 = yb * p.bh * p.stride - p.pad, b0 = bbk * p.bb;
                const int o0 = tn * p.BN;
                // channel chunk, tap and weight column of stage kb
                const int tap0 = kb / p.nck;
                int c0 = (kb - tap0 * p.nck) * p.ck, ky = tap0 / p.kw, kx = tap0 - (tap0 / p.kw) * p.kw;
                int kcol = kb * p.ck;
                for (int ks = kb; ks < ke; ks += p.kps, ++g) {
                    const bool mine = g % nissue == myid;
                    // slot reuse: wait until the MMAs of the previous lap released it
                    if (mine && lap > 0 && !mbar_wait(&empty[s], (lap - 1) & 1, p.wait_cycles)) { alive = false; break; }
                    uint8_t *sa = smem + (size_t)s * p.stage_bytes;
                    const int nb = min(p.kps, ke - ks);           // K blocks in this stage
                    if (mine && arrive) mbar_expect_tx(&full[s], (uint32_t)nb * bytes * (PAIR ? 2u : 1u));
                    const uint32_t fb = (PAIR && mine) ? cta0_addr(&full[s]) : 0u;
                    for (int j = 0; j < nb; ++j) {
                        // tensor-map x coordinates: elements, or bytes for packed E2M1
                        const int cx = FMT == 2 ? c0 >> 1 : c0, kx_ = FMT == 2 ? kcol >> 1 : kcol;
                        if (mine) {
                            if constexpr (PAIR) {
                                if (act)
                                    tma_load_4d_pair(sa + (size_t)j * p.a_bytes, &tmA, fb, cx, x0 + kx, y0 + ky, b0);
                                else
                                    tma_load_2d_pair(sa + (size_t)p.kps * p.a_bytes + (size_t)j * p.b_bytes, &tmB, fb,
                                                     kx_, o0 + crank * bslice);
                            } else if (act)
                                tma_load_4d(sa + (size_t)j * p.a_bytes, &tmA, &full[s], cx, x0 + kx, y0 + ky, b0);
                            else {
                                uint8_t *sb = sa + (size_t)p.kps * p.a_bytes + (size_t)j * p.b_bytes;
                                tma_load_2d(sb, &tmB, &full[s], kx_, o0);
                                if (p.dup) tma_load_2d(sb + (size_t)64 * p.cb, &tmB, &full[s], kx_, o0);
                            }
                        }
                        kcol += p.ck;
                        c0 += p.ck;
                        if (c0 == p.C) {
                            c0 = 0;
                            if (++kx == p.kw) { kx = 0; ++ky; }
                        }
                    }
                    if (++s == p.S) { s = 0; ++lap; }
                }
            }
            // drain: every load this lane issued has landed before the CTA can exit
            // (pairs: the MMAs that read the last stages have completed)
            for (int j = g > p.S ? g - p.S : 0; j < g; ++j)
                if (j % nissue == myid &&
                    !(PAIR ? mbar_wait(&empty[j % p.S], (j / p.S) & 1, p.wait_cycles)
                           : mbar_wait(&full[j % p.S], (j / p.S) & 1, p.wait_cycles)))
                    break;
            if (p.wres && wwarp && lane == 0 && (!PAIR || crank == 0)) mbar_wait(wfull, 0u, p.wait_cycles);
        }
    } else if (warp == 1) {
        if (!PAIR || crank == 0) {
            // ---------------- MMA issuer (pairs: CTA 0 issues for both) ----------------
            // The whole warp runs this loop with warp-uniform values; one elected
            // lane issues each MMA and commit (see mma_f8).  Every wait's outcome
            // is made warp-uniform, so the warp stays converged.
            int s = 0, i = 0;
            uint32_t fphase = 0;
            bool alive = true;
            // descriptors advance by a constant per ring slot, the K = 32 steps are unrolled
            const uint32_t sbase = smem_u32(smem);
            const uint64_t adesc0 = sw_desc(sbase, p.cb), bdesc0 = sw_desc(sbase + p.kps * p.a_bytes, p.cb);
            const uint64_t wdesc0 = sw_desc(sbase + p.wres_off, p.cb);     // resident weights, K block 0
            const uint32_t dstep = p.stage_bytes >> 4;     // start-address step of one ring slot
            const uint32_t astep = p.a_bytes >> 4, bstep = p.b_bytes >> 4;   // second K block of a stage
            const bool k128 = p.cb == 128;                 // four 32-byte K steps per K block, else two
            const uint32_t idesc = p.idesc;
            const uint32_t sfa = tmem_base + p.sf_col, sfb = sfa + 32u;
            // timeout-path test (single CTAs): a wait that runs out; every other
            // warp's next wait then runs out too, and the kernel winds down
            if (!PAIR && p.stall && !__all_sync(0xffffffffu, mbar_wait(tstall, 0u, p.wait_cycles))) alive = false;
            if (FMT == 2 && alive &&
                !__all_sync(0xffffffffu, PAIR ? mbar_wait_cluster(sfready, 0u, p.wait_cycles)
                                              : mbar_wait(sfready, 0u, p.wait_cycles)))
                alive = false;
            fence_after();
            if (p.wres && alive && !__all_sync(0xffffffffu, PAIR ? mbar_wait_cluster(wfull, 0u, p.wait_cycles)
                                                                 : mbar_wait(wfull, 0u, p.wait_cycles)))
                alive = false;
            for (int n = 0, w; alive && (w = cta_item(p, n, items, tiles_m, crank)) >= 0; ++n, ++i) {
                const int ab = p.nacc == 2 ? (i & 1) : 0, use = p.nacc == 2 ? (i >> 1) : i;
                const int t = w / p.ksplit, kp = w - t * p.ksplit;
                const int kb = (int)((long long)kp * p.nk / p.ksplit), ke = (int)((long long)(kp + 1) * p.nk / p.ksplit);
                if (use > 0 && !__all_sync(0xffffffffu, PAIR ? mbar_wait_cluster(&tempty[ab], (use - 1) & 1, p.wait_cycles)
                                                             : mbar_wait(&tempty[ab], (use - 1) & 1, p.wait_cycles)))
                    break;
                fence_after();
                const uint32_t tmem_d = tmem_base + (uint32_t)(ab * p.acc_cols);
                uint32_t acc = 0u;
                auto mma = [&](uint64_t ad_, uint64_t bd_, uint32_t a_) {
                    if constexpr (PAIR && FMT == 1)
                        mma_bf16_pair(tmem_d, ad_, bd_, idesc, a_);
                    else if constexpr (PAIR && FMT == 2)
                        mma_f4_pair(tmem_d, ad_, bd_, idesc, a_, sfa, sfb);
                    else if constexpr (PAIR)
                        mma_f8_pair(tmem_d, ad_, bd_, idesc, a_);
                    else if constexpr (FMT == 1)
                        mma_bf16(tmem_d, ad_, bd_, idesc, a_);
                    else if constexpr (FMT == 2)
                        mma_f4(tmem_d, ad_, bd_, idesc, a_, sfa, sfb);
                    else
                        mma_f8(tmem_d, ad_, bd_, idesc, a_);
                };
                for (int ks = kb; ks < ke; ks += p.kps) {
                    if (!__all_sync(0xffffffffu, mbar_wait(&full[s], fphase, p.wait_cycles))) { alive = false; break; }
                    fence_after();
                    const uint64_t off = (uint64_t)((uint32_t)s * dstep);
                    uint64_t ad = adesc0 + off;
                    uint64_t bd = p.wres ? wdesc0 + (uint64_t)((uint32_t)ks * bstep) : bdesc0 + off;
                    if (p.trans) {            // weights are the MMA's A operand (M = channels)
                        const uint64_t t_ = ad;
                        ad = bd;
                        bd = t_;
                    }
                    const uint32_t as_ = p.trans ? bstep : astep, bs_ = p.trans ? astep : bstep;
                    mma(ad, bd, acc);
                    mma(ad + 2, bd + 2, 1u);
                    if (k128) {
                        mma(ad + 4, bd + 4, 1u);
                        mma(ad + 6, bd + 6, 1u);
                    }
                    if (p.kps == 2 && ks + 1 < ke) {
                        ad += as_;
                        bd += bs_;
                        mma(ad, bd, 1u);
                        mma(ad + 2, bd + 2, 1u);
                        if (k128) {
                            mma(ad + 4, bd + 4, 1u);
                            mma(ad + 6, bd + 6, 1u);
                        }
                    }
                    acc = 1u;
                    if constexpr (PAIR)
                        mma_commit_pair(&empty[s]);              // both CTAs' slots are free
                    else
                        mma_commit(&empty[s]);
                    if (++s == p.S) { s = 0; fphase ^= 1; }
                }
                if constexpr (PAIR)
                    mma_commit_pair(&tfull[ab]);
                else
                    mma_commit(&tfull[ab]);
            }
        }
    } else if (warp < B_WARP) {
        // ---------------- epilogue: warps 2..9 ----------------
        const int et = threadIdx.x - 64;          // 0 .. 255
        if constexpr (FMT == 2) {
            // unit scale factors (UE8M0 0x7F = 2^0) in 64 columns from sf_col, written
            // by one warp per TMEM lane quarter (a pair: each CTA in its own tensor memory)
            if (warp < 6) {
                const uint32_t ta = tmem_base + ((uint32_t)((warp & 3) * 32) << 16) + p.sf_col;
#pragma unroll
                for (int c = 0; c < 64; c += 8)
                    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %1, %1, %1, %1, %1, %1, %1};\n" ::"r"(
                                     ta + (uint32_t)c),
                                 "r"(0x7F7F7F7Fu));
                asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory");
                fence_before();
                __syncwarp();
                if (lane == 0) {
                    if (PAIR && crank == 1)
                        mbar_arrive_cluster(cta0_addr(sfready));
                    else
                        mbar_arrive(sfready);
                }
            }
        }
        // output-quantizer breakpoints of every channel, in shared memory
        if constexpr (OUTB > 0) {
            // held as (-T_1 .. -T_{n-1}, sigma) with -0 stored as +0, so that
            // fmaf(acc, sigma, -T) is never -0 and its sign bit is [sigma * acc < T]
            // rows u = 0 .. NL - 1 of O32 channels each (channel fastest: four channels per 128-bit load)
            if (p.thr != nullptr) {
                for (int i = et; i < p.O * NL; i += EPI_WARPS * 32) {
                    const float x = __ldg(p.thr + i);
                    const int o = i / NL, u = i - o * NL;
                    sthr[u * O32 + o] = (u == NL - 1) ? x : mask_breakpoint(x);
                }
            } else if (p.res_codes == nullptr && p.res_f32 == nullptr) {
                // (a residual block quantizes y + shortcut: no per-channel breakpoints on acc)
                for (int o = et; o < p.O; o += EPI_WARPS * 32) {
                    float t[8];
                    channel_thresholds(__ldg(p.scale + o), __ldg(p.shift + o), p.qo, t);
                    for (int u = 0; u < NL; ++u) sthr[u * O32 + o] = (u == NL - 1) ? t[u] : mask_breakpoint(t[u]);
                }
            }
            for (int i = p.O * NL + et; i < thr_floats; i += EPI_WARPS * 32) {      // padding channels
                const int k = i - p.O * NL, o = p.O + k / NL, u = k % NL;
                sthr[u * O32 + o] = (u == NL - 1) ? 1.0f : 0.0f;
            }
            if (p.res_codes != nullptr || p.res_f32 != nullptr) {       // level of y = #{u : y >= T_u}
                if (p.ythr != nullptr) {
                    if (et < NL - 1) syt[et] = mask_breakpoint(__ldg(p.ythr + et));
                } else if (et == 0) {
                    float t[8];
                    channel_thresholds_f32(1.0f, 0.0f, p.qo, t);         // a long serial search: callers cache it
                    for (int u = 0; u < NL - 1; ++u) syt[u] = mask_breakpoint(t[u]);
                }
            }
            // sigma of a channel: the sign of its BN scale (+1 for 0); one warp per
            // 32-channel word, a lane per channel (one load latency for the word)
            for (int g = warp - 2; g < sig_words; g += EPI_WARPS) {
                const int o = g * 32 + lane;
                const float sg = o < p.O ? (p.thr != nullptr ? __ldg(p.thr + o * NL + NL - 1)
                                                             : (__ldg(p.scale + o) < 0.0f ? -1.0f : 1.0f))
                                         : 1.0f;
                const uint32_t m = __ballot_sync(0xffffffffu, sg > 0.0f);
                if (lane == 0) ssig[g] = m;
            }
        }
        asm volatile("bar.sync 1, %0;\n" ::"n"(EPI_WARPS * 32) : "memory");   // breakpoints in place
        pdl_wait();                               // outputs, shortcuts and partial sums are shared with other kernels
        const int q = warp & 3;                   // TMEM lane quarter of this warp
        const int half_cols = (warp - 2) >> 2;    // which half of the accumulator columns
        const int r = q * 32 + lane;              // tile row = output pixel
        const int Hp = p.pool ? p.Ho / 2 : p.Ho, Wp = p.pool ? p.Wo / 2 : p.Wo;
        const int NWo = (p.O + 31) >> 5;
        const int rb = r / (p.bh * p.bw), ry = (r / p.bw) % p.bh, rx = r % p.bw;
        // this warp's 16-column groups: the first or second half of BN/16
        // (split at an even group so that no 32-channel plane word straddles the halves)
        const int ngrp = p.BN / 16;
        const int gmid = min(ngrp, (((ngrp + 1) / 2) + 1) & ~1);
        const int gbeg = half_cols ? gmid : 0, gend = half_cols ? ngrp : gmid;
        // mask epilogue (a layer whose only output is the next layer's levels):
        // this warp's 32-column chunks
        const bool resid = p.res_codes != nullptr || p.res_f32 != nullptr || p.y_nhwc != nullptr;
        // the accumulator is drained: CTA 1 of a pair tells CTA 0, which issues the MMAs
        auto tempty_arrive = [&](uint64_t *bar) {
            if (PAIR && crank == 1)
                mbar_arrive_cluster(cta0_addr(bar));
            else
                mbar_arrive(bar);
        };
        const bool masked = OUTB > 0 && p.ksplit == 1 && p.acc_out == nullptr && p.y_out == nullptr && !resid;
        // residual epilogue without per-element fp32 outputs: the same chunks
        const bool rmasked = p.ksplit == 1 && p.acc_out == nullptr && p.y_out == nullptr && !p.pool && resid &&
                             p.O % 16 == 0;
        const int nch = (p.BN + 31) >> 5, cmid = (nch + 1) >> 1;
        const int cbeg = half_cols ? cmid : 0, cend = half_cols ? nch : cmid;
        int i = 0;
        bool dead = false;           // a bounded wait ran out: skip work, keep the barrier sequence
        if constexpr (OUTB > 0) {
            if (p.trans) {
                // tile = 128 channels (TMEM lanes) x 256 pixels (columns): this warp holds
                // channels 32 q + lane of pixel columns [128 half, 128 half + 128); with the
                // weights loaded twice (64 channels), channels 32 (q & 1) + lane of the 64
                // columns [64 (2 (q >> 1) + half), + 64)
                const int oq = 32 * (p.dup ? (q & 1) : q);
                const int cq = p.dup ? 2 : 4, cb = p.dup ? 2 * (2 * (q >> 1) + half_cols) : 4 * half_cols;
                // this lane's pixel of each of the warp's chunks, relative to the tile (tiles-invariant)
                int crb[4], cry[4], crx[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int r = (cb + k) * 32 + lane;
                    crb[k] = r / (p.bh * p.bw);
                    cry[k] = (r / p.bw) % p.bh;
                    crx[k] = r % p.bw;
                }
                for (int n = 0, w; (w = cta_item(p, n, items, tiles_m, crank)) >= 0; ++n, ++i) {
                    const int ab = p.nacc == 2 ? (i & 1) : 0, use = p.nacc == 2 ? (i >> 1) : i;
                    const int tn = w / tiles_m, tm = w - tn * tiles_m;
                    const int xb = tm % p.nbx, yb = (tm / p.nbx) % p.nby, bbk = tm / (p.nbx * p.nby);
                    const int oc = tn * p.BN + oq + lane;          // this lane's channel
                    const bool qlive = tn * p.BN + oq < p.O;       // 64-channel layers: half the lanes are padding
                    float nt[NL - 1], sg = 1.0f;
                    uint32_t sig = 0u;
#pragma unroll
                    for (int u = 0; u < NL - 1; ++u) nt[u] = 0.0f;
                    if (qlive) {
#pragma unroll
                        for (int u = 0; u < NL - 1; ++u) nt[u] = sthr[u * O32 + oc];
                        sg = sthr[(NL - 1) * O32 + oc];
                        sig = ssig[(tn * p.BN + oq) >> 5];
                    }
                    if (!dead && !mbar_wait(&tfull[ab], use & 1, p.wait_cycles)) dead = true;
                    fence_after();
                    const bool tres = p.res_codes != nullptr || p.res_f32 != nullptr;
                    float sc = 0.0f, sh = 0.0f, ny[NL - 1];
#pragma unroll
                    for (int u = 0; u < NL - 1; ++u) ny[u] = syt[u];
                    if (tres && qlive) {
                        sc = __ldg(p.scale + oc);
                        sh = __ldg(p.shift + oc);
                    }
                    // plain block epilogue of 1- and 2-bit outputs: two chunks at a time, their loads,
                    // sign chains, transposes, pooling and stores interleaved (a 3-bit output's six
                    // mask chains per chunk already overlap)
#pragma unroll
                    for (int k = 0; k < 4; k += 2) {
                        if (NL > 3 || k >= cq || dead || !qlive || tres) break;
                        __syncwarp();
                        uint32_t v0[32], v1[32];
                        const uint32_t ta = tmem_base + ((uint32_t)oq << 16) + (uint32_t)(ab * p.acc_cols + (cb + k) * 32);
                        tmem_ld32_nw(ta, v0);
                        tmem_ld32_nw(ta + 32u, v1);
                        tmem_wait_ld();
                        uint32_t M0[NL - 1], M1[NL - 1];
#pragma unroll
                        for (int u = 0; u < NL - 1; ++u) {
                            float d0[32], d1[32];      // sigma * acc - T_u: sign bit j = [sigma * acc < T_u] at column j
#pragma unroll
                            for (int j = 0; j < 32; ++j) {
                                d0[j] = fmaf(__uint_as_float(v0[j]), sg, nt[u]);
                                d1[j] = fmaf(__uint_as_float(v1[j]), sg, nt[u]);
                            }
                            M0[u] = transpose32(sign_word(d0), lane);   // lane j: bit k = channel oq + k at column j
                            M1[u] = transpose32(sign_word(d1), lane);
                        }
                        if (p.pool) {
#pragma unroll
                            for (int u = 0; u < NL - 1; ++u) {
                                const uint32_t m0 = M0[u], m1 = M1[u];
                                const uint32_t n0 = __shfl_xor_sync(0xffffffffu, m0, 1), n1 = __shfl_xor_sync(0xffffffffu, m1, 1);
                                const uint32_t a0 = m0 & n0, o0 = m0 | n0, a1 = m1 & n1, o1 = m1 | n1;
                                const uint32_t a0b = a0 & __shfl_xor_sync(0xffffffffu, a0, p.bw);
                                const uint32_t a1b = a1 & __shfl_xor_sync(0xffffffffu, a1, p.bw);
                                const uint32_t o0b = o0 | __shfl_xor_sync(0xffffffffu, o0, p.bw);
                                const uint32_t o1b = o1 | __shfl_xor_sync(0xffffffffu, o1, p.bw);
                                M0[u] = (sig & a0b) | (~sig & o0b);
                                M1[u] = (sig & a1b) | (~sig & o1b);
                            }
                        }
#pragma unroll
                        for (int h2 = 0; h2 < 2; ++h2) {
                            const int b = bbk * p.bb + crb[k + h2];
                            const int y = yb * p.bh + cry[k + h2];
                            const int x = xb * p.bw + crx[k + h2];
                            const bool valid = b < p.B && y < p.Ho && x < p.Wo;
                            if (valid && (!p.pool || ((x & 1) == 0 && (y & 1) == 0))) {
                                const int yp = p.pool ? y / 2 : y, xp = p.pool ? x / 2 : x;
                                const long long opix = ((long long)b * Hp + yp) * Wp + xp;
                                const int ob = tn * p.BN + oq;
                                store_level_masks<OUTB>(h2 ? M1 : M0, 32, 32,
                                                        p.planes_out ? p.planes_out + (opix * OUTB) * NWo + (ob >> 5) : nullptr,
                                                        NWo, p.codes_out ? p.codes_out + ((opix * p.O + ob) >> p.out4) : nullptr,
                                                        p.out4 != 0);
                            }
                        }
                    }
                    for (int c = cb; c < cb + cq && !dead && qlive && (tres || NL > 3); ++c) {
                        __syncwarp();
                        uint32_t v[32];
                        tmem_ld32(tmem_base + ((uint32_t)oq << 16) + (uint32_t)(ab * p.acc_cols + c * 32), v);
                        const int r = c * 32 + lane;                    // tile row (pixel) of this lane
                        const int b = bbk * p.bb + r / (p.bh * p.bw);
                        const int y = yb * p.bh + (r / p.bw) % p.bh;
                        const int x = xb * p.bw + r % p.bw;
                        const bool valid = b < p.B && y < p.Ho && x < p.Wo;
                        uint32_t M[NL - 1];
                        if (tres) {
                            // residual block: y = BN(acc) + shortcut at (pixel j, this lane's channel), then the
                            // quantizer's breakpoints on y; pixel j's index comes from lane j
                            // (all 32 loads issue before the first use; a pixel past the batch reads pixel 0)
                            const long long pix = valid ? (((long long)b * p.Ho + y) * p.Wo + x) * p.O : 0;
                            float yv[32];
                            if (p.res_codes != nullptr && p.res4) {
                                uint32_t cb[32];
#pragma unroll
                                for (int j = 0; j < 32; ++j)
                                    cb[j] = __ldg(p.res_codes + ((oc + __shfl_sync(0xffffffffu, pix, j)) >> 1));
#pragma unroll
                                for (int j = 0; j < 32; ++j)
                                    yv[j] = fmaf(__uint_as_float(v[j]), sc, sh) +
                                            code_units_e2m1(cb[j] >> (4 * (oc & 1))) * p.res_unit;
                            } else if (p.res_codes != nullptr) {
                                uint32_t cb[32];
#pragma unroll
                                for (int j = 0; j < 32; ++j) cb[j] = __ldg(p.res_codes + oc + __shfl_sync(0xffffffffu, pix, j));
#pragma unroll
                                for (int j = 0; j < 32; ++j)
                                    yv[j] = fmaf(__uint_as_float(v[j]), sc, sh) + code_units(cb[j]) * p.res_unit;
                            } else {
#pragma unroll
                                for (int j = 0; j < 32; ++j) yv[j] = __ldg(p.res_f32 + oc + __shfl_sync(0xffffffffu, pix, j));
#pragma unroll
                                for (int j = 0; j < 32; ++j) yv[j] = fmaf(__uint_as_float(v[j]), sc, sh) + yv[j];
                            }
#pragma unroll
                            for (int u = 0; u < NL - 1; ++u) {
                                uint32_t wd = 0u;
#pragma unroll
                                for (int j = 31; j >= 0; --j) wd = __funnelshift_l(__float_as_uint(yv[j] + ny[u]), wd, 1);
                                M[u] = transpose32(wd, lane);
                            }
                        } else {
#pragma unroll
                            for (int u = 0; u < NL - 1; ++u) {
                                uint32_t wd = 0u;          // bit j: [sigma * acc < T_u] at pixel column 32 c + j
#pragma unroll
                                for (int j = 31; j >= 0; --j)
                                    wd = __funnelshift_l(__float_as_uint(fmaf(__uint_as_float(v[j]), sg, nt[u])), wd, 1);
                                M[u] = transpose32(wd, lane);     // lane j: bit k = channel oq + k at column 32 c + j
                            }
                        }
                        if (p.pool) {
#pragma unroll
                            for (int u = 0; u < NL - 1; ++u) {
                                const uint32_t m = M[u];
                                const uint32_t n1 = __shfl_xor_sync(0xffffffffu, m, 1);
                                const uint32_t a1 = m & n1, o1 = m | n1;
                                const uint32_t a2 = a1 & __shfl_xor_sync(0xffffffffu, a1, p.bw);
                                const uint32_t o2 = o1 | __shfl_xor_sync(0xffffffffu, o1, p.bw);
                                M[u] = (sig & a2) | (~sig & o2);
                            }
                        }
                        const bool writer = valid && (!p.pool || ((x & 1) == 0 && (y & 1) == 0));
                        if (writer) {
                            const int yp = p.pool ? y / 2 : y, xp = p.pool ? x / 2 : x;
                            const long long opix = ((long long)b * Hp + yp) * Wp + xp;
                            const int ob = tn * p.BN + oq;
                            store_level_masks<OUTB>(M, 32, 32,
                                                    p.planes_out ? p.planes_out + (opix * OUTB) * NWo + (ob >> 5) : nullptr,
                                                    NWo, p.codes_out ? p.codes_out + ((opix * p.O + ob) >> p.out4) : nullptr,
                                                    p.out4 != 0);
                        }
                    }
                    fence_before();
                    __syncwarp();
                    if (lane == 0 && !dead) tempty_arrive(&tempty[ab]);
                }
            }
        }
        for (int n = 0, w; !p.trans && (w = cta_item(p, n, items, tiles_m, crank)) >= 0; ++n, ++i) {
            const int ab = p.nacc == 2 ? (i & 1) : 0, use = p.nacc == 2 ? (i >> 1) : i;
            const int t = w / p.ksplit, kp = w - t * p.ksplit;
            const int tn = t / tiles_m, tm = t - tn * tiles_m;
            const int xb = tm % p.nbx, yb = (tm / p.nbx) % p.nby, bbk = tm / (p.nbx * p.nby);
            const int b = bbk * p.bb + rb;
            const int y = yb * p.bh + ry;
            const int x = xb * p.bw + rx;
            const int o0 = tn * p.BN;
            const bool valid = b < p.B && y < p.Ho && x < p.Wo;
            const bool writer = valid && (!p.pool || ((x & 1) == 0 && (y & 1) == 0));
            const int yp = p.pool ? y / 2 : y, xp = p.pool ? x / 2 : x;
            const long long opix = ((long long)b * Hp + yp) * Wp + xp;
            uint32_t pw[3] = {0u, 0u, 0u};

            if constexpr (OUTB > 0) {
                if (masked) {
                    if (!dead && !mbar_wait(&tfull[ab], use & 1, p.wait_cycles)) dead = true;
                    fence_after();
                    for (int c = cbeg; c < cend && !dead; ++c) {
                        const int ob = o0 + c * 32;
                        if (ob >= p.O) break;                      // no channel of this tile left
                        __syncwarp();
                        mask_chunk<OUTB>(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * p.BN + c * 32),
                                         c * 32 + 32 <= p.BN, sthr + ob, O32, p.pool ? ssig[ob >> 5] : 0u, p.pool,
                                         p.bw, writer, p.O - ob,
                                         p.planes_out ? p.planes_out + (opix * OUTB) * NWo + (ob >> 5) : nullptr,
                                         NWo, p.codes_out ? p.codes_out + ((opix * p.O + ob) >> p.out4) : nullptr,
                                         p.out4 != 0);
                    }
                    fence_before();
                    __syncwarp();
                    if (lane == 0 && !dead) tempty_arrive(&tempty[ab]);
                    continue;
                }
            }
            if (rmasked) {
                if (!dead && !mbar_wait(&tfull[ab], use & 1, p.wait_cycles)) dead = true;
                fence_after();
                for (int c = cbeg; c < cend && !dead; ++c) {
                    const int ob = o0 + c * 32;
                    if (ob >= p.O) break;
                    __syncwarp();
                    resid_chunk<OUTB>(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * p.BN + c * 32),
                                      c * 32 + 32 <= p.BN, p, ob, opix, writer, syt, NWo);
                }
                fence_before();
                __syncwarp();
                if (lane == 0 && !dead) tempty_arrive(&tempty[ab]);
                continue;
            }

            // the fused block epilogue of one 16-column group of exact accumulators
            auto finish = [&](float (&a)[16], int ch) {
                if (p.pool) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        a[j] = fmaxf(a[j], __shfl_xor_sync(0xffffffffu, a[j], 1));
                        a[j] = fmaxf(a[j], __shfl_xor_sync(0xffffffffu, a[j], p.bw));
                    }
                }
                const int ob = o0 + ch * 16;
                if (p.acc_out != nullptr && valid) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        if (ob + j < p.O)
                            p.acc_out[(((long long)b * p.O + ob + j) * p.Ho + y) * p.Wo + x] = __float2int_rn(a[j]);
                }
                const bool resid = p.res_codes != nullptr || p.res_f32 != nullptr || p.y_nhwc != nullptr;
                if (p.y_out != nullptr && writer && !resid) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int o = ob + j;
                        if (o < p.O) {
                            float yv = fmaf(a[j], __ldg(p.scale + o), __ldg(p.shift + o));
                            if (OUTB > 0) yv = fminf(fmaxf(yv, -1.0f), 1.0f);
                            p.y_out[(((long long)b * p.O + o) * Hp + yp) * Wp + xp] = yv;
                        }
                    }
                }
                if (p.hb_out != nullptr && writer) {
                    // weight-only networks: HardTanh(BN(acc) [+ shortcut]) (the fp32 fmaf, one fp32
                    // add, the two clamps, one rounding to bf16) into this pixel's NHWC row, 16
                    // channels of it [and the fp32 value into NCHW]
                    uint32_t pk[8];
                    if (p.hb_res == nullptr && p.hb_z == nullptr) {
#pragma unroll
                        for (int j = 0; j < 16; j += 2) {
                            uint32_t h2[2];
#pragma unroll
                            for (int e = 0; e < 2; ++e) {
                                const int o = min(ob + j + e, p.O - 1);
                                const float yv = fmaf(a[j + e], __ldg(p.scale + o), __ldg(p.shift + o));
                                h2[e] = __bfloat16_as_ushort(__float2bfloat16_rn(fminf(fmaxf(yv, -1.0f), 1.0f)));
                            }
                            pk[j >> 1] = h2[0] | (h2[1] << 16);
                        }
                    } else {
                        const long long nchw = ((long long)b * p.O * p.Ho + y) * p.Wo + x;     // channel 0
                        const long long cst = (long long)p.Ho * p.Wo;
                        float rv[16];
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            rv[j] = p.hb_res != nullptr ? __ldg(p.hb_res + nchw + min(ob + j, p.O - 1) * cst) : 0.0f;
#pragma unroll
                        for (int j = 0; j < 16; j += 2) {
                            uint32_t h2[2];
#pragma unroll
                            for (int e = 0; e < 2; ++e) {
                                const int o = min(ob + j + e, p.O - 1);
                                float yv = fmaf(a[j + e], __ldg(p.scale + o), __ldg(p.shift + o));
                                if (p.hb_res != nullptr) yv = yv + rv[j + e];
                                yv = fminf(fmaxf(yv, -1.0f), 1.0f);
                                if (p.hb_z != nullptr && ob + j + e < p.O) p.hb_z[nchw + o * cst] = yv;
                                h2[e] = __bfloat16_as_ushort(__float2bfloat16_rn(yv));
                            }
                            pk[j >> 1] = h2[0] | (h2[1] << 16);
                        }
                    }
                    uint16_t *dst = p.hb_out + opix * p.hb_ld + p.hb_off + ob;
                    const uintptr_t al = reinterpret_cast<uintptr_t>(dst);
                    if (ob + 16 <= p.O && (al & 15) == 0) {
                        reinterpret_cast<uint4 *>(dst)[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                        reinterpret_cast<uint4 *>(dst)[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
                    } else if ((al & 7) == 0) {
#pragma unroll
                        for (int g = 0; g < 4; ++g) {
                            if (ob + 4 * g + 4 <= p.O)
                                reinterpret_cast<uint2 *>(dst)[g] = make_uint2(pk[2 * g], pk[2 * g + 1]);
                            else
                                for (int j = 4 * g; j < 4 * g + 4 && ob + j < p.O; ++j)
                                    dst[j] = (uint16_t)(pk[j >> 1] >> (16 * (j & 1)));
                        }
                    } else {
                        for (int j = 0; j < 16 && ob + j < p.O; ++j) dst[j] = (uint16_t)(pk[j >> 1] >> (16 * (j & 1)));
                    }
                }
                if (resid) {
                    // residual block: y = BN(acc) [+ shortcut], HardTanh, quantize,
                    // element by element in the fp32 order of the block
                    if (writer) {
                        uint32_t cw[4] = {0u, 0u, 0u, 0u}, cw4[2] = {0u, 0u};
                        uint32_t bits16[3] = {0u, 0u, 0u};
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            const int o = ob + j;
                            if (o >= p.O) continue;
                            float yv = fmaf(a[j], __ldg(p.scale + o), __ldg(p.shift + o));
                            if (p.y_nhwc != nullptr) p.y_nhwc[opix * p.O + o] = yv;
                            if (p.res_codes != nullptr && p.res4)
                                yv += code_units_e2m1(__ldg(p.res_codes + ((opix * p.O + o) >> 1)) >> (4 * (o & 1))) *
                                      p.res_unit;
                            else if (p.res_codes != nullptr)
                                yv += code_units(__ldg(p.res_codes + opix * p.O + o)) * p.res_unit;
                            else if (p.res_f32 != nullptr) yv += __ldg(p.res_f32 + opix * p.O + o);
                            if (p.y_out != nullptr)
                                p.y_out[(((long long)b * p.O + o) * Hp + yp) * Wp + xp] =
                                    (OUTB > 0) ? fminf(fmaxf(yv, -1.0f), 1.0f) : yv;
                            if constexpr (OUTB > 0) {
                                const int k = level_index_of_y(yv, p.qo);
                                cw[j >> 2] |= code_k<OUTB>(k) << ((j & 3) * 8);
                                cw4[j >> 3] |= code4_k<OUTB>(k) << ((j & 7) * 4);
                                const uint32_t pb = planes_k<OUTB>(k);
#pragma unroll
                                for (int u = 0; u < OUTB; ++u) bits16[u] |= ((pb >> u) & 1u) << j;
                            }
                        }
                        if constexpr (OUTB > 0) {
                            if (p.codes_out != nullptr && p.out4)
                                *reinterpret_cast<uint2 *>(p.codes_out + ((opix * p.O + ob) >> 1)) = make_uint2(cw4[0], cw4[1]);
                            else if (p.codes_out != nullptr)
                                *reinterpret_cast<uint4 *>(p.codes_out + opix * p.O + ob) =
                                    make_uint4(cw[0], cw[1], cw[2], cw[3]);
                            if (p.planes_out != nullptr) {
                                const int half = (ob >> 4) & 1;
#pragma unroll
                                for (int u = 0; u < OUTB; ++u) pw[u] |= bits16[u] << (16 * half);
                                if (half == 1 || ch == p.BN / 16 - 1 || ob + 16 >= p.O) {
                                    uint32_t *dst = p.planes_out + (opix * OUTB) * NWo + (ob >> 5);
#pragma unroll
                                    for (int u = 0; u < OUTB; ++u) {
                                        dst[u * NWo] = pw[u];
                                        pw[u] = 0u;
                                    }
                                }
                            }
                        }
                    }
                } else if constexpr (OUTB > 0) {
                    if (writer) {
                        int kq[16];
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            const int o = min(ob + j, p.O - 1);
                            const float vv = a[j] * sthr[(NL - 1) * O32 + o];
                            int k = 0;
#pragma unroll
                            for (int u = 0; u < NL - 1; ++u) k += (vv + sthr[u * O32 + o] >= 0.0f) ? 1 : 0;   // -T
                            kq[j] = k;
                        }
                        if (p.codes_out != nullptr && p.out4) {
                            uint32_t cw4[2] = {0u, 0u};
#pragma unroll
                            for (int j = 0; j < 16; ++j) cw4[j >> 3] |= code4_k<OUTB>(kq[j]) << ((j & 7) * 4);
                            *reinterpret_cast<uint2 *>(p.codes_out + ((opix * p.O + ob) >> 1)) = make_uint2(cw4[0], cw4[1]);
                        } else if (p.codes_out != nullptr) {
                            uint32_t cw[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                            for (int j = 0; j < 16; ++j) cw[j >> 2] |= code_k<OUTB>(kq[j]) << ((j & 3) * 8);
                            *reinterpret_cast<uint4 *>(p.codes_out + opix * p.O + ob) =
                                make_uint4(cw[0], cw[1], cw[2], cw[3]);
                        }
                        if (p.planes_out != nullptr) {
                            uint32_t bits16[3] = {0u, 0u, 0u};
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                const uint32_t pb = (ob + j < p.O) ? planes_k<OUTB>(kq[j]) : 0u;
#pragma unroll
                                for (int u = 0; u < OUTB; ++u) bits16[u] |= ((pb >> u) & 1u) << j;
                            }
                            const int half = (ob >> 4) & 1;
#pragma unroll
                            for (int u = 0; u < OUTB; ++u) pw[u] |= bits16[u] << (16 * half);
                            if (half == 1 || ch == p.BN / 16 - 1 || ob + 16 >= p.O) {
                                uint32_t *dst = p.planes_out + (opix * OUTB) * NWo + (ob >> 5);
#pragma unroll
                                for (int u = 0; u < OUTB; ++u) {
                                    dst[u * NWo] = pw[u];
                                    pw[u] = 0u;
                                }
                            }
                        }
                    }
                }
            };

            // fully connected fp32 output: this warp's BN values, four columns a lane,
            // loaded before the accumulator is ready (the loads overlap the MMAs)
            float bsc[4] = {1.0f, 1.0f, 1.0f, 1.0f}, bsh[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            if (p.ksplit == 1 && p.rowst) {
                const int oc = o0 + gbeg * 16 + 4 * lane;
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (4 * lane + e < (gend - gbeg) * 16 && oc + e < p.O) {
                        bsc[e] = __ldg(p.scale + oc + e);
                        bsh[e] = __ldg(p.shift + oc + e);
                    }
                if (p.upd && b < p.B) {
                    // the latent weights of this lane's row into L2 while the MMAs run
                    const int o1 = o0 + gbeg * 16;
                    const int ncol = min((gend - gbeg) * 16, p.O - o1);
                    const float *wrow = p.y_out + (long long)b * p.O + o1;
                    for (int off = 0; off < ncol; off += 32)
                        asm volatile("prefetch.global.L2 [%0];\n" ::"l"(wrow + off));
                }
            }
            if (!dead && !mbar_wait(&tfull[ab], use & 1, p.wait_cycles)) dead = true;
            fence_after();
            int32_t *prow = p.part + (((size_t)kp * tiles + t) * 128 + r) * p.BN;
            uint32_t v32[32];
            for (int ch = gbeg; ch < gend && !dead; ++ch) {
                __syncwarp();
                // two groups per TMEM load where possible (one wait for 32 columns)
                const int sub = (ch - gbeg) & 1;
                if (sub == 0) {
                    if (ch + 1 < gend)
                        tmem_ld32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * p.BN + ch * 16), v32);
                    else {
                        uint32_t v16[16];
                        tmem_ld16(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * p.BN + ch * 16), v16);
#pragma unroll
                        for (int j = 0; j < 16; ++j) v32[j] = v16[j];
                    }
                }
                float a[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) a[j] = __uint_as_float(sub ? v32[16 + j] : v32[j]);
                uint32_t *sw = sy + (warp - 2) * (32 * 16);
                if (p.ksplit == 1 && p.rowst) {
                    // fully connected output y[b][o]: rows b0 + rr of this warp, row-contiguous
                    const int ob = o0 + ch * 16;
                    uint32_t u[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) u[j] = __float_as_uint(a[j]);
                    // the BN values of columns 4 (lane & 3) .. + 3 of this group
                    const int src = (ch - gbeg) * 4 + (lane & 3);
                    float sc[4], sh[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        sc[e] = __shfl_sync(0xffffffffu, bsc[e], src);
                        sh[e] = __shfl_sync(0xffffffffu, bsh[e], src);
                    }
                    const int b0 = b - lane;
                    rows_store16(sw, u, lane, reinterpret_cast<uint32_t *>(p.y_out) + (long long)b0 * p.O + ob, p.O,
                                 p.B - b0, p.O - ob, sc, sh, p.upd != 0, p.upd_lr, p.upd_2a);
                } else if (p.ksplit == 1) {
                    finish(a, ch);
                } else if (p.rowst) {
                    // partial sums of this K slice (exact integers, or fp32 sums of bf16 products),
                    // summed by splitk_reduce_kernel
                    uint32_t u[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) u[j] = FMT == 1 ? __float_as_uint(a[j]) : (uint32_t)__float2int_rn(a[j]);
                    rows_store16(sw, u, lane,
                                 reinterpret_cast<uint32_t *>(p.part) + (((size_t)kp * tiles + t) * 128 + q * 32) * p.BN +
                                     ch * 16,
                                 p.BN, 32, 16);
                } else {
                    int4 *dst = reinterpret_cast<int4 *>(prow + ch * 16);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        int v[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            v[e] = FMT == 1 ? __float_as_int(a[4 * j + e]) : __float2int_rn(a[4 * j + e]);
                        dst[j] = make_int4(v[0], v[1], v[2], v[3]);
                    }
                }
            }
            fence_before();
            __syncwarp();
            if (lane == 0 && !dead) tempty_arrive(&tempty[ab]);      // the accumulator can be reused
        }
    }
    __syncthreads();
    if constexpr (PAIR) {
        // both CTAs are done with the pair's tensor memory and barriers; one warp of each frees it
        cluster_sync_all();
        if (warp == 1) {
            fence_after();
            asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(p.tmem_cols));
        }
    } else {
        if (warp == 1) {
            fence_after();
            asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_base), "r"(p.tmem_cols));
        }
    }
}

// Split-K second pass: sums the K slices of every accumulator and runs the
// block epilogue (no pooling).  Thread = one tile row (output pixel) x four
// channels; eight consecutive lanes cover 32 channels of one row, so the
// partial-sum loads coalesce and plane words assemble with shuffles.
template <int OUTB>
__global__ void __launch_bounds__(256) splitk_reduce_kernel(const Params p, const float *__restrict__ thr) {
    pdl_wait();
    pdl_trigger();
    constexpr int NL = OUTB == 0 ? 1 : (OUTB == 1 ? 2 : (OUTB == 2 ? 3 : 7));
    const int tiles_m = p.nbx * p.nby * p.nbb;
    const int tiles = tiles_m * p.ntn;
    const int g32 = (p.O + 31) >> 5;                 // 32-channel groups
    // 32-bit index arithmetic: the host launches fewer than 2^31 threads
    const uint32_t total = (uint32_t)tiles_m * 128u * (uint32_t)g32 * 8u;
    const uint32_t idx = blockIdx.x * blockDim.x + threadIdx.x;
    const int lane8 = threadIdx.x & 7;
    if (idx - lane8 >= total) return;               // whole 8-lane groups leave together
    const uint32_t rowgrp = idx >> 3;
    const int g = (int)(rowgrp % (uint32_t)g32);
    const uint32_t rr = rowgrp / (uint32_t)g32;
    const int tm = (int)(rr >> 7), r = (int)(rr & 127);
    const int o = g * 32 + lane8 * 4;                // first of this thread's four channels
    const bool live = o < p.O;
    const int tn = live ? o / p.BN : 0, col = live ? o - tn * p.BN : 0;
    const int t = tn * tiles_m + tm;
    const int xb = tm % p.nbx, yb = (tm / p.nbx) % p.nby, bbk = tm / (p.nbx * p.nby);
    const int b = bbk * p.bb + r / (p.bh * p.bw);
    const int y = yb * p.bh + (r / p.bw) % p.bh;
    const int x = xb * p.bw + r % p.bw;
    const bool inside = b < p.B && y < p.Ho && x < p.Wo;
    const bool valid = live && inside;
    int acc[4] = {0, 0, 0, 0};
    float accf[4] = {0.0f, 0.0f, 0.0f, 0.0f};      // the accumulators as fp32
    if (valid) {
        const size_t slice4 = (size_t)tiles * 128 * p.BN / 4;
        const int4 *src = reinterpret_cast<const int4 *>(p.part + ((size_t)t * 128 + r) * p.BN + col);
        // four slices' loads in flight before their adds (the adds keep slice order)
        if (p.esize == 2) {
            // fp32 partial sums of bf16 products, added in slice order
            const float4 *src4 = reinterpret_cast<const float4 *>(src);
            int kp = 0;
            for (; kp + 4 <= p.ksplit; kp += 4) {
                float4 v[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) v[e] = __ldcs(src4 + (kp + e) * slice4);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    accf[0] += v[e].x; accf[1] += v[e].y; accf[2] += v[e].z; accf[3] += v[e].w;
                }
            }
            for (; kp < p.ksplit; ++kp) {
                const float4 v = __ldcs(src4 + kp * slice4);
                accf[0] += v.x; accf[1] += v.y; accf[2] += v.z; accf[3] += v.w;
            }
        } else {
            int kp = 0;
            for (; kp + 4 <= p.ksplit; kp += 4) {
                int4 v[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) v[e] = __ldcs(src + (kp + e) * slice4);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    acc[0] += v[e].x; acc[1] += v[e].y; acc[2] += v[e].z; acc[3] += v[e].w;
                }
            }
            for (; kp < p.ksplit; ++kp) {
                const int4 v = __ldcs(src + kp * slice4);
                acc[0] += v.x; acc[1] += v.y; acc[2] += v.z; acc[3] += v.w;
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) accf[j] = (float)acc[j];
        }
    }
    const long long HoWo = (long long)p.Ho * p.Wo;
    const long long pix = ((long long)b * p.Ho + y) * p.Wo + x;
    if (valid && p.acc_out != nullptr)
        for (int j = 0; j < 4; ++j)
            if (o + j < p.O) p.acc_out[((long long)b * p.O + o + j) * HoWo + (long long)y * p.Wo + x] = acc[j];
    // residual blocks: y = BN(acc) [+ shortcut], element by element as in the
    // single-pass epilogue; yres holds the HardTanh input
    const bool resid = p.res_codes != nullptr || p.res_f32 != nullptr || p.y_nhwc != nullptr;
    float yres[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (valid && resid)
        for (int j = 0; j < 4; ++j)
            if (o + j < p.O) {
                float yv = fmaf(accf[j], __ldg(p.scale + o + j), __ldg(p.shift + o + j));
                if (p.y_nhwc != nullptr) p.y_nhwc[pix * p.O + o + j] = yv;
                if (p.res_codes != nullptr && p.res4)
                    yv += code_units_e2m1(__ldg(p.res_codes + ((pix * p.O + o + j) >> 1)) >> (4 * ((o + j) & 1))) *
                          p.res_unit;
                else if (p.res_codes != nullptr)
                    yv += code_units(__ldg(p.res_codes + pix * p.O + o + j)) * p.res_unit;
                else if (p.res_f32 != nullptr) yv += __ldg(p.res_f32 + pix * p.O + o + j);
                yres[j] = yv;
            }
    if (valid && p.y_out != nullptr) {
        float yv4[4];
        for (int j = 0; j < 4; ++j) {
            const int oj = min(o + j, p.O - 1);
            yv4[j] = resid ? yres[j] : fmaf(accf[j], __ldg(p.scale + oj), __ldg(p.shift + oj));
            if (OUTB > 0) yv4[j] = fminf(fmaxf(yv4[j], -1.0f), 1.0f);
        }
        if (HoWo == 1 && o + 4 <= p.O && ((reinterpret_cast<uintptr_t>(p.y_out + (long long)b * p.O + o) & 15) == 0)) {
            // fully connected output: four consecutive channels of one row
            *reinterpret_cast<float4 *>(p.y_out + (long long)b * p.O + o) = make_float4(yv4[0], yv4[1], yv4[2], yv4[3]);
        } else {
            for (int j = 0; j < 4; ++j)
                if (o + j < p.O) p.y_out[((long long)b * p.O + o + j) * HoWo + (long long)y * p.Wo + x] = yv4[j];
        }
    }
    if constexpr (OUTB > 0) {
        uint32_t code = 0u, code4 = 0u, bits[3] = {0u, 0u, 0u};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (valid && o + j < p.O) {
                int k = 0;
                if (resid) {
                    k = level_index_of_y(yres[j], p.qo);
                } else {
                    const float *th = thr + (o + j) * NL;
                    const float v = accf[j] * __ldg(th + NL - 1);
#pragma unroll
                    for (int u = 0; u < NL - 1; ++u) k += (v >= __ldg(th + u)) ? 1 : 0;
                }
                code |= code_k<OUTB>(k) << (8 * j);
                code4 |= code4_k<OUTB>(k) << (4 * j);
                const uint32_t pb = planes_k<OUTB>(k);
#pragma unroll
                for (int u = 0; u < OUTB; ++u) bits[u] |= ((pb >> u) & 1u) << (lane8 * 4 + j);
            }
        }
        if (p.codes_out != nullptr && valid) {
            if (p.out4)
                *reinterpret_cast<uint16_t *>(p.codes_out + ((pix * p.O + o) >> 1)) = (uint16_t)code4;
            else
                *reinterpret_cast<uint32_t *>(p.codes_out + pix * p.O + o) = code;
        }
        if (p.planes_out != nullptr) {
#pragma unroll
            for (int u = 0; u < OUTB; ++u) {
                bits[u] |= __shfl_xor_sync(__activemask(), bits[u], 1);
                bits[u] |= __shfl_xor_sync(__activemask(), bits[u], 2);
                bits[u] |= __shfl_xor_sync(__activemask(), bits[u], 4);
            }
            if (lane8 == 0 && inside) {
                const int NWo = (p.O + 31) >> 5;
                uint32_t *dst = p.planes_out + (pix * OUTB) * NWo + g;
#pragma unroll
                for (int u = 0; u < OUTB; ++u) dst[u * NWo] = bits[u];
            }
        }
    }
}

// Breakpoints of every channel (see channel_thresholds): one thread per channel.
__global__ void thresholds_kernel(const float *__restrict__ scale, const float *__restrict__ shift, int O,
                                  QParams q, float *__restrict__ out) {
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o < O) channel_thresholds(scale[o], shift[o], q, out + o * num_levels(q.bits));
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

static int pow2_ceil(int v) {
    int p = 1;
    while (p < v) p <<= 1;
    return p;
}

struct Plan {
    Params p;
    CUtensorMap tmA, tmB;
    dim3 grid;
    size_t smem;
    float *thr_ws;      // split-K: breakpoints computed into the workspace (nullable)
};

static bool plan_shape(const ConvArgs &a, Params &p, int rows = 128) {
    if ((a.stride != 1 && a.stride != 2) || a.C % 64 != 0 || a.pad >= a.kh || a.pad >= a.kw) return false;
    int bw = pow2_ceil(a.Wo);
    if (bw > rows) bw = rows;
    if (bw > 128) bw = 128;
    if (a.pool && bw > 16) bw = 16;
    int bh = pow2_ceil(a.Ho);
    if (bh > rows / bw) bh = rows / bw;
    const int bb = rows / (bw * bh);
    if (a.pool && (bw < 2 || bh < 2)) return false;
    p.bw = bw; p.bh = bh; p.bb = bb;
    p.nbx = (a.Wo + bw - 1) / bw;
    p.nby = (a.Ho + bh - 1) / bh;
    int BN = ((a.O + 15) / 16) * 16;
    if (BN > 256) BN = 256;
    p.BN = BN;
    return true;
}

// Split-K: a shape with fewer output tiles than a third of the SMs and a long
// K loop (>= 16 stages) splits it into slices of at least four stages, up to
// one work item per SM.  Short K loops gain less than the second launch costs,
// and a split in two gains less than its second epilogue round (the partial
// sums) and the reduction cost.
static int auto_ksplit(int tiles, int nk, int sms) {
    if (tiles * 3 > sms || nk < 16) return 1;
    int ks = sms / tiles;
    if (ks > nk / 4) ks = nk / 4;
    return ks < 3 ? 1 : ks;
}
// channels of one K chunk: 128-byte rows of E4M3 codes (64-byte rows when C is
// not a multiple of 128), or 64 bf16 values
static int chunk_channels(const ConvArgs &a) {
    if (a.fp4) return (a.C % 256 == 0) ? 256 : 128;    // 128- or 64-byte rows of E2M1 pairs
    return a.bf16 ? 64 : ((a.C % 128 == 0) ? 128 : 64);
}
static size_t slice_bytes(int tiles, int BN) { return (size_t)tiles * 128 * BN * sizeof(int32_t); }
static size_t thr_ws_bytes(int O, int nlev) { return (((size_t)O * nlev * sizeof(float)) + 255) & ~(size_t)255; }

// Plan options (runtime.cu): channel-major 64-channel tiles with the weight
// rows loaded twice (else zero rows), CTA pairs for 256-channel layers with
// long K loops, K blocks per stage, channel-major tiles for 64- and
// 128-channel layers.
static int dup_pref() { return minw_host::plan_options().dup_weights != 0; }
static int pair_pref() { return minw_host::plan_options().cta_pairs != 0; }
static int kps_pref() { return minw_host::plan_options().kblocks_per_stage; }
static int trans_pref() { return minw_host::plan_options().channel_major != 0; }

// Tile of 256 pixels (bb images x bh rows x bw columns) that covers the output
// image exactly, widest rows first; pooling keeps 2x2 windows inside a warp.
static bool trans_shape(const ConvArgs &a, Params &p) {
    if ((a.stride != 1 && a.stride != 2) || a.C % 64 != 0 || a.pad >= a.kh || a.pad >= a.kw) return false;
    for (int bw = 128; bw >= 1; bw >>= 1) {
        if (a.Wo % bw != 0 || (a.pool && (bw > 16 || bw < 2))) continue;
        for (int bh = 256 / bw; bh >= 1; bh >>= 1) {
            if (a.Ho % bh != 0 || (a.pool && bh < 2)) continue;
            p.bw = bw; p.bh = bh; p.bb = 256 / (bw * bh);
            p.nbx = a.Wo / bw;
            p.nby = a.Ho / bh;
            p.BN = 128;
            return true;
        }
    }
    return false;
}

static bool trans_eligible(const ConvArgs &a) {
    return trans_pref() && (a.O == 128 || a.O == 64) && a.quant_out && (a.codes_out != nullptr || a.planes_out != nullptr) &&
           a.acc_out == nullptr && a.y_out == nullptr && a.y_nhwc == nullptr && a.ksplit <= 1 &&
           (a.res_codes == nullptr && a.res_f32 == nullptr ||
            ((a.O == 128 || (a.O == 64 && dup_pref())) && !a.pool));   // residual: all 8 warps hold channels
}

// encode = false plans the tiles and the split only (no tensor maps: no driver call).
static minw_status make_plan(const ConvArgs &a, Plan &pl, bool encode = true) {
    Params &p = pl.p;
    p = Params{};
    p.trans = 0;
    if (trans_eligible(a)) {
        // only when the 256-pixel tiles cover the image without padding and leave
        // at least channel_major_min_tiles_per_sm tiles per SM, else the 128-pixel tiles
        // balance better
        Params q{};
        const int sms_ = minw_host::num_sms() > 0 ? minw_host::num_sms() : 148;
        const int min_tiles = minw_host::plan_options().channel_major_min_tiles_per_sm;
        if (trans_shape(a, q) && (long long)q.nbx * q.nby * ((a.B + q.bb - 1) / q.bb) >= (long long)min_tiles * sms_)
            p.trans = 1;
    }
    p.mrows = p.trans ? 256 : 128;
    if (p.trans ? !trans_shape(a, p) : !plan_shape(a, p)) return MINW_EUNSUPPORTED;
    p.dup = (p.trans && a.O == 64 && dup_pref()) ? 1 : 0;
    p.B = a.B; p.C = a.C; p.H = a.H; p.W = a.W; p.O = a.O; p.kh = a.kh; p.kw = a.kw; p.pad = a.pad;
    p.Ho = a.Ho; p.Wo = a.Wo;
    p.stride = a.stride;
    p.esize = a.bf16 ? 2 : 1;
    p.fp4 = a.fp4 ? 1 : 0;
    p.out4 = a.codes_out4 ? 1 : 0;
    p.res4 = a.res_codes4 ? 1 : 0;
    // bytes of one pixel's channels: E2M1 packs two channels per byte
    const int rowb = p.fp4 ? a.C / 2 : a.C * p.esize;
    p.cb = (rowb % 128 == 0) ? 128 : 64;
    p.ck = p.fp4 ? 2 * p.cb : p.cb / p.esize;
    p.a_bytes = (uint32_t)(p.mrows * p.cb);
    p.nck = a.C / p.ck;
    p.nk = a.kh * a.kw * p.nck;
    p.nbb = (a.B + p.bb - 1) / p.bb;
    p.ntn = (a.O + p.BN - 1) / p.BN;
    // E2M1 tiles of 128 channels on single CTAs (request n128): a 256-channel E2M1 tile holds one
    // accumulator beside the scale factors, a 128-channel one two, so that each tile's epilogue
    // overlaps the next tile's MMAs (at half the MMA width)
    if (a.n128 && a.fp4 && !p.trans && !a.pair_n128 && p.BN > 128) {
        p.BN = 128;
        p.ntn = (a.O + 127) / 128;
    }
    p.nlev = a.quant_out ? num_levels(a.qo.bits) : 0;
    p.thr = a.thr;
    // CTA pairs (MINW_TC_PAIR): 256-channel tiles of a layer that is not split along K
    {
        const int sms_ = minw_host::num_sms() > 0 ? minw_host::num_sms() : 148;
        const int tiles_ = p.nbx * p.nby * p.nbb * p.ntn;
        const int ks_ = (a.workspace != nullptr && !a.pool && !a.upd) ? (a.ksplit > 0 ? a.ksplit : auto_ksplit(tiles_, p.nk, sms_))
                                                            : 1;
        p.pair = (pair_pref() && !p.trans && p.BN == 256 && a.O % 256 == 0 && p.nk >= 18 && ks_ <= 1) ? 1 : 0;
        // E2M1 pairs of 128-channel tiles: each CTA accumulates 128 pixels x 128 channels, so two
        // accumulators fit beside the scale factors (a 256-channel E2M1 tile has one)
        if (a.pair_n128 && p.fp4 && !p.trans && a.O % 128 == 0 && ks_ <= 1 && !a.upd) {
            p.BN = 128;
            p.ntn = (a.O + 127) / 128;
            p.pair = 1;
        }
    }
    p.b_bytes = (uint32_t)((p.pair ? p.BN / 2 : p.BN) * p.cb);   // pairs: each CTA holds half the weight rows
    const size_t o32 = ((size_t)a.O + 31) & ~(size_t)31;
    const size_t thr_bytes = a.quant_out ? (o32 * p.nlev + o32 / 32 + 10) * sizeof(float) : 0;
    // staging tiles of the row-contiguous stores: a layer that may split along K,
    // or whose fp32 output is a fully connected one (1 x 1 images)
    const bool resid_ = a.res_codes != nullptr || a.res_f32 != nullptr || a.y_nhwc != nullptr;
    const bool rowst_fc = !p.trans && a.y_out != nullptr && a.Ho == 1 && a.Wo == 1 && !a.pool && !a.quant_out &&
                          a.acc_out == nullptr && !resid_;
    const bool may_split = a.workspace != nullptr && !a.pool && !p.trans && !p.pair && !a.upd;
    if (a.upd && !rowst_fc) return MINW_EUNSUPPORTED;     // the update runs in the row-contiguous epilogue
    p.ystage = (rowst_fc || may_split) ? 8 * 32 * 16 : 0;
    size_t budget = 224 * 1024 - 1024 - 256 - thr_bytes - (p.ystage ? (size_t)p.ystage * 4 + 16 : 0);
    // resident weights (plan option resident_weights): a layer not split along K
    // whose weights per CTA fit beside at least three activation stages, with
    // at least as many CTA units as channel tiles and two or more pixel tiles
    // per unit; it halves the loads per K block and frees the weight warp to
    // issue activation stages
    p.wres = 0;
    p.wres_off = 0;
    {
        const int sms_ = minw_host::num_sms() > 0 ? minw_host::num_sms() : 148;
        const int tiles_ = p.nbx * p.nby * p.nbb * p.ntn;
        const int ks_ = may_split ? (a.ksplit > 0 ? a.ksplit : auto_ksplit(tiles_, p.nk, sms_)) : 1;
        const int cl_ = p.pair ? 2 : 1;
        const int units = sms_ / cl_;
        const int tiles_mp_ = (p.nbx * p.nby * p.nbb + cl_ - 1) / cl_ * cl_;
        const size_t wbytes = (size_t)p.nk * p.b_bytes;
        if (minw_host::plan_options().resident_weights && ks_ <= 1 && !rowst_fc && !a.upd && p.ntn <= units &&
            tiles_mp_ / cl_ >= 2 * (units / p.ntn) && wbytes + 3 * (size_t)p.a_bytes <= budget) {
            p.wres = 1;
            budget -= wbytes;
        }
    }
    // two K blocks per stage (one commit per 8 or 4 MMAs) when three such stages fit
    const size_t blk = (size_t)p.a_bytes + (p.wres ? 0 : p.b_bytes);
    p.kps = (kps_pref() != 1 && p.nk >= 2 && budget / (2 * blk) >= 3) ? 2 : 1;
    p.stage_bytes = (uint32_t)(p.kps * blk);
    int S = (int)(budget / p.stage_bytes);
    if (S > 8) S = 8;
    if (S < 2) return MINW_EUNSUPPORTED;
    p.S = S;
    if (p.wres) p.wres_off = (uint32_t)S * p.stage_bytes;
    // lanes issuing TMA loads per producer warp (plan option tma_lanes), at most one per ring slot
    p.tlanes = minw_host::plan_options().tma_lanes;
    if (p.tlanes > p.S) p.tlanes = p.S;
    if (p.tlanes < 1) p.tlanes = 1;
    // MMA N: the output channels, or the 256 pixels of a channel-major tile (M = 128 either way)
    const int mma_n = p.trans ? 256 : p.BN;
    p.acc_cols = mma_n;
    // D fp32; A and B E4M3 (kind::f8f6f4), bf16 (kind::f16), or E2M1 with UE8M0
    // block scales (kind::mxf4: formats E2M1 = 1, scale type bit 23)
    const uint32_t mrows = (uint32_t)(p.pair ? 256 : 128);
    if (p.fp4) {
        p.idesc = (1u << 7) | (1u << 10) | ((uint32_t)(mma_n >> 3) << 17) | (1u << 23) | ((mrows >> 4) << 24);
        // all 512 columns: the accumulators below column 448, the unit scale
        // factors of A at 448 and of B at 480
        p.tmem_cols = 512;
        p.sf_col = 448;
        p.nacc = 2 * mma_n <= 448 ? 2 : 1;
    } else {
        const uint32_t fmt = a.bf16 ? 1u : 0u;
        p.idesc = (1u << 4) | (fmt << 7) | (fmt << 10) | ((uint32_t)(mma_n >> 3) << 17) | ((mrows >> 4) << 24);
        uint32_t cols = 32;
        while ((int)cols < 2 * mma_n) cols <<= 1;         // two accumulators
        p.tmem_cols = cols;
        p.sf_col = 0;
        p.nacc = 2;
    }
    p.acc_out = a.acc_out; p.y_out = a.y_out; p.scale = a.scale; p.shift = a.shift;
    p.upd = a.upd; p.upd_lr = a.upd_lr; p.upd_2a = a.upd_2a;
    p.pool = a.pool; p.quant_out = a.quant_out; p.qo = a.qo;
    p.planes_out = a.planes_out; p.codes_out = a.codes_out;
    p.res_codes = a.res_codes; p.res_unit = a.res_unit; p.res_f32 = a.res_f32; p.y_nhwc = a.y_nhwc;
    p.ythr = a.ythr;
    p.hb_out = a.hb_out; p.hb_ld = a.hb_ld; p.hb_off = a.hb_off; p.hb_res = a.hb_res; p.hb_z = a.hb_z;

    const int tiles = p.nbx * p.nby * p.nbb * p.ntn;
    const int sms = minw_host::num_sms() > 0 ? minw_host::num_sms() : 148;
    p.ksplit = 1;
    pl.thr_ws = nullptr;
    if (a.workspace != nullptr && !a.pool && !p.trans && !p.pair && !a.upd) {
        // workspace: [breakpoints, when not given][ksplit partial-sum slices]
        const size_t tb = (a.quant_out && a.thr == nullptr) ? thr_ws_bytes(a.O, p.nlev) : 0;
        const size_t sb = slice_bytes(tiles, p.BN);
        int ks = a.ksplit > 0 ? a.ksplit : auto_ksplit(tiles, p.nk, sms);
        if (a.workspace_bytes > tb) {
            const size_t cap = (a.workspace_bytes - tb) / sb;
            if ((size_t)ks > cap) ks = (int)cap;
        } else {
            ks = 1;
        }
        if (ks > p.nk) ks = p.nk;
        // the reduction's threads (one per four channels of a tile row) index in 32 bits
        if ((long long)p.nbx * p.nby * p.nbb * 128 * ((a.O + 31) / 32) * 8 >= (1ll << 31)) ks = 1;
        if (ks > 1) {
            p.ksplit = ks;
            uint8_t *w = reinterpret_cast<uint8_t *>(a.workspace);
            if (tb) pl.thr_ws = reinterpret_cast<float *>(w);
            p.part = reinterpret_cast<int32_t *>(w + tb);
        }
    }
    p.rowst = (p.ystage > 0 && (p.ksplit > 1 || rowst_fc)) ? 1 : 0;
    const int tiles_m = p.nbx * p.nby * p.nbb;
    // CTA pairs walk pixel tiles two by two (an odd count gets one padded tile)
    p.cl = p.pair ? 2 : 1;
    p.tiles_mp = (tiles_m + p.cl - 1) / p.cl * p.cl;
    if (!encode) return MINW_OK;
    minw_host::EncodeTiledFn enc = minw_host::tensor_map_encoder();
    if (enc == nullptr) return MINW_ECUDA;
    const CUtensorMapSwizzle swz = p.cb == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
    const CUtensorMapDataType dt = a.bf16 ? CU_TENSOR_MAP_DATA_TYPE_UINT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8;
    const cuuint64_t es_ = (cuuint64_t)p.esize;
    // tensor-map elements per pixel row and per K block: bytes for packed E2M1
    const cuuint64_t cel = (cuuint64_t)(p.fp4 ? a.C / 2 : a.C);
    const cuuint32_t kel = (cuuint32_t)(p.fp4 ? p.cb : p.ck);
    {
        const cuuint64_t rel = (a.bf16 && a.ldc) ? (cuuint64_t)a.ldc : cel;     // elements per pixel row
        const cuuint64_t dims[4] = {cel, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.B};
        const cuuint64_t strides[3] = {rel * es_, (cuuint64_t)a.W * rel * es_, (cuuint64_t)a.H * a.W * rel * es_};
        const cuuint32_t sd = (cuuint32_t)p.stride;
        const cuuint32_t box[4] = {kel, (cuuint32_t)p.bw * sd, (cuuint32_t)p.bh * sd, (cuuint32_t)p.bb};
        const cuuint32_t es[4] = {1u, sd, sd, 1u};
        if (enc(&pl.tmA, dt, 4, const_cast<uint8_t *>(a.act8), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return MINW_ECUDA;
    }
    {
        const long long K = (long long)a.kh * a.kw * cel;
        const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)a.O};
        const cuuint64_t strides[1] = {(cuuint64_t)K * es_};
        const cuuint32_t box[2] = {kel, (cuuint32_t)(p.dup ? 64 : p.BN / p.cl)};
        const cuuint32_t es[2] = {1u, 1u};
        if (enc(&pl.tmB, dt, 2, const_cast<uint8_t *>(a.wgt8), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return MINW_ECUDA;
    }
    const int items = p.tiles_mp * p.ntn * p.ksplit;
    int grid = items < sms ? items : sms;
    grid -= grid % p.cl;
    if (p.wres) grid = (sms / p.cl / p.ntn) * p.ntn * p.cl;     // whole units per channel tile
    pl.grid = dim3((unsigned)grid);
    pl.smem = (size_t)p.S * p.stage_bytes + (p.wres ? (size_t)p.nk * p.b_bytes : 0) + 1024 + 256 + thr_bytes +
              (p.ystage ? (size_t)p.ystage * 4 + 16 : 0);
    // more than half of an SM's shared memory: exactly one CTA (and one TMEM
    // allocation) per SM
    if (pl.smem < 120 * 1024) pl.smem = 120 * 1024;
    return MINW_OK;
}

// Resident clusters of cl CTAs for a launch of kern with smem bytes (cached:
// the answer depends only on these three).
static int max_active_clusters(const void *kern, int cl, size_t smem, const cudaLaunchConfig_t &cfg) {
    struct Entry { const void *k; int cl; size_t smem; int n; };
    static Entry cache[32];
    static int used = 0;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < used; ++i)
        if (cache[i].k == kern && cache[i].cl == cl && cache[i].smem == smem) return cache[i].n;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
    }
    if (used < 32) cache[used++] = Entry{kern, cl, smem, n};
    return n;
}

}  // namespace tc

size_t conv_tc_workspace_bytes(const ConvArgs &a) {
    tc::Params p{};
    if (a.pool || !tc::plan_shape(a, p)) return 0;
    const int nbb = (a.B + p.bb - 1) / p.bb;
    const int tiles = p.nbx * p.nby * nbb * ((a.O + p.BN - 1) / p.BN);
    const int nk = a.kh * a.kw * (a.C / tc::chunk_channels(a));
    const int sms = minw_host::num_sms() > 0 ? minw_host::num_sms() : 148;
    const int ks = tc::auto_ksplit(tiles, nk, sms);
    if (ks < 2) return 0;
    return tc::thr_ws_bytes(a.O, 7) + (size_t)ks * tc::slice_bytes(tiles, p.BN);
}

size_t conv_tc_min_split_bytes(const ConvArgs &a) {
    tc::Params p{};
    if (a.pool || !tc::plan_shape(a, p)) return 0;
    const int nbb = (a.B + p.bb - 1) / p.bb;
    const int tiles = p.nbx * p.nby * nbb * ((a.O + p.BN - 1) / p.BN);
    const int nk = a.kh * a.kw * (a.C / tc::chunk_channels(a));
    const int sms = minw_host::num_sms() > 0 ? minw_host::num_sms() : 148;
    if (tc::auto_ksplit(tiles, nk, sms) < 2) return 0;
    return tc::thr_ws_bytes(a.O, 7) + 2 * tc::slice_bytes(tiles, p.BN);
}

static bool conv_tc_residual(const ConvArgs &a) {
    return a.res_codes != nullptr || a.res_f32 != nullptr || a.y_nhwc != nullptr;
}

bool conv_tc_supported(const ConvArgs &a) {
    tc::Params p{};
    if (!tc::plan_shape(a, p)) return false;
    // E2M1 operands: rows of 64 or 128 bytes (128 or 256 channels)
    if (a.fp4 && (a.bf16 || a.C % 128 != 0)) return false;
    // bf16 operands: real-valued accumulators, so fp32 BN outputs only
    if (a.bf16 && (a.quant_out || a.acc_out != nullptr || (a.y_out == nullptr) == (a.hb_out == nullptr) ||
                   conv_tc_residual(a)))
        return false;
    if (a.hb_out != nullptr && (!a.bf16 || a.pool || a.workspace != nullptr || a.upd)) return false;
    if (a.quant_out && (size_t)a.O * num_levels(a.qo.bits) * sizeof(float) > 64 * 1024) return false;
    if (a.quant_out && a.codes_out != nullptr && a.O % 16 != 0) return false;
    if (a.acc_out != nullptr && a.pool) return false;
    return true;
}


int conv_tc_ksplit(const ConvArgs &a) {
    if (!conv_tc_supported(a)) return 0;
    tc::Plan pl;
    return tc::make_plan(a, pl, false) == MINW_OK ? pl.p.ksplit : 0;
}

bool conv_tc_pairs128(const ConvArgs &a) {
    if (!conv_tc_supported(a)) return false;
    tc::Plan pl;
    return tc::make_plan(a, pl, false) == MINW_OK && pl.p.pair && pl.p.BN == 128;
}

bool conv_tc_n128(const ConvArgs &a) {
    if (!conv_tc_supported(a) || !a.n128 || !a.fp4) return false;
    ConvArgs b = a;
    b.n128 = 0;
    tc::Plan pl, pl0;
    // a change of tiling only: the default plan has wider single-CTA tiles
    return tc::make_plan(a, pl, false) == MINW_OK && tc::make_plan(b, pl0, false) == MINW_OK && !pl.p.pair &&
           !pl.p.trans && pl.p.BN == 128 && pl0.p.BN > 128;
}

int conv_tc_launches(const ConvArgs &a) {
    if (a.workspace == nullptr || a.pool) return 1;
    tc::Plan pl;
    if (tc::make_plan(a, pl) != MINW_OK || pl.p.ksplit < 2) return 1;
    // main pass + reduction, plus the breakpoints when the reduction needs them
    return (a.quant_out && a.thr == nullptr && !conv_tc_residual(a)) ? 3 : 2;
}

minw_status launch_thresholds(const float *scale, const float *shift, int O, const QParams &q, float *out,
                              cudaStream_t s) {
    tc::thresholds_kernel<<<(O + 127) / 128, 128, 0, s>>>(scale, shift, O, q, out);
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

minw_status launch_conv_tc(const ConvArgs &a, cudaStream_t s) {
    if (!a.act8 || !a.wgt8) return MINW_EINVAL;
    if (!conv_tc_supported(a)) return MINW_EUNSUPPORTED;
    tc::Plan pl;
    minw_status st = tc::make_plan(a, pl);
    if (st != MINW_OK) return st;
    const int outb = a.quant_out ? a.qo.bits : 0;
    const bool split = pl.p.ksplit > 1;
    const int kout = split ? 0 : outb;            // the split main pass writes only partial sums
    typedef void (*TcKernel)(const CUtensorMap, const CUtensorMap, const tc::Params);
    // [pair][E2M1][output bits]; bf16 operands have fp32 outputs only
    static const TcKernel kernels[2][2][4] = {
        {{tc::conv_tc_kernel<0, false, 0>, tc::conv_tc_kernel<1, false, 0>, tc::conv_tc_kernel<2, false, 0>,
          tc::conv_tc_kernel<3, false, 0>},
         {tc::conv_tc_kernel<0, false, 2>, tc::conv_tc_kernel<1, false, 2>, tc::conv_tc_kernel<2, false, 2>,
          tc::conv_tc_kernel<3, false, 2>}},
        {{tc::conv_tc_kernel<0, true, 0>, tc::conv_tc_kernel<1, true, 0>, tc::conv_tc_kernel<2, true, 0>,
          tc::conv_tc_kernel<3, true, 0>},
         {tc::conv_tc_kernel<0, true, 2>, tc::conv_tc_kernel<1, true, 2>, tc::conv_tc_kernel<2, true, 2>,
          tc::conv_tc_kernel<3, true, 2>}}};
    static size_t configured[2][2][4] = {}, configured_bf16[2] = {0, 0};
    const int kp = pl.p.pair ? 1 : 0, kf = pl.p.fp4 ? 1 : 0;
    TcKernel kern = a.bf16 ? (kp ? tc::conv_tc_kernel<0, true, 1> : tc::conv_tc_kernel<0, false, 1>)
                           : kernels[kp][kf][kout];
    size_t &conf = a.bf16 ? configured_bf16[kp] : configured[kp][kf][kout];
    if (pl.smem > conf) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl.smem) != cudaSuccess)
            return MINW_ECUDA;
        conf = pl.smem;
    }
    const float *thr = a.thr;
    if (split && a.quant_out && thr == nullptr && !conv_tc_residual(a)) {
        tc::thresholds_kernel<<<(a.O + 127) / 128, 128, 0, s>>>(a.scale, a.shift, a.O, a.qo, pl.thr_ws);
        thr = pl.thr_ws;
    }
    tc::Params pm = pl.p;
    pm.wait_cycles = (long long)minw_host::plan_options().wait_cycles;
    pm.stall = pl.p.pair ? 0 : minw_host::take_stall(MINW_STALL_CONV_TC);
    if (split) {
        pm.quant_out = 0;
        pm.acc_out = nullptr;
        pm.y_out = nullptr;
    }
    if (pm.cl == 1) {
        if (minw_host::launch_pdl(kern, pl.grid, dim3(tc::NT), pl.smem, s, pl.tmA, pl.tmB, pm) != cudaSuccess) return MINW_ECUDA;
    } else {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = pl.grid;
        cfg.blockDim = dim3(tc::NT);
        cfg.dynamicSmemBytes = pl.smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[2];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = (unsigned)pm.cl;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[1].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        minw_host::max_shared_carveout(reinterpret_cast<const void *>(kern));
        // a persistent grid: no more clusters than can be resident at once
        const int maxc = tc::max_active_clusters(reinterpret_cast<const void *>(kern), pm.cl, pl.smem, cfg);
        if (maxc < 1) return MINW_EUNSUPPORTED;
        if ((int)cfg.gridDim.x > maxc * pm.cl) cfg.gridDim.x = (unsigned)(maxc * pm.cl);
        cfg.numAttrs = minw_host::pdl_enabled() ? 2 : 1;
        if (cudaLaunchKernelEx(&cfg, kern, pl.tmA, pl.tmB, pm) != cudaSuccess) return MINW_ECUDA;
    }
    if (split) {
        const int tiles_m = pl.p.nbx * pl.p.nby * pl.p.nbb;
        const long long threads = (long long)tiles_m * 128 * ((a.O + 31) / 32) * 8;
        if (threads >= (1ll << 31)) return MINW_EUNSUPPORTED;     // the reduction indexes in 32 bits
        const unsigned blocks = (unsigned)((threads + 255) / 256);
        switch (outb) {
            case 1: minw_host::launch_pdl(tc::splitk_reduce_kernel<1>, dim3(blocks), dim3(256), 0, s, pl.p, thr); break;
            case 2: minw_host::launch_pdl(tc::splitk_reduce_kernel<2>, dim3(blocks), dim3(256), 0, s, pl.p, thr); break;
            case 3: minw_host::launch_pdl(tc::splitk_reduce_kernel<3>, dim3(blocks), dim3(256), 0, s, pl.p, thr); break;
            default: minw_host::launch_pdl(tc::splitk_reduce_kernel<0>, dim3(blocks), dim3(256), 0, s, pl.p, thr); break;
        }
    }
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

}  // namespace minw

extern "C" minw_status minw_get_last_device_error(void *stream) {
    if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return MINW_ECUDA;
    int flag = 0;
    if (cudaMemcpyFromSymbol(&flag, minw::g_device_error, sizeof(int)) != cudaSuccess) return MINW_ECUDA;
    if (flag) {
        const int zero = 0;
        if (cudaMemcpyToSymbol(minw::g_device_error, &zero, sizeof(int)) != cudaSuccess) return MINW_ECUDA;
    }
    const int first = minw::take_first_error();
    const int first_tc = minw::take_first_tc_error();
    if (first < 0 || first_tc < 0) return MINW_ECUDA;
    return (flag || first || first_tc) ? MINW_ETIMEOUT : MINW_OK;
}

minw_host::EncodeTiledFn minw_host::tensor_map_encoder() {
    static EncodeTiledFn fn = nullptr;
    if (fn == nullptr) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    }
    return fn;
}
