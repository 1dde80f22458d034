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
// Warp roles (192 threads): warp 0 issues TMA, warp 1 owns TMEM and issues
// MMAs (4 x K=32 per stage), warps 2-5 drain TMEM (one lane quarter each) and
// run the fused epilogue: exact int conversion, 2x2 max pool via warp
// shuffles, BN fmaf, HardTanh, quantize, and stores of the next layer's codes
// or bit-planes (or raw int32 / fp32 NCHW outputs).
//
// Every mbarrier wait is bounded (about one second of clock64); a wait that
// runs out sets the device error flag read by minw_get_last_device_error, the
// CTA stops issuing work, drains its own TMA loads and frees its TMEM.
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace minw {

__device__ int g_device_error = 0;

namespace tc {

constexpr int NT = 192;
constexpr int A_BYTES = 128 * 128;
constexpr long long WAIT_CYCLES = 1ll << 31;

struct Params {
    int B, C, H, W, O, kh, kw, pad, Ho, Wo;
    int bw, bh, bb, nbx, nby;
    int BN, nck, nk, S;
    uint32_t stage_bytes, idesc, tmem_cols;
    int32_t *acc_out;
    float *y_out;
    const float *scale, *shift;
    int pool, quant_out;
    QParams qo;
    uint32_t *planes_out;
    uint8_t *codes_out;
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
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait for the phase with the given parity; false (and the device
// error flag set) when it does not complete within WAIT_CYCLES.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > WAIT_CYCLES) {
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

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];\n" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
        : "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile stored as rows of
// 128 bytes with the 128-byte swizzle: 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);   // start address
    d |= (uint64_t)1 << 16;                             // leading byte offset (unused here)
    d |= (uint64_t)(1024 >> 4) << 32;                   // stride byte offset: next 8 rows
    d |= (uint64_t)1 << 46;                             // descriptor version
    d |= (uint64_t)2 << 61;                             // 128-byte swizzle
    return d;
}

__device__ __forceinline__ void mma_f8(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

__device__ __forceinline__ void mma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                     smem_u32(bar))
                 : "memory");
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

__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

__global__ void __launch_bounds__(NT, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + (size_t)p.S * p.stage_bytes);
    uint64_t *empty = full + p.S;
    uint64_t *accum = empty + p.S;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(accum + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tile_m = blockIdx.x, tile_n = blockIdx.y;
    const int xb = tile_m % p.nbx;
    const int yb = (tile_m / p.nbx) % p.nby;
    const int bbk = tile_m / (p.nbx * p.nby);
    const int x0 = xb * p.bw, y0 = yb * p.bh, b0 = bbk * p.bb;
    const int o0 = tile_n * p.BN;

    if (threadIdx.x == 0) {
        for (int s = 0; s < p.S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(accum, 1);
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(tmem_slot)),
                     "r"(p.tmem_cols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem_d = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer ----------------
            asm volatile("prefetch.tensormap [%0];\n" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
            asm volatile("prefetch.tensormap [%0];\n" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
            int issued = 0;
            for (int ks = 0; ks < p.nk; ++ks) {
                const int s = ks % p.S, u = ks / p.S;
                if (u > 0 && !mbar_wait(&empty[s], (u - 1) & 1)) break;
                const int tap = ks / p.nck;
                const int c0 = (ks - tap * p.nck) * 128;
                const int ky = tap / p.kw, kx = tap - (tap / p.kw) * p.kw;
                uint8_t *sa = smem + (size_t)s * p.stage_bytes;
                mbar_expect_tx(&full[s], p.stage_bytes);
                tma_load_4d(sa, &tmA, &full[s], c0, x0 - p.pad + kx, y0 - p.pad + ky, b0);
                tma_load_2d(sa + A_BYTES, &tmB, &full[s], tap * p.C + c0, o0);
                ++issued;
            }
            // drain: every issued load has landed before the CTA can exit
            for (int j = issued > p.S ? issued - p.S : 0; j < issued; ++j)
                if (!mbar_wait(&full[j % p.S], (j / p.S) & 1)) break;
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer ----------------
            for (int ks = 0; ks < p.nk; ++ks) {
                const int s = ks % p.S, u = ks / p.S;
                if (!mbar_wait(&full[s], u & 1)) break;
                fence_after();
                const uint32_t sa = smem_u32(smem + (size_t)s * p.stage_bytes);
                const uint64_t adesc = sw128_desc(sa);
                const uint64_t bdesc = sw128_desc(sa + A_BYTES);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    mma_f8(tmem_d, adesc + 2 * kk, bdesc + 2 * kk, p.idesc, (ks | kk) != 0);
                mma_commit(&empty[s]);
            }
            mma_commit(accum);
        }
    } else {
        // ---------------- epilogue: warps 2..5 ----------------
        const int q = warp & 3;                   // TMEM lane quarter of this warp
        const int r = q * 32 + lane;              // tile row = output pixel
        const int b = b0 + r / (p.bh * p.bw);
        const int y = y0 + (r / p.bw) % p.bh;
        const int x = x0 + r % p.bw;
        const bool valid = b < p.B && y < p.Ho && x < p.Wo;
        const bool ok = mbar_wait(accum, 0);
        fence_after();
        const bool writer = valid && (!p.pool || ((x & 1) == 0 && (y & 1) == 0));
        const int Hp = p.pool ? p.Ho / 2 : p.Ho, Wp = p.pool ? p.Wo / 2 : p.Wo;
        const int yp = p.pool ? y / 2 : y, xp = p.pool ? x / 2 : x;
        const long long opix = ((long long)b * Hp + yp) * Wp + xp;
        const int NWo = (p.O + 31) >> 5;
        uint32_t pw[3] = {0u, 0u, 0u};
        if (ok) {
            for (int ch = 0; ch < p.BN / 16; ++ch) {
                __syncwarp();
                uint32_t v[16];
                tmem_ld16(tmem_d + ((uint32_t)(q * 32) << 16) + (uint32_t)(ch * 16), v);
                int a[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) a[j] = __float2int_rn(__uint_as_float(v[j]));
                if (p.pool) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        a[j] = max(a[j], __shfl_xor_sync(0xffffffffu, a[j], 1));
                        a[j] = max(a[j], __shfl_xor_sync(0xffffffffu, a[j], p.bw));
                    }
                }
                const int ob = o0 + ch * 16;
                if (p.acc_out != nullptr && valid) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        if (ob + j < p.O)
                            p.acc_out[(((long long)b * p.O + ob + j) * p.Ho + y) * p.Wo + x] = a[j];
                }
                if (writer && (p.y_out != nullptr || p.quant_out)) {
                uint32_t cw[4] = {0u, 0u, 0u, 0u};
                uint32_t bits16[3] = {0u, 0u, 0u};
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int o = ob + j;
                    if (o >= p.O) break;
                    float yv = fmaf((float)a[j], __ldg(p.scale + o), __ldg(p.shift + o));
                    if (p.quant_out) {
                        yv = fminf(fmaxf(yv, -1.0f), 1.0f);
                        const int lv = level_units(yv * p.qo.scale, p.qo);
                        cw[j >> 2] |= (uint32_t)level_code_e4m3(lv) << ((j & 3) * 8);
                        const uint32_t pb = level_plane_bits(lv, p.qo.bits);
                        bits16[0] |= (pb & 1u) << j;
                        bits16[1] |= ((pb >> 1) & 1u) << j;
                        bits16[2] |= ((pb >> 2) & 1u) << j;
                    }
                    if (p.y_out != nullptr)
                        p.y_out[(((long long)b * p.O + o) * Hp + yp) * Wp + xp] = yv;
                }
                if (p.quant_out && p.codes_out != nullptr)
                    *reinterpret_cast<uint4 *>(p.codes_out + opix * p.O + ob) = make_uint4(cw[0], cw[1], cw[2], cw[3]);
                if (p.quant_out && p.planes_out != nullptr) {
                    const int half = (ob >> 4) & 1;
#pragma unroll
                    for (int k = 0; k < 3; ++k) pw[k] |= bits16[k] << (16 * half);
                    if (half == 1 || ch == p.BN / 16 - 1 || ob + 16 >= p.O) {
                        uint32_t *dst = p.planes_out + (opix * p.qo.bits) * NWo + (ob >> 5);
                        for (int k = 0; k < p.qo.bits; ++k) dst[k * NWo] = pw[k];
                        pw[0] = pw[1] = pw[2] = 0u;
                    }
                }
                }  // writer
            }
        }
        __syncwarp();
        fence_before();
    }
    __syncthreads();
    if (warp == 1) {
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem_d), "r"(p.tmem_cols));
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
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
};

static bool plan_shape(const ConvArgs &a, Params &p) {
    if (a.stride != 1 || a.C % 128 != 0 || a.pad >= a.kh || a.pad >= a.kw) return false;
    int bw = pow2_ceil(a.Wo);
    if (bw > 128) bw = 128;
    if (a.pool && bw > 16) bw = 16;
    int bh = pow2_ceil(a.Ho);
    if (bh > 128 / bw) bh = 128 / bw;
    const int bb = 128 / (bw * bh);
    if (a.pool && (bw < 2 || bh < 2)) return false;
    p.bw = bw; p.bh = bh; p.bb = bb;
    p.nbx = (a.Wo + bw - 1) / bw;
    p.nby = (a.Ho + bh - 1) / bh;
    int BN = ((a.O + 15) / 16) * 16;
    if (BN > 256) BN = 256;
    p.BN = BN;
    return true;
}

static minw_status make_plan(const ConvArgs &a, Plan &pl) {
    Params &p = pl.p;
    p = Params{};
    if (!plan_shape(a, p)) return MINW_EUNSUPPORTED;
    p.B = a.B; p.C = a.C; p.H = a.H; p.W = a.W; p.O = a.O; p.kh = a.kh; p.kw = a.kw; p.pad = a.pad;
    p.Ho = a.Ho; p.Wo = a.Wo;
    p.nck = a.C / 128;
    p.nk = a.kh * a.kw * p.nck;
    p.stage_bytes = (uint32_t)(A_BYTES + p.BN * 128);
    const size_t budget = (p.BN <= 128) ? 110 * 1024 : 200 * 1024;
    int S = (int)(budget / p.stage_bytes);
    if (S > 6) S = 6;
    if (S < 2) S = 2;
    p.S = S;
    p.idesc = (1u << 4) | (0u << 7) | (0u << 10) | ((uint32_t)(p.BN >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
    uint32_t cols = 32;
    while ((int)cols < p.BN) cols <<= 1;
    p.tmem_cols = cols;
    p.acc_out = a.acc_out; p.y_out = a.y_out; p.scale = a.scale; p.shift = a.shift;
    p.pool = a.pool; p.quant_out = a.quant_out; p.qo = a.qo;
    p.planes_out = a.planes_out; p.codes_out = a.codes_out;

    EncodeTiledFn enc = encode_fn();
    if (enc == nullptr) return MINW_ECUDA;
    {
        const cuuint64_t dims[4] = {(cuuint64_t)a.C, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.B};
        const cuuint64_t strides[3] = {(cuuint64_t)a.C, (cuuint64_t)a.W * a.C, (cuuint64_t)a.H * a.W * a.C};
        const cuuint32_t box[4] = {128u, (cuuint32_t)p.bw, (cuuint32_t)p.bh, (cuuint32_t)p.bb};
        const cuuint32_t es[4] = {1u, 1u, 1u, 1u};
        if (enc(&pl.tmA, CU_TENSOR_MAP_DATA_TYPE_UINT8, 4, const_cast<uint8_t *>(a.act8), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return MINW_ECUDA;
    }
    {
        const long long K = (long long)a.kh * a.kw * a.C;
        const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)a.O};
        const cuuint64_t strides[1] = {(cuuint64_t)K};
        const cuuint32_t box[2] = {128u, (cuuint32_t)p.BN};
        const cuuint32_t es[2] = {1u, 1u};
        if (enc(&pl.tmB, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(a.wgt8), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return MINW_ECUDA;
    }
    const int nbb = (a.B + p.bb - 1) / p.bb;
    pl.grid = dim3((unsigned)(p.nbx * p.nby * nbb), (unsigned)((a.O + p.BN - 1) / p.BN));
    pl.smem = (size_t)p.S * p.stage_bytes + 1024 + 256;
    return MINW_OK;
}

}  // namespace tc

bool conv_tc_supported(const ConvArgs &a) {
    tc::Params p{};
    if (!tc::plan_shape(a, p)) return false;
    if (a.quant_out && a.codes_out != nullptr && a.O % 16 != 0) return false;
    if (a.acc_out != nullptr && a.pool) return false;
    return true;
}

minw_status launch_conv_tc(const ConvArgs &a, cudaStream_t s) {
    if (!a.act8 || !a.wgt8) return MINW_EINVAL;
    if (!conv_tc_supported(a)) return MINW_EUNSUPPORTED;
    tc::Plan pl;
    minw_status st = tc::make_plan(a, pl);
    if (st != MINW_OK) return st;
    static size_t configured = 0;
    if (pl.smem > configured) {
        if (cudaFuncSetAttribute(tc::conv_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl.smem) !=
            cudaSuccess)
            return MINW_ECUDA;
        configured = pl.smem;
    }
    tc::conv_tc_kernel<<<pl.grid, tc::NT, pl.smem, s>>>(pl.tmA, pl.tmB, pl.p);
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
        return MINW_ETIMEOUT;
    }
    return MINW_OK;
}
