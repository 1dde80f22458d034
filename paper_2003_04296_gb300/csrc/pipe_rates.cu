// pipe_rates.cu -- measured throughput of the pipes the quantized
// convolution can run on (minw_measure_pipe_rates): the integer pipe's
// XOR + POPC + add loop (the bit-serial path of Table I), the legacy binary
// and int8 MMAs the sm_103a toolchain exposes (mma.sync b1 xor.popc, s8),
// the tcgen05 tensor-core kinds the library uses (E4M3 kind::f8f6f4, E2M1
// kind::mxf4 with unit scales, bf16 kind::f16) issued warp-uniformly at
// M = 128, N = 128 and 256 with a commit every four MMAs, and the time one
// thread spends per 32 KB TMA box from L2.  These rates are the evidence
// behind the choice of path per shape; every wait is bounded.
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "kernels.cuh"

namespace {

__device__ int g_rate_timeout = 0;

__device__ __forceinline__ uint32_t s32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ bool rwait(uint64_t *bar, uint32_t parity) {
    const long long t0 = clock64();
    while (true) {
        uint32_t ok;
        asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
                     : "=r"(ok)
                     : "r"(s32(bar)), "r"(parity)
                     : "memory");
        if (ok) return true;
        if (clock64() - t0 > (1ll << 31)) {
            atomicExch(&g_rate_timeout, 1);
            return false;
        }
    }
}

// 16 independent XOR + POPC + add chains per thread
__global__ void popc_rate_kernel(uint32_t *out, int iters, uint32_t seed) {
    uint32_t a[4], w[4];
    int acc[16];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        a[i] = seed * (threadIdx.x + 1) + i;
        w[i] = seed ^ (blockIdx.x * 977u + i * 31u);
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) acc[i] = 0;
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[i * 4 + j] += __popc(a[i] ^ w[j]);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            a[i] += 0x9E3779B9u;
            w[i] ^= a[i];
        }
    }
    int s = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) s += acc[i];
    out[blockIdx.x * blockDim.x + threadIdx.x] = (uint32_t)s;
}

// four independent accumulator sets of the legacy warp MMAs
template <bool B1>
__global__ void warp_mma_rate_kernel(uint32_t *out, int iters, uint32_t seed) {
    const uint32_t a0 = seed * threadIdx.x, a1 = a0 ^ 0x55u, a2 = a0 + 7u, a3 = a0 * 3u;
    const uint32_t b0 = seed ^ threadIdx.x, b1 = b0 + 11u;
    int c[4][4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int i = 0; i < 4; ++i) c[k][i] = 0;
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if constexpr (B1)
                asm volatile("mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.xor.popc "
                             "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
                             : "+r"(c[k][0]), "+r"(c[k][1]), "+r"(c[k][2]), "+r"(c[k][3])
                             : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
            else
                asm volatile("mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 "
                             "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
                             : "+r"(c[k][0]), "+r"(c[k][1]), "+r"(c[k][2]), "+r"(c[k][3])
                             : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
        }
    }
    int s = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int i = 0; i < 4; ++i) s += c[k][i];
    out[blockIdx.x * blockDim.x + threadIdx.x] = (uint32_t)s;
}

// K-major operand in 128-byte rows with the 128-byte swizzle
__device__ __forceinline__ uint64_t rdesc(uint32_t a) {
    return (uint64_t)((a & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// KIND: 0 E4M3 (kind::f8f6f4), 1 E2M1 (kind::mxf4, unit UE8M0 scales), 2 bf16 (kind::f16);
// each MMA consumes 32 bytes of K of each operand row
template <int KIND>
__device__ __forceinline__ void rate_mma(uint32_t d, uint64_t a, uint64_t b, uint32_t id, uint32_t acc, uint32_t sf) {
    if constexpr (KIND == 1)
        asm volatile("{\n .reg .pred p, e;\n .reg .b32 r;\n setp.ne.b32 p, %4, 0;\n elect.sync r|e, 0xffffffff;\n"
                     " @e tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%0], %1, %2, %3, [%5], [%6], p;\n}\n"
                     ::"r"(d), "l"(a), "l"(b), "r"(id), "r"(acc), "r"(sf), "r"(sf + 32u));
    else if constexpr (KIND == 2)
        asm volatile("{\n .reg .pred p, e;\n .reg .b32 r;\n setp.ne.b32 p, %4, 0;\n elect.sync r|e, 0xffffffff;\n"
                     " @e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
                     ::"r"(d), "l"(a), "l"(b), "r"(id), "r"(acc));
    else
        asm volatile("{\n .reg .pred p, e;\n .reg .b32 r;\n setp.ne.b32 p, %4, 0;\n elect.sync r|e, 0xffffffff;\n"
                     " @e tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n"
                     ::"r"(d), "l"(a), "l"(b), "r"(id), "r"(acc));
}

constexpr int RATE_RING = 4;

// one CTA per SM; warp 0 issues iters x 4 MMAs with a commit (and, after the
// ring's first lap, a bounded wait) per four; the other warps only set up
template <int KIND>
__global__ void __launch_bounds__(128, 1) tc_rate_kernel(int N, int iters, long long *cycles) {
    extern __shared__ __align__(1024) uint8_t sm_raw[];
    uint8_t *base = sm_raw + ((1024u - (s32(sm_raw) & 1023u)) & 1023u);
    uint64_t *bar = reinterpret_cast<uint64_t *>(base + 49152);
    uint32_t *slot = reinterpret_cast<uint32_t *>(base + 49152 + 64);
    for (int i = threadIdx.x; i < 49152 / 4; i += blockDim.x) {       // +-1 levels of the kind
        uint32_t h = (uint32_t)i * 2654435761u ^ (blockIdx.x * 97u + 12345u);
        h ^= h >> 13;
        h *= 0x5bd1e995u;
        h ^= h >> 15;
        uint32_t v;
        if (KIND == 0) v = 0x38383838u | (h & 0x80808080u);
        else if (KIND == 1) v = 0x22222222u | (h & 0x88888888u);
        else v = 0x3F803F80u | (h & 0x80008000u);
        reinterpret_cast<uint32_t *>(base)[i] = v;
    }
    if (threadIdx.x == 0) {
        for (int r = 0; r <= RATE_RING; ++r) asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(s32(bar + r)));
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (threadIdx.x < 32) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;\n" ::"r"(s32(slot)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n");
    }
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    const uint32_t tmem = *slot;
    {   // unit scale factors (UE8M0 0x7F) in columns 448 .. 511
        const uint32_t w = threadIdx.x >> 5;
        for (int c = 448; c < 512; c += 4)
            asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1, %1, %1, %1};\n" ::"r"(tmem + ((w * 32) << 16) + c),
                         "r"(0x7F7F7F7Fu));
        asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    if (threadIdx.x < 32) {
        uint32_t id;
        if (KIND == 1)
            id = (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | (1u << 23) | ((128u >> 4) << 24);
        else
            id = (1u << 4) | ((KIND == 2 ? 1u : 0u) << 7) | ((KIND == 2 ? 1u : 0u) << 10) | ((uint32_t)(N >> 3) << 17) |
                 ((128u >> 4) << 24);
        const uint64_t ad = rdesc(s32(base)), bd = rdesc(s32(base + 16384));
        bool ok = true;
        const long long t0 = clock64();
        for (int i = 0; i < iters && ok; ++i) {
            if (i >= RATE_RING) ok = __all_sync(0xffffffffu, rwait(&bar[i % RATE_RING], (uint32_t)(((i / RATE_RING) - 1) & 1)));
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) rate_mma<KIND>(tmem, ad + 2 * kk, bd + 2 * kk, id, (i | kk) != 0, tmem + 448);
            asm volatile("{\n .reg .pred e;\n .reg .b32 r;\n elect.sync r|e, 0xffffffff;\n"
                         " @e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}\n" ::"r"(
                             s32(&bar[i % RATE_RING]))
                         : "memory");
        }
        asm volatile("{\n .reg .pred e;\n .reg .b32 r;\n elect.sync r|e, 0xffffffff;\n"
                     " @e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}\n" ::"r"(
                         s32(&bar[RATE_RING]))
                     : "memory");
        rwait(&bar[RATE_RING], 0u);
        for (int i = iters > RATE_RING ? iters - RATE_RING : 0; i < iters; ++i)
            rwait(&bar[i % RATE_RING], (uint32_t)((i / RATE_RING) & 1));
        if (threadIdx.x == 0) cycles[blockIdx.x] = clock64() - t0;
    }
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    if (threadIdx.x < 32) {
        asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;\n" ::"r"(tmem));
    }
}

// one thread per CTA loads iters 4D boxes {128 B, 32, 8, 1} (32 KB) through a
// ring of three buffers; cycles per box = the issue-to-issue time
__global__ void __launch_bounds__(32, 1) tma_rate_kernel(const __grid_constant__ CUtensorMap tm, int iters, int nb,
                                                         long long *cycles) {
    extern __shared__ __align__(1024) uint8_t sm_raw[];
    uint8_t *base = sm_raw + ((1024u - (s32(sm_raw) & 1023u)) & 1023u);
    constexpr int S = 3, BOX = 32768;
    uint64_t *bar = reinterpret_cast<uint64_t *>(base + S * BOX);
    if (threadIdx.x != 0) return;
    for (int s = 0; s < S; ++s) asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(s32(bar + s)));
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    const long long t0 = clock64();
    bool ok = true;
    int b = blockIdx.x % nb, y = 0;
    for (int i = 0; i < iters + S && ok; ++i) {
        const int s = i % S;
        if (i >= S) ok = rwait(&bar[s], (uint32_t)(((i / S) - 1) & 1));
        if (i < iters) {
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(s32(bar + s)), "r"(BOX) : "memory");
            asm volatile("cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
                         " [%0], [%1, {%2, %3, %4, %5}], [%6];\n" ::"r"(s32(base + (size_t)s * BOX)),
                         "l"(reinterpret_cast<uint64_t>(&tm)), "r"(0), "r"(0), "r"(y), "r"(b), "r"(s32(bar + s))
                         : "memory");
            y += 8;
            if (y == 32) {
                y = 0;
                b = (b + 152) % nb;
            }
        }
    }
    cycles[blockIdx.x] = clock64() - t0;
}

struct Timer {
    cudaEvent_t a = nullptr, b = nullptr;
    Timer() {
        cudaEventCreate(&a);
        cudaEventCreate(&b);
    }
    ~Timer() {
        cudaEventDestroy(a);
        cudaEventDestroy(b);
    }
};

double mean_cycles(const long long *dev, int n) {
    std::vector<long long> h((size_t)n);
    if (cudaMemcpy(h.data(), dev, sizeof(long long) * n, cudaMemcpyDeviceToHost) != cudaSuccess) return 0.0;
    double s = 0.0;
    for (long long v : h) s += (double)v;
    return s / n;
}

template <int KIND>
minw_status tc_rate(int sms, int N, long long *cyc, cudaStream_t st, double *flops, double *mhz) {
    const int smem = 120 * 1024, iters = 4000;
    if (cudaFuncSetAttribute(tc_rate_kernel<KIND>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
        return MINW_ECUDA;
    Timer t;
    float ms = 0.0f;
    for (int rep = 0; rep < 2; ++rep) {
        cudaEventRecord(t.a, st);
        tc_rate_kernel<KIND><<<sms, 128, smem, st>>>(N, iters, cyc);
        cudaEventRecord(t.b, st);
        if (cudaEventSynchronize(t.b) != cudaSuccess) return MINW_ECUDA;
    }
    cudaEventElapsedTime(&ms, t.a, t.b);
    const double kper = KIND == 0 ? 32.0 : KIND == 1 ? 64.0 : 16.0;
    *flops = 2.0 * 128 * N * kper * 4.0 * iters * sms / (ms * 1e-3);
    if (mhz) *mhz = mean_cycles(cyc, sms) / (ms * 1e3);
    return MINW_OK;
}

}  // namespace

extern "C" minw_status minw_measure_pipe_rates(minw_pipe_rates *out, void *stream) {
    if (!out) return MINW_EINVAL;
    *out = minw_pipe_rates{};
    cudaStream_t st = (cudaStream_t)stream;
    const int sms = minw_host::num_sms();
    if (sms <= 0) return MINW_ECUDA;
    const int threads = 256, blocks = sms * 8;
    uint32_t *buf = nullptr;
    long long *cyc = nullptr;
    uint8_t *tbuf = nullptr;
    const size_t tbytes = (size_t)64 * 32 * 32 * 128;      // 8 MB: L2-resident boxes
    if (cudaMalloc(&buf, sizeof(uint32_t) * blocks * threads) != cudaSuccess) return MINW_ECUDA;
    if (cudaMalloc(&cyc, sizeof(long long) * 1024) != cudaSuccess || cudaMalloc(&tbuf, tbytes) != cudaSuccess) {
        cudaFree(buf);
        cudaFree(cyc);
        return MINW_ECUDA;
    }
    minw_status rc = MINW_OK;
    do {
        Timer t;
        float ms = 0.0f;
        const int iters = 1 << 14;
        for (int rep = 0; rep < 2; ++rep) {
            cudaEventRecord(t.a, st);
            popc_rate_kernel<<<blocks, threads, 0, st>>>(buf, iters, 12345u + rep);
            cudaEventRecord(t.b, st);
            if (cudaEventSynchronize(t.b) != cudaSuccess) { rc = MINW_ECUDA; break; }
        }
        if (rc != MINW_OK) break;
        cudaEventElapsedTime(&ms, t.a, t.b);
        out->popc_per_s = 16.0 * iters * blocks * threads / (ms * 1e-3);
        for (int kind = 0; kind < 2; ++kind) {
            for (int rep = 0; rep < 2; ++rep) {
                cudaEventRecord(t.a, st);
                if (kind == 0)
                    warp_mma_rate_kernel<true><<<blocks, threads, 0, st>>>(buf, iters, 777u + rep);
                else
                    warp_mma_rate_kernel<false><<<blocks, threads, 0, st>>>(buf, iters, 999u + rep);
                cudaEventRecord(t.b, st);
                if (cudaEventSynchronize(t.b) != cudaSuccess) { rc = MINW_ECUDA; break; }
            }
            if (rc != MINW_OK) break;
            cudaEventElapsedTime(&ms, t.a, t.b);
            const double per = 4.0 * iters * (blocks * threads / 32) * 16.0 * 8.0;
            if (kind == 0) out->bmma_b1_mac_per_s = per * 256.0 / (ms * 1e-3);
            else out->imma_s8_mac_per_s = per * 32.0 / (ms * 1e-3);
        }
        if (rc != MINW_OK) break;
        const int Ns[2] = {128, 256};
        for (int j = 0; j < 2 && rc == MINW_OK; ++j) {
            double mhz = 0.0;
            if ((rc = tc_rate<0>(sms, Ns[j], cyc, st, &out->tc_e4m3_flop_per_s[j], &mhz)) != MINW_OK) break;
            if (j == 1) out->sm_clock_mhz = mhz;
            if ((rc = tc_rate<1>(sms, Ns[j], cyc, st, &out->tc_e2m1_flop_per_s[j], nullptr)) != MINW_OK) break;
            rc = tc_rate<2>(sms, Ns[j], cyc, st, &out->tc_bf16_flop_per_s[j], nullptr);
        }
        if (rc != MINW_OK) break;
        // TMA: 32 KB boxes of an 8 MB NHWC byte tensor [64][32][32][128]
        minw_host::EncodeTiledFn enc = minw_host::tensor_map_encoder();
        if (enc == nullptr) { rc = MINW_ECUDA; break; }
        cudaMemsetAsync(tbuf, 1, tbytes, st);
        CUtensorMap tm;
        const cuuint64_t dims[4] = {128, 32, 32, 64};
        const cuuint64_t strides[3] = {128, 32 * 128, 32 * 32 * 128};
        const cuuint32_t box[4] = {128, 32, 8, 1};
        const cuuint32_t es[4] = {1, 1, 1, 1};
        if (enc(&tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 4, tbuf, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
            rc = MINW_ECUDA;
            break;
        }
        const int smem = 3 * 32768 + 2048, biters = 2000;
        if (cudaFuncSetAttribute(tma_rate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess) {
            rc = MINW_ECUDA;
            break;
        }
        for (int rep = 0; rep < 2; ++rep) tma_rate_kernel<<<sms, 32, smem, st>>>(tm, biters, 64, cyc);
        if (cudaStreamSynchronize(st) != cudaSuccess) { rc = MINW_ECUDA; break; }
        out->tma_box_cycles = mean_cycles(cyc, sms) / biters;
        int to = 0;
        if (cudaMemcpyFromSymbol(&to, g_rate_timeout, sizeof(int)) != cudaSuccess) { rc = MINW_ECUDA; break; }
        if (to) rc = MINW_ETIMEOUT;
    } while (false);
    cudaFree(buf);
    cudaFree(cyc);
    cudaFree(tbuf);
    if (rc == MINW_OK && cudaGetLastError() != cudaSuccess) rc = MINW_ECUDA;
    return rc;
}
