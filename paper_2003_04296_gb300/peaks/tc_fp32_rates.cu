// Issue rate of tcgen05.mma kind::f8f6f4 from one thread (M = 128, N = 64,
// 128, 256; with and without a commit + wait per four MMAs) and the FP32 FMA
// rate of scalar fmaf and packed fma.rn.f32x2.  These figures explain the
// tensor-core kernel's tile shape (N = 256 reaches the peak; each MMA costs
// the issuing thread about a hundred cycles) and set the FP32 roofline of the
// first layer.  Build and run:
//   nvcc -gencode arch=compute_103a,code=sm_103a -O3 -o tc_fp32_rates tc_fp32_rates.cu && ./tc_fp32_rates
// One CTA per SM (120 KB of shared memory); operands are fixed random FP8
// level codes in shared memory; every wait is bounded.
#include <cstdio>
#include <cstdint>
#include <cuda_runtime.h>

#define CK(x) do { cudaError_t e = (x); if (e != cudaSuccess) { printf("CUDA %s at %d\n", cudaGetErrorString(e), __LINE__); return 1; } } while (0)

__device__ int g_timeout = 0;

__device__ __forceinline__ uint32_t saddr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

// K-major operand, rows of 128 bytes, 128-byte swizzle, 8-row groups 1024 bytes apart
__device__ __forceinline__ uint64_t sdesc(uint32_t a) {
    return (uint64_t)((a & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

__device__ __forceinline__ bool wait_phase(uint64_t *bar, uint32_t parity) {
    const long long t0 = clock64();
    while (true) {
        uint32_t ok;
        asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
                     : "=r"(ok) : "r"(saddr(bar)), "r"(parity) : "memory");
        if (ok) return true;
        if (clock64() - t0 > (1ll << 31)) { atomicExch(&g_timeout, 1); return false; }
    }
}

constexpr int RING = 4;

__global__ void __launch_bounds__(128, 1) mma_rate(int N, int iters, int ring, long long *cycles) {
    extern __shared__ __align__(1024) uint8_t sm[];
    uint8_t *base = sm + ((1024u - (saddr(sm) & 1023u)) & 1023u);
    uint64_t *bar = reinterpret_cast<uint64_t *>(base + 49152);          // [RING + 1]
    uint32_t *slot = reinterpret_cast<uint32_t *>(base + 49152 + 64);
    for (int i = threadIdx.x; i < 49152 / 4; i += blockDim.x) {          // random +-1 levels
        uint32_t h = (uint32_t)i * 2654435761u ^ (blockIdx.x * 97u + 12345u);
        h ^= h >> 13; h *= 0x5bd1e995u; h ^= h >> 15;
        reinterpret_cast<uint32_t *>(base)[i] = 0x38383838u | (h & 0x80808080u);
    }
    if (threadIdx.x == 0) {
        for (int r = 0; r <= RING; ++r) asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(saddr(bar + r)));
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (threadIdx.x < 32) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 256;\n" ::"r"(saddr(slot)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n");
    }
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    const uint32_t tmem = *slot;
    if (threadIdx.x == 0) {
        const uint32_t id = (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((128u >> 4) << 24);   // E4M3 x E4M3 -> f32
        const uint64_t ad = sdesc(saddr(base)), bd = sdesc(saddr(base + 16384));
        bool ok = true;
        const long long t0 = clock64();
        for (int i = 0; i < iters && ok; ++i) {
            if (ring && i >= RING) ok = wait_phase(&bar[i % RING], (uint32_t)(((i / RING) - 1) & 1));
            for (int kk = 0; kk < 4; ++kk) {
                const uint32_t acc = (i | kk) != 0;
                asm volatile("{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                             " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem),
                             "l"(ad + 2 * kk), "l"(bd + 2 * kk), "r"(id), "r"(acc));
            }
            if (ring)
                asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                                 saddr(bar + i % RING)) : "memory");
        }
        asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                         saddr(bar + RING)) : "memory");
        wait_phase(&bar[RING], 0u);
        if (ring)     // every ring commit has arrived before the CTA leaves
            for (int i = iters > RING ? iters - RING : 0; i < iters; ++i) wait_phase(&bar[i % RING], (uint32_t)((i / RING) & 1));
        cycles[blockIdx.x] = clock64() - t0;
    }
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    if (threadIdx.x < 32) {
        asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 256;\n" ::"r"(tmem));
    }
}

__global__ void ffma_rate(float *out, int iters) {
    float a[16];
    for (int i = 0; i < 16; ++i) a[i] = threadIdx.x * 1e-3f + i;
    const float b = 1.0000001f, c = 1e-7f;
    for (int it = 0; it < iters; ++it)
#pragma unroll
        for (int i = 0; i < 16; ++i) a[i] = fmaf(a[i], b, c);
    float s = 0.0f;
    for (int i = 0; i < 16; ++i) s += a[i];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

__global__ void ffma2_rate(float *out, int iters) {
    unsigned long long a[8], b, c;
    for (int i = 0; i < 8; ++i) { const float x = threadIdx.x * 1e-3f + i; asm("mov.b64 %0, {%1, %1};" : "=l"(a[i]) : "f"(x)); }
    { const float x = 1.0000001f, y = 1e-7f; asm("mov.b64 %0, {%1, %1};" : "=l"(b) : "f"(x)); asm("mov.b64 %0, {%1, %1};" : "=l"(c) : "f"(y)); }
    for (int it = 0; it < iters; ++it)
#pragma unroll
        for (int i = 0; i < 8; ++i) asm volatile("fma.rn.f32x2 %0, %0, %1, %2;" : "+l"(a[i]) : "l"(b), "l"(c));
    float s = 0.0f;
    for (int i = 0; i < 8; ++i) { float lo, hi; asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(a[i])); s += lo + hi; }
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

int main() {
    int sms = 0, clk_khz = 0;
    CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0));
    CK(cudaDeviceGetAttribute(&clk_khz, cudaDevAttrClockRate, 0));
    long long *cyc;
    CK(cudaMalloc(&cyc, sms * sizeof(long long)));
    const int smem = 120 * 1024;
    CK(cudaFuncSetAttribute(mma_rate, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    printf("%d SMs\n", sms);
    for (int N : {64, 128, 256})
        for (int ring : {0, 1}) {
            const int iters = 4000;
            cudaEvent_t e0, e1;
            CK(cudaEventCreate(&e0)); CK(cudaEventCreate(&e1));
            for (int rep = 0; rep < 2; ++rep) {
                CK(cudaEventRecord(e0));
                mma_rate<<<sms, 128, smem>>>(N, iters, ring, cyc);
                CK(cudaEventRecord(e1));
                CK(cudaEventSynchronize(e1));
            }
            float ms; CK(cudaEventElapsedTime(&ms, e0, e1));
            long long h[1024]; CK(cudaMemcpy(h, cyc, sms * sizeof(long long), cudaMemcpyDeviceToHost));
            double c = 0; for (int b = 0; b < sms; ++b) c += h[b]; c /= sms;
            const double flop = 2.0 * 128 * N * 128 * (double)iters * sms;
            printf("tcgen05 f8f6f4 M=128 N=%3d %s: %6.1f cycles per MMA, %6.0f TFLOP/s\n", N,
                   ring ? "commit+wait per 4" : "no commit         ", c / iters / 4, flop / (ms * 1e-3) / 1e12);
        }
    float *d;
    CK(cudaMalloc(&d, (size_t)sms * 2 * 1024 * sizeof(float)));
    for (int kind = 0; kind < 2; ++kind) {
        const int iters = 20000, bs = 1024;
        cudaEvent_t e0, e1;
        CK(cudaEventCreate(&e0)); CK(cudaEventCreate(&e1));
        for (int rep = 0; rep < 2; ++rep) {
            CK(cudaEventRecord(e0));
            if (kind == 0) ffma_rate<<<sms * 2, bs>>>(d, iters); else ffma2_rate<<<sms * 2, bs>>>(d, iters);
            CK(cudaEventRecord(e1));
            CK(cudaEventSynchronize(e1));
        }
        float ms; CK(cudaEventElapsedTime(&ms, e0, e1));
        const double fma = (double)sms * 2 * bs * 16.0 * iters;
        printf("%s: %.1f TFMA/s = %.1f FMA/clk/SM at %.0f MHz\n", kind ? "fma.rn.f32x2" : "fmaf        ",
               fma / (ms * 1e-3) / 1e12, fma / (ms * 1e-3) / sms / (clk_khz * 1e3), clk_khz / 1e3);
    }
    int to = 0;
    CK(cudaMemcpyFromSymbol(&to, g_timeout, sizeof(int)));
    printf("bounded waits timed out: %d\n", to);
    return 0;
}
