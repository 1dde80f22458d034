// Integer-pipe and legacy-MMA throughput of the GPU: XOR + POPC + IADD (the
// popcount path's inner loop), mma.sync b1 (xor.popc) and mma.sync s8.  These
// figures set the "alu" roofline of the popcount convolution and decide
// against the legacy binary MMA.  Build and run:
//   nvcc -gencode arch=compute_103a,code=sm_103a -O3 -o pipe_rates pipe_rates.cu && ./pipe_rates
// Grid/threads fixed; every store index < nblocks*nthreads (buffer sized for it).
#include <cstdio>
#include <cstdint>
#include <cuda_runtime.h>

#define CK(x) do { cudaError_t e = (x); if (e != cudaSuccess) { printf("CUDA %s at %d\n", cudaGetErrorString(e), __LINE__); return 1; } } while (0)

__global__ void popc_kernel(uint32_t* out, int iters, uint32_t seed) {
    uint32_t a[4], w[4];
    int acc[16];
    #pragma unroll
    for (int i = 0; i < 4; ++i) { a[i] = seed * (threadIdx.x + 1) + i; w[i] = seed ^ (blockIdx.x * 977 + i * 31); }
    #pragma unroll
    for (int i = 0; i < 16; ++i) acc[i] = 0;
    for (int it = 0; it < iters; ++it) {
        #pragma unroll
        for (int i = 0; i < 4; ++i)
            #pragma unroll
            for (int j = 0; j < 4; ++j) acc[i * 4 + j] += __popc(a[i] ^ w[j]);
        #pragma unroll
        for (int i = 0; i < 4; ++i) { a[i] += 0x9E3779B9u; w[i] ^= a[i]; }
    }
    int s = 0;
    #pragma unroll
    for (int i = 0; i < 16; ++i) s += acc[i];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

__global__ void mma_b1_kernel(uint32_t* out, int iters, uint32_t seed) {
    uint32_t a0 = seed * threadIdx.x, a1 = a0 ^ 0x55, a2 = a0 + 7, a3 = a0 * 3;
    uint32_t b0 = seed ^ threadIdx.x, b1 = b0 + 11;
    int c[4][4];
    #pragma unroll
    for (int k = 0; k < 4; ++k) for (int i = 0; i < 4; ++i) c[k][i] = 0;
    for (int it = 0; it < iters; ++it) {
        #pragma unroll
        for (int k = 0; k < 4; ++k) {
            asm volatile("mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.xor.popc "
                         "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
                         : "+r"(c[k][0]), "+r"(c[k][1]), "+r"(c[k][2]), "+r"(c[k][3])
                         : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
        }
    }
    int s = 0;
    for (int k = 0; k < 4; ++k) for (int i = 0; i < 4; ++i) s += c[k][i];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

__global__ void mma_s8_kernel(uint32_t* out, int iters, uint32_t seed) {
    uint32_t a0 = seed * threadIdx.x, a1 = a0 ^ 0x55, a2 = a0 + 7, a3 = a0 * 3;
    uint32_t b0 = seed ^ threadIdx.x, b1 = b0 + 11;
    int c[4][4];
    #pragma unroll
    for (int k = 0; k < 4; ++k) for (int i = 0; i < 4; ++i) c[k][i] = 0;
    for (int it = 0; it < iters; ++it) {
        #pragma unroll
        for (int k = 0; k < 4; ++k) {
            asm volatile("mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 "
                         "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
                         : "+r"(c[k][0]), "+r"(c[k][1]), "+r"(c[k][2]), "+r"(c[k][3])
                         : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
        }
    }
    int s = 0;
    for (int k = 0; k < 4; ++k) for (int i = 0; i < 4; ++i) s += c[k][i];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

__global__ void clock_kernel(long long* out, int iters) {
    long long t0 = clock64();
    uint32_t x = threadIdx.x;
    for (int i = 0; i < iters; ++i) x = x * 1664525u + 1013904223u;
    long long t1 = clock64();
    if (threadIdx.x == 0) out[blockIdx.x] = t1 - t0 + (x == 12345 ? 1 : 0);
}

int main() {
    int dev = 0; cudaDeviceProp p; CK(cudaGetDeviceProperties(&p, dev));
    int sms = p.multiProcessorCount;
    printf("{\"gpu\": \"%s\", \"sms\": %d, \"cc\": \"%d.%d\"}\n", p.name, sms, p.major, p.minor);
    const int threads = 256;
    const int blocks = sms * 8;
    uint32_t* out; CK(cudaMalloc(&out, sizeof(uint32_t) * blocks * threads));
    long long* clk; CK(cudaMalloc(&clk, sizeof(long long) * blocks));
    cudaEvent_t e0, e1; cudaEventCreate(&e0); cudaEventCreate(&e1);
    float ms;
    // clock rate estimate
    for (int rep = 0; rep < 2; ++rep) {
        int iters = 1 << 22;
        cudaEventRecord(e0); clock_kernel<<<sms, 32>>>(clk, iters); cudaEventRecord(e1); CK(cudaEventSynchronize(e1));
        cudaEventElapsedTime(&ms, e0, e1);
        long long c0; CK(cudaMemcpy(&c0, clk, sizeof(long long), cudaMemcpyDeviceToHost));
        printf("{\"probe\": \"clock\", \"cycles\": %lld, \"ms\": %.3f, \"mhz\": %.1f}\n", c0, ms, c0 / (ms * 1e3));
    }
    for (int rep = 0; rep < 3; ++rep) {
        int iters = 1 << 14;
        cudaEventRecord(e0); popc_kernel<<<blocks, threads>>>(out, iters, 12345u + rep); cudaEventRecord(e1); CK(cudaEventSynchronize(e1));
        cudaEventElapsedTime(&ms, e0, e1);
        double popcs = 16.0 * iters * blocks * threads;
        printf("{\"probe\": \"xor_popc_add\", \"ms\": %.3f, \"popc_per_s\": %.4e, \"bin_mac_per_s\": %.4e}\n", ms, popcs / (ms * 1e-3), 32 * popcs / (ms * 1e-3));
    }
    for (int rep = 0; rep < 3; ++rep) {
        int iters = 1 << 14;
        cudaEventRecord(e0); mma_b1_kernel<<<blocks, threads>>>(out, iters, 777u + rep); cudaEventRecord(e1); CK(cudaEventSynchronize(e1));
        cudaEventElapsedTime(&ms, e0, e1);
        double macs = 4.0 * iters * (blocks * threads / 32) * 16.0 * 8.0 * 256.0;
        printf("{\"probe\": \"mma_b1_xor\", \"ms\": %.3f, \"bin_mac_per_s\": %.4e}\n", ms, macs / (ms * 1e-3));
    }
    for (int rep = 0; rep < 3; ++rep) {
        int iters = 1 << 14;
        cudaEventRecord(e0); mma_s8_kernel<<<blocks, threads>>>(out, iters, 999u + rep); cudaEventRecord(e1); CK(cudaEventSynchronize(e1));
        cudaEventElapsedTime(&ms, e0, e1);
        double macs = 4.0 * iters * (blocks * threads / 32) * 16.0 * 8.0 * 32.0;
        printf("{\"probe\": \"mma_s8\", \"ms\": %.3f, \"mac_per_s\": %.4e}\n", ms, macs / (ms * 1e-3));
    }
    CK(cudaDeviceSynchronize());
    cudaFree(out); cudaFree(clk);
    return 0;
}
