// conv_tc.cu -- tensor-core path of the quantized convolution (tcgen05).
// Placeholder until the kernel lands: no shape is covered yet, so the
// per-shape choice always takes the popcount path.
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace minw {

// Device error flag: set by a bounded wait that gave up.
__device__ int g_device_error = 0;

bool conv_tc_supported(const ConvArgs &) { return false; }

minw_status launch_conv_tc(const ConvArgs &, cudaStream_t) { return MINW_EUNSUPPORTED; }

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
