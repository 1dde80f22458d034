// fc_noalloc.cu -- minw_fc_codes for callers that cannot allocate device
// memory.
//
// Some callers have no way to obtain device memory for scratch: a plugin run
// by a host framework that owns all device memory and passes in only the
// tensors of the call, or a service that reserves its memory at start-up and
// forbids allocations afterwards (cudaMalloc may also synchronise the
// device, which such a caller cannot accept).  For them the split-K scratch
// of the fully connected layer lives in a fixed array inside the library.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds MINW_FC_NOALLOC_SCRATCH_BYTES of it until the process exits.
// Host code cannot hand the array's name to a kernel (in host code the name
// is only a host-side stand-in for the device symbol), so the first call on
// each device asks the runtime for the array's device address with
// cudaGetSymbolAddress, with that device current, and caches it.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "kernels.cuh"

using namespace minw;
using namespace minw_host;

namespace {

__device__ __align__(256) uint8_t g_fc_scratch[MINW_FC_NOALLOC_SCRATCH_BYTES];

constexpr int MAX_DEVICES = 64;
void *g_scratch_addr[MAX_DEVICES] = {};
std::mutex g_scratch_mu;

// Device address of the scratch array on the current device (looked up once
// per device).
minw_status scratch_address(void **out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return MINW_ECUDA;
    if (dev < 0 || dev >= MAX_DEVICES) return MINW_EDEVICE;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (g_scratch_addr[dev] == nullptr) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_fc_scratch) != cudaSuccess || ptr == nullptr) return MINW_ECUDA;
        g_scratch_addr[dev] = ptr;
    }
    *out = g_scratch_addr[dev];
    return MINW_OK;
}

}  // namespace

extern "C" minw_status minw_fc_codes_noalloc(const uint8_t *act, int32_t B, int32_t K, int32_t bits_a,
                                             const uint8_t *wgt, int32_t O, int32_t bits_w, const float *scale,
                                             const float *shift, const minw_quant *q_out, uint8_t *codes_out,
                                             uint32_t *planes_out, float *y_out, int32_t *acc_out, void *stream) {
    if (B <= 0 || K <= 0 || O <= 0) return MINW_EINVAL;
    if (K % 128 != 0) return MINW_EUNSUPPORTED;
    // the smallest split this shape would use must fit in the fixed array
    ConvArgs a{};
    a.B = B; a.C = K; a.H = 1; a.W = 1; a.O = O; a.kh = 1; a.kw = 1; a.stride = 1; a.pad = 0;
    a.Ho = 1; a.Wo = 1; a.NW = K / 32; a.M = B;
    if (conv_tc_min_split_bytes(a) > (size_t)MINW_FC_NOALLOC_SCRATCH_BYTES) return MINW_EUNSUPPORTED;
    void *scratch = nullptr;
    const minw_status st = scratch_address(&scratch);
    if (st != MINW_OK) return st;
    return minw_fc_codes(act, B, K, bits_a, wgt, O, bits_w, scale, shift, q_out, codes_out, planes_out, y_out,
                         acc_out, scratch, (size_t)MINW_FC_NOALLOC_SCRATCH_BYTES, stream);
}
