// runtime.cu -- process-wide plan options of the library and the test hook
// of the bounded-wait timeout path.
//
// The plan options pick between kernel variants that compute the same result
// (CTA pairs, channel-major tiles, the 64-channel weight duplication, K blocks
// per pipeline stage, TMA first-layer patches, the tensor-core first layer,
// programmatic dependent launch,
// graph replay of a network forward) and set the limit of every bounded wait.
// The defaults are the measured fastest choices; they are read when a launch
// is planned, so a change applies to standalone calls made after it and to
// networks created after it.  Tests turn each option off to check that every
// variant gives the same bits.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>
#include <unordered_set>

#include "kernels.cuh"

namespace {

minw_plan_options defaults() {
    minw_plan_options o;
    o.cta_pairs = 1;
    o.channel_major = 1;
    o.channel_major_min_tiles_per_sm = 2;
    o.dup_weights = 1;
    o.kblocks_per_stage = 2;
    o.first_tma = 1;
    o.pdl = 1;
    o.graph = 1;
    o.tma_lanes = 1;
    o.resident_weights = 0;
    o.first_tensor_cores = 1;
    o.wait_cycles = (int64_t)1 << 31;
    return o;
}

std::mutex g_mu;
minw_plan_options g_opt = defaults();
std::atomic<int> g_stall{0};

}  // namespace

namespace minw_host {

minw_plan_options plan_options() {
    std::lock_guard<std::mutex> lock(g_mu);
    return g_opt;
}

bool pdl_enabled() { return plan_options().pdl != 0; }

int take_stall(int which) {
    int expected = which;
    return g_stall.compare_exchange_strong(expected, 0) ? 1 : 0;
}

void max_shared_carveout(const void *kern) {
    static std::mutex mu;
    static std::unordered_set<const void *> done;
    std::lock_guard<std::mutex> lock(mu);
    if (done.insert(kern).second)
        cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
}

}  // namespace minw_host

extern "C" {

minw_status minw_get_plan_options(minw_plan_options *out) {
    if (!out) return MINW_EINVAL;
    *out = minw_host::plan_options();
    return MINW_OK;
}

minw_status minw_set_plan_options(const minw_plan_options *opt) {
    minw_plan_options o = opt ? *opt : defaults();
    if (o.kblocks_per_stage != 1 && o.kblocks_per_stage != 2) return MINW_EINVAL;
    if (o.channel_major_min_tiles_per_sm < 0 || o.wait_cycles <= 0 || o.tma_lanes < 1 || o.tma_lanes > 8)
        return MINW_EINVAL;
    std::lock_guard<std::mutex> lock(g_mu);
    g_opt = o;
    return MINW_OK;
}

minw_status minw_test_stall_next_launch(int32_t kernel) {
    if (kernel != 0 && kernel != MINW_STALL_CONV_TC && kernel != MINW_STALL_CONV_FIRST) return MINW_EINVAL;
    g_stall.store(kernel);
    return MINW_OK;
}

}  // extern "C"
