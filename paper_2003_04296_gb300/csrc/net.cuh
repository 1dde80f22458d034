// net.cuh -- the network object shared by the sequential builder (net.cu)
// and the residual builder (resnet.cu).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "kernels.cuh"

struct LayerPlan {
    minw_layer_desc d;        // shape fields only; pointers are not kept
    int C, H, W, O, kh, kw, stride, pad, pool;
    int Ho, Wo, Hp, Wp;
    uint32_t *wplanes = nullptr;   // packed weights (popcount layers)
    uint8_t *wcodes = nullptr;     // weight codes (tensor-core layers)
    float *thr = nullptr;          // output-quantizer breakpoints (first layer: fp32 [O][8];
                                   // tensor-core layers: integer-valued [O][levels])
    int in_codes = 0;              // input arrives in the codes layout
    int in4 = 0;                   // ... as E2M1 codes (two channels per byte; weights too)
    int pair128 = 0;               // E2M1 tensor-core layer as CTA pairs of 128-channel tiles (measured choice)
    int n128 = 0;                  // E2M1 tensor-core layer on single-CTA 128-channel tiles (measured choice)
    float cand_ms[5] = {-1.0f, -1.0f, -1.0f, -1.0f, -1.0f};   // creation-time times of the candidates
                                   // (MINW_VARIANT_AUTO): E4M3, E2M1, E2M1 pairs, popcount, E2M1 128-channel
                                   // tiles; -1 where not a candidate
    float *wlatent = nullptr;      // fp32 weights (first layer)
    float *wt = nullptr;           // first layer: weights prepared as [K][O] levels
    float *wscale = nullptr;       // per-channel weight prescale (first layer)
    float *scale = nullptr;
    float *shift = nullptr;
    minw_quant qw{}, qo{};
    int variant = MINW_VARIANT_POPC;
};

struct ResNetPlan;   // resnet.cu
struct WResPlan;     // wonly_nets.cu
struct WDensePlan;   // wonly_nets.cu

struct minw_net {
    int kind = 0;                     // 0: sequential (minw_net_create), 1: residual (minw_resnet18_create),
                                      // 2: weight-only residual (minw_wresnet_create),
                                      // 3: weight-only DenseNet-BC (minw_wdense_create)
    ResNetPlan *res = nullptr;
    WResPlan *wres = nullptr;
    WDensePlan *wdense = nullptr;
    std::vector<LayerPlan> L;
    int max_batch = 0;
    uint32_t *buf[2] = {nullptr, nullptr};
    size_t buf_words = 0;
    std::vector<void *> owned;
    float *x_stage = nullptr;         // device staging of minw_forward_host
    float *logits_stage = nullptr;
    size_t x_elems = 0, logit_elems = 0;
    void *ws = nullptr;               // split-K workspace shared by the layers
    size_t ws_bytes = 0;
    std::vector<cudaEvent_t> events;  // [0] before the first layer, [l+1] after layer l
    bool timing = false;
    // the forward captured once as a CUDA graph (per input, logits and batch) and replayed
    cudaStream_t cap_stream = nullptr;
    cudaGraphExec_t gexec = nullptr;
    const float *gx = nullptr;
    float *glogits = nullptr;
    int gB = 0;
};


// Enqueue the residual network's forward (resnet.cu).
minw_status resnet_forward(minw_net *net, const float *x, int B, float *logits, cudaStream_t s);
int32_t resnet_ops(const minw_net *net);
void resnet_variants(const minw_net *net, int32_t *variants);
int32_t resnet_kernels(const minw_net *net);
void resnet_free(minw_net *net);

// The weight-only residual network (wonly_nets.cu).
minw_status wresnet_forward(minw_net *net, const float *x, int B, float *logits, cudaStream_t s);
int32_t wresnet_ops(const minw_net *net);
void wresnet_variants(const minw_net *net, int32_t *variants);
int32_t wresnet_kernels(const minw_net *net);
void wresnet_free(minw_net *net);

// The weight-only DenseNet-BC (wonly_nets.cu).
minw_status wdense_forward(minw_net *net, const float *x, int B, float *logits, cudaStream_t s);
int32_t wdense_ops(const minw_net *net);
void wdense_variants(const minw_net *net, int32_t *variants);
int32_t wdense_kernels(const minw_net *net);
void wdense_free(minw_net *net);
