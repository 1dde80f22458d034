// net.cu -- whole-network forward of a sequential MINW-Net (Algorithm 1,
// inference branch, with the layer constructs of Sec. III-E).
//
// minw_net_create packs every quantized weight tensor once (W^ = h(W)),
// copies the BN affine maps, plans one kernel per layer and allocates two
// ping-pong activation buffers holding packed planes.  minw_forward then
// enqueues one kernel per layer: the fp32 first layer, then quantized
// convolution blocks whose epilogues write the next layer's packed input, and
// a last layer that writes fp32 logits.  Fully connected layers run as
// convolutions whose kernel covers the whole input map (flatten order
// (c, h, w) = OIHW weight order).
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdlib.h>

#include <algorithm>
#include <vector>

#include "net.cuh"

using namespace minw;
using namespace minw_host;

static void net_free(minw_net *n) {
    if (!n) return;
    if (n->res) resnet_free(n);
    if (n->wres) wresnet_free(n);
    if (n->wdense) wdense_free(n);
    for (void *p : n->owned) cudaFree(p);
    for (cudaEvent_t e : n->events) cudaEventDestroy(e);
    if (n->gexec) cudaGraphExecDestroy(n->gexec);
    if (n->cap_stream) cudaStreamDestroy(n->cap_stream);
    delete n;
}

template <typename T>
static minw_status net_alloc(minw_net *n, T **p, size_t count) {
    void *q = nullptr;
    if (cudaMalloc(&q, count * sizeof(T) + 16) != cudaSuccess) return MINW_ECUDA;
    n->owned.push_back(q);
    *p = reinterpret_cast<T *>(q);
    return MINW_OK;
}

// Time one convolution launch on either path: one warm-up, then the least of
// three runs (ms).
static minw_status time_conv(const ConvArgs &a, bool popc, cudaStream_t s, cudaEvent_t e0, cudaEvent_t e1,
                             float *ms) {
    minw_status st = popc ? launch_conv_popc(a, s) : launch_conv_tc(a, s);
    if (st != MINW_OK) return st;
    float best = 1e30f;
    for (int r = 0; r < 3; ++r) {
        if (cudaEventRecord(e0, s) != cudaSuccess) return MINW_ECUDA;
        if ((st = popc ? launch_conv_popc(a, s) : launch_conv_tc(a, s)) != MINW_OK) return st;
        if (cudaEventRecord(e1, s) != cudaSuccess || cudaEventSynchronize(e1) != cudaSuccess) return MINW_ECUDA;
        float t = 0.0f;
        cudaEventElapsedTime(&t, e0, e1);
        if (t < best) best = t;
    }
    *ms = best;
    return MINW_OK;
}

// The measured choice of kernel, operands and tiling for every layer the
// tensor cores cover: E4M3 operands, E2M1 operands, E2M1 as CTA pairs of
// 128-channel tiles, or bit-planes on the popcount path (pipe rates alone do
// not decide: the layer's tiling, its accumulator count and its epilogue do;
// on GB300 E2M1 wins on most layers but not on all).  Each candidate runs on
// the layer's shape at the net's batch with its own weight codes or planes,
// breakpoints and split workspace, into scratch buffers; the fastest is kept
// (P.variant, P.in4, P.pair128), every candidate's time is kept in P.cand_ms,
// and the shared workspace is sized for the choices.
static minw_status tune_formats(minw_net *n, const minw_layer_desc *layers, int n_layers, int max_batch,
                                cudaStream_t s) {
    size_t in_b = 0, out_b = 0, w_b = 0, ws_b = 0;
    std::vector<int> cand;
    for (int l = 1; l < n_layers; ++l) {
        const LayerPlan &P = n->L[l];
        if (P.variant != MINW_VARIANT_TC || layers[l].variant != 0) continue;
        cand.push_back(l);
        // codes (one byte per channel at most) or bit-planes (3 bits per channel at most) in;
        // codes, planes or fp32 logits out
        in_b = std::max(in_b, (size_t)max_batch * P.H * P.W * P.C);
        out_b = std::max(out_b, (size_t)max_batch * P.Hp * P.Wp * P.O * sizeof(float));
        w_b = std::max(w_b, (size_t)P.O * P.kh * P.kw * P.C);
    }
    if (cand.empty()) return MINW_OK;
    std::vector<void *> tmp;
    auto talloc = [&](size_t bytes, void **p) -> minw_status {
        if (cudaMalloc(p, bytes + 256) != cudaSuccess) return MINW_ECUDA;
        tmp.push_back(*p);
        return MINW_OK;
    };
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    minw_status st = MINW_OK;
    void *xin = nullptr, *yout = nullptr, *w8 = nullptr, *w4 = nullptr, *thr = nullptr, *ws = nullptr;
    void *wpl = nullptr;
    do {
        if (cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) { st = MINW_ECUDA; break; }
        if ((st = talloc(in_b, &xin)) != MINW_OK || (st = talloc(out_b, &yout)) != MINW_OK ||
            (st = talloc(w_b, &w8)) != MINW_OK || (st = talloc(w_b, &w4)) != MINW_OK ||
            (st = talloc(w_b, &wpl)) != MINW_OK || (st = talloc(4096 * 8 * sizeof(float), &thr)) != MINW_OK)
            break;
        // +1 levels in both formats (E4M3 0x38; E2M1 0x2 in each nibble)
        if (cudaMemsetAsync(xin, 0x22, in_b, s) != cudaSuccess) { st = MINW_ECUDA; break; }
        for (int l : cand) {
            LayerPlan &P = n->L[l];
            const minw_layer_desc &d = layers[l];
            const bool last = l == n_layers - 1;
            ConvArgs a{};
            a.B = max_batch; a.C = P.C; a.H = P.H; a.W = P.W; a.O = P.O; a.kh = P.kh; a.kw = P.kw;
            a.stride = P.stride; a.pad = P.pad; a.Ho = P.Ho; a.Wo = P.Wo; a.NW = P.C / 32;
            a.bits_a = d.bits_in; a.bits_w = d.bits_w;
            a.M = (long long)max_batch * P.Ho * P.Wo;
            a.scale = P.scale; a.shift = P.shift; a.pool = P.pool;
            a.quant_out = !last;
            if (!last) {
                a.qo = to_qparams(&P.qo);
                if (P.O > 4096) { st = MINW_EUNSUPPORTED; break; }
                if ((st = launch_thresholds(P.scale, P.shift, P.O, a.qo, (float *)thr, s)) != MINW_OK) break;
                a.thr = (const float *)thr;
                a.codes_out = (uint8_t *)yout;
            } else {
                a.y_out = (float *)yout;
            }
            // candidates: E4M3 operands, E2M1 operands, E2M1 as CTA pairs of 128-channel tiles,
            // bit-planes on the popcount path (its input: the same bytes read as planes; its
            // output: planes, or the fp32 logits of the last layer)
            float t[5] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
            for (int f = 0; f < 5 && st == MINW_OK; ++f) {
                if (f == 3) {
                    ConvArgs b = a;
                    b.thr = nullptr;
                    b.codes_out = nullptr;
                    if (!last) b.planes_out = (uint32_t *)yout;
                    if ((st = minw_pack_weights(d.w, P.O, P.C, P.kh, P.kw, &P.qw, d.w_scale, (uint32_t *)wpl, s)) !=
                        MINW_OK)
                        break;
                    b.act = (const uint32_t *)xin;
                    b.wgt = (const uint32_t *)wpl;
                    st = time_conv(b, true, s, e0, e1, &t[f]);
                    continue;
                }
                ConvArgs b = a;
                b.fp4 = f ? 1 : 0;
                b.pair_n128 = f == 2 ? 1 : 0;
                b.n128 = f == 4 ? 1 : 0;
                b.codes_out4 = f && !last;
                if (!conv_tc_supported(b)) { t[f] = 1e30f; continue; }
                // the tiling the layer would run with: at run time it gets the net's split workspace
                // (a layer that splits along K runs no CTA pairs); planning only reads the size
                {
                    ConvArgs c = b;
                    const size_t wsn = conv_tc_workspace_bytes(c);
                    c.workspace = wsn ? reinterpret_cast<void *>(256) : nullptr;
                    c.workspace_bytes = wsn;
                    if ((f == 2 && !conv_tc_pairs128(c)) || (f == 4 && !conv_tc_n128(c))) { t[f] = 1e30f; continue; }
                }
                void *wq = f ? w4 : w8;
                if (f < 2)
                    st = f ? minw_pack_weight_codes_e2m1(d.w, P.O, P.C, P.kh, P.kw, &P.qw, d.w_scale, (uint8_t *)wq, s)
                           : minw_pack_weight_codes(d.w, P.O, P.C, P.kh, P.kw, &P.qw, d.w_scale, (uint8_t *)wq, s);
                if (st != MINW_OK) break;
                b.act8 = (const uint8_t *)xin;
                b.wgt8 = (const uint8_t *)wq;
                const size_t need = conv_tc_workspace_bytes(b);
                if (need > ws_b) {
                    if (ws) { cudaStreamSynchronize(s); cudaFree(ws); tmp.erase(std::find(tmp.begin(), tmp.end(), ws)); ws = nullptr; }
                    if ((st = talloc(need, &ws)) != MINW_OK) break;
                    if (cudaMemsetAsync(ws, 0, need, s) != cudaSuccess) { st = MINW_ECUDA; break; }
                    ws_b = need;
                }
                b.workspace = ws;
                b.workspace_bytes = ws_b;
                st = time_conv(b, false, s, e0, e1, &t[f]);
            }
            if (st != MINW_OK) break;
            int best = 0;
            for (int f = 1; f < 5; ++f)
                if (t[f] < t[best]) best = f;
            for (int f = 0; f < 5; ++f) P.cand_ms[f] = t[f] < 1e29f ? t[f] : -1.0f;
            P.variant = best == 3 ? MINW_VARIANT_POPC : MINW_VARIANT_TC;
            P.in4 = (best == 1 || best == 2 || best == 4) ? 1 : 0;
            P.pair128 = best == 2 ? 1 : 0;
            P.n128 = best == 4 ? 1 : 0;
        }
    } while (false);
    cudaStreamSynchronize(s);
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    for (void *p : tmp) cudaFree(p);
    if (st != MINW_OK) return st;
    // the shared split workspace, for the chosen formats
    n->ws_bytes = 0;
    for (int l = 1; l < n_layers; ++l) {
        const LayerPlan &P = n->L[l];
        if (P.variant != MINW_VARIANT_TC) continue;
        ConvArgs a{};
        a.B = max_batch; a.C = P.C; a.H = P.H; a.W = P.W; a.O = P.O; a.kh = P.kh; a.kw = P.kw;
        a.stride = P.stride; a.pad = P.pad; a.Ho = P.Ho; a.Wo = P.Wo; a.NW = P.C / 32;
        a.M = (long long)max_batch * P.Ho * P.Wo; a.pool = P.pool; a.quant_out = l + 1 < n_layers;
        a.fp4 = P.in4;
        a.pair_n128 = P.pair128;
        a.n128 = P.n128;
        n->ws_bytes = std::max(n->ws_bytes, conv_tc_workspace_bytes(a));
    }
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

extern "C" {

minw_status minw_net_create(const minw_layer_desc *layers, int32_t n_layers, int32_t max_batch,
                            int32_t variant, void *stream, minw_net **out) {
    if (!layers || n_layers < 2 || max_batch <= 0 || !out) return MINW_EINVAL;
    if (variant < 0 || variant > MINW_VARIANT_TC_E2M1_N128) return MINW_EINVAL;
    *out = nullptr;
    cudaStream_t s = (cudaStream_t)stream;
    minw_net *n = new minw_net();
    n->max_batch = max_batch;
    int pc = 0, ph = 0, pw = 0, pbits = 0;     // previous output shape and bits
    size_t max_words = 0;
    for (int l = 0; l < n_layers; ++l) {
        const minw_layer_desc &d = layers[l];
        LayerPlan P;
        P.d = d;
        P.d.w = nullptr; P.d.w_scale = nullptr; P.d.scale = nullptr; P.d.shift = nullptr;
        const bool first = l == 0, last = l == n_layers - 1;
        // this layer's request, in the values minw_net_layer_variants reports (there
        // MINW_VARIANT_TC is a layer on E4M3 operands), else the network's
        const int req = d.variant != 0 ? (d.variant == MINW_VARIANT_TC ? MINW_VARIANT_TC_E4M3 : d.variant) : variant;
        if (!d.w || !d.scale || !d.shift || d.O <= 0 || d.C <= 0 || d.H <= 0 || d.W <= 0 || d.variant < 0 ||
            d.variant > MINW_VARIANT_TC_E2M1_N128) {
            net_free(n);
            return MINW_EINVAL;
        }
        if ((first && (d.bits_in != 0 || d.kind != MINW_LAYER_CONV)) || (!first && d.bits_in != pbits) ||
            (last && d.bits_out != 0) || (!last && (d.bits_out < 1 || d.bits_out > 3)) ||
            (!first && (d.bits_w < 1 || d.bits_w > 3)) || (first && (d.bits_w < 0 || d.bits_w > 3)) ||
            (!first && (d.C != pc || d.H != ph || d.W != pw))) {
            net_free(n);
            return MINW_EINVAL;
        }
        P.C = d.C; P.H = d.H; P.W = d.W; P.O = d.O;
        if (d.kind == MINW_LAYER_FC) {
            P.kh = d.H; P.kw = d.W; P.stride = 1; P.pad = 0; P.pool = 0;
        } else {
            P.kh = d.kh; P.kw = d.kw; P.stride = d.stride; P.pad = d.pad; P.pool = d.pool;
        }
        if (P.kh <= 0 || P.kw <= 0 || P.stride <= 0 || P.pad < 0) { net_free(n); return MINW_EINVAL; }
        P.Ho = (P.H + 2 * P.pad - P.kh) / P.stride + 1;
        P.Wo = (P.W + 2 * P.pad - P.kw) / P.stride + 1;
        if (P.Ho <= 0 || P.Wo <= 0 || (P.pool && ((P.Ho & 1) || (P.Wo & 1)))) {
            net_free(n);
            return MINW_EINVAL;
        }
        P.Hp = P.pool ? P.Ho / 2 : P.Ho;
        P.Wp = P.pool ? P.Wo / 2 : P.Wo;
        P.qw.bits = d.bits_w; P.qw.scale = 1.0f;
        for (int i = 0; i < 3; ++i) P.qw.thr[i] = d.thr_w[i];
        P.qo.bits = d.bits_out; P.qo.scale = 1.0f;
        for (int i = 0; i < 3; ++i) P.qo.thr[i] = d.thr_out[i];
        if ((d.bits_w > 0 && !valid_quant(&P.qw)) || (!last && !valid_quant(&P.qo))) {
            net_free(n);
            return MINW_EINVAL;
        }
        minw_status st = MINW_OK;
        if ((st = net_alloc(n, &P.scale, P.O)) != MINW_OK || (st = net_alloc(n, &P.shift, P.O)) != MINW_OK) {
            net_free(n);
            return st;
        }
        cudaMemcpyAsync(P.scale, d.scale, sizeof(float) * P.O, cudaMemcpyDeviceToDevice, s);
        cudaMemcpyAsync(P.shift, d.shift, sizeof(float) * P.O, cudaMemcpyDeviceToDevice, s);
        const size_t K = (size_t)P.C * P.kh * P.kw;
        if (first) {
            if (!last) {
                if ((st = net_alloc(n, &P.thr, (size_t)P.O * 8)) != MINW_OK) { net_free(n); return st; }
                if ((st = launch_thresholds_f32(P.scale, P.shift, P.O, to_qparams(&P.qo), P.thr, s)) != MINW_OK) {
                    net_free(n);
                    return st;
                }
            }
            if ((st = net_alloc(n, &P.wlatent, (size_t)P.O * K)) != MINW_OK) { net_free(n); return st; }
            cudaMemcpyAsync(P.wlatent, d.w, sizeof(float) * P.O * K, cudaMemcpyDeviceToDevice, s);
            if (d.w_scale) {
                if ((st = net_alloc(n, &P.wscale, P.O)) != MINW_OK) { net_free(n); return st; }
                cudaMemcpyAsync(P.wscale, d.w_scale, sizeof(float) * P.O, cudaMemcpyDeviceToDevice, s);
            }
            if ((st = net_alloc(n, &P.wt, (size_t)P.O * K)) != MINW_OK) { net_free(n); return st; }
            if ((st = launch_first_weights(P.wlatent, P.O, (int)K, d.bits_w > 0, to_qparams(&P.qw), P.wscale, P.wt,
                                           s)) != MINW_OK) {
                net_free(n);
                return st;
            }
        } else {
            if (P.C % 32 != 0) { net_free(n); return MINW_EUNSUPPORTED; }
            if (P.pad >= P.kh || P.pad >= P.kw) { net_free(n); return MINW_EUNSUPPORTED; }
            ConvArgs a{};
            a.B = max_batch; a.C = P.C; a.H = P.H; a.W = P.W; a.O = P.O; a.kh = P.kh; a.kw = P.kw;
            a.stride = P.stride; a.pad = P.pad; a.Ho = P.Ho; a.Wo = P.Wo; a.NW = P.C / 32;
            a.bits_a = d.bits_in; a.bits_w = d.bits_w;
            a.M = (long long)max_batch * P.Ho * P.Wo;
            a.pool = P.pool;
            a.quant_out = !last;
            if (!last) a.qo = to_qparams(&P.qo);
            P.variant = choose_variant(a, req >= MINW_VARIANT_TC ? MINW_VARIANT_TC : req);
            if (P.variant == MINW_VARIANT_TC && !conv_tc_supported(a)) { net_free(n); return MINW_EUNSUPPORTED; }
            if (P.variant == MINW_VARIANT_TC && req != MINW_VARIANT_TC_E4M3) {
                // E2M1 operands wherever the channels fill 64-byte rows
                a.fp4 = 1;
                P.in4 = conv_tc_supported(a) ? 1 : 0;
                a.fp4 = P.in4;
                // requested tilings, planned with the split workspace the layer gets at run time
                // (a layer that splits along K runs no CTA pairs)
                ConvArgs c = a;
                const size_t wsn = conv_tc_workspace_bytes(c);
                c.workspace = wsn ? reinterpret_cast<void *>(256) : nullptr;
                c.workspace_bytes = wsn;
                if (req == MINW_VARIANT_TC_E2M1_PAIRS && P.in4) {
                    c.pair_n128 = 1;
                    P.pair128 = conv_tc_pairs128(c) ? 1 : 0;
                    a.pair_n128 = P.pair128;
                }
                if (req == MINW_VARIANT_TC_E2M1_N128 && P.in4) {
                    c.n128 = 1;
                    P.n128 = conv_tc_n128(c) ? 1 : 0;
                    a.n128 = P.n128;
                }
            }
            if (P.variant == MINW_VARIANT_TC) {
                const size_t wb = conv_tc_workspace_bytes(a);
                if (wb > n->ws_bytes) n->ws_bytes = wb;
            }
        }
        pc = P.O; ph = P.Hp; pw = P.Wp; pbits = d.bits_out;
        n->L.push_back(P);
    }
    // MINW_VARIANT_AUTO: the operand format of each tensor-core layer that can
    // take both is chosen by measurement (tune_formats)
    if (variant == MINW_VARIANT_AUTO) {
        minw_status st = tune_formats(n, layers, n_layers, max_batch, s);
        if (st != MINW_OK) { net_free(n); return st; }
    }
    // input layouts follow the consumer's kernel; weights are quantized once
    for (int l = 1; l < n_layers; ++l) {
        LayerPlan &P = n->L[l];
        const minw_layer_desc &d = layers[l];
        P.in_codes = P.variant == MINW_VARIANT_TC;
        minw_status st;
        // the weights are [O][C][kh][kw]; an FC weight [O][K] with K in
        // (c, h, w) order is the same array
        if (P.in_codes) {
            const size_t bytes = (size_t)P.O * P.kh * P.kw * P.C;
            if ((st = net_alloc(n, &P.wcodes, bytes)) != MINW_OK) { net_free(n); return st; }
            st = P.in4 ? minw_pack_weight_codes_e2m1(d.w, P.O, P.C, P.kh, P.kw, &P.qw, d.w_scale, P.wcodes, stream)
                       : minw_pack_weight_codes(d.w, P.O, P.C, P.kh, P.kw, &P.qw, d.w_scale, P.wcodes, stream);
            if (st == MINW_OK && l + 1 < n_layers) {
                const QParams qo = to_qparams(&P.qo);
                st = net_alloc(n, &P.thr, (size_t)P.O * num_levels(qo.bits));
                if (st == MINW_OK) st = launch_thresholds(P.scale, P.shift, P.O, qo, P.thr, s);
            }
        } else {
            const size_t words = (size_t)P.O * P.kh * P.kw * d.bits_w * (P.C / 32);
            if ((st = net_alloc(n, &P.wplanes, words)) != MINW_OK) { net_free(n); return st; }
            st = minw_pack_weights(d.w, P.O, P.C, P.kh, P.kw, &P.qw, d.w_scale, P.wplanes, stream);
        }
        if (st != MINW_OK) { net_free(n); return st; }
    }
    for (int l = 0; l + 1 < n_layers; ++l) {
        const LayerPlan &P = n->L[l];
        const bool codes = n->L[l + 1].in_codes;
        const size_t cbytes = (size_t)max_batch * P.Hp * P.Wp * P.O / (n->L[l + 1].in4 ? 2 : 1);
        const size_t words = codes ? (cbytes + 3) / 4
                                   : (size_t)max_batch * P.Hp * P.Wp * P.d.bits_out * ((P.O + 31) / 32);
        if (words > max_words) max_words = words;
    }
    for (int i = 0; i < 2; ++i) {
        minw_status st = net_alloc(n, &n->buf[i], max_words);
        if (st != MINW_OK) { net_free(n); return st; }
    }
    n->buf_words = max_words;
    if (n->ws_bytes) {
        uint8_t *w = nullptr;
        minw_status st = net_alloc(n, &w, n->ws_bytes);
        if (st != MINW_OK) { net_free(n); return st; }
        if (cudaMemsetAsync(w, 0, n->ws_bytes, s) != cudaSuccess) { net_free(n); return MINW_ECUDA; }
        n->ws = w;
    }
    n->x_elems = (size_t)max_batch * layers[0].C * layers[0].H * layers[0].W;
    const LayerPlan &PL = n->L.back();
    n->logit_elems = (size_t)max_batch * PL.O * PL.Hp * PL.Wp;
    {
        minw_status st = net_alloc(n, &n->x_stage, n->x_elems);
        if (st == MINW_OK) st = net_alloc(n, &n->logits_stage, n->logit_elems);
        if (st != MINW_OK) { net_free(n); return st; }
    }
    if (cudaStreamSynchronize(s) != cudaSuccess) { net_free(n); return MINW_ECUDA; }
    *out = n;
    return MINW_OK;
}

// Plan option graph = 0 enqueues every kernel on every call instead of
// replaying the captured forward.
static bool graphs_enabled() { return minw_host::plan_options().graph != 0; }

static minw_status forward_enqueue(minw_net *net, const float *x, int32_t B, float *logits, cudaStream_t cs) {
    if (net->kind == 1) return resnet_forward(net, x, B, logits, cs);
    if (net->kind == 2) return wresnet_forward(net, x, B, logits, cs);
    if (net->kind == 3) return wdense_forward(net, x, B, logits, cs);
    const int nl = (int)net->L.size();
    int cur = 0;
    if (net->timing && cudaEventRecord(net->events[0], cs) != cudaSuccess) return MINW_ECUDA;
    for (int l = 0; l < nl; ++l) {
        const LayerPlan &P = net->L[l];
        const bool last = l == nl - 1;
        const bool out_codes = !last && net->L[l + 1].in_codes;
        void *dst = last ? nullptr : (void *)net->buf[cur];
        minw_status st;
        if (l == 0) {
            FirstArgs a{};
            a.x = x; a.w = P.wlatent; a.cscale = P.wscale;
            a.quant_w = P.d.bits_w > 0;
            if (a.quant_w) a.qw = to_qparams(&P.qw);
            a.B = B; a.C = P.C; a.H = P.H; a.W = P.W; a.O = P.O; a.kh = P.kh; a.kw = P.kw;
            a.stride = P.stride; a.pad = P.pad; a.Ho = P.Ho; a.Wo = P.Wo;
            a.scale = P.scale; a.shift = P.shift;
            a.quant_out = !last;
            if (!last) a.qo = to_qparams(&P.qo);
            a.planes_out = out_codes ? nullptr : (uint32_t *)dst;
            a.codes_out = out_codes ? (uint8_t *)dst : nullptr;
            a.codes4 = out_codes && net->L[l + 1].in4;
            a.y_out = last ? logits : nullptr;
            a.thr = P.thr;
            a.wt = P.wt;
            st = launch_conv_first(a, cs);
        } else {
            const void *src = net->buf[cur ^ 1];
            ConvArgs a{};
            a.B = B; a.C = P.C; a.H = P.H; a.W = P.W; a.O = P.O; a.kh = P.kh; a.kw = P.kw;
            a.stride = P.stride; a.pad = P.pad; a.Ho = P.Ho; a.Wo = P.Wo; a.NW = P.C / 32;
            a.bits_a = P.d.bits_in; a.bits_w = P.d.bits_w;
            a.M = (long long)B * P.Ho * P.Wo;
            a.scale = P.scale; a.shift = P.shift; a.pool = P.pool;
            a.quant_out = !last;
            if (!last) a.qo = to_qparams(&P.qo);
            a.planes_out = (!last && !out_codes) ? (uint32_t *)dst : nullptr;
            a.codes_out = out_codes ? (uint8_t *)dst : nullptr;
            a.codes_out4 = out_codes && net->L[l + 1].in4;
            a.y_out = last ? logits : nullptr;
            a.fp4 = P.in4;
            a.pair_n128 = P.pair128;
            a.n128 = P.n128;
            if (P.in_codes) {
                a.act8 = (const uint8_t *)src;
                a.wgt8 = P.wcodes;
                a.thr = P.thr;
                a.workspace = net->ws;
                a.workspace_bytes = net->ws_bytes;
                st = launch_conv_tc(a, cs);
            } else {
                a.act = (const uint32_t *)src;
                a.wgt = P.wplanes;
                st = launch_conv_popc(a, cs);
            }
        }
        if (st != MINW_OK) return st;
        if (net->timing && cudaEventRecord(net->events[l + 1], cs) != cudaSuccess) return MINW_ECUDA;
        cur ^= 1;
    }
    return MINW_OK;
}

// The forward's kernels are captured once into a CUDA graph on a stream the
// net owns and replayed on the caller's stream while the input and logits
// pointers and the batch stay the same (any change re-captures); per-layer
// timing enqueues the kernels directly, and so does a call made while the
// caller's stream is itself being captured.
minw_status minw_forward(minw_net *net, const float *x, int32_t B, float *logits, void *stream) {
    if (!net || !x || !logits || B <= 0 || B > net->max_batch) return MINW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (net->timing || !graphs_enabled() || cudaStreamIsCapturing(s, &cap) != cudaSuccess ||
        cap != cudaStreamCaptureStatusNone)
        return forward_enqueue(net, x, B, logits, s);
    if (net->gexec == nullptr || net->gx != x || net->glogits != logits || net->gB != B) {
        if (net->cap_stream == nullptr &&
            cudaStreamCreateWithFlags(&net->cap_stream, cudaStreamNonBlocking) != cudaSuccess)
            return MINW_ECUDA;
        if (cudaStreamBeginCapture(net->cap_stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
            return MINW_ECUDA;
        const minw_status st = forward_enqueue(net, x, B, logits, net->cap_stream);
        cudaGraph_t g = nullptr;
        const cudaError_t ce = cudaStreamEndCapture(net->cap_stream, &g);
        if (st != MINW_OK || ce != cudaSuccess || g == nullptr) {
            if (g) cudaGraphDestroy(g);
            cudaGetLastError();
            return st != MINW_OK ? st : MINW_ECUDA;
        }
        if (net->gexec) cudaGraphExecDestroy(net->gexec);
        net->gexec = nullptr;
        const cudaError_t ie = cudaGraphInstantiate(&net->gexec, g, 0);
        cudaGraphDestroy(g);
        if (ie != cudaSuccess) {
            net->gexec = nullptr;
            return MINW_ECUDA;
        }
        net->gx = x;
        net->glogits = logits;
        net->gB = B;
    }
    return cudaGraphLaunch(net->gexec, s) == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

minw_status minw_forward_host(minw_net *net, const float *x_host, int32_t B, float *logits_host,
                              void *stream) {
    if (!net || !x_host || !logits_host || B <= 0 || B > net->max_batch) return MINW_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    const size_t xin = net->x_elems / net->max_batch * B;
    const size_t lout = net->logit_elems / net->max_batch * B;
    if (cudaMemcpyAsync(net->x_stage, x_host, xin * sizeof(float), cudaMemcpyHostToDevice, s) != cudaSuccess)
        return MINW_ECUDA;
    minw_status st = minw_forward(net, net->x_stage, B, net->logits_stage, stream);
    if (st != MINW_OK) return st;
    if (cudaMemcpyAsync(logits_host, net->logits_stage, lout * sizeof(float), cudaMemcpyDeviceToHost, s) !=
        cudaSuccess)
        return MINW_ECUDA;
    return cudaStreamSynchronize(s) == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

minw_status minw_net_enable_timing(minw_net *net, int32_t on) {
    if (!net) return MINW_EINVAL;
    if (on && net->events.empty()) {
        net->events.resize((size_t)minw_net_launches(net) + 1);
        for (auto &e : net->events)
            if (cudaEventCreate(&e) != cudaSuccess) return MINW_ECUDA;
    }
    net->timing = on != 0;
    return MINW_OK;
}

minw_status minw_net_layer_times(minw_net *net, float *ms) {
    if (!net || !ms || net->events.empty()) return MINW_EINVAL;
    if (cudaEventSynchronize(net->events.back()) != cudaSuccess) return MINW_ECUDA;
    for (size_t l = 0; l + 1 < net->events.size(); ++l)
        if (cudaEventElapsedTime(&ms[l], net->events[l], net->events[l + 1]) != cudaSuccess) return MINW_ECUDA;
    return MINW_OK;
}

minw_status minw_net_layer_candidates(const minw_net *net, int32_t layer, float *ms) {
    if (!net || !ms) return MINW_EINVAL;
    if (net->kind != 0) return MINW_EUNSUPPORTED;
    if (layer < 0 || layer >= (int32_t)net->L.size()) return MINW_EINVAL;
    for (int f = 0; f < 5; ++f) ms[f] = net->L[layer].cand_ms[f];
    return MINW_OK;
}

minw_status minw_net_layer_variants(const minw_net *net, int32_t *variants) {
    if (!net || !variants) return MINW_EINVAL;
    if (net->kind == 1) {
        resnet_variants(net, variants);     // stem, pool, the block convolutions, head
        return MINW_OK;
    }
    if (net->kind == 2) {
        wresnet_variants(net, variants);    // stem, its pass, per block conv1, pass, [shortcut], conv2, pass; head
        return MINW_OK;
    }
    if (net->kind == 3) {
        wdense_variants(net, variants);     // stem, its pass, per layer 1x1, pass, 3x3, pass; transitions; head
        return MINW_OK;
    }
    for (size_t l = 0; l < net->L.size(); ++l)
        variants[l] = l == 0 ? 0
                      : net->L[l].n128 ? MINW_VARIANT_TC_E2M1_N128
                      : net->L[l].pair128 ? MINW_VARIANT_TC_E2M1_PAIRS
                      : net->L[l].in4 ? MINW_VARIANT_TC_E2M1 : net->L[l].variant;
    return MINW_OK;
}

int32_t minw_net_launches(const minw_net *net) {
    if (!net) return 0;
    return net->kind == 1   ? resnet_ops(net)
           : net->kind == 2 ? wresnet_ops(net)
           : net->kind == 3 ? wdense_ops(net)
                            : (int32_t)net->L.size();
}

// Kernels one minw_forward issues (a split-K layer issues two).
int32_t minw_net_kernels(const minw_net *net) {
    if (!net) return 0;
    if (net->kind == 1) return resnet_kernels(net);
    if (net->kind == 2) return wresnet_kernels(net);
    if (net->kind == 3) return wdense_kernels(net);
    int32_t k = 0;
    for (size_t l = 0; l < net->L.size(); ++l) {
        const LayerPlan &P = net->L[l];
        if (l == 0 || !P.in_codes) { ++k; continue; }
        ConvArgs a{};
        a.B = net->max_batch; a.C = P.C; a.H = P.H; a.W = P.W; a.O = P.O; a.kh = P.kh; a.kw = P.kw;
        a.stride = P.stride; a.pad = P.pad; a.Ho = P.Ho; a.Wo = P.Wo; a.NW = P.C / 32;
        a.M = (long long)net->max_batch * P.Ho * P.Wo; a.pool = P.pool;
        a.quant_out = l + 1 < net->L.size();
        if (a.quant_out) a.qo = to_qparams(&P.qo);
        a.act8 = P.wcodes; a.wgt8 = P.wcodes; a.thr = P.thr; a.fp4 = P.in4;
        a.pair_n128 = P.pair128; a.n128 = P.n128;
        a.workspace = net->ws; a.workspace_bytes = net->ws_bytes;
        k += conv_tc_launches(a);
    }
    return k;
}

void minw_net_destroy(minw_net *net) {
    if (!net) return;
    cudaDeviceSynchronize();
    net_free(net);
}

}  // extern "C"
