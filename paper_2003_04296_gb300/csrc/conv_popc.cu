// conv_popc.cu -- bit-serial implicit-GEMM convolution on the integer pipe
// (the XNOR / SHIFT inference of Table I and Sec. III-C on packed bit-planes).
//
// GEMM view: M = B*Ho*Wo output pixels, N = O output channels,
// K = kh*kw*C taken tap by tap in chunks of KC words (32*KC channels) of every
// bit-plane.  A CTA owns a 128-pixel x 64-channel tile; 256 threads each hold
// 4 pixels (lane + 32 i) x 8 channels (8 warp + j) of int32 accumulators.
// Chunks stream through a 3-stage cp.async pipeline (zero fill for padded taps
// and for channels >= O).
//
// Per 32-channel word the signed dot product of two level words follows from
// popcounts (exact integer arithmetic):
//   sign plane S, magnitude one-hot planes E_e with |level| = 2^e units
//   (1-bit: E_0 = "tap is valid", 2-bit: E_0 = non-zero mask,
//    3-bit: E_0..E_2 decoded from the 2-bit magnitude code),
//   dot = sum_{ea,ew} 2^(ea+ew) [popc(E_ea & E_ew) - 2 popc(E_ea & E_ew & (Sa ^ Sw))].
// 1-bit x 1-bit is the XNOR identity dot = valid*32 - 2 popc((Sa ^ Sw) & valid).
//
// Epilogue (one pass through shared memory): optional raw int32 output, 2x2
// max pool on the accumulator, BN as fmaf(acc, scale, shift), HardTanh and
// quantize + pack of the next layer's planes (Sec. III-E block order).
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace minw {

namespace popc {

constexpr int BM = 128;
constexpr int BN = 64;
constexpr int NT = 256;
constexpr int NSTAGE = 3;

template <int PA, int PW, int KC>
struct Smem {
    uint32_t a[NSTAGE][BM][PA][KC];
    uint32_t b[NSTAGE][BN][PW][KC];
};

constexpr int ACC_LD = BM + 1;   // padded row of the staged accumulator tile

template <int BYTES>
__device__ __forceinline__ void cp_async_zfill(void *smem, const void *gmem, bool valid) {
    const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
    const int src_bytes = valid ? BYTES : 0;
    if constexpr (BYTES == 16) {
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(src_bytes));
    } else {
        asm volatile("cp.async.ca.shared.global [%0], [%1], %2, %3;\n" ::"r"(s), "l"(gmem), "n"(BYTES), "r"(src_bytes));
    }
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

template <int KC>
__device__ __forceinline__ void lds_words(uint32_t (&d)[KC], const uint32_t *s) {
    if constexpr (KC == 4) {
        const uint4 v = *reinterpret_cast<const uint4 *>(s);
        d[0] = v.x; d[1] = v.y; d[2] = v.z; d[3] = v.w;
    } else if constexpr (KC == 2) {
        const uint2 v = *reinterpret_cast<const uint2 *>(s);
        d[0] = v.x; d[1] = v.y;
    } else {
        d[0] = s[0];
    }
}

// Magnitude one-hot planes of an operand word (P = bits).
template <int P>
__device__ __forceinline__ void magnitudes(const uint32_t *pl, uint32_t valid, uint32_t *E) {
    if constexpr (P == 1) {
        E[0] = valid;
    } else if constexpr (P == 2) {
        E[0] = pl[1];
    } else {
        const uint32_t c0 = pl[1], c1 = pl[2];
        E[0] = c0 & ~c1;      // code 1: 1/4  -> 1 unit
        E[1] = ~c0 & c1;      // code 2: 1/2  -> 2 units
        E[2] = c0 & c1;       // code 3: 1    -> 4 units
    }
}

template <int PA, int PW, int KC>
__global__ void __launch_bounds__(NT) conv_popc_kernel(const ConvArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    Smem<PA, PW, KC> &S = *reinterpret_cast<Smem<PA, PW, KC> *>(smem_raw);
    int32_t *sAcc = reinterpret_cast<int32_t *>(smem_raw);   // reused after the main loop
    __shared__ int sPix[BM];
    __shared__ int sY0[BM];
    __shared__ int sX0[BM];

    constexpr int NEA = (PA == 3) ? 3 : 1;
    constexpr int NEW = (PW == 3) ? 3 : 1;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const long long m0 = (long long)blockIdx.x * BM;
    const int o0 = blockIdx.y * BN;
    const int HoWo = a.Ho * a.Wo;

    for (int r = tid; r < BM; r += NT) {
        const long long m = m0 + r;
        if (m < a.M) {
            const int b = (int)(m / HoWo);
            const int rem = (int)(m - (long long)b * HoWo);
            const int yo = rem / a.Wo, xo = rem - (rem / a.Wo) * a.Wo;
            sPix[r] = b * a.H * a.W;
            sY0[r] = yo * a.stride - a.pad;
            sX0[r] = xo * a.stride - a.pad;
        } else {
            sPix[r] = -1;
            sY0[r] = 0;
            sX0[r] = 0;
        }
    }
    __syncthreads();

    const int nwc = a.NW / KC;
    const int ntaps = a.kh * a.kw;
    const int nchunks = ntaps * nwc;

    int py0[4], px0[4];
    bool pin[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = lane + 32 * i;
        pin[i] = sPix[r] >= 0;
        py0[i] = sY0[r];
        px0[i] = sX0[r];
    }

    auto load_stage = [&](int st, int chunk) {
        const int tap = chunk / nwc, wg = chunk - (chunk / nwc) * nwc;
        const int ky = tap / a.kw, kx = tap - (tap / a.kw) * a.kw;
        for (int u = tid; u < BM * PA; u += NT) {
            const int r = u / PA, p = u - (u / PA) * PA;
            const int yi = sY0[r] + ky, xi = sX0[r] + kx;
            const bool v = sPix[r] >= 0 && yi >= 0 && yi < a.H && xi >= 0 && xi < a.W;
            const uint32_t *src = a.act;
            if (v) src = a.act + ((long long)(sPix[r] + yi * a.W + xi) * PA + p) * a.NW + wg * KC;
            cp_async_zfill<KC * 4>(&S.a[st][r][p][0], src, v);
        }
        for (int u = tid; u < BN * PW; u += NT) {
            const int r = u / PW, p = u - (u / PW) * PW;
            const int o = o0 + r;
            const bool v = o < a.O;
            const uint32_t *src = a.wgt;
            if (v) src = a.wgt + ((long long)(o * ntaps + tap) * PW + p) * a.NW + wg * KC;
            cp_async_zfill<KC * 4>(&S.b[st][r][p][0], src, v);
        }
    };

    int32_t acc[4][8];
    int32_t cnt[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        cnt[i] = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0;
    }

#pragma unroll
    for (int s = 0; s < NSTAGE - 1; ++s) {
        if (s < nchunks) load_stage(s, s);
        cp_async_commit();
    }

    for (int chunk = 0; chunk < nchunks; ++chunk) {
        cp_async_wait<NSTAGE - 2>();
        __syncthreads();
        {
            const int nx = chunk + NSTAGE - 1;
            if (nx < nchunks) load_stage(nx % NSTAGE, nx);
            cp_async_commit();
        }
        const int st = chunk % NSTAGE;
        const int tap = chunk / nwc;
        const int ky = tap / a.kw, kx = tap - (tap / a.kw) * a.kw;

        // weights of this thread's 8 channels for the chunk
        uint32_t wv[8][PW][KC];
#pragma unroll
        for (int j = 0; j < 8; ++j)
#pragma unroll
            for (int p = 0; p < PW; ++p) lds_words<KC>(wv[j][p], &S.b[st][warp * 8 + j][p][0]);

        // per-channel magnitude counts (1-bit activations x multi-level weights)
        int32_t cw[8];
        if constexpr (PA == 1 && PW > 1) {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                int32_t c = 0;
#pragma unroll
                for (int kk = 0; kk < KC; ++kk) {
                    uint32_t pl[PW], E[NEW];
#pragma unroll
                    for (int p = 0; p < PW; ++p) pl[p] = wv[j][p][kk];
                    magnitudes<PW>(pl, 0xffffffffu, E);
#pragma unroll
                    for (int e = 0; e < NEW; ++e) c += __popc(E[e]) << e;
                }
                cw[j] = c;
            }
        }

#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int yi = py0[i] + ky, xi = px0[i] + kx;
            const bool valid = pin[i] && yi >= 0 && yi < a.H && xi >= 0 && xi < a.W;
            const uint32_t vm = valid ? 0xffffffffu : 0u;
            uint32_t av[PA][KC];
#pragma unroll
            for (int p = 0; p < PA; ++p) lds_words<KC>(av[p], &S.a[st][lane + 32 * i][p][0]);

            if constexpr (PA == 1 && PW == 1) {
                cnt[i] += valid ? 32 * KC : 0;
#pragma unroll
                for (int j = 0; j < 8; ++j)
#pragma unroll
                    for (int kk = 0; kk < KC; ++kk)
                        acc[i][j] -= __popc((av[0][kk] ^ wv[j][0][kk]) & vm) << 1;
            } else if constexpr (PW == 1) {
                uint32_t E[KC][NEA];
#pragma unroll
                for (int kk = 0; kk < KC; ++kk) {
                    uint32_t pl[PA];
#pragma unroll
                    for (int p = 0; p < PA; ++p) pl[p] = av[p][kk];
                    magnitudes<PA>(pl, vm, E[kk]);
#pragma unroll
                    for (int e = 0; e < NEA; ++e) cnt[i] += __popc(E[kk][e]) << e;
                }
#pragma unroll
                for (int j = 0; j < 8; ++j)
#pragma unroll
                    for (int kk = 0; kk < KC; ++kk) {
                        const uint32_t X = av[0][kk] ^ wv[j][0][kk];
#pragma unroll
                        for (int e = 0; e < NEA; ++e) acc[i][j] -= __popc(E[kk][e] & X) << (e + 1);
                    }
            } else if constexpr (PA == 1) {
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    acc[i][j] += valid ? cw[j] : 0;
#pragma unroll
                    for (int kk = 0; kk < KC; ++kk) {
                        uint32_t pl[PW], E[NEW];
#pragma unroll
                        for (int p = 0; p < PW; ++p) pl[p] = wv[j][p][kk];
                        magnitudes<PW>(pl, 0xffffffffu, E);
                        const uint32_t X = (av[0][kk] ^ wv[j][0][kk]) & vm;
#pragma unroll
                        for (int e = 0; e < NEW; ++e) acc[i][j] -= __popc(E[e] & X) << (e + 1);
                    }
                }
            } else {
                uint32_t Ea[KC][NEA];
#pragma unroll
                for (int kk = 0; kk < KC; ++kk) {
                    uint32_t pl[PA];
#pragma unroll
                    for (int p = 0; p < PA; ++p) pl[p] = av[p][kk];
                    magnitudes<PA>(pl, vm, Ea[kk]);
                }
#pragma unroll
                for (int j = 0; j < 8; ++j)
#pragma unroll
                    for (int kk = 0; kk < KC; ++kk) {
                        uint32_t pl[PW], Ew[NEW];
#pragma unroll
                        for (int p = 0; p < PW; ++p) pl[p] = wv[j][p][kk];
                        magnitudes<PW>(pl, 0xffffffffu, Ew);
                        const uint32_t X = av[0][kk] ^ wv[j][0][kk];
#pragma unroll
                        for (int k = 0; k < NEA + NEW - 1; ++k) {
                            uint32_t T = 0u;
#pragma unroll
                            for (int ea = 0; ea < NEA; ++ea) {
                                const int ew = k - ea;
                                if (ew >= 0 && ew < NEW) T |= Ea[kk][ea] & Ew[ew];
                            }
                            acc[i][j] += (__popc(T) - (__popc(T & X) << 1)) << k;
                        }
                    }
            }
        }
    }
    cp_async_wait<0>();
    __syncthreads();

    // ---- stage the accumulator tile: sAcc[channel][pixel] ----
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) sAcc[(warp * 8 + j) * ACC_LD + lane + 32 * i] = acc[i][j] + cnt[i];
    __syncthreads();

    // ---- raw accumulator output (unpooled, NCHW) ----
    if (a.acc_out != nullptr) {
        const int r = tid & (BM - 1);
        const long long m = m0 + r;
        if (m < a.M) {
            const long long b = m / HoWo;
            const long long pix = m - b * HoWo;
            for (int c = tid >> 7; c < BN; c += NT / BM) {
                const int o = o0 + c;
                if (o < a.O) a.acc_out[(b * a.O + o) * HoWo + pix] = sAcc[c * ACC_LD + r];
            }
        }
    }
    if (a.y_out == nullptr && !a.quant_out) return;

    // ---- pooled / unpooled output pixels: BN, HardTanh, quantize + pack ----
    const int Wp = a.pool ? a.Wo / 2 : a.Wo;
    const int HpWp = a.pool ? (a.Ho / 2) * Wp : HoWo;
    const int nq = a.pool ? BM / 4 : BM;        // output pixels owned by this tile
    const int groups = BN / 32;
    const int NWo = (a.O + 31) >> 5;
    for (int t = tid; t < nq * groups; t += NT) {
        const int q = t % nq, g = t / nq;
        int r00;
        if (a.pool) {
            const int half = a.Wo / 2;
            const int prow = q / half, pc = q - (q / half) * half;
            r00 = 2 * prow * a.Wo + 2 * pc;
        } else {
            r00 = q;
        }
        const long long m = m0 + r00;
        if (m >= a.M) continue;
        const long long b = m / HoWo;
        const int pix = (int)(m - b * HoWo);
        const int yo = pix / a.Wo, xo = pix - (pix / a.Wo) * a.Wo;
        const int opix = a.pool ? (yo / 2) * Wp + (xo / 2) : pix;
        uint32_t words[3] = {0u, 0u, 0u};
        uint32_t cw[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
        for (int c = 0; c < 32; ++c) {
            const int cc = g * 32 + c;
            const int o = o0 + cc;
            if (o >= a.O) break;
            int32_t v = sAcc[cc * ACC_LD + r00];
            if (a.pool) {
                v = max(v, sAcc[cc * ACC_LD + r00 + 1]);
                v = max(v, sAcc[cc * ACC_LD + r00 + a.Wo]);
                v = max(v, sAcc[cc * ACC_LD + r00 + a.Wo + 1]);
            }
            float y = fmaf((float)v, __ldg(a.scale + o), __ldg(a.shift + o));
            if (a.quant_out) {
                y = fminf(fmaxf(y, -1.0f), 1.0f);
                const int lv = level_units(y * a.qo.scale, a.qo);
                const uint32_t pb = level_plane_bits(lv, a.qo.bits);
                cw[c >> 2] |= (uint32_t)level_code_e4m3(lv) << ((c & 3) * 8);
                words[0] |= (pb & 1u) << c;
                words[1] |= ((pb >> 1) & 1u) << c;
                words[2] |= ((pb >> 2) & 1u) << c;
            }
            if (a.y_out != nullptr) a.y_out[(b * a.O + o) * HpWp + opix] = y;
        }
        if (a.quant_out && a.codes_out != nullptr) {
            const int ob = o0 + g * 32;
            uint4 *dst = reinterpret_cast<uint4 *>(a.codes_out + (b * HpWp + opix) * a.O + ob);
            if (ob < a.O) dst[0] = make_uint4(cw[0], cw[1], cw[2], cw[3]);
            if (ob + 16 < a.O) dst[1] = make_uint4(cw[4], cw[5], cw[6], cw[7]);
        }
        if (a.quant_out && a.planes_out != nullptr) {
            const int wi = (o0 >> 5) + g;
            if (wi < NWo) {
                uint32_t *dst = a.planes_out + ((b * HpWp + opix) * a.qo.bits) * NWo + wi;
                for (int p = 0; p < a.qo.bits; ++p) dst[p * NWo] = words[p];
            }
        }
    }
}

template <int PA, int PW, int KC>
minw_status launch_t(const ConvArgs &a, cudaStream_t s) {
    const size_t pipe = sizeof(Smem<PA, PW, KC>);
    const size_t epi = sizeof(int32_t) * BN * ACC_LD;
    const size_t smem = pipe > epi ? pipe : epi;
    static bool configured = false;
    if (!configured) {
        if (cudaFuncSetAttribute(conv_popc_kernel<PA, PW, KC>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
            return MINW_ECUDA;
        configured = true;
    }
    const dim3 grid((unsigned)((a.M + BM - 1) / BM), (unsigned)((a.O + BN - 1) / BN));
    conv_popc_kernel<PA, PW, KC><<<grid, NT, smem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? MINW_OK : MINW_ECUDA;
}

template <int PA, int PW>
minw_status launch_kc(const ConvArgs &a, cudaStream_t s) {
    if (a.NW % 4 == 0) return launch_t<PA, PW, 4>(a, s);
    if (a.NW % 2 == 0) return launch_t<PA, PW, 2>(a, s);
    return launch_t<PA, PW, 1>(a, s);
}

}  // namespace popc

minw_status launch_conv_popc(const ConvArgs &a, cudaStream_t s) {
    if (a.pool && (popc::BM % (2 * a.Wo) != 0 || (a.Ho & 1) || (a.Wo & 1))) return MINW_EUNSUPPORTED;
    if (a.M > (1ll << 31) * popc::BM) return MINW_EUNSUPPORTED;
    switch (a.bits_a * 4 + a.bits_w) {
        case 5: return popc::launch_kc<1, 1>(a, s);
        case 6: return popc::launch_kc<1, 2>(a, s);
        case 7: return popc::launch_kc<1, 3>(a, s);
        case 9: return popc::launch_kc<2, 1>(a, s);
        case 10: return popc::launch_kc<2, 2>(a, s);
        case 11: return popc::launch_kc<2, 3>(a, s);
        case 13: return popc::launch_kc<3, 1>(a, s);
        case 14: return popc::launch_kc<3, 2>(a, s);
        case 15: return popc::launch_kc<3, 3>(a, s);
    }
    return MINW_EINVAL;
}

}  // namespace minw
