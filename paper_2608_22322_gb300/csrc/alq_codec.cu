// alq_codec.cu -- stand-alone AL (Sec. 4.1, Eq. (3)-(5)) and UF8 (Sec. 4.3)
// codec kernels and their C-ABI entry points. One HBM pass each: the encoder
// reduces each block's minimum positive value and maximum with warp
// reductions, derives (l_min, Delta) once per block and writes codes and
// metadata; the decoder rebuilds each block's level tables and writes fp32.
// the level and bound passes' exp2/log2 tables from per-CTA shared copies
#define ALQ_SMEM_TABLES 1
#include "alq_kernels.cuh"

namespace alq {

template <typename Kernel>
static int grid_for(Kernel kernel, int64_t ntiles) {
    return persistent_grid((const void*)kernel, kThreads, 0, ntiles);
}

// ------------------------------------------------------------- AL encode --
// Three CTAs per SM (at most 80 registers; four, 64 registers, for blocks of
// 512): the per-block chain (reduction, two-float log2, constants) is
// latency bound, and more resident warps hide more of it.
template <int CPB, int BITS>
__global__ void __launch_bounds__(kThreads, CPB == 4 ? 4 : 3)
al_encode_kernel(const float* __restrict__ x, int64_t n, int block, float log_floor,
                 void* __restrict__ codes, float* __restrict__ meta, int64_t ntiles) {
    constexpr int NB = 4 / CPB;
    constexpr float Lm2 = BITS == 8 ? 254.0f : 65534.0f;
    __shared__ uint32_t s_part[2][kThreads / 32];
    const int warp = __shfl_sync(0xFFFFFFFFu, (int)(threadIdx.x >> 5), 0), lane = threadIdx.x & 31;
    const int wpb = CPB == 4 && block > kSeg ? block / kSeg : 1;
    const int bshift = block_shift<CPB, 4>(block);
    const int64_t nblk = (n + (1 << bshift) - 1) >> bshift;
    for (int i = threadIdx.x; i < 1024; i += kThreads) {
        s_kExp2Hi[i] = kExp2HiD[i];
        s_kExp2Lo[i] = kExp2LoD[i];
        s_kLog2C[i] = kLog2CD[i];
        s_kLog2Hi[i] = kLog2HiD[i];
        s_kLog2Lo[i] = kLog2LoD[i];
    }
    __syncthreads();
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int64_t seg0 = tile * kTile + (int64_t)warp * kSeg;
        const bool full = seg0 + kSeg <= n;  // warp-uniform: unmasked I/O
        float4 v[4];
        uint32_t cmin[4], cmax[4];
        if (full) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                v[c] = __ldcs(reinterpret_cast<const float4*>(x + chunk_index(seg0, c, lane)));
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c) v[c] = load4f(x, chunk_index(seg0, c, lane), n);
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            cmin[c] = 0xFFFFFFFFu;
            cmax[c] = 0u;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t b = f2u(f4get(v[c], i)) & 0x7FFFFFFFu;  // -0 -> 0
                cmin[c] = umix<false>(cmin[c], b - 1u);               // 0 -> max
                cmax[c] = umix<true>(cmax[c], b);
            }
        }
        uint32_t bmin[NB], bmax[NB];
        warp_blocks_reduce<CPB, false>(cmin, bmin);
        warp_blocks_reduce<CPB, true>(cmax, bmax);
        if (wpb > 1) {
            bmin[0] = cta_group_reduce<false>(bmin[0], s_part[0], wpb);
            bmax[0] = cta_group_reduce<true>(bmax[0], s_part[1], wpb);
        }
        float mn[NB], mx[NB], lmin[NB], delta[NB];
        AlEncConsts ek[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            mn[b] = u2f(bmin[b] + 1u);
            mx[b] = u2f(bmax[b]);
        }
        al_blocks_params<NB>(mn, mx, log_floor, lmin, delta);
#pragma unroll
        for (int b = 0; b < NB; ++b) ek[b] = al_encode_consts(lmin[b], delta[b], Lm2);
        float xv[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) xv[e] = f4get(v[e / 4], e % 4);
        uint32_t q[16];
        al_encode_chunks<BITS, CPB, NB, 4>(xv, mn, lmin, delta, ek, q);
        uint32_t wq[4 * BITS / 8];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            if constexpr (BITS == 8) {
                wq[c] = q[4 * c] | (q[4 * c + 1] << 8) | (q[4 * c + 2] << 16) | (q[4 * c + 3] << 24);
            } else {
                wq[2 * c] = q[4 * c] | (q[4 * c + 1] << 16);
                wq[2 * c + 1] = q[4 * c + 2] | (q[4 * c + 3] << 16);
            }
        }
        if (full) {
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int64_t idx = chunk_index(seg0, c, lane);
                if constexpr (BITS == 8)
                    __stcs(reinterpret_cast<unsigned int*>((uint8_t*)codes + idx), wq[c]);
                else
                    __stcs(reinterpret_cast<uint2*>((uint16_t*)codes + idx),
                           make_uint2(wq[2 * c], wq[2 * c + 1]));
            }
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int64_t idx = chunk_index(seg0, c, lane);
                if constexpr (BITS == 8)
                    store4b((uint8_t*)codes, idx, n, wq[c]);
                else
                    store4h((uint16_t*)codes, idx, n, make_uint2(wq[2 * c], wq[2 * c + 1]));
            }
        }
        if (lane == 0 && (warp % wpb) == 0) {
            const int64_t gb0 = seg0 >> bshift;
#pragma unroll
            for (int b = 0; b < NB; ++b)
                if (gb0 + b < nblk)
                    reinterpret_cast<float2*>(meta)[gb0 + b] = make_float2(lmin[b], delta[b]);
        }
    }
}

// ------------------------------------------------------------- AL decode --
template <int CPB, int BITS>
__global__ void __launch_bounds__(kThreads)
al_decode_kernel(const void* __restrict__ codes, const float* __restrict__ meta, int64_t n,
                 int block, float* __restrict__ out, int64_t ntiles, Opaque2 k) {
    constexpr int NB = 4 / CPB;
    __shared__ __align__(16) float2 s_tab[kThreads / 32][NB * 32];
    __shared__ float s_val[kThreads / 32][BITS == 8 ? NB * 256 : 1];
    const int warp = __shfl_sync(0xFFFFFFFFu, (int)(threadIdx.x >> 5), 0), lane = threadIdx.x & 31;
    const float kf = al8_table_k(lane);
    const int bshift = block_shift<CPB, 4>(block);
    const int64_t nblk = (n + (1 << bshift) - 1) >> bshift;
    for (int i = threadIdx.x; i < 1024; i += kThreads) {
        s_kExp2Hi[i] = kExp2HiD[i];
        s_kExp2Lo[i] = kExp2LoD[i];
        s_kLog2C[i] = kLog2CD[i];
        s_kLog2Hi[i] = kLog2HiD[i];
        s_kLog2Lo[i] = kLog2LoD[i];
    }
    __syncthreads();
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int64_t seg0 = tile * kTile + (int64_t)warp * kSeg;
        const bool full = seg0 + kSeg <= n;  // warp-uniform: unmasked I/O
        uint32_t w[4 * BITS / 8];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int64_t idx = chunk_index(seg0, c, lane);
            if (BITS == 8) {
                w[c] = full ? __ldcs(reinterpret_cast<const unsigned int*>((const uint8_t*)codes + idx))
                            : load4b((const uint8_t*)codes, idx, n);
            } else {
                const uint2 h = full ? __ldcs(reinterpret_cast<const uint2*>((const uint16_t*)codes + idx))
                                     : load4h((const uint16_t*)codes, idx, n);
                w[2 * c] = h.x;
                w[2 * c + 1] = h.y;
            }
        }
        float lmin[NB], delta[NB];
        const int64_t gb0 = seg0 >> bshift;
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            float2 mt = make_float2(0.f, 0.f);
            if (gb0 + b < nblk) mt = __ldg(reinterpret_cast<const float2*>(meta) + gb0 + b);
            lmin[b] = mt.x;
            delta[b] = mt.y;
        }
        // AL8: the blocks' 256 exactly rounded values in shared memory, then
        // one lookup per element; AL16: each level directly
        if constexpr (BITS == 8) {
            float* ts = reinterpret_cast<float*>(s_tab[warp]);  // 64 floats per block (SoA)
            if constexpr (NB >= 2) {
#pragma unroll
                for (int b = 0; b < NB; b += 2)
                    al8_build_tables2_soa(ts + 64 * b, ts + 64 * (b + 1), lmin[b], delta[b],
                                          lmin[b + 1], delta[b + 1], kf, k);
            } else {
                al8_build_tables_soa(ts, lmin[0], delta[0], kf);
            }
#pragma unroll
            for (int b = 0; b < NB; ++b)
                al8_values_from_tables_soa(s_val[warp] + 256 * b, ts + 64 * b, lmin[b], delta[b]);
        }
        float4 r4[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int b = c / CPB;
            float r[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t q = code_of<BITS>(w, c, i);
                if constexpr (BITS == 8)
                    r[i] = s_val[warp][256 * b + q];
                else
                    r[i] = al16_decode(q, lmin[b], delta[b]);
            }
            r4[c] = make_float4(r[0], r[1], r[2], r[3]);
        }
        if (full) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                __stcs(reinterpret_cast<float4*>(out + chunk_index(seg0, c, lane)), r4[c]);
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c) store4f(out, chunk_index(seg0, c, lane), n, r4[c]);
        }
        __syncwarp();
    }
}

// ------------------------------------------------------------ UF8 encode --
template <int CPB>
__global__ void __launch_bounds__(kThreads)
uf8_encode_kernel(const float* __restrict__ m, int64_t n, int block, int8_t* __restrict__ codes,
                  float* __restrict__ absmax, int64_t ntiles) {
    constexpr int NB = 4 / CPB;
    __shared__ uint32_t s_part[kThreads / 32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int wpb = CPB == 4 && block > kSeg ? block / kSeg : 1;
    const int bshift = block_shift<CPB, 4>(block);
    const int64_t nblk = (n + (1 << bshift) - 1) >> bshift;
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int64_t seg0 = tile * kTile + (int64_t)warp * kSeg;
        const bool full = seg0 + kSeg <= n;  // warp-uniform: unmasked I/O
        float4 v[4];
        uint32_t ca[4];
        if (full) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                v[c] = __ldcs(reinterpret_cast<const float4*>(m + chunk_index(seg0, c, lane)));
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c) v[c] = load4f(m, chunk_index(seg0, c, lane), n);
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            ca[c] = 0u;
#pragma unroll
            for (int i = 0; i < 4; ++i) ca[c] = umix<true>(ca[c], f2u(f4get(v[c], i)) & 0x7FFFFFFFu);
        }
        uint32_t ba[NB];
        warp_blocks_reduce<CPB, true>(ca, ba);
        if (wpb > 1) ba[0] = cta_group_reduce<true>(ba[0], s_part, wpb);
        float s[NB], sc[NB], inv[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            s[b] = u2f(ba[b]);
            sc[b] = 1.0f;
            inv[b] = 0.0f;
            if (s[b] > 0.0f) uf8_encode_consts(s[b], sc[b], inv[b]);
        }
        uint32_t wd[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int b = c / CPB;
            wd[c] = 0;
            if (s[b] > 0.0f) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    wd[c] |= ((uint32_t)uf8_quantize(f4get(v[c], i), sc[b], inv[b]) & 0xFFu) << (8 * i);
            }
        }
        if (full) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                __stcs(reinterpret_cast<unsigned int*>((uint8_t*)codes + chunk_index(seg0, c, lane)), wd[c]);
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c) store4b((uint8_t*)codes, chunk_index(seg0, c, lane), n, wd[c]);
        }
        if (lane == 0 && (warp % wpb) == 0) {
            const int64_t gb0 = seg0 >> bshift;
#pragma unroll
            for (int b = 0; b < NB; ++b)
                if (gb0 + b < nblk) absmax[gb0 + b] = s[b];
        }
    }
}

// ------------------------------------------------------------ UF8 decode --
template <int CPB>
__global__ void __launch_bounds__(kThreads)
uf8_decode_kernel(const int8_t* __restrict__ codes, const float* __restrict__ absmax, int64_t n,
                  int block, float* __restrict__ out, int64_t ntiles) {
    constexpr int NB = 4 / CPB;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int bshift = block_shift<CPB, 4>(block);
    const int64_t nblk = (n + (1 << bshift) - 1) >> bshift;
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int64_t seg0 = tile * kTile + (int64_t)warp * kSeg;
        float d[NB];
        const int64_t gb0 = seg0 >> bshift;
#pragma unroll
        for (int b = 0; b < NB; ++b)
            d[b] = (gb0 + b < nblk) ? __ldg(absmax + gb0 + b) / 127.0f : 0.0f;
        const bool full = seg0 + kSeg <= n;  // warp-uniform: unmasked I/O
        uint32_t w[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int64_t idx = chunk_index(seg0, c, lane);
            w[c] = full ? __ldcs(reinterpret_cast<const unsigned int*>((const uint8_t*)codes + idx))
                        : load4b((const uint8_t*)codes, idx, n);
        }
        float4 r[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int b = c / CPB;
            r[c].x = s8_to_float(w[c] & 0xFFu) * d[b];
            r[c].y = s8_to_float((w[c] >> 8) & 0xFFu) * d[b];
            r[c].z = s8_to_float((w[c] >> 16) & 0xFFu) * d[b];
            r[c].w = s8_to_float(w[c] >> 24) * d[b];
        }
        if (full) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                __stcs(reinterpret_cast<float4*>(out + chunk_index(seg0, c, lane)), r[c]);
        } else {
#pragma unroll
            for (int c = 0; c < 4; ++c) store4f(out, chunk_index(seg0, c, lane), n, r[c]);
        }
    }
}

// ------------------------------------------------------------- launchers --
static int cpb_of(int block) { return block >= 512 ? 4 : block / 128; }

#define ALQ_DISPATCH_CPB(block, KERNEL_TMPL, ...)                 \
    switch (cpb_of(block)) {                                      \
        case 1: { auto k = KERNEL_TMPL<1 __VA_ARGS__>; LAUNCH(k); } break; \
        case 2: { auto k = KERNEL_TMPL<2 __VA_ARGS__>; LAUNCH(k); } break; \
        default: { auto k = KERNEL_TMPL<4 __VA_ARGS__>; LAUNCH(k); } break; \
    }

}  // namespace alq

using namespace alq;

extern "C" {

int al_encode(const float* x, int64_t n, int block, int bits, float log_floor, void* codes,
              float* meta, void* stream) {
    if (n < 0) return ALQ_ERR_INVALID_ARG;
    if (!valid_block(block) || (bits != 8 && bits != 16)) return ALQ_ERR_UNSUPPORTED;
    if (n == 0) return ALQ_OK;
    if (!x || !codes || !meta) return ALQ_ERR_INVALID_ARG;
    if (!aligned(x, 16) || !aligned(codes, 16) || !aligned(meta, 8)) return ALQ_ERR_ALIGN;
    const int64_t ntiles = blocks_of(n, kTile);
    cudaStream_t s = (cudaStream_t)stream;
#define LAUNCH(k) k<<<grid_for(k, ntiles), kThreads, 0, s>>>(x, n, block, log_floor, codes, meta, ntiles)
    if (bits == 8) {
        ALQ_DISPATCH_CPB(block, al_encode_kernel, , 8)
    } else {
        ALQ_DISPATCH_CPB(block, al_encode_kernel, , 16)
    }
#undef LAUNCH
    return check_launch();
}

int al_decode(const void* codes, const float* meta, int64_t n, int block, int bits, float* out,
              void* stream) {
    if (n < 0) return ALQ_ERR_INVALID_ARG;
    if (!valid_block(block) || (bits != 8 && bits != 16)) return ALQ_ERR_UNSUPPORTED;
    if (n == 0) return ALQ_OK;
    if (!codes || !meta || !out) return ALQ_ERR_INVALID_ARG;
    if (!aligned(out, 16) || !aligned(codes, 16) || !aligned(meta, 8)) return ALQ_ERR_ALIGN;
    const int64_t ntiles = blocks_of(n, kTile);
    cudaStream_t s = (cudaStream_t)stream;
#define LAUNCH(k)                                                                      \
    k<<<grid_for(k, ntiles), kThreads, 0, s>>>(codes, meta, n, block, out, ntiles,         \
                                               Opaque2{make_float2(1.0f, 1.0f), make_float2(0.0f, 0.0f)})
    if (bits == 8) {
        ALQ_DISPATCH_CPB(block, al_decode_kernel, , 8)
    } else {
        ALQ_DISPATCH_CPB(block, al_decode_kernel, , 16)
    }
#undef LAUNCH
    return check_launch();
}

int uf8_encode(const float* m, int64_t n, int block, int8_t* codes, float* absmax, void* stream) {
    if (n < 0) return ALQ_ERR_INVALID_ARG;
    if (!valid_block(block)) return ALQ_ERR_UNSUPPORTED;
    if (n == 0) return ALQ_OK;
    if (!m || !codes || !absmax) return ALQ_ERR_INVALID_ARG;
    if (!aligned(m, 16) || !aligned(codes, 16) || !aligned(absmax, 4)) return ALQ_ERR_ALIGN;
    const int64_t ntiles = blocks_of(n, kTile);
    cudaStream_t s = (cudaStream_t)stream;
#define LAUNCH(k) k<<<grid_for(k, ntiles), kThreads, 0, s>>>(m, n, block, codes, absmax, ntiles)
    ALQ_DISPATCH_CPB(block, uf8_encode_kernel, )
#undef LAUNCH
    return check_launch();
}

int uf8_decode(const int8_t* codes, const float* absmax, int64_t n, int block, float* out,
               void* stream) {
    if (n < 0) return ALQ_ERR_INVALID_ARG;
    if (!valid_block(block)) return ALQ_ERR_UNSUPPORTED;
    if (n == 0) return ALQ_OK;
    if (!codes || !absmax || !out) return ALQ_ERR_INVALID_ARG;
    if (!aligned(out, 16) || !aligned(codes, 16) || !aligned(absmax, 4)) return ALQ_ERR_ALIGN;
    const int64_t ntiles = blocks_of(n, kTile);
    cudaStream_t s = (cudaStream_t)stream;
#define LAUNCH(k) k<<<grid_for(k, ntiles), kThreads, 0, s>>>(codes, absmax, n, block, out, ntiles)
    ALQ_DISPATCH_CPB(block, uf8_decode_kernel, )
#undef LAUNCH
    return check_launch();
}

}  // extern "C"
