// alq_apollo.cu -- APOLLO step with quantized projected moments (Sec. 3.1:
// moments in a low-rank projected space give a channel-wise scale applied to
// the original gradient; rank 256, channel-wise scaling in Sec. 6.1).
//
// Launch sequence of one step:
//   project   R = bf16(G) * P^T on the tensor cores, one persistent CTA per
//             SM over 128-channel tiles: sixteen converter warps read G
//             (fp32, prefetched into L2 by TMA a few jobs ahead) and write
//             it as bf16 (round to nearest even) into a 4-stage shared-
//             memory ring in the 128-byte-swizzled K-major layout,
//             transposing when the channels are G's columns; TMA loads the
//             matching P tiles; one thread issues tcgen05.mma (bf16 x bf16 ->
//             fp32) into one of two 128 x rank accumulators in tensor
//             memory; four epilogue warps read the other back with
//             tcgen05.ld and write R [channels][rank].
//   moments   per channel (one quantization block = rank values): decode
//             UF8 M^P and AL8 V^P, Adam EMAs with bias correction, channel
//             norms of Rt and R (fp32 sums: they move p only) -> s_j,
//             re-encode.
//   limiter   (optional) ||G s|| and the norm-growth cap: sums of squares
//             per chunk of kNormChunk update tiles (a partition of each
//             matrix that does not depend on the grid), summed in chunk
//             order by the limiter kernel, so the grouped step limits every
//             matrix exactly as the single-matrix step does.
//   update    p = p (1 - lr wd) - (lr alpha) g s_j.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "alq_async.cuh"
// the level and bound passes' exp2/log2 tables from per-CTA shared copies
#define ALQ_SMEM_TABLES 1
#include "alq_kernels.cuh"

namespace alq {

constexpr int kGM = 128;      // UMMA M (rows of A per CTA)
constexpr int kGK = 64;       // K per stage (64 bf16 = one 128-byte swizzle row)
constexpr int kAStage = kGM * kGK * 2;     // 16 KB
constexpr int kBStage = 256 * kGK * 2;     // 32 KB (rank <= 256)

// ------------------------------------------------------------ workspace --
struct ApWs {
    float* R;        // [L][rank]
    float* scale;    // [L]
    double* npart;   // [norm_chunks(n)] limiter partials
    float* lim;      // [2]: limiter factor
    int* err;        // [1]: projection pipeline timeout flag
    size_t bytes;
};

// Limiter partials: one per chunk of kNormChunk update tiles of a matrix.
constexpr int kNormChunk = 8;
static __host__ __device__ int64_t norm_chunks(int64_t n) {
    return (((n + kTile - 1) / kTile) + kNormChunk - 1) / kNormChunk;
}

static size_t r256(size_t x) { return (x + 255) & ~(size_t)255; }

static ApWs ap_layout(void* base, int64_t rows, int64_t cols, int rank) {
    const int64_t s = rows <= cols ? rows : cols, L = rows <= cols ? cols : rows;
    ApWs w;
    size_t off = 0;
    char* p = (char*)base;
    auto take = [&](size_t b) {
        char* r = p ? p + off : nullptr;
        off += r256(b);
        return r;
    };
    (void)s;
    w.R = (float*)take(4 * (size_t)L * rank);
    w.scale = (float*)take(4 * (size_t)L);
    w.npart = (double*)take(8 * (size_t)norm_chunks(rows * cols));
    w.lim = (float*)take(8);
    w.err = (int*)take(4);
    w.bytes = off;
    return w;
}

int al_apollo_workspace(int64_t rows, int64_t cols, int rank, size_t* bytes) {
    *bytes = ap_layout(nullptr, rows, cols, rank).bytes;
    return ALQ_OK;
}

// ------------------------------------------------------ PTX primitives --
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"((uint64_t)map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// L2 prefetch of one box of a tensor map (no shared memory, no barrier).
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap* map, int x, int y) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global [%0, {%1, %2}];" ::"l"((uint64_t)map),
                 "r"(x), "r"(y)
                 : "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile stored in the
// 128-byte-swizzled layout TMA writes: rows of 128 bytes, 8-row groups 1024
// bytes apart (SBO), descriptor version 1, swizzle mode 128B.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr) {
    uint64_t d = (uint64_t)((addr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;            // LBO (not used by swizzled K-major layouts)
    d |= (uint64_t)(1024 >> 4) << 32;  // SBO
    d |= (uint64_t)1 << 46;            // descriptor version
    d |= (uint64_t)2 << 61;            // 128-byte swizzle
    return d;
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                          uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
        "%28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Instruction descriptor of tcgen05.mma kind::f16: bf16 A and B (K-major),
// fp32 accumulator, M x N.
__host__ __device__ constexpr uint32_t umma_idesc_bf16(int M, int N) {
    return (1u << 4)                         // D format: f32
           | (1u << 7)                       // A format: bf16
           | (1u << 10)                      // B format: bf16
           | ((uint32_t)(N >> 3) << 17)      // N / 8
           | ((uint32_t)(M >> 4) << 24);     // M / 16
}

// ---------------------------------------------------------- projection --
struct GemmArgs {     // G as the projection's operand
    const float* g;   // G [rows][cols] fp32
    int64_t cols;     // row pitch of G
    int64_t K;        // short side s: the reduction length
    int L;            // channels (the long side)
    int kblocks;      // K blocks of 64
    int rows_short;   // channels are G's columns (rows <= cols)
};

// bf16 (round to nearest even) of two values, lo in the low half.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&b);
}

// One converter warp's share (256 / NW values per lane, NW converter
// warps) of K block kb of the 128-channel tile at m0. Channels are G's rows
// (RS false: K contiguous; warp c takes tile rows (128 / NW) c onwards, two
// rows per load, 16 lanes x 16 bytes along K) or G's columns (RS true: K
// strided; warp c takes K rows (64 / NW) c onwards, lane l the channels
// l + 32 q, each load a 128-byte row slice). Outside G the values are 0.
template <bool RS, int NW>
__device__ __forceinline__ void conv_load(const GemmArgs& a, int m0, int kb, int c, int lane,
                                          float (&v)[256 / NW]) {
    if constexpr (!RS) {
        const int64_t k = (int64_t)kb * kGK + 4 * (lane & 15);
#pragma unroll
        for (int i = 0; i < 64 / NW; ++i) {
            const int64_t j = m0 + (128 / NW) * c + 2 * i + (lane >> 4);
            float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
            if (j < a.L && k < a.K) x = __ldcs(reinterpret_cast<const float4*>(a.g + j * a.cols + k));
            v[4 * i] = x.x;
            v[4 * i + 1] = x.y;
            v[4 * i + 2] = x.z;
            v[4 * i + 3] = x.w;
        }
    } else {
        constexpr int KR = 64 / NW;  // K rows of a warp
#pragma unroll
        for (int kk = 0; kk < KR; ++kk) {
            const int64_t k = (int64_t)kb * kGK + KR * c + kk;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int64_t j = m0 + lane + 32 * q;
                v[KR * q + kk] = (k < a.K && j < a.L) ? __ldcs(a.g + k * a.cols + j) : 0.0f;
            }
        }
    }
}

// The same share as bf16 into an operand stage in the layout a 128-byte
// swizzled TMA load writes (row r of 128 bytes, 16-byte chunk x stored at
// chunk x ^ (r & 7)): K-major, as the MMA's shared-memory descriptor reads.
template <bool RS, int NW>
__device__ __forceinline__ void conv_store(uint8_t* sa, int c, int lane,
                                           const float (&v)[256 / NW]) {
    if constexpr (!RS) {
        const int kq = lane & 15;
#pragma unroll
        for (int i = 0; i < 64 / NW; ++i) {
            const int r = (128 / NW) * c + 2 * i + (lane >> 4);
            const uint2 w = make_uint2(pack_bf16x2(v[4 * i], v[4 * i + 1]),
                                       pack_bf16x2(v[4 * i + 2], v[4 * i + 3]));
            *reinterpret_cast<uint2*>(sa + r * 128 + (((kq >> 1) ^ (r & 7)) << 4) + ((kq & 1) << 3)) = w;
        }
    } else {
        constexpr int KR = 64 / NW;  // K rows of a warp: 2 KR bytes of each 128-byte row
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int r = lane + 32 * q;
            const float* x = v + KR * q;
            if constexpr (KR == 16) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const float* y = x + 8 * h;
                    const uint4 w = make_uint4(pack_bf16x2(y[0], y[1]), pack_bf16x2(y[2], y[3]),
                                               pack_bf16x2(y[4], y[5]), pack_bf16x2(y[6], y[7]));
                    *reinterpret_cast<uint4*>(sa + r * 128 + (((2 * c + h) ^ (r & 7)) << 4)) = w;
                }
            } else if constexpr (KR == 8) {
                const uint4 w = make_uint4(pack_bf16x2(x[0], x[1]), pack_bf16x2(x[2], x[3]),
                                           pack_bf16x2(x[4], x[5]), pack_bf16x2(x[6], x[7]));
                *reinterpret_cast<uint4*>(sa + r * 128 + ((c ^ (r & 7)) << 4)) = w;
            } else {
                static_assert(KR == 4, "4, 8 or 16 converter warps");
                const uint2 w = make_uint2(pack_bf16x2(x[0], x[1]), pack_bf16x2(x[2], x[3]));
                *reinterpret_cast<uint2*>(sa + r * 128 + (((c >> 1) ^ (r & 7)) << 4) + ((c & 1) << 3)) = w;
            }
        }
    }
}

// ------------------------------------------------------------- moments --
// Projected Adam moments, one quantization block per channel (block = rank).
struct MomentArgs {
    const float* R;
    int64_t n;  // L * rank
    int8_t* m_codes;
    float* m_absmax;
    void* v_codes;
    float* v_meta;
    int block;
    float* scale;
    float beta1, beta2, omb1, omb2, ic1, c2, eps, log_floor;
    float one;   // 1 and 0, opaque to the compiler: f * one + c rounds as
    float zero;  // f + c, fma(x, y, zero) as x y
};

// Geometry of the moments pass: a warp owns a 512-element segment (four
// 4-element chunks per lane, 128 elements apart), so two rank-256 channels
// (or four rank-128 channels), their levels two channels per paired pass; a
// CTA owns a 4096-element tile (16 values a lane: 2.997 against 3.018 ms per
// grouped step with 8).
constexpr int kMCH = 4;
constexpr int kMSeg = 128 * kMCH;
constexpr int kMTile = 8 * kMSeg;

// One tile of the moments pass. tab and vals are this warp's shared slots
// for the AL8 decode tables (NB * 32 pairs) and the blocks' 256 decoded
// values (NB * 256); lane 0 writes the blocks' channel scales.
template <int CPB, int VBITS>
__device__ __forceinline__ void moments_tile(const MomentArgs& m, int64_t tile, float2* tab,
                                             float* vals) {
    constexpr int NB = kMCH / CPB;
    constexpr int NE = 4 * kMCH;
    constexpr float Lm2 = VBITS == 8 ? 254.0f : 65534.0f;
    const int warp = __shfl_sync(0xFFFFFFFFu, (int)(threadIdx.x >> 5), 0), lane = threadIdx.x & 31;
    const float kf = al8_table_k(lane);
    const int bshift = block_shift<CPB, kMCH>(m.block);  // rank = 128 CPB
    const int64_t nblk = (m.n + (1 << bshift) - 1) >> bshift;
    const int64_t seg0 = tile * kMTile + (int64_t)warp * kMSeg;
    const int64_t b0 = seg0 >> bshift;
    float4 r[kMCH];
    uint32_t mw[kMCH], vw[kMCH * VBITS / 8];
    const bool full = seg0 + kMSeg <= m.n;  // warp-uniform: unmasked I/O
    if (full) {
#pragma unroll
        for (int c = 0; c < kMCH; ++c) {
            const int64_t idx = chunk_index(seg0, c, lane);
            r[c] = __ldcs(reinterpret_cast<const float4*>(m.R + idx));
            mw[c] = __ldcs(reinterpret_cast<const unsigned int*>((const uint8_t*)m.m_codes + idx));
            if constexpr (VBITS == 8) {
                vw[c] = __ldcs(reinterpret_cast<const unsigned int*>((const uint8_t*)m.v_codes + idx));
            } else {
                const uint2 h = __ldcs(reinterpret_cast<const uint2*>((const uint16_t*)m.v_codes + idx));
                vw[2 * c] = h.x;
                vw[2 * c + 1] = h.y;
            }
        }
    } else {
#pragma unroll
        for (int c = 0; c < kMCH; ++c) {
            const int64_t idx = chunk_index(seg0, c, lane);
            r[c] = load4f(m.R, idx, m.n);
            mw[c] = load4b((const uint8_t*)m.m_codes, idx, m.n);
            if constexpr (VBITS == 8) {
                vw[c] = load4b((const uint8_t*)m.v_codes, idx, m.n);
            } else {
                const uint2 h = load4h((const uint16_t*)m.v_codes, idx, m.n);
                vw[2 * c] = h.x;
                vw[2 * c + 1] = h.y;
            }
        }
    }
    float olmin[NB], odelta[NB], dm[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        float2 mt = make_float2(0.f, 0.f);
        float sa = 0.0f;
        if (b0 + b < nblk) {
            mt = __ldg(reinterpret_cast<const float2*>(m.v_meta) + b0 + b);
            sa = __ldg(m.m_absmax + b0 + b);
        }
        olmin[b] = mt.x;
        odelta[b] = mt.y;
        dm[b] = sa / 127.0f;
    }
    // previous V: AL8 through the blocks' tables of exactly rounded values
    float vh[NE];
    if constexpr (VBITS == 8) {
        float* ts = reinterpret_cast<float*>(tab);  // 64 floats per block (SoA)
        if constexpr (NB >= 2) {
            const Opaque2 ok2{make_float2(m.one, m.one), make_float2(m.zero, m.zero)};
#pragma unroll
            for (int b = 0; b < NB; b += 2)
                al8_build_tables2_soa(ts + 64 * b, ts + 64 * (b + 1), olmin[b], odelta[b],
                                      olmin[b + 1], odelta[b + 1], kf, ok2);
        } else {
            al8_build_tables_soa(ts, olmin[0], odelta[0], kf);
        }
#pragma unroll
        for (int b = 0; b < NB; ++b)
            al8_values_from_tables_soa(vals + 256 * b, ts + 64 * b, olmin[b], odelta[b]);
#pragma unroll
        for (int e = 0; e < NE; ++e)
            vh[e] = vals[256 * (e / 4 / CPB) + ((vw[e / 4] >> (8 * (e % 4))) & 0xFFu)];
    } else {
#pragma unroll
        for (int e = 0; e < NE; ++e)
            vh[e] = al16_decode(code_of<VBITS>(vw, e / 4, e % 4), olmin[e / 4 / CPB],
                                odelta[e / 4 / CPB]);
    }
    // Moments and channel norms on pairs of elements (paired fp32
    // instructions, each component rounded as the scalar operation; a sum
    // of two rounded products is a fused multiply-add by the opaque one, so
    // that no product is contracted into it). The channel norms, like the
    // bias-corrected ratio they measure, move only the parameters: fp32
    // sums of squares (relative error below 2^-19 over a channel).
    const float2 one = make_float2(m.one, m.one);
    const float2 b1 = make_float2(m.beta1, m.beta1), o1 = make_float2(m.omb1, m.omb1);
    const float2 b2 = make_float2(m.beta2, m.beta2), o2 = make_float2(m.omb2, m.omb2);
    const float2 ic1 = make_float2(m.ic1, m.ic1), c2 = make_float2(m.c2, m.c2);
    const float2 eps = make_float2(m.eps, m.eps);
    float vf[NE];
    float2 mf2[NE / 2];
    uint32_t cvmin[kMCH], cvmax[kMCH];
    float cmabs[kMCH];
    float2 nr2[NB], ng2[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) nr2[b] = ng2[b] = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int c = 0; c < kMCH; ++c) {
        const int b = c / CPB;
        const float2 dm2 = make_float2(dm[b], dm[b]);
        const uint32_t mx = mw[c] ^ 0x80808080u;
        cvmin[c] = 0xFFFFFFFFu;
        cvmax[c] = 0u;
        cmabs[c] = 0.0f;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            // momentum bytes as exact floats (see s8_to_float)
            const float2 qf = make_float2(u2f(__byte_perm(mx, 0x4B400000u, 0x7640u | (2 * i))),
                                          u2f(__byte_perm(mx, 0x4B400000u, 0x7640u | (2 * i + 1))));
            const float2 mh = mul2(add2(qf, make_float2(-12583040.0f, -12583040.0f)), dm2);
            const float2 rv = i == 0 ? make_float2(r[c].x, r[c].y) : make_float2(r[c].z, r[c].w);
            const float2 vh2 = make_float2(vh[4 * c + 2 * i], vh[4 * c + 2 * i + 1]);
            const float2 mq = fma2(mul2(b1, mh), one, mul2(o1, rv));
            const float2 vq = fma2(mul2(b2, vh2), one, mul2(o2, mul2(rv, rv)));
            // the bias-corrected ratio feeds only the channel scales (so
            // only p): approximate square root and reciprocal
            const float2 den = fma2(mul2(make_float2(sqrt_approx(vq.x), sqrt_approx(vq.y)), c2), one, eps);
            const float2 num = mul2(mq, ic1);
            const float2 rt = mul2(num, make_float2(rcp_approx(den.x), rcp_approx(den.y)));
            mf2[2 * c + i] = mq;
            vf[4 * c + 2 * i] = vq.x;
            vf[4 * c + 2 * i + 1] = vq.y;
            nr2[b] = fma2(rt, rt, nr2[b]);
            ng2[b] = fma2(rv, rv, ng2[b]);
            const uint32_t vbx = f2u(vq.x), vby = f2u(vq.y);
            cvmin[c] = umix<false>(cvmin[c], umix<false>(vbx - 1u, vby - 1u));
            cvmax[c] = umix<true>(cvmax[c], umix<true>(vbx, vby));
            cmabs[c] = fmaxf(cmabs[c], fmaxf(fabsf(mq.x), fabsf(mq.y)));
        }
    }
    float nrs[NB], ngs[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        nrs[b] = nr2[b].x + nr2[b].y;
        ngs[b] = ng2[b].x + ng2[b].y;
    }
    uint32_t cmabs_u[kMCH];
#pragma unroll
    for (int c = 0; c < kMCH; ++c) cmabs_u[c] = f2u(cmabs[c]);
    uint32_t bvmin[NB], bvmax[NB], bmabs[NB];
    warp_blocks_reduce<CPB, false>(cvmin, bvmin);
    warp_blocks_reduce<CPB, true>(cvmax, bvmax);
    warp_blocks_reduce<CPB, true>(cmabs_u, bmabs);
#pragma unroll
    for (int k = 16; k >= 1; k >>= 1) {
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            nrs[b] += __shfl_xor_sync(0xFFFFFFFFu, nrs[b], k);
            ngs[b] += __shfl_xor_sync(0xFFFFFFFFu, ngs[b], k);
        }
    }
    float vmn[NB], vmx[NB], nlmin[NB], ndelta[NB], ms[NB], sc[NB], inv[NB];
    AlEncConsts ek[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        vmn[b] = u2f(bvmin[b] + 1u);
        vmx[b] = u2f(bvmax[b]);
        ms[b] = u2f(bmabs[b]);
        uf8_encode_consts(ms[b] > 0.0f ? ms[b] : 1.0f, sc[b], inv[b]);
        inv[b] = ms[b] > 0.0f ? inv[b] : 0.0f;  // an all-zero block codes as 0
    }
    // (m sc) inv: sc is 1 except in blocks whose absmax is below 2^-120
#pragma unroll
    for (int c = 0; c < kMCH; ++c) {
        const int b = c / CPB;
        if (__builtin_expect(sc[b] != 1.0f, 0)) {
            const float2 s2 = make_float2(sc[b], sc[b]);
            mf2[2 * c] = mul2(mf2[2 * c], s2);
            mf2[2 * c + 1] = mul2(mf2[2 * c + 1], s2);
        }
    }
    al_blocks_params<NB>(vmn, vmx, m.log_floor, nlmin, ndelta);
#pragma unroll
    for (int b = 0; b < NB; ++b) ek[b] = al_encode_consts(nlmin[b], ndelta[b], Lm2);
    uint32_t qv[NE];
    al_encode_chunks<VBITS, CPB, NB, kMCH, true>(vf, vmn, nlmin, ndelta, ek, qv);
#pragma unroll
    for (int c = 0; c < kMCH; ++c) {
        const int b = c / CPB;
        const int64_t idx = chunk_index(seg0, c, lane);
        // q = rint((m sc) inv) as the low byte of 1.5 * 2^23 + q (two's
        // complement for q < 0); the rounding add by the opaque one
        const float2 inv2 = make_float2(inv[b], inv[b]);
        uint32_t rb[4];
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const float2 f = mul2(mf2[2 * c + i], inv2);
            const float2 rr = fma2(f, one, make_float2(12582912.0f, 12582912.0f));
            rb[2 * i] = f2u(rr.x);
            rb[2 * i + 1] = f2u(rr.y);
        }
        const uint32_t qm = __byte_perm(__byte_perm(rb[0], rb[1], 0x0040u),
                                        __byte_perm(rb[2], rb[3], 0x0040u), 0x5410u);
        if (full) {
            __stcs(reinterpret_cast<unsigned int*>((uint8_t*)m.m_codes + idx), qm);
            if constexpr (VBITS == 8)
                __stcs(reinterpret_cast<unsigned int*>((uint8_t*)m.v_codes + idx),
                       qv[4 * c] | (qv[4 * c + 1] << 8) | (qv[4 * c + 2] << 16) | (qv[4 * c + 3] << 24));
            else
                __stcs(reinterpret_cast<uint2*>((uint16_t*)m.v_codes + idx),
                       make_uint2(qv[4 * c] | (qv[4 * c + 1] << 16), qv[4 * c + 2] | (qv[4 * c + 3] << 16)));
        } else {
            store4b((uint8_t*)m.m_codes, idx, m.n, qm);
            if constexpr (VBITS == 8)
                store4b((uint8_t*)m.v_codes, idx, m.n,
                        qv[4 * c] | (qv[4 * c + 1] << 8) | (qv[4 * c + 2] << 16) | (qv[4 * c + 3] << 24));
            else
                store4h((uint16_t*)m.v_codes, idx, m.n,
                        make_uint2(qv[4 * c] | (qv[4 * c + 1] << 16), qv[4 * c + 2] | (qv[4 * c + 3] << 16)));
        }
    }
    if (lane == 0) {
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            if (b0 + b >= nblk) continue;
            reinterpret_cast<float2*>(m.v_meta)[b0 + b] = make_float2(nlmin[b], ndelta[b]);
            m.m_absmax[b0 + b] = ms[b];
        }
    }
    // s_j = ||Rt_j|| / (||R_j|| + 1e-8)
    if (lane == 0) {
#pragma unroll
        for (int b = 0; b < NB; ++b)
            if (b0 + b < nblk) m.scale[b0 + b] = sqrtf(nrs[b]) / (sqrtf(ngs[b]) + 1e-8f);
    }
    __syncwarp();
}

template <int CPB, int VBITS>
__global__ void __launch_bounds__(kThreads, 3)
apollo_moments_kernel(MomentArgs m, int64_t ntiles) {
    constexpr int NB = kMCH / CPB;
    __shared__ __align__(16) float2 s_tab[kThreads / 32][NB * 32];
    __shared__ float s_val[kThreads / 32][VBITS == 8 ? NB * 256 : 1];
    const int warp = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < 1024; i += kThreads) {
        s_kExp2Hi[i] = kExp2HiD[i];
        s_kExp2Lo[i] = kExp2LoD[i];
        s_kLog2C[i] = kLog2CD[i];
        s_kLog2Hi[i] = kLog2HiD[i];
        s_kLog2Lo[i] = kLog2LoD[i];
    }
    __syncthreads();
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x)
        moments_tile<CPB, VBITS>(m, tile, s_tab[warp], s_val[warp]);
}

// ------------------------------------------------------ limiter, update --
struct ApUpdateArgs {
    float* p;
    const float* g;
    int64_t n;
    Divider dv;
    int rows_short;  // 1: channel = column; 0: channel = row
    const float* scale;
    const float* lim;  // nullptr when the limiter is off
    float decay, lr_a;
};

// Sum of (g s_j)^2 over chunk `chunk` (update tiles chunk * kNormChunk ..
// + kNormChunk - 1 of a matrix of ntiles tiles), computed by the whole CTA
// in a fixed order (each warp its segments tile by tile in two-float, the
// warps merged in order in double) and written to part[chunk]. s_w holds
// kThreads / 32 doubles; every thread of the CTA calls this.
__device__ __forceinline__ void gnorm_chunk(const ApUpdateArgs& u, int64_t chunk, int64_t ntiles,
                                            double* __restrict__ part, double* s_w) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float hi = 0.0f, lo = 0.0f;
    const int64_t t1 = min(ntiles, (chunk + 1) * kNormChunk);
    for (int64_t tile = chunk * kNormChunk; tile < t1; ++tile) {
        const int64_t seg0 = tile * kTile + (int64_t)warp * kSeg;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int64_t idx = chunk_index(seg0, c, lane);
            if (idx >= u.n) continue;
            const uint32_t row = divide((uint32_t)idx, u.dv);
            const uint32_t col = (uint32_t)idx - row * u.dv.d;
            const float4 gv = __ldcs(reinterpret_cast<const float4*>(u.g + idx));
            float4 sv;
            if (u.rows_short) {
                sv = __ldg(reinterpret_cast<const float4*>(u.scale + col));
            } else {
                const float sc = __ldg(u.scale + row);
                sv = make_float4(sc, sc, sc, sc);
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float gt = f4get(gv, j) * f4get(sv, j);
                float h, l;
                two_prod(gt, gt, h, l);
                ff_acc(hi, lo, h, l);
            }
        }
    }
    ff_warp_sum(hi, lo);
    __syncthreads();  // s_w of the previous chunk has been read
    if (lane == 0) s_w[warp] = (double)hi + (double)lo;
    __syncthreads();
    if (threadIdx.x == 0) {
        double sum = 0.0;
        for (int w = 0; w < kThreads / 32; ++w) sum += s_w[w];
        part[chunk] = sum;
    }
}

__global__ void __launch_bounds__(kThreads)
apollo_gnorm_kernel(ApUpdateArgs u, int64_t ntiles, int64_t nchunks, double* __restrict__ part) {
    __shared__ double s_w[kThreads / 32];
    for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x) gnorm_chunk(u, c, ntiles, part, s_w);
}

// The limiter of one matrix from its chunk partials (summed in chunk order):
// ||G s|| against gamma times the previous norm.
__device__ __forceinline__ void limit_one(const double* __restrict__ part, int64_t nparts,
                                          float gamma, float* __restrict__ prev_norm,
                                          float* __restrict__ lim) {
    double ss = 0.0;
    for (int64_t i = 0; i < nparts; ++i) ss += part[i];
    const double nt = sqrt(ss);
    const double prev = (double)*prev_norm;
    const double cap = (double)gamma * prev;
    if (prev > 0.0 && nt > cap) {
        lim[0] = (float)(cap / nt);
        *prev_norm = (float)cap;
    } else {
        lim[0] = 1.0f;
        *prev_norm = (float)nt;
    }
}

__global__ void apollo_limit_kernel(const double* __restrict__ part, int64_t nparts, float gamma,
                                    float* __restrict__ prev_norm, float* __restrict__ lim) {
    if (threadIdx.x == 0) limit_one(part, nparts, gamma, prev_norm, lim);
}

// One tile (kTile parameters) of p = p (1 - lr wd) - (lr alpha) lim (g s_j).
__device__ __forceinline__ void update_tile(const ApUpdateArgs& u, int64_t tile, float lim) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    {
        const int64_t seg0 = tile * kTile + (int64_t)warp * kSeg;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int64_t idx = chunk_index(seg0, c, lane);
            if (idx >= u.n) continue;
            const uint32_t row = divide((uint32_t)idx, u.dv);
            const uint32_t col = (uint32_t)idx - row * u.dv.d;
            const float4 gv = __ldcs(reinterpret_cast<const float4*>(u.g + idx));
            const float4 pv = __ldcs(reinterpret_cast<const float4*>(u.p + idx));
            float4 sv;
            if (u.rows_short) {
                sv = __ldg(reinterpret_cast<const float4*>(u.scale + col));
            } else {
                const float s = __ldg(u.scale + row);
                sv = make_float4(s, s, s, s);
            }
            float pn[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float gt = f4get(gv, j) * f4get(sv, j);
                if (u.lim) gt = gt * lim;
                pn[j] = f4get(pv, j) * u.decay - u.lr_a * gt;
            }
            __stcs(reinterpret_cast<float4*>(u.p + idx), make_float4(pn[0], pn[1], pn[2], pn[3]));
        }
    }
}

__global__ void __launch_bounds__(kThreads)
apollo_update_kernel(ApUpdateArgs u, int64_t ntiles) {
    const float lim = u.lim ? __ldg(u.lim) : 1.0f;
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) update_tile(u, tile, lim);
}

// ------------------------------------------------------- grouped step --
// Plan of a grouped step: a header, then one 64-byte-aligned entry per
// matrix (its TMA descriptors first), then the projection tile -> matrix map.
constexpr uint32_t kApPlanMagic = 0x41504C31u;  // "APL1"

struct ApPlanHeader {
    uint32_t magic;
    int32_t nmat, rank, v_bits;
    int64_t gemm_tiles, mom_tiles, upd_tiles;
    int64_t total_params, total_channels;
    int64_t norm_chunks;
    int32_t limiter_ok, reserved0;
    int64_t reserved;
};
static_assert(sizeof(ApPlanHeader) == 80, "plan header layout");

struct ApEntry {  // aligned as CUtensorMap (at least 64 bytes)
    CUtensorMap tmB;  // bf16 P [rank][s], box [rank][64]
    CUtensorMap tmG;  // fp32 G, box = one 128-channel x 64-K projection job (L2 prefetch)
    float* p;
    const float* g;
    int8_t* m_codes;
    float* m_absmax;
    void* v_codes;
    float* v_meta;
    float* R;
    float* scale;
    int64_t rows, cols, n, L, s, npj;
    Divider dv;
    int32_t rows_short, kblocks;
    int64_t gemm_t0, mom_t0, upd_t0;  // first tile of each pass
    int64_t nrm_t0;                   // first limiter chunk
    double* npart;                    // limiter partials [norm_chunks(n)]
    float* lim;                       // limiter factor
    float* prev_norm;                 // previous update norm (device scalar)
};

constexpr size_t kApEntryOffset = 128;  // header rounded up to the entry alignment
static_assert(kApEntryOffset % alignof(ApEntry) == 0 && sizeof(ApEntry) % 64 == 0,
              "plan entries keep their tensor maps 64-byte aligned");

__device__ __forceinline__ int entry_for(const ApEntry* __restrict__ tab, int nmat, int64_t tile,
                                         int cur, int64_t ApEntry::*t0) {
    while (cur + 1 < nmat && tab[cur + 1].*t0 <= tile) ++cur;
    return cur;
}

// ----------------------------------------------------------- projection --
// R = bf16(G) P^T by a persistent kernel: one CTA per SM walks 128-channel
// tiles with a stride of the grid. Each tile is kblocks jobs of 64 K; a job
// is one 4-stage ring slot holding the tile's G slice as bf16 (converted by
// the converter warps) and P's slice (a TMA load). The ring's stages and
// phases run on across tiles, and the two accumulators in tensor memory
// alternate between tiles, so the epilogue of one tile overlaps the operand
// stream of the next. Warp 0 issues the TMA loads of P and an L2 prefetch of
// G kPrefetch jobs ahead (so that the converters' loads hit L2), warp 1 the
// MMAs, warps 2 .. 1 + kPConv convert G, the last kPEpi warps drain the
// accumulators into R.
constexpr int kPStages = 4;
constexpr int kPrefetch = 4;  // G jobs prefetched into L2 ahead of the P loads
constexpr int kPConv = 16;
constexpr int kPEpi = 4;
constexpr int kPThreads = 64 + 32 * (kPConv + kPEpi);
constexpr int kPSmem = kPStages * (kAStage + kBStage) + 1024 + 256;
constexpr int kPV = 256 / kPConv;  // values per converter lane and job

// Matrix of tile t: from the plan's tile map, or the one matrix of a
// single-matrix launch.
template <bool kOne>
__device__ __forceinline__ const ApEntry* tile_entry(const ApEntry* tab,
                                                     const uint16_t* __restrict__ tile_mat,
                                                     int64_t t) {
    return kOne ? tab : tab + tile_mat[t];
}

// One (tile, K block) job of a converter warp's walk.
struct PJob {
    GemmArgs a;
    int m0, kb;
    bool valid;
};

template <bool kOne>
__device__ __forceinline__ PJob pjob_at(const ApEntry* tab, const uint16_t* __restrict__ tile_mat,
                                        int64_t ntiles, int64_t t) {
    PJob j;
    j.valid = t < ntiles;
    j.kb = 0;
    j.m0 = 0;
    if (j.valid) {
        const ApEntry* e = tile_entry<kOne>(tab, tile_mat, t);
        j.a = GemmArgs{e->g, e->cols, e->s, (int)e->L, e->kblocks, e->rows_short};
        j.m0 = (int)(t - e->gemm_t0) * kGM;
    }
    return j;
}

__device__ __forceinline__ void pjob_load(const PJob& j, int c, int lane, float (&v)[kPV]) {
    if (j.a.rows_short) conv_load<true, kPConv>(j.a, j.m0, j.kb, c, lane, v);
    else conv_load<false, kPConv>(j.a, j.m0, j.kb, c, lane, v);
}

// Job kc of the walk into its ring slot: wait until the MMAs that read the
// slot's previous contents retired, write it, make the writes visible to the
// tensor cores and arrive (one arrival per converter warp).
__device__ __forceinline__ bool pjob_stage(const PJob& j, const float (&v)[kPV], uint32_t kc,
                                           uint8_t* sA, uint32_t afull0, uint32_t empty0, int c,
                                           int lane) {
    const uint32_t s = kc % kPStages;
    if (kc >= (uint32_t)kPStages && !mbar_wait(empty0 + 8 * s, ((kc / kPStages) - 1) & 1))
        return false;
    if (j.a.rows_short) conv_store<true, kPConv>(sA + s * kAStage, c, lane, v);
    else conv_store<false, kPConv>(sA + s * kAStage, c, lane, v);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(afull0 + 8 * s);
    return true;
}

// A converter warp's walk: the loads of the next job (the next K block, or
// the first of the next tile) are issued before the current job is stored
// (two register buffers used in turn).
template <bool kOne>
__device__ __forceinline__ bool pconv_walk(const ApEntry* tab, const uint16_t* __restrict__ tile_mat,
                                           int64_t ntiles, uint8_t* sA, uint32_t afull0,
                                           uint32_t empty0, int c, int lane) {
    const int64_t G = gridDim.x;
    int64_t t = blockIdx.x;
    PJob ja = pjob_at<kOne>(tab, tile_mat, ntiles, t), jb;
    float va[kPV], vb[kPV];
    if (!ja.valid) return true;
    pjob_load(ja, c, lane, va);
    uint32_t kc = 0;
    for (;;) {
        if (ja.kb + 1 < ja.a.kblocks) {
            jb = ja;
            ++jb.kb;
        } else {
            t += G;
            jb = pjob_at<kOne>(tab, tile_mat, ntiles, t);
        }
        if (jb.valid) pjob_load(jb, c, lane, vb);
        if (!pjob_stage(ja, va, kc++, sA, afull0, empty0, c, lane)) return false;
        if (!jb.valid) return true;
        if (jb.kb + 1 < jb.a.kblocks) {
            ja = jb;
            ++ja.kb;
        } else {
            t += G;
            ja = pjob_at<kOne>(tab, tile_mat, ntiles, t);
        }
        if (ja.valid) pjob_load(ja, c, lane, va);
        if (!pjob_stage(jb, vb, kc++, sA, afull0, empty0, c, lane)) return false;
        if (!ja.valid) return true;
    }
}

// kOne: a single matrix whose descriptor (tensor maps included) is the
// kernel parameter `one`; otherwise the plan's table `tab` and tile map.
template <bool kOne>
__global__ void __launch_bounds__(kPThreads, 1)
apollo_project_kernel(const ApEntry* __restrict__ plan_tab, const uint16_t* __restrict__ tile_mat,
                      int64_t ntiles, int rank, int* err, const __grid_constant__ ApEntry one) {
    extern __shared__ uint8_t smem_raw[];
    const ApEntry* tab = kOne ? &one : plan_tab;
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sA = smem;
    uint8_t* sB = smem + kPStages * kAStage;
    // bfull, afull, empty per stage; tfull, tempty per accumulator
    uint64_t* bars = (uint64_t*)(sB + kPStages * kBStage);
    uint32_t* tmem_slot = (uint32_t*)(bars + 3 * kPStages + 4);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t bfull0 = smem_u32(bars), afull0 = smem_u32(bars + kPStages);
    const uint32_t empty0 = smem_u32(bars + 2 * kPStages);
    const uint32_t tfull0 = smem_u32(bars + 3 * kPStages), tempty0 = tfull0 + 16;
    const uint32_t acc_cols = rank <= 128 ? 128u : 256u;
    const uint32_t ncols = 2 * acc_cols;
    const int64_t G = gridDim.x;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kPStages; ++s) {
            mbar_init(bfull0 + 8 * s, 1);
            mbar_init(afull0 + 8 * s, kPConv);
            mbar_init(empty0 + 8 * s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(tfull0 + 8 * b, 1);
            mbar_init(tempty0 + 8 * b, kPEpi);
        }
        mbar_init_fence();
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(ncols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;
    const uint32_t b_bytes = (uint32_t)rank * kGK * 2;

    bool ok = true;
    if (warp == 0) {
        if (lane == 0) {
            // TMA producer of P: stage s is refilled once the MMAs that read
            // it retire
            // and L2 prefetcher of G: the job kPrefetch ahead of the one
            // whose P it loads (tile pt, K block pkb) is fetched into L2, so
            // that the converter warps' loads of it hit L2
            uint32_t kc = 0;
            const ApEntry* last = nullptr;
            int64_t pt = blockIdx.x;
            int pkb = 0;
            const ApEntry* pe = pt < ntiles ? tile_entry<kOne>(tab, tile_mat, pt) : nullptr;
            const ApEntry* plast = nullptr;
            auto prefetch_next = [&]() {
                if (!pe) return;
                if (!kOne && pe != plast) {
                    asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(
                                     &pe->tmG)
                                 : "memory");
                    plast = pe;
                }
                const int m0 = (int)(pt - pe->gemm_t0) * kGM;
                if (pe->rows_short) tma_prefetch_2d(&pe->tmG, m0, pkb * kGK);
                else tma_prefetch_2d(&pe->tmG, pkb * kGK, m0);
                if (++pkb == pe->kblocks) {
                    pkb = 0;
                    pt += G;
                    pe = pt < ntiles ? tile_entry<kOne>(tab, tile_mat, pt) : nullptr;
                }
            };
            for (int i = 0; i < kPrefetch; ++i) prefetch_next();
            for (int64_t t = blockIdx.x; t < ntiles && ok; t += G) {
                const ApEntry* e = tile_entry<kOne>(tab, tile_mat, t);
                if (!kOne && e != last) {
                    // a plan's descriptor was written through the generic
                    // proxy (a copy to device memory): make it visible to the
                    // tensor-map proxy
                    asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(
                                     &e->tmB)
                                 : "memory");
                    last = e;
                }
                const int kblocks = e->kblocks;
                for (int kb = 0; kb < kblocks; ++kb, ++kc) {
                    prefetch_next();
                    const uint32_t s = kc % kPStages;
                    if (kc >= (uint32_t)kPStages)
                        ok = mbar_wait(empty0 + 8 * s, ((kc / kPStages) - 1) & 1);
                    if (!ok) break;
                    mbar_expect_tx(bfull0 + 8 * s, b_bytes);
                    tma_load_2d(smem_u32(sB + s * kBStage), &e->tmB, kb * kGK, 0, bfull0 + 8 * s);
                }
            }
            if (!ok) {
                // a wait gave up: let this thread's copies in flight land
                // (bounded waits) before the CTA releases its shared memory
                for (uint32_t k = kc > (uint32_t)kPStages ? kc - kPStages : 0u; k < kc; ++k)
                    mbar_wait(bfull0 + 8 * (k % kPStages), (k / kPStages) & 1);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // MMA issuer: four K = 16 steps per stage, 32 bytes apart in the
            // row; accumulator it & 1 of tile number it
            const uint32_t idesc = umma_idesc_bf16(kGM, rank);
            uint32_t kc = 0, it = 0;
            for (int64_t t = blockIdx.x; t < ntiles && ok; t += G, ++it) {
                const int kblocks = tile_entry<kOne>(tab, tile_mat, t)->kblocks;
                const uint32_t acc = it & 1;
                if (it >= 2) ok = mbar_wait(tempty0 + 8 * acc, ((it / 2) - 1) & 1);
                if (!ok) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t d = tmem + acc * acc_cols;
                for (int kb = 0; kb < kblocks; ++kb, ++kc) {
                    const uint32_t s = kc % kPStages;
                    const uint32_t par = (kc / kPStages) & 1;
                    ok = mbar_wait(afull0 + 8 * s, par) && mbar_wait(bfull0 + 8 * s, par);
                    if (!ok) break;
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t a0 = smem_u32(sA + s * kAStage), b0 = smem_u32(sB + s * kBStage);
#pragma unroll
                    for (int k = 0; k < kGK / 16; ++k)
                        umma_bf16(d, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), idesc,
                                  (kb | k) != 0);
                    umma_commit(empty0 + 8 * s);
                }
                if (ok) umma_commit(tfull0 + 8 * acc);
            }
            if (!ok && kc > 0) {
                // a wait gave up: let the MMAs already issued retire
                // (bounded wait on the last commit) before the tensor memory
                // is released
                mbar_wait(empty0 + 8 * ((kc - 1) % kPStages), ((kc - 1) / kPStages) & 1);
            }
        }
    } else if (warp < 2 + kPConv) {
        ok = pconv_walk<kOne>(tab, tile_mat, ntiles, sA, afull0, empty0, warp - 2, lane);
    } else {
        // epilogue: a warp may read TMEM lanes 32 (warp % 4) .. + 31 (tile
        // rows), 32 columns at a time
        const int q = warp & 3;
        uint32_t it = 0;
        for (int64_t t = blockIdx.x; t < ntiles && ok; t += G, ++it) {
            const ApEntry* e = tile_entry<kOne>(tab, tile_mat, t);
            const uint32_t acc = it & 1;
            ok = mbar_wait(tfull0 + 8 * acc, (it / 2) & 1);
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const int64_t row = (t - e->gemm_t0) * kGM + q * 32 + lane;
            float* R = e->R;
            const int64_t L = e->L;
            for (int c0 = 0; c0 < rank; c0 += 32) {
                float v[32];
                if (ok) {
                    tmem_ld32(tmem + acc * acc_cols + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, v);
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = __int_as_float(0x7FC00000);  // NaN marks a failure
                }
                if (row < L) {
                    float4* dst = reinterpret_cast<float4*>(R + row * rank + c0);
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
        }
    }
    if (!ok) atomicExch(err, 1);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(ncols)
                     : "memory");
}

template <int CPB, int VBITS>
__global__ void __launch_bounds__(kThreads, 3)
apollo_moments_multi_kernel(const ApEntry* __restrict__ tab, int nmat, int64_t ntiles,
                            MomentArgs base) {
    constexpr int NB = kMCH / CPB;
    __shared__ __align__(16) float2 s_tab[kThreads / 32][NB * 32];
    __shared__ float s_val[kThreads / 32][VBITS == 8 ? NB * 256 : 1];
    const int warp = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < 1024; i += kThreads) {
        s_kExp2Hi[i] = kExp2HiD[i];
        s_kExp2Lo[i] = kExp2LoD[i];
        s_kLog2C[i] = kLog2CD[i];
        s_kLog2Hi[i] = kLog2HiD[i];
        s_kLog2Lo[i] = kLog2LoD[i];
    }
    __syncthreads();
    int cur = 0;
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        cur = entry_for(tab, nmat, tile, cur, &ApEntry::mom_t0);
        const ApEntry& e = tab[cur];
        MomentArgs m = base;
        m.R = e.R;
        m.n = e.npj;
        m.m_codes = e.m_codes;
        m.m_absmax = e.m_absmax;
        m.v_codes = e.v_codes;
        m.v_meta = e.v_meta;
        m.scale = e.scale;
        moments_tile<CPB, VBITS>(m, tile - e.mom_t0, s_tab[warp], s_val[warp]);
    }
}

// limited: every matrix's update is scaled by its limiter factor.
__global__ void __launch_bounds__(kThreads)
apollo_update_multi_kernel(const ApEntry* __restrict__ tab, int nmat, int64_t ntiles,
                           ApUpdateArgs base, int limited) {
    int cur = 0;
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        cur = entry_for(tab, nmat, tile, cur, &ApEntry::upd_t0);
        const ApEntry& e = tab[cur];
        ApUpdateArgs u = base;
        u.p = e.p;
        u.g = e.g;
        u.n = e.n;
        u.dv = e.dv;
        u.rows_short = e.rows_short;
        u.scale = e.scale;
        u.lim = limited ? e.lim : nullptr;
        update_tile(u, tile - e.upd_t0, limited ? __ldg(e.lim) : 1.0f);
    }
}

// Limiter partials of every matrix: one chunk per iteration, the chunks of
// all matrices in one launch.
__global__ void __launch_bounds__(kThreads)
apollo_gnorm_multi_kernel(const ApEntry* __restrict__ tab, int nmat, int64_t nchunks) {
    __shared__ double s_w[kThreads / 32];
    int cur = 0;
    for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x) {
        cur = entry_for(tab, nmat, c, cur, &ApEntry::nrm_t0);
        const ApEntry& e = tab[cur];
        ApUpdateArgs u{};
        u.g = e.g;
        u.n = e.n;
        u.dv = e.dv;
        u.rows_short = e.rows_short;
        u.scale = e.scale;
        gnorm_chunk(u, c - e.nrm_t0, (e.n + kTile - 1) / kTile, e.npart, s_w);
    }
}

// One thread per matrix: its limiter factor and new previous norm.
__global__ void apollo_limit_multi_kernel(const ApEntry* __restrict__ tab, int nmat,
                                          float gamma) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= nmat) return;
    const ApEntry& e = tab[i];
    limit_one(e.npart, norm_chunks(e.n), gamma, e.prev_norm, e.lim);
}

// ------------------------------------------------------------- host side --
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static std::mutex mu;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
    }
    return fn;
}

// 2-D bf16 tensor map over a row-major [rows][k] matrix, box [box_rows][64],
// 128-byte swizzle, zero fill out of bounds.
static bool make_map(CUtensorMap* map, const void* base, uint64_t k, uint64_t rows,
                     uint32_t box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {k, rows};
    const cuuint64_t strides[1] = {k * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kGK, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D fp32 tensor map over G [rows][cols] whose box is one projection job:
// 128 channels by 64 K (channels are G's rows, box [128][64], or its columns,
// box [64][128]). Used only to prefetch jobs into L2.
static bool make_gmap(CUtensorMap* map, const float* g, int64_t rows, int64_t cols,
                      bool rows_short) {
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)cols * 4};
    const cuuint32_t box[2] = {rows_short ? (cuuint32_t)kGM : (cuuint32_t)kGK,
                               rows_short ? (cuuint32_t)kGK : (cuuint32_t)kGM};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(g), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static int launch_project(const float* g, int64_t rows, int64_t cols, const uint16_t* P,
                          int rank, float* R, int* err, cudaStream_t st) {
    const int rows_short = rows <= cols;
    ApEntry e;
    memset(&e, 0, sizeof(e));
    e.g = g;
    e.R = R;
    e.rows = rows;
    e.cols = cols;
    e.s = rows_short ? rows : cols;
    e.L = rows_short ? cols : rows;
    e.rows_short = rows_short;
    e.kblocks = (int32_t)blocks_of(e.s, kGK);
    if (!make_map(&e.tmB, P, (uint64_t)e.s, (uint64_t)rank, (uint32_t)rank) ||
        !make_gmap(&e.tmG, g, rows, cols, rows_short))
        return record_cuda(cudaErrorInvalidValue);
    const int64_t ntiles = blocks_of(e.L, kGM);
    apollo_project_kernel<true><<<persistent_grid((const void*)apollo_project_kernel<true>,
                                                  kPThreads, kPSmem, ntiles),
                                  kPThreads, kPSmem, st>>>(nullptr, nullptr, ntiles, rank, err, e);
    return check_launch();
}

// The checks al_apollo_step applies to one matrix.
static int check_apollo_matrix(const al_apollo_matrix& m, int rank, int v_bits) {
    if (!m.p || !m.g || !m.proj || !m.m_codes || !m.m_absmax || !m.v_codes || !m.v_meta ||
        m.rows < 1 || m.cols < 1)
        return ALQ_ERR_INVALID_ARG;
    const int64_t s = m.rows <= m.cols ? m.rows : m.cols, L = m.rows <= m.cols ? m.cols : m.rows;
    if ((rank != 128 && rank != 256) || (v_bits != 8 && v_bits != 16) || m.cols % 4 != 0 ||
        s % 8 != 0 || m.rows * m.cols >= (int64_t)1 << 31 || L > (1 << 30))
        return ALQ_ERR_UNSUPPORTED;
    if (!aligned(m.p, 16) || !aligned(m.g, 16) || !aligned(m.proj, 16) ||
        !aligned(m.m_codes, 16) || !aligned(m.v_codes, 16) || !aligned(m.v_meta, 8) ||
        !aligned(m.m_absmax, 4))
        return ALQ_ERR_ALIGN;
    return ALQ_OK;
}

// Moment-pass scalars of step t (bias corrections in double, rounded once).
static MomentArgs moment_scalars(const al_apollo_hp* hp, int64_t t, int rank) {
    const double bc1 = 1.0 - pow((double)hp->beta1, (double)t);
    const double bc2 = 1.0 - pow((double)hp->beta2, (double)t);
    MomentArgs m{};
    m.block = rank;
    m.beta1 = hp->beta1;
    m.beta2 = hp->beta2;
    m.omb1 = (float)(1.0 - (double)hp->beta1);
    m.omb2 = (float)(1.0 - (double)hp->beta2);
    m.ic1 = (float)(1.0 / bc1);
    m.c2 = (float)(1.0 / sqrt(bc2));
    m.eps = hp->eps;
    m.log_floor = hp->log_floor;
    m.one = 1.0f;
    m.zero = 0.0f;
    return m;
}

template <int CPB, int VBITS>
static void launch_moments_t(const MomentArgs& m, cudaStream_t st) {
    const int64_t ntiles = blocks_of(m.n, kMTile);
    auto k = apollo_moments_kernel<CPB, VBITS>;
    k<<<persistent_grid((const void*)k, kThreads, 0, ntiles), kThreads, 0, st>>>(m, ntiles);
}

}  // namespace alq

using namespace alq;

extern "C" int al_apollo_step(float* p, const float* g, int64_t rows, int64_t cols,
                              const uint16_t* proj, int8_t* m_codes, float* m_absmax, int m_block,
                              void* v_codes, float* v_meta, int v_bits, int v_block,
                              float* prev_norm, const al_apollo_hp* hp, int64_t t,
                              void* workspace, size_t ws_bytes, void* stream) {
    if (!hp || t < 1) return ALQ_ERR_INVALID_ARG;
    const int rank = hp->rank;
    if (m_block != rank || v_block != rank) return ALQ_ERR_UNSUPPORTED;
    const al_apollo_matrix mat{p, g, rows, cols, proj, m_codes, m_absmax, v_codes, v_meta};
    int rc0 = check_apollo_matrix(mat, rank, v_bits);
    if (rc0) return rc0;
    const int64_t L = rows <= cols ? cols : rows;
    if (hp->norm_growth_gamma > 0.0f && !prev_norm) return ALQ_ERR_INVALID_ARG;
    const ApWs w = ap_layout(workspace, rows, cols, rank);
    if (!workspace || ws_bytes < w.bytes || !aligned(workspace, 256)) return ALQ_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    const int rows_short = rows <= cols;

    int rc = launch_project(g, rows, cols, proj, rank, w.R, w.err, st);
    if (rc) return rc;

    MomentArgs m = moment_scalars(hp, t, rank);
    m.R = w.R;
    m.n = L * rank;
    m.m_codes = m_codes;
    m.m_absmax = m_absmax;
    m.v_codes = v_codes;
    m.v_meta = v_meta;
    m.scale = w.scale;
    if (rank == 128) {
        if (v_bits == 8) launch_moments_t<1, 8>(m, st); else launch_moments_t<1, 16>(m, st);
    } else {
        if (v_bits == 8) launch_moments_t<2, 8>(m, st); else launch_moments_t<2, 16>(m, st);
    }
    rc = check_launch();
    if (rc) return rc;

    ApUpdateArgs u;
    u.p = p;
    u.g = g;
    u.n = rows * cols;
    u.dv = make_divider((uint32_t)cols);
    u.rows_short = rows_short;
    u.scale = w.scale;
    u.lim = nullptr;
    u.decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    u.lr_a = (float)((double)hp->lr * (double)hp->alpha);
    const int64_t ntiles = blocks_of(u.n, kTile);
    if (hp->norm_growth_gamma > 0.0f) {
        const int64_t nch = norm_chunks(u.n);
        apollo_gnorm_kernel<<<persistent_grid((const void*)apollo_gnorm_kernel, kThreads, 0, nch),
                              kThreads, 0, st>>>(u, ntiles, nch, w.npart);
        apollo_limit_kernel<<<1, 32, 0, st>>>(w.npart, nch, hp->norm_growth_gamma, prev_norm,
                                               w.lim);
        u.lim = w.lim;
    }
    apollo_update_kernel<<<persistent_grid((const void*)apollo_update_kernel, kThreads, 0, ntiles),
                           kThreads, 0, st>>>(u, ntiles);
    return check_launch();
}

// ------------------------------------------------------- grouped step --
namespace alq {

struct ApShape {
    int64_t s, L, n;
    int rows_short;
};

static ApShape ap_shape(const al_apollo_matrix& m) {
    ApShape a;
    a.rows_short = m.rows <= m.cols;
    a.s = a.rows_short ? m.rows : m.cols;
    a.L = a.rows_short ? m.cols : m.rows;
    a.n = m.rows * m.cols;
    return a;
}

// Per-matrix scratch of a grouped step: R, scale, limiter partials and
// factor, each 256-byte aligned.
static size_t multi_ws_bytes(const al_apollo_matrix& m, int rank) {
    const ApShape a = ap_shape(m);
    return r256(4 * (size_t)a.L * rank) + r256(4 * (size_t)a.L) +
           r256(8 * (size_t)norm_chunks(a.n)) + r256(8);
}

static int check_matrices(const al_apollo_matrix* mats, int nmat) {
    if (!mats || nmat < 1 || nmat > 65535) return ALQ_ERR_INVALID_ARG;
    return ALQ_OK;
}

static size_t plan_size(const al_apollo_matrix* mats, int nmat) {
    int64_t gemm = 0;
    for (int i = 0; i < nmat; ++i) gemm += blocks_of(ap_shape(mats[i]).L, kGM);
    return kApEntryOffset + (size_t)nmat * sizeof(ApEntry) + r256(2 * (size_t)gemm);
}

}  // namespace alq

extern "C" int al_apollo_plan_bytes(const al_apollo_matrix* mats, int nmat, size_t* bytes) {
    if (!bytes) return ALQ_ERR_INVALID_ARG;
    const int rc = check_matrices(mats, nmat);
    if (rc) return rc;
    for (int i = 0; i < nmat; ++i)
        if (mats[i].rows < 1 || mats[i].cols < 1) return ALQ_ERR_INVALID_ARG;
    *bytes = plan_size(mats, nmat);
    return ALQ_OK;
}

extern "C" int al_apollo_workspace_multi(const al_apollo_matrix* mats, int nmat, int rank,
                                         size_t* bytes) {
    if (!bytes) return ALQ_ERR_INVALID_ARG;
    int rc = check_matrices(mats, nmat);
    if (rc) return rc;
    if (rank != 128 && rank != 256) return ALQ_ERR_UNSUPPORTED;
    size_t tot = 256;  // the projection's timeout flag
    for (int i = 0; i < nmat; ++i) {
        if (mats[i].rows < 1 || mats[i].cols < 1) return ALQ_ERR_INVALID_ARG;
        tot += multi_ws_bytes(mats[i], rank);
    }
    *bytes = tot;
    return ALQ_OK;
}

extern "C" int al_apollo_plan(const al_apollo_matrix* mats, int nmat, int rank, int v_bits,
                              void* workspace, size_t ws_bytes, void* plan_host,
                              size_t plan_bytes, al_apollo_info* info) {
    int rc = check_matrices(mats, nmat);
    if (rc) return rc;
    if (!plan_host || !info) return ALQ_ERR_INVALID_ARG;
    for (int i = 0; i < nmat; ++i) {
        rc = check_apollo_matrix(mats[i], rank, v_bits);
        if (rc) return rc;
    }
    size_t need = 0;
    al_apollo_workspace_multi(mats, nmat, rank, &need);
    if (!workspace || ws_bytes < need || !aligned(workspace, 256)) return ALQ_ERR_WORKSPACE;
    if (plan_bytes < plan_size(mats, nmat)) return ALQ_ERR_INVALID_ARG;

    char* base = (char*)plan_host;
    memset(base, 0, plan_size(mats, nmat));
    uint16_t* tile_mat =
        (uint16_t*)(base + kApEntryOffset + (size_t)nmat * sizeof(ApEntry));
    char* ws = (char*)workspace + 256;  // first 256 bytes: timeout flag
    ApPlanHeader h{};
    h.magic = kApPlanMagic;
    h.limiter_ok = 1;
    h.nmat = nmat;
    h.rank = rank;
    h.v_bits = v_bits;
    for (int i = 0; i < nmat; ++i) {
        const al_apollo_matrix& m = mats[i];
        const ApShape a = ap_shape(m);
        ApEntry e;
        memset(&e, 0, sizeof(e));
        e.p = m.p;
        e.g = m.g;
        e.m_codes = m.m_codes;
        e.m_absmax = m.m_absmax;
        e.v_codes = m.v_codes;
        e.v_meta = m.v_meta;
        e.R = (float*)ws;
        e.scale = (float*)(ws + r256(4 * (size_t)a.L * rank));
        e.npart = (double*)(ws + r256(4 * (size_t)a.L * rank) + r256(4 * (size_t)a.L));
        e.lim = (float*)((char*)e.npart + r256(8 * (size_t)norm_chunks(a.n)));
        e.prev_norm = m.prev_norm;
        ws += multi_ws_bytes(m, rank);
        e.rows = m.rows;
        e.cols = m.cols;
        e.n = a.n;
        e.L = a.L;
        e.s = a.s;
        e.npj = a.L * rank;
        e.dv = make_divider((uint32_t)m.cols);
        e.rows_short = a.rows_short;
        e.kblocks = (int32_t)blocks_of(a.s, kGK);
        e.gemm_t0 = h.gemm_tiles;
        e.mom_t0 = h.mom_tiles;
        e.upd_t0 = h.upd_tiles;
        e.nrm_t0 = h.norm_chunks;
        if (!make_map(&e.tmB, m.proj, (uint64_t)a.s, (uint64_t)rank, (uint32_t)rank) ||
            !make_gmap(&e.tmG, m.g, m.rows, m.cols, a.rows_short))
            return record_cuda(cudaErrorInvalidValue);
        const int64_t gt = blocks_of(a.L, kGM);
        for (int64_t k = 0; k < gt; ++k) tile_mat[h.gemm_tiles + k] = (uint16_t)i;
        h.gemm_tiles += gt;
        h.mom_tiles += blocks_of(e.npj, kMTile);
        h.upd_tiles += blocks_of(a.n, kTile);
        h.norm_chunks += norm_chunks(a.n);
        if (!m.prev_norm) h.limiter_ok = 0;
        h.total_params += a.n;
        h.total_channels += a.L;
        memcpy(base + kApEntryOffset + (size_t)i * sizeof(ApEntry), &e, sizeof(e));
    }
    memcpy(base, &h, sizeof(h));
    info->nmat = nmat;
    info->rank = rank;
    info->v_bits = v_bits;
    info->limiter_ok = h.limiter_ok;
    info->norm_chunks = h.norm_chunks;
    info->total_params = h.total_params;
    info->total_channels = h.total_channels;
    info->gemm_tiles = h.gemm_tiles;
    info->mom_tiles = h.mom_tiles;
    info->upd_tiles = h.upd_tiles;
    info->workspace = workspace;
    return ALQ_OK;
}

extern "C" int al_apollo_step_multi(const void* plan_dev, const al_apollo_info* info,
                                    const al_apollo_hp* hp, int64_t t, void* stream) {
    if (!plan_dev || !info || !hp || t < 1 || info->nmat < 1 || !info->workspace)
        return ALQ_ERR_INVALID_ARG;
    if (!aligned(plan_dev, 64)) return ALQ_ERR_ALIGN;
    if (hp->rank != info->rank) return ALQ_ERR_INVALID_ARG;
    const bool limited = hp->norm_growth_gamma > 0.0f;
    if (limited && !info->limiter_ok) return ALQ_ERR_INVALID_ARG;  // a matrix has no prev_norm
    cudaStream_t st = (cudaStream_t)stream;
    const ApEntry* tab = (const ApEntry*)((const char*)plan_dev + kApEntryOffset);
    const uint16_t* tile_mat = (const uint16_t*)((const char*)plan_dev + kApEntryOffset +
                                                 (size_t)info->nmat * sizeof(ApEntry));
    int* err = (int*)info->workspace;

    int rc;
    ApEntry none;
    memset(&none, 0, sizeof(none));
    apollo_project_kernel<false><<<persistent_grid((const void*)apollo_project_kernel<false>,
                                                   kPThreads, kPSmem, info->gemm_tiles),
                                   kPThreads, kPSmem, st>>>(tab, tile_mat, info->gemm_tiles,
                                                            info->rank, err, none);
    rc = check_launch();
    if (rc) return rc;

    const MomentArgs m = moment_scalars(hp, t, info->rank);
    const int64_t nt = info->mom_tiles;
#define ALQ_MOM(CPB, VB)                                                                     \
    apollo_moments_multi_kernel<CPB, VB><<<                                                  \
        persistent_grid((const void*)apollo_moments_multi_kernel<CPB, VB>, kThreads, 0, nt), \
        kThreads, 0, st>>>(tab, info->nmat, nt, m)
    if (info->rank == 128) {
        if (info->v_bits == 8) ALQ_MOM(1, 8); else ALQ_MOM(1, 16);
    } else {
        if (info->v_bits == 8) ALQ_MOM(2, 8); else ALQ_MOM(2, 16);
    }
#undef ALQ_MOM
    rc = check_launch();
    if (rc) return rc;

    if (limited) {
        const int64_t nch = info->norm_chunks;
        apollo_gnorm_multi_kernel<<<persistent_grid((const void*)apollo_gnorm_multi_kernel,
                                                    kThreads, 0, nch),
                                    kThreads, 0, st>>>(tab, info->nmat, nch);
        apollo_limit_multi_kernel<<<(info->nmat + 127) / 128, 128, 0, st>>>(
            tab, info->nmat, hp->norm_growth_gamma);
        rc = check_launch();
        if (rc) return rc;
    }
    ApUpdateArgs u{};
    u.lim = nullptr;
    u.decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    u.lr_a = (float)((double)hp->lr * (double)hp->alpha);
    apollo_update_multi_kernel<<<persistent_grid((const void*)apollo_update_multi_kernel,
                                                 kThreads, 0, info->upd_tiles),
                                 kThreads, 0, st>>>(tab, info->nmat, info->upd_tiles, u,
                                                    limited ? 1 : 0);
    return check_launch();
}
