// alq_factored.cu -- Adafactor and CAME steps with AL-coded factored states
// (Sec. 3.1: row/column statistics reconstruct the second moment; CAME adds
// factored confidence states tracking a residual) and UF8 momentum.
//
// Launch sequence of one step (all on the caller's stream, no host sync):
//   sumsq      G read once: per 64-row x 256-column tile, exact float-float
//              sums of g^2 per row (over the tile's columns) and per column
//              (over its rows) -> fp64 partials in the workspace.
//   factor     one CTA per factor block: finish r_i / c_j (fp64, fixed order),
//              decode the old factor, EMA, AL-encode the fresh factor.
//   scale      a_i = 1/sqrt(R_i / mean(R)), b_j = 1/sqrt(C_j).
//   usq        G read again: u = (g a_i) b_j, exact float-float sum of u^2,
//              one fp64 partial per 4096-element tile (fixed order). The CTA
//              that finishes a matrix's last tile adds its partials and
//              writes the clip factor 1 / max(1, RMS(u) / d).
//   update     G read a third time: u_hat, optional UF8 momentum, p update.
// CAME inserts, before its update, a second sumsq pass over the residual
// (u_hat - m)^2 + eps2 (recomputing m from the old momentum codes), a second
// factor pass (confidence, beta3) and a second scale pass; its update uses
// m / sqrt(S) with S from the confidence factors.
// Every reduction is deterministic: error-free fp32 transforms inside a
// thread, fixed shuffle and tree orders, fp64 merges; no float atomics.
//
// Each pass is a per-tile device function; the single-matrix kernels and
// the grouped ones (one launch per pass over many matrices, tiles never
// crossing a matrix) call the same functions, so a matrix's results do not
// depend on which path stepped it.
#include "alq_async.cuh"
#include "alq_kernels.cuh"

namespace alq {

// ------------------------------------------- programmatic dependent launch --
// The passes of a step form a dependent chain on one stream. Each is launched
// with programmatic stream serialization: every CTA first allows the next
// pass to be launched (its CTAs take SM slots as this pass's CTAs retire, and
// its launch latency overlaps this pass), then waits until the previous
// grid has completed and its memory operations are visible. Every memory
// access of a pass comes after that wait, so the order of reads and writes
// is the order of the stream.
__device__ __forceinline__ void pdl_entry() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// The grouped passes (several matrices per launch, groups on several
// streams) launch without the attribute: there, dependent CTAs waiting on SM
// slots took them from the other streams' passes (measured slower); the
// instructions of pdl_entry() are then no-ops.
template <typename... KArgs, typename... Args>
static void pdl_launch(bool dependent, void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = dependent ? 1 : 0;
    cudaLaunchKernelEx(&cfg, k, args...);  // errors surface through check_launch()
}


constexpr int kFR = 64;   // rows per sumsq tile
constexpr int kFC = 256;  // columns per sumsq tile
constexpr int kFCH = kFC / 128;  // 4-column chunks per lane
constexpr int kUsqChunk = 8;  // tiles of kTile elements per RMS partial

// ------------------------------------------------------------ workspace --
struct FacWs {
    double* rowpart;  // [ncb][rows]
    double* colpart;  // [nrb][cols]
    double* upart;    // [chunks of kUsqChunk tiles]: RMS partials
    float* fr;        // fresh row factor (V)
    float* fc;        // fresh column factor (V)
    float* fr2;       // fresh row factor (C)
    float* fc2;       // fresh column factor (C)
    float* a;         // [rows]
    float* b;         // [cols]
    float* a2;        // [rows]
    float* b2;        // [cols]
    float* scal;      // [4]: icf
    double* rsum;     // [rows / 128 + 1]: per-block sums of the fresh row factor (V)
    double* rsum2;    // same for the confidence row factor (C)
    unsigned int* ticket;  // CTAs of the RMS pass that have finished
    size_t bytes;
};

static size_t round256(size_t x) { return (x + 255) & ~(size_t)255; }

static FacWs fac_layout(void* base, int64_t rows, int64_t cols) {
    const int64_t ncb = blocks_of(cols, kFC), nrb = blocks_of(rows, kFR);
    FacWs w;
    size_t off = 0;
    char* p = (char*)base;
    auto take = [&](size_t bytes) {
        char* r = p ? p + off : nullptr;
        off += round256(bytes);
        return r;
    };
    w.rowpart = (double*)take(sizeof(double) * ncb * rows);
    w.colpart = (double*)take(sizeof(double) * nrb * cols);
    w.upart = (double*)take(sizeof(double) * blocks_of(blocks_of(rows * cols, kTile), kUsqChunk));
    w.fr = (float*)take(sizeof(float) * rows);
    w.fc = (float*)take(sizeof(float) * cols);
    w.fr2 = (float*)take(sizeof(float) * rows);
    w.fc2 = (float*)take(sizeof(float) * cols);
    w.a = (float*)take(sizeof(float) * rows);
    w.b = (float*)take(sizeof(float) * cols);
    w.a2 = (float*)take(sizeof(float) * rows);
    w.b2 = (float*)take(sizeof(float) * cols);
    w.scal = (float*)take(sizeof(float) * 4);
    w.rsum = (double*)take(sizeof(double) * (rows / 128 + 1));
    w.rsum2 = (double*)take(sizeof(double) * (rows / 128 + 1));
    w.ticket = (unsigned int*)take(sizeof(unsigned int));
    w.bytes = off;
    return w;
}

// ------------------------------------------------------------ residual --
// CAME's residual inputs: old momentum codes, scales, clip factor.
struct ResidualArgs {
    const int8_t* m_codes;
    const float* m_absmax;
    int m_shift;  // log2(m_block)
    const float* a;
    const float* b;
    const float* scal;  // scal[0] = 1 / max(1, RMS(u)/d)
    float beta1, omb1, eps2;
    float one, zero;    // 1 and 0 from the kernel's parameters (see ff_sq2)
};

// ----------------------------------------------------------------- sumsq --
// MODE 0: terms g^2 (exact two-float squares). MODE 1: terms CAME's
// residual (u_hat - m)^2 + eps2 rounded to fp32 as the update defines it.
// One 64-row x kFC-column tile (bx over columns, by over rows); every
// thread of the CTA calls it, with the CTA's dynamic shared memory (see
// SumsqSmem). Each warp walks its eight rows two at a time; the next pair's
// loads go to shared memory by per-thread asynchronous copies while the
// current pair is summed (each thread reads back only what it copied, so no
// barrier is needed), which keeps the loads of two row pairs in flight
// without holding them in registers.
template <int MODE>
struct SumsqSmem {
    // per stage, warp, row of the pair, chunk and lane: g (16 bytes), and for
    // MODE 1 the momentum codes and the block absmax (4 bytes each)
    static constexpr int kSlots = 2 * (kThreads / 32) * 2 * kFCH * 32;
    static constexpr size_t kG = sizeof(float4) * kSlots;
    static constexpr size_t kBytes = kG + (MODE == 1 ? 2 * sizeof(uint32_t) * kSlots : 0);
    static_assert(kBytes >= sizeof(float2) * (kThreads / 32) * kFC, "s_col aliases the stages");
};

template <int MODE>
__device__ __forceinline__ void sumsq_tile(const float* __restrict__ g, int rows, int cols,
                                           const ResidualArgs& ra, double* __restrict__ rowpart,
                                           double* __restrict__ colpart, int bx, int by,
                                           unsigned char* smem) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c0 = bx * kFC, r0 = by * kFR;
    float4* sg = reinterpret_cast<float4*>(smem);
    uint32_t* sm = reinterpret_cast<uint32_t*>(smem + SumsqSmem<MODE>::kG);
    uint32_t* sa = sm + SumsqSmem<MODE>::kSlots;
    // this thread's slot of (stage, row q of the pair, chunk k)
    auto slot = [&](int st, int q, int k) {
        return (((st * (kThreads / 32) + warp) * 2 + q) * kFCH + k) * 32 + lane;
    };
    // copies of the row pair starting at warp row 2 * it into stage it & 1
    auto issue = [&](int it) {
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int row = r0 + warp + 8 * (2 * it + q);
#pragma unroll
            for (int k = 0; k < kFCH; ++k) {
                const int col = c0 + 128 * k + 4 * lane;
                const bool ok = row < rows && col < cols;
                const int64_t idx = ok ? (int64_t)row * cols + col : 0;
                const int sl = slot(it & 1, q, k);
                cp_async16(smem_u32(sg + sl), g + idx, ok);
                if (MODE == 1) {
                    cp_async4(smem_u32(sm + sl), ra.m_codes + idx, ok);
                    cp_async4(smem_u32(sa + sl), ra.m_absmax + (idx >> ra.m_shift), ok);
                }
            }
        }
        cp_async_commit();
    };
    // column sums of this lane's 4 kFCH columns as pairs; each row's sum as
    // two (even and odd elements) merged before the warp sum
    float2 ch[2 * kFCH], cl[2 * kFCH];
#pragma unroll
    for (int k = 0; k < 2 * kFCH; ++k) ch[k] = cl[k] = make_float2(0.0f, 0.0f);
    const float2 one = make_float2(ra.one, ra.one), zero = make_float2(ra.zero, ra.zero);
    const float2 neg = make_float2(-1.0f, -1.0f);
    float icf = 0.0f;
    float4 bv[kFCH];  // column scales of this lane's columns (CAME residual)
    if (MODE == 1) {
        icf = __ldg(ra.scal);
#pragma unroll
        for (int k = 0; k < kFCH; ++k) {
            const int col = c0 + 128 * k + 4 * lane;
            bv[k] = col < cols ? __ldg(reinterpret_cast<const float4*>(ra.b + col))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    // this warp's eight row sums, row k's in lane k, converted to fp64 in
    // one instruction at the end (FP64 is slow on this part)
    float keep_h = 0.0f, keep_l = 0.0f;
    constexpr int kIters = kFR / 16;  // row pairs per warp
    issue(0);
    for (int it = 0; it < kIters; ++it) {
        if (it + 1 < kIters) issue(it + 1); else cp_async_commit();
        cp_async_wait<1>();
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int row = r0 + warp + 8 * (2 * it + q);
            const float ai = (MODE == 1 && row < rows) ? __ldg(ra.a + row) : 0.0f;
            float2 rh2 = make_float2(0.0f, 0.0f), rl2 = make_float2(0.0f, 0.0f);
            if (row < rows) {
#pragma unroll
                for (int k = 0; k < kFCH; ++k) {
                    const int col = c0 + 128 * k + 4 * lane;
                    if (col < cols) {
                        const int sl = slot(it & 1, q, k);
                        const float4 gv = sg[sl];
                        uint32_t mx = 0;
                        float dm = 0.0f;
                        if (MODE == 1) {
                            mx = sm[sl] ^ 0x80808080u;
                            dm = __uint_as_float(sa[sl]) / 127.0f;
                        }
#pragma unroll
                        for (int jp = 0; jp < 2; ++jp) {
                            const float2 x = jp == 0 ? make_float2(gv.x, gv.y)
                                                     : make_float2(gv.z, gv.w);
                            float2 h, nl;
                            if (MODE == 0) {
                                ff_sq2(x, neg, zero, h, nl);
                            } else {
                                // the update's residual, each product rounded
                                // before it enters a sum (opaque one)
                                const float2 bj = jp == 0 ? make_float2(bv[k].x, bv[k].y)
                                                          : make_float2(bv[k].z, bv[k].w);
                                const float2 u = mul2(mul2(x, make_float2(ai, ai)), bj);
                                const float2 uh = mul2(u, make_float2(icf, icf));
                                const float2 qf = make_float2(
                                    u2f(__byte_perm(mx, 0x4B400000u, 0x7640u | (2 * jp))),
                                    u2f(__byte_perm(mx, 0x4B400000u, 0x7640u | (2 * jp + 1))));
                                const float2 mh = mul2(add2(qf, make_float2(-12583040.0f, -12583040.0f)),
                                                       make_float2(dm, dm));
                                const float2 nmk = fma2(mul2(make_float2(-ra.beta1, -ra.beta1), mh), one,
                                                        mul2(make_float2(-ra.omb1, -ra.omb1), uh));
                                const float2 d = fma2(uh, one, nmk);  // uh - mk
                                h = fma2(mul2(d, d), one, make_float2(ra.eps2, ra.eps2));
                                nl = make_float2(0.0f, 0.0f);
                            }
                            ff_acc2(ch[2 * k + jp], cl[2 * k + jp], h, nl);
                            ff_acc2(rh2, rl2, h, nl);
                        }
                    }
                }
            }
            float rh, rl;
            ff_merge2(rh2, rl2, rh, rl);
            ff_warp_sum(rh, rl);
            if (lane == 2 * it + q) {
                keep_h = rh;
                keep_l = rl;
            }
        }
    }
    cp_async_wait<0>();
    {
        const int row = r0 + warp + 8 * lane;  // lane k holds row warp + 8 k
        if (lane < kFR / 8 && row < rows)
            rowpart[(int64_t)bx * rows + row] = (double)keep_h + (double)keep_l;
    }
    // column sums: the warps' two-float sums merged in warp order, one fp64
    // conversion per column (the merge buffer reuses the stages)
    float2 (*s_col)[kFC] = reinterpret_cast<float2 (*)[kFC]>(smem);
    __syncthreads();
#pragma unroll
    for (int k = 0; k < kFCH; ++k)
#pragma unroll
        for (int jp = 0; jp < 2; ++jp) {
            const float2 h = ch[2 * k + jp], l = cl[2 * k + jp];
            s_col[warp][128 * k + 4 * lane + 2 * jp] = make_float2(h.x, l.x);
            s_col[warp][128 * k + 4 * lane + 2 * jp + 1] = make_float2(h.y, l.y);
        }
    __syncthreads();
    for (int t = threadIdx.x; t < kFC; t += kThreads) {
        if (c0 + t >= cols) continue;
        float hi = s_col[0][t].x, lo = s_col[0][t].y;
#pragma unroll
        for (int w = 1; w < kThreads / 32; ++w) ff_acc(hi, lo, s_col[w][t].x, s_col[w][t].y);
        colpart[(int64_t)by * cols + c0 + t] = (double)hi + (double)lo;
    }
}

template <int MODE>
__global__ void __launch_bounds__(kThreads)
sumsq_kernel(const float* __restrict__ g, int rows, int cols, ResidualArgs ra,
             double* __restrict__ rowpart, double* __restrict__ colpart) {
    pdl_entry();
    extern __shared__ __align__(16) unsigned char s_sumsq[];
    sumsq_tile<MODE>(g, rows, cols, ra, rowpart, colpart, blockIdx.x, blockIdx.y, s_sumsq);
}

// ---------------------------------------------------------------- factor --
// One factor vector's update: stat_i = sum_p part[p][i] / mean_len + add_eps
// (fp64, fixed order: partial p into accumulator p mod 4, the four added
// pairwise; rounded once), fresh = beta * decode(old) + omb * stat, then AL
// re-encoding of each block.
struct FactorDesc {
    const double* part;
    int nparts;
    int64_t len;
    double mean_len;
    double add_eps;
    float beta, omb;
    void* codes;
    float* meta;
    int bits;
    int block;
    float log_floor;
    float* fresh;
};

__device__ __forceinline__ uint32_t fac_code(const FactorDesc& f, int64_t i) {
    return f.bits == 8 ? (uint32_t)((const uint8_t*)f.codes)[i] : (uint32_t)((const uint16_t*)f.codes)[i];
}

// KPT = elements per thread (block / 256, at least 1). rsum (nullable)
// receives, for the blocks of f0, the fp64 sum of the block's fresh values in
// a fixed order (the scale pass builds mean(R) from them).
// Block b of factor f, by one CTA; rsum (nullable) as above.
template <int KPT>
__device__ __forceinline__ void factor_block(const FactorDesc& f, int64_t b,
                                             double* __restrict__ rsum) {
    __shared__ uint32_t s_part[2][kThreads / 32];
    __shared__ double s_sum[kThreads / 32];
    const bool first = rsum != nullptr;
    const int64_t lo = b * f.block;
    const int64_t hi = lo + f.block < f.len ? lo + f.block : f.len;
    const bool raw = f.bits == 32;  // the unquantized fp32 role: no metadata
    const float2 om = raw ? make_float2(0.f, 0.f) : __ldg(reinterpret_cast<const float2*>(f.meta) + b);
    const float Lm2 = f.bits == 8 ? 254.0f : 65534.0f;
    float v[KPT];
    uint32_t vmin = 0xFFFFFFFFu, vmax = 0u;
#pragma unroll
    for (int k = 0; k < KPT; ++k) {
        const int64_t i = lo + threadIdx.x + (int64_t)kThreads * k;
        v[k] = 0.0f;
        if (i < hi) {
            // partials in a fixed order: loads issued 32 at a time (one
            // memory round trip per 32 partials), summed into four
            // accumulators (partial p into accumulator p mod 4, in index
            // order), which are then added as (a0 + a1) + (a2 + a3)
            double a[4] = {0.0, 0.0, 0.0, 0.0};
            const double* pp = f.part + i;
            int p = 0;
            for (; p + 32 <= f.nparts; p += 32) {
                double t32[32];
#pragma unroll
                for (int q = 0; q < 32; ++q) t32[q] = pp[(int64_t)(p + q) * f.len];
#pragma unroll
                for (int q = 0; q < 32; ++q) a[q & 3] += t32[q];
            }
            for (; p + 4 <= f.nparts; p += 4) {
#pragma unroll
                for (int q = 0; q < 4; ++q) a[q] += pp[(int64_t)(p + q) * f.len];
            }
            // p is a multiple of 4 here: the last 0-3 partials
#pragma unroll
            for (int q = 0; q < 3; ++q)
                if (p + q < f.nparts) a[q] += pp[(int64_t)(p + q) * f.len];
            const double s = (a[0] + a[1]) + (a[2] + a[3]);
            const float stat = (float)(s / f.mean_len + f.add_eps);
            const float old = raw ? ((const float*)f.codes)[i]
                                  : al_decode_direct(fac_code(f, i), om.x, om.y, Lm2);
            v[k] = f.beta * old + f.omb * stat;
            f.fresh[i] = v[k];
            const uint32_t vb = f2u(v[k]);
            vmin = umix<false>(vmin, vb - 1u);
            vmax = umix<true>(vmax, vb);
        }
    }
    if (first) {
        // fixed order: per thread, then shuffle tree, then warps in order
        double t = 0.0;
#pragma unroll
        for (int k = 0; k < KPT; ++k) t += (double)v[k];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xFFFFFFFFu, t, o);
        if ((threadIdx.x & 31) == 0) s_sum[threadIdx.x >> 5] = t;
    }
    if (raw) {
        // the fresh factor is the stored state
        __syncthreads();
        if (first && threadIdx.x == 0) {
            double t = 0.0;
            for (int w = 0; w < kThreads / 32; ++w) t += s_sum[w];
            rsum[b] = t;
        }
#pragma unroll
        for (int k = 0; k < KPT; ++k) {
            const int64_t i = lo + threadIdx.x + (int64_t)kThreads * k;
            if (i < hi) ((float*)f.codes)[i] = v[k];
        }
        return;
    }
    vmin = __reduce_min_sync(0xFFFFFFFFu, vmin);
    vmax = __reduce_max_sync(0xFFFFFFFFu, vmax);
    vmin = cta_group_reduce<false>(vmin, s_part[0], kThreads / 32);
    vmax = cta_group_reduce<true>(vmax, s_part[1], kThreads / 32);
    if (first && threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < kThreads / 32; ++w) t += s_sum[w];
        rsum[b] = t;
    }
    float lmin, delta;
    al_block_params(u2f(vmin + 1u), u2f(vmax), f.log_floor, lmin, delta);
    const AlEncConsts ek = al_encode_consts(lmin, delta, Lm2);
#pragma unroll
    for (int k = 0; k < KPT; ++k) {
        const int64_t i = lo + threadIdx.x + (int64_t)kThreads * k;
        if (i < hi) {
            uint32_t q = 0;
            if (v[k] != 0.0f) {
                bool fb;
                q = al_quantize_fast(v[k], ek, Lm2, fb);
                if (fb) q = al_quantize_refine(v[k], lmin, delta, Lm2);
            }
            if (f.bits == 8)
                ((uint8_t*)f.codes)[i] = (uint8_t)q;
            else
                ((uint16_t*)f.codes)[i] = (uint16_t)q;
        }
    }
    if (threadIdx.x == 0) reinterpret_cast<float2*>(f.meta)[b] = make_float2(lmin, delta);
}

// Blocks 0 .. nb0 - 1 of f0 (with the block sums into rsum), then f1's.
template <int KPT>
__global__ void __launch_bounds__(kThreads)
factor_kernel(FactorDesc f0, FactorDesc f1, int nb0, double* __restrict__ rsum) {
    pdl_entry();
    const bool first = (int)blockIdx.x < nb0;
    factor_block<KPT>(first ? f0 : f1, first ? blockIdx.x : blockIdx.x - nb0,
                      first ? rsum : nullptr);
}

// ----------------------------------------------------------------- scale --
// a_i = 1/sqrt(R_i / mean(R)), b_j = 1/sqrt(C_j). mean(R) in fp64 from the
// factor pass's per-block sums, added in block order by every CTA (the same
// value everywhere), rounded once. One element per thread over rows + cols.
__device__ __forceinline__ void scale_tile(const float* __restrict__ R, int rows,
                                           const float* __restrict__ C, int cols,
                                           const double* __restrict__ rsum, int nrb,
                                           float* __restrict__ a, float* __restrict__ b,
                                           unsigned int* __restrict__ ticket, int tile) {
    __shared__ float s_mean;
    if (ticket && tile == 0 && threadIdx.x == 0) *ticket = 0u;  // for the RMS pass
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int k = 0; k < nrb; ++k) t += rsum[k];
        s_mean = (float)(t / (double)rows);
    }
    __syncthreads();
    const float meanR = s_mean;
    const int i = tile * kThreads + threadIdx.x;
    if (i < rows)
        a[i] = 1.0f / sqrtf(R[i] / meanR);
    else if (i < rows + cols)
        b[i - rows] = 1.0f / sqrtf(C[i - rows]);
}

__global__ void __launch_bounds__(kThreads)
scale_kernel(const float* __restrict__ R, int rows, const float* __restrict__ C, int cols,
             const double* __restrict__ rsum, int nrb, float* __restrict__ a,
             float* __restrict__ b, unsigned int* __restrict__ ticket) {
    pdl_entry();
    scale_tile(R, rows, C, cols, rsum, nrb, a, b, ticket, blockIdx.x);
}

// ------------------------------------------------------------------- usq --
// Sum of u^2, u = (g a_i) b_j, over the whole matrix: exact squares in
// two-float per thread, fixed warp/CTA order, one fp64 partial per chunk of
// kUsqChunk tiles (4096 elements each, a partition of the matrix that does
// not depend on the grid). The CTA that finishes a matrix's last chunk (an
// atomic ticket, zeroed by the scale pass) adds the partials in chunk order
// and writes the clip factor scal[0] = 1 / max(1, sqrt(sum / count) / clip_d).
struct UsqArgs {
    const float* g;
    int64_t n;
    Divider dv;
    const float* a;
    const float* b;
    double* upart;
    unsigned int* ticket;
    float* scal;
    float zero;  // 0 from the kernel's parameters (see ff_sq2)
};

__device__ __forceinline__ int64_t usq_chunks(int64_t n) {
    return blocks_of_dev(blocks_of_dev(n, kTile), kUsqChunk);
}

// The chunk's partial (every thread of the CTA calls it; thread 0 gets it).
__device__ __forceinline__ double usq_chunk_sum(const UsqArgs& q, int64_t chunk, float2* s_w) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const float2 zero = make_float2(q.zero, q.zero), neg = make_float2(-1.0f, -1.0f);
    float2 hi2 = make_float2(0.0f, 0.0f), lo2 = make_float2(0.0f, 0.0f);
    // the gradient loads of two tiles in flight per step (the row and column
    // scales, small and cached, are read as they are used), accumulated in
    // tile, chunk and element order: the order of one tile at a time
    for (int k = 0; k < kUsqChunk; k += 2) {
        float4 gv[2][4];
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const int64_t seg0 = (chunk * kUsqChunk + k + kk) * kTile + (int64_t)warp * kSeg;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int64_t idx = chunk_index(seg0, c, lane);
                gv[kk][c] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (idx < q.n) gv[kk][c] = __ldcg(reinterpret_cast<const float4*>(q.g + idx));
            }
        }
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const int64_t seg0 = (chunk * kUsqChunk + k + kk) * kTile + (int64_t)warp * kSeg;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int64_t idx = chunk_index(seg0, c, lane);
                if (idx < q.n) {
                    const uint32_t row = divide((uint32_t)idx, q.dv);
                    const uint32_t col = (uint32_t)idx - row * q.dv.d;
                    const float4 bv = __ldg(reinterpret_cast<const float4*>(q.b + col));
                    const float2 ai = make_float2(__ldg(q.a + row), __ldg(q.a + row));
                    const float4& g4 = gv[kk][c];
#pragma unroll
                    for (int jp = 0; jp < 2; ++jp) {
                        const float2 x = jp == 0 ? make_float2(g4.x, g4.y) : make_float2(g4.z, g4.w);
                        const float2 bj = jp == 0 ? make_float2(bv.x, bv.y) : make_float2(bv.z, bv.w);
                        ff_acc_sq2(hi2, lo2, mul2(mul2(x, ai), bj), neg, zero);  // u = (g a_i) b_j
                    }
                }
            }
        }
    }
    float hi, lo;
    ff_merge2(hi2, lo2, hi, lo);
    ff_warp_sum(hi, lo);
    __syncthreads();  // s_w may still be read by the previous chunk's finish
    if (lane == 0) s_w[warp] = make_float2(hi, lo);
    __syncthreads();
    double t = 0.0;
    if (threadIdx.x == 0) {
        float h = s_w[0].x, l = s_w[0].y;
        for (int w = 1; w < kThreads / 32; ++w) ff_acc(h, l, s_w[w].x, s_w[w].y);
        t = (double)h + (double)l;
    }
    return t;
}

// One chunk of the RMS pass: its partial, and the clip factor if this CTA
// completes the matrix.
__device__ __forceinline__ void usq_chunk(const UsqArgs& q, int64_t chunk, float clip_d,
                                          float2* s_w, double* s_d, bool* s_last) {
    const int64_t nchunks = usq_chunks(q.n);
    const double t = usq_chunk_sum(q, chunk, s_w);
    if (threadIdx.x == 0) {
        q.upart[chunk] = t;
        __threadfence();
        *s_last = atomicAdd(q.ticket, 1u) == (unsigned int)(nchunks - 1);
    }
    __syncthreads();
    if (!*s_last) return;
    __threadfence();
    // fixed order: per thread over a stride of kThreads, then a tree
    double acc = 0.0;
    for (int64_t i = threadIdx.x; i < nchunks; i += kThreads) acc += ((volatile double*)q.upart)[i];
    s_d[threadIdx.x] = acc;
    __syncthreads();
    for (int st = kThreads / 2; st > 0; st >>= 1) {
        if ((int)threadIdx.x < st) s_d[threadIdx.x] += s_d[threadIdx.x + st];
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        const double rms = sqrt(s_d[0] / (double)q.n);
        double cf = rms / (double)clip_d;
        if (cf < 1.0) cf = 1.0;
        q.scal[0] = (float)(1.0 / cf);
    }
}

__global__ void __launch_bounds__(kThreads)
usq_kernel(UsqArgs q, float clip_d) {
    pdl_entry();
    __shared__ float2 s_w[kThreads / 32];
    __shared__ double s_d[kThreads];
    __shared__ bool s_last;
    const int64_t nchunks = usq_chunks(q.n);
    for (int64_t chunk = blockIdx.x; chunk < nchunks; chunk += gridDim.x)
        usq_chunk(q, chunk, clip_d, s_w, s_d, &s_last);
}


// ---------------------------------------------------------------- update --
// MODE 0: Adafactor without momentum; 1: Adafactor with UF8 momentum;
// 2: CAME (UF8 momentum, p -= lr (m a2_i) b2_j).
struct UpdateArgs {
    float* p;
    const float* g;
    int64_t n;
    Divider dv;
    const float* a;
    const float* b;
    const float* a2;
    const float* b2;
    const float* scal;
    int8_t* m_codes;
    float* m_absmax;
    int m_block;
    float beta1, omb1, decay, lr;
};

// One tile of the update; every thread of the CTA calls it (momentum blocks
// wider than a warp's segment meet in s_part).
template <int MODE, int CPBM>
__device__ __forceinline__ void update_tile(const UpdateArgs& u, int64_t tile, uint32_t* s_part) {
    constexpr int NBM = 4 / CPBM;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int wpbm = CPBM == 4 && u.m_block > kSeg ? u.m_block / kSeg : 1;
    const float icf = __ldg(u.scal);
    const int mshift = block_shift<CPBM, 4>(u.m_block);
    const int64_t nmb = (u.n + (1 << mshift) - 1) >> mshift;
    {
        const int64_t seg0 = tile * kTile + (int64_t)warp * kSeg;
        const int64_t mb0 = seg0 >> mshift;
        float dm[NBM];
#pragma unroll
        for (int b = 0; b < NBM; ++b)
            dm[b] = (MODE > 0 && mb0 + b < nmb) ? __ldg(u.m_absmax + mb0 + b) / 127.0f : 0.0f;
        float mf[16];
        uint32_t cabs[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int64_t idx = chunk_index(seg0, c, lane);
            cabs[c] = 0u;
#pragma unroll
            for (int j = 0; j < 4; ++j) mf[4 * c + j] = 0.0f;
            if (idx >= u.n) continue;
            const uint32_t row = divide((uint32_t)idx, u.dv);
            const uint32_t col = (uint32_t)idx - row * u.dv.d;
            const float4 gv = __ldcs(reinterpret_cast<const float4*>(u.g + idx));
            const float4 pv = __ldcs(reinterpret_cast<const float4*>(u.p + idx));
            const float4 bv = __ldg(reinterpret_cast<const float4*>(u.b + col));
            const float ai = __ldg(u.a + row);
            uint32_t mw = 0;
            float4 b2v = make_float4(0.f, 0.f, 0.f, 0.f);
            float a2i = 0.0f;
            if (MODE > 0) mw = __ldcs(reinterpret_cast<const unsigned int*>(u.m_codes + idx));
            if (MODE == 2) {
                b2v = __ldg(reinterpret_cast<const float4*>(u.b2 + col));
                a2i = __ldg(u.a2 + row);
            }
            float pn[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float uu = (f4get(gv, j) * ai) * f4get(bv, j);
                const float uh = uu * icf;
                float upd = uh;
                if (MODE > 0) {
                    const float mh = s8_to_float((mw >> (8 * j)) & 0xFFu) * dm[c / CPBM];
                    const float mk = u.beta1 * mh + u.omb1 * uh;
                    mf[4 * c + j] = mk;
                    cabs[c] = umix<true>(cabs[c], f2u(mk) & 0x7FFFFFFFu);
                    upd = MODE == 2 ? (mk * a2i) * f4get(b2v, j) : mk;
                }
                pn[j] = f4get(pv, j) * u.decay - u.lr * upd;
            }
            __stcs(reinterpret_cast<float4*>(u.p + idx), make_float4(pn[0], pn[1], pn[2], pn[3]));
        }
        if (MODE == 0) return;
        uint32_t babs[NBM];
        warp_blocks_reduce<CPBM, true>(cabs, babs);
        if (wpbm > 1) babs[0] = cta_group_reduce<true>(babs[0], s_part, wpbm);
        float ms[NBM], sc[NBM], inv[NBM];
#pragma unroll
        for (int b = 0; b < NBM; ++b) {
            ms[b] = u2f(babs[b]);
            sc[b] = 1.0f;
            inv[b] = 0.0f;
            if (ms[b] > 0.0f) uf8_encode_consts(ms[b], sc[b], inv[b]);
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int64_t idx = chunk_index(seg0, c, lane);
            const int b = c / CPBM;
            uint32_t qm = 0;
            if (ms[b] > 0.0f) {
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    qm |= ((uint32_t)uf8_quantize(mf[4 * c + j], sc[b], inv[b]) & 0xFFu) << (8 * j);
            }
            if (idx < u.n) __stcs(reinterpret_cast<unsigned int*>(u.m_codes + idx), qm);
        }
        if (lane == 0 && (warp % wpbm) == 0) {
#pragma unroll
            for (int b = 0; b < NBM; ++b)
                if (mb0 + b < nmb) u.m_absmax[mb0 + b] = ms[b];
        }
    }
}

template <int MODE, int CPBM>
__global__ void __launch_bounds__(kThreads)
update_kernel(UpdateArgs u, int64_t ntiles) {
    pdl_entry();
    __shared__ uint32_t s_part[kThreads / 32];
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x)
        update_tile<MODE, CPBM>(u, tile, s_part);
}

// ------------------------------------------------------------- host side --
// The sums kernels' dynamic shared memory (above the 48 KB default: one
// opt-in per kernel; a refusal shows up as a failed launch).
template <typename K>
static size_t sumsq_smem_optin(K kernel, size_t bytes) {
    cudaFuncSetAttribute((const void*)kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)bytes);
    return bytes;
}

template <int MODE>
static void launch_sumsq(dim3 grid, const float* g, int rows, int cols, const ResidualArgs& ra,
                         double* rowpart, double* colpart, cudaStream_t st) {
    static const size_t smem = sumsq_smem_optin(sumsq_kernel<MODE>, SumsqSmem<MODE>::kBytes);
    pdl_launch(true, sumsq_kernel<MODE>, dim3(grid), dim3(kThreads), smem, st, g, rows, cols, ra,
               rowpart, colpart);
}
static int cpb_of(int block) { return block >= 512 ? 4 : block / 128; }

template <int MODE>
static int launch_update(const UpdateArgs& u, cudaStream_t st) {
    const int64_t ntiles = blocks_of(u.n, kTile);
    const int cpb = MODE == 0 ? 4 : cpb_of(u.m_block);
    const void* k = cpb == 1 ? (const void*)update_kernel<MODE, 1>
                  : cpb == 2 ? (const void*)update_kernel<MODE, 2>
                             : (const void*)update_kernel<MODE, 4>;
    const int grid = persistent_grid(k, kThreads, 0, ntiles);
    if (cpb == 1) pdl_launch(true, update_kernel<MODE, 1>, dim3(grid), dim3(kThreads), 0, st, u,
                             ntiles);
    else if (cpb == 2) pdl_launch(true, update_kernel<MODE, 2>, dim3(grid), dim3(kThreads), 0, st,
                                  u, ntiles);
    else pdl_launch(true, update_kernel<MODE, 4>, dim3(grid), dim3(kThreads), 0, st, u, ntiles);
    return check_launch();
}

static int check_matrix(const float* p, const float* g, int64_t rows, int64_t cols) {
    if (!p || !g || rows < 1 || cols < 1) return ALQ_ERR_INVALID_ARG;
    if (cols % 4 != 0 || rows * cols >= (int64_t)1 << 31) return ALQ_ERR_UNSUPPORTED;
    if (!aligned(p, 16) || !aligned(g, 16)) return ALQ_ERR_ALIGN;
    return ALQ_OK;
}

// bits 8 or 16: AL codes with block metadata; 32: the unquantized fp32 role
// (codes point to fp32 values, meta is unused and may be NULL).
static int check_factor(const void* codes, const float* meta, int bits, int block) {
    if (!codes || (bits != 32 && !meta)) return ALQ_ERR_INVALID_ARG;
    if ((bits != 8 && bits != 16 && bits != 32) || !valid_block(block)) return ALQ_ERR_UNSUPPORTED;
    if (!aligned(codes, 16) || (bits != 32 && !aligned(meta, 8))) return ALQ_ERR_ALIGN;
    return ALQ_OK;
}

static int check_momentum(const int8_t* codes, const float* absmax, int block) {
    if (!codes || !absmax) return ALQ_ERR_INVALID_ARG;
    if (!valid_block(block)) return ALQ_ERR_UNSUPPORTED;
    if (!aligned(codes, 16) || !aligned(absmax, 4)) return ALQ_ERR_ALIGN;
    return ALQ_OK;
}

static FactorDesc factor_desc(const double* part, int nparts, int64_t len, int64_t mean_len,
                              double add_eps, float beta, float omb, void* codes, float* meta,
                              int bits, int block, float floor_, float* fresh) {
    FactorDesc f;
    f.part = part;
    f.nparts = nparts;
    f.len = len;
    f.mean_len = (double)mean_len;
    f.add_eps = add_eps;
    f.beta = beta;
    f.omb = omb;
    f.codes = codes;
    f.meta = meta;
    f.bits = bits;
    f.block = block;
    f.log_floor = floor_;
    f.fresh = fresh;
    return f;
}

// One launch of the factor pass for a row and a column factor (same block).
static void launch_factor(const FactorDesc& fr, const FactorDesc& fc, double* rsum,
                          cudaStream_t st) {
    const int nb0 = (int)blocks_of(fr.len, fr.block), nb1 = (int)blocks_of(fc.len, fc.block);
    const int kpt = fr.block <= kThreads ? 1 : fr.block / kThreads;
    const unsigned grid = (unsigned)(nb0 + nb1);
    switch (kpt) {
        case 1: pdl_launch(true, factor_kernel<1>, dim3(grid), dim3(kThreads), 0, st, fr, fc, nb0,
                           rsum); break;
        case 2: pdl_launch(true, factor_kernel<2>, dim3(grid), dim3(kThreads), 0, st, fr, fc, nb0,
                           rsum); break;
        case 4: pdl_launch(true, factor_kernel<4>, dim3(grid), dim3(kThreads), 0, st, fr, fc, nb0,
                           rsum); break;
        case 8: pdl_launch(true, factor_kernel<8>, dim3(grid), dim3(kThreads), 0, st, fr, fc, nb0,
                           rsum); break;
        default: pdl_launch(true, factor_kernel<16>, dim3(grid), dim3(kThreads), 0, st, fr, fc, nb0,
                            rsum); break;
    }
}

// G pass 1 (g^2 sums), factor update, scales, G pass 2 (RMS) -> a, b, icf.
static int second_moment_passes(const float* g, int64_t rows, int64_t cols, const FacWs& w,
                                FactorDesc fr, FactorDesc fc, float clip_d, cudaStream_t st,
                                float* a, float* b) {
    const int ncb = (int)blocks_of(cols, kFC), nrb = (int)blocks_of(rows, kFR);
    ResidualArgs none{};
    none.one = 1.0f;
    launch_sumsq<0>(dim3(ncb, nrb), g, (int)rows, (int)cols, none, w.rowpart, w.colpart, st);
    const int nb0 = (int)blocks_of(rows, fr.block);
    launch_factor(fr, fc, w.rsum, st);
    pdl_launch(true, scale_kernel, dim3((unsigned)blocks_of(rows + cols, kThreads)),
               dim3(kThreads), 0, st, fr.fresh, (int)rows, fc.fresh, (int)cols, w.rsum, nb0, a, b,
               w.ticket);
    const int64_t n = rows * cols;
    const int64_t ntiles = blocks_of(n, kTile);
    const UsqArgs q{g, n, make_divider((uint32_t)cols), a, b, w.upart, w.ticket, w.scal, 0.0f};
    const int64_t nchunks = blocks_of(ntiles, kUsqChunk);
    pdl_launch(true, usq_kernel,
               dim3(persistent_grid((const void*)usq_kernel, kThreads, 0, nchunks)),
               dim3(kThreads), 0, st, q, clip_d);
    return check_launch();
}

}  // namespace alq

using namespace alq;

extern "C" {

int al_workspace_size(int op, int64_t rows, int64_t cols, int rank, size_t* bytes) {
    if (!bytes || rows < 1 || cols < 1) return ALQ_ERR_INVALID_ARG;
    if (op == AL_OP_ADAFACTOR || op == AL_OP_CAME) {
        *bytes = fac_layout(nullptr, rows, cols).bytes;
        return ALQ_OK;
    }
    if (op == AL_OP_APOLLO) {
        if (rank < 1) return ALQ_ERR_INVALID_ARG;
        return al_apollo_workspace(rows, cols, rank, bytes);
    }
    return ALQ_ERR_INVALID_ARG;
}

int al_adafactor_step(float* p, const float* g, int64_t rows, int64_t cols, void* r_codes,
                      float* r_meta, void* c_codes, float* c_meta, int fac_bits, int fac_block,
                      int8_t* m_codes, float* m_absmax, int m_block,
                      const al_adafactor_hp* hp, int64_t t, void* workspace, size_t ws_bytes,
                      void* stream) {
    int st = check_matrix(p, g, rows, cols);
    if (st) return st;
    if (!hp || t < 1 || !(hp->eps1 > 0.0f) || !(hp->clip_d > 0.0f)) return ALQ_ERR_INVALID_ARG;
    st = check_factor(r_codes, r_meta, fac_bits, fac_block);
    if (!st) st = check_factor(c_codes, c_meta, fac_bits, fac_block);
    if (!st && m_codes) st = check_momentum(m_codes, m_absmax, m_block);
    if (st) return st;
    const FacWs w = fac_layout(workspace, rows, cols);
    if (!workspace || ws_bytes < w.bytes || !aligned(workspace, 256)) return ALQ_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;

    const double omr_d = pow((double)t, (double)hp->decay_rate);
    const float omr = (float)omr_d, rho = (float)(1.0 - omr_d);
    const int ncb = (int)blocks_of(cols, kFC), nrb = (int)blocks_of(rows, kFR);
    FactorDesc fr = factor_desc(w.rowpart, ncb, rows, cols, hp->eps1, rho, omr, r_codes, r_meta,
                                fac_bits, fac_block, hp->log_floor, w.fr);
    FactorDesc fc = factor_desc(w.colpart, nrb, cols, rows, hp->eps1, rho, omr, c_codes, c_meta,
                                fac_bits, fac_block, hp->log_floor, w.fc);
    st = second_moment_passes(g, rows, cols, w, fr, fc, hp->clip_d, s, w.a, w.b);
    if (st) return st;

    UpdateArgs u{};
    u.p = p;
    u.g = g;
    u.n = rows * cols;
    u.dv = make_divider((uint32_t)cols);
    u.a = w.a;
    u.b = w.b;
    u.scal = w.scal;
    u.m_codes = m_codes;
    u.m_absmax = m_absmax;
    u.m_block = m_codes ? m_block : 4096;
    u.beta1 = hp->beta1;
    u.omb1 = (float)(1.0 - (double)hp->beta1);
    u.decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    u.lr = hp->lr;
    return m_codes ? launch_update<1>(u, s) : launch_update<0>(u, s);
}

int al_came_step(float* p, const float* g, int64_t rows, int64_t cols, void* vr_codes,
                 float* vr_meta, void* vc_codes, float* vc_meta, int v_bits, int v_block,
                 void* cr_codes, float* cr_meta, void* cc_codes, float* cc_meta, int c_bits,
                 int c_block, int8_t* m_codes, float* m_absmax, int m_block,
                 const al_came_hp* hp, int64_t t, void* workspace, size_t ws_bytes,
                 void* stream) {
    int st = check_matrix(p, g, rows, cols);
    if (st) return st;
    if (!hp || t < 1 || !(hp->eps1 > 0.0f) || !(hp->eps2 > 0.0f) || !(hp->clip_d > 0.0f))
        return ALQ_ERR_INVALID_ARG;
    st = check_factor(vr_codes, vr_meta, v_bits, v_block);
    if (!st) st = check_factor(vc_codes, vc_meta, v_bits, v_block);
    if (!st) st = check_factor(cr_codes, cr_meta, c_bits, c_block);
    if (!st) st = check_factor(cc_codes, cc_meta, c_bits, c_block);
    if (!st) st = check_momentum(m_codes, m_absmax, m_block);
    if (st) return st;
    const FacWs w = fac_layout(workspace, rows, cols);
    if (!workspace || ws_bytes < w.bytes || !aligned(workspace, 256)) return ALQ_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;

    const float omb1 = (float)(1.0 - (double)hp->beta1);
    const float omb2 = (float)(1.0 - (double)hp->beta2);
    const float omb3 = (float)(1.0 - (double)hp->beta3);
    const int ncb = (int)blocks_of(cols, kFC), nrb = (int)blocks_of(rows, kFR);
    FactorDesc fr = factor_desc(w.rowpart, ncb, rows, cols, hp->eps1, hp->beta2, omb2, vr_codes,
                                vr_meta, v_bits, v_block, hp->log_floor_v, w.fr);
    FactorDesc fc = factor_desc(w.colpart, nrb, cols, rows, hp->eps1, hp->beta2, omb2, vc_codes,
                                vc_meta, v_bits, v_block, hp->log_floor_v, w.fc);
    st = second_moment_passes(g, rows, cols, w, fr, fc, hp->clip_d, s, w.a, w.b);
    if (st) return st;

    // residual (u_hat - m)^2 + eps2 from the old momentum codes, its factored
    // confidence (beta3) and the confidence scales
    ResidualArgs ra{m_codes, m_absmax, 0, w.a, w.b, w.scal, hp->beta1, omb1, hp->eps2, 1.0f, 0.0f};
    while ((1 << ra.m_shift) < m_block) ++ra.m_shift;
    launch_sumsq<1>(dim3(ncb, nrb), g, (int)rows, (int)cols, ra, w.rowpart, w.colpart, s);
    FactorDesc cr = factor_desc(w.rowpart, ncb, rows, cols, 0.0, hp->beta3, omb3, cr_codes,
                                cr_meta, c_bits, c_block, hp->log_floor_c, w.fr2);
    FactorDesc cc = factor_desc(w.colpart, nrb, cols, rows, 0.0, hp->beta3, omb3, cc_codes,
                                cc_meta, c_bits, c_block, hp->log_floor_c, w.fc2);
    const int nb0 = (int)blocks_of(rows, c_block), nb1 = (int)blocks_of(cols, c_block);
    launch_factor(cr, cc, w.rsum2, s);
    pdl_launch(true, scale_kernel, dim3((unsigned)blocks_of(rows + cols, kThreads)),
               dim3(kThreads), 0, s, w.fr2, (int)rows, w.fc2, (int)cols, w.rsum2,
               (int)blocks_of(rows, cr.block), w.a2, w.b2, nullptr);
    st = check_launch();
    if (st) return st;

    UpdateArgs u{};
    u.p = p;
    u.g = g;
    u.n = rows * cols;
    u.dv = make_divider((uint32_t)cols);
    u.a = w.a;
    u.b = w.b;
    u.a2 = w.a2;
    u.b2 = w.b2;
    u.scal = w.scal;
    u.m_codes = m_codes;
    u.m_absmax = m_absmax;
    u.m_block = m_block;
    u.beta1 = hp->beta1;
    u.omb1 = omb1;
    u.decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    u.lr = hp->lr;
    return launch_update<2>(u, s);
}

}  // extern "C"

// ------------------------------------------------------- grouped step --
namespace alq {

constexpr uint32_t kFacPlanMagic = 0x46504C31u;  // "FPL1"

struct FacPlanHeader {
    uint32_t magic;
    int32_t nmat, op, reserved;
};
constexpr size_t kFacEntryOffset = 64;

// One matrix of a grouped plan: its arguments, its scratch, and the first
// tile of each pass in the launch that covers all matrices.
struct FacEntry {
    float* p;
    const float* g;
    int64_t rows, cols, n, ntiles;
    Divider dv;
    void* vr_codes;
    float* vr_meta;
    void* vc_codes;
    float* vc_meta;
    void* cr_codes;
    float* cr_meta;
    void* cc_codes;
    float* cc_meta;
    int8_t* m_codes;
    float* m_absmax;
    FacWs w;
    int32_t ncb, nrb;  // the sums passes' tile grid (columns, rows)
    int64_t sq_t0, fac_t0, fac2_t0, sc_t0, usq_t0, upd_t0;  // usq_t0 in RMS chunks
};

// Per-step scalars of the grouped passes.
struct FacStep {
    int op;
    int v_bits, v_block, c_bits, c_block, m_block, m_shift;
    float rho_v, omb_v;   // second-moment factor EMA (Adafactor: rho_t)
    float rho_c, omb_c;   // confidence factor EMA (CAME: beta3)
    double eps1;
    float log_floor_v, log_floor_c;
    float clip_d;
    float beta1, omb1, eps2, decay, lr;
    float one, zero;  // opaque 1 and 0 for the paired sums (see ff_sq2)
};

// The entry whose pass (first tile t0) holds a launch-wide tile: entries are
// in increasing t0 and every matrix has at least one tile in every pass.
__device__ __forceinline__ const FacEntry& fac_entry(const FacEntry* __restrict__ tab, int nmat,
                                                     int64_t tile, int64_t FacEntry::*t0) {
    int lo = 0, hi = nmat - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (tab[mid].*t0 <= tile) lo = mid; else hi = mid - 1;
    }
    return tab[lo];
}

// Forward cursor for persistent loops (a CTA's tiles only increase).
__device__ __forceinline__ int fac_advance(const FacEntry* __restrict__ tab, int nmat, int64_t tile,
                                           int cur, int64_t FacEntry::*t0) {
    while (cur + 1 < nmat && tab[cur + 1].*t0 <= tile) ++cur;
    return cur;
}

template <int MODE>
__global__ void __launch_bounds__(kThreads)
sumsq_multi_kernel(const FacEntry* __restrict__ tab, int nmat, FacStep fs) {
    pdl_entry();
    extern __shared__ __align__(16) unsigned char s_sumsq[];
    const FacEntry& e = fac_entry(tab, nmat, blockIdx.x, &FacEntry::sq_t0);
    const int64_t lt = blockIdx.x - e.sq_t0;
    ResidualArgs ra{};
    if (MODE == 1)
        ra = ResidualArgs{e.m_codes, e.m_absmax, fs.m_shift, e.w.a, e.w.b, e.w.scal,
                          fs.beta1, fs.omb1, fs.eps2, fs.one, fs.zero};
    ra.one = fs.one;
    ra.zero = fs.zero;
    sumsq_tile<MODE>(e.g, (int)e.rows, (int)e.cols, ra, e.w.rowpart, e.w.colpart,
                     (int)(lt % e.ncb), (int)(lt / e.ncb), s_sumsq);
}

// which = 0: the second-moment factors; 1: CAME's confidence factors.
template <int KPT>
__global__ void __launch_bounds__(kThreads)
factor_multi_kernel(const FacEntry* __restrict__ tab, int nmat, FacStep fs, int which) {
    pdl_entry();
    const FacEntry& e = fac_entry(tab, nmat, blockIdx.x, which ? &FacEntry::fac2_t0 : &FacEntry::fac_t0);
    const int64_t lt = blockIdx.x - (which ? e.fac2_t0 : e.fac_t0);
    const int block = which ? fs.c_block : fs.v_block;
    const int64_t nbr = blocks_of_dev(e.rows, block);
    const bool row = lt < nbr;
    FactorDesc f;
    f.part = row ? e.w.rowpart : e.w.colpart;
    f.nparts = row ? e.ncb : e.nrb;
    f.len = row ? e.rows : e.cols;
    f.mean_len = (double)(row ? e.cols : e.rows);
    f.add_eps = which ? 0.0 : fs.eps1;
    f.beta = which ? fs.rho_c : fs.rho_v;
    f.omb = which ? fs.omb_c : fs.omb_v;
    f.codes = which ? (row ? e.cr_codes : e.cc_codes) : (row ? e.vr_codes : e.vc_codes);
    f.meta = which ? (row ? e.cr_meta : e.cc_meta) : (row ? e.vr_meta : e.vc_meta);
    f.bits = which ? fs.c_bits : fs.v_bits;
    f.block = block;
    f.log_floor = which ? fs.log_floor_c : fs.log_floor_v;
    f.fresh = which ? (row ? e.w.fr2 : e.w.fc2) : (row ? e.w.fr : e.w.fc);
    double* rsum = row ? (which ? e.w.rsum2 : e.w.rsum) : nullptr;
    factor_block<KPT>(f, row ? lt : lt - nbr, rsum);
}

__global__ void __launch_bounds__(kThreads)
scale_multi_kernel(const FacEntry* __restrict__ tab, int nmat, FacStep fs, int which) {
    pdl_entry();
    const FacEntry& e = fac_entry(tab, nmat, blockIdx.x, &FacEntry::sc_t0);
    const int lt = (int)(blockIdx.x - e.sc_t0);
    if (which == 0)
        scale_tile(e.w.fr, (int)e.rows, e.w.fc, (int)e.cols, e.w.rsum,
                   (int)blocks_of_dev(e.rows, fs.v_block), e.w.a, e.w.b, e.w.ticket, lt);
    else
        scale_tile(e.w.fr2, (int)e.rows, e.w.fc2, (int)e.cols, e.w.rsum2,
                   (int)blocks_of_dev(e.rows, fs.c_block), e.w.a2, e.w.b2, nullptr, lt);
}

__global__ void __launch_bounds__(kThreads)
usq_multi_kernel(const FacEntry* __restrict__ tab, int nmat, int64_t nchunks, float clip_d,
                 float zero) {
    pdl_entry();
    __shared__ float2 s_w[kThreads / 32];
    __shared__ double s_d[kThreads];
    __shared__ bool s_last;
    int cur = 0;
    for (int64_t chunk = blockIdx.x; chunk < nchunks; chunk += gridDim.x) {
        cur = fac_advance(tab, nmat, chunk, cur, &FacEntry::usq_t0);
        const FacEntry& e = tab[cur];
        const UsqArgs q{e.g, e.n, e.dv, e.w.a, e.w.b, e.w.upart, e.w.ticket, e.w.scal, zero};
        usq_chunk(q, chunk - e.usq_t0, clip_d, s_w, s_d, &s_last);
    }
}

template <int MODE, int CPBM>
__global__ void __launch_bounds__(kThreads)
update_multi_kernel(const FacEntry* __restrict__ tab, int nmat, int64_t ntiles, FacStep fs) {
    pdl_entry();
    __shared__ uint32_t s_part[kThreads / 32];
    int cur = 0;
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        cur = fac_advance(tab, nmat, tile, cur, &FacEntry::upd_t0);
        const FacEntry& e = tab[cur];
        UpdateArgs u{};
        u.p = e.p;
        u.g = e.g;
        u.n = e.n;
        u.dv = e.dv;
        u.a = e.w.a;
        u.b = e.w.b;
        u.a2 = e.w.a2;
        u.b2 = e.w.b2;
        u.scal = e.w.scal;
        u.m_codes = e.m_codes;
        u.m_absmax = e.m_absmax;
        u.m_block = MODE > 0 ? fs.m_block : 4096;
        u.beta1 = fs.beta1;
        u.omb1 = fs.omb1;
        u.decay = fs.decay;
        u.lr = fs.lr;
        update_tile<MODE, CPBM>(u, tile - e.upd_t0, s_part);
    }
}

static size_t fac_plan_size(int nmat) {
    return kFacEntryOffset + (size_t)nmat * sizeof(FacEntry);
}

static int check_factored_matrices(const al_factored_matrix* mats, int nmat) {
    if (!mats || nmat < 1) return ALQ_ERR_INVALID_ARG;
    for (int i = 0; i < nmat; ++i)
        if (mats[i].rows < 1 || mats[i].cols < 1) return ALQ_ERR_INVALID_ARG;
    return ALQ_OK;
}

template <int KPT>
static void launch_factor_multi(const FacEntry* tab, int nmat, const FacStep& fs, int which,
                                int64_t tiles, cudaStream_t st) {
    pdl_launch(false, factor_multi_kernel<KPT>, dim3((unsigned)tiles), dim3(kThreads), 0, st, tab,
               nmat, fs, which);
}

static void factor_multi(const FacEntry* tab, int nmat, const FacStep& fs, int which,
                         int64_t tiles, cudaStream_t st) {
    const int block = which ? fs.c_block : fs.v_block;
    const int kpt = block <= kThreads ? 1 : block / kThreads;
    switch (kpt) {
        case 1: launch_factor_multi<1>(tab, nmat, fs, which, tiles, st); break;
        case 2: launch_factor_multi<2>(tab, nmat, fs, which, tiles, st); break;
        case 4: launch_factor_multi<4>(tab, nmat, fs, which, tiles, st); break;
        case 8: launch_factor_multi<8>(tab, nmat, fs, which, tiles, st); break;
        default: launch_factor_multi<16>(tab, nmat, fs, which, tiles, st); break;
    }
}

template <int MODE>
static void update_multi(const FacEntry* tab, int nmat, int64_t tiles, const FacStep& fs,
                         cudaStream_t st) {
    const int cpb = MODE == 0 ? 4 : cpb_of(fs.m_block);
    const void* k = cpb == 1 ? (const void*)update_multi_kernel<MODE, 1>
                  : cpb == 2 ? (const void*)update_multi_kernel<MODE, 2>
                             : (const void*)update_multi_kernel<MODE, 4>;
    const int grid = persistent_grid(k, kThreads, 0, tiles);
    if (cpb == 1) pdl_launch(false, update_multi_kernel<MODE, 1>, dim3(grid), dim3(kThreads), 0, st,
                             tab, nmat, tiles, fs);
    else if (cpb == 2) pdl_launch(false, update_multi_kernel<MODE, 2>, dim3(grid), dim3(kThreads),
                                  0, st, tab, nmat, tiles, fs);
    else pdl_launch(false, update_multi_kernel<MODE, 4>, dim3(grid), dim3(kThreads), 0, st, tab,
                    nmat, tiles, fs);
}

// The passes both optimizers share: g^2 sums, second-moment factors, their
// scales (which also zero the RMS tickets), the RMS pass.
static void second_moment_multi(const FacEntry* tab, const al_factored_info* info,
                                const FacStep& fs, cudaStream_t st) {
    static const size_t smem0 = sumsq_smem_optin(sumsq_multi_kernel<0>, SumsqSmem<0>::kBytes);
    pdl_launch(false, sumsq_multi_kernel<0>,
               dim3((unsigned)info->sumsq_tiles), dim3(kThreads), smem0, st, tab, info->nmat, fs);
    factor_multi(tab, info->nmat, fs, 0, info->factor_tiles, st);
    pdl_launch(false, scale_multi_kernel,
               dim3((unsigned)info->scale_tiles), dim3(kThreads), 0, st, tab, info->nmat, fs, 0);
    pdl_launch(false, usq_multi_kernel,
               dim3(persistent_grid((const void*)usq_multi_kernel, kThreads, 0, info->rms_chunks)), dim3(kThreads), 0, st, tab, info->nmat, info->rms_chunks, fs.clip_d, fs.zero);
}

static int check_multi_call(const void* plan_dev, const al_factored_info* info, int op) {
    if (!plan_dev || !info || info->nmat < 1 || !info->workspace) return ALQ_ERR_INVALID_ARG;
    if (!aligned(plan_dev, 64)) return ALQ_ERR_ALIGN;
    if (info->op != op) return ALQ_ERR_INVALID_ARG;
    return ALQ_OK;
}

}  // namespace alq

extern "C" {

int al_factored_plan_bytes(const al_factored_matrix* mats, int nmat, size_t* bytes) {
    if (!bytes) return ALQ_ERR_INVALID_ARG;
    const int rc = check_factored_matrices(mats, nmat);
    if (rc) return rc;
    *bytes = fac_plan_size(nmat);
    return ALQ_OK;
}

int al_factored_workspace_multi(const al_factored_matrix* mats, int nmat, size_t* bytes) {
    if (!bytes) return ALQ_ERR_INVALID_ARG;
    const int rc = check_factored_matrices(mats, nmat);
    if (rc) return rc;
    size_t tot = 0;
    for (int i = 0; i < nmat; ++i) tot += fac_layout(nullptr, mats[i].rows, mats[i].cols).bytes;
    *bytes = tot;
    return ALQ_OK;
}

int al_factored_plan(int op, const al_factored_matrix* mats, int nmat, int v_bits, int v_block,
                     int c_bits, int c_block, int m_block, void* workspace, size_t ws_bytes,
                     void* plan_host, size_t plan_bytes, al_factored_info* info) {
    int rc = check_factored_matrices(mats, nmat);
    if (rc) return rc;
    if (!plan_host || !info || (op != AL_OP_ADAFACTOR && op != AL_OP_CAME))
        return ALQ_ERR_INVALID_ARG;
    const bool came = op == AL_OP_CAME;
    const bool has_m = mats[0].m_codes != nullptr;
    for (int i = 0; i < nmat; ++i) {
        const al_factored_matrix& m = mats[i];
        rc = check_matrix(m.p, m.g, m.rows, m.cols);
        if (!rc) rc = check_factor(m.vr_codes, m.vr_meta, v_bits, v_block);
        if (!rc) rc = check_factor(m.vc_codes, m.vc_meta, v_bits, v_block);
        if (!rc && came) rc = check_factor(m.cr_codes, m.cr_meta, c_bits, c_block);
        if (!rc && came) rc = check_factor(m.cc_codes, m.cc_meta, c_bits, c_block);
        if (!rc && (m.m_codes != nullptr) != has_m) rc = ALQ_ERR_INVALID_ARG;
        if (!rc && came && !has_m) rc = ALQ_ERR_INVALID_ARG;
        if (!rc && has_m) rc = check_momentum(m.m_codes, m.m_absmax, m_block);
        if (rc) return rc;
    }
    size_t need = 0;
    al_factored_workspace_multi(mats, nmat, &need);
    if (!workspace || ws_bytes < need || !aligned(workspace, 256)) return ALQ_ERR_WORKSPACE;
    if (plan_bytes < fac_plan_size(nmat)) return ALQ_ERR_INVALID_ARG;

    char* base = (char*)plan_host;
    memset(base, 0, fac_plan_size(nmat));
    FacPlanHeader h{kFacPlanMagic, nmat, op, 0};
    memcpy(base, &h, sizeof(h));
    char* ws = (char*)workspace;
    memset(info, 0, sizeof(*info));
    for (int i = 0; i < nmat; ++i) {
        const al_factored_matrix& m = mats[i];
        FacEntry e;
        memset(&e, 0, sizeof(e));
        e.p = m.p;
        e.g = m.g;
        e.rows = m.rows;
        e.cols = m.cols;
        e.n = m.rows * m.cols;
        e.ntiles = blocks_of(e.n, kTile);
        e.dv = make_divider((uint32_t)m.cols);
        e.vr_codes = m.vr_codes;
        e.vr_meta = m.vr_meta;
        e.vc_codes = m.vc_codes;
        e.vc_meta = m.vc_meta;
        e.cr_codes = came ? m.cr_codes : nullptr;
        e.cr_meta = came ? m.cr_meta : nullptr;
        e.cc_codes = came ? m.cc_codes : nullptr;
        e.cc_meta = came ? m.cc_meta : nullptr;
        e.m_codes = has_m ? m.m_codes : nullptr;
        e.m_absmax = has_m ? m.m_absmax : nullptr;
        e.w = fac_layout(ws, m.rows, m.cols);
        ws += e.w.bytes;
        e.ncb = (int32_t)blocks_of(m.cols, kFC);
        e.nrb = (int32_t)blocks_of(m.rows, kFR);
        e.sq_t0 = info->sumsq_tiles;
        e.fac_t0 = info->factor_tiles;
        e.fac2_t0 = info->factor2_tiles;
        e.sc_t0 = info->scale_tiles;
        e.usq_t0 = info->rms_chunks;
        e.upd_t0 = info->tiles;
        info->sumsq_tiles += (int64_t)e.ncb * e.nrb;
        info->factor_tiles += blocks_of(m.rows, v_block) + blocks_of(m.cols, v_block);
        if (came) info->factor2_tiles += blocks_of(m.rows, c_block) + blocks_of(m.cols, c_block);
        info->scale_tiles += blocks_of(m.rows + m.cols, kThreads);
        info->tiles += e.ntiles;
        info->rms_chunks += blocks_of(e.ntiles, kUsqChunk);
        info->total_params += e.n;
        memcpy(base + kFacEntryOffset + (size_t)i * sizeof(FacEntry), &e, sizeof(e));
    }
    // one launch per pass: its grid must fit a launch
    if (info->sumsq_tiles > INT32_MAX || info->factor_tiles > INT32_MAX ||
        info->factor2_tiles > INT32_MAX || info->scale_tiles > INT32_MAX)
        return ALQ_ERR_UNSUPPORTED;
    info->nmat = nmat;
    info->op = op;
    info->v_bits = v_bits;
    info->v_block = v_block;
    info->c_bits = came ? c_bits : 0;
    info->c_block = came ? c_block : 0;
    info->m_block = has_m ? m_block : 0;
    info->has_momentum = has_m ? 1 : 0;
    info->workspace = workspace;
    return ALQ_OK;
}

int al_adafactor_step_multi(const void* plan_dev, const al_factored_info* info,
                            const al_adafactor_hp* hp, int64_t t, void* stream) {
    int rc = check_multi_call(plan_dev, info, AL_OP_ADAFACTOR);
    if (rc) return rc;
    if (!hp || t < 1 || !(hp->eps1 > 0.0f) || !(hp->clip_d > 0.0f)) return ALQ_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    const FacEntry* tab = (const FacEntry*)((const char*)plan_dev + kFacEntryOffset);
    const double omr_d = pow((double)t, (double)hp->decay_rate);
    FacStep fs{};
    fs.op = AL_OP_ADAFACTOR;
    fs.v_bits = info->v_bits;
    fs.v_block = info->v_block;
    fs.m_block = info->has_momentum ? info->m_block : 4096;
    fs.rho_v = (float)(1.0 - omr_d);
    fs.omb_v = (float)omr_d;
    fs.eps1 = hp->eps1;
    fs.log_floor_v = hp->log_floor;
    fs.clip_d = hp->clip_d;
    fs.beta1 = hp->beta1;
    fs.omb1 = (float)(1.0 - (double)hp->beta1);
    fs.decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    fs.lr = hp->lr;
    fs.one = 1.0f;
    second_moment_multi(tab, info, fs, st);
    if (info->has_momentum)
        update_multi<1>(tab, info->nmat, info->tiles, fs, st);
    else
        update_multi<0>(tab, info->nmat, info->tiles, fs, st);
    return check_launch();
}

int al_came_step_multi(const void* plan_dev, const al_factored_info* info, const al_came_hp* hp,
                       int64_t t, void* stream) {
    int rc = check_multi_call(plan_dev, info, AL_OP_CAME);
    if (rc) return rc;
    if (!hp || t < 1 || !(hp->eps1 > 0.0f) || !(hp->eps2 > 0.0f) || !(hp->clip_d > 0.0f))
        return ALQ_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    const FacEntry* tab = (const FacEntry*)((const char*)plan_dev + kFacEntryOffset);
    FacStep fs{};
    fs.op = AL_OP_CAME;
    fs.v_bits = info->v_bits;
    fs.v_block = info->v_block;
    fs.c_bits = info->c_bits;
    fs.c_block = info->c_block;
    fs.m_block = info->m_block;
    while ((1 << fs.m_shift) < fs.m_block) ++fs.m_shift;
    fs.rho_v = hp->beta2;
    fs.omb_v = (float)(1.0 - (double)hp->beta2);
    fs.rho_c = hp->beta3;
    fs.omb_c = (float)(1.0 - (double)hp->beta3);
    fs.eps1 = hp->eps1;
    fs.eps2 = hp->eps2;
    fs.log_floor_v = hp->log_floor_v;
    fs.log_floor_c = hp->log_floor_c;
    fs.clip_d = hp->clip_d;
    fs.beta1 = hp->beta1;
    fs.omb1 = (float)(1.0 - (double)hp->beta1);
    fs.decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    fs.lr = hp->lr;
    fs.one = 1.0f;
    second_moment_multi(tab, info, fs, st);
    // residual sums, confidence factors and their scales, update
    static const size_t smem1 = sumsq_smem_optin(sumsq_multi_kernel<1>, SumsqSmem<1>::kBytes);
    pdl_launch(false, sumsq_multi_kernel<1>,
               dim3((unsigned)info->sumsq_tiles), dim3(kThreads), smem1, st, tab, info->nmat, fs);
    factor_multi(tab, info->nmat, fs, 1, info->factor2_tiles, st);
    pdl_launch(false, scale_multi_kernel,
               dim3((unsigned)info->scale_tiles), dim3(kThreads), 0, st, tab, info->nmat, fs, 1);
    update_multi<2>(tab, info->nmat, info->tiles, fs, st);
    return check_launch();
}

}  // extern "C"
