// alq_adamw.cu -- fused AdamW step with UF8 momentum and AL-coded second
// moment (Sec. 3.1 Eq. (1); Sec. 6.2; fused as in Sec. 7.1).
//
// One HBM pass per element: read p, g (fp32), the momentum and second-moment
// codes and their per-block metadata; decode; update m, v and p in fp32; write
// p; reduce each block's absmax (momentum) and minimum-positive / maximum
// (second moment) with warp reductions; derive the new block constants; encode
// and write the codes and metadata. 16.09 bytes per parameter for AL8/UF8
// with 256-element blocks.
//
// Every state value, code and block constant is the exact fp32 result of the
// oracle's operation order. The update direction u = m / (sqrt(v) c2 + eps),
// which moves only p, takes the hardware's approximate square root and
// reciprocal: a parameter differs from the IEEE result by a few ulp of its
// step lr |u|, far inside the 1e-5 relative parameter tolerance.
//
// The same kernel serves one tensor (descriptor passed by value) or a plan of
// many tensors (descriptor table in device memory, tiles never crossing a
// tensor boundary). The grid is persistent: each CTA walks tiles with a
// stride of gridDim.x and a forward-only cursor into the descriptor table.
// The exp2/log2 tables of the codec's two-float levels and block bounds are
// read from shared memory in this translation unit (copied once per CTA).
#define ALQ_SMEM_TABLES 1
#include "alq_kernels.cuh"

namespace alq {

// Geometry of this kernel: 4 chunks per lane (16 elements), 512-element
// segments per warp (two blocks of 256), 4096-element tiles per CTA; blocks
// of 128..4096.
constexpr int kCH = 4;
constexpr int kASeg = 128 * kCH;
constexpr int kATile = 8 * kASeg;

// ------------------------------------------------ ragged-segment I/O --
// Masked loads and stores of a segment that crosses the end of its tensor
// (one per tensor), out of line so that the fused loop body stays compact.
template <int VBITS>
struct SegIn {
    float4 g[kCH], p[kCH];
    uint32_t mw[kCH], vw[kCH * VBITS / 8];
};

template <int VBITS>
static __device__ __noinline__ SegIn<VBITS> load_seg_masked(const float* g, const float* p,
                                                            const int8_t* m_codes,
                                                            const void* v_codes, int64_t e0,
                                                            int64_t n) {
    SegIn<VBITS> r;
#pragma unroll
    for (int c = 0; c < kCH; ++c) {
        const int64_t idx = e0 + 128 * c;
        r.g[c] = load4f(g, idx, n);
        r.p[c] = load4f(p, idx, n);
        r.mw[c] = load4b((const uint8_t*)m_codes, idx, n);
        if constexpr (VBITS == 8) {
            r.vw[c] = load4b((const uint8_t*)v_codes, idx, n);
        } else {
            const uint2 h = load4h((const uint16_t*)v_codes, idx, n);
            r.vw[2 * c] = h.x;
            r.vw[2 * c + 1] = h.y;
        }
    }
    return r;
}

static __device__ __noinline__ void store_p_masked(float* p, int64_t idx, int64_t n, float4 v) {
    store4f(p, idx, n, v);
}

template <int VBITS>
static __device__ __noinline__ void store_codes_masked(int8_t* m_codes, void* v_codes, int64_t idx,
                                                       int64_t n, uint32_t qm, uint2 qv) {
    store4b((uint8_t*)m_codes, idx, n, qm);
    if constexpr (VBITS == 8)
        store4b((uint8_t*)v_codes, idx, n, qv.x);
    else
        store4h((uint16_t*)v_codes, idx, n, qv);
}

// Step scalars as broadcast pairs: the element arithmetic runs on pairs of
// elements with the paired fp32 instructions (each component rounded exactly
// as the scalar operation), and a pair operand held in the kernel's
// parameter space costs no registers.
struct AdamWPairs {
    float2 decay, nstep, c2, omb1, omb2, beta1, beta2, eps;
    float2 one;   // (1, 1) and (0, 0), opaque to the compiler: f * one + c
    float2 zero;  // rounds as f + c, fma(x, y, zero) as x y
    float log_floor;
};

static AdamWPairs adamw_pairs(const AdamWScalars& s) {
    AdamWPairs q;
    q.decay = make_float2(s.decay, s.decay);
    q.nstep = make_float2(-s.step, -s.step);  // p1 + (-step) q == p1 - step q exactly
    q.c2 = make_float2(s.c2, s.c2);
    q.omb1 = make_float2(s.omb1, s.omb1);
    q.omb2 = make_float2(s.omb2, s.omb2);
    q.beta1 = make_float2(s.beta1, s.beta1);
    q.beta2 = make_float2(s.beta2, s.beta2);
    q.eps = make_float2(s.eps, s.eps);
    q.one = make_float2(1.0f, 1.0f);
    q.zero = make_float2(0.0f, 0.0f);
    q.log_floor = s.log_floor;
    return q;
}

// Barrier of the nwarps warps of a group (named barrier id; a group of
// every warp of the CTA is the whole CTA).
__device__ __forceinline__ void group_sync(int id, int nwarps) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(32 * nwarps) : "memory");
}

__device__ __forceinline__ PlanEntry plan_entry(const PlanEntry* table, int ntensors,
                                                const PlanEntry& single, int64_t tile,
                                                int& cur) {
    if (!table) return single;
    while (cur + 1 < ntensors && table[cur + 1].first_tile <= tile) ++cur;
    return table[cur];
}

// Three CTAs per SM (80 registers, no spills): 16 elements a lane halve
// the per-segment work of the block constants, plan walk and reductions
// (two 256-blocks' bounds in one lane pass, their levels in one paired
// pass); 8 elements a lane at four CTAs per SM ran 0.7% slower at blocks of
// 256 and 15% slower at blocks of 2048.
// WIDE (AL8, WPBV > 1): blocks wider than a segment (1024 .. 4096
// elements), whose value table is built once per block by the warps that
// share it.
// WPBV: warps per V block (v_block / 512 for blocks of at least a segment,
// else 1), a compile-time constant of each instantiation.
template <int CPBV, int CPBM, int VBITS, int WPBV = 1>
__global__ void __launch_bounds__(kThreads, 3)
adamw_fused_kernel(const PlanEntry* __restrict__ table, int ntensors, int64_t total_tiles,
                   PlanEntry single, int v_block, int m_block, AdamWPairs s) {
    // a block narrower than a segment is 128 CPB elements: its geometry is
    // the instantiation's (v_block and m_block are then those sizes)
    constexpr bool WIDE = VBITS == 8 && WPBV > 1;
    const int v_shift = CPBV < kCH ? 7 + ilog2c(CPBV) : 7 + ilog2c(kCH) + ilog2c(WPBV);
    const int m_shift = CPBM < kCH ? 7 + ilog2c(CPBM) : __ffs(m_block) - 1;
    constexpr int NBV = kCH / CPBV;
    constexpr int NBM = kCH / CPBM;
    constexpr int NE = 4 * kCH;
    constexpr float Lm2 = VBITS == 8 ? 254.0f : 65534.0f;
    // level tables; one block per segment: two slots, alternating between
    // iterations, written by the even warp of each pair
    __shared__ __align__(16) float2 s_tab[kThreads / 32][NBV == 1 ? 2 : 1][NBV * 32];
    __shared__ float s_val[kThreads / 32][VBITS == 8 ? NBV * 256 : 1];
    __shared__ uint32_t s_part[2][3][kThreads / 32];
    // the warp index through a shuffle from lane 0: the compiler then knows it
    // is the same for the whole warp, and every branch on the segment's
    // position is a uniform one
    const int warp = __shfl_sync(0xFFFFFFFFu, (int)(threadIdx.x >> 5), 0), lane = threadIdx.x & 31;
    constexpr int wpbv = WPBV;
    const int wpbm = CPBM == kCH && m_block > kASeg ? m_block / kASeg : 1;
    const float kf = al8_table_k(lane);
    const Opaque2 ok2{s.one, s.zero};
    const int G = gridDim.x;
    // the 2^(j/1024) and log2 reduction tables of the level and bound
    // computations, 20 KB, into shared memory (their lookups sit on the
    // level pass's dependent chain)
    for (int i = threadIdx.x; i < 1024; i += kThreads) {
        s_kExp2Hi[i] = kExp2HiD[i];
        s_kExp2Lo[i] = kExp2LoD[i];
        s_kLog2C[i] = kLog2CD[i];
        s_kLog2Hi[i] = kLog2HiD[i];
        s_kLog2Lo[i] = kLog2LoD[i];
    }
    __syncthreads();
    int cur = 0;
    int parity = 0;  // slot of the next cross-warp block reduction
    int tslot = 0;   // level-table slot of this iteration
    int wit = 0;     // WIDE: this iteration's index within its look-ahead round
    int curL = 0;    // WIDE: descriptor cursor of the look-ahead lookups
    for (int64_t tile = blockIdx.x; tile < total_tiles; tile += G) {
        const PlanEntry d = plan_entry(table, ntensors, single, tile, cur);
        const int64_t n = d.n;
        const int64_t t0 = (tile - d.first_tile) * kATile;
        const int64_t seg0 = t0 + (int64_t)warp * kASeg;
        // ---- p, g and the codes of this lane's chunks
        const bool full = seg0 + kASeg <= n;  // warp-uniform: unmasked I/O
        const int64_t e0 = seg0 + 4 * lane;   // this lane's first element
        float4 g[kCH], p[kCH];
        uint32_t mw[kCH], vw[kCH * VBITS / 8];
        if (full) {
            // chunk c starts 128 c elements further: immediate offsets
            const float4* gp = reinterpret_cast<const float4*>(d.g + e0);
            const float4* pp = reinterpret_cast<const float4*>(d.p + e0);
            const unsigned* mp = reinterpret_cast<const unsigned*>(d.m_codes + e0);
#pragma unroll
            for (int c = 0; c < kCH; ++c) {
                g[c] = __ldcs(gp + 32 * c);
                p[c] = __ldcs(pp + 32 * c);
                mw[c] = __ldcs(mp + 32 * c);
                if constexpr (VBITS == 8) {
                    vw[c] = __ldcs(reinterpret_cast<const unsigned*>((const uint8_t*)d.v_codes + e0) + 32 * c);
                } else {
                    const uint2 h = __ldcs(reinterpret_cast<const uint2*>((const uint16_t*)d.v_codes + e0) + 32 * c);
                    vw[2 * c] = h.x;
                    vw[2 * c + 1] = h.y;
                }
            }
        } else {
            const SegIn<VBITS> r = load_seg_masked<VBITS>(d.g, d.p, d.m_codes, d.v_codes, e0, n);
#pragma unroll
            for (int c = 0; c < kCH; ++c) {
                g[c] = r.g[c];
                p[c] = r.p[c];
                mw[c] = r.mw[c];
            }
#pragma unroll
            for (int k = 0; k < kCH * VBITS / 8; ++k) vw[k] = r.vw[k];
        }

        // ---- previous block constants
        const int64_t nvb = (n + (1 << v_shift) - 1) >> v_shift, nmb = (n + (1 << m_shift) - 1) >> m_shift;
        const int64_t vb0 = seg0 >> v_shift, mb0 = seg0 >> m_shift;
        float olmin[NBV], odelta[NBV], dm[NBM];
#pragma unroll
        for (int b = 0; b < NBV; ++b) {
            float2 mt = make_float2(0.f, 0.f);
            if (vb0 + b < nvb) mt = __ldg(reinterpret_cast<const float2*>(d.v_meta) + vb0 + b);
            olmin[b] = mt.x;
            odelta[b] = mt.y;
        }
#pragma unroll
        for (int b = 0; b < NBM; ++b)
            dm[b] = (mb0 + b < nmb) ? __ldg(d.m_absmax + mb0 + b) / 127.0f : 0.0f;

        // ---- decode the previous states
        float vh[NE];
        if constexpr (VBITS == 8) {
            if constexpr (WIDE) {
                // every wpbv iterations, warp r of a group computes the levels
                // of the group's block at tile + r G (all at once, one
                // barrier); every iteration, each warp of the group its share
                // of the 255 values. A block's constants change only when
                // its own tile is processed, after they have been used.
                const int g0 = (warp / wpbv) * wpbv, r = warp - g0;
                if (wit == 0) {
                    float la[1] = {olmin[0]}, da[1] = {odelta[0]};
                    if (r > 0) {
                        la[0] = da[0] = 0.0f;
                        const int64_t tx = tile + (int64_t)r * G;
                        if (tx < total_tiles) {
                            const PlanEntry dx = plan_entry(table, ntensors, single, tx, curL);
                            const int64_t sx = (tx - dx.first_tile) * kATile + (int64_t)g0 * kASeg;
                            if (sx < dx.n) {
                                const float2 mt = __ldg(reinterpret_cast<const float2*>(dx.v_meta) + (sx >> v_shift));
                                la[0] = mt.x;
                                da[0] = mt.y;
                            }
                        }
                    }
                    al8_build_tables_soa(reinterpret_cast<float*>(s_tab[warp][0]), la[0], da[0], kf);
                    group_sync(1 + warp / wpbv, wpbv);
                }
                al8_values_part_soa(s_val[g0], reinterpret_cast<const float*>(s_tab[g0 + wit][0]),
                                    olmin[0], odelta[0], r, wpbv);
                group_sync(1 + warp / wpbv, wpbv);
                wit = wit + 1 == wpbv ? 0 : wit + 1;
            } else if constexpr (NBV == 1) {
                // warps 2k and 2k + 1 hold adjacent blocks of one tensor: the
                // even warp computes both blocks' levels in one paired pass
                // (the scalar pass's roundings, so the same entries) and the
                // pair meets at a 64-thread barrier. The slots alternate, so
                // the even warp never overwrites a table the odd one reads.
                if ((warp & 1) == 0) {
                    float l1 = 0.0f, d1 = 0.0f;
                    if (seg0 + kASeg < n) {
                        const float2 mt = __ldg(reinterpret_cast<const float2*>(d.v_meta) + vb0 + 1);
                        l1 = mt.x;
                        d1 = mt.y;
                    }
                    al8_build_tables2_soa(reinterpret_cast<float*>(s_tab[warp][tslot]),
                                          reinterpret_cast<float*>(s_tab[warp + 1][tslot]),
                                          olmin[0], odelta[0], l1, d1, kf, ok2);
                }
                asm volatile("bar.sync %0, 64;" ::"r"(1 + (warp >> 1)) : "memory");
                al8_values_from_tables_soa(s_val[warp],
                                           reinterpret_cast<const float*>(s_tab[warp][tslot]),
                                           olmin[0], odelta[0]);
                tslot ^= 1;
            } else {
                // two or four blocks per segment: their levels two blocks per
                // paired pass
                float* ts = reinterpret_cast<float*>(s_tab[warp][0]);
#pragma unroll
                for (int b = 0; b < NBV; b += 2)
                    al8_build_tables2_soa(ts + 64 * b, ts + 64 * (b + 1), olmin[b], odelta[b],
                                          olmin[b + 1], odelta[b + 1], kf, ok2);
#pragma unroll
                for (int b = 0; b < NBV; ++b)
                    al8_values_from_tables_soa(s_val[warp] + 256 * b, ts + 64 * b, olmin[b],
                                               odelta[b]);
            }
            const float* vt = s_val[WIDE ? (warp / wpbv) * wpbv : warp];
#pragma unroll
            for (int e = 0; e < NE; ++e)
                vh[e] = vt[256 * (e / 4 / CPBV) + ((vw[e / 4] >> (8 * (e % 4))) & 0xFFu)];
        } else {
#pragma unroll
            for (int e = 0; e < NE; ++e)
                vh[e] = al16_decode(code_of<VBITS>(vw, e / 4, e % 4), olmin[e / 4 / CPBV],
                                    odelta[e / 4 / CPBV]);
        }

        // ---- update, write p; keep the fresh m and v (element pairs)
        float2 mf[NE / 2], vf2[NE / 2];
        uint32_t cvmin[kCH], cvmax[kCH];
        float cmabs[kCH];  // |m| >= 0: float and unsigned order agree
#pragma unroll
        for (int c = 0; c < kCH; ++c) {
            const int bm = c / CPBM;
            const float2 dm2 = make_float2(dm[bm], dm[bm]);
            // momentum bytes as exact floats: (q + 128) placed in the low
            // mantissa of 1.5 * 2^23, then shifted back by 1.5 * 2^23 + 128
            const uint32_t mx = mw[c] ^ 0x80808080u;
            float2 pn[2];
            cvmin[c] = 0xFFFFFFFFu;
            cvmax[c] = 0u;
            cmabs[c] = 0.0f;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const float2 qf = make_float2(u2f(__byte_perm(mx, 0x4B400000u, 0x7640u | (2 * h))),
                                              u2f(__byte_perm(mx, 0x4B400000u, 0x7640u | (2 * h + 1))));
                const float2 mh = mul2(add2(qf, make_float2(-12583040.0f, -12583040.0f)), dm2);
                const float2 gi = h == 0 ? make_float2(g[c].x, g[c].y) : make_float2(g[c].z, g[c].w);
                const float2 pi = h == 0 ? make_float2(p[c].x, p[c].y) : make_float2(p[c].z, p[c].w);
                // products enter sums only through fma2: a paired product
                // feeding a paired add could be contracted by the compiler
                const float2 p1 = mul2(pi, s.decay);
                const float2 mm = fma2(s.beta1, mh, mul2(s.omb1, gi));
                const float2 vh2 = make_float2(vh[4 * c + 2 * h], vh[4 * c + 2 * h + 1]);
                const float2 vv = fma2(s.beta2, vh2, mul2(s.omb2, mul2(gi, gi)));
                // the update direction, approximately (moves p only)
                const float2 den = fma2(make_float2(sqrt_approx(vv.x), sqrt_approx(vv.y)), s.c2, s.eps);
                const float2 u = mul2(mm, make_float2(rcp_approx(den.x), rcp_approx(den.y)));
                pn[h] = fma2(s.nstep, u, p1);
                mf[2 * c + h] = mm;
                vf2[2 * c + h] = vv;
                const uint32_t vbx = f2u(vv.x), vby = f2u(vv.y);
                cvmin[c] = umix<false>(cvmin[c], umix<false>(vbx - 1u, vby - 1u));  // 0 -> max: min positive
                cvmax[c] = umix<true>(cvmax[c], umix<true>(vbx, vby));
                cmabs[c] = fmaxf(cmabs[c], fmaxf(fabsf(mm.x), fabsf(mm.y)));
            }
            const float4 pv = make_float4(pn[0].x, pn[0].y, pn[1].x, pn[1].y);
            if (full)
                __stcs(reinterpret_cast<float4*>(d.p + e0) + 32 * c, pv);
            else
                store_p_masked(d.p, e0 + 128 * c, n, pv);
        }
        float vf[NE];
#pragma unroll
        for (int j = 0; j < NE / 2; ++j) {
            vf[2 * j] = vf2[j].x;
            vf[2 * j + 1] = vf2[j].y;
        }

        // ---- new block statistics
        uint32_t bvmin[NBV], bvmax[NBV], bmabs[NBM];
        warp_blocks_reduce<CPBV, false>(cvmin, bvmin);
        warp_blocks_reduce<CPBV, true>(cvmax, bvmax);
        uint32_t cmabs_u[kCH];
#pragma unroll
        for (int c = 0; c < kCH; ++c) cmabs_u[c] = f2u(cmabs[c]);
        warp_blocks_reduce<CPBM, true>(cmabs_u, bmabs);
        // (only instantiations whose V or M blocks span whole segments can
        // have blocks wider than a segment)
        if (((CPBV == kCH) || (CPBM == kCH)) && (wpbv > 1 || wpbm > 1)) {
            // blocks wider than a segment (then one block per warp): one
            // shared round for all three statistics, one barrier; the slots
            // alternate between iterations, so a warp one iteration ahead
            // never overwrites values another warp has yet to read
            uint32_t(*sp)[kThreads / 32] = s_part[parity];
            parity ^= 1;
            if (lane == 0) {
                sp[0][warp] = bvmin[0];
                sp[1][warp] = bvmax[0];
                sp[2][warp] = bmabs[0];
            }
            const int gmax = wpbv > wpbm ? wpbv : wpbm;
            group_sync(5 + warp / gmax, gmax);
            if (wpbv > 1) {
                const int g0 = (warp / wpbv) * wpbv;
                uint32_t a = sp[0][g0], b = sp[1][g0];
                for (int k = 1; k < wpbv; ++k) {
                    a = umix<false>(a, sp[0][g0 + k]);
                    b = umix<true>(b, sp[1][g0 + k]);
                }
                bvmin[0] = a;
                bvmax[0] = b;
            }
            if (wpbm > 1) {
                const int g0 = (warp / wpbm) * wpbm;
                uint32_t a = sp[2][g0];
                for (int k = 1; k < wpbm; ++k) a = umix<true>(a, sp[2][g0 + k]);
                bmabs[0] = a;
            }
        }

        float vmn[NBV], vmx[NBV], nlmin[NBV], ndelta[NBV];
        AlEncConsts ek[NBV];
#pragma unroll
        for (int b = 0; b < NBV; ++b) {
            vmn[b] = u2f(bvmin[b] + 1u);
            vmx[b] = u2f(bvmax[b]);
        }
        al_blocks_params<NBV>(vmn, vmx, s.log_floor, nlmin, ndelta);
#pragma unroll
        for (int b = 0; b < NBV; ++b) ek[b] = al_encode_consts(nlmin[b], ndelta[b], Lm2);
        float ms[NBM], msc[NBM], minv[NBM];
#pragma unroll
        for (int b = 0; b < NBM; ++b) {
            ms[b] = u2f(bmabs[b]);
            uf8_encode_consts(ms[b] > 0.0f ? ms[b] : 1.0f, msc[b], minv[b]);
            minv[b] = ms[b] > 0.0f ? minv[b] : 0.0f;  // an all-zero block codes as 0
        }
        // (m sc) inv: sc is 1 except in blocks whose absmax is below 2^-120,
        // where the fresh m values are scaled (exactly) first
#pragma unroll
        for (int c = 0; c < kCH; ++c) {
            const int bm = c / CPBM;
            if (__builtin_expect(msc[bm] != 1.0f, 0)) {
                const float2 sc2 = make_float2(msc[bm], msc[bm]);
                mf[2 * c] = mul2(mf[2 * c], sc2);
                mf[2 * c + 1] = mul2(mf[2 * c + 1], sc2);
            }
        }

        // ---- encode and write the codes and block constants
        uint32_t qv[NE];
        al_encode_chunks<VBITS, CPBV, NBV, kCH, true>(vf, vmn, nlmin, ndelta, ek, qv);
#pragma unroll
        for (int c = 0; c < kCH; ++c) {
            const int bm = c / CPBM;
            const int64_t idx = e0 + 128 * c;
            // q = rint((m sc) inv) as the low byte of 1.5 * 2^23 + q, the
            // two's complement byte for q < 0; all codes are 0 when the
            // block's absmax is 0 (inv = 0). The rounding add is a fused
            // multiply-add by the opaque one, so the product rounds first.
            const float2 inv2 = make_float2(minv[bm], minv[bm]);
            uint32_t rb[4];
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const float2 f = mul2(mf[2 * c + i], inv2);
                const float2 r = fma2(f, s.one, make_float2(12582912.0f, 12582912.0f));
                rb[2 * i] = f2u(r.x);
                rb[2 * i + 1] = f2u(r.y);
            }
            const uint32_t qm = __byte_perm(__byte_perm(rb[0], rb[1], 0x0040u),
                                            __byte_perm(rb[2], rb[3], 0x0040u), 0x5410u);
            if (full) {
                __stcs(reinterpret_cast<unsigned int*>(d.m_codes + e0) + 32 * c, qm);
                if constexpr (VBITS == 8)
                    __stcs(reinterpret_cast<unsigned int*>((uint8_t*)d.v_codes + e0) + 32 * c,
                           qv[4 * c] | (qv[4 * c + 1] << 8) | (qv[4 * c + 2] << 16) | (qv[4 * c + 3] << 24));
                else
                    __stcs(reinterpret_cast<uint2*>((uint16_t*)d.v_codes + e0) + 32 * c,
                           make_uint2(qv[4 * c] | (qv[4 * c + 1] << 16), qv[4 * c + 2] | (qv[4 * c + 3] << 16)));
            } else {
                const uint2 w = VBITS == 8
                    ? make_uint2(qv[4 * c] | (qv[4 * c + 1] << 8) | (qv[4 * c + 2] << 16) | (qv[4 * c + 3] << 24), 0u)
                    : make_uint2(qv[4 * c] | (qv[4 * c + 1] << 16), qv[4 * c + 2] | (qv[4 * c + 3] << 16));
                store_codes_masked<VBITS>(d.m_codes, d.v_codes, idx, n, qm, w);
            }
        }
        if (lane == 0) {
            if ((warp % wpbv) == 0) {
#pragma unroll
                for (int b = 0; b < NBV; ++b)
                    if (vb0 + b < nvb)
                        reinterpret_cast<float2*>(d.v_meta)[vb0 + b] = make_float2(nlmin[b], ndelta[b]);
            }
            if ((warp % wpbm) == 0) {
#pragma unroll
                for (int b = 0; b < NBM; ++b)
                    if (mb0 + b < nmb) d.m_absmax[mb0 + b] = ms[b];
            }
        }
        __syncwarp();
    }
}

// ------------------------------------------------ unquantized reference --
// v_bits 32: AdamW with dense fp32 m and v (Sec. 4.5's FP32 state role, the
// unquantized reference): the per-element arithmetic of the fused kernel
// with m_hat = m and v_hat = v, no codec, and the IEEE square root and
// division (bit for bit the oracle's); 28 bytes per parameter. The same
// tiles and descriptors (m_codes and v_codes hold fp32 m and v).
__global__ void __launch_bounds__(kThreads)
adamw_fp32_kernel(const PlanEntry* __restrict__ table, int ntensors, int64_t total_tiles,
                  PlanEntry single, AdamWPairs s) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int cur = 0;
    for (int64_t tile = blockIdx.x; tile < total_tiles; tile += gridDim.x) {
        const PlanEntry d = plan_entry(table, ntensors, single, tile, cur);
        const int64_t e0 = (tile - d.first_tile) * kATile + (int64_t)warp * kASeg + 4 * lane;
        float* m = reinterpret_cast<float*>(d.m_codes);
        float* v = reinterpret_cast<float*>(d.v_codes);
#pragma unroll
        for (int c = 0; c < kCH; ++c) {
            const int64_t idx = e0 + 128 * c;
            if (idx >= d.n) continue;
            const float4 g4 = load4f(d.g, idx, d.n), p4 = load4f(d.p, idx, d.n);
            const float4 m4 = load4f(m, idx, d.n), v4 = load4f(v, idx, d.n);
            float2 pn[2], mn[2], vn[2];
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const float2 gi = i == 0 ? make_float2(g4.x, g4.y) : make_float2(g4.z, g4.w);
                const float2 pi = i == 0 ? make_float2(p4.x, p4.y) : make_float2(p4.z, p4.w);
                const float2 mi = i == 0 ? make_float2(m4.x, m4.y) : make_float2(m4.z, m4.w);
                const float2 vi = i == 0 ? make_float2(v4.x, v4.y) : make_float2(v4.z, v4.w);
                const float2 p1 = mul2(pi, s.decay);
                const float2 mm = fma2(s.beta1, mi, mul2(s.omb1, gi));
                const float2 vv = fma2(s.beta2, vi, mul2(s.omb2, mul2(gi, gi)));
                const float2 den = fma2(make_float2(sqrtf(vv.x), sqrtf(vv.y)), s.c2, s.eps);
                pn[i] = fma2(s.nstep, make_float2(mm.x / den.x, mm.y / den.y), p1);
                mn[i] = mm;
                vn[i] = vv;
            }
            store4f(d.p, idx, d.n, make_float4(pn[0].x, pn[0].y, pn[1].x, pn[1].y));
            store4f(m, idx, d.n, make_float4(mn[0].x, mn[0].y, mn[1].x, mn[1].y));
            store4f(v, idx, d.n, make_float4(vn[0].x, vn[0].y, vn[1].x, vn[1].y));
        }
    }
}

// ------------------------------------------------------------- dispatch --
static int cpb_of(int block) { return block >= kASeg ? kCH : block / 128; }
static bool adamw_block_ok(int block) { return valid_block(block) && block <= kATile; }

template <int CPBV, int CPBM, int VBITS>
static int launch_adamw_t(const PlanEntry* table, int ntensors, int64_t total_tiles,
                          const PlanEntry& single, int v_block, int m_block,
                          const AdamWScalars& s, cudaStream_t stream) {
    auto k = adamw_fused_kernel<CPBV, CPBM, VBITS, 1>;
    if constexpr (CPBV == kCH) {
        if (v_block == 2 * kASeg) k = adamw_fused_kernel<CPBV, CPBM, VBITS, 2>;
        if (v_block == 4 * kASeg) k = adamw_fused_kernel<CPBV, CPBM, VBITS, 4>;
        if (v_block == 8 * kASeg) k = adamw_fused_kernel<CPBV, CPBM, VBITS, 8>;
    }
    const int grid = persistent_grid((const void*)k, kThreads, 0, total_tiles);
    k<<<grid, kThreads, 0, stream>>>(table, ntensors, total_tiles, single, v_block, m_block,
                                     adamw_pairs(s));
    return check_launch();
}

template <int VBITS>
static int launch_adamw_v(int cv, int cm, const PlanEntry* table, int ntensors,
                          int64_t total_tiles, const PlanEntry& single, int v_block,
                          int m_block, const AdamWScalars& s, cudaStream_t st) {
#define ALQ_CASE(A, B)                                                                      \
    if (cv == A && cm == B)                                                                 \
        return launch_adamw_t<A, B, VBITS>(table, ntensors, total_tiles, single, v_block, \
                                           m_block, s, st);
    ALQ_CASE(1, 1) ALQ_CASE(1, 2) ALQ_CASE(1, 4) ALQ_CASE(2, 1) ALQ_CASE(2, 2) ALQ_CASE(2, 4)
    ALQ_CASE(4, 1) ALQ_CASE(4, 2) ALQ_CASE(4, 4)
#undef ALQ_CASE
    return ALQ_ERR_UNSUPPORTED;
}

static int launch_adamw(const PlanEntry* table, int ntensors, int64_t total_tiles,
                        const PlanEntry& single, int v_block, int m_block, int v_bits,
                        const al_adamw_hp* hp, int64_t t, cudaStream_t st) {
    const AdamWScalars s = adamw_scalars(hp, t);
    if (v_bits == 32) {
        const int grid = persistent_grid((const void*)adamw_fp32_kernel, kThreads, 0, total_tiles);
        adamw_fp32_kernel<<<grid, kThreads, 0, st>>>(table, ntensors, total_tiles, single,
                                                      adamw_pairs(s));
        return check_launch();
    }
    const int cv = cpb_of(v_block), cm = cpb_of(m_block);
    if (v_bits == 8)
        return launch_adamw_v<8>(cv, cm, table, ntensors, total_tiles, single, v_block, m_block, s, st);
    return launch_adamw_v<16>(cv, cm, table, ntensors, total_tiles, single, v_block, m_block, s, st);
}

static int check_hp(const al_adamw_hp* hp) {
    if (!hp) return ALQ_ERR_INVALID_ARG;
    if (!(hp->beta1 >= 0.0f && hp->beta1 < 1.0f) || !(hp->beta2 >= 0.0f && hp->beta2 < 1.0f) ||
        !(hp->eps > 0.0f) || !(hp->lr >= 0.0f))
        return ALQ_ERR_INVALID_ARG;
    return ALQ_OK;
}

// v_bits 32: m_codes and v_codes are fp32 m and v; m_absmax and v_meta are
// unused (may be NULL).
static int check_tensor(const PlanEntry& e, int v_bits) {
    if (e.n < 0) return ALQ_ERR_INVALID_ARG;
    if (e.n == 0) return ALQ_OK;
    const bool raw = v_bits == 32;
    if (!e.p || !e.g || !e.m_codes || !e.v_codes || (!raw && (!e.m_absmax || !e.v_meta)))
        return ALQ_ERR_INVALID_ARG;
    if (!aligned(e.p, 16) || !aligned(e.g, 16) || !aligned(e.m_codes, 16) ||
        !aligned(e.v_codes, 16))
        return ALQ_ERR_ALIGN;
    if (!raw && (!aligned(e.v_meta, 8) || !aligned(e.m_absmax, 4))) return ALQ_ERR_ALIGN;
    return ALQ_OK;
}

// Bit widths and block sizes of a call: blocks are ignored for v_bits 32.
static bool adamw_config_ok(int m_block, int v_block, int v_bits) {
    if (v_bits == 32) return true;
    return adamw_block_ok(m_block) && adamw_block_ok(v_block) && (v_bits == 8 || v_bits == 16);
}

}  // namespace alq

using namespace alq;

extern "C" {

int al_adamw_step(float* p, const float* g, int8_t* m_codes, float* m_absmax, void* v_codes,
                  float* v_meta, int64_t n, int m_block, int v_block, int v_bits,
                  const al_adamw_hp* hp, int64_t t, void* stream) {
    if (!adamw_config_ok(m_block, v_block, v_bits)) return ALQ_ERR_UNSUPPORTED;
    if (t < 1) return ALQ_ERR_INVALID_ARG;
    int st = check_hp(hp);
    if (st) return st;
    PlanEntry e{p, g, m_codes, m_absmax, v_codes, v_meta, n, 0};
    st = check_tensor(e, v_bits);
    if (st) return st;
    if (n == 0) return ALQ_OK;
    return launch_adamw(nullptr, 1, blocks_of(n, kATile), e, v_block, m_block, v_bits, hp, t,
                        (cudaStream_t)stream);
}

int al_adamw_plan(const al_adamw_tensor* tensors, int ntensors, int m_block, int v_block,
                  int v_bits, void* plan_host, size_t plan_bytes, al_multi_info* info) {
    if (!tensors || ntensors <= 0 || !plan_host || !info) return ALQ_ERR_INVALID_ARG;
    if (!adamw_config_ok(m_block, v_block, v_bits)) return ALQ_ERR_UNSUPPORTED;
    size_t need = 0;
    al_adamw_plan_bytes(ntensors, &need);
    if (plan_bytes < need) return ALQ_ERR_INVALID_ARG;
    PlanHeader* h = (PlanHeader*)plan_host;
    PlanEntry* ent = (PlanEntry*)((char*)plan_host + sizeof(PlanHeader));
    int64_t tiles = 0, elems = 0;
    for (int i = 0; i < ntensors; ++i) {
        const al_adamw_tensor& t = tensors[i];
        PlanEntry e{t.p, t.g, t.m_codes, t.m_absmax, t.v_codes, t.v_meta, t.n, tiles};
        int st = check_tensor(e, v_bits);
        if (st) return st;
        ent[i] = e;
        tiles += blocks_of(t.n, kATile);
        elems += t.n;
    }
    memset(h, 0, sizeof(PlanHeader));
    h->magic = kPlanMagic;
    h->ntensors = ntensors;
    h->m_block = m_block;
    h->v_block = v_block;
    h->v_bits = v_bits;
    h->tile = kATile;
    h->total_tiles = tiles;
    h->total_elems = elems;
    info->ntensors = ntensors;
    info->m_block = m_block;
    info->v_block = v_block;
    info->v_bits = v_bits;
    info->total_tiles = tiles;
    info->total_elems = elems;
    return ALQ_OK;
}

int al_adamw_step_multi(const void* plan_dev, const al_multi_info* info, const al_adamw_hp* hp,
                        int64_t t, void* stream) {
    if (!plan_dev || !info || t < 1) return ALQ_ERR_INVALID_ARG;
    if (!aligned(plan_dev, 16)) return ALQ_ERR_ALIGN;
    if (info->ntensors <= 0 || info->total_tiles < 0) return ALQ_ERR_INVALID_ARG;
    if (!adamw_config_ok(info->m_block, info->v_block, info->v_bits)) return ALQ_ERR_UNSUPPORTED;
    int st = check_hp(hp);
    if (st) return st;
    if (info->total_tiles == 0) return ALQ_OK;
    const PlanEntry* table =
        (const PlanEntry*)((const char*)plan_dev + sizeof(PlanHeader));
    PlanEntry none{};
    return launch_adamw(table, info->ntensors, info->total_tiles, none, info->v_block,
                        info->m_block, info->v_bits, hp, t, (cudaStream_t)stream);
}

}  // extern "C"
