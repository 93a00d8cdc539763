// alq_kernels.cuh -- device building blocks of the element-wise kernels:
// masked chunk loads/stores, per-block reductions, per-block AL/UF8
// constants, and the AL8 decode tables.
//
// Geometry (see alq_internal.h): a warp owns a 512-element segment; lane l
// owns chunk c = 0..3 = elements [128 c + 4 l, 128 c + 4 l + 4) of it. For a
// block size B = 128 * CPB (CPB = 1, 2, 4 chunks per block) a segment holds
// NB = 4 / CPB blocks, each spanning all 32 lanes; for B > 512 a block spans
// B / 512 consecutive warps and its statistics are combined through shared
// memory.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "alq_internal.h"
#include "alq_numerics.h"

namespace alq {

// ----------------------------------------------- paired fp32 arithmetic --
// Two independent fp32 operations per instruction (sm_100 and later). The
// explicit .rn modifier makes each component round exactly like the scalar
// operation and forbids contraction into a fused multiply-add.
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
    float2 r;
    asm("{\n.reg .b64 a, b, d;\nmov.b64 a, {%2, %3};\nmov.b64 b, {%4, %5};\n"
        "mul.rn.f32x2 d, a, b;\nmov.b64 {%0, %1}, d;\n}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    float2 r;
    asm("{\n.reg .b64 a, b, d;\nmov.b64 a, {%2, %3};\nmov.b64 b, {%4, %5};\n"
        "add.rn.f32x2 d, a, b;\nmov.b64 {%0, %1}, d;\n}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 sub2(float2 a, float2 b) {
    float2 r;
    asm("{\n.reg .b64 a, b, d;\nmov.b64 a, {%2, %3};\nmov.b64 b, {%4, %5};\n"
        "sub.rn.f32x2 d, a, b;\nmov.b64 {%0, %1}, d;\n}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    float2 r;
    asm("{\n.reg .b64 a, b, c, d;\nmov.b64 a, {%2, %3};\nmov.b64 b, {%4, %5};\n"
        "mov.b64 c, {%6, %7};\nfma.rn.f32x2 d, a, b, c;\nmov.b64 {%0, %1}, d;\n}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return r;
}

// ------------------------------------------------------------- chunk I/O --
// ---------------------------------------- approximate update direction --
// The hardware's approximate square root and reciprocal (a few ulp each).
// The fused AdamW step forms its update direction u = m / (sqrt(v) c2 + eps)
// with them: u moves only the parameters and feeds no optimizer state, so
// every code and block constant stays exact, and a step's parameter differs
// from the IEEE result by a few ulp of lr |u| at most.
__device__ __forceinline__ float sqrt_approx(float x) {
    float r;
    asm("sqrt.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

__device__ __forceinline__ float rcp_approx(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// log2 of a power of two, at compile time
__host__ __device__ constexpr int ilog2c(int x) { return x <= 1 ? 0 : 1 + ilog2c(x / 2); }

// Shift of a kernel's block size: a block narrower than a segment of CH
// chunks is 128 CPB elements, known when the kernel is instantiated;
// otherwise the runtime size.
template <int CPB, int CH>
__device__ __forceinline__ int block_shift(int block) {
    return CPB < CH ? 7 + ilog2c(CPB) : __ffs(block) - 1;
}

__device__ __forceinline__ int64_t blocks_of_dev(int64_t n, int block) {
    return (n + block - 1) / block;
}

__device__ __forceinline__ int64_t chunk_index(int64_t seg0, int c, int lane) {
    return seg0 + 128 * c + 4 * lane;
}

__device__ __forceinline__ float4 load4f(const float* p, int64_t i, int64_t n) {
    if (i + 4 <= n) return __ldcs(reinterpret_cast<const float4*>(p + i));
    float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i < n) r.x = p[i];
    if (i + 1 < n) r.y = p[i + 1];
    if (i + 2 < n) r.z = p[i + 2];
    return r;
}

__device__ __forceinline__ void store4f(float* p, int64_t i, int64_t n, float4 v) {
    if (i + 4 <= n) {
        __stcs(reinterpret_cast<float4*>(p + i), v);
        return;
    }
    if (i < n) p[i] = v.x;
    if (i + 1 < n) p[i + 1] = v.y;
    if (i + 2 < n) p[i + 2] = v.z;
}

// Four 8-bit codes as one little-endian word.
__device__ __forceinline__ uint32_t load4b(const uint8_t* p, int64_t i, int64_t n) {
    if (i + 4 <= n) return __ldcs(reinterpret_cast<const unsigned int*>(p + i));
    uint32_t r = 0;
    if (i < n) r |= (uint32_t)p[i];
    if (i + 1 < n) r |= (uint32_t)p[i + 1] << 8;
    if (i + 2 < n) r |= (uint32_t)p[i + 2] << 16;
    return r;
}

__device__ __forceinline__ void store4b(uint8_t* p, int64_t i, int64_t n, uint32_t w) {
    if (i + 4 <= n) {
        __stcs(reinterpret_cast<unsigned int*>(p + i), w);
        return;
    }
    if (i < n) p[i] = (uint8_t)w;
    if (i + 1 < n) p[i + 1] = (uint8_t)(w >> 8);
    if (i + 2 < n) p[i + 2] = (uint8_t)(w >> 16);
}

// Four 16-bit codes as two words (w0 = codes 0,1; w1 = codes 2,3).
__device__ __forceinline__ uint2 load4h(const uint16_t* p, int64_t i, int64_t n) {
    if (i + 4 <= n) return __ldcs(reinterpret_cast<const uint2*>(p + i));
    uint2 r = make_uint2(0u, 0u);
    if (i < n) r.x |= (uint32_t)p[i];
    if (i + 1 < n) r.x |= (uint32_t)p[i + 1] << 16;
    if (i + 2 < n) r.y |= (uint32_t)p[i + 2];
    return r;
}

__device__ __forceinline__ void store4h(uint16_t* p, int64_t i, int64_t n, uint2 w) {
    if (i + 4 <= n) {
        __stcs(reinterpret_cast<uint2*>(p + i), w);
        return;
    }
    if (i < n) p[i] = (uint16_t)w.x;
    if (i + 1 < n) p[i + 1] = (uint16_t)(w.x >> 16);
    if (i + 2 < n) p[i + 2] = (uint16_t)w.y;
}

__device__ __forceinline__ float f4get(const float4& v, int i) {
    return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// Code i (0..3) of a chunk: 8-bit codes packed in one word, 16-bit in two.
template <int BITS>
__device__ __forceinline__ uint32_t code_of(const uint32_t* w, int c, int i) {
    if (BITS == 8) return (w[c] >> (8 * i)) & 0xFFu;
    return (w[2 * c + (i >> 1)] >> (16 * (i & 1))) & 0xFFFFu;
}

// --------------------------------------------------------- block reductions --
template <bool kMax>
__device__ __forceinline__ uint32_t umix(uint32_t a, uint32_t b) {
    return kMax ? (a > b ? a : b) : (a < b ? a : b);
}

// Per-block warp-wide min or max of per-chunk values (unsigned order): a lane
// holds CH chunks, CPB consecutive chunks form one block.
template <int CPB, bool kMax, int CH>
__device__ __forceinline__ void warp_blocks_reduce(const uint32_t (&chunk)[CH],
                                                   uint32_t (&out)[CH / CPB]) {
#pragma unroll
    for (int b = 0; b < CH / CPB; ++b) {
        uint32_t v = chunk[b * CPB];
#pragma unroll
        for (int c = 1; c < CPB; ++c) v = umix<kMax>(v, chunk[b * CPB + c]);
        out[b] = kMax ? __reduce_max_sync(0xFFFFFFFFu, v) : __reduce_min_sync(0xFFFFFFFFu, v);
    }
}

// Blocks wider than a segment: combine the per-warp results of the `wpb`
// warps that share a block. Every thread of the CTA must call this.
template <bool kMax>
__device__ __forceinline__ uint32_t cta_group_reduce(uint32_t v, uint32_t* s_part,
                                                     int wpb) {
    const int warp = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) s_part[warp] = v;
    __syncthreads();
    const int g0 = (warp / wpb) * wpb;
    uint32_t r = s_part[g0];
    for (int k = 1; k < wpb; ++k) r = umix<kMax>(r, s_part[g0 + k]);
    __syncthreads();
    return r;
}

// ------------------------------------------------------- AL block constants --
// (l_min, Delta) of the NB blocks of a segment from their minimum positive
// value mn and maximum mx (Eq. (3)). The 2 NB fp32-rounded logs are spread
// over the lanes (one log per lane) and exchanged by shuffles; each is
// first taken from the hardware log2 with its rounding certified
// (log2_rn_fast), and the lanes it cannot certify (about one in ten) take
// the two-float log2_rn under one warp-uniform branch.
template <int NB>
__device__ __forceinline__ void al_blocks_params(const float (&mn)[NB], const float (&mx)[NB],
                                                 float log_floor, float (&lmin)[NB],
                                                 float (&delta)[NB]) {
    const int lane = threadIdx.x & 31;
    const int v = lane & (2 * NB - 1);
    float x = 0.0f;
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        if (v == 2 * b) x = mn[b];
        if (v == 2 * b + 1) x = mx[b];
    }
    bool ok;
    float L = log2_rn_fast(x > 0.0f ? x : 1.0f, ok);
    ok = ok || !(x > 0.0f);
    L = (x > 0.0f) ? L : 0.0f;
    if (__builtin_expect(__any_sync(0xFFFFFFFFu, !ok), 0)) L = log2_rn_fixup(x, L, ok);
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        const float l0 = __shfl_sync(0xFFFFFFFFu, L, 2 * b);
        const float l1 = __shfl_sync(0xFFFFFFFFu, L, 2 * b + 1);
        al_block_params_from_logs(mx[b], l0, l1, log_floor, lmin[b], delta[b]);
    }
}

// ------------------------------------------------------ AL8 decode tables --
// The two 16-entry level tables of each of the NB blocks of a segment
// (Eq. (5)): entry b < 16 holds T_lo[b] = 2^((b-1) d), entries 16..31 hold
// T_hi[a] = 2^(l_min + 16 a d), d = Delta / 254, as two-float pairs; code
// q = 16 a + b decodes to T_hi[a] * T_lo[b]. T_hi is stored even a first
// (slots 16..23), then odd a (24..31): lane l decodes the codes l + 32 k,
// whose factors T_hi[2 k + (l >> 4)] are then contiguous. One entry per lane
// per block. Blocks whose l_min is below -96 (or that are empty) take the
// FP64 path.
// Level index of this lane's table entry: k = b - 1 for lanes b < 16,
// k = 16 (lane - 16) for the others (as a float).
__device__ __forceinline__ float al8_table_k(int lane) {
    return int_to_float_small(lane >= 16 ? 16 * (lane - 16) : lane - 1);
}

__device__ __forceinline__ int al8_hi_slot(uint32_t a) {
    return 16 + (int)((a & 1u) << 3) + (int)(a >> 1);
}

__device__ __forceinline__ bool al8_fast_ok(float lmin, float delta) {
    return delta > 0.0f && lmin >= -96.0f;
}

// ------------------------------------------- paired two-float AL levels --
// al_level_ff (alq_numerics.h) for two (l_min, Delta) at once, step for step
// in paired instructions: every rounding of the scalar routine happens here
// too (the steps that routine documents as exact may fuse), so the results
// are the scalar ones. A product that enters a sum is formed by a fused
// multiply-add with zero, or enters it through a fused multiply-add by one,
// both values the compiler cannot see (k.x, k.y from the kernel's
// parameters): a paired product feeding a paired add could otherwise be
// contracted. The table lookups and the integer parts stay scalar.
struct Opaque2 {
    float2 one, zero;
};

__device__ __forceinline__ float2 rint_small2(float2 x, const Opaque2& k, int& i0, int& i1) {
    const float2 magic = make_float2(12582912.0f, 12582912.0f);
    const float2 r = fma2(x, k.one, magic);
    i0 = (int)(f2u(r.x) - 0x4B400000u);
    i1 = (int)(f2u(r.y) - 0x4B400000u);
    return sub2(r, magic);
}

__device__ __forceinline__ void two_sum2(float2 a, float2 b, float2& s, float2& e) {
    s = add2(a, b);
    const float2 bb = sub2(s, a);
    e = add2(sub2(a, sub2(s, bb)), sub2(b, bb));
}

__device__ __forceinline__ void exp2_ff2(float2 fh, float2 fl, const Opaque2& k, float2& rh,
                                         float2& rl, int& eo0, int& eo1) {
    int n0, n1;
    const float2 ns = rint_small2(mul2(fh, make_float2(1024.0f, 1024.0f)), k, n0, n1);
    const float2 f0 = fma2(ns, make_float2(-1.0f / 1024.0f, -1.0f / 1024.0f), fh);  // exact
    float2 gh, gl;
    two_sum2(f0, fl, gh, gl);
    const float2 ln2h = make_float2(ALQ_LN2_HI, ALQ_LN2_HI), ln2l = make_float2(ALQ_LN2_LO, ALQ_LN2_LO);
    const float2 wh = fma2(gh, ln2h, k.zero);
    const float2 nwh = mul2(gh, make_float2(-ALQ_LN2_HI, -ALQ_LN2_HI));
    const float2 wl = add2(fma2(gh, ln2h, nwh), fma2(mul2(gh, ln2l), k.one, mul2(gl, ln2h)));
    const float2 a = fma2(mul2(wh, make_float2(1.0f / 6.0f, 1.0f / 6.0f)), k.one,
                          make_float2(0.5f, 0.5f));
    const float2 c = fma2(mul2(mul2(wh, wh), a), k.one, wl);
    const int j0 = n0 & 1023, j1 = n1 & 1023;
    eo0 = n0 >> 10;
    eo1 = n1 >> 10;
    const float2 th = make_float2(ALQ_TAB(kExp2Hi, j0), ALQ_TAB(kExp2Hi, j1));
    const float2 tl = make_float2(ALQ_TAB(kExp2Lo, j0), ALQ_TAB(kExp2Lo, j1));
    const float2 ph = fma2(th, wh, k.zero);
    const float2 pl = fma2(th, wh, mul2(th, make_float2(-wh.x, -wh.y)));
    const float2 sh = fma2(ph, k.one, th);
    const float2 sl = fma2(ph, k.one, sub2(th, sh));  // ph - (sh - th)
    const float2 lo = add2(sl, add2(pl, add2(tl, fma2(mul2(tl, wh), k.one, mul2(th, c)))));
    rh = add2(sh, lo);
    rl = sub2(lo, sub2(rh, sh));
}

__device__ __forceinline__ void al_level_ff2(float2 lmin, float2 delta, float kf, float Lm2,
                                             float inv_Lm2, const Opaque2& k, float2& rh,
                                             float2& rl) {
    int I00, I01, N0, N1;
    const float2 I0f = rint_small2(lmin, k, I00, I01);
    const float2 F0 = sub2(lmin, I0f);  // exact
    const float2 kf2 = make_float2(kf, kf);
    const float2 ph = fma2(kf2, delta, k.zero);
    const float2 pl = fma2(kf2, delta, mul2(kf2, make_float2(-delta.x, -delta.y)));
    const float2 inv = make_float2(inv_Lm2, inv_Lm2);
    const float2 Nf = rint_small2(mul2(ph, inv), k, N0, N1);
    const float2 r0 = fma2(Nf, make_float2(-Lm2, -Lm2), ph);  // exact
    float2 Rh, Rl;
    two_sum2(r0, pl, Rh, Rl);
    const float2 q1 = fma2(Rh, inv, k.zero);
    const float2 rem = fma2(mul2(Rh, make_float2(-inv_Lm2, -inv_Lm2)), make_float2(Lm2, Lm2), Rh);
    const float2 q2 = fma2(add2(rem, Rl), inv, k.zero);
    float2 Fh, Fe;
    two_sum2(F0, q1, Fh, Fe);
    const float2 Fl = add2(Fe, q2);
    int eo0, eo1;
    exp2_ff2(Fh, Fl, k, rh, rl, eo0, eo1);
    const float2 sc = make_float2(pow2i(I00 + N0 + eo0), pow2i(I01 + N1 + eo1));
    rh = mul2(rh, sc);
    rl = mul2(rl, sc);
}

// al8_decode_pair (alq_numerics.h) on two values with the same low factor
// (bh, bl), step for step in paired instructions (each component rounds as
// the scalar operation does).
__device__ __forceinline__ float2 al8_decode_pair2(float2 ah, float2 al, float2 bh, float2 bl,
                                                   float2 nbh, bool& fb0, bool& fb1) {
    const float2 c = fma2(ah, bl, mul2(al, bh));
    const float2 r = fma2(ah, bh, c);
    const float2 t = fma2(ah, nbh, r);
    const float2 res = sub2(c, t);
    const float2 z = fma2(res, make_float2(kZivFactor, kZivFactor), r);
    fb0 = z.x != r.x;
    fb1 = z.y != r.y;
    return r;
}


// ------------------------------------------------------ AL8 level tables --
// An AL8 block's codes q = 16 a + b factor through two 16-entry tables of
// two-float levels (the high factor T_hi[a] and the low factor T_lo[b]),
// stored as 64 floats: the high parts at [slot], the low parts at
// [32 + slot] (slots 0-15 the low factors, al8_hi_slot(a) the high ones), so
// that the paired products read the high parts of two entries, and their
// low parts, as adjacent pairs. Each lane computes one entry; a block
// outside the fast range gets zeros. Two blocks per paired pass:
__device__ __forceinline__ void al8_build_tables2_soa(float* tab0, float* tab1, float lmin0,
                                                      float delta0, float lmin1, float delta1,
                                                      float kf, const Opaque2& k) {
    const int lane = threadIdx.x & 31;
    const bool hi = lane >= 16;
    const int slot = hi ? al8_hi_slot((uint32_t)(lane - 16)) : lane;
    const bool f0 = al8_fast_ok(lmin0, delta0), f1 = al8_fast_ok(lmin1, delta1);
    const float2 lm = make_float2(hi && f0 ? lmin0 : 0.0f, hi && f1 ? lmin1 : 0.0f);
    const float2 dl = make_float2(f0 ? delta0 : 1.0f, f1 ? delta1 : 1.0f);
    float2 rh, rl;
    al_level_ff2(lm, dl, kf, 254.0f, 1.0f / 254.0f, k, rh, rl);
    tab0[slot] = f0 ? rh.x : 0.0f;
    tab0[32 + slot] = f0 ? rl.x : 0.0f;
    tab1[slot] = f1 ? rh.y : 0.0f;
    tab1[32 + slot] = f1 ? rl.y : 0.0f;
    __syncwarp();
}

// One block's level tables in the same layout, one level per lane (scalar).
__device__ __forceinline__ void al8_build_tables_soa(float* tab, float lmin, float delta,
                                                     float kf) {
    const int lane = threadIdx.x & 31;
    const bool hi = lane >= 16;
    const int slot = hi ? al8_hi_slot((uint32_t)(lane - 16)) : lane;
    float rh = 0.0f, rl = 0.0f;
    if (al8_fast_ok(lmin, delta))
        al_level_ff(hi ? lmin : 0.0f, delta, kf, 254.0f, 1.0f / 254.0f, rh, rl);
    tab[slot] = rh;
    tab[32 + slot] = rl;
    __syncwarp();
}

// Rare path of al8_values_from_tables_soa, out of line so that the hot loop
// stays compact: redo this lane's eight boundary tests of one block and
// recompute the flagged values in FP64.
static __device__ __noinline__ void al8_values_fixup_soa(float* vals, const float* tab, float lmin,
                                                         float delta) {
    const int lane = threadIdx.x & 31;
    const bool fast = al8_fast_ok(lmin, delta);
    for (int k = 0; k < 8; ++k) {
        const uint32_t q = (uint32_t)(lane + 32 * k);
        const int sa = al8_hi_slot(q >> 4), sb = (int)(q & 15u);
        bool fb;
        al8_decode_pair(tab[sa], tab[32 + sa], tab[sb], tab[32 + sb], fb);
        if ((q != 0u) && (fb || !fast)) vals[q] = al_dequantize_fp64(q, lmin, delta, 254.0);
    }
}

// The 256 decoded values of one block (Eq. (5), code 0 -> 0), exactly as
// the double expression rounds them, in shared memory: lane l computes codes
// l, l + 32, ..., l + 224 from the block's level tables (T_hi[q >> 4] *
// T_lo[q & 15], two codes per paired step: T_lo[l & 15] is the same for all
// eight); entries whose two-float product lies too close to an fp32 rounding
// boundary, and blocks outside the fast range, are recomputed in FP64 under
// one warp-uniform branch. An element decode is then a single shared-memory
// load. tab must be 8-byte aligned.
__device__ __forceinline__ void al8_values_from_tables_soa(float* vals, const float* tab,
                                                           float lmin, float delta) {
    const int lane = threadIdx.x & 31;
    const bool fast = al8_fast_ok(lmin, delta);
    const float bv = tab[lane & 15], blv = tab[32 + (lane & 15)];
    const float2 bh = make_float2(bv, bv), bl = make_float2(blv, blv);
    const float2 nbh = make_float2(-bv, -bv);
    const float2* Ah = reinterpret_cast<const float2*>(tab + 16 + 8 * (lane >> 4));
    const float2* Al = reinterpret_cast<const float2*>(tab + 48 + 8 * (lane >> 4));
    bool any_fb = !fast;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        bool f0, f1;
        const float2 r = al8_decode_pair2(Ah[j], Al[j], bh, bl, nbh, f0, f1);
        const uint32_t q0 = (uint32_t)(lane + 64 * j);
        vals[q0] = q0 == 0u ? 0.0f : r.x;
        vals[q0 + 32] = r.y;
        any_fb |= ((q0 != 0u) & f0) | f1;
    }
    if (__builtin_expect(__any_sync(0xFFFFFFFFu, any_fb), 0)) al8_values_fixup_soa(vals, tab, lmin, delta);
    __syncwarp();
}

// Fixed-size arrays passed by value to the out-of-line rare paths (so that
// the hot path's register arrays never need an address).
template <typename T, int N>
struct Arr {
    T v[N];
};

// Rare path of al_encode_chunks, out of line: zero codes for zeros, redo the
// boundary tests (with the subnormal test) and recompute the flagged codes
// in two-float arithmetic (FP64 for the few that cannot be decided so).
template <int BITS, int CPB, int NB, int CH>
static __device__ __noinline__ Arr<uint32_t, 4 * CH> al_encode_fixup(
    Arr<float, 4 * CH> x, Arr<float, NB> lmin, Arr<float, NB> delta, Arr<AlEncConsts, NB> k,
    Arr<uint32_t, 4 * CH> q) {
    constexpr float Lm2 = BITS == 8 ? 254.0f : 65534.0f;
#pragma unroll
    for (int e = 0; e < 4 * CH; ++e) {
        const int b = e / 4 / CPB;
        bool fb;
        al_quantize_fast(x.v[e], k.v[b], Lm2, fb);
        if (x.v[e] == 0.0f)
            q.v[e] = 0u;
        else if (fb)
            q.v[e] = al_quantize_refine(x.v[e], lmin.v[b], delta.v[b], Lm2);
    }
    return q;
}

// Eq. (4) for the 4 CH values of a lane's chunks: al_quantize_fast on pairs
// of values in paired instructions (the clamping fused multiply-adds
// scalar), branch-free, with the same fixup in FP64 for values near a
// half-integer of t. mn is each block's minimum positive value (0 for a
// block without one); a block with a subnormal minimum sends the whole
// segment through the fixup, so that the fast path needs no per-value
// subnormal test. Zero codes as 0: its exponent field 0 gives tau <=
// -(127 + l_min) / Delta < 0 (l_min >= -126 without subnormals), so
// q = rint(Lm2 clip(tau)) + [x != 0] = 0. POS: every x has its sign bit
// clear (no -0), so the exponent field needs no mask.
template <int BITS, int CPB, int NB, int CH, bool POS = false>
__device__ __forceinline__ void al_encode_chunks(const float (&x)[4 * CH], const float (&mn)[NB],
                                                 const float (&lmin)[NB],
                                                 const float (&delta)[NB],
                                                 const AlEncConsts (&k)[NB],
                                                 uint32_t (&q)[4 * CH]) {
    constexpr float Lm2 = BITS == 8 ? 254.0f : 65534.0f;
    bool any_fb = false;
#pragma unroll
    for (int b = 0; b < NB; ++b) any_fb |= (mn[b] > 0.0f) & (mn[b] < 0x1p-126f);
    // POS: q = rint(Lm2 t1) + 1 comes out of the rounding constant
    // 1.5 * 2^23 + 1 (exact ties, where that constant could round the other
    // way, always take the fixup), and min(q, bits of x) makes a zero 0
    // (every positive x the fast path codes is normal: bits >= 2^23 > q)
    const float cr = POS ? 12582913.0f : 12582912.0f;
    const uint32_t cb = POS ? 0x4B400000u : 0x4B400000u;
    const float2 rc = make_float2(cr, cr);
    const float2 l2 = make_float2(Lm2, Lm2);
    float dmax[NB];  // the largest |t - rint(t)| distance to the tie of each block
#pragma unroll
    for (int b = 0; b < NB; ++b) dmax[b] = 0.0f;
#pragma unroll
    for (int e = 0; e < 4 * CH; e += 2) {
        const int b = e / 4 / CPB;
        const uint32_t x0 = f2u(x[e]), x1 = f2u(x[e + 1]);
        // 2^23 + the biased exponent: one funnel shift when the sign is clear
        const float2 eb = POS ? make_float2(u2f(__funnelshift_r(x0, 0x4B000000u >> 9, 23)),
                                            u2f(__funnelshift_r(x1, 0x4B000000u >> 9, 23)))
                              : make_float2(u2f(0x4B000000u | ((x0 >> 23) & 0xFFu)),
                                            u2f(0x4B000000u | ((x1 >> 23) & 0xFFu)));
        const float2 lg = make_float2(lg2_mant(u2f((x0 & 0x007FFFFFu) | 0x3F800000u)),
                                      lg2_mant(u2f((x1 & 0x007FFFFFu) | 0x3F800000u)));
        const float2 iD = make_float2(k[b].iD, k[b].iD);
        const float2 s1 = sub2(eb, make_float2(k[b].e0p, k[b].e0p));  // e - I, exact
        const float2 u = fma2(lg, iD, make_float2(k[b].nFiD, k[b].nFiD));
        const float2 t1 = make_float2(fma_sat(s1.x, iD.x, u.x), fma_sat(s1.y, iD.y, u.y));
        const float2 rr = fma2(t1, l2, rc);  // rint(Lm2 t1) + the rounding constant
        const float2 df = fma2(t1, l2, sub2(rc, rr));
        dmax[b] = fmaxf(dmax[b], fmaxf(fabsf(df.x), fabsf(df.y)));
        if (POS) {
            q[e] = min(f2u(rr.x) - cb, x0);
            q[e + 1] = min(f2u(rr.y) - cb, x1);
        } else {
            q[e] = (f2u(rr.x) - cb) + min(x0 << 1, 1u);
            q[e + 1] = (f2u(rr.y) - cb) + min(x1 << 1, 1u);
        }
    }
#pragma unroll
    for (int b = 0; b < NB; ++b) any_fb |= dmax[b] > 0.5f - k[b].E;
    if (__builtin_expect(__any_sync(0xFFFFFFFFu, any_fb), 0)) {
        Arr<float, 4 * CH> xa;
        Arr<uint32_t, 4 * CH> qa;
        Arr<float, NB> la, da;
        Arr<AlEncConsts, NB> ka;
#pragma unroll
        for (int e = 0; e < 4 * CH; ++e) {
            xa.v[e] = x[e];
            qa.v[e] = q[e];
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            la.v[b] = lmin[b];
            da.v[b] = delta[b];
            ka.v[b] = k[b];
        }
        qa = al_encode_fixup<BITS, CPB, NB, CH>(xa, la, da, ka, qa);
#pragma unroll
        for (int e = 0; e < 4 * CH; ++e) q[e] = qa.v[e];
    }
}

// Rare path of al8_values_part_soa: this warp's share of codes (steps j0 ..
// j0 + nsteps - 1, halves in hmask) recomputed in FP64 where the product
// could not be certified or the block is outside the fast range.
static __device__ __noinline__ void al8_values_part_fixup_soa(float* vals, const float* tab,
                                                              float lmin, float delta, int j0,
                                                              int nsteps, uint32_t hmask) {
    const int lane = threadIdx.x & 31;
    const bool fast = al8_fast_ok(lmin, delta);
    for (int j = j0; j < j0 + nsteps; ++j) {
        for (int h = 0; h < 2; ++h) {
            if (!((hmask >> h) & 1u)) continue;
            const uint32_t q = (uint32_t)(lane + 64 * j + 32 * h);
            const int sa = al8_hi_slot(q >> 4), sb = (int)(q & 15u);
            bool fb;
            al8_decode_pair(tab[sa], tab[32 + sa], tab[sb], tab[32 + sb], fb);
            if ((q != 0u) && (fb || !fast)) vals[q] = al_dequantize_fp64(q, lmin, delta, 254.0);
        }
    }
}

// One block's value table shared by the wpb (2, 4 or 8) warps whose segments
// it spans: warp r of the group computes its share of the pair steps of
// al8_values_from_tables_soa (step j covers codes l + 64 j and l + 64 j + 32;
// wpb 2: steps 2 r, 2 r + 1; wpb 4: step r; wpb 8: one half of step r / 2),
// with the same products, the same certification and the same FP64
// recomputation, so every value is the one al8_values_from_tables_soa
// stores. The caller synchronises the group before and after.
__device__ __forceinline__ void al8_values_part_soa(float* vals, const float* tab, float lmin,
                                                    float delta, int r, int wpb) {
    const int lane = threadIdx.x & 31;
    const int nsteps = wpb == 2 ? 2 : 1;
    const int j0 = wpb == 8 ? (r >> 1) : r * nsteps;
    const uint32_t hmask = wpb == 8 ? (1u << (r & 1)) : 3u;
    const float bv = tab[lane & 15], blv = tab[32 + (lane & 15)];
    const float2 bh = make_float2(bv, bv), bl = make_float2(blv, blv);
    const float2 nbh = make_float2(-bv, -bv);
    const float2* Ah = reinterpret_cast<const float2*>(tab + 16 + 8 * (lane >> 4));
    const float2* Al = reinterpret_cast<const float2*>(tab + 48 + 8 * (lane >> 4));
    bool any_fb = !al8_fast_ok(lmin, delta);
#pragma unroll
    for (int s = 0; s < 2; ++s) {
        if (s >= nsteps) break;
        const int j = j0 + s;
        bool f0, f1;
        const float2 v = al8_decode_pair2(Ah[j], Al[j], bh, bl, nbh, f0, f1);
        const uint32_t q0 = (uint32_t)(lane + 64 * j);
        if (hmask & 1u) {
            vals[q0] = q0 == 0u ? 0.0f : v.x;
            any_fb |= (q0 != 0u) & f0;
        }
        if (hmask & 2u) {
            vals[q0 + 32] = v.y;
            any_fb |= f1;
        }
    }
    if (__builtin_expect(__any_sync(0xFFFFFFFFu, any_fb), 0))
        al8_values_part_fixup_soa(vals, tab, lmin, delta, j0, nsteps, hmask);
}

// Element decode with the level computed directly in two-float form (any
// bit width; used for AL16 and for the small factor vectors).
__device__ __forceinline__ float al_decode_direct(uint32_t q, float lmin, float delta,
                                                  float Lm2) {
    if (q == 0u) return 0.0f;
    if (lmin >= -96.0f && delta > 0.0f) {
        float rh, rl;
        al_level_ff(lmin, delta, int_to_float_small((int)q - 1), Lm2, 1.0f / Lm2, rh, rl);
        if (!ziv_fails(rh, rl)) return rh;  // rh + rl: relative error below 2^-45
    }
    return al_dequantize_fp64(q, lmin, delta, (double)Lm2);
}

__device__ __forceinline__ float al16_decode(uint32_t q, float lmin, float delta) {
    return al_decode_direct(q, lmin, delta, 65534.0f);
}

// Eq. (4) element encode with the FP64 fallback near rounding boundaries.
template <int BITS>
__device__ __forceinline__ uint32_t al_encode_elem(float x, float lmin, float delta,
                                                   const AlEncConsts& k) {
    if (x == 0.0f) return 0u;
    constexpr float Lm2 = BITS == 8 ? 254.0f : 65534.0f;
    bool fb;
    uint32_t q = al_quantize_fast(x, k, Lm2, fb);
    if (fb) q = al_quantize_refine(x, lmin, delta, Lm2);
    return q;
}

// Signed 8-bit code (two's complement byte) to float, exactly, without an
// int-to-float conversion: (byte ^ 0x80) is q + 128 in [0, 255]; placed in
// the low mantissa of 1.5 * 2^23 it reads as 1.5 * 2^23 + q + 128.
__device__ __forceinline__ float s8_to_float(uint32_t byte) {
    return __uint_as_float(0x4B400000u | ((byte & 0xFFu) ^ 0x80u)) - 12583040.0f;
}

// ------------------------------------------- division by an invariant int --
// Unsigned 32-bit division by a run-time invariant d >= 2 through one
// multiply-high (Granlund and Montgomery, "Division by invariant integers
// using multiplication", PLDI 1994, Fig. 4.1).
struct Divider {
    uint32_t m, s1, s2, d;
};

inline Divider make_divider(uint32_t d) {
    uint32_t l = 0;
    while ((1ull << l) < d) ++l;
    Divider v;
    v.m = (uint32_t)(((1ull << 32) * ((1ull << l) - d)) / d + 1);
    v.s1 = l > 0 ? 1 : 0;
    v.s2 = l > 0 ? l - 1 : 0;
    v.d = d;
    return v;
}

__device__ __forceinline__ uint32_t divide(uint32_t n, const Divider& v) {
    const uint32_t t1 = __umulhi(v.m, n);
    return (t1 + ((n - t1) >> v.s1)) >> v.s2;
}

// ----------------------------------------------------- float-float add-in --
__device__ __forceinline__ void ff_acc(float& hi, float& lo, float h, float l) {
    float s, e;
    two_sum(hi, h, s, e);
    hi = s;
    lo = lo + (e + l);
}

// Paired two-float accumulation (two independent sums): adds h + l, given
// h and nl = -l, to (hi, lo) by Knuth's TwoSum of hi and h.
__device__ __forceinline__ void ff_acc2(float2& hi, float2& lo, float2 h, float2 nl) {
    const float2 s = add2(hi, h);
    const float2 bb = sub2(s, hi);
    const float2 e = add2(sub2(hi, sub2(s, bb)), sub2(h, bb));
    hi = s;
    lo = add2(lo, sub2(e, nl));
}

// Exact squares of a pair of values: x^2 = h + l with h = RN(x x) and
// nl = -l = RN(h - x x) (exact); neg = (-1, -1). h is a fused multiply-add
// with zero, a value the compiler cannot see (from the kernel's parameters):
// a paired product feeding the sums could otherwise be contracted into them.
__device__ __forceinline__ void ff_sq2(float2 x, float2 neg, float2 zero, float2& h, float2& nl) {
    h = fma2(x, x, zero);
    nl = fma2(mul2(x, neg), x, h);
}

__device__ __forceinline__ void ff_acc_sq2(float2& hi, float2& lo, float2 x, float2 neg,
                                           float2 zero) {
    float2 h, nl;
    ff_sq2(x, neg, zero, h, nl);
    ff_acc2(hi, lo, h, nl);
}

// The two sums of a pair merged into one (hi, lo).
__device__ __forceinline__ void ff_merge2(float2 hi2, float2 lo2, float& hi, float& lo) {
    hi = hi2.x;
    lo = lo2.x;
    ff_acc(hi, lo, hi2.y, lo2.y);
}

__device__ __forceinline__ void ff_warp_sum(float& hi, float& lo) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float oh = __shfl_xor_sync(0xFFFFFFFFu, hi, o);
        const float ol = __shfl_xor_sync(0xFFFFFFFFu, lo, o);
        ff_acc(hi, lo, oh, ol);
    }
}

}  // namespace alq
