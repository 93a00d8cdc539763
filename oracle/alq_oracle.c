/*
 * alq_oracle.c -- CPU oracle of the AL-quantized optimizer step.
 *
 * TEST INFRASTRUCTURE: see alq_oracle.h. Only the tests, the smoke check and
 * the benchmark's CPU-baseline leg use it.
 *
 * Sources, by function:
 *   AL codec          Sec. 4.1, Eq. (3) bounds, Eq. (4) codes, Eq. (5) values,
 *                     degenerate handling and the l_max cap of 126 in the last
 *                     paragraph of Sec. 4.1; AL8/AL16 code counts in Sec. 4.1
 *                     and Sec. 4.4.
 *   storage           Sec. 4.4, Eq. (7).
 *   UF8               Sec. 4.3 ("uniform 8-bit quantization" of signed
 *                     momentum), momentum block 256 in Sec. 6.2.
 *   AdamW             Sec. 3.1, Eq. (1), with the decoupled weight decay and
 *                     bias correction of the AdamW algorithm the paper cites.
 *   Adafactor         Sec. 3.1 (row/column statistics reconstructing the
 *                     preconditioner), following the published Adafactor
 *                     algorithm: factored second moment with rho_t = 1 -
 *                     t^decay, update clipping by RMS(u)/d.
 *   CAME              Sec. 3.1 (dense M, factored V and confidence C),
 *                     following the published CAME algorithm: residual
 *                     (u_hat - m)^2 + eps2 tracked by factored beta3-EMAs.
 *   APOLLO            Sec. 3.1 (projected moments give a channel-wise scale of
 *                     the original gradient), rank 256 and channel-wise
 *                     scaling in Sec. 6.1.
 *   update error      Sec. 3.2, Eq. (2).
 *
 * Threads: the file also builds with -fopenmp (the benchmark's all-core CPU
 * baseline). Only loops whose iterations are independent carry an OpenMP
 * pragma -- blocks, elements, rows, columns, channels, each summed in its
 * own fixed order -- and every reduction across them stays a sequential
 * loop, so both builds give the same bits; without -fopenmp the pragmas are
 * ignored.
 *
 * Every function is pinned by tests that do not re-derive it: invariants and
 * closed forms of the paper (exact zero, endpoint codes, half-step round-trip
 * bound, monotone codes, brute force at 4 bits, storage numbers printed in
 * Sec. 5.5 and Sec. 6.2) and independent library optimizers (torch AdamW,
 * torch Adafactor, torch Adam for the projected moments) in the special cases
 * where they coincide with the quantized step's fp32 form.
 */
#include "alq_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ===================================================================== AL */

static int64_t nblocks_of(int64_t n, int block) {
    return (n + block - 1) / block;
}

static uint32_t code_get(const void* codes, int bits, int64_t i) {
    if (bits <= 8) return ((const uint8_t*)codes)[i];
    return ((const uint16_t*)codes)[i];
}

static void code_set(void* codes, int bits, int64_t i, uint32_t q) {
    if (bits <= 8)
        ((uint8_t*)codes)[i] = (uint8_t)q;
    else
        ((uint16_t*)codes)[i] = (uint16_t)q;
}

/* Eq. (3): l_min = max(l_floor, min_{x>0} log2 x), l_max = max_{x>0} log2 x,
 * each log rounded once to fp32. Sec. 4.1: l_max is capped at 126; a
 * collapsed interval (all positive values equal, or all below the floor) is
 * widened by one unit, l_max = l_min + 1; the width is at least 1e-12. */
int ora_al_block_meta(const float* x, int64_t len, float log_floor,
                      float* lmin_out, float* delta_out) {
    float mn = INFINITY, mx = 0.0f;
    int any = 0;
    for (int64_t i = 0; i < len; ++i) {
        float v = x[i];
        if (v > 0.0f) {
            any = 1;
            if (v < mn) mn = v;
            if (v > mx) mx = v;
        }
    }
    if (!any) {
        *lmin_out = 0.0f;
        *delta_out = 0.0f;
        return 0;
    }
    float lmin = (float)log2((double)mn);
    if (lmin < log_floor) lmin = log_floor;
    float lmax = (float)log2((double)mx);
    if (lmax > 126.0f) lmax = 126.0f;
    if (lmax <= lmin) lmax = lmin + 1.0f;
    float delta = lmax - lmin;
    if (delta < 1e-12f) delta = 1e-12f;
    *lmin_out = lmin;
    *delta_out = delta;
    return 1;
}

/* Eq. (4): q = 0 for x = 0, else 1 + round((L-2) z) with
 * z = clip((log2 x - l_min) / Delta, 0, 1); round half to even. */
uint32_t ora_al_quantize(float x, float lmin, float delta, int bits) {
    if (x == 0.0f) return 0u;
    const double Lm2 = (double)((1u << bits) - 2u);
    double t = (Lm2 * (log2((double)x) - (double)lmin)) / (double)delta;
    if (t < 0.0) t = 0.0;
    if (t > Lm2) t = Lm2;
    return 1u + (uint32_t)rint(t);
}

/* Eq. (5): x_hat = 0 for q = 0, else 2^(l_min + (q-1) Delta / (L-2)). */
float ora_al_dequantize(uint32_t q, float lmin, float delta, int bits) {
    if (q == 0u) return 0.0f;
    const double Lm2 = (double)((1u << bits) - 2u);
    double y = (double)lmin + ((double)(q - 1u) * (double)delta) / Lm2;
    return (float)exp2(y);
}

void ora_al_encode(const float* x, int64_t n, int block, int bits,
                   float log_floor, void* codes, float* meta) {
    int64_t nb = nblocks_of(n, block);
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < nb; ++b) {
        int64_t lo = b * block;
        int64_t len = (n - lo < block) ? (n - lo) : block;
        float lmin, delta;
        int any = ora_al_block_meta(x + lo, len, log_floor, &lmin, &delta);
        meta[2 * b] = lmin;
        meta[2 * b + 1] = delta;
        for (int64_t i = 0; i < len; ++i) {
            uint32_t q = any ? ora_al_quantize(x[lo + i], lmin, delta, bits) : 0u;
            code_set(codes, bits, lo + i, q);
        }
    }
}

void ora_al_decode(const void* codes, const float* meta, int64_t n, int block,
                   int bits, float* out) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        int64_t b = i / block;
        out[i] = ora_al_dequantize(code_get(codes, bits, i), meta[2 * b],
                                   meta[2 * b + 1], bits);
    }
}

/* A state kept in a role's precision (Sec. 4.5, state policy): AL8/AL16
 * codes with block metadata, or bits == 32, the unquantized fp32 state
 * (codes then point to fp32 values; there is no metadata). */
static void state_decode(const void* codes, const float* meta, int64_t n,
                         int block, int bits, float* out) {
    if (bits == 32)
        memcpy(out, codes, sizeof(float) * (size_t)n);
    else
        ora_al_decode(codes, meta, n, block, bits, out);
}

static void state_encode(const float* x, int64_t n, int block, int bits,
                         float log_floor, void* codes, float* meta) {
    if (bits == 32)
        memcpy(codes, x, sizeof(float) * (size_t)n);
    else
        ora_al_encode(x, n, block, bits, log_floor, codes, meta);
}

/* Eq. (7): code bytes plus two fp32 values per block. */
int64_t ora_al_state_bytes(int64_t n, int block, int bits) {
    int64_t code_bytes = (bits <= 8) ? n : 2 * n;
    return code_bytes + 8 * nblocks_of(n, block);
}

/* ==================================================================== UF8 */

/* Symmetric per-block absmax code: q = rint(m * (127 / s)), s = max |m|.
 * For s < 2^-120 both m and s are scaled by 2^64 (exact) first. */
void ora_uf8_encode(const float* m, int64_t n, int block, int8_t* codes,
                    float* absmax) {
    int64_t nb = nblocks_of(n, block);
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < nb; ++b) {
        int64_t lo = b * block;
        int64_t len = (n - lo < block) ? (n - lo) : block;
        float s = 0.0f;
        for (int64_t i = 0; i < len; ++i) {
            float a = fabsf(m[lo + i]);
            if (a > s) s = a;
        }
        absmax[b] = s;
        if (s == 0.0f) {
            for (int64_t i = 0; i < len; ++i) codes[lo + i] = 0;
            continue;
        }
        float sc = (s < 0x1p-120f) ? 0x1p64f : 1.0f;
        float inv = 127.0f / (s * sc);
        for (int64_t i = 0; i < len; ++i) {
            float f = (m[lo + i] * sc) * inv;
            codes[lo + i] = (int8_t)(int)rintf(f);
        }
    }
}

void ora_uf8_decode(const int8_t* codes, const float* absmax, int64_t n,
                    int block, float* out) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        float d = absmax[i / block] / 127.0f;
        out[i] = (float)codes[i] * d;
    }
}

/* ================================================================== AdamW */

void ora_adamw_update_fp32(float* p, const float* g, float* m, float* v,
                           int64_t n, const ora_adamw_hp* hp, int64_t t) {
    const double bc1 = 1.0 - pow((double)hp->beta1, (double)t);
    const double bc2 = 1.0 - pow((double)hp->beta2, (double)t);
    const float decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    const float step = (float)((double)hp->lr / bc1);
    const float c2 = (float)(1.0 / sqrt(bc2));
    const float omb1 = (float)(1.0 - (double)hp->beta1);
    const float omb2 = (float)(1.0 - (double)hp->beta2);
    const float b1 = hp->beta1, b2 = hp->beta2, eps = hp->eps;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        float gi = g[i];
        /* Eq. (1) in fp32; a product that is added is fused with the sum
         * (one rounding), every other operation rounds on its own */
        float p1 = p[i] * decay;
        float mi = fmaf(b1, m[i], omb1 * gi);
        float vi = fmaf(b2, v[i], omb2 * (gi * gi));
        float den = fmaf(sqrtf(vi), c2, eps);
        p[i] = fmaf(-step, mi / den, p1);
        m[i] = mi;
        v[i] = vi;
    }
}

void ora_adamw_step(float* p, const float* g, int8_t* m_codes,
                    float* m_absmax, void* v_codes, float* v_meta, int64_t n,
                    int m_block, int v_block, int v_bits,
                    const ora_adamw_hp* hp, int64_t t, float* m_fresh,
                    float* v_fresh) {
    /* v_bits == 32: the unquantized reference, m and v dense fp32 (m_codes
     * and v_codes point to fp32 arrays; m_absmax and v_meta are unused) */
    float* m = (float*)malloc(sizeof(float) * (size_t)(n > 0 ? n : 1));
    float* v = (float*)malloc(sizeof(float) * (size_t)(n > 0 ? n : 1));
    if (v_bits == 32)
        memcpy(m, m_codes, sizeof(float) * (size_t)n);
    else
        ora_uf8_decode(m_codes, m_absmax, n, m_block, m);
    state_decode(v_codes, v_meta, n, v_block, v_bits, v);
    ora_adamw_update_fp32(p, g, m, v, n, hp, t);
    if (m_fresh) memcpy(m_fresh, m, sizeof(float) * (size_t)n);
    if (v_fresh) memcpy(v_fresh, v, sizeof(float) * (size_t)n);
    if (v_bits == 32)
        memcpy(m_codes, m, sizeof(float) * (size_t)n);
    else
        ora_uf8_encode(m, n, m_block, m_codes, m_absmax);
    state_encode(v, n, v_block, v_bits, hp->log_floor, v_codes, v_meta);
    free(m);
    free(v);
}

/* ====================================================== factored helpers */

/* mean_j(g_ij^2 + eps1) for every row, exact squares summed in double. */
static void row_sq_means(const float* g, int64_t rows, int64_t cols,
                         float eps1, float* r) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows; ++i) {
        double s = 0.0;
        for (int64_t j = 0; j < cols; ++j) {
            double x = (double)g[i * cols + j];
            s += x * x;
        }
        r[i] = (float)(s / (double)cols + (double)eps1);
    }
}

static void col_sq_means(const float* g, int64_t rows, int64_t cols,
                         float eps1, float* c) {
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < cols; ++j) {
        double s = 0.0;
        for (int64_t i = 0; i < rows; ++i) {
            double x = (double)g[i * cols + j];
            s += x * x;
        }
        c[j] = (float)(s / (double)rows + (double)eps1);
    }
}

static float mean_f(const float* x, int64_t n) {
    double s = 0.0;
    for (int64_t i = 0; i < n; ++i) s += (double)x[i];
    return (float)(s / (double)n);
}

/* a_i = 1/sqrt(R_i / mean(R)), b_j = 1/sqrt(C_j): the factors of
 * 1/sqrt(V_hat) with V_hat_ij = R_i C_j / mean(R). */
static void inv_sqrt_factors(const float* R, int64_t rows, const float* C,
                             int64_t cols, float* a, float* b) {
    float meanR = mean_f(R, rows);
    for (int64_t i = 0; i < rows; ++i) a[i] = 1.0f / sqrtf(R[i] / meanR);
    for (int64_t j = 0; j < cols; ++j) b[j] = 1.0f / sqrtf(C[j]);
}

/* u = (g * a_i) * b_j and the clip factor 1/max(1, RMS(u)/d). */
static float scaled_update(const float* g, int64_t rows, int64_t cols,
                           const float* a, const float* b, float clip_d,
                           float* u) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows; ++i)
        for (int64_t j = 0; j < cols; ++j) u[i * cols + j] = (g[i * cols + j] * a[i]) * b[j];
    double ss = 0.0;  /* in element order */
    for (int64_t k = 0; k < rows * cols; ++k) ss += (double)u[k] * (double)u[k];
    double rms = sqrt(ss / ((double)rows * (double)cols));
    double cf = rms / (double)clip_d;
    if (cf < 1.0) cf = 1.0;
    return (float)(1.0 / cf);
}

static void* xmalloc(size_t bytes) { return malloc(bytes > 0 ? bytes : 1); }

/* ============================================================== Adafactor */

void ora_adafactor_update_fp32(float* p, const float* g, int64_t rows,
                               int64_t cols, float* R, float* C, float* M,
                               const ora_adafactor_hp* hp, int64_t t) {
    const int64_t n = rows * cols;
    const double omr_d = pow((double)t, (double)hp->decay_rate);
    const float omr = (float)omr_d;
    const float rho = (float)(1.0 - omr_d);
    const float decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    const float omb1 = (float)(1.0 - (double)hp->beta1);

    float* r = (float*)xmalloc(sizeof(float) * (size_t)rows);
    float* c = (float*)xmalloc(sizeof(float) * (size_t)cols);
    float* a = (float*)xmalloc(sizeof(float) * (size_t)rows);
    float* b = (float*)xmalloc(sizeof(float) * (size_t)cols);
    float* u = (float*)xmalloc(sizeof(float) * (size_t)n);

    row_sq_means(g, rows, cols, hp->eps1, r);
    col_sq_means(g, rows, cols, hp->eps1, c);
    for (int64_t i = 0; i < rows; ++i) R[i] = rho * R[i] + omr * r[i];
    for (int64_t j = 0; j < cols; ++j) C[j] = rho * C[j] + omr * c[j];
    inv_sqrt_factors(R, rows, C, cols, a, b);
    const float icf = scaled_update(g, rows, cols, a, b, hp->clip_d, u);
#pragma omp parallel for schedule(static)
    for (int64_t k = 0; k < n; ++k) {
        float uh = u[k] * icf;
        float upd = uh;
        if (M) {
            float mk = hp->beta1 * M[k] + omb1 * uh;
            M[k] = mk;
            upd = mk;
        }
        p[k] = p[k] * decay - hp->lr * upd;
    }
    free(r); free(c); free(a); free(b); free(u);
}

void ora_adafactor_step(float* p, const float* g, int64_t rows, int64_t cols,
                        void* r_codes, float* r_meta, void* c_codes,
                        float* c_meta, int fac_bits, int fac_block,
                        int8_t* m_codes, float* m_absmax, int m_block,
                        const ora_adafactor_hp* hp, int64_t t, float* R_fresh,
                        float* C_fresh, float* M_fresh) {
    const int64_t n = rows * cols;
    float* R = (float*)xmalloc(sizeof(float) * (size_t)rows);
    float* C = (float*)xmalloc(sizeof(float) * (size_t)cols);
    float* M = m_codes ? (float*)xmalloc(sizeof(float) * (size_t)n) : NULL;
    state_decode(r_codes, r_meta, rows, fac_block, fac_bits, R);
    state_decode(c_codes, c_meta, cols, fac_block, fac_bits, C);
    if (M) ora_uf8_decode(m_codes, m_absmax, n, m_block, M);
    ora_adafactor_update_fp32(p, g, rows, cols, R, C, M, hp, t);
    if (R_fresh) memcpy(R_fresh, R, sizeof(float) * (size_t)rows);
    if (C_fresh) memcpy(C_fresh, C, sizeof(float) * (size_t)cols);
    if (M_fresh && M) memcpy(M_fresh, M, sizeof(float) * (size_t)n);
    state_encode(R, rows, fac_block, fac_bits, hp->log_floor, r_codes, r_meta);
    state_encode(C, cols, fac_block, fac_bits, hp->log_floor, c_codes, c_meta);
    if (M) ora_uf8_encode(M, n, m_block, m_codes, m_absmax);
    free(R); free(C); free(M);
}

/* =================================================================== CAME */

void ora_came_update_fp32(float* p, const float* g, int64_t rows, int64_t cols,
                          float* Vr, float* Vc, float* Cr, float* Cc, float* M,
                          const ora_came_hp* hp, int64_t t) {
    (void)t; /* CAME uses constant EMA rates and no bias correction */
    const int64_t n = rows * cols;
    const float omb1 = (float)(1.0 - (double)hp->beta1);
    const float omb2 = (float)(1.0 - (double)hp->beta2);
    const float omb3 = (float)(1.0 - (double)hp->beta3);
    const float decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);

    float* r = (float*)xmalloc(sizeof(float) * (size_t)rows);
    float* c = (float*)xmalloc(sizeof(float) * (size_t)cols);
    float* a = (float*)xmalloc(sizeof(float) * (size_t)rows);
    float* b = (float*)xmalloc(sizeof(float) * (size_t)cols);
    float* u = (float*)xmalloc(sizeof(float) * (size_t)n);
    float* res = (float*)xmalloc(sizeof(float) * (size_t)n);

    /* second-moment factors */
    row_sq_means(g, rows, cols, hp->eps1, r);
    col_sq_means(g, rows, cols, hp->eps1, c);
    for (int64_t i = 0; i < rows; ++i) Vr[i] = hp->beta2 * Vr[i] + omb2 * r[i];
    for (int64_t j = 0; j < cols; ++j) Vc[j] = hp->beta2 * Vc[j] + omb2 * c[j];
    inv_sqrt_factors(Vr, rows, Vc, cols, a, b);
    const float icf = scaled_update(g, rows, cols, a, b, hp->clip_d, u);

    /* momentum of the clipped update and its residual */
#pragma omp parallel for schedule(static)
    for (int64_t k = 0; k < n; ++k) {
        float uh = u[k] * icf;
        float mk = hp->beta1 * M[k] + omb1 * uh;
        M[k] = mk;
        float d = uh - mk;
        res[k] = d * d + hp->eps2;
    }

    /* confidence factors: beta3-EMAs of the residual's row/column means */
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows; ++i) {
        double s = 0.0;
        for (int64_t j = 0; j < cols; ++j) s += (double)res[i * cols + j];
        r[i] = (float)(s / (double)cols);
    }
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < cols; ++j) {
        double s = 0.0;
        for (int64_t i = 0; i < rows; ++i) s += (double)res[i * cols + j];
        c[j] = (float)(s / (double)rows);
    }
    for (int64_t i = 0; i < rows; ++i) Cr[i] = hp->beta3 * Cr[i] + omb3 * r[i];
    for (int64_t j = 0; j < cols; ++j) Cc[j] = hp->beta3 * Cc[j] + omb3 * c[j];
    inv_sqrt_factors(Cr, rows, Cc, cols, a, b);

#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows; ++i)
        for (int64_t j = 0; j < cols; ++j) {
            int64_t k = i * cols + j;
            float upd = (M[k] * a[i]) * b[j];
            p[k] = p[k] * decay - hp->lr * upd;
        }
    free(r); free(c); free(a); free(b); free(u); free(res);
}

void ora_came_step(float* p, const float* g, int64_t rows, int64_t cols,
                   void* vr_codes, float* vr_meta, void* vc_codes,
                   float* vc_meta, int v_bits, int v_block, void* cr_codes,
                   float* cr_meta, void* cc_codes, float* cc_meta, int c_bits,
                   int c_block, int8_t* m_codes, float* m_absmax, int m_block,
                   const ora_came_hp* hp, int64_t t, float* fresh) {
    const int64_t n = rows * cols;
    float* Vr = (float*)xmalloc(sizeof(float) * (size_t)rows);
    float* Vc = (float*)xmalloc(sizeof(float) * (size_t)cols);
    float* Cr = (float*)xmalloc(sizeof(float) * (size_t)rows);
    float* Cc = (float*)xmalloc(sizeof(float) * (size_t)cols);
    float* M = (float*)xmalloc(sizeof(float) * (size_t)n);
    state_decode(vr_codes, vr_meta, rows, v_block, v_bits, Vr);
    state_decode(vc_codes, vc_meta, cols, v_block, v_bits, Vc);
    state_decode(cr_codes, cr_meta, rows, c_block, c_bits, Cr);
    state_decode(cc_codes, cc_meta, cols, c_block, c_bits, Cc);
    ora_uf8_decode(m_codes, m_absmax, n, m_block, M);
    ora_came_update_fp32(p, g, rows, cols, Vr, Vc, Cr, Cc, M, hp, t);
    if (fresh) {
        float* f = fresh;
        memcpy(f, Vr, sizeof(float) * (size_t)rows); f += rows;
        memcpy(f, Vc, sizeof(float) * (size_t)cols); f += cols;
        memcpy(f, Cr, sizeof(float) * (size_t)rows); f += rows;
        memcpy(f, Cc, sizeof(float) * (size_t)cols); f += cols;
        memcpy(f, M, sizeof(float) * (size_t)n);
    }
    state_encode(Vr, rows, v_block, v_bits, hp->log_floor_v, vr_codes, vr_meta);
    state_encode(Vc, cols, v_block, v_bits, hp->log_floor_v, vc_codes, vc_meta);
    state_encode(Cr, rows, c_block, c_bits, hp->log_floor_c, cr_codes, cr_meta);
    state_encode(Cc, cols, c_block, c_bits, hp->log_floor_c, cc_codes, cc_meta);
    ora_uf8_encode(M, n, m_block, m_codes, m_absmax);
    free(Vr); free(Vc); free(Cr); free(Cc); free(M);
}

/* ================================================================= APOLLO */

uint16_t ora_f32_to_bf16(float x) {
    uint32_t u;
    memcpy(&u, &x, 4);
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7fffu + lsb;
    return (uint16_t)(u >> 16);
}

float ora_bf16_to_f32(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float x;
    memcpy(&x, &u, 4);
    return x;
}

/* If rows <= cols the rows are the short side: R[j][k] = sum_i P[k][i] g[i][j]
 * with channels j over the columns; otherwise R[j][k] = sum_i P[k][i] g[j][i]
 * with channels over the rows. Both operands are rounded to bf16 once, into
 * double copies laid out with the short side contiguous; every sum runs over
 * i in ascending order. */
void ora_apollo_project(const float* g, int64_t rows, int64_t cols,
                        const uint16_t* proj, int rank, float* R) {
    const int rows_short = rows <= cols;
    const int64_t s = rows_short ? rows : cols;
    const int64_t L = rows_short ? cols : rows;
    double* gb = (double*)malloc(sizeof(double) * (size_t)(L * s));   /* [L][s] */
    double* pb = (double*)malloc(sizeof(double) * (size_t)(rank * s)); /* [rank][s] */
    for (int64_t j = 0; j < L; ++j)
        for (int64_t i = 0; i < s; ++i) {
            float gv = rows_short ? g[i * cols + j] : g[j * cols + i];
            gb[j * s + i] = (double)ora_bf16_to_f32(ora_f32_to_bf16(gv));
        }
    for (int64_t q = 0; q < (int64_t)rank * s; ++q)
        pb[q] = (double)ora_bf16_to_f32(proj[q]);
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < L; ++j)
        for (int k = 0; k < rank; ++k) {
            const double* gj = gb + j * s;
            const double* pk = pb + (int64_t)k * s;
            double acc = 0.0;
            for (int64_t i = 0; i < s; ++i) acc += pk[i] * gj[i];
            R[j * rank + k] = (float)acc;
        }
    free(gb);
    free(pb);
}

/* Everything after the projection, for a given R [c x rank]. */
void ora_apollo_update_given_R(float* p, const float* g, int64_t rows,
                               int64_t cols, const float* R, float* MP,
                               float* VP, float* prev_norm,
                               const ora_apollo_hp* hp, int64_t t,
                               float* scale_out) {
    const int rank = hp->rank;
    const int rows_short = rows <= cols;
    const int64_t L = rows_short ? cols : rows;
    const double bc1 = 1.0 - pow((double)hp->beta1, (double)t);
    const double bc2 = 1.0 - pow((double)hp->beta2, (double)t);
    const float ic1 = (float)(1.0 / bc1);
    const float c2 = (float)(1.0 / sqrt(bc2));
    const float omb1 = (float)(1.0 - (double)hp->beta1);
    const float omb2 = (float)(1.0 - (double)hp->beta2);
    const float decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    const float lr_a = (float)((double)hp->lr * (double)hp->alpha);

    float* s = (float*)xmalloc(sizeof(float) * (size_t)L);
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < L; ++j) {
        double nr = 0.0, ng = 0.0;
        for (int k = 0; k < rank; ++k) {
            int64_t q = j * rank + k;
            float rv = R[q];
            float mq = hp->beta1 * MP[q] + omb1 * rv;
            float vq = hp->beta2 * VP[q] + omb2 * (rv * rv);
            MP[q] = mq;
            VP[q] = vq;
            float rt = (mq * ic1) / (sqrtf(vq) * c2 + hp->eps);
            nr += (double)rt * (double)rt;
            ng += (double)rv * (double)rv;
        }
        s[j] = (float)(sqrt(nr) / (sqrt(ng) + 1e-8));
    }
    if (scale_out) memcpy(scale_out, s, sizeof(float) * (size_t)L);

    /* optional norm-growth limiter on the scaled gradient */
    float lim = 1.0f;
    if (hp->norm_growth_gamma > 0.0f) {
        double ss = 0.0;
        for (int64_t i = 0; i < rows; ++i)
            for (int64_t j = 0; j < cols; ++j) {
                float gt = g[i * cols + j] * s[rows_short ? j : i];
                ss += (double)gt * (double)gt;
            }
        double nt = sqrt(ss);
        double prev = (double)*prev_norm;
        double cap = (double)hp->norm_growth_gamma * prev;
        if (prev > 0.0 && nt > cap) {
            lim = (float)(cap / nt);
            *prev_norm = (float)cap;
        } else {
            *prev_norm = (float)nt;
        }
    }

#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows; ++i)
        for (int64_t j = 0; j < cols; ++j) {
            int64_t k = i * cols + j;
            float gt = g[k] * s[rows_short ? j : i];
            if (hp->norm_growth_gamma > 0.0f) gt = gt * lim;
            p[k] = p[k] * decay - lr_a * gt;
        }
    free(s);
}

void ora_apollo_update_fp32(float* p, const float* g, int64_t rows,
                            int64_t cols, const uint16_t* proj, float* MP,
                            float* VP, float* prev_norm,
                            const ora_apollo_hp* hp, int64_t t,
                            float* scale_out) {
    const int64_t L = rows <= cols ? cols : rows;
    float* R = (float*)xmalloc(sizeof(float) * (size_t)(L * hp->rank));
    ora_apollo_project(g, rows, cols, proj, hp->rank, R);
    ora_apollo_update_given_R(p, g, rows, cols, R, MP, VP, prev_norm, hp, t, scale_out);
    free(R);
}

/* Quantized APOLLO for a given projection R (decode, update, encode). */
void ora_apollo_step_given_R(float* p, const float* g, int64_t rows,
                             int64_t cols, const float* R, int8_t* m_codes,
                             float* m_absmax, int m_block, void* v_codes,
                             float* v_meta, int v_bits, int v_block,
                             float* prev_norm, const ora_apollo_hp* hp,
                             int64_t t, float* scale_out) {
    const int64_t L = rows <= cols ? cols : rows;
    const int64_t np = L * hp->rank;
    float* MP = (float*)xmalloc(sizeof(float) * (size_t)np);
    float* VP = (float*)xmalloc(sizeof(float) * (size_t)np);
    ora_uf8_decode(m_codes, m_absmax, np, m_block, MP);
    ora_al_decode(v_codes, v_meta, np, v_block, v_bits, VP);
    ora_apollo_update_given_R(p, g, rows, cols, R, MP, VP, prev_norm, hp, t, scale_out);
    ora_uf8_encode(MP, np, m_block, m_codes, m_absmax);
    ora_al_encode(VP, np, v_block, v_bits, hp->log_floor, v_codes, v_meta);
    free(MP);
    free(VP);
}

void ora_apollo_step(float* p, const float* g, int64_t rows, int64_t cols,
                     const uint16_t* proj, int8_t* m_codes, float* m_absmax,
                     int m_block, void* v_codes, float* v_meta, int v_bits,
                     int v_block, float* prev_norm, const ora_apollo_hp* hp,
                     int64_t t, float* scale_out, float* MP_fresh,
                     float* VP_fresh) {
    const int64_t L = rows <= cols ? cols : rows;
    const int64_t np = L * hp->rank;
    float* MP = (float*)xmalloc(sizeof(float) * (size_t)np);
    float* VP = (float*)xmalloc(sizeof(float) * (size_t)np);
    ora_uf8_decode(m_codes, m_absmax, np, m_block, MP);
    ora_al_decode(v_codes, v_meta, np, v_block, v_bits, VP);
    ora_apollo_update_fp32(p, g, rows, cols, proj, MP, VP, prev_norm, hp, t,
                           scale_out);
    if (MP_fresh) memcpy(MP_fresh, MP, sizeof(float) * (size_t)np);
    if (VP_fresh) memcpy(VP_fresh, VP, sizeof(float) * (size_t)np);
    ora_uf8_encode(MP, np, m_block, m_codes, m_absmax);
    ora_al_encode(VP, np, v_block, v_bits, hp->log_floor, v_codes, v_meta);
    free(MP);
    free(VP);
}

/* ================================================================ Eq. (2) */

double ora_update_error(const float* u_hat, const float* u_ref, int64_t n,
                        double eps) {
    double num = 0.0, den = 0.0;
    for (int64_t i = 0; i < n; ++i) {
        double d = (double)u_hat[i] - (double)u_ref[i];
        num += d * d;
        den += (double)u_ref[i] * (double)u_ref[i];
    }
    return sqrt(num) / (sqrt(den) + eps);
}
