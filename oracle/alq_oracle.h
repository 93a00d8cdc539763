/*
 * alq_oracle.h -- CPU oracle of the AL-quantized optimizer step.
 *
 * TEST INFRASTRUCTURE. Only the tests, the package smoke check and the
 * benchmark's CPU-baseline leg may load or call this code; the product path
 * never does. It shares no code with the CUDA implementation.
 *
 * Plain, slow, single-threaded C. Transcendentals (log2, exp2) and all
 * reductions are computed in double and rounded once to fp32; the state EMAs
 * and parameter updates are fp32 in the operation order stated in the source
 * (the file is compiled with -ffp-contract=off: a multiply-add is fused only
 * where the source calls fmaf).
 *
 * Codes are stored as uint8_t when bits <= 8 and uint16_t when bits > 8.
 * Metadata is (l_min, Delta) per block, interleaved.
 */
#ifndef ALQ_ORACLE_H_
#define ALQ_ORACLE_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- AL codec: Sec. 4.1, Eq. (3)-(5); bits in [2, 16], L = 2^bits ------- */

/* Per-block (l_min, Delta) of Eq. (3) plus the degenerate handling of
 * Sec. 4.1. Returns 0 (and writes (0, 0)) when the block has no positive
 * value, 1 otherwise. */
int ora_al_block_meta(const float* x, int64_t len, float log_floor,
                      float* lmin, float* delta);

/* Code of one value under given (l_min, Delta): Eq. (4). */
uint32_t ora_al_quantize(float x, float lmin, float delta, int bits);

/* Value of one code under given (l_min, Delta): Eq. (5). */
float ora_al_dequantize(uint32_t q, float lmin, float delta, int bits);

void ora_al_encode(const float* x, int64_t n, int block, int bits,
                   float log_floor, void* codes, float* meta);
void ora_al_decode(const void* codes, const float* meta, int64_t n, int block,
                   int bits, float* out);

/* Logical bytes of an AL state (Sec. 4.4, Eq. (7)). */
int64_t ora_al_state_bytes(int64_t n, int block, int bits);

/* ---- UF8 signed momentum code: Sec. 4.3 ---------------------------------- */
void ora_uf8_encode(const float* m, int64_t n, int block, int8_t* codes,
                    float* absmax);
void ora_uf8_decode(const int8_t* codes, const float* absmax, int64_t n,
                    int block, float* out);

/* ---- AdamW: Sec. 3.1 Eq. (1), Sec. 6.2 ----------------------------------- */
typedef struct {
    float lr, beta1, beta2, eps, weight_decay, log_floor;
} ora_adamw_hp;

/* fp32-state AdamW (m, v are fp32 arrays updated in place):
 * p1 = p decay; m = fma(b1, m, (1-b1) g); v = fma(b2, v, (1-b2) g^2);
 * p = fma(-step, m / fma(sqrt(v), c2, eps), p1). */
void ora_adamw_update_fp32(float* p, const float* g, float* m, float* v,
                           int64_t n, const ora_adamw_hp* hp, int64_t t);

/* Quantized AdamW: UF8 m, AL v. m_fresh / v_fresh (nullable) receive the
 * fresh fp32 states before re-encoding. */
void ora_adamw_step(float* p, const float* g, int8_t* m_codes,
                    float* m_absmax, void* v_codes, float* v_meta, int64_t n,
                    int m_block, int v_block, int v_bits,
                    const ora_adamw_hp* hp, int64_t t, float* m_fresh,
                    float* v_fresh);

/* ---- Adafactor: Sec. 3.1 (factored second moment) ------------------------- */
typedef struct {
    float lr, eps1, clip_d, decay_rate, beta1, weight_decay, log_floor;
} ora_adafactor_hp;

/* fp32-state Adafactor; R [rows], C [cols] in place; M [rows*cols] or NULL. */
void ora_adafactor_update_fp32(float* p, const float* g, int64_t rows,
                               int64_t cols, float* R, float* C, float* M,
                               const ora_adafactor_hp* hp, int64_t t);

/* Quantized Adafactor: AL factors (fac_bits, fac_block), optional UF8 M.
 * R_fresh, C_fresh, M_fresh (nullable) receive the fresh fp32 states. */
void ora_adafactor_step(float* p, const float* g, int64_t rows, int64_t cols,
                        void* r_codes, float* r_meta, void* c_codes,
                        float* c_meta, int fac_bits, int fac_block,
                        int8_t* m_codes, float* m_absmax, int m_block,
                        const ora_adafactor_hp* hp, int64_t t, float* R_fresh,
                        float* C_fresh, float* M_fresh);

/* ---- CAME: Sec. 3.1 (dense M, factored V and confidence C) ---------------- */
typedef struct {
    float lr, beta1, beta2, beta3, eps1, eps2, clip_d, weight_decay,
        log_floor_v, log_floor_c;
} ora_came_hp;

void ora_came_update_fp32(float* p, const float* g, int64_t rows, int64_t cols,
                          float* Vr, float* Vc, float* Cr, float* Cc, float* M,
                          const ora_came_hp* hp, int64_t t);

/* fresh (nullable): [rows] Vr, [cols] Vc, [rows] Cr, [cols] Cc,
 * [rows*cols] M, packed in that order. */
void ora_came_step(float* p, const float* g, int64_t rows, int64_t cols,
                   void* vr_codes, float* vr_meta, void* vc_codes,
                   float* vc_meta, int v_bits, int v_block, void* cr_codes,
                   float* cr_meta, void* cc_codes, float* cc_meta, int c_bits,
                   int c_block, int8_t* m_codes, float* m_absmax, int m_block,
                   const ora_came_hp* hp, int64_t t, float* fresh);

/* ---- APOLLO: Sec. 3.1 (projected moments, channel-wise scale) ------------- */
typedef struct {
    float lr, beta1, beta2, eps, alpha, weight_decay, norm_growth_gamma,
        log_floor;
    int32_t rank;
} ora_apollo_hp;

/* Projection R = P * bf16(G) over the short side, channel-major [c x rank],
 * accumulated in double and rounded once to fp32. */
void ora_apollo_project(const float* g, int64_t rows, int64_t cols,
                        const uint16_t* proj, int rank, float* R);

/* fp32-state APOLLO: MP, VP [c x rank] in place; prev_norm in place;
 * scale_out (nullable) receives s_j [c]. */
void ora_apollo_update_fp32(float* p, const float* g, int64_t rows,
                            int64_t cols, const uint16_t* proj, float* MP,
                            float* VP, float* prev_norm,
                            const ora_apollo_hp* hp, int64_t t,
                            float* scale_out);

/* Everything after the projection, for a given R [c x rank] (fp32 states). */
void ora_apollo_update_given_R(float* p, const float* g, int64_t rows,
                               int64_t cols, const float* R, float* MP,
                               float* VP, float* prev_norm,
                               const ora_apollo_hp* hp, int64_t t,
                               float* scale_out);

/* Quantized APOLLO for a given projection R. */
void ora_apollo_step_given_R(float* p, const float* g, int64_t rows,
                             int64_t cols, const float* R, int8_t* m_codes,
                             float* m_absmax, int m_block, void* v_codes,
                             float* v_meta, int v_bits, int v_block,
                             float* prev_norm, const ora_apollo_hp* hp,
                             int64_t t, float* scale_out);

/* Quantized APOLLO: UF8 M^P, AL V^P over the flattened [c x rank] arrays. */
void ora_apollo_step(float* p, const float* g, int64_t rows, int64_t cols,
                     const uint16_t* proj, int8_t* m_codes, float* m_absmax,
                     int m_block, void* v_codes, float* v_meta, int v_bits,
                     int v_block, float* prev_norm, const ora_apollo_hp* hp,
                     int64_t t, float* scale_out, float* MP_fresh,
                     float* VP_fresh);

/* bf16 helpers (round to nearest even; finite inputs). */
uint16_t ora_f32_to_bf16(float x);
float ora_bf16_to_f32(uint16_t b);

/* ---- Eq. (2): relative update error ---------------------------------------- */
double ora_update_error(const float* u_hat, const float* u_ref, int64_t n,
                        double eps);

#ifdef __cplusplus
}
#endif

#endif /* ALQ_ORACLE_H_ */
