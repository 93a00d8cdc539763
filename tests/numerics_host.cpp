// Host build of the CUDA library's codec arithmetic (alq_numerics.h), for CPU
// tests only. Exposes C entry points so pytest can drive the exact-rounding
// fast paths over millions of inputs and compare them with the oracle.
#include "alq_numerics.h"

using namespace alq;

extern "C" {

float alqn_log2_rn(float x) { return log2_rn(x); }

// The certified fast path alone: ok = 1 when it vouches for its result.
float alqn_log2_rn_fast(float x, int* ok) {
    bool o;
    const float r = log2_rn_fast(x, o);
    *ok = o ? 1 : 0;
    return r;
}

void alqn_block_params(float mn, float mx, float floor_, float* lmin, float* delta) {
    al_block_params(mn, mx, floor_, *lmin, *delta);
}

// Level k (two-float) of a block, as the decode tables build it.
void alqn_level(float lmin, float delta, int k, float Lm2, float* hi, float* lo) {
    al_level_ff(lmin, delta, (float)k, Lm2, 1.0f / Lm2, *hi, *lo);
}

// AL8 decode through the two 16-entry tables; fb_count accumulates fallbacks.
void alqn_al8_decode(const uint8_t* q, int64_t n, float lmin, float delta,
                     float* out, int64_t* fb_count) {
    float th[16], tl[16], uh[16], ul[16];
    const float inv = 1.0f / 254.0f;
    for (int a = 0; a < 16; ++a) al_level_ff(lmin, delta, (float)(16 * a), 254.0f, inv, th[a], tl[a]);
    for (int b = 0; b < 16; ++b) al_level_ff(0.0f, delta, (float)(b - 1), 254.0f, inv, uh[b], ul[b]);
    for (int64_t i = 0; i < n; ++i) {
        uint32_t c = q[i];
        if (c == 0) { out[i] = 0.0f; continue; }
        bool fb;
        float v = al8_decode_pair(th[c >> 4], tl[c >> 4], uh[c & 15], ul[c & 15], fb);
        if (fb) {
            ++*fb_count;
            v = al_dequantize_fp64(c, lmin, delta, 254.0);
        }
        out[i] = v;
    }
}

// Fast Eq. (4) with FP64 fallback; fb_count accumulates fallbacks.
void alqn_al_quantize(const float* x, int64_t n, float lmin, float delta,
                      int bits, uint32_t* codes, int64_t* fb_count) {
    float Lm2 = (float)((1u << bits) - 2u);
    const AlEncConsts ek = al_encode_consts(lmin, delta, Lm2);
    for (int64_t i = 0; i < n; ++i) {
        if (x[i] == 0.0f) { codes[i] = 0; continue; }
        bool fb;
        uint32_t q = al_quantize_fast(x[i], ek, Lm2, fb);
        if (fb) {
            ++*fb_count;
            q = al_quantize_refine(x[i], lmin, delta, Lm2);
        }
        codes[i] = q;
    }
}

// Two-float Eq. (4) alone for every nonzero value (FP64 where it cannot
// decide); undecided counts those.
void alqn_al_quantize_ff(const float* x, int64_t n, float lmin, float delta, int bits,
                         uint32_t* codes, int64_t* undecided) {
    float Lm2 = (float)((1u << bits) - 2u);
    for (int64_t i = 0; i < n; ++i) {
        if (x[i] == 0.0f) { codes[i] = 0; continue; }
        bool ok;
        uint32_t q = al_quantize_ff(x[i], lmin, delta, Lm2, ok);
        if (!ok) {
            ++*undecided;
            q = al_quantize_fp64(x[i], lmin, delta, (double)Lm2);
        }
        codes[i] = q;
    }
}

}  // extern "C"
