// alq_factored.cu -- Adafactor / CAME / APOLLO steps and their workspace sizes.
#include "alq_internal.h"

using namespace alq;

extern "C" {

int al_workspace_size(int op, int64_t rows, int64_t cols, int rank, size_t* bytes) {
    (void)op; (void)rows; (void)cols; (void)rank;
    if (!bytes) return ALQ_ERR_INVALID_ARG;
    *bytes = 0;
    return ALQ_ERR_UNSUPPORTED;
}

int al_adafactor_step(float*, const float*, int64_t, int64_t, void*, float*, void*, float*, int, int,
                      int8_t*, float*, int, const al_adafactor_hp*, int64_t, void*, size_t, void*) {
    return ALQ_ERR_UNSUPPORTED;
}

int al_came_step(float*, const float*, int64_t, int64_t, void*, float*, void*, float*, int, int, void*,
                 float*, void*, float*, int, int, int8_t*, float*, int, const al_came_hp*, int64_t,
                 void*, size_t, void*) {
    return ALQ_ERR_UNSUPPORTED;
}

int al_apollo_step(float*, const float*, int64_t, int64_t, const uint16_t*, int8_t*, float*, int, void*,
                   float*, int, int, float*, const al_apollo_hp*, int64_t, void*, size_t, void*) {
    return ALQ_ERR_UNSUPPORTED;
}

}  // extern "C"
