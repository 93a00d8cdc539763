// alq_noalloc.cu -- an Adafactor step for callers that cannot allocate GPU
// memory.
//
// Some callers cannot call cudaMalloc (or any allocator) at the point where
// they run an optimizer step: code running inside a framework that owns all
// device memory through its own pool, code that must not allocate after
// start-up (fixed memory budgets, real-time loops), or callers without access
// to the CUDA allocator through their language binding. al_adafactor_step
// needs a workspace for its row/column partial sums; this variant takes it
// from a fixed array that lives in the library's device image instead, so the
// caller passes only its inputs and outputs.
//
// The array is a file-scope __device__ variable: every GPU that loads this
// library holds kNoAllocScratchBytes of device memory for it until the
// process exits. Host code cannot use the array's name as a device address:
// each call looks the address up with cudaGetSymbolAddress, with the
// calling thread's device and context current. The lookup is a host-side
// table read once the library's device code is loaded (the first call on a
// device may load it), and doing it per call means the address can never be
// stale after cudaDeviceReset or under another context on the same device.
#include "alq_internal.h"

namespace alq {

constexpr size_t kNoAllocScratchBytes = size_t(4) << 20;  // 4 MiB
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of g_noalloc_scratch in the current context. Returns
// nullptr (and records the CUDA error) on failure.
static void* scratch_address() {
    void* p = nullptr;
    if (record_cuda(cudaGetSymbolAddress(&p, g_noalloc_scratch)) != ALQ_OK) return nullptr;
    return p;
}

}  // namespace alq

using namespace alq;

extern "C" {

size_t al_adafactor_noalloc_capacity(void) { return kNoAllocScratchBytes; }

int al_adafactor_step_noalloc(float* p, const float* g, int64_t rows, int64_t cols,
                              void* r_codes, float* r_meta, void* c_codes, float* c_meta,
                              int fac_bits, int fac_block, int8_t* m_codes, float* m_absmax,
                              int m_block, const al_adafactor_hp* hp, int64_t t, void* stream) {
    size_t need = 0;
    int st = al_workspace_size(AL_OP_ADAFACTOR, rows, cols, 0, &need);
    if (st != ALQ_OK) return st;
    if (need > kNoAllocScratchBytes) return ALQ_ERR_WORKSPACE;  // matrix too large
    void* scratch = scratch_address();
    if (!scratch) return ALQ_ERR_CUDA;
    return al_adafactor_step(p, g, rows, cols, r_codes, r_meta, c_codes, c_meta, fac_bits,
                             fac_block, m_codes, m_absmax, m_block, hp, t, scratch,
                             kNoAllocScratchBytes, stream);
}

}  // extern "C"
