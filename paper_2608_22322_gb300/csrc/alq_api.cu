// alq_api.cu -- host-side entry points of the C ABI that launch nothing:
// status strings, error text, sizes, workspace sizes, and the AdamW scalar
// precomputation shared by the single- and multi-tensor steps.
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <map>
#include <mutex>
#include <utility>
#include <vector>

#include "alq_internal.h"

namespace alq {

static thread_local char g_last_error[256] = "";

int record_cuda(cudaError_t e) {
    if (e == cudaSuccess) return ALQ_OK;
    snprintf(g_last_error, sizeof(g_last_error), "%s: %s", cudaGetErrorName(e),
             cudaGetErrorString(e));
    return ALQ_ERR_CUDA;
}

int check_launch() { return record_cuda(cudaGetLastError()); }

bool valid_block(int block) {
    return block >= 128 && block <= 4096 && (block & (block - 1)) == 0;
}

bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

int64_t blocks_of(int64_t n, int block) { return (n + block - 1) / block; }

int sm_count() {
    static std::mutex mu;
    static std::vector<int> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    std::lock_guard<std::mutex> lock(mu);
    if ((int)cache.size() <= dev) cache.resize(dev + 1, 0);
    if (cache[dev] == 0) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        cache[dev] = v > 0 ? v : 1;
    }
    return cache[dev];
}

int persistent_grid(const void* kernel, int threads, size_t smem, int64_t ntiles) {
    static std::mutex mu;
    static std::map<std::pair<const void*, int>, int> cache;
    int dev = 0;
    cudaGetDevice(&dev);
    int occ = 0;
    {
        std::lock_guard<std::mutex> lock(mu);
        auto it = cache.find({kernel, dev});
        if (it != cache.end()) occ = it->second;
    }
    if (occ == 0) {
        // dynamic shared memory beyond the default 48 KB needs an opt-in per
        // kernel and device; the launch reports a failure if it is refused
        if (smem > 0) cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel, threads, smem) != cudaSuccess ||
            occ < 1)
            occ = 1;
        std::lock_guard<std::mutex> lock(mu);
        cache[{kernel, dev}] = occ;
    }
    const int64_t g = (int64_t)sm_count() * occ;
    return (int)(ntiles < g ? ntiles : g);
}

// Bias corrections and step sizes of the AdamW step, in double from the
// integer step t, rounded once to fp32 (the kernels never call pow).
AdamWScalars adamw_scalars(const al_adamw_hp* hp, int64_t t) {
    const double bc1 = 1.0 - pow((double)hp->beta1, (double)t);
    const double bc2 = 1.0 - pow((double)hp->beta2, (double)t);
    AdamWScalars s;
    s.decay = (float)(1.0 - (double)hp->lr * (double)hp->weight_decay);
    s.step = (float)((double)hp->lr / bc1);
    s.c2 = (float)(1.0 / sqrt(bc2));
    s.omb1 = (float)(1.0 - (double)hp->beta1);
    s.omb2 = (float)(1.0 - (double)hp->beta2);
    s.beta1 = hp->beta1;
    s.beta2 = hp->beta2;
    s.eps = hp->eps;
    s.log_floor = hp->log_floor;
    return s;
}

}  // namespace alq

using namespace alq;

extern "C" {

const char* alq_status_string(int status) {
    switch (status) {
        case ALQ_OK: return "ALQ_OK";
        case ALQ_ERR_INVALID_ARG: return "ALQ_ERR_INVALID_ARG";
        case ALQ_ERR_UNSUPPORTED: return "ALQ_ERR_UNSUPPORTED";
        case ALQ_ERR_ALIGN: return "ALQ_ERR_ALIGN";
        case ALQ_ERR_WORKSPACE: return "ALQ_ERR_WORKSPACE";
        case ALQ_ERR_CUDA: return "ALQ_ERR_CUDA";
        default: return "ALQ_ERR_UNKNOWN";
    }
}

const char* alq_last_cuda_error(void) { return g_last_error; }

const char* al_last_cuda_error(void) { return g_last_error; }

int alq_version(void) { return 100; }

int64_t al_num_blocks(int64_t n, int block) {
    if (n < 0 || block <= 0) return -1;
    return blocks_of(n, block);
}

int64_t al_meta_count(int64_t n, int block) {
    if (n < 0 || block <= 0) return -1;
    return 2 * blocks_of(n, block);
}

int64_t al_state_bytes(int64_t n, int block, int bits) {
    if (n < 0 || block <= 0 || (bits != 8 && bits != 16)) return -1;
    return n * (bits / 8) + 8 * blocks_of(n, block);
}

int al_adamw_plan_bytes(int ntensors, size_t* bytes) {
    if (ntensors <= 0 || !bytes) return ALQ_ERR_INVALID_ARG;
    *bytes = sizeof(PlanHeader) + (size_t)ntensors * sizeof(PlanEntry);
    return ALQ_OK;
}

}  // extern "C"
