// alq_internal.h -- definitions shared by the library's translation units:
// the tile geometry of the element-wise kernels, the multi-tensor plan
// layout, argument validation and error reporting.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/alq.h"

namespace alq {

// Element-wise kernels process tiles of kTile elements with 256 threads:
// warp w owns the 512-element segment [512 w, 512 w + 512) of the tile and
// lane l owns, for chunk c = 0..3, the four consecutive elements at
// 128 c + 4 l of the segment. A quantization block of B >= 128 elements thus
// spans whole chunks of every lane of a warp (B <= 512) or whole segments
// of B / 512 warps (B >= 512).
constexpr int kThreads = 256;
constexpr int kTile = 4096;
constexpr int kSeg = 512;

// ------------------------------------------------------ multi-tensor plan --
constexpr uint32_t kPlanMagic = 0x414C5131u;  // "ALQ1"

struct PlanHeader {
    uint32_t magic;
    int32_t ntensors;
    int32_t m_block;
    int32_t v_block;
    int32_t v_bits;
    int32_t tile;
    int64_t total_tiles;
    int64_t total_elems;
    int64_t reserved[3];
};
static_assert(sizeof(PlanHeader) == 64, "plan header is 64 bytes");

struct PlanEntry {
    float* p;
    const float* g;
    int8_t* m_codes;
    float* m_absmax;
    void* v_codes;
    float* v_meta;
    int64_t n;
    int64_t first_tile;
};
static_assert(sizeof(PlanEntry) == 64, "plan entry is 64 bytes");

// AdamW scalars, computed on the host in double and rounded once.
struct AdamWScalars {
    float decay, step, c2, omb1, omb2, beta1, beta2, eps, log_floor;
};

AdamWScalars adamw_scalars(const al_adamw_hp* hp, int64_t t);

// -------------------------------------------------------------- checking --
bool valid_block(int block);  // power of two in [128, 4096]
bool aligned(const void* p, size_t a);
int record_cuda(cudaError_t e);       // ALQ_OK or ALQ_ERR_CUDA (and records text)
int check_launch();                   // cudaGetLastError -> status
int sm_count();                       // multiprocessors of the current device
// Persistent-grid size: min(ntiles, SMs x resident CTAs of `kernel`), the
// residency queried once per kernel and device (which also opts the kernel
// in to `smem` bytes of dynamic shared memory; every launch of a kernel must
// pass the same `smem`).
int persistent_grid(const void* kernel, int threads, size_t smem, int64_t ntiles);
int64_t blocks_of(int64_t n, int block);

// APOLLO workspace bytes (alq_apollo.cu).
int al_apollo_workspace(int64_t rows, int64_t cols, int rank, size_t* bytes);

}  // namespace alq
