/*
 * alq.h -- C ABI of the Adaptive Log-Space (AL) quantized optimizer step for
 * NVIDIA GB300 (sm_103a).
 *
 * Method: "Beyond Dense Adam States: Adaptive Log-Space Quantization for
 * Memory-Efficient Optimizers". Non-negative optimizer states (AdamW second
 * moment, Adafactor row/column factors, CAME confidence factors, APOLLO
 * projected second moment) are stored as AL codes (Sec. 4.1, Eq. (3)-(5)):
 * code 0 is reserved for exact zero (Eq. (6)), codes 1..L-1 are spread
 * uniformly in log2 space over each block's observed positive interval.
 * Signed momentum is stored as uniform 8-bit codes (UF8, Sec. 4.3 and
 * Sec. 5.6). Each optimizer step decodes the states, updates them from the
 * gradient, updates the parameters and re-encodes the states, in fused
 * kernels (Sec. 7.1).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every array pointer is DEVICE-accessible memory owned by the caller,
 *    unless the argument is documented as host memory: device memory, or
 *    pinned host memory through its device mapping (the kernels then read
 *    and write it across the host link; a host-offloaded optimizer can step
 *    its host-resident arrays in place). Plans themselves live in device
 *    memory. The library allocates, frees and
 *    synchronises nothing; work is enqueued on `stream` (a cudaStream_t passed
 *    as void*; NULL is the legacy default stream) and the call returns without
 *    waiting for it.
 *  - Arguments are validated on the host before any launch. A call that
 *    returns a non-zero status launched nothing, except ALQ_ERR_CUDA, which
 *    reports a failed launch (see alq_last_cuda_error()).
 *  - Element counts are int64_t. n == 0 is valid and launches nothing.
 *  - Quantization blocks are consecutive runs of `block` elements of one
 *    tensor; the last block of a tensor may be partial, and elements past the
 *    end never enter a block statistic. `block` must be a power of two in
 *    [128, 4096], the fused AdamW step included. The paper's block
 *    sizes (256 and 2048, Sec. 6.2; 128 for the AL16 factors) are all of
 *    this form. The kernels give each lane whole 4-element chunks of 128
 *    consecutive elements per warp and locate blocks by shifts, so a block
 *    never splits a chunk; other sizes return ALQ_ERR_UNSUPPORTED (the
 *    oracle accepts any size).
 *  - AL metadata is two fp32 values per block, interleaved:
 *    meta[2b] = l_min, meta[2b+1] = Delta (Sec. 4.1, "each block also stores
 *    l_min and Delta"). An all-zero block stores (0, 0) and all-zero codes.
 *  - AL8 codes are uint8_t (L = 256); AL16 codes are uint16_t (L = 65536),
 *    read as unsigned (Sec. 4.4). UF8 codes are int8_t in [-127, 127] with one
 *    fp32 absmax per block.
 *  - A freshly initialised state is all codes 0 and all metadata 0; it decodes
 *    to exact zeros, the same as a zero-initialised fp32 optimizer state.
 *  - Alignment: fp32 arrays and code arrays that are streamed element-wise must
 *    be 16-byte aligned; metadata arrays 8-byte aligned. Misalignment returns
 *    ALQ_ERR_ALIGN.
 *  - Floating-point contract: state EMAs and updates are IEEE fp32 in the
 *    operation order documented per entry point, with a fused multiply-add
 *    (one rounding) exactly where the order writes fma(a, b, c) and no other
 *    contraction; log2/exp2 in the codec are evaluated as if in double and
 *    rounded once to fp32. Within that contract the results are reproducible
 *    run to run (no floating-point atomics).
 *  - Scalar step counters `t` start at 1.
 */
#ifndef ALQ_H_
#define ALQ_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---------------------------------------------------------------- status -- */
#define ALQ_OK 0
#define ALQ_ERR_INVALID_ARG (-1) /* null pointer, bad size, bad hyperparameter */
#define ALQ_ERR_UNSUPPORTED (-2) /* bit width or block size not supported     */
#define ALQ_ERR_ALIGN (-3)       /* pointer not aligned as documented          */
#define ALQ_ERR_WORKSPACE (-4)   /* workspace missing or smaller than required */
#define ALQ_ERR_CUDA (-5)        /* a CUDA runtime call or launch failed       */

/* The same status codes under the AL_ prefix. */
#define AL_OK ALQ_OK
#define AL_ERR_INVALID_ARG ALQ_ERR_INVALID_ARG
#define AL_ERR_UNSUPPORTED ALQ_ERR_UNSUPPORTED
#define AL_ERR_ALIGN ALQ_ERR_ALIGN
#define AL_ERR_WORKSPACE ALQ_ERR_WORKSPACE
#define AL_ERR_CUDA ALQ_ERR_CUDA

/* Human-readable name of a status code (static string). */
const char* alq_status_string(int status);

/* Text of the last CUDA error seen by this library on the calling thread, or
 * "" if none. al_last_cuda_error is the same function under the al_ prefix. */
const char* alq_last_cuda_error(void);
const char* al_last_cuda_error(void);

/* Library ABI version: 100 * major + minor. */
int alq_version(void);

/* Number of quantization blocks of `block` elements covering n elements,
 * ceil(n / block). Host-only; returns -1 for invalid arguments. */
int64_t al_num_blocks(int64_t n, int block);

/* Number of fp32 metadata values of an AL-coded state of n elements: two
 * (l_min, Delta) per block, 2 * ceil(n / block). Host-only; returns -1 for
 * invalid arguments. */
int64_t al_meta_count(int64_t n, int block);

/* Logical storage of one AL-coded state of n elements in bytes: codes plus
 * 8 bytes of metadata per block (Sec. 4.4, Eq. (7): c_AL8 = 1 + 8/B bytes per
 * element, c_AL16 = 2 + 8/B). Host-only; returns -1 for invalid arguments. */
int64_t al_state_bytes(int64_t n, int block, int bits);

/* ------------------------------------------------------------ AL codec -- */
/*
 * al_encode -- Sec. 4.1, Eq. (3)-(4), degenerate handling in the last
 * paragraph of Sec. 4.1.
 *   x         [n] fp32, non-negative, finite (negative values are outside the
 *             contract and are not checked; -0.0 counts as zero).
 *   block     elements per block (power of two, 128..4096).
 *   bits      8 (AL8, L = 256, codes uint8_t) or 16 (AL16, L = 65536,
 *             codes uint16_t).
 *   log_floor l_floor of Eq. (3), the lower bound of l_min.
 *   codes     [n] output codes.
 *   meta      [2 * ceil(n/block)] output (l_min, Delta) per block.
 * Per block: mn = min{x > 0}, mx = max x; l_min = max(l_floor, log2 mn),
 * l_max = min(log2 mx, 126); if l_max <= l_min then l_max = l_min + 1;
 * Delta = max(l_max - l_min, 1e-12). q = 0 for x == 0, otherwise
 * q = 1 + rint((L - 2) * clip((log2 x - l_min) / Delta, 0, 1)), ties to even.
 */
int al_encode(const float* x, int64_t n, int block, int bits, float log_floor,
              void* codes, float* meta, void* stream);

/*
 * al_decode -- Sec. 4.1, Eq. (5).
 *   codes [n] uint8_t (bits = 8) or uint16_t (bits = 16); meta [2*nblocks].
 *   out   [n] fp32: 0 for q == 0, otherwise 2^(l_min + (q-1) * Delta / (L-2))
 *         rounded once to fp32.
 */
int al_decode(const void* codes, const float* meta, int64_t n, int block,
              int bits, float* out, void* stream);

/* ----------------------------------------------------------- UF8 codec -- */
/*
 * uf8_encode -- uniform signed 8-bit momentum code (Sec. 4.3; momentum block
 * size 256 in Sec. 6.2). Per block: s = max |m|. If s == 0 every code is 0
 * and absmax = 0. Otherwise q = rint(m * (127 / s)) in fp32, ties to even;
 * |q| <= 127 and q never has the opposite sign of m. When s < 2^-120 both m
 * and s are first multiplied by 2^64 (exact), so that 127 / s stays finite.
 *   m      [n] fp32 (finite).
 *   codes  [n] int8_t output.
 *   absmax [ceil(n/block)] fp32 output.
 */
int uf8_encode(const float* m, int64_t n, int block, int8_t* codes,
               float* absmax, void* stream);

/* uf8_decode -- m_hat = (float)q * (s / 127), with s / 127 rounded to fp32
 * once per block. */
int uf8_decode(const int8_t* codes, const float* absmax, int64_t n, int block,
               float* out, void* stream);

/* ----------------------------------------------------------------- AdamW -- */
/* Hyperparameters (host struct). */
typedef struct {
    float lr;           /* learning rate                                   */
    float beta1;        /* first-moment EMA rate                           */
    float beta2;        /* second-moment EMA rate                          */
    float eps;          /* added to the bias-corrected sqrt(V)             */
    float weight_decay; /* decoupled weight decay                          */
    float log_floor;    /* l_floor for V (the paper uses log2 of eps^2)    */
} al_adamw_hp;

/*
 * al_adamw_step -- one AdamW step with UF8 momentum M and AL-coded second
 * moment V (Sec. 3.1, Eq. (1); Sec. 6.2 "AL8 second moments with UF8
 * momentum"; fused as in Sec. 7.1). In place:
 *   p        [n] fp32 parameters (read and written).
 *   g        [n] fp32 gradient.
 *   m_codes  [n] int8 UF8 codes, m_absmax [ceil(n/m_block)] fp32.
 *   m_block, v_block  block sizes, powers of two in [128, 4096].
 *   v_codes  [n] uint8 (v_bits = 8) or uint16 (v_bits = 16) AL codes,
 *   v_meta   [2*ceil(n/v_block)] fp32.
 *   v_bits = 32 is the unquantized FP32 role (Sec. 4.5, "AL8, AL16, or
 *            FP32 according to state sensitivity"): m_codes and v_codes
 *            then point to dense fp32 m and v [n], m_absmax, v_meta,
 *            m_block and v_block are unused (m_absmax and v_meta may be
 *            NULL), and the step is the same arithmetic without the codec.
 *   hp       host pointer; t >= 1.
 * Scalars computed on the host in double and rounded to fp32 once:
 *   decay = 1 - lr*wd, step = lr / (1 - beta1^t), c2 = 1 / sqrt(1 - beta2^t),
 *   omb1 = 1 - beta1, omb2 = 1 - beta2.
 * Per element, in fp32, in this order (fma: one rounding):
 *   p1 = p*decay;  m = fma(beta1, m_hat, omb1*g);
 *   v = fma(beta2, v_hat, omb2*(g*g));  den = fma(sqrt(v), c2, eps);
 *   p = fma(-step, m/den, p1);
 * then m is UF8-encoded (m_block) and v is AL-encoded (v_block, log_floor).
 * The parameter update uses the fresh fp32 m and v, not their re-decoded
 * values. m, v, their codes and block constants are exact in this order.
 * With v_bits 8 or 16, sqrt(v) and the division m/den are the hardware's
 * approximations (a few ulp), so p differs from the IEEE result by a few ulp
 * of step*|m/den|; with v_bits 32 they are IEEE and p is exact too.
 */
int al_adamw_step(float* p, const float* g, int8_t* m_codes, float* m_absmax,
                  void* v_codes, float* v_meta, int64_t n, int m_block,
                  int v_block, int v_bits, const al_adamw_hp* hp, int64_t t,
                  void* stream);

/* One tensor of a multi-tensor AdamW step; pointers as in al_adamw_step. */
typedef struct {
    float* p;
    const float* g;
    int8_t* m_codes;
    float* m_absmax;
    void* v_codes;
    float* v_meta;
    int64_t n;
} al_adamw_tensor;

/* Summary of a multi-tensor plan (host struct, filled by al_adamw_plan). */
typedef struct {
    int32_t ntensors;
    int32_t m_block;
    int32_t v_block;
    int32_t v_bits;
    int64_t total_tiles; /* 4096-element tiles of the fused kernel  */
    int64_t total_elems; /* sum of n over the tensors               */
} al_multi_info;

/* Size in bytes of the plan buffer for `ntensors` tensors. */
int al_adamw_plan_bytes(int ntensors, size_t* bytes);

/*
 * al_adamw_plan -- build, in HOST memory `plan_host` (plan_bytes long), the
 * table that al_adamw_step_multi reads. The caller copies it once to device
 * memory (any 16-byte aligned buffer of the same size) and reuses it for
 * every step while the tensors' pointers and sizes stay the same. Blocks
 * never cross tensor boundaries (Sec. 4.4, "ignoring tensor-boundary
 * padding"). Every tensor is validated as in al_adamw_step.
 */
int al_adamw_plan(const al_adamw_tensor* tensors, int ntensors, int m_block,
                  int v_block, int v_bits, void* plan_host, size_t plan_bytes,
                  al_multi_info* info);

/* al_adamw_step_multi -- one fused launch of al_adamw_step over every tensor
 * of a plan. `plan_dev` is the device copy of the plan; `info` the host
 * summary returned by al_adamw_plan. */
int al_adamw_step_multi(const void* plan_dev, const al_multi_info* info,
                        const al_adamw_hp* hp, int64_t t, void* stream);

/* ------------------------------------------------------------- workspace -- */
#define AL_OP_ADAFACTOR 1
#define AL_OP_CAME 2
#define AL_OP_APOLLO 3

/* Steps of independent matrices may run concurrently on different streams,
 * each call with its own workspace; for many small matrices this overlaps
 * one matrix's short passes with another's streaming passes.
 *
 * Scratch bytes that al_adafactor_step / al_came_step / al_apollo_step need
 * for a rows x cols matrix (rank is used by APOLLO only). Host-only. */
int al_workspace_size(int op, int64_t rows, int64_t cols, int rank,
                      size_t* bytes);

/* ------------------------------------------------------------- Adafactor -- */
typedef struct {
    float lr;           /* learning rate                                     */
    float eps1;         /* added to g^2 in the factored statistics (> 0)     */
    float clip_d;       /* update clipping threshold d (> 0)                 */
    float decay_rate;   /* rho_t = 1 - t^decay_rate, e.g. -0.8               */
    float beta1;        /* momentum EMA rate, used when m_codes != NULL      */
    float weight_decay; /* decoupled weight decay                            */
    float log_floor;    /* l_floor of the factor codes (typically log2 eps1) */
} al_adafactor_hp;

/*
 * al_adafactor_step -- Adafactor with a factored second moment (Sec. 3.1,
 * "row and column statistics"; lr 1e-3 in Sec. 6.1) whose row factor R [rows]
 * and column factor C [cols] are AL-coded (fac_bits 8 or 16, fac_block), and
 * optional UF8 momentum. p and g are row-major [rows x cols] fp32.
 * fac_bits = 32 keeps the factors unquantized (Sec. 4.5's FP32 role):
 * r_codes and c_codes then point to fp32 factors, r_meta and c_meta are
 * unused (may be NULL). The same holds for v_bits and c_bits of
 * al_came_step (c_bits = 32 with AL-coded V is the paper's "FP32 C" CAME).
 *   r_i = mean_j(g_ij^2 + eps1), c_j = mean_i(g_ij^2 + eps1)  (exact sums,
 *         rounded once to fp32);
 *   R = rho*R_hat + (1-rho)*r,  C = rho*C_hat + (1-rho)*c;
 *   a_i = 1/sqrt(R_i/mean(R)), b_j = 1/sqrt(C_j);  u_ij = (g_ij*a_i)*b_j;
 *   u_hat = u * (1/max(1, RMS(u)/d));  optional M = beta1*M_hat+(1-beta1)*u_hat;
 *   p = p*(1 - lr*wd) - lr*(M or u_hat).
 * Momentum is disabled by m_codes == NULL (then m_absmax and m_block are
 * ignored). workspace: al_workspace_size(AL_OP_ADAFACTOR, ...) bytes of device
 * memory, contents need not be initialised.
 */
int al_adafactor_step(float* p, const float* g, int64_t rows, int64_t cols,
                      void* r_codes, float* r_meta, void* c_codes,
                      float* c_meta, int fac_bits, int fac_block,
                      int8_t* m_codes, float* m_absmax, int m_block,
                      const al_adafactor_hp* hp, int64_t t, void* workspace,
                      size_t ws_bytes, void* stream);

/*
 * al_adafactor_step_noalloc -- al_adafactor_step for callers that cannot
 * allocate GPU memory (no counterpart in the paper; an interface addition).
 * Some callers cannot call cudaMalloc when they step the optimizer: code
 * running under a framework that owns all device memory, code with a fixed
 * memory budget after start-up, or bindings without access to the CUDA
 * allocator. This variant takes the step's scratch space from a fixed array
 * inside the library (al_adafactor_noalloc_capacity() bytes, 4 MiB, enough
 * for matrices up to 4096 x 4096) and allocates nothing; arguments and
 * results are exactly those of al_adafactor_step without the workspace.
 *   - Every GPU that loads the library reserves that array until the process
 *     exits.
 *   - Every call looks up the array's device address (cudaGetSymbolAddress,
 *     with the calling thread's current device and context), so the address
 *     stays valid after cudaDeviceReset or under another context on the same
 *     device. The first call on a device may load the library's device code:
 *     make that first call before capturing any stream.
 *   - Every call on a device shares the one array: calls that may run
 *     concurrently on the GPU (different streams, no ordering between them)
 *     race and corrupt each other's results. Serialise them on one stream.
 *     The array keeps the previous call's contents; every scratch word a call
 *     reads it has written first in the same call, so nothing needs clearing.
 *   - Returns ALQ_ERR_WORKSPACE when the matrix needs more scratch than the
 *     array holds (see al_workspace_size(AL_OP_ADAFACTOR, ...)), and every
 *     status of al_adafactor_step otherwise.
 */
int al_adafactor_step_noalloc(float* p, const float* g, int64_t rows,
                              int64_t cols, void* r_codes, float* r_meta,
                              void* c_codes, float* c_meta, int fac_bits,
                              int fac_block, int8_t* m_codes, float* m_absmax,
                              int m_block, const al_adafactor_hp* hp,
                              int64_t t, void* stream);

/* Bytes of the fixed scratch array that al_adafactor_step_noalloc uses. */
size_t al_adafactor_noalloc_capacity(void);

/* ------------------------------------------------------------------ CAME -- */
typedef struct {
    float lr;
    float beta1;        /* momentum EMA rate                               */
    float beta2;        /* factored second-moment EMA rate                 */
    float beta3;        /* factored confidence EMA rate (0.9999, Sec. 6.1) */
    float eps1;         /* added to g^2 (> 0)                              */
    float eps2;         /* added to the residual (> 0)                     */
    float clip_d;       /* update clipping threshold d (> 0)               */
    float weight_decay;
    float log_floor_v;  /* l_floor of the second-moment factor codes       */
    float log_floor_c;  /* l_floor of the confidence factor codes          */
} al_came_hp;

/*
 * al_came_step -- CAME (Sec. 3.1: dense momentum M, factored second moment
 * V^(r), V^(c), factored confidence C^(r), C^(c); beta3 = 0.9999 in Sec. 6.1)
 * with AL-coded factors and UF8 momentum (Sec. 6.2, "AL16 for both V and C").
 *   u and u_hat as in al_adafactor_step but with a constant beta2 EMA;
 *   M = beta1*M_hat + (1-beta1)*u_hat;
 *   U_ij = (u_hat_ij - M_ij)^2 + eps2;  Cr/Cc = beta3-EMA of the row/column
 *   means of U;  S_ij = Cr_i*Cc_j/mean(Cr);
 *   p = p*(1 - lr*wd) - lr * M/sqrt(S)  (as (M*ar_i)*bc_j with
 *   ar_i = 1/sqrt(Cr_i/mean(Cr)), bc_j = 1/sqrt(Cc_j)).
 * The momentum codes are required (m_codes != NULL).
 */
int al_came_step(float* p, const float* g, int64_t rows, int64_t cols,
                 void* vr_codes, float* vr_meta, void* vc_codes,
                 float* vc_meta, int v_bits, int v_block, void* cr_codes,
                 float* cr_meta, void* cc_codes, float* cc_meta, int c_bits,
                 int c_block, int8_t* m_codes, float* m_absmax, int m_block,
                 const al_came_hp* hp, int64_t t, void* workspace,
                 size_t ws_bytes, void* stream);

/* --------------------------------------------- grouped Adafactor / CAME -- */
/*
 * One Adafactor or CAME step over many matrices with one launch per pass
 * (Adafactor: g^2 sums, factors, scales, RMS, update = 5 launches; CAME adds
 * the residual sums, the confidence factors and their scales = 8 launches)
 * instead of those launches per matrix. Every pass works in tiles that never
 * cross a matrix, with the per-tile code of al_adafactor_step / al_came_step,
 * so each matrix's results are bit-identical to the per-matrix call. The
 * grouping is the library's; the paper steps matrix by matrix.
 *
 * Usage: al_factored_workspace_multi -> allocate the workspace (256-byte
 * aligned); al_factored_plan_bytes -> allocate a host buffer and a device
 * buffer (64-byte aligned) of that size; al_factored_plan fills the host
 * buffer; copy it to the device buffer once; then call
 * al_adafactor_step_multi or al_came_step_multi every step. The plan records
 * the matrices' pointers and the workspace: rebuild it if any of them
 * changes.
 */
typedef struct {
    float* p;             /* [rows x cols] fp32, row-major                   */
    const float* g;
    int64_t rows, cols;   /* cols % 4 == 0, rows * cols < 2^31               */
    void* vr_codes;       /* second-moment row factor [rows] (Adafactor R)   */
    float* vr_meta;
    void* vc_codes;       /* second-moment column factor [cols] (C)          */
    float* vc_meta;
    void* cr_codes;       /* CAME confidence row factor [rows]; NULL for      */
    float* cr_meta;       /* Adafactor                                       */
    void* cc_codes;       /* CAME confidence column factor [cols]            */
    float* cc_meta;
    int8_t* m_codes;      /* UF8 momentum [rows x cols]; NULL for Adafactor  */
    float* m_absmax;      /* without momentum (then for every matrix)        */
} al_factored_matrix;

/* Summary of a grouped factored plan (host struct, filled by
 * al_factored_plan). */
typedef struct {
    int32_t nmat;
    int32_t op;           /* AL_OP_ADAFACTOR or AL_OP_CAME                   */
    int32_t v_bits, v_block, c_bits, c_block, m_block;
    int32_t has_momentum;
    int64_t total_params;
    int64_t sumsq_tiles;  /* 64 x 256 tiles of the sums passes               */
    int64_t factor_tiles; /* factor blocks (rows and columns) of V           */
    int64_t factor2_tiles;/* factor blocks of CAME's confidence (else 0)     */
    int64_t scale_tiles;  /* 256-entry tiles of the scale passes             */
    int64_t tiles;        /* 4096-parameter tiles of the update              */
    int64_t rms_chunks;   /* 8-tile chunks of the RMS pass (one partial each) */
    void* workspace;      /* the workspace the plan is bound to              */
} al_factored_info;

/* Bytes of a plan over these matrices (host and device copies alike). */
int al_factored_plan_bytes(const al_factored_matrix* mats, int nmat, size_t* bytes);

/* Scratch bytes of a grouped step: every matrix's al_workspace_size
 * scratch side by side. */
int al_factored_workspace_multi(const al_factored_matrix* mats, int nmat, size_t* bytes);

/* Validates every matrix as al_adafactor_step (op AL_OP_ADAFACTOR: v_bits
 * and v_block are fac_bits and fac_block, c_* ignored) or al_came_step (op
 * AL_OP_CAME) does, with one set of bit widths and block sizes for all, and
 * writes the plan into plan_host. Momentum must be present in every matrix
 * or in none (CAME: in every matrix). Returns ALQ_ERR_WORKSPACE when the
 * workspace is missing, misaligned or too small. */
int al_factored_plan(int op, const al_factored_matrix* mats, int nmat, int v_bits,
                     int v_block, int c_bits, int c_block, int m_block, void* workspace,
                     size_t ws_bytes, void* plan_host, size_t plan_bytes,
                     al_factored_info* info);

/* One grouped step. plan_dev is the device copy of the plan; info and hp are
 * host pointers; the plan's op must match the call. */
int al_adafactor_step_multi(const void* plan_dev, const al_factored_info* info,
                            const al_adafactor_hp* hp, int64_t t, void* stream);
int al_came_step_multi(const void* plan_dev, const al_factored_info* info,
                       const al_came_hp* hp, int64_t t, void* stream);

/* ---------------------------------------------------------------- APOLLO -- */
typedef struct {
    float lr;
    float beta1, beta2; /* projected-moment EMA rates                         */
    float eps;          /* added to the bias-corrected sqrt(V^P)              */
    float alpha;        /* scale applied to the channel-scaled gradient       */
    float weight_decay;
    float norm_growth_gamma; /* norm-growth limit; <= 0 disables the limiter */
    float log_floor;    /* l_floor of the V^P codes                           */
    int32_t rank;       /* projection rank r (256 in Sec. 6.1)                */
} al_apollo_hp;

/*
 * al_apollo_step -- APOLLO with channel-wise scaling (Sec. 3.1, "moments in a
 * low-rank gradient space ... scale applied to the original gradient"; rank
 * 256, channel-wise, projection gap 200 in Sec. 6.1), with UF8 M^P and
 * AL-coded V^P.
 *   p, g      row-major [rows x cols] fp32.
 *   proj      bf16 bit patterns [rank x s], s = min(rows, cols), row-major:
 *             the random projection of the short side. The caller draws and
 *             refreshes it; the projected moments are kept across refreshes.
 *   m_codes/m_absmax, v_codes/v_meta: projected moments, channel-major
 *             [c x rank] with c = max(rows, cols) channels; blocks run along
 *             that flattened array.
 *   prev_norm device fp32 scalar, the limiter's previous update norm; 0 at
 *             the first step. Read and written only when the limiter is on.
 * R = P * bf16(G) over the short side (fp32 accumulation on tensor cores);
 * M = beta1*M_hat + (1-beta1)*R;  V = beta2*V_hat + (1-beta2)*R*R;
 * Rt = (M*(1/(1-beta1^t))) / (sqrt(V)*(1/sqrt(1-beta2^t)) + eps);
 * s_j = ||Rt_j|| / (||R_j|| + 1e-8) per channel j;  Gt = G scaled by s_j;
 * optional limiter Gt *= min(1, gamma*prev_norm/||Gt||) when prev_norm > 0;
 * p = p*(1 - lr*wd) - (lr*alpha)*Gt.
 */
int al_apollo_step(float* p, const float* g, int64_t rows, int64_t cols,
                   const uint16_t* proj, int8_t* m_codes, float* m_absmax,
                   int m_block, void* v_codes, float* v_meta, int v_bits,
                   int v_block, float* prev_norm, const al_apollo_hp* hp,
                   int64_t t, void* workspace, size_t ws_bytes, void* stream);

/* ---------------------------------------------------- grouped APOLLO step -- */
/*
 * One APOLLO step over many matrices in three launches (one persistent
 * projection launch whose CTAs walk every matrix's 128-channel tiles, one
 * moments launch, one update launch) instead of three launches per matrix. Each matrix gets exactly the arithmetic of al_apollo_step (the
 * results are bit-identical). This grouping is the library's; the paper
 * applies the method matrix by matrix.
 *
 * Usage: al_apollo_workspace_multi -> allocate the workspace (256-byte
 * aligned); al_apollo_plan_bytes -> allocate a host buffer and a device
 * buffer (64-byte aligned) of that size; al_apollo_plan fills the host
 * buffer; copy it to the device buffer once; then call al_apollo_step_multi
 * every step. The plan records the matrices' pointers, the workspace and the
 * TMA descriptors of the projections: rebuild it if any of them
 * changes (a refreshed projection written into the same proj buffer needs no
 * rebuild). The norm-growth limiter (hp->norm_growth_gamma > 0) limits
 * every matrix by its own previous norm (prev_norm, one device scalar per
 * matrix, as in al_apollo_step); it returns ALQ_ERR_INVALID_ARG when a
 * matrix of the plan has no prev_norm. Each matrix's results, limiter
 * included, are bit for bit those of al_apollo_step.
 */
typedef struct {
    float* p;              /* [rows x cols] fp32, as in al_apollo_step      */
    const float* g;
    int64_t rows, cols;
    const uint16_t* proj;  /* bf16 bits [rank x min(rows, cols)]            */
    int8_t* m_codes;       /* [max(rows, cols) x rank] UF8, block = rank    */
    float* m_absmax;
    void* v_codes;         /* [max(rows, cols) x rank] AL8 or AL16          */
    float* v_meta;
    float* prev_norm;      /* device scalar, the limiter's previous norm
                              (nullable when the limiter is never used)     */
} al_apollo_matrix;

/* Summary of a grouped plan (host struct, filled by al_apollo_plan). */
typedef struct {
    int32_t nmat, rank, v_bits;
    int32_t limiter_ok;     /* 1 when every matrix has a prev_norm           */
    int64_t total_params;   /* sum of rows * cols                            */
    int64_t total_channels; /* sum of max(rows, cols)                        */
    int64_t gemm_tiles;     /* 128-channel tiles of the grouped projection   */
    int64_t mom_tiles;      /* 4096-value tiles of the moments pass          */
    int64_t upd_tiles;      /* 4096-parameter tiles of the update pass       */
    void* workspace;        /* the workspace the plan is bound to            */
    int64_t norm_chunks;    /* limiter partial sums (8 update tiles each)    */
} al_apollo_info;

/* Bytes of a plan over these matrices (host and device copies alike). */
int al_apollo_plan_bytes(const al_apollo_matrix* mats, int nmat, size_t* bytes);

/* Scratch bytes of a grouped step: every matrix's projection R and channel
 * scales side by side. */
int al_apollo_workspace_multi(const al_apollo_matrix* mats, int nmat, int rank,
                              size_t* bytes);

/* Validates every matrix as al_apollo_step does (rank 128 or 256, v_bits 8
 * or 16) and writes the plan into plan_host. Returns ALQ_ERR_WORKSPACE when
 * the workspace is missing, misaligned or too small, ALQ_ERR_CUDA when a TMA
 * descriptor cannot be encoded. */
int al_apollo_plan(const al_apollo_matrix* mats, int nmat, int rank,
                   int v_bits, void* workspace, size_t ws_bytes,
                   void* plan_host, size_t plan_bytes, al_apollo_info* info);

/* One grouped step. plan_dev is the device copy of the plan; info and hp
 * are host pointers; hp->rank must equal the plan's rank. */
int al_apollo_step_multi(const void* plan_dev, const al_apollo_info* info,
                         const al_apollo_hp* hp, int64_t t, void* stream);

#ifdef __cplusplus
} /* extern "C" */
#endif

#endif /* ALQ_H_ */
