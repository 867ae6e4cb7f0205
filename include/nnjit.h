/*
 * nnjit.h -- C ABI of a JIT-tuned dense MatMul / BatchMatMul library for one NVIDIA
 * GB300 (sm_103a).
 *
 * The operator is the one every kernel experiment of nnJIT (arXiv 2309.08978) tunes:
 * MatMul (Sec. 2.2; Table 3, K0/K1) and BatchMatMul (Table 3, K2/K3):
 *
 *     C[b,i,j] = sum_k A[b,i,k] * Bt[b,k,j] (+ bias[j]),   Bt = B or B^T (see nnjit_blayout)
 *
 * The library keeps the paper's JIT scheme (Sec. 3): for each (kernel type, shape, device)
 * it builds a small "lite" space of kernel configurations pruned by tile-based hardware
 * usage formulas (Sec. 5.2, Table 1), times the candidates on the device, keeps the
 * fastest, and caches it under a key made of the kernel type, shape and device (Sec. 5.3).
 *
 * Conventions for every function below:
 *   - Every call returns an nnjit_status; no C++ exception crosses this boundary.  On
 *     failure nnjit_last_error() returns a thread-local, human-readable detail string.
 *   - Device pointers are plain CUDA device addresses (e.g. from cudaMalloc or a PyTorch
 *     tensor's data_ptr()) on the device that was current when the plan was made; the
 *     caller owns them.  `stream` is a cudaStream_t passed as void* (NULL = legacy
 *     default stream).
 *   - All sizes, leading dimensions and batch strides are in ELEMENTS, not bytes.
 *   - Matrices are row-major.  A is [batch][M][K] (row i at A + b*stride_a + i*lda).
 *     C is [batch][M][N] float32 (row i at C + b*stride_c + i*ldc).
 *   - Operand element types: NNJIT_F32_FFMA and NNJIT_TF32 take float32 A and B;
 *     NNJIT_BF16 takes bfloat16 A and B (16-bit patterns).  bias and C are always float32;
 *     accumulation is always float32.
 */
#ifndef NNJIT_H
#define NNJIT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
typedef enum {
    NNJIT_OK = 0,
    NNJIT_ERR_INVALID_ARG = 1,   /* bad shape (<0), NULL operand, unknown enum, bad stride */
    NNJIT_ERR_UNSUPPORTED = 2,   /* legal request this library does not serve, e.g. a
                                    tensor-core path whose row stride or pointer is not
                                    16-byte aligned */
    NNJIT_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed (detail in last_error) */
    NNJIT_ERR_OOM = 4,           /* device or host allocation failed */
    NNJIT_ERR_TIMEOUT = 5,       /* a kernel's bounded wait expired and it stopped early
                                    (device watchdog word set); results are invalid */
    NNJIT_ERR_BUDGET = 6         /* tuning budget too small to evaluate any candidate;
                                    only returned when NNJIT_PLAN_REQUIRE_TIMED is set */
} nnjit_status;

/* Arithmetic path.  C and bias are float32 for all three. */
typedef enum {
    NNJIT_F32_FFMA = 0,  /* float32 operands, exact float32 fused multiply-add (SIMT) */
    NNJIT_TF32 = 1,      /* float32 operands consumed as TF32 by the tensor cores
                            (tcgen05 .kind::tf32), float32 accumulation */
    NNJIT_BF16 = 2,      /* bfloat16 operands, float32 accumulation (tcgen05 .kind::f16,
                            or the split-K GEMV when M <= 8) */
    NNJIT_W4_BF16 = 3    /* bfloat16 A, 4-bit weights B with bfloat16 group scales (the
                            "4-bit quantization" of the paper's Llama 2 result, Sec. 7:
                            decode, M <= 8, B as [N][K] only); float32 accumulation.  B
                            points to a weight blob laid out as described below. */
} nnjit_dtype;

/*
 * 4-bit weight blob (NNJIT_W4_BF16).  Weight w[n][k] = (q[n][k] - 8) * s[k / 128][n]:
 *   - q are unsigned 4-bit codes, two per byte, row n at byte n * ldb / 2, code k in byte
 *     k / 2, the low nibble holding the even k.  ldb (in codes) >= K and a multiple of 32
 *     (16-byte rows).
 *   - s are bfloat16 scales, one per row and group of 128 consecutive k, stored
 *     group-major: s[g][n] at element g * N + n of the scale block, which starts at byte
 *     nnjit_w4_layout()'s scale_offset (the code block rounded up to 256 bytes).  N must be
 *     a multiple of 8.
 * The blob is read-only for the library; like any B it is owned by the caller.
 */
nnjit_status nnjit_w4_layout(int64_t N, int64_t K, int64_t ldb, int64_t* scale_offset_bytes,
                             int64_t* total_bytes);

/* Storage of B. */
typedef enum {
    NNJIT_B_KN = 0,      /* B is [K][N] row-major (ldb >= N): Bt = B */
    NNJIT_B_NK = 1       /* B is [N][K] row-major (ldb >= K): Bt = B^T.  This is the
                            PyTorch Linear weight layout and K^T of attention QK^T. */
} nnjit_blayout;

/*
 * Elementwise activation applied to every output after the bias, inside the kernel that
 * writes C (the epilogue fusion of a Linear with its activation; in split-K plans the
 * reduction applies it once the slices are summed):  C = act(A * Bt + bias).
 * Or-ed with NNJIT_EPI_RESIDUAL, the kernel that writes C also adds the value C held
 * before the call (a residual connection; C must then be initialised by the caller):
 *   C = act(A * Bt + bias) + C.
 * Partial sums of split-K plans go to the plan's workspace; C is read and written once.
 */
typedef enum {
    NNJIT_EPI_NONE = 0,
    NNJIT_EPI_RELU = 1,  /* max(x, 0) */
    NNJIT_EPI_GELU = 2,  /* x * Phi(x) = 0.5 x (1 + erf(x / sqrt(2)))  (exact, erf form) */
    NNJIT_EPI_SILU = 3,  /* x * sigmoid(x) = x / (1 + exp(-x)) */
    NNJIT_EPI_RESIDUAL = 0x10
} nnjit_epilogue;

/* Kernel families of the lite space. */
typedef enum {
    NNJIT_FAMILY_FFMA = 0,  /* register-tiled SIMT GEMM, exact FP32 */
    NNJIT_FAMILY_TC = 1,    /* TMA + tcgen05/TMEM tensor-core GEMM, persistent */
    NNJIT_FAMILY_GEMV = 2   /* streaming split-K GEMV for M <= 8 (BF16 weights) */
} nnjit_family;

/* Plan descriptor flags. */
#define NNJIT_PLAN_NO_CACHE      0x1u  /* neither read nor write the process plan cache */
#define NNJIT_PLAN_EXHAUSTIVE    0x2u  /* time every candidate, ignoring the budget */
#define NNJIT_PLAN_REQUIRE_TIMED 0x4u  /* fail with NNJIT_ERR_BUDGET instead of taking the
                                          top-ranked candidate untimed */
#define NNJIT_PLAN_B_CONSTANT    0x8u  /* promise: B (e.g. Linear weights) is never written by
                                          a kernel launched earlier in the same stream, so the
                                          kernels may start reading B while that kernel still
                                          runs (programmatic dependent launch); A and bias are
                                          read only after it has completed */

/*
 * Full problem description.  Zero leading dimensions / strides mean "packed":
 * lda = K, ldb = (B_KN ? N : K), ldc = N, stride_a = M*lda, stride_b = (B_KN ? K : N)*ldb,
 * stride_c = M*ldc.  batch >= 1.  M, N, K >= 0 (an empty M or N is a no-op; K = 0 gives
 * C = bias, or 0 without bias).
 */
typedef struct {
    int64_t M, N, K;
    int64_t batch;
    int32_t dtype;        /* nnjit_dtype */
    int32_t b_layout;     /* nnjit_blayout */
    int64_t lda, ldb, ldc;
    int64_t stride_a, stride_b, stride_c;
    int32_t has_bias;     /* 1: run() takes a float32 bias[N] added to every row */
    uint32_t flags;       /* NNJIT_PLAN_* */
    int32_t epilogue;     /* nnjit_epilogue, applied after the bias (0 = none) */
} nnjit_matmul_desc;

/*
 * Device resources the lite space is built against (the "hardware constraints" that
 * the formulas of Table 1 take: registers, L1/shared memory and warps per core), plus
 * the Blackwell-specific tensor-memory column count.
 */
typedef struct {
    int32_t sm_count;
    int32_t smem_per_sm;           /* bytes of shared memory per SM */
    int32_t smem_per_block_optin;  /* bytes a CTA may opt in to */
    int32_t regs_per_sm;
    int32_t max_threads_per_sm;
    int32_t max_blocks_per_sm;
    int32_t tmem_cols_per_sm;      /* tensor-memory columns per SM (512 on sm_10x) */
    int32_t l2_bytes;
    int32_t cc_major, cc_minor;
} nnjit_device_limits;

/*
 * One candidate of the lite space (the "sequence of primitives and configurations"
 * of Sec. 2.2; tile symbols follow Table 1: x1, y1, r1 = bm, bn, bk; x0, y0 = tm, tn).
 */
typedef struct {
    int32_t family;          /* nnjit_family */
    int32_t bm, bn, bk;      /* CTA tile (TC: bm = 256 is a tile of a CTA pair; bk = K elements
                                per ring slot, 2 k-blocks of 128 bytes when it is 256 bytes;
                                GEMV: bm = M, bn = weight rows per CTA or stage, bk = K slice
                                or K elements per ring stage) */
    int32_t tm, tn;          /* FFMA: thread tile; GEMV: tm = rows per warp */
    int32_t stages;          /* TC: shared-memory ring depth; GEMV: loads in flight per row,
                                or ring stages of the TMA-fed kernels (instance >= 8) */
    int32_t split_k;         /* K slices reduced in a fixed order afterwards (1 = none) */
    int32_t raster;          /* TC tile order: 0 = M fastest, 1 = N fastest */
    int32_t threads;         /* threads per CTA */
    int32_t smem_bytes;      /* shared memory per CTA */
    int32_t tmem_cols;       /* TMEM columns per CTA (TC only) */
    int32_t regs_per_thread; /* register figure used by the usage model */
    int32_t blocks_per_sm;   /* Block_core of Table 1 */
    int32_t grid;            /* CTAs per launch of the main kernel */
    int32_t wave_eff_ppm;    /* predicted wave efficiency, parts per million */
    int32_t instance;        /* index of the precompiled kernel instance */
    int64_t predicted_cost;  /* model cost used for ordering (arbitrary units, lower first) */
    int32_t reduce;          /* split-K reduction: 0 = partials in the plan's workspace, summed
                                by a second kernel; 1 = TC only, inside a thread-block cluster
                                of split_k CTAs through distributed shared memory; 2 = CTA
                                pairs only, stream-K over the last waves (split_k 1) */
    int32_t cluster_m;       /* TC only: 2 = a cluster of two CTAs on two SMs computing one
                                256-row tile (bm = 256) with tcgen05 cta_group::2 MMAs;
                                else 1 */
} nnjit_candidate;

typedef struct nnjit_plan_s* nnjit_plan;

/*
 * Fixed settings (the primitive vector of Sec. 5.1): settings that offline
 * microbenchmarks found consistently better are fixed before the lite space is built,
 * which shrinks the space.  Each field is NNJIT_SETTING_FREE (searched; the default) or
 * the one value kept.  They act on the tensor-core family only:
 *   raster     tile order: 0 = M fastest, 1 = N fastest;
 *   kgroup     k-blocks per ring slot (candidate bk / one 128-byte k-block): 1 or 2;
 *   reduce     split-K reduction: 0 = second kernel, 1 = inside a cluster (DSMEM),
 *              2 = CTA-pair stream-K over the last waves.
 * A fixed value removes a candidate only where the same candidate with the fixed value
 * (every other searched field equal: bm, bn, split_k and the other two settings) is
 * in the space, so a setting never empties the space and never removes the only legal
 * choice (for example kgroup = 2 keeps bn = 256 tiles, which exist only with 1).  The
 * axes are applied in the order above.
 */
#define NNJIT_SETTING_FREE (-1)
typedef struct {
    int32_t raster;
    int32_t kgroup;
    int32_t reduce;
} nnjit_settings;

/* ---------------------------------------------------------------------------------- */

/* Static string for a status code.  Never NULL. */
const char* nnjit_status_string(nnjit_status s);

/* Detail of the last failing call on this thread ("" if none).  Valid until the next
 * call on this thread. */
const char* nnjit_last_error(void);

/* Library version, major*10000 + minor*100 + patch. */
int32_t nnjit_version(void);

/* Query the limits of CUDA device `device` (host call; needs a GPU). */
nnjit_status nnjit_device_limits_query(int32_t device, nnjit_device_limits* out);

/*
 * Build the lite space for `d` against `lim` (host only; needs no GPU).  Sec. 5.2 and
 * Table 1: enumerate power-of-two tiles (heuristic 2), keep those whose shared memory,
 * TMEM, register and thread usage fit the device, compute Block_core =
 * min(RegLimit, L1Limit, WarpLimit, ...), and order the survivors from most to fewest
 * blocks per core, then by the predicted cost; then drop what the process-wide fixed
 * settings (nnjit_settings_set) exclude.  Writes at most `capacity` candidates to
 * `out` (may be NULL when capacity is 0), the full count to *count, and the size of the
 * unpruned space (every tile/stage/split combination of the family's axes before the
 * usage rules and heuristics) to *naive_count (may be NULL).
 * INVALID_ARG for a bad descriptor; UNSUPPORTED when no family serves it.
 */
nnjit_status nnjit_space_enumerate(const nnjit_matmul_desc* d, const nnjit_device_limits* lim,
                                   nnjit_candidate* out, int32_t capacity, int32_t* count,
                                   int64_t* naive_count);

/*
 * Set (or, with s = NULL, clear) the process-wide fixed settings used by every later
 * nnjit_space_enumerate and plan call; the plan cache keys include them.  INVALID_ARG for
 * a value outside the field's range (FREE or the values listed above).  Thread-safe.
 */
nnjit_status nnjit_settings_set(const nnjit_settings* s);

/* The current process-wide fixed settings. */
nnjit_status nnjit_settings_get(nnjit_settings* out);

/*
 * One-variable-at-a-time microbenchmark (Sec. 5.1) over the products `descs[0..count)`
 * on the current device: each product's full space (every setting searched, the current
 * fixed settings ignored) is timed exhaustively as by NNJIT_PLAN_EXHAUSTIVE; then, from
 * its fastest candidate, each setting is flipped alone and the two times compared.  A
 * flip more than 2 % slower is a decisive vote for the fastest candidate's value; a
 * smaller difference is a tie; a setting whose flipped twin is not in the space has no
 * vote.  *out receives, per setting, the value every decisive vote agreed on, or FREE
 * when there was no decisive vote or the votes disagreed.  Nothing is applied: pass *out
 * to nnjit_settings_set.  `report` (may be NULL) receives a JSON object with each
 * product's space size, fastest candidate and per-setting times and verdicts; the
 * length it needs (with the NUL) is stored in *report_needed (may be NULL).  The plan
 * cache is neither read nor written.  Synchronises the device.  INVALID_ARG for
 * count < 1 or a bad descriptor; the first failing product's status otherwise.
 */
nnjit_status nnjit_settings_study(const nnjit_matmul_desc* descs, int32_t count, nnjit_settings* out,
                                  char* report, size_t report_len, size_t* report_needed);

/*
 * JIT-tune a plan for C[M,N] = A[M,K] . B[K,N] (B_KN, batch 1, packed, with a bias slot
 * that may be NULL at run time).  Shorthand for nnjit_matmul_plan_ex.
 */
nnjit_status nnjit_matmul_plan(int64_t M, int64_t N, int64_t K, nnjit_dtype dt,
                               double tune_budget_ms, nnjit_plan* out);

/*
 * JIT-tune a plan (Sec. 3: compose the lite space, evaluate candidates on the device,
 * keep the fastest).  Candidates are evaluated in space order on device scratch buffers
 * the call allocates and frees itself, while the wall-clock time spent stays under
 * tune_budget_ms (at least one candidate is timed when the budget is > 0).  Budget 0
 * takes the top-ranked candidate untimed (unless NNJIT_PLAN_REQUIRE_TIMED).  The choice
 * is the fastest median time; ties go to the lower space index.  The result is cached
 * per (type, shape, layout, strides, dtype, device) unless NNJIT_PLAN_NO_CACHE; a cache
 * hit returns at once.  Uses the current CUDA device.  Synchronises the device.
 * The plan owns its split-K workspace and its kernel-watchdog word.
 */
nnjit_status nnjit_matmul_plan_ex(const nnjit_matmul_desc* d, double tune_budget_ms,
                                  nnjit_plan* out);

/*
 * Plan that uses candidate `index` of the space nnjit_space_enumerate builds for `d` on
 * the current device, without tuning and without the cache (testing every candidate;
 * exhaustive sweeps).  INVALID_ARG if index is out of range.
 */
nnjit_status nnjit_matmul_plan_candidate(const nnjit_matmul_desc* d, int32_t index,
                                         nnjit_plan* out);

/*
 * Online plan (Sec. 3: kernels are evaluated on the device between inferences, and a
 * newly measured kernel replaces the registered one only if it is significantly faster).
 * No tuning happens here: the plan serves every nnjit_matmul_run / _run_batched call at
 * once, with the top-ranked candidate at first.  While the queue (the lite space in
 * evaluation order) lasts, each call is run instead with the candidate under evaluation
 * and timed with CUDA events recorded around that call's own launches; the timings are
 * read back on later calls without synchronising.  After 3 timed calls a candidate
 * replaces the incumbent if its median is more than 2 % lower.  Every call's result is
 * correct whichever candidate ran.  When the queue is exhausted the choice is stored in
 * the plan cache (unless NNJIT_PLAN_NO_CACHE), so later nnjit_matmul_plan_ex calls hit.
 * Calls on one online plan must not overlap on the GPU (share one stream); synchronise
 * before nnjit_plan_destroy.  Allocates the plan's workspace (for the widest candidate),
 * watchdog word and 16 CUDA events.
 */
nnjit_status nnjit_matmul_plan_online(const nnjit_matmul_desc* d, nnjit_plan* out);

/* Progress of an online plan: candidates fully evaluated, space size, the index of the
 * candidate now serving calls, and whether the queue is exhausted (1).  For other plans:
 * evaluated = space size, done = 1. */
nnjit_status nnjit_plan_online_progress(nnjit_plan p, int32_t* evaluated, int32_t* space_size,
                                        int32_t* current_index, int32_t* done);

/*
 * C = A . Bt (+ bias) with the plan's kernel, asynchronously on `stream`.
 * A, B: device pointers (float32 or bf16 per the plan's dtype); bias: float32[N] device
 * pointer or NULL (NULL means no bias even if the plan was made with has_bias);
 * C: float32 device pointer.  C must not overlap A, B or bias.  Tensor-core and GEMV
 * paths need A, B (and C for the GEMV's vector stores) 16-byte aligned, else
 * UNSUPPORTED.  Never synchronises.  A kernel watchdog expiry is reported by
 * nnjit_plan_check.  Batched plans run all batch items.
 */
nnjit_status nnjit_matmul_run(nnjit_plan p, const void* A, const void* B, const float* bias,
                              float* C, void* stream);

/* Batched form of nnjit_matmul_run for attention QK^T / PV (Table 3, K2/K3): no bias. */
nnjit_status nnjit_matmul_run_batched(nnjit_plan p, const void* A, const void* B, float* C,
                                      void* stream);

/*
 * End-to-end form with HOST buffers: copies A, B (and bias when non-NULL) host->device
 * into device staging buffers the plan owns (allocated on first use, packed layout),
 * runs the plan, and copies C device->host, all asynchronously on `stream`; the caller
 * synchronises the stream before reading hC.  Host buffers should be page-locked for
 * asynchronous copies.  Plans with non-packed strides are UNSUPPORTED here.
 */
nnjit_status nnjit_matmul_run_host(nnjit_plan p, const void* hA, const void* hB,
                                   const float* hbias, float* hC, void* stream);

/*
 * End-to-end form over a sequence of `count` products with HOST buffers (for instance the
 * Linears of a layer whose weights and activations come from host memory): product i is
 * nnjit_matmul_run_host(plans[i], hA[i], hB[i], hbias ? hbias[i] : NULL, hC[i]), but the
 * transfers of different products overlap each other and the kernels: the inputs of the
 * products are copied in, in order, on a host-to-device stream of the library, and each
 * result is copied out, in order, on a device-to-host stream of the library as soon as
 * its kernels finish, while the kernels run on `stream`.  The sequence's whole cost is
 * about the longer of the two copy directions plus one product's exposed head and tail,
 * instead of the sum of every copy and kernel.
 * Ordering: nothing of the call starts before the work already queued on `stream`, and
 * work queued on `stream` after the call starts after the last result has reached the
 * host, so the caller synchronises `stream` before reading any hC[i].  Within the call
 * the inputs of later products may be read before earlier results are written: no hC[i]
 * may overlap any hA[j], hB[j] or hbias[j].  A plan may appear more than once (its
 * staging buffers are then reused in order).  Every plan must belong to the current
 * device and be packed (else INVALID_ARG / UNSUPPORTED, checked before anything is
 * queued); hbias may be NULL (no bias anywhere) and hbias[i] may be NULL.  Host buffers
 * should be page-locked.  The copy streams and events are created on the first call on a
 * device and kept until exit; calls from several threads on one device are serialised
 * while they queue their work.  Never synchronises.
 */
nnjit_status nnjit_matmul_run_host_seq(int32_t count, const nnjit_plan* plans, const void* const* hA,
                                       const void* const* hB, const float* const* hbias,
                                       float* const* hC, void* stream);

/* Synchronise the plan's device and read its watchdog word: TIMEOUT if any kernel of
 * this plan stopped on an expired wait since the last check (the word is then reset). */
nnjit_status nnjit_plan_check(nnjit_plan p);

/*
 * JSON description of the plan: shape, family and parameters of the chosen candidate,
 * space size, naive count, tuning wall time, and every timed candidate with its median
 * microseconds.  Truncated to len-1 characters (always NUL-terminated when len > 0);
 * *needed (may be NULL) receives the full length + 1.
 */
nnjit_status nnjit_plan_describe(nnjit_plan p, char* buf, size_t len, size_t* needed);

/* The chosen candidate. */
nnjit_status nnjit_plan_candidate(nnjit_plan p, nnjit_candidate* out);

/* Free the plan and everything it owns.  NULL is a no-op.  The caller must ensure no
 * launch of this plan is still running (e.g. synchronise the stream first). */
nnjit_status nnjit_plan_destroy(nnjit_plan p);

/*
 * Fused attention (the QK^T -> softmax -> PV neighbours of the attention BatchMatMuls of
 * Table 3, K2 and K3): for each of `batch` independent problems (batch x heads),
 *   S = scale * Q K^T,  P = softmax over each row of S (keys j masked off are left out),
 *   O = P V,
 * without writing S or P to memory.  Q [batch][Lq][d], K and V [batch][Lk][d] packed
 * bfloat16, O [batch][Lq][d] packed float32, all device pointers the caller owns, 16-byte
 * aligned.  d is 64 or 128.  With causal = 1 query i sees keys j <= i + (Lk - Lq) (the
 * causal mask aligned to the last key, as in decoding with a cache); a query that sees no
 * key gets O = 0.  The scores are accumulated in float32 from exact bfloat16 products;
 * P is rounded to bfloat16 for the P V product, whose sums are float32.  Lq, Lk >= 0
 * (Lq = 0 is a no-op), batch >= 1, Lq, Lk, batch < 2^31.  `kernel` selects the
 * implementation: NNJIT_ATTN_AUTO (0) and NNJIT_ATTN_TCGEN05 (1) run the tensor-memory
 * kernel (128 queries per CTA, scores and outputs in TMEM, bounded waits), NNJIT_ATTN_MMA
 * (2) the warp-level MMA kernel (64 queries per CTA, no waits), NNJIT_ATTN_TCGEN05_2T (3)
 * the tensor-memory kernel with two 128-query tiles per CTA sharing each key and value
 * block (the tensor cores alternate between the tiles; bounded waits; when there are more
 * work items than CTAs, the CTAs take them from a work counter in device memory: each
 * call uses the next of 64 counter slots, which the call leaves at zero, so calls that
 * run at the same time on different streams use different slots, while one captured
 * graph replayed on two streams at once would share its slot and is not supported); AUTO takes the
 * kernel that nnjit_attention_tune recorded as fastest for the same (batch, Lq, Lk, d,
 * causal) on the current device, else the two-tile kernel (3) when batch * ceil(Lq / 256)
 * is at least half the device's SM count and the tensor-memory kernel (1) otherwise.  INVALID_ARG for a bad
 * descriptor or NULL pointer, UNSUPPORTED for another d or unaligned pointers.
 * Asynchronous on `stream`; allocates nothing.  An expired wait inside the tensor-memory
 * kernel is reported by nnjit_attention_check.
 */
typedef enum {
    NNJIT_ATTN_AUTO = 0,
    NNJIT_ATTN_TCGEN05 = 1,
    NNJIT_ATTN_MMA = 2,
    NNJIT_ATTN_TCGEN05_2T = 3
} nnjit_attention_kernel;

typedef struct {
    int64_t batch, Lq, Lk, d;
    int32_t causal;
    float scale;
    int32_t kernel;  /* nnjit_attention_kernel */
} nnjit_attention_desc;

nnjit_status nnjit_attention(const nnjit_attention_desc* desc, const void* Q, const void* K,
                             const void* V, float* O, void* stream);

/* Synchronise the current device and report whether any tensor-memory attention kernel
 * since the last check gave up on a wait (NNJIT_ERR_TIMEOUT, with the wait's code in
 * nnjit_last_error); clears the record.  The record is one word per device, shared by
 * every attention call on that device (unlike a matmul plan's own watchdog word): with
 * calls from several streams or threads, one caller's check can report, and clears,
 * another caller's expired wait, so callers that need to tell their calls apart must
 * serialise them with their checks (nnjit_attention_tune checks, and clears, it too). */
nnjit_status nnjit_attention_check(void);

/*
 * JIT selection for fused attention (Sec. 3: evaluate the candidates on the device, keep
 * the fastest): runs each kernel on the caller's buffers (O is overwritten; the inputs
 * are only read), once to warm up and then `reps` (1..100) times per trial for three
 * trials, on a stream of its own, and records the one with the lowest median time for
 * (batch, Lq, Lk, d, causal) on the current device, where later calls with kernel = AUTO
 * find it.  *times_us (may be NULL; three doubles) receives the medians of kernels 1, 2
 * and 3 (tensor-memory, warp-MMA, tensor-memory with two tiles), *chosen (may be NULL) the
 * recorded kernel.  Synchronous.  Errors as nnjit_attention;
 * NNJIT_ERR_TIMEOUT if a tensor-memory wait expired while timing.
 */
nnjit_status nnjit_attention_tune(const nnjit_attention_desc* desc, const void* Q, const void* K,
                                  const void* V, float* O, int32_t reps, double* times_us,
                                  int32_t* chosen);

/*
 * Decode GEMV that allocates nothing (the paper has no counterpart; this serves callers
 * that cannot allocate device memory when they run a product, e.g. a process whose
 * device memory a framework's caching allocator has already reserved, or a decode loop
 * that must not pay for cudaMalloc / cudaFree, which may synchronise the device).
 *
 * C[m,n] = sum_k x[m,k] * W[n,k] (+ bias[n]) for 1 <= M <= 8, with x [M][K] and W [N][K]
 * packed bf16, C [M][N] packed float32, bias float32[N] or NULL, all device pointers the
 * caller owns; K % 8 == 0, x and W 16-byte aligned, C and bias 4-byte aligned (else
 * UNSUPPORTED).  K is split into split_k slices
 * (1..64) whose float32 partial sums are kept in one fixed device array inside the
 * library of NNJIT_NOALLOC_SCRATCH_FLOATS floats (4 MiB, held by every GPU that loads
 * the library until the process exits) and then added in slice order.  Requests with
 * split_k * M * N above that size, or whose x slice (M * K / split_k bf16 values) exceeds
 * 96 KiB of shared memory, fail with UNSUPPORTED and a message in nnjit_last_error().
 * On success the call makes no allocation: it calls no cudaMalloc, cudaMallocAsync,
 * cudaFree or other allocating routine, and no host heap allocation of its own; it makes
 * no plan and does no tuning (one fixed GEMV configuration).  The first call on a device looks
 * up the array's device address (cudaGetSymbolAddress) and keeps it; make that first
 * call before any stream capture.  Every call on a device shares the one array: calls
 * that may overlap on the GPU (different streams, or another thread) race on it and
 * must be serialised by the caller.  Every partial is written before it is read, so the
 * array's previous contents never matter.  Asynchronous on `stream`.
 */
#define NNJIT_NOALLOC_SCRATCH_FLOATS (1 << 20)
nnjit_status nnjit_gemv_bf16_noalloc(int64_t M, int64_t N, int64_t K, const void* x, const void* W,
                                     const float* bias, float* C, int32_t split_k, void* stream);

/* Drop every cached plan choice of this process. */
nnjit_status nnjit_cache_clear(void);

/* Number of choices currently in the process plan cache. */
int32_t nnjit_cache_size(void);

/*
 * Persist the plan cache -- the kernel database of Sec. 5.3, keyed by kernel type, shape,
 * layout, strides, dtype and device (name, compute capability, SM count) -- to a text
 * file at `path` (overwritten), so that tuning results outlive the process.
 * NNJIT_ERR_INVALID_ARG if the file cannot be written.
 */
nnjit_status nnjit_cache_save(const char* path);

/*
 * Merge the entries of a file written by nnjit_cache_save into the plan cache (entries
 * already present are replaced); *loaded (may be NULL) receives the number read.  An entry
 * is used by nnjit_matmul_plan_ex only if its candidate is still a member of the lite
 * space this library builds for that problem on this device; otherwise the problem is
 * tuned afresh.  INVALID_ARG if the file cannot be read or is not a cache file.
 */
nnjit_status nnjit_cache_load(const char* path, int32_t* loaded);

#ifdef __cplusplus
}
#endif

#endif /* NNJIT_H */
