/*
 * Oracle for the dense MatMul / BatchMatMul operator -- TEST INFRASTRUCTURE ONLY.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may load this
 * code.  The GPU library never calls it and shares no code with it.
 *
 * What it computes (the operator every experiment of the paper tunes: MatMul in the
 * preliminary study of Sec. 2.2, the MatMul / BatchMatMul kernels K0-K3 of Table 3):
 *
 *     C[b,i,j] = sum_{k=0}^{K-1} A[b,i,k] * Bt[b,k,j]  (+ bias[j])
 *
 * with Bt = B when B is stored [K,N] (row-major, "KN") and Bt[k,j] = B[j,k] when B is
 * stored [N,K] (the Linear-weight layout, "NK").  The tiled loop nest of Table 1 and of
 * the tile/memory-hierarchy figure in Sec. 5.2 is a re-ordering of this sum; the oracle
 * is the sum itself: FP64, k ascending, one accumulator per output element, bias added
 * once after the sum.  Inputs are handed over already widened to double (every f32 and
 * bf16 value is exactly representable in double), so the oracle sees exactly the values
 * the GPU path is given.
 *
 * Rows are split across POSIX threads; each output element is still produced by one
 * thread in the order above, so the result does not depend on the thread count.
 */
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

#define ORACLE_B_KN 0
#define ORACLE_B_NK 1

typedef struct {
    int64_t batch, M, N, K;
    const double* A; int64_t lda, strideA;
    const double* B; int b_layout; int64_t ldb, strideB;
    const double* bias;
    double* C; int64_t ldc, strideC;
    int64_t row_begin, row_end; /* over the flattened (b, i) index */
} oracle_job;

/* One output row C[b,i,:].  KN: i-k-j order with a row of accumulators (still k
 * ascending per element).  NK: i-j-k dot products, contiguous in k for both operands. */
static void oracle_row(const oracle_job* jb, int64_t b, int64_t i, double* acc) {
    const double* a = jb->A + b * jb->strideA + i * jb->lda;
    const double* bm = jb->B + b * jb->strideB;
    double* c = jb->C + b * jb->strideC + i * jb->ldc;
    int64_t N = jb->N, K = jb->K;
    if (jb->b_layout == ORACLE_B_KN) {
        for (int64_t j = 0; j < N; ++j) acc[j] = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            const double aik = a[k];
            const double* brow = bm + k * jb->ldb;
            for (int64_t j = 0; j < N; ++j) acc[j] += aik * brow[j];
        }
    } else {
        for (int64_t j = 0; j < N; ++j) {
            const double* bcol = bm + j * jb->ldb;
            double s = 0.0;
            for (int64_t k = 0; k < K; ++k) s += a[k] * bcol[k];
            acc[j] = s;
        }
    }
    for (int64_t j = 0; j < N; ++j) c[j] = jb->bias ? acc[j] + jb->bias[j] : acc[j];
}

static void* oracle_worker(void* p) {
    oracle_job* jb = (oracle_job*)p;
    double* acc = (double*)malloc((size_t)(jb->N > 0 ? jb->N : 1) * sizeof(double));
    if (!acc) return (void*)1;
    for (int64_t r = jb->row_begin; r < jb->row_end; ++r) {
        int64_t b = r / jb->M, i = r % jb->M;
        oracle_row(jb, b, i, acc);
    }
    free(acc);
    return NULL;
}

/* Number of hardware threads the oracle uses when asked for 0. */
int oracle_hw_threads(void) {
    long n = sysconf(_SC_NPROCESSORS_ONLN);
    return n > 0 ? (int)n : 1;
}

/*
 * C (double, [batch][M][ldc]) = A . Bt (+ bias).  Returns 0 on success, 1 on a bad
 * argument, 2 on an allocation or thread failure.  nthreads <= 0 means all hardware
 * threads.  Strides and leading dimensions are in elements.
 */
int oracle_matmul_f64(int64_t batch, int64_t M, int64_t N, int64_t K,
                      const double* A, int64_t lda, int64_t strideA,
                      const double* B, int b_layout, int64_t ldb, int64_t strideB,
                      const double* bias, double* C, int64_t ldc, int64_t strideC,
                      int nthreads) {
    if (batch < 0 || M < 0 || N < 0 || K < 0) return 1;
    if (b_layout != ORACLE_B_KN && b_layout != ORACLE_B_NK) return 1;
    if (batch == 0 || M == 0 || N == 0) return 0;
    if (!C || (K > 0 && (!A || !B))) return 1;
    if (nthreads <= 0) nthreads = oracle_hw_threads();
    int64_t rows = batch * M;
    if (nthreads > rows) nthreads = (int)rows;

    oracle_job base;
    base.batch = batch; base.M = M; base.N = N; base.K = K;
    base.A = A; base.lda = lda; base.strideA = strideA;
    base.B = B; base.b_layout = b_layout; base.ldb = ldb; base.strideB = strideB;
    base.bias = bias; base.C = C; base.ldc = ldc; base.strideC = strideC;

    oracle_job* jobs = (oracle_job*)calloc((size_t)nthreads, sizeof(oracle_job));
    pthread_t* th = (pthread_t*)calloc((size_t)nthreads, sizeof(pthread_t));
    if (!jobs || !th) { free(jobs); free(th); return 2; }
    int rc = 0, started = 0;
    for (int t = 0; t < nthreads; ++t) {
        jobs[t] = base;
        jobs[t].row_begin = rows * t / nthreads;
        jobs[t].row_end = rows * (t + 1) / nthreads;
        if (t == nthreads - 1) break; /* the last slice runs on the calling thread */
        if (pthread_create(&th[t], NULL, oracle_worker, &jobs[t]) != 0) { rc = 2; break; }
        ++started;
    }
    if (rc == 0 && oracle_worker(&jobs[nthreads - 1]) != NULL) rc = 2;
    for (int t = 0; t < started; ++t) {
        void* ret = NULL;
        pthread_join(th[t], &ret);
        if (ret != NULL) rc = 2;
    }
    free(jobs); free(th);
    return rc;
}

/*
 * Widen bf16 bit patterns to double.  A bf16 value is the upper half of an IEEE-754
 * binary32 value, so shifting the 16 bits into the high half of a 32-bit word gives the
 * float exactly; the float widens to double exactly.
 */
void oracle_bf16_to_f64(const uint16_t* src, double* dst, int64_t n) {
    for (int64_t i = 0; i < n; ++i) {
        uint32_t w = ((uint32_t)src[i]) << 16;
        float f;
        memcpy(&f, &w, sizeof f);
        dst[i] = (double)f;
    }
}
