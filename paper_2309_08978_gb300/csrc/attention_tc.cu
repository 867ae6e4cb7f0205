// Fused attention on the 5th-generation tensor cores (nnjit_attention, kernel 1):
// O = softmax(scale Q K^T) V per batch x head without writing the scores.
//
// A persistent CTA per SM loops over (problem, 128-query block) items; 10 warps:
//   warp 0     TMA producer: an item's Q tile (two Q buffers), then its key and value
//              blocks of 128 rows through separate key and value rings (128-byte
//              swizzle; keys K-major, values MN-major), values one key block behind;
//   warp 1     allocates TMEM and issues (the warp converged, one lane elected by
//              elect.sync) S_g = Q K_g^T (M = 128,
//              N = 128, K = d) into TMEM score buffer g % 2, a block ahead, and
//              O += P_g V_g (M = 128, N = d, K = 128) with P_g read from TMEM as the A
//              operand, into the item's TMEM output;
//   warps 2-9  softmax: the two warps w, w + 4 share TMEM lane quarter w % 4 (32 query
//              rows) and split each row in two parts of 64 keys and d / 2 output
//              columns.  Row maximum over S_g (first pass; the parts' maxima meet
//              through shared memory behind a barrier of the two warps), then
//              p = 2^(s - m) stored as bf16 pairs into TMEM P buffer g % 2 (second
//              pass).  A row keeps its base m until a block's maximum exceeds it by
//              more than 2^8; only then is its TMEM output rescaled in place.
// The score and P buffers are double-buffered so that the tensor cores work on block
// g + 1 while the softmax warps work on block g.  Keys past Lk and, with the causal mask,
// keys past i + (Lk - Lq) score -inf; blocks a query block cannot see are skipped.  Every
// wait is bounded: on expiry the watchdog word is set, the CTA's abort flag raised, and
// every role leaves after draining what it issued.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>

#include "../../include/nnjit.h"
#include "launch.h"
#include "ptx.cuh"

namespace nnjit {

namespace {

__device__ int g_attn_watchdog;  // first expired wait's code (0: none)

// Work counters of the two-tile kernel: a launch uses slot Params::sched (the launcher
// cycles through the slots).  CTA b takes item b first, then (when there are more items
// than CTAs) items G + [0]++ in turn, so a CTA whose items run long takes fewer; a CTA
// that has taken its last item counts itself in [1], and the last one zeroes both for the
// slot's next launch.  Launches that run at the same time need different slots.
constexpr int kSchedSlots = 64;
__device__ unsigned g_attn_sched[kSchedSlots][2];

constexpr int kQ = 128;   // queries per work item (a CTA loops over items)
// Bytes of Q, K, V and O that one group of problems may touch (about 3/4 of the 129 MB L2).
constexpr long long kGroupL2Bytes = 96ll << 20;
constexpr int kKV = 128;  // keys per block
// Softmax warps per TMEM lane quarter.  Two: one (whole rows per thread, no exchange of
// maxima) measured 60.7 against 55.4 us on the Llama prefill heads, four (d = 64) slower
// too, the extra barriers and per-part overhead outweighing the extra warps.
template <int D>
__host__ __device__ constexpr int split_of() { return 2; }
template <int D>
__host__ __device__ constexpr int threads_of() { return 64 + 128 * split_of<D>(); }
constexpr int kErrProd = 0x301, kErrMmaQ = 0x311, kErrMmaKv = 0x312, kErrMmaP = 0x314;
constexpr int kErrSoftS = 0x321, kErrSoftO = 0x322, kErrItem = 0x323, kErrDrain = 0x331;

template <int D>
struct Cfg {
    // key and value ring slots (a third key slot with d = 128 measured no faster)
    static constexpr int kKStages = D == 64 ? 4 : 2;
    static constexpr int kVStages = D == 64 ? 4 : 2;
    static constexpr uint32_t kQBytes = kQ * D * 2;
    // two Q buffers, so that the next item's Q tile loads during this item
    static constexpr int kQBuf = 2;
    static constexpr uint32_t kKBytes = kKV * D * 2;
    static constexpr uint32_t kVBytes = kKV * D * 2;
    // output staging: one 32 x 32 f32 tile (4 KB, 128-byte swizzle) per softmax warp, stored
    // to global memory by TMA (whole 128-byte row segments instead of one row per lane)
    static constexpr uint32_t kOStage = 4096;
    static constexpr uint32_t kSmem =
        1024 + kQBuf * kQBytes + kKStages * kKBytes + kVStages * kVBytes + 8 * kOStage;
};

struct Params {
    CUtensorMap tq, tk, tv, to;
    CUtensorMap to16;  // O in 32 x 16 pieces (64-byte rows, 64-byte swizzle): the two-tile kernel
    float* O;
    int Lq, Lk, causal, qblocks, batch;
    int group;  // problems per item group (divides batch)
    float scale_log2;
    int sched;  // two-tile kernel: its work-counter slot
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Packed pairs of f32 (the Blackwell f32x2 add and multiply: one instruction for two lanes
// worth of work, each half rounded as the scalar operation would be), and the three-input
// maximum.
__device__ __forceinline__ uint64_t f2(uint32_t lo, uint32_t hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(lo), "r"(hi));
    return r;
}
__device__ __forceinline__ void f2_split(uint64_t v, uint32_t& lo, uint32_t& hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=r"(lo), "=r"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// 32 lanes x 64 consecutive 32-bit TMEM columns in one load, and its wait.
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, uint32_t (&r)[64]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x64.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%64];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait64(uint32_t (&r)[64]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31]), "+r"(r[32]), "+r"(r[33]), "+r"(r[34]), "+r"(r[35]), "+r"(r[36]), "+r"(r[37]), "+r"(r[38]), "+r"(r[39]), "+r"(r[40]), "+r"(r[41]), "+r"(r[42]), "+r"(r[43]), "+r"(r[44]), "+r"(r[45]), "+r"(r[46]), "+r"(r[47]), "+r"(r[48]), "+r"(r[49]), "+r"(r[50]), "+r"(r[51]), "+r"(r[52]), "+r"(r[53]), "+r"(r[54]), "+r"(r[55]), "+r"(r[56]), "+r"(r[57]), "+r"(r[58]), "+r"(r[59]), "+r"(r[60]), "+r"(r[61]), "+r"(r[62]), "+r"(r[63])
                 :
                 : "memory");
}

__device__ __forceinline__ void st_shared_f4(uint32_t addr, float a, float b, float c, float d) {
    asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
                 : "memory");
}

// 32 lanes x 32 consecutive 32-bit TMEM columns stored from registers, and the wait for
// this thread's outstanding stores.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
                 : "memory");
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
                 : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

template <int D>
__global__ void __launch_bounds__(threads_of<D>(), 1) attention_tc_kernel(const __grid_constant__ Params p) {
    using C = Cfg<D>;
    constexpr int kSplit = split_of<D>();
    constexpr int kCols = kKV / kSplit;  // score columns of a row per softmax thread
    constexpr int SK = C::kKStages, SV = C::kVStages;
    constexpr int kDB = D / 64;  // 64-element (128-byte) column blocks of d
    extern __shared__ uint8_t raw[];
    // q_full, q_empty (2 each), drain, k_full, k_empty (SK each), v_full, v_empty (SV
    // each), s_full, p_full, o_full (2 each)
    __shared__ __align__(8) uint64_t bars[5 + 2 * C::kKStages + 2 * C::kVStages + 6];
    static_assert(C::kQBuf <= 2, "two Q barrier pairs");
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_word;
    // [part][row]: partial row maxima, then sums.  One buffer is enough: a group barrier
    // (the vote on the next wait) separates each read from the next write.
    __shared__ float red[kSplit][kQ];
    volatile int* abort_flag = &abort_word;
    int* err = &g_attn_watchdog;

    const uint32_t base = (ptx::smem_u32(raw) + 1023u) & ~1023u;
    // separate key and value rings of S slots each: a key slot is free once its score
    // product has completed, well before the value slot of the same block
    constexpr int QB = C::kQBuf;
    auto sQ = [&](int i) { return base + (uint32_t)i * C::kQBytes; };
    const uint32_t sKR = base + QB * C::kQBytes, sVR = sKR + SK * C::kKBytes;
    auto sK = [&](int s) { return sKR + (uint32_t)s * C::kKBytes; };
    auto sV = [&](int s) { return sVR + (uint32_t)s * C::kVBytes; };
    const uint32_t sO = sVR + SV * C::kVBytes;  // 8 output staging tiles
    auto bar = [&](int i) { return ptx::smem_u32(&bars[i]); };
    const uint32_t drain_bar = bar(4);
    auto q_full = [&](int i) { return bar(i); };
    auto q_empty = [&](int i) { return bar(2 + i); };
    auto k_full = [&](int s) { return bar(5 + s); };
    auto k_empty = [&](int s) { return bar(5 + SK + s); };
    constexpr int kVB = 5 + 2 * SK, kSB = kVB + 2 * SV;
    auto v_full = [&](int s) { return bar(kVB + s); };
    auto v_empty = [&](int s) { return bar(kVB + SV + s); };
    auto s_full = [&](int i) { return bar(kSB + i); };
    auto p_full = [&](int i) { return bar(kSB + 2 + i); };
    auto o_full = [&](int i) { return bar(kSB + 4 + i); };

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int shift = p.Lk - p.Lq;
    const int items = p.qblocks * p.batch;
    // Work item -> (problem, first query, key blocks).  The problems run in groups of
    // p.group, sized on the host so that a group's Q, K, V and O fit in L2 together: the
    // key and value blocks a problem's query blocks share are then read from DRAM once.
    // Within a group the items run heaviest first: with the causal mask the last query
    // blocks see the most keys.
    auto decode = [&](int it, int& bb, int& qq0) {
        const int per = p.group * p.qblocks;
        const int g = it / per, r = it - g * per;
        bb = g * p.group + r % p.group;
        qq0 = (p.qblocks - 1 - r / p.group) * kQ;
        int kv_end = p.Lk;
        if (p.causal) kv_end = min(p.Lk, max(0, min(qq0 + kQ, p.Lq) - 1 + shift + 1));
        return (kv_end + kKV - 1) / kKV;
    };

    if (threadIdx.x == 0) {
        for (int i = 0; i < QB; ++i) {
            ptx::mbar_init(q_full(i), 1);
            ptx::mbar_init(q_empty(i), 1);
        }
        for (int s = 0; s < SK; ++s) {
            ptx::mbar_init(k_full(s), 1);
            ptx::mbar_init(k_empty(s), 1);
        }
        for (int s = 0; s < SV; ++s) {
            ptx::mbar_init(v_full(s), 1);
            ptx::mbar_init(v_empty(s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(s_full(i), 1);
            ptx::mbar_init(p_full(i), 4 * kSplit);  // one arrival per softmax warp
            ptx::mbar_init(o_full(i), 1);
        }
        ptx::mbar_init(drain_bar, 1);
        abort_word = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(&tmem_slot), 512);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = tmem_slot;
    ptx::griddep_wait();
    if (threadIdx.x == 0) ptx::griddep_launch_dependents();

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            ptx::prefetch_tmap(&p.tq);
            ptx::prefetch_tmap(&p.tk);
            ptx::prefetch_tmap(&p.tv);
            uint32_t k_armed = 0, k_par = 0, v_armed = 0, v_par = 0, q_armed = 0, q_par = 0;
            int g = 0, nq = 0;  // key blocks and Q tiles loaded so far
            bool ok = true;
            // the value block of global block gv (problem vb, first key vk0): issued one key
            // block behind, so that a wait for a value slot never holds back the next keys
            int gv = -1, vb = 0, vk0 = 0;
            auto load_v = [&]() -> bool {
                const int st = gv % SV;
                const uint32_t ph = (uint32_t)(gv / SV) & 1u;
                if (!ptx::mbar_wait(v_empty(st), ph ^ 1u, abort_flag, err, kErrProd)) return false;
                ptx::mbar_arrive_expect_tx(v_full(st), C::kVBytes);
                for (int kb = 0; kb < 2; ++kb)       // 64 keys per K-block of P V
                    for (int a = 0; a < kDB; ++a)    // 64 columns of d per swizzle atom
                        ptx::tma_load_3d(sV(st) + kb * (D * 128u) + a * 8192u, &p.tv, a * 64, vk0 + kb * 64, vb,
                                         v_full(st));
                v_armed |= 1u << st;
                v_par = (v_par & ~(1u << st)) | (ph << st);
                gv = -1;
                return true;
            };
            for (int it = blockIdx.x; ok && it < items; it += gridDim.x) {
                int bb, qq0;
                const int nblocks = decode(it, bb, qq0);
                if (nblocks == 0) continue;
                // a Q buffer is free once the score MMAs of the item that used it have completed
                const int qi = nq % QB;
                const uint32_t qph = (uint32_t)(nq / QB) & 1u;
                if (nq >= QB && !ptx::mbar_wait(q_empty(qi), qph ^ 1u, abort_flag, err, kErrProd)) break;
                ptx::mbar_arrive_expect_tx(q_full(qi), C::kQBytes);
                for (int kb = 0; kb < kDB; ++kb)
                    ptx::tma_load_3d(sQ(qi) + kb * 16384u, &p.tq, kb * 64, qq0, bb, q_full(qi));
                q_armed |= 1u << qi;
                q_par = (q_par & ~(1u << qi)) | (qph << qi);
                ++nq;
                for (int j = 0; j < nblocks; ++j, ++g) {
                    const int st = g % SK;
                    const uint32_t ph = (uint32_t)(g / SK) & 1u;
                    if (!ptx::mbar_wait(k_empty(st), ph ^ 1u, abort_flag, err, kErrProd)) {
                        ok = false;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(k_full(st), C::kKBytes);
                    for (int kb = 0; kb < kDB; ++kb)
                        ptx::tma_load_3d(sK(st) + kb * 16384u, &p.tk, kb * 64, j * kKV, bb, k_full(st));
                    k_armed |= 1u << st;
                    k_par = (k_par & ~(1u << st)) | (ph << st);
                    if (gv >= 0 && !load_v()) {
                        ok = false;
                        break;
                    }
                    gv = g;
                    vb = bb;
                    vk0 = j * kKV;
                }
                // the item's last value block before the next item's Q tile and keys
                if (ok && gv >= 0 && !load_v()) ok = false;
            }
            // drain: every copy issued here has landed before the CTA may exit
            volatile int no_abort = 0;
            for (int i = 0; i < QB; ++i)
                if (q_armed & (1u << i))
                    ptx::mbar_wait(q_full(i), (q_par >> i) & 1u, &no_abort, err, kErrDrain, ptx::kWaitLimitNs / 4);
            for (int st = 0; st < SK; ++st)
                if (k_armed & (1u << st))
                    ptx::mbar_wait(k_full(st), (k_par >> st) & 1u, &no_abort, err, kErrDrain, ptx::kWaitLimitNs / 4);
            for (int st = 0; st < SV; ++st)
                if (v_armed & (1u << st))
                    ptx::mbar_wait(v_full(st), (v_par >> st) & 1u, &no_abort, err, kErrDrain, ptx::kWaitLimitNs / 4);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        // The whole warp runs the loop converged: every lane waits (the results are voted,
        // so the warp leaves as one) and elect.sync picks the lane that issues.
        auto wait_all = [&](uint32_t bar, uint32_t parity, int code) {
            return __all_sync(0xffffffffu, ptx::mbar_wait(bar, parity, abort_flag, err, code));
        };
        constexpr uint32_t kIdescS = ptx::instr_desc(1u, false, kQ, kKV);
        constexpr uint32_t kIdescO = ptx::instr_desc(1u, true, kQ, D);
        uint32_t q_addr = sQ(0);  // the current item's Q tile
        // S_g = Q K_g^T into score buffer g % 2
        auto issue_s = [&](int g) -> bool {
            const int sb = g & 1, st = g % SK;
            // Score buffer g % 2 is free: the softmax read S_{g-2} before releasing P_{g-2},
            // and P_{g-2} V_{g-2} was issued (after that release) before this product.
            if (!wait_all(k_full(st), (uint32_t)((g / SK) & 1), kErrMmaKv)) return false;
            ptx::tc_fence_after();
            const uint32_t d_tmem = tmem + (uint32_t)sb * kKV;
#pragma unroll
            for (int kb = 0; kb < kDB; ++kb) {
                const uint64_t ad = ptx::smem_desc(q_addr + kb * 16384u, 16, 1024);
                const uint64_t bd = ptx::smem_desc(sK(st) + kb * 16384u, 16, 1024);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    ptx::mma_ss_elect<0>(d_tmem, ad + 2 * kk, bd + 2 * kk, kIdescS, (kb | kk) ? 1u : 0u);
            }
            ptx::tc_commit_elect(s_full(sb));
            ptx::tc_commit_elect(k_empty(st));  // the key slot is free once S_g has completed
            return true;
        };
        int g = 0, nq = 0;
        bool ok = true;
        for (int it = blockIdx.x; ok && it < items; it += gridDim.x) {
            int bb, qq0;
            const int nblocks = decode(it, bb, qq0);
            if (nblocks == 0) continue;
            const int qi = nq % QB;
            if (!wait_all(q_full(qi), (uint32_t)(nq / QB) & 1u, kErrMmaQ)) break;
            q_addr = sQ(qi);
            ++nq;
            ptx::tc_fence_after();
            if (!issue_s(g)) break;
            for (int j = 0; j < nblocks; ++j, ++g) {
                if (j + 1 < nblocks) {
                    if (!issue_s(g + 1)) {
                        ok = false;
                        break;
                    }
                } else {
                    ptx::tc_commit_elect(q_empty(qi));  // every score MMA of the item is issued
                }
                const int st = g % SV;
                if (!wait_all(p_full(g & 1), (g >> 1) & 1, kErrMmaP) ||
                    !wait_all(v_full(st), (uint32_t)((g / SV) & 1), kErrMmaKv)) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t o_tmem = tmem + 2u * kKV;  // O accumulates over the item's blocks
                const uint32_t p_tmem = o_tmem + D + (uint32_t)(g & 1) * (kKV / 2);  // P_g, bf16 pairs
#pragma unroll
                for (int kb = 0; kb < 2; ++kb) {
                    const uint64_t bd = ptx::smem_desc(sV(st) + kb * (D * 128u), 8192, 1024, ptx::kLayoutSw128);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)  // keys kb * 64 + kk * 16 .. + 15: 8 columns of P
                        ptx::mma_ts_f16_elect(o_tmem, p_tmem + kb * 32 + kk * 8, bd + 128 * kk, kIdescO,
                                              (j | kb | kk) ? 1u : 0u);
                }
                ptx::tc_commit_elect(o_full(g & 1));
                ptx::tc_commit_elect(v_empty(st));
            }
        }
        // every MMA issued here has completed before TMEM is freed
        __syncwarp();
        ptx::tc_commit_elect(drain_bar);
        volatile int no_abort = 0;
        ptx::mbar_wait(drain_bar, 0, &no_abort, err, kErrDrain, ptx::kWaitLimitNs / 4);
    } else {
        // ------------------------------------------------------------ softmax warps
        const int q = warp & 3;                 // TMEM lane quarter
        const int part = (warp - 2) >> 2;       // which kCols columns of the row
        const int row = q * 32 + lane;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        constexpr int kOP = D / kSplit;         // output columns of this part
        // barrier of the kSplit warps of lane quarter q; the vote keeps them leaving together
        auto group_any = [&](bool v) -> bool {
            uint32_t r;
            asm volatile(
                "{\n\t.reg .pred a, b;\n\t"
                "setp.ne.u32 a, %1, 0;\n\t"
                "barrier.cta.red.or.pred b, %2, %3, a;\n\t"
                "selp.u32 %0, 1, 0, b;\n\t}"
                : "=r"(r)
                : "r"((uint32_t)v), "r"(1 + q), "n"(32 * kSplit)
                : "memory");
            return r != 0;
        };
        auto group_sync = [&]() { asm volatile("bar.sync %0, %1;" ::"r"(1 + q), "n"(32 * kSplit) : "memory"); };
        // the maximum (op 0) or sum (op 1) of the row's kSplit partial values
        auto row_reduce = [&](float v, int op) -> float {
            if constexpr (kSplit == 1) return v;
            red[part][row] = v;
            group_sync();
            float r = v;
#pragma unroll
            for (int k = 1; k < kSplit; ++k) {
                const float w = red[(part + k) % kSplit][row];
                r = op == 0 ? fmaxf(r, w) : r + w;
            }
            return r;
        };
        int g = 0;
        bool ok = true;
        for (int it = blockIdx.x; it < items; it += gridDim.x) {
            int bb, qq0;
            const int nblocks = decode(it, bb, qq0);
            const int qrow = qq0 + row;
            const int last = p.causal ? qrow + shift : p.Lk - 1;  // last key this row sees
            // The output accumulates in TMEM (the P V products add onto it); the row keeps
            // its base m (p = 2^(x - m)) until a block's maximum exceeds it by more than
            // 2^8, and only then is the TMEM row rescaled by 2^(m_old - m_new) (values up
            // to 2^8 are harmless to bf16 P and float32 sums).
            float m = -INFINITY, l = 0.0f;
            const uint32_t orow = tmem + lane_base + 2u * kKV + (uint32_t)(part * kOP);
            for (int j = 0; ok && j < nblocks; ++j, ++g) {
                const int sb = g & 1;
                const bool ready = ptx::mbar_wait(s_full(sb), (g >> 1) & 1, abort_flag, err, kErrSoftS);
                if (group_any(!ready)) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t sa = tmem + lane_base + (uint32_t)sb * kKV + (uint32_t)(part * kCols);
                // this part of the row's scores, in one TMEM load kept for both passes
                uint32_t sr[kCols];
#pragma unroll
                for (int c = 0; c < kCols; c += 64) tmem_ld64(sa + c, *reinterpret_cast<uint32_t(*)[64]>(sr + c));
#pragma unroll
                for (int c = 0; c < kCols; c += 64) tmem_wait64(*reinterpret_cast<uint32_t(*)[64]>(sr + c));
                ptx::tc_fence_before();
                // columns 0..lim of this part are visible
                const int lim = min(last, p.Lk - 1) - j * kKV - part * kCols;
                // pass 1: scale to base 2 in place (-inf where masked), this part's maximum
                // (four independent partial maxima), then the row's
                float mxv[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                const uint32_t cb = __float_as_uint(p.scale_log2);
                const uint64_t c2 = f2(cb, cb);
                if (lim >= kCols - 1) {  // every column of this part is visible
#pragma unroll
                    for (int i = 0; i < kCols; i += 2) {  // two columns per packed multiply
                        f2_split(f2_mul(f2(sr[i], sr[i + 1]), c2), sr[i], sr[i + 1]);
                        mxv[(i >> 1) & 3] =
                            max3(mxv[(i >> 1) & 3], __uint_as_float(sr[i]), __uint_as_float(sr[i + 1]));
                    }
                } else {
                    const uint32_t ninf = __float_as_uint(-INFINITY);
#pragma unroll
                    for (int i = 0; i < kCols; i += 2) {
                        f2_split(f2_mul(f2(sr[i], sr[i + 1]), c2), sr[i], sr[i + 1]);
                        if (i > lim) sr[i] = ninf;
                        if (i + 1 > lim) sr[i + 1] = ninf;
                        mxv[(i >> 1) & 3] =
                            max3(mxv[(i >> 1) & 3], __uint_as_float(sr[i]), __uint_as_float(sr[i + 1]));
                    }
                }
                const float mx = row_reduce(fmaxf(fmaxf(mxv[0], mxv[1]), fmaxf(mxv[2], mxv[3])), 0);
                // a new base only when the maximum outgrows the current one by 2^8
                const bool rebase = mx > m + 8.0f;  // (always for the first visible key: m = -inf)
                float alpha = 1.0f;
                if (rebase) {
                    alpha = ex2(m - mx);  // 0 while m = -inf
                    m = mx;
                    l *= alpha;
                }
                const float basev = m == -INFINITY ? 0.0f : m;  // no visible key yet: every p is 0
                // pass 2: p = 2^(s - m) as bf16 into P in TMEM (the row's lane; keys 2c, 2c + 1
                // of the block in column c of P buffer g % 2), the A operand of P V
                const uint32_t pcol = tmem + lane_base + 2u * kKV + D + (uint32_t)sb * (kKV / 2) +
                                      (uint32_t)(part * kCols / 2);
                // packed partial sums: two pairs of lanes (shorter dependency chains)
                uint64_t lv2[2] = {0ull, 0ull};
                const uint32_t nb = __float_as_uint(-basev);  // x + (-m) rounds as x - m
                const uint64_t nb2 = f2(nb, nb);
#pragma unroll
                for (int c0 = 0; c0 < kCols; c0 += 64) {  // 64 keys = 32 columns of P per store
                    uint32_t pk[32];
#pragma unroll
                    for (int i = 0; i < 64; i += 2) {
                        // the maximum gives exactly 2^0 = 1 when it is the base; masked 2^-inf = 0
                        uint32_t d0, d1;
                        f2_split(f2_add(f2(sr[c0 + i], sr[c0 + i + 1]), nb2), d0, d1);
                        const float p0 = ex2(__uint_as_float(d0)), p1 = ex2(__uint_as_float(d1));
                        lv2[(i >> 1) & 1] = f2_add(lv2[(i >> 1) & 1], f2(__float_as_uint(p0), __float_as_uint(p1)));
                        pk[i >> 1] = pack_bf16(p0, p1);
                    }
                    tmem_st32(pcol + (uint32_t)(c0 / 2), pk);
                }
                {
                    uint32_t a0, a1, b0, b1;
                    f2_split(lv2[0], a0, a1);
                    f2_split(lv2[1], b0, b1);
                    l += (__uint_as_float(a0) + __uint_as_float(a1)) + (__uint_as_float(b0) + __uint_as_float(b1));
                }
                // O (the P V products of this item's earlier blocks) is complete in TMEM; P_g went to
                // the other P buffer meanwhile
                if (j >= 1) {
                    const bool done = ptx::mbar_wait(o_full((g - 1) & 1), ((g - 1) >> 1) & 1, abort_flag, err, kErrSoftO);
                    if (group_any(!done)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    // rescale the warp's rows of O in TMEM when any of them took a new base
                    if (__any_sync(0xffffffffu, rebase)) {
#pragma unroll
                        for (int c0 = 0; c0 < kOP; c0 += 32) {
                            uint32_t r[32];
                            ptx::tmem_ld32(orow + c0, r);
                            ptx::tmem_wait_ld(r);
#pragma unroll
                            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
                            tmem_st32(orow + c0, r);
                        }
                    }
                }
                tmem_wait_st();
                ptx::tc_fence_before();  // P_g and the rescaled O are stored before P V_g runs
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(p_full(sb));  // one arrival per warp
            }
            // the row sum is the parts' sums (all relative to the same base)
            l = row_reduce(l, 1);
            // the item's output: O from TMEM once its last P V product has completed
            bool have_o = false;
            if (ok && nblocks > 0) {
                const bool done = ptx::mbar_wait(o_full((g - 1) & 1), ((g - 1) >> 1) & 1, abort_flag, err, kErrSoftO);
                ok = !group_any(!done);
                have_o = ok;
                if (ok) ptx::tc_fence_after();
            }
            const float inv = (have_o && l > 0.0f) ? 1.0f / l : 0.0f;
            // 32 x 32 tiles of the warp's rows and this part's columns: staged with the
            // 128-byte swizzle (16-byte chunk c of row r at c ^ (r % 8)) and stored by TMA,
            // which leaves rows past Lq unwritten
            const uint32_t stage = sO + (uint32_t)(warp - 2) * C::kOStage;
#pragma unroll
            for (int c0 = 0; c0 < kOP; c0 += 32) {
                uint32_t r[32];
                if (have_o) {
                    ptx::tmem_ld32(orow + c0, r);
                    ptx::tmem_wait_ld(r);
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) r[i] = 0u;
                }
                if (lane == 0) ptx::bulk_wait_all_read();  // the tile's previous store has read it
                __syncwarp();
#pragma unroll
                for (int c = 0; c < 8; ++c)
                    st_shared_f4(stage + (uint32_t)lane * 128u + ((uint32_t)(c ^ (lane & 7)) << 4),
                                 __uint_as_float(r[4 * c]) * inv, __uint_as_float(r[4 * c + 1]) * inv,
                                 __uint_as_float(r[4 * c + 2]) * inv, __uint_as_float(r[4 * c + 3]) * inv);
                ptx::fence_proxy_async_smem();  // the tile is read by the TMA (async proxy)
                __syncwarp();
                if (lane == 0) {
                    ptx::tma_store_3d(&p.to, stage, part * kOP + c0, qq0 + q * 32, bb);
                    ptx::bulk_commit();
                }
            }
            ptx::tc_fence_before();  // the next item's first P V overwrites O
            // the next item's first maximum is written only after every part read this sum
            group_sync();
            if (!ok) break;
        }
        if (lane == 0) ptx::bulk_wait_all();  // every output store has completed
        __syncwarp();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------------------------
// Kernel 3: two query tiles per work item.  An item is 256 queries of one problem, tiles
// A (rows 0..127) and B (rows 128..255), sharing every key and value block.  The tensor
// cores alternate between the tiles: while the softmax warps of tile A turn S_A(j) into
// P_A(j), the MMAs compute S_B(j) or P_B V, and the other way round.  TMEM holds S_A, S_B,
// O_A and O_B (512 columns with d = 128); P_X(j) is written over the columns of S_X(j)
// it was computed from (the softmax has read them), and S_X(j + 1) is issued only after
// P_X(j) V(j), so the in-order tensor pipe reads P_X(j) before overwriting it.  Each
// softmax thread owns a whole row (no exchange of row maxima), read from TMEM in 32-column
// pieces.
//   warp 0     TMA producer: takes the items (its own index first, then from the launch's
//              work counter) and publishes them in the item ring; per item Q_A, the first
//              key block, Q_B (each tile's Q buffer with its own barriers), then the key
//              and value blocks through the key and value rings;
//   warp 1     TMEM owner and MMA issuer (converged warp, elected lane);
//   warps 2-5  softmax of tile A (TMEM lane quarter = warp % 4), warps 6-9 of tile B.
// The MMA and softmax warps read the items from the ring in the producer's order.  Every
// wait is bounded, as in kernel 1.
template <int D>
struct Cfg2 {
    static constexpr int kKStages = 2;
    static constexpr int kVStages = 2;
    static constexpr uint32_t kQBytes = kQ * D * 2;  // one tile
    static constexpr uint32_t kKBytes = kKV * D * 2;
    static constexpr uint32_t kVBytes = kKV * D * 2;
    static constexpr uint32_t kOStage = 4096;
    static constexpr uint32_t kSmem = 1024 + 2 * kQBytes + kKStages * kKBytes + kVStages * kVBytes + 8 * kOStage;
};

template <int D>
__global__ void __launch_bounds__(320, 1) attention_tc2_kernel(const __grid_constant__ Params p) {
    using C = Cfg2<D>;
    constexpr int SK = C::kKStages, SV = C::kVStages;
    constexpr int kDB = D / 64;  // 64-element (128-byte) column blocks of d
    extern __shared__ uint8_t raw[];
    constexpr int kIR = 4;  // item ring: the items the producer has taken ahead
    // q_full[X], q_empty[X], drain, k_full/k_empty (SK each), v_full/v_empty (SV each),
    // per tile X: s_full[X], p_full[X], o_full[X]; then i_full/i_empty (kIR each)
    __shared__ __align__(8) uint64_t bars[5 + 2 * SK + 2 * SV + 6 + 2 * kIR];
    __shared__ int item_ring[kIR];
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_word;
    volatile int* abort_flag = &abort_word;
    int* err = &g_attn_watchdog;

    const uint32_t base = (ptx::smem_u32(raw) + 1023u) & ~1023u;
    auto sQ = [&](int x) { return base + (uint32_t)x * C::kQBytes; };
    const uint32_t sKR = base + 2 * C::kQBytes, sVR = sKR + SK * C::kKBytes;
    auto sK = [&](int s) { return sKR + (uint32_t)s * C::kKBytes; };
    auto sV = [&](int s) { return sVR + (uint32_t)s * C::kVBytes; };
    const uint32_t sO = sVR + SV * C::kVBytes;  // 8 output staging tiles
    auto bar = [&](int i) { return ptx::smem_u32(&bars[i]); };
    // each tile's Q buffer has its own pair of barriers, so that tile A's next Q tile
    // loads as soon as A's last score product of the current item has completed
    auto q_full = [&](int x) { return bar(x); };
    auto q_empty = [&](int x) { return bar(2 + x); };
    const uint32_t drain_bar = bar(4);
    auto k_full = [&](int s) { return bar(5 + s); };
    auto k_empty = [&](int s) { return bar(5 + SK + s); };
    constexpr int kVB = 5 + 2 * SK, kXB = kVB + 2 * SV;
    auto v_full = [&](int s) { return bar(kVB + s); };
    auto v_empty = [&](int s) { return bar(kVB + SV + s); };
    auto s_full = [&](int x) { return bar(kXB + x); };
    auto p_full = [&](int x) { return bar(kXB + 2 + x); };
    auto o_full = [&](int x) { return bar(kXB + 4 + x); };
    auto i_full = [&](int s) { return bar(kXB + 6 + s); };
    auto i_empty = [&](int s) { return bar(kXB + 6 + kIR + s); };
    // TMEM: S_A at column 0, S_B at 128, O_A at 256, O_B at 256 + D
    auto s_col = [&](int x) { return (uint32_t)x * kKV; };
    auto o_col = [&](int x) { return 2u * kKV + (uint32_t)x * D; };

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int shift = p.Lk - p.Lq;
    const int items = p.qblocks * p.batch;  // qblocks: 256-query blocks here
    // Work item -> (problem, first query) and the key blocks tiles A and B see: as kernel
    // 1's order (problem groups that fit in L2, heaviest first within a group).
    auto decode = [&](int it, int& bb, int& qq0, int& na, int& nb) {
        const int per = p.group * p.qblocks;
        const int g = it / per, r = it - g * per;
        bb = g * p.group + r % p.group;
        qq0 = (p.qblocks - 1 - r / p.group) * (2 * kQ);
        auto blocks = [&](int q0) {  // key blocks the rows q0 .. q0 + 127 (below Lq) see
            if (q0 >= p.Lq) return 0;
            int kv_end = p.Lk;
            if (p.causal) kv_end = min(p.Lk, max(0, min(q0 + kQ, p.Lq) - 1 + shift + 1));
            return (kv_end + kKV - 1) / kKV;
        };
        na = blocks(qq0);
        nb = blocks(qq0 + kQ);
    };

    // Items are handed out dynamically: the producer takes the next item index from the
    // launch's work counter and publishes it in the item ring; the other roles read the
    // same sequence from the ring (an index past the last item ends every role's loop).
    auto next_item = [&](int n) -> int {  // the n-th item of this CTA (MMA and softmax warps)
        const int s = n % kIR;
        if (!__all_sync(0xffffffffu, ptx::mbar_wait(i_full(s), (uint32_t)(n / kIR) & 1u, abort_flag, err, kErrItem)))
            return -1;
        const int it = *reinterpret_cast<volatile int*>(&item_ring[s]);
        __syncwarp();
        if ((threadIdx.x & 31) == 0) ptx::mbar_arrive(i_empty(s));
        return it;
    };

    if (threadIdx.x == 0) {
        for (int x = 0; x < 2; ++x) {
            ptx::mbar_init(q_full(x), 1);
            ptx::mbar_init(q_empty(x), 1);
        }
        ptx::mbar_init(drain_bar, 1);
        for (int s = 0; s < SK; ++s) {
            ptx::mbar_init(k_full(s), 1);
            ptx::mbar_init(k_empty(s), 1);
        }
        for (int s = 0; s < SV; ++s) {
            ptx::mbar_init(v_full(s), 1);
            ptx::mbar_init(v_empty(s), 1);
        }
        for (int x = 0; x < 2; ++x) {
            ptx::mbar_init(s_full(x), 1);
            ptx::mbar_init(p_full(x), 4);  // one arrival per softmax warp of the tile
            ptx::mbar_init(o_full(x), 1);
        }
        for (int s = 0; s < kIR; ++s) {
            ptx::mbar_init(i_full(s), 1);
            ptx::mbar_init(i_empty(s), 9);  // the MMA warp and the eight softmax warps
        }
        abort_word = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(&tmem_slot), 512);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = tmem_slot;
    ptx::griddep_wait();
    if (threadIdx.x == 0) ptx::griddep_launch_dependents();

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            ptx::prefetch_tmap(&p.tq);
            ptx::prefetch_tmap(&p.tk);
            ptx::prefetch_tmap(&p.tv);
            uint32_t k_armed = 0, k_par = 0, v_armed = 0, v_par = 0, q_armed = 0, q_par = 0;
            int g = 0;                 // key blocks loaded so far
            int nqt[2] = {0, 0};       // Q tiles loaded so far, per tile
            bool ok = true;
            // tile x's Q buffer is free once the last score product of its previous item
            // has completed
            auto load_q = [&](int x, int bb, int row0) -> bool {
                const uint32_t ph = (uint32_t)nqt[x] & 1u;
                if (nqt[x] >= 1 && !ptx::mbar_wait(q_empty(x), ph ^ 1u, abort_flag, err, kErrProd)) return false;
                ptx::mbar_arrive_expect_tx(q_full(x), C::kQBytes);
                for (int kb = 0; kb < kDB; ++kb)
                    ptx::tma_load_3d(sQ(x) + kb * 16384u, &p.tq, kb * 64, row0, bb, q_full(x));
                q_armed |= 1u << x;
                q_par = (q_par & ~(1u << x)) | (ph << x);
                ++nqt[x];
                return true;
            };
            int gv = -1, vb = 0, vk0 = 0;  // the value block issued one key block behind
            auto load_v = [&]() -> bool {
                const int st = gv % SV;
                const uint32_t ph = (uint32_t)(gv / SV) & 1u;
                if (!ptx::mbar_wait(v_empty(st), ph ^ 1u, abort_flag, err, kErrProd)) return false;
                ptx::mbar_arrive_expect_tx(v_full(st), C::kVBytes);
                for (int kb = 0; kb < 2; ++kb)       // 64 keys per K-block of P V
                    for (int a = 0; a < kDB; ++a)    // 64 columns of d per swizzle atom
                        ptx::tma_load_3d(sV(st) + kb * (D * 128u) + a * 8192u, &p.tv, a * 64, vk0 + kb * 64, vb,
                                         v_full(st));
                v_armed |= 1u << st;
                v_par = (v_par & ~(1u << st)) | (ph << st);
                gv = -1;
                return true;
            };
            for (int n = 0; ok; ++n) {
                // take the next item: its ring slot is free once every role has read item n - kIR
                const int s = n % kIR;
                if (n >= kIR && !ptx::mbar_wait(i_empty(s), ((uint32_t)(n / kIR) & 1u) ^ 1u, abort_flag, err, kErrProd))
                    break;
                // the first item is the CTA's own index (no wait on the counter before the
                // first loads); the later ones come from the counter, which counts past the grid
                int it = -1;
                if (n == 0)
                    it = (int)blockIdx.x;
                else if (items > (int)gridDim.x)
                    it = (int)gridDim.x + (int)atomicAdd(&g_attn_sched[p.sched][0], 1u);
                if (it >= items) it = -1;
                item_ring[s] = it;
                ptx::mbar_arrive(i_full(s));  // (release: the index is visible to the waiters)
                if (it < 0) break;
                int bb, qq0, na, nb;
                decode(it, bb, qq0, na, nb);
                const int nmax = max(na, nb);
                if (nmax == 0) continue;
                // order: Q_A, the first key block, Q_B (tile B's previous item ends a block
                // later than tile A's), then the item's key and value blocks
                if (na > 0 && !load_q(0, bb, qq0)) break;
                for (int j = 0; j < nmax; ++j, ++g) {
                    const int st = g % SK;
                    const uint32_t ph = (uint32_t)(g / SK) & 1u;
                    if (!ptx::mbar_wait(k_empty(st), ph ^ 1u, abort_flag, err, kErrProd)) {
                        ok = false;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(k_full(st), C::kKBytes);
                    for (int kb = 0; kb < kDB; ++kb)
                        ptx::tma_load_3d(sK(st) + kb * 16384u, &p.tk, kb * 64, j * kKV, bb, k_full(st));
                    k_armed |= 1u << st;
                    k_par = (k_par & ~(1u << st)) | (ph << st);
                    if (j == 0 && nb > 0 && !load_q(1, bb, qq0 + kQ)) {
                        ok = false;
                        break;
                    }
                    if (gv >= 0 && !load_v()) {
                        ok = false;
                        break;
                    }
                    gv = g;
                    vb = bb;
                    vk0 = j * kKV;
                }
                if (ok && gv >= 0 && !load_v()) ok = false;  // the item's last value block
            }
            if (items > (int)gridDim.x) {
                // this CTA takes no more items; the last CTA to get here zeroes the counter
                // for the slot's next launch (every other CTA has taken its last item)
                unsigned* c = g_attn_sched[p.sched];
                __threadfence();
                if (atomicAdd(&c[1], 1u) == gridDim.x - 1) {
                    __threadfence();
                    atomicExch(&c[0], 0u);
                    atomicExch(&c[1], 0u);
                }
            }
            // drain: every copy issued here has landed before the CTA may exit
            volatile int no_abort = 0;
            for (int x = 0; x < 2; ++x)
                if (q_armed & (1u << x))
                    ptx::mbar_wait(q_full(x), (q_par >> x) & 1u, &no_abort, err, kErrDrain, ptx::kWaitLimitNs / 4);
            for (int st = 0; st < SK; ++st)
                if (k_armed & (1u << st))
                    ptx::mbar_wait(k_full(st), (k_par >> st) & 1u, &no_abort, err, kErrDrain, ptx::kWaitLimitNs / 4);
            for (int st = 0; st < SV; ++st)
                if (v_armed & (1u << st))
                    ptx::mbar_wait(v_full(st), (v_par >> st) & 1u, &no_abort, err, kErrDrain, ptx::kWaitLimitNs / 4);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        auto wait_all = [&](uint32_t b, uint32_t parity, int code) {
            return __all_sync(0xffffffffu, ptx::mbar_wait(b, parity, abort_flag, err, code));
        };
        constexpr uint32_t kIdescS = ptx::instr_desc(1u, false, kQ, kKV);
        constexpr uint32_t kIdescO = ptx::instr_desc(1u, true, kQ, D);
        // S_X = Q_X K^T of the key block in slot st into tile X's score columns
        auto issue_s = [&](int x, int st) {
            const uint32_t d_tmem = tmem + s_col(x);
#pragma unroll
            for (int kb = 0; kb < kDB; ++kb) {
                const uint64_t ad = ptx::smem_desc(sQ(x) + kb * 16384u, 16, 1024);
                const uint64_t bd = ptx::smem_desc(sK(st) + kb * 16384u, 16, 1024);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    ptx::mma_ss_elect<0>(d_tmem, ad + 2 * kk, bd + 2 * kk, kIdescS, (kb | kk) ? 1u : 0u);
            }
            ptx::tc_commit_elect(s_full(x));
        };
        // O_X += P_X V of the value block in slot st (P_X: bf16 pairs over S_X's columns)
        auto issue_pv = [&](int x, int st, bool acc) {
            const uint32_t o_tmem = tmem + o_col(x), p_tmem = tmem + s_col(x);
#pragma unroll
            for (int kb = 0; kb < 2; ++kb) {
                const uint64_t bd = ptx::smem_desc(sV(st) + kb * (D * 128u), 8192, 1024, ptx::kLayoutSw128);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)  // keys kb * 64 + kk * 16 .. + 15: 8 columns of P
                    ptx::mma_ts_f16_elect(o_tmem, p_tmem + kb * 32 + kk * 8, bd + 128 * kk, kIdescO,
                                          (acc || kb || kk) ? 1u : 0u);
            }
            ptx::tc_commit_elect(o_full(x));
        };
        int g = 0;
        int nqt[2] = {0, 0};  // Q tiles used so far, per tile
        int gx[2] = {0, 0};   // blocks of tile A / B so far (the parity of its barriers)
        bool ok = true;
        for (int ni = 0; ok; ++ni) {
            const int it = next_item(ni);
            if (it < 0) break;
            int bb, qq0, na, nb;
            decode(it, bb, qq0, na, nb);
            const int n[2] = {na, nb};
            const int nmax = max(na, nb);
            if (nmax == 0) continue;
            // block 0's score products, tile by tile as its Q tile lands
            if (!wait_all(k_full(g % SK), (uint32_t)((g / SK) & 1), kErrMmaKv)) break;
            for (int x = 0; x < 2 && ok; ++x) {
                if (n[x] == 0) continue;
                if (!wait_all(q_full(x), (uint32_t)nqt[x] & 1u, kErrMmaQ)) {
                    ok = false;
                    break;
                }
                ++nqt[x];
                ptx::tc_fence_after();
                issue_s(x, g % SK);
                if (n[x] == 1) ptx::tc_commit_elect(q_empty(x));  // the tile's only score product
            }
            if (!ok) break;
            ptx::tc_commit_elect(k_empty(g % SK));
            for (int j = 0; j < nmax; ++j, ++g) {
                const int sv = g % SV, sk1 = (g + 1) % SK;
                if (!wait_all(v_full(sv), (uint32_t)((g / SV) & 1), kErrMmaKv)) {
                    ok = false;
                    break;
                }
                const bool next = j + 1 < nmax;
                bool k_ready = false;  // key block j + 1 landed (waited for before its first use)
                for (int x = 0; x < 2 && ok; ++x) {
                    if (j >= n[x]) continue;
                    if (!wait_all(p_full(x), (uint32_t)gx[x] & 1u, kErrMmaP)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    issue_pv(x, sv, j > 0);
                    ++gx[x];
                    if (j + 1 < n[x]) {  // after P_X(j) V: the in-order pipe reads P_X(j) first
                        if (!k_ready && !wait_all(k_full(sk1), (uint32_t)(((g + 1) / SK) & 1), kErrMmaKv)) {
                            ok = false;
                            break;
                        }
                        k_ready = true;
                        ptx::tc_fence_after();
                        issue_s(x, sk1);
                        if (j + 2 == n[x]) ptx::tc_commit_elect(q_empty(x));  // the tile's last score product
                    }
                }
                if (!ok) break;
                ptx::tc_commit_elect(v_empty(sv));
                if (next) ptx::tc_commit_elect(k_empty(sk1));
            }
        }
        // every MMA issued here has completed before TMEM is freed
        __syncwarp();
        ptx::tc_commit_elect(drain_bar);
        volatile int no_abort = 0;
        ptx::mbar_wait(drain_bar, 0, &no_abort, err, kErrDrain, ptx::kWaitLimitNs / 4);
    } else {
        // ------------------------------------------------------------ softmax warps
        const int x = (warp - 2) >> 2;  // tile A (0) or B (1)
        const int q = warp & 3;         // TMEM lane quarter
        const int row = q * 32 + lane;  // row of the tile
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const uint32_t srow = tmem + lane_base + s_col(x), orow = tmem + lane_base + o_col(x);
        auto wait_warp = [&](uint32_t b, uint32_t parity, int code) {
            return __all_sync(0xffffffffu, ptx::mbar_wait(b, parity, abort_flag, err, code));
        };
        int gx = 0;  // this tile's blocks so far (the parity of its barriers)
        bool ok = true;
        for (int ni = 0; ok; ++ni) {
            const int it = next_item(ni);
            if (it < 0) break;
            int bb, qq0, na, nb;
            decode(it, bb, qq0, na, nb);
            if (max(na, nb) == 0) continue;
            const int nx = x ? nb : na;
            const int qrow = qq0 + x * kQ + row;
            const int last = p.causal ? qrow + shift : p.Lk - 1;  // last key this row sees
            // The output accumulates in TMEM; the row keeps its base m, a raw score
            // (p = 2^((s - m) c), c = scale log2(e)), until a block's maximum exceeds it by
            // more than 8 / c (p > 2^8), and only then is its TMEM row of O rescaled by
            // 2^((m_old - m_new) c).  s - m is formed first: the maximum gives exactly 1.
            float m = -INFINITY, l = 0.0f;
            const float c = p.scale_log2, rebase_gap = 8.0f / c;
            for (int j = 0; j < nx; ++j, ++gx) {
                if (!wait_warp(s_full(x), (uint32_t)gx & 1u, kErrSoftS)) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                // The row's 128 scores are read from TMEM twice, in 32-column pieces with the
                // next piece's load in flight while one is worked on (a few registers, no
                // spills): pass 1 takes the maximum of the raw scores, pass 2 computes p.
                uint32_t ra[32], rb[32];
                const int lim = min(last, p.Lk - 1) - j * kKV;  // columns 0..lim are visible
                float mxv[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                ptx::tmem_ld32(srow, ra);
                ptx::tmem_wait_ld(ra);
                // the branch is taken by the whole warp: the TMEM loads and stores in it are
                // warp-collective (.sync.aligned), and lim differs between rows
                if (__all_sync(0xffffffffu, lim >= kKV - 1)) {
#pragma unroll
                    for (int k = 0; k < kKV / 32; ++k) {
                        uint32_t(&cur)[32] = (k & 1) ? rb : ra;
                        uint32_t(&nxt)[32] = (k & 1) ? ra : rb;
                        if (k + 1 < kKV / 32) ptx::tmem_ld32(srow + 32u * (k + 1), nxt);
#pragma unroll
                        for (int i = 0; i < 32; i += 2)
                            mxv[(i >> 1) & 3] = max3(mxv[(i >> 1) & 3], __uint_as_float(cur[i]), __uint_as_float(cur[i + 1]));
                        if (k + 1 < kKV / 32) ptx::tmem_wait_ld(nxt);
                    }
                } else {
                    // a block on the mask's edge: masked scores become -inf, written back to
                    // TMEM (so that pass 2 reads p = 0 there) before the second read
                    const uint32_t ninf = __float_as_uint(-INFINITY);
#pragma unroll
                    for (int k = 0; k < kKV / 32; ++k) {
                        uint32_t(&cur)[32] = (k & 1) ? rb : ra;
                        uint32_t(&nxt)[32] = (k & 1) ? ra : rb;
                        if (k + 1 < kKV / 32) ptx::tmem_ld32(srow + 32u * (k + 1), nxt);
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (32 * k + i > lim) cur[i] = ninf;
#pragma unroll
                        for (int i = 0; i < 32; i += 2)
                            mxv[(i >> 1) & 3] = max3(mxv[(i >> 1) & 3], __uint_as_float(cur[i]), __uint_as_float(cur[i + 1]));
                        tmem_st32(srow + 32u * k, cur);
                        if (k + 1 < kKV / 32) ptx::tmem_wait_ld(nxt);
                    }
                    tmem_wait_st();
                }
                const float mx = fmaxf(fmaxf(mxv[0], mxv[1]), fmaxf(mxv[2], mxv[3]));
                const bool rebase = mx > m + rebase_gap;  // (always for the first visible key: m = -inf)
                float alpha = 1.0f;
                if (rebase) {
                    alpha = ex2((m - mx) * c);  // 0 while m = -inf
                    m = mx;
                    l *= alpha;
                }
                const float basev = m == -INFINITY ? 0.0f : m;  // no visible key yet: every p is 0
                // pass 2: p as bf16 pairs over the first 64 score columns (keys 2c, 2c + 1 in
                // column c), the A operand of P V.  Piece k's p go to columns 16k..16k+15, whose
                // scores were read before.
                uint64_t lv2[2] = {0ull, 0ull};
                const uint32_t cb = __float_as_uint(c), nb2u = __float_as_uint(-basev);
                const uint64_t c2 = f2(cb, cb), nb2 = f2(nb2u, nb2u);
                ptx::tmem_ld32(srow, ra);
                ptx::tmem_wait_ld(ra);
#pragma unroll
                for (int k = 0; k < kKV / 32; ++k) {
                    uint32_t(&cur)[32] = (k & 1) ? rb : ra;
                    uint32_t(&nxt)[32] = (k & 1) ? ra : rb;
                    if (k + 1 < kKV / 32) ptx::tmem_ld32(srow + 32u * (k + 1), nxt);
                    uint32_t pk[16];
#pragma unroll
                    for (int i = 0; i < 32; i += 2) {
                        uint32_t d0, d1;
                        f2_split(f2_mul(f2_add(f2(cur[i], cur[i + 1]), nb2), c2), d0, d1);
                        const float p0 = ex2(__uint_as_float(d0)), p1 = ex2(__uint_as_float(d1));
                        lv2[(i >> 1) & 1] = f2_add(lv2[(i >> 1) & 1], f2(__float_as_uint(p0), __float_as_uint(p1)));
                        pk[i >> 1] = pack_bf16(p0, p1);
                    }
                    tmem_st16(srow + 16u * k, pk);
                    if (k + 1 < kKV / 32) ptx::tmem_wait_ld(nxt);
                }
                {
                    uint32_t a0, a1, b0, b1;
                    f2_split(lv2[0], a0, a1);
                    f2_split(lv2[1], b0, b1);
                    l += (__uint_as_float(a0) + __uint_as_float(a1)) + (__uint_as_float(b0) + __uint_as_float(b1));
                }
                // O (the P V products of this item's earlier blocks) is complete in TMEM
                if (j >= 1) {
                    if (!wait_warp(o_full(x), (uint32_t)(gx - 1) & 1u, kErrSoftO)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    if (__any_sync(0xffffffffu, rebase)) {  // rescale the warp's rows of O
#pragma unroll
                        for (int c0 = 0; c0 < D; c0 += 32) {
                            uint32_t r[32];
                            ptx::tmem_ld32(orow + c0, r);
                            ptx::tmem_wait_ld(r);
#pragma unroll
                            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
                            tmem_st32(orow + c0, r);
                        }
                    }
                }
                tmem_wait_st();
                ptx::tc_fence_before();  // P_X(j) and the rescaled O are stored before P V runs
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(p_full(x));
            }
            if (!ok) break;
            // the item's output: O from TMEM once its last P V product has completed
            const bool have_o = nx > 0;
            if (have_o) {
                if (!wait_warp(o_full(x), (uint32_t)(gx - 1) & 1u, kErrSoftO)) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
            }
            const float inv = (have_o && l > 0.0f) ? 1.0f / l : 0.0f;
            // 32 x 16 pieces of the warp's rows, staged alternately in the two 2 KB halves of
            // the warp's buffer with the 64-byte swizzle (16-byte chunk c of row r at
            // c ^ (r / 2 % 4)) and stored by TMA, which leaves rows past Lq unwritten: a store
            // may still be reading one half while the warp fills the other
            // (the row's D output columns come from TMEM in one round trip first)
            const uint32_t stage = sO + (uint32_t)(warp - 2) * C::kOStage;
            uint32_t ro[D];
            if (have_o) {
#pragma unroll
                for (int c0 = 0; c0 < D; c0 += 32)
                    ptx::tmem_ld32(orow + c0, *reinterpret_cast<uint32_t(*)[32]>(ro + c0));
#pragma unroll
                for (int c0 = 0; c0 < D; c0 += 32) ptx::tmem_wait_ld(*reinterpret_cast<uint32_t(*)[32]>(ro + c0));
            } else {
#pragma unroll
                for (int i = 0; i < D; ++i) ro[i] = 0u;
            }
#pragma unroll
            for (int c0 = 0; c0 < D; c0 += 16) {
                const uint32_t* r = ro + c0;
                const uint32_t buf = stage + (uint32_t)((c0 / 16) & 1) * 2048u;
                if (lane == 0) ptx::bulk_wait_read<1>();  // the store before last (this half) has read it
                __syncwarp();
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    st_shared_f4(buf + (uint32_t)lane * 64u + ((uint32_t)(c ^ ((lane >> 1) & 3)) << 4),
                                 __uint_as_float(r[4 * c]) * inv, __uint_as_float(r[4 * c + 1]) * inv,
                                 __uint_as_float(r[4 * c + 2]) * inv, __uint_as_float(r[4 * c + 3]) * inv);
                ptx::fence_proxy_async_smem();  // the piece is read by the TMA (async proxy)
                __syncwarp();
                if (lane == 0) {
                    ptx::tma_store_3d(&p.to16, buf, c0, qq0 + x * kQ + q * 32, bb);
                    ptx::bulk_commit();
                }
            }
            ptx::tc_fence_before();  // the next item's first P V overwrites O
        }
        if (lane == 0) ptx::bulk_wait_all();  // every output store has completed
        __syncwarp();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, 512);
}

}  // namespace

cudaError_t attention_watchdog_take(int* word) {
    cudaError_t e = cudaMemcpyFromSymbol(word, g_attn_watchdog, sizeof(int));
    if (e != cudaSuccess || *word == 0) return e;
    const int zero = 0;
    return cudaMemcpyToSymbol(g_attn_watchdog, &zero, sizeof(int));
}

cudaError_t launch_attention_tc(const nnjit_attention_desc& d, const void* Q, const void* K, const void* V,
                                float* O, cudaStream_t stream, bool two_tiles) {
    const int item_q = two_tiles ? 2 * kQ : kQ;  // queries per work item
    const int qblocks = (int)((d.Lq + item_q - 1) / item_q);
    const long long ctas = (long long)qblocks * d.batch;
    if (ctas <= 0) return cudaSuccess;
    if (ctas >= (1LL << 31)) return cudaErrorInvalidValue;
    if (d.Lk == 0) return cudaMemsetAsync(O, 0, (size_t)d.batch * d.Lq * d.d * sizeof(float), stream);
    EncodeTiledFn enc = get_encode_fn();
    if (!enc) return cudaErrorNotSupported;
    Params p;
    const cuuint32_t estr[3] = {1, 1, 1};
    auto encode = [&](CUtensorMap* m, const void* ptr, long long rows, cuuint32_t box_rows) {
        const cuuint64_t dims[3] = {(cuuint64_t)d.d, (cuuint64_t)rows, (cuuint64_t)d.batch};
        const cuuint64_t strides[2] = {(cuuint64_t)(d.d * 2), (cuuint64_t)(rows * d.d * 2)};
        const cuuint32_t box[3] = {64, box_rows, 1};
        return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
    };
    if (!encode(&p.tq, Q, d.Lq, kQ) || !encode(&p.tk, K, d.Lk, kKV) || !encode(&p.tv, V, d.Lk, 64))
        return cudaErrorInvalidValue;
    {  // O: f32 [batch, Lq, d], stored in 32 x 32 tiles (128-byte rows, 128-byte swizzle)
        const cuuint64_t dims[3] = {(cuuint64_t)d.d, (cuuint64_t)d.Lq, (cuuint64_t)d.batch};
        const cuuint64_t strides[2] = {(cuuint64_t)(d.d * 4), (cuuint64_t)(d.Lq * d.d * 4)};
        const cuuint32_t box[3] = {32, 32, 1};
        if (enc(&p.to, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, O, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        const cuuint32_t box16[3] = {16, 32, 1};
        if (enc(&p.to16, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, O, dims, strides, box16, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    p.O = O;
    p.Lq = (int)d.Lq;
    p.Lk = (int)d.Lk;
    p.causal = d.causal;
    p.qblocks = qblocks;
    p.batch = (int)d.batch;
    // item groups: halve the group (while it divides the batch) until one group's Q, K, V
    // (bf16) and O (f32) take at most kGroupL2Bytes
    const long long per_problem = (long long)d.Lq * d.d * (2 + 4) + 2LL * d.Lk * d.d * 2;
    long long group = d.batch;
    while (group % 2 == 0 && group * per_problem > kGroupL2Bytes) group /= 2;
    p.group = (int)group;
    p.scale_log2 = d.scale * 1.4426950408889634f;
    static std::atomic<unsigned> next_sched{0};
    p.sched = two_tiles ? (int)(next_sched.fetch_add(1u) % kSchedSlots) : 0;
    // persistent: one CTA per SM (the CTA holds all of the SM's tensor memory)
    const int sms = current_sm_count();
    const unsigned grid = (unsigned)std::min<long long>(ctas, sms);
    void (*kern)(Params);
    int smem, threads;
    if (two_tiles) {
        kern = d.d == 64 ? attention_tc2_kernel<64> : attention_tc2_kernel<128>;
        smem = d.d == 64 ? (int)Cfg2<64>::kSmem : (int)Cfg2<128>::kSmem;
        threads = 320;
    } else {
        kern = d.d == 64 ? attention_tc_kernel<64> : attention_tc_kernel<128>;
        smem = d.d == 64 ? (int)Cfg<64>::kSmem : (int)Cfg<128>::kSmem;
        threads = d.d == 64 ? threads_of<64>() : threads_of<128>();
    }
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(kern), smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(grid), dim3(threads), (size_t)smem, stream, p);
}

}  // namespace nnjit
