// Fused attention (nnjit_attention): O = softmax(scale Q K^T) V per batch x head, the two
// attention BatchMatMuls of Table 3 (K2, K3) with the softmax between them, without
// writing the scores.
//
// One CTA takes 64 queries of one problem; its 4 warps own 16 query rows each.  The key
// and value blocks (64 rows x d) stream through a two-slot shared-memory ring
// (cp.async, 16-byte chunks, chunk c of row r stored at c ^ (r % 8) so that ldmatrix
// reads are conflict-free).  Per block, on warp-level tensor-core MMAs (m16n8k16, bf16 x
// bf16 -> f32):
//   S = Q K^T                (Q fragments kept in registers, K via ldmatrix)
//   online softmax in base 2 (row maxima across the 4 lanes that share a row; the
//                             running output and row sums rescaled by 2^(m_old - m_new))
//   O += P V                 (P re-packed from the S accumulators straight into A
//                             fragments: the accumulator layout of an m16n8 tile pair is
//                             the A layout of an m16k16 tile; V via ldmatrix.trans)
// P is rounded to bf16 for the second product.  Keys past Lk and, with the causal mask,
// keys past i + (Lk - Lq) score -inf; blocks a CTA cannot see are skipped.  The output is
// O / (row sum), 0 for a query that sees no key.
#include <cuda_runtime.h>


#include <cmath>
#include <cstdint>

#include "../../include/nnjit.h"
#include "launch.h"

namespace nnjit {

namespace {

constexpr int kBQ = 64;    // queries per CTA
constexpr int kBKV = 64;   // keys per block
constexpr int kWarps = 4;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// 16-byte async copy global -> shared; src_bytes = 0 fills zeros (no global read).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// 2^x (the PTX approximate base-2 exponential; 2^-inf = 0)
__device__ __forceinline__ float exp2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

struct AttnParams {
    const uint16_t* Q;
    const uint16_t* K;
    const uint16_t* V;
    float* O;
    int Lq, Lk, causal, qblocks;
    float scale_log2;  // scale * log2(e)
};

// Shared-memory byte offset of 16-byte chunk c of row r of a [rows][D] bf16 tile.
template <int D>
__device__ __forceinline__ uint32_t swz(int r, int c) {
    return (uint32_t)(r * (D * 2) + ((c ^ (r & 7)) << 4));
}

// Copy rows [row0, row0 + 64) of a [L][D] bf16 matrix into a swizzled tile; rows past L
// are zero-filled.
template <int D>
__device__ __forceinline__ void load_tile(uint32_t tile, const uint16_t* src, int row0, int L) {
    constexpr int kChunks = D / 8;  // 16-byte chunks per row
    for (int i = threadIdx.x; i < 64 * kChunks; i += kWarps * 32) {
        const int r = i / kChunks, c = i % kChunks;
        const int gr = row0 + r;
        const bool in = gr < L;
        const uint16_t* g = src + (size_t)(in ? gr : 0) * D + c * 8;
        cp_async16(tile + swz<D>(r, c), g, in ? 16 : 0);
    }
}

template <int D>
__global__ void __launch_bounds__(kWarps * 32) attention_kernel(const AttnParams p) {
    extern __shared__ __align__(128) uint8_t sm[];
    constexpr int kTile = 64 * D * 2;  // bytes of one 64-row tile
    const uint32_t sQ = smem_u32(sm);
    const uint32_t sK0 = sQ + kTile, sV0 = sQ + 3 * kTile;  // K slots at 1, 2; V slots at 3, 4
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, t = lane & 3;
    // consecutive CTAs take the query blocks of one problem (they share its K and V in L2)
    const int b = (int)(blockIdx.x / p.qblocks);
    const int q0 = (int)(blockIdx.x % p.qblocks) * kBQ;
    const uint16_t* Qb = p.Q + (size_t)b * p.Lq * D;
    const uint16_t* Kb = p.K + (size_t)b * p.Lk * D;
    const uint16_t* Vb = p.V + (size_t)b * p.Lk * D;
    float* Ob = p.O + (size_t)b * p.Lq * D;

    // keys this CTA can see: [0, kv_end)
    const int shift = p.Lk - p.Lq;
    int kv_end = p.Lk;
    if (p.causal) kv_end = min(p.Lk, max(0, min(q0 + kBQ, p.Lq) - 1 + shift + 1));
    const int nblocks = (kv_end + kBKV - 1) / kBKV;

    load_tile<D>(sQ, Qb, q0, p.Lq);
    if (nblocks > 0) {
        load_tile<D>(sK0, Kb, 0, p.Lk);
        load_tile<D>(sV0, Vb, 0, p.Lk);
    }
    cp_async_commit();

    constexpr int kK = D / 16;  // k-steps of S = Q K^T
    constexpr int kN = D / 8;   // n-tiles of O
    uint32_t qf[kK][4];
    float o[kN][4];
#pragma unroll
    for (int n = 0; n < kN; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.0f;
    float m0 = -INFINITY, m1 = -INFINITY;  // running maxima of rows g and g + 8 (base-2 units)
    float l0 = 0.0f, l1 = 0.0f;            // this lane's part of the running row sums
    const int qr0 = q0 + warp * 16 + g, qr1 = qr0 + 8;  // the two query rows of this lane

    for (int blk = 0; blk < nblocks; ++blk) {
        const int slot = blk & 1;
        if (blk + 1 < nblocks) {
            load_tile<D>(sK0 + (slot ^ 1) * kTile, Kb, (blk + 1) * kBKV, p.Lk);
            load_tile<D>(sV0 + (slot ^ 1) * kTile, Vb, (blk + 1) * kBKV, p.Lk);
        }
        cp_async_commit();
        cp_async_wait<1>();  // everything but the group just issued has landed
        __syncthreads();
        if (blk == 0) {
            // Q fragments (A of m16k16): lane l addresses row l % 16, chunk 2kk + l / 16
#pragma unroll
            for (int kk = 0; kk < kK; ++kk)
                ldsm_x4(sQ + swz<D>(warp * 16 + (lane & 15), 2 * kk + (lane >> 4)), qf[kk][0], qf[kk][1],
                        qf[kk][2], qf[kk][3]);
        }
        const uint32_t sK = sK0 + slot * kTile, sV = sV0 + slot * kTile;
        // ---- S = Q K^T for this warp's 16 rows x 64 keys
        float s[8][4];
#pragma unroll
        for (int n = 0; n < 8; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.0f;
#pragma unroll
        for (int kk = 0; kk < kK; ++kk) {
#pragma unroll
            for (int np = 0; np < 4; ++np) {  // key tiles 2np, 2np + 1
                // lanes 0-7: keys of tile 2np, chunk 2kk; 8-15: same keys, chunk 2kk + 1;
                // 16-23 / 24-31: tile 2np + 1
                const int key = np * 16 + ((lane >> 4) << 3) + (lane & 7);
                const int ch = 2 * kk + ((lane >> 3) & 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4(sK + swz<D>(key, ch), b0, b1, b2, b3);
                mma16816(s[2 * np], qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], b0, b1);
                mma16816(s[2 * np + 1], qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], b2, b3);
            }
        }
        // ---- masks, online softmax (base 2)
        const int kbase = blk * kBKV;
        const int last0 = p.causal ? qr0 + shift : p.Lk - 1;  // last key row g may see
        const int last1 = p.causal ? qr1 + shift : p.Lk - 1;
        float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
        for (int n = 0; n < 8; ++n) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int key = kbase + 8 * n + 2 * t + e;
                const bool ok0 = key <= last0 && key < p.Lk, ok1 = key <= last1 && key < p.Lk;
                s[n][e] = ok0 ? s[n][e] * p.scale_log2 : -INFINITY;
                s[n][2 + e] = ok1 ? s[n][2 + e] * p.scale_log2 : -INFINITY;
                mx0 = fmaxf(mx0, s[n][e]);
                mx1 = fmaxf(mx1, s[n][2 + e]);
            }
        }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        // a row with no visible key so far keeps m = -inf: use 0 as its base (all p = 0)
        const float base0 = mn0 == -INFINITY ? 0.0f : mn0, base1 = mn1 == -INFINITY ? 0.0f : mn1;
        const float alpha0 = exp2_approx(m0 - base0), alpha1 = exp2_approx(m1 - base1);
        m0 = mn0;
        m1 = mn1;
        l0 *= alpha0;
        l1 *= alpha1;
#pragma unroll
        for (int n = 0; n < kN; ++n) {
            o[n][0] *= alpha0; o[n][1] *= alpha0;
            o[n][2] *= alpha1; o[n][3] *= alpha1;
        }
        uint32_t pa[4][4];  // P as A fragments, 4 k-steps of 16 keys
#pragma unroll
        for (int n = 0; n < 8; ++n) {
            const float p0 = exp2_approx(s[n][0] - base0), p1 = exp2_approx(s[n][1] - base0);
            const float p2 = exp2_approx(s[n][2] - base1), p3 = exp2_approx(s[n][3] - base1);
            l0 += p0 + p1;
            l1 += p2 + p3;
            // key tile n = 2kk + h: h = 0 -> a0 (row g) / a1 (row g + 8); h = 1 -> a2 / a3
            pa[n >> 1][(n & 1) * 2 + 0] = pack_bf16(p0, p1);
            pa[n >> 1][(n & 1) * 2 + 1] = pack_bf16(p2, p3);
        }
        // ---- O += P V
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
            for (int np = 0; np < kN / 2; ++np) {  // output tiles 2np, 2np + 1 (d columns)
                // lanes 0-7: keys 16kk + 0..7 at chunk 2np; 8-15: keys + 8..15, same chunk;
                // 16-23 / 24-31: chunk 2np + 1
                const int key = kk * 16 + ((lane >> 3) & 1) * 8 + (lane & 7);
                const int ch = 2 * np + (lane >> 4);
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(sV + swz<D>(key, ch), b0, b1, b2, b3);
                mma16816(o[2 * np], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], b0, b1);
                mma16816(o[2 * np + 1], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], b2, b3);
            }
        }
        __syncthreads();  // the slot is refilled by the next iteration's copies
    }
    cp_async_wait<0>();
    // ---- O / row sum
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    const float r0 = l0 > 0.0f ? 1.0f / l0 : 0.0f, r1 = l1 > 0.0f ? 1.0f / l1 : 0.0f;
#pragma unroll
    for (int n = 0; n < kN; ++n) {
        const int c = 8 * n + 2 * t;
        if (qr0 < p.Lq)
            *reinterpret_cast<float2*>(Ob + (size_t)qr0 * D + c) = make_float2(o[n][0] * r0, o[n][1] * r0);
        if (qr1 < p.Lq)
            *reinterpret_cast<float2*>(Ob + (size_t)qr1 * D + c) = make_float2(o[n][2] * r1, o[n][3] * r1);
    }
}

}  // namespace

cudaError_t launch_attention(const nnjit_attention_desc& d, const void* Q, const void* K, const void* V,
                             float* O, cudaStream_t stream) {
    AttnParams p;
    p.Q = static_cast<const uint16_t*>(Q);
    p.K = static_cast<const uint16_t*>(K);
    p.V = static_cast<const uint16_t*>(V);
    p.O = O;
    p.Lq = (int)d.Lq;
    p.Lk = (int)d.Lk;
    p.causal = d.causal;
    p.scale_log2 = d.scale * 1.4426950408889634f;
    p.qblocks = (int)((d.Lq + kBQ - 1) / kBQ);
    const long long ctas = (long long)p.qblocks * d.batch;
    if (ctas <= 0) return cudaSuccess;
    if (ctas >= (1LL << 31)) return cudaErrorInvalidValue;
    const int smem = 5 * 64 * (int)d.d * 2;  // Q tile + two K and two V slots
    const int i = d.d == 64 ? 0 : 1;
    cudaError_t e = ensure_dynamic_smem(
        i == 0 ? reinterpret_cast<const void*>(attention_kernel<64>) : reinterpret_cast<const void*>(attention_kernel<128>),
        smem);
    if (e != cudaSuccess) return e;
    if (i == 0)
        attention_kernel<64><<<(unsigned)ctas, kWarps * 32, smem, stream>>>(p);
    else
        attention_kernel<128><<<(unsigned)ctas, kWarps * 32, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace nnjit
