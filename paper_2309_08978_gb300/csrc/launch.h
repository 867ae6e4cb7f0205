// Internal interface between the C-ABI layer (capi.cu) and the kernel translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <utility>

#include "space.h"

namespace nnjit {

// Launch `kernel` with programmatic stream serialization (PDL): the kernel may begin
// while the previous kernel in the stream finishes; every kernel of this library calls
// griddepcontrol.wait before it touches global memory.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Everything one launch of the plan's main kernel needs.
struct LaunchArgs {
    const Problem* p = nullptr;
    const nnjit_candidate* c = nullptr;
    const void* A = nullptr;
    const void* B = nullptr;
    const float* bias = nullptr;   // NULL: no bias
    float* C = nullptr;
    float* ws = nullptr;           // split-K partials [split][batch][M][N], or NULL if split == 1
    int* err = nullptr;            // device watchdog word
    cudaStream_t stream = nullptr;
    const CUtensorMap* tmap_a = nullptr;  // TC family only
    const CUtensorMap* tmap_b = nullptr;
    const CUtensorMap* tmap_c = nullptr;  // TC output map (C, or partials when split > 1);
                                          // NULL: the epilogue stores directly
};

// Main kernels.  Each returns the launch status (cudaGetLastError after the launch).
cudaError_t launch_ffma(const LaunchArgs& a);
cudaError_t launch_gemv(const LaunchArgs& a);
cudaError_t launch_tc(const LaunchArgs& a);
// CTA-pair (cta_group::2) tensor-core instances kTcPairFirstInstance.. (bf16, tf32).  A
// stream-K candidate (reduce 2) takes its flags and partial sums from LaunchArgs::ws.
cudaError_t launch_tc_pair(const LaunchArgs& a);
// Workspace of a stream-K pair candidate over `pairs` pairs: 2 CTAs x 4 warps of flags
// per pair (padded to 256 bytes in all), then one 256 x 256 f32 partial tile per pair.
// The flags must be zero before the first launch; every launch that completes leaves
// them zero.
inline int64_t tc2_sk_flag_floats(int64_t pairs) { return (pairs * 8 + 63) / 64 * 64; }
inline int64_t tc2_sk_ws_bytes(int64_t pairs) { return (tc2_sk_flag_floats(pairs) + pairs * 256 * 256) * 4; }

// C[b,m,n] = sum_{s < split} ws[s][b][m][n] (+ bias[n]), s ascending.
cudaError_t launch_splitk_reduce(const float* ws, int split, const Problem& p, const float* bias,
                                 float* C, cudaStream_t s);

// C = bias broadcast over rows (or 0 when bias is NULL): the K = 0 product.
cudaError_t launch_fill_bias(const Problem& p, const float* bias, float* C, cudaStream_t s);

// Arbitrary finite data for tuning scratch buffers (not the test inputs).
cudaError_t launch_fill_scratch(void* dst, int64_t n_elems, int elem_bytes, uint32_t seed,
                                cudaStream_t s);

// Write `bytes` of `buf` (evicts the L2 between timed repetitions).
cudaError_t launch_l2_flush(void* buf, int64_t bytes, cudaStream_t s);

// Opt-in dynamic shared memory of `func` on the current device.  The attribute belongs to
// a device's context, so the sizes already set are recorded per (device, function):
// cudaFuncSetAttribute runs the first time a device needs a size beyond the default or
// beyond what was set there before.  Thread-safe; idempotent.
cudaError_t ensure_dynamic_smem(const void* func, int smem_bytes);
// Number of SMs of the current device (looked up once per device).
int current_sm_count();

// Kernel attribute setup of one instance on the current device (ensure_dynamic_smem).
cudaError_t prepare_tc_instance(int instance, int smem_bytes);
cudaError_t prepare_gemv_instance(int instance, int smem_bytes);

// Output tensor map for the TC epilogue's TMA stores: C (partials = false) or the split-K
// partials buffer.  *ok is false when the output's alignment or strides rule TMA out.
cudaError_t encode_tc_output_map(const Problem& p, const nnjit_candidate& c, float* out,
                                 bool partials, CUtensorMap* tc_map, bool* ok);

// Detail string for nnjit_last_error() (defined with the C ABI).
void set_last_error(const char* msg);

// Driver entry point for cuTensorMapEncodeTiled, fetched through the runtime so the
// library does not link against libcuda (NULL if unavailable).
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn get_encode_fn();

// GEMV candidates whose weights are streamed by TMA (instances kGemvTmaFirstInstance..+5).
bool gemv_uses_tma(const nnjit_candidate& c);
cudaError_t launch_gemv_tma(const LaunchArgs& a);
// GEMV candidates over 4-bit weights (instances kGemvW4FirstInstance..+1); LaunchArgs'
// tmap_a, tmap_b, tmap_c are the maps of x, the codes and the group scales.
bool gemv_uses_w4(const nnjit_candidate& c);
cudaError_t launch_gemv_w4(const LaunchArgs& a);
cudaError_t encode_gemv_w4_maps(const Problem& p, const nnjit_candidate& c, const void* A, const void* B,
                                CUtensorMap* tx, CUtensorMap* tw, CUtensorMap* ts, const char** why);
// Tensor maps of x (*tx, from A) and the weights (*tw, from B) for a TMA GEMV candidate.
cudaError_t encode_gemv_tensor_maps(const Problem& p, const nnjit_candidate& c, const void* A,
                                    const void* B, CUtensorMap* tx, CUtensorMap* tw,
                                    const char** why);

// Tensor maps for the TC family (host; uses the driver entry point).
cudaError_t encode_tc_tensor_maps(const Problem& p, const nnjit_candidate& c, const void* A,
                                  const void* B, CUtensorMap* ta, CUtensorMap* tb,
                                  const char** why);

// Fused attention (nnjit_attention); the descriptor is validated by the caller.  The
// warp-level MMA kernel, and the tensor-memory kernel with its watchdog word.
cudaError_t launch_attention(const nnjit_attention_desc& d, const void* Q, const void* K, const void* V,
                             float* O, cudaStream_t stream);
// two_tiles: 256-query items of two 128-row tiles sharing the key and value blocks (kernel
// NNJIT_ATTN_TCGEN05_2T); else 128-query items (NNJIT_ATTN_TCGEN05).
cudaError_t launch_attention_tc(const nnjit_attention_desc& d, const void* Q, const void* K, const void* V,
                                float* O, cudaStream_t stream, bool two_tiles = false);
// Read and clear the tensor-memory kernel's watchdog word (synchronous).
cudaError_t attention_watchdog_take(int* word);

}  // namespace nnjit
