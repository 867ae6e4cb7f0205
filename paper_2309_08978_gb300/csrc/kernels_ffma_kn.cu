// FP32-FFMA GEMM instances with B stored [K][N]: the 12 (thread tile, block tile)
// pairs of the lite space (BK = 16), in the order of ffma_instance().
#include "ffma.cuh"

namespace nnjit {

using FfmaKernel = void (*)(FfmaParams);

#define NNJIT_FFMA_PAIR(TM, BM, BN) ffma_gemm_kernel<BM, BN, 16, TM, TM, false>

static const FfmaKernel kFfma_kn[12] = {
    NNJIT_FFMA_PAIR(4, 32, 32),  NNJIT_FFMA_PAIR(4, 32, 64),  NNJIT_FFMA_PAIR(4, 32, 128),
    NNJIT_FFMA_PAIR(4, 64, 32),  NNJIT_FFMA_PAIR(4, 64, 64),  NNJIT_FFMA_PAIR(4, 128, 32),
    NNJIT_FFMA_PAIR(8, 32, 128), NNJIT_FFMA_PAIR(8, 64, 64),  NNJIT_FFMA_PAIR(8, 64, 128),
    NNJIT_FFMA_PAIR(8, 128, 32), NNJIT_FFMA_PAIR(8, 128, 64), NNJIT_FFMA_PAIR(8, 128, 128),
};

FfmaKernel ffma_kernel_kn(int i) { return (i >= 0 && i < 12) ? kFfma_kn[i] : nullptr; }

}  // namespace nnjit
