// laq_gemm_prologue.cu -- the GEMM kernel instances whose X staging applies a fused prologue
// (RMSNorm of the residual sum, or SiLU(gate) * up), compiled apart from the plain instances so
// the two sets build in parallel.
#include "laq_gemm_kernel.cuh"

namespace laq {

const void* gemm_prologue_kernel(int bits, int mp, int nt) {
    return bits == 4 ? pick_mp<4, true>(mp, nt) : pick_mp<3, true>(mp, nt);
}

}  // namespace laq
