// laq_internal.cuh -- declarations shared by the library's translation units (not installed).
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace laq {

cudaError_t launch_quantize_rtn(const uint16_t* W, int64_t K, int64_t N, int bits,
                                uint8_t* codes, uint16_t* s, uint8_t* z, cudaStream_t stream);
cudaError_t launch_pack(const uint8_t* codes, int64_t K, int64_t N, int bits, uint32_t* packed,
                        cudaStream_t stream);
cudaError_t launch_unpack(const uint32_t* packed, int64_t K, int64_t N, int bits, uint8_t* codes,
                          cudaStream_t stream);

// One GEMM launch, fully resolved on the host.
struct GemmLaunch {
    const uint16_t* X;
    const uint8_t* packed;
    const uint16_t* s;
    const uint8_t* z;
    uint16_t* Y;
    int M, K, N, bits;
    int tiles_per_cta, warps, cluster, stages, pdl;
    // X prologue (kPro*): the GEMV's input is RMSNorm(X + R) * w, or SiLU(gate) * up of X
    int pro = 0;
    float eps = 0.f;
    const uint16_t* R = nullptr;
    uint16_t* R_out = nullptr;
    const uint16_t* w = nullptr;
};
constexpr int kProNone = 0, kProRmsNorm = 1, kProSiluMul = 2;

// Staged X in the GEMM's shared memory, in 16-byte chunks (chunk j holds x[8j .. 8j+7]).  For
// M <= 2 (MP <= 2) chunk j of group lg of batch row b sits at b * 16 gpp + 16 lg + j; at most 4
// lanes of a load phase read X then.  For MP >= 4, where 8 lanes of a phase read 4 chunk columns
// of 2 batch rows, the chunk sits at b * xs_row_chunks + 17 lg + j + j / 8: the pad between a
// group's halves and a row stride of 2 mod 8 chunks put those 8 lanes on 8 different bank slots.
__host__ __device__ constexpr bool xs_padded(int mp) { return mp >= 4; }
__host__ __device__ constexpr int xs_group_chunks(int mp) { return xs_padded(mp) ? 17 : 16; }
__host__ __device__ constexpr int xs_row_chunks(int gpp, int mp) {
    return xs_padded(mp) ? gpp * 17 + (((2 - gpp * 17) % 8) + 8) % 8 : gpp * 16;
}

// Dynamic shared memory the GEMM kernel needs for this launch (bytes), and the groups of X it
// stages per phase.
size_t gemm_smem_bytes(const GemmLaunch& L, int* groups_per_phase);
cudaError_t launch_gemm(const GemmLaunch& L, size_t smem_limit, cudaStream_t stream);

// One persistent launch of a GEMV chain, fully resolved on the host.
constexpr int kChainMax = 384;  // = LAQ_CHAIN_MAX
struct ChainEntry {
    const uint16_t* X;
    const uint8_t* packed;
    const uint16_t* s;
    const uint8_t* z;
    uint16_t* Y;
    int K, N;
    int xoff;   // X offset in the stage's shared X area, 16-byte units
    int psoff;  // offset in the stage's (S, P) table, one per (row, group)
};
struct ChainStage {
    int e0, ne, records;
    int split;  // CTA shares by records (tiles may straddle CTAs) instead of whole tiles
};
// Chain workspace bytes for `count` entries (counters, per-CTA flags and published parts for
// grids of up to 256 CTAs), and the leading bytes that must be zero before a launch.
size_t chain_workspace_bytes(int count);
size_t chain_workspace_zeroed_bytes(int count);
struct ChainLaunch {
    const ChainEntry* e;
    const ChainStage* st;
    int count, nstages, M, bits, xs_bytes;
    uint32_t* ws;
};
// Dynamic shared memory of the chain kernel (its ring depth is fixed per bit width).
size_t chain_smem_bytes(int bits, int M, int xs_bytes, int nstages, int count);
cudaError_t launch_chain(const ChainLaunch& L, int num_sms, cudaStream_t stream);

}  // namespace laq
