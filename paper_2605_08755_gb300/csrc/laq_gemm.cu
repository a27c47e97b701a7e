// laq_gemm.cu -- launch of the dequantize-fused GEMM (kernel template in laq_gemm_kernel.cuh):
// shared-memory sizing, kernel choice, launch attributes; and the plain-X kernel instances.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "laq_gemm_kernel.cuh"

namespace laq {

namespace {

int mp_class(int M) { return M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : M <= 8 ? 8 : 16; }
int mp_index(int mp) { return mp == 1 ? 0 : mp == 2 ? 1 : mp == 4 ? 2 : mp == 8 ? 3 : 4; }
int nt_index(int nt) { return nt == 1 ? 0 : nt == 2 ? 1 : nt == 4 ? 2 : 3; }

std::atomic<size_t> g_attr_limit[2][2][5][4];  // max dynamic smem granted per kernel instance

constexpr size_t kXsBudget = 64 * 1024;  // shared memory for staged X (and its tables) per phase

}  // namespace

size_t gemm_smem_bytes(const GemmLaunch& L, int* groups_per_phase) {
    const size_t rec = L.bits == 4 ? 1024 : 768;
    const size_t ring = (size_t)L.warps * L.stages * rec;
    const int G = L.K / 128;
    const int gc = (G + L.cluster - 1) / L.cluster;
    // staged X (xs_row_chunks) and (S, P) of one group, and the zero block of the unpadded form
    const int mp = mp_class(L.M);
    const size_t per_group = (size_t)L.M * (xs_group_chunks(mp) * 16 + 8);
    int gpp = (int)(kXsBudget / per_group);
    if (gpp > gc) gpp = gc;
    if (gpp < 1) gpp = 1;
    if (groups_per_phase) *groups_per_phase = gpp;
    const size_t xs = (size_t)L.M * xs_row_chunks(gpp, mp) * 16 + (size_t)L.M * gpp * 8 +
                      (xs_padded(mp) ? 0 : 64);
    const size_t sz = (size_t)(gc > 0 ? gc : 1) * L.tiles_per_cta * 48;  // s (32 B) + z (16 B)
    const size_t pro = L.pro != kProNone ? 128 : 0;  // inv_rms [16] + warp sums [16], fp32
    return ring + xs + sz + (size_t)L.tiles_per_cta * mp * 16 * 4 + pro;
}

cudaError_t launch_gemm(const GemmLaunch& L, size_t smem_limit, cudaStream_t stream) {
    int gpp = 1;
    const size_t smem = gemm_smem_bytes(L, &gpp);
    if (smem > smem_limit) return cudaErrorInvalidConfiguration;
    const int mp = mp_class(L.M);
    const bool pro = L.pro != kProNone;
    const void* fn = pro ? gemm_prologue_kernel(L.bits, mp, L.tiles_per_cta)
                   : L.bits == 4 ? pick_mp<4, false>(mp, L.tiles_per_cta)
                                 : pick_mp<3, false>(mp, L.tiles_per_cta);
    std::atomic<size_t>& granted =
        g_attr_limit[pro][L.bits == 4][mp_index(mp)][nt_index(L.tiles_per_cta)];
    if (granted.load() < smem) {
        // Every instance asks for the largest shared-memory carveout, so kernels of different
        // shapes following each other in a decode step never reconfigure L1 / shared memory.
        cudaError_t e = cudaFuncSetAttribute(
            fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_limit);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(fn,
                                 cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        granted.store(smem_limit);
    }
    Params prm;
    prm.pro = L.pro;
    prm.eps = L.eps;
    prm.R = L.R;
    prm.R_out = L.R_out;
    prm.w = L.w;
    prm.X = L.X;
    prm.packed = L.packed;
    prm.s = L.s;
    prm.z = L.z;
    prm.Y = L.Y;
    prm.M = L.M;
    prm.K = L.K;
    prm.N = L.N;
    prm.G = L.K / 128;
    prm.T = L.N / 16;
    prm.stages = L.stages;
    prm.gpp = gpp;
    prm.gc = (prm.G + L.cluster - 1) / L.cluster;
    prm.exps = exps_for(L.bits);

    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((prm.T + L.tiles_per_cta - 1) / L.tiles_per_cta),
                       (unsigned)L.cluster, 1);
    cfg.blockDim = dim3((unsigned)(L.warps * 32), 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attrs[2];
    int na = 0;
    if (L.cluster > 1) {
        attrs[na].id = cudaLaunchAttributeClusterDimension;
        attrs[na].val.clusterDim.x = 1;
        attrs[na].val.clusterDim.y = (unsigned)L.cluster;
        attrs[na].val.clusterDim.z = 1;
        ++na;
    }
    if (L.pdl) {
        attrs[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attrs[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    cfg.attrs = attrs;
    cfg.numAttrs = na;
    void* args[] = {&prm};
    const cudaError_t e = cudaLaunchKernelExC(&cfg, fn, args);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace laq
