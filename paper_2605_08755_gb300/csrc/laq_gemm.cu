// laq_gemm.cu -- Y[M][N] = X[M][K] * W_hat[K][N] with W_hat = s * (q - z) per group of 128 rows
// of K (Eq. (1) of LAQuant), M = 1..16, for sm_103a.
//
// Design (the paper's own INT3 GEMV, App. H, is prior art for a different GPU; this is not it):
//
//  * Weights stream from HBM exactly once.  Each warp runs a private cp.async ring of `stages`
//    slots in shared memory; slot i holds the warp's current 16-column x 128-row record of
//    each of its NT tiles (768 B at b = 3, 1024 B at b = 4).  Every lane copies and later
//    reads only its own 16 + 8 (b = 3) or 16 + 16 (b = 4) bytes, so the ring needs no barrier.
//
//  * Dequantization is folded into a tensor-core contraction.  A code q at bit position p of
//    an fp16 mantissa becomes the exact fp16 value 1024 + q * 2^p with one LOP3 (two codes per
//    32-bit register).  X is pre-scaled per row of K by 2^-p, so the m16n8k16 MMA (fp16 in, fp32
//    accumulate) of these registers against x' = x * 2^-p yields, per group g and column n,
//        D = sum_k (1024 + q 2^p) x 2^-p = 1024 * S'_g + sum_k q x,     S'_g = sum_k x'.
//    The group epilogue applies Eq. (1):  y_n += s_gn * (D - 1024 S'_g - z_gn * S_g),
//    S_g = sum_k x_k, which equals sum_k x_k * s_gn * (q - z_gn).  No per-weight subtract or
//    multiply is needed; the unpack is ~0.7 integer ops per weight.
//
//  * The MMA's 8 output columns are shared between batch rows and groups: with MP = M rounded
//    up to a power of two (<= 8), column col = b * (8/MP) + (group index mod 8/MP).  At M = 1
//    one accumulator collects 8 groups in its 8 columns, so every fp32 result of the MMA is
//    used and the group epilogue runs once per 8 groups.  M = 9..16 issues two MMAs per step.
//
//  * Split-K: the warps of a CTA take interleaved groups of the CTA's K range; their partial
//    sums meet in shared memory.  The CTAs of a thread-block cluster split K further and reduce
//    through distributed shared memory, in fixed order (deterministic, no atomics, no global
//    scratch).  Within a warp, the 8/MP group columns of one batch row are summed with warp
//    shuffles.
#include <cooperative_groups.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "laq_internal.cuh"

namespace cg = cooperative_groups;

namespace laq {

namespace {

constexpr uint32_t kMagic = 0x64006400u;  // fp16 1024.0 in both halves
constexpr int kMaxWarps = 8;

template <int BITS>
struct RecordFmt;
template <>
struct RecordFmt<4> {
    static constexpr int kBytes = 1024;  // 32 lanes x 32 B
    static constexpr int kChunk1 = 16;   // second copy per lane
};
template <>
struct RecordFmt<3> {
    static constexpr int kBytes = 768;   // 32 lanes x 24 B
    static constexpr int kChunk1 = 8;
};

struct Params {
    const uint16_t* X;
    const uint8_t* packed;
    const uint16_t* s;
    const uint8_t* z;
    uint16_t* Y;
    int M, K, N, G, T;
    int stages;  // cp.async ring depth per warp
    int gpp;     // groups of X staged in shared memory per phase
};

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async8(uint32_t dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;\n" ::: "memory");
}
// Wait until at most n of this thread's committed cp.async groups are pending (n = 0..7).
__device__ __forceinline__ void cp_async_wait(int n) {
    switch (n) {
        case 0: asm volatile("cp.async.wait_group 0;\n" ::: "memory"); break;
        case 1: asm volatile("cp.async.wait_group 1;\n" ::: "memory"); break;
        case 2: asm volatile("cp.async.wait_group 2;\n" ::: "memory"); break;
        case 3: asm volatile("cp.async.wait_group 3;\n" ::: "memory"); break;
        case 4: asm volatile("cp.async.wait_group 4;\n" ::: "memory"); break;
        case 5: asm volatile("cp.async.wait_group 5;\n" ::: "memory"); break;
        case 6: asm volatile("cp.async.wait_group 6;\n" ::: "memory"); break;
        default: asm volatile("cp.async.wait_group 7;\n" ::: "memory"); break;
    }
}

__device__ __forceinline__ void pdl_wait() {
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

// D += A * B, m16n8k16, A row-major fp16 (16 columns of W x 16 rows of K), B fp16 (16 rows of
// K x 8 columns), fp32 accumulate.
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Pre-scale exponent p of pair index i = 2j + h (the bit position its codes occupy inside the
// fp16 mantissa after extraction).  b = 4: h = 0 -> 0, h = 1 -> 4.  b = 3: fields at bits 0 / 3 /
// 6 for i < 6 / < 12 / < 15, and the assembled spare-bit code at bit 4 for i = 15.
template <int BITS>
__device__ __forceinline__ int pair_shift(int i) {
    if (BITS == 4) return (i & 1) ? 4 : 0;
    return i < 6 ? 0 : (i < 12 ? 3 : (i < 15 ? 6 : 4));
}

// Extract the A fragments of one record (one lane's words) into a[j][0..3] for the 8 k16 steps:
// a0 = (row r, k 2c..2c+1), a1 = (row r+8, same k), a2 = (row r, k 2c+8..), a3 = (row r+8, ...).
template <int BITS>
__device__ __forceinline__ void extract(const uint32_t (&wd)[BITS == 4 ? 8 : 6],
                                        uint32_t (&a)[8][4]) {
    if constexpr (BITS == 4) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const uint32_t w = wd[j], t = w >> 8;
            a[j][0] = (w & 0x000f000fu) | kMagic;  // pair (j, 0, r)      p = 0
            a[j][2] = (w & 0x00f000f0u) | kMagic;  // pair (j, 1, r)      p = 4
            a[j][1] = (t & 0x000f000fu) | kMagic;  // pair (j, 0, r + 8)  p = 0
            a[j][3] = (t & 0x00f000f0u) | kMagic;  // pair (j, 1, r + 8)  p = 4
        }
    } else {
        uint32_t u[6];
#pragma unroll
        for (int w = 0; w < 6; ++w) u[w] = wd[w] >> 9;
        uint32_t rp[16][2];
#pragma unroll
        for (int w = 0; w < 6; ++w) {
            rp[w][0] = (wd[w] & 0x00070007u) | kMagic;      // bits 0-2    p = 0
            rp[w][1] = (u[w] & 0x00070007u) | kMagic;       // bits 9-11   p = 0
            rp[6 + w][0] = (wd[w] & 0x00380038u) | kMagic;  // bits 3-5    p = 3
            rp[6 + w][1] = (u[w] & 0x00380038u) | kMagic;   // bits 12-14  p = 3
        }
#pragma unroll
        for (int q = 0; q < 3; ++q) {
            rp[12 + q][0] = (wd[2 * q] & 0x01c001c0u) | kMagic;      // bits 6-8  p = 6
            rp[12 + q][1] = (wd[2 * q + 1] & 0x01c001c0u) | kMagic;
        }
        // pair 15: bit 15 of words 0,1,2 (row r) / 3,4,5 (row r+8) -> code bits 0,1,2 at p = 4
        rp[15][0] = kMagic | ((u[0] >> 2) & 0x00100010u) | ((u[1] >> 1) & 0x00200020u) |
                    (u[2] & 0x00400040u);
        rp[15][1] = kMagic | ((u[3] >> 2) & 0x00100010u) | ((u[4] >> 1) & 0x00200020u) |
                    (u[5] & 0x00400040u);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            a[j][0] = rp[2 * j][0];
            a[j][1] = rp[2 * j][1];
            a[j][2] = rp[2 * j + 1][0];
            a[j][3] = rp[2 * j + 1][1];
        }
    }
}

template <int BITS, int MP, int NT>
__global__ void __launch_bounds__(kMaxWarps * 32, 2) gemm_kernel(const Params p) {
    using F = RecordFmt<BITS>;
    constexpr int WPL = BITS == 4 ? 8 : 6;
    constexpr int GPA = MP >= 8 ? 1 : 8 / MP;  // groups sharing one accumulator (columns)
    constexpr int NH = MP > 8 ? 2 : 1;          // MMAs per step (batch rows 0-7, 8-15)

    extern __shared__ __align__(128) uint8_t smem[];
    const int W = blockDim.x >> 5;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = lane & 3, R = lane >> 2;
    const int M = p.M, GP = p.gpp, S = p.stages;
    const int T0 = blockIdx.x * NT;
    const int ntv = min(NT, p.T - T0);
    const int C = gridDim.y, rank = blockIdx.y;
    const int g0 = (int)((long long)p.G * rank / C);
    const int g1 = (int)((long long)p.G * (rank + 1) / C);

    // shared memory: ring | xs | zero block | S | P | part
    uint8_t* ring = smem;
    uint4* xs = reinterpret_cast<uint4*>(smem + (size_t)W * S * NT * F::kBytes);
    uint4* zblk = xs + (size_t)M * GP * 16;
    float* ssum = reinterpret_cast<float*>(zblk + 16);
    float* psum = ssum + M * GP;
    float* part = psum + M * GP;
    if (threadIdx.x < 16) zblk[threadIdx.x] = make_uint4(0u, 0u, 0u, 0u);

    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(ring) +
                            (uint32_t)(warp * S * NT * F::kBytes);
    const uint8_t* ring_w = ring + (size_t)warp * S * NT * F::kBytes;

    float yacc[NT][NH][4];
#pragma unroll
    for (int t = 0; t < NT; ++t)
#pragma unroll
        for (int h = 0; h < NH; ++h)
#pragma unroll
            for (int v = 0; v < 4; ++v) yacc[t][h][v] = 0.f;

    bool waited = false;
    for (int pa = g0; pa < g1; pa += GP) {
        const int pb = min(g1, pa + GP);
        const int nw = (pb - pa - warp + W - 1) / W;  // groups of this warp (may be <= 0)

        // Issue the copies of the warp's i-th group (records of all valid tiles) into slot i % S.
        auto issue = [&](int i) {
            if (i < nw) {
                const int g = pa + warp + i * W;
                const uint32_t slot = ring_s + (uint32_t)((i % S) * NT * F::kBytes);
#pragma unroll
                for (int t = 0; t < NT; ++t) {
                    if (t < ntv) {
                        const uint8_t* src =
                            p.packed + ((size_t)(T0 + t) * p.G + g) * F::kBytes;
                        const uint32_t dst = slot + t * F::kBytes;
                        cp_async16(dst + lane * 16, src + lane * 16);
                        if (F::kChunk1 == 16)
                            cp_async16(dst + 512 + lane * 16, src + 512 + lane * 16);
                        else
                            cp_async8(dst + 512 + lane * 8, src + 512 + lane * 8);
                    }
                }
            }
            cp_async_commit();
        };

        for (int i = 0; i < S - 1; ++i) issue(i);

        if (!waited) {  // X (and Y) belong to the preceding kernel until it completes
            pdl_wait();
            pdl_launch_dependents();
            waited = true;
        }
        if (pa != g0) __syncthreads();  // every warp is done reading the previous phase's xs

        // Stage x' = x * 2^-p in MMA B-fragment order, plus S_g = sum x and 1024 * S'_g.
        {
            const int ng = pb - pa;
            const int sc = lane >> 3, sj = lane & 7;  // staging lane -> (c, j)
            const int pA = pair_shift<BITS>(2 * sj), pB = pair_shift<BITS>(2 * sj + 1);
            const __half2 fA = __float2half2_rn(__int_as_float((127 - pA) << 23));
            const __half2 fB = __float2half2_rn(__int_as_float((127 - pB) << 23));
            for (int e = warp; e < M * ng; e += W) {
                const int b = e / ng, gl = e - b * ng;
                const uint16_t* xrow = p.X + (size_t)b * p.K + (size_t)(pa + gl) * 128;
                const uint32_t xa = *reinterpret_cast<const uint32_t*>(xrow + 16 * sj + 2 * sc);
                const uint32_t xb =
                    *reinterpret_cast<const uint32_t*>(xrow + 16 * sj + 8 + 2 * sc);
                const __half2 ha = *reinterpret_cast<const __half2*>(&xa);
                const __half2 hb = *reinterpret_cast<const __half2*>(&xb);
                const __half2 sa = __hmul2(ha, fA), sb = __hmul2(hb, fB);
                const float2 fa = __half22float2(ha), fb = __half22float2(hb);
                const float2 ga = __half22float2(sa), gb = __half22float2(sb);
                float sum = (fa.x + fa.y) + (fb.x + fb.y);
                float psc = (ga.x + ga.y) + (gb.x + gb.y);
                uint2 v;
                v.x = *reinterpret_cast<const uint32_t*>(&sa);
                v.y = *reinterpret_cast<const uint32_t*>(&sb);
                reinterpret_cast<uint2*>(xs)[2 * (((b * GP + gl) * 4 + (sj >> 1)) * 4 + sc) +
                                             (sj & 1)] = v;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    sum += __shfl_xor_sync(0xffffffffu, sum, o);
                    psc += __shfl_xor_sync(0xffffffffu, psc, o);
                }
                if (lane == 0) {
                    ssum[b * GP + gl] = sum;
                    psum[b * GP + gl] = 1024.f * psc;
                }
            }
        }
        __syncthreads();

        // Batch row and group column of this lane's B fragment (MMA column R).
        const int bl = MP <= 8 ? R / GPA : R;
        const int gil = MP <= 8 ? R % GPA : 0;

        float D[NT][NH][4];
        uint32_t sz[NT][4];  // s bits | z << 16 for the block's epilogue
        for (int i = 0; i < nw; ++i) {
            issue(i + S - 1);
            cp_async_wait(S - 1);

            const int gi = GPA > 1 ? i % GPA : 0;
            const int gl = warp + i * W;  // group index within the phase
            if (gi == 0) {
                // Start of an accumulator block: zero D, fetch s and z for its epilogue.
#pragma unroll
                for (int t = 0; t < NT; ++t) {
#pragma unroll
                    for (int h = 0; h < NH; ++h)
#pragma unroll
                        for (int v = 0; v < 4; ++v) D[t][h][v] = 0.f;
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        const int col = 2 * c + (v & 1);
                        const int giv = MP <= 8 ? col % GPA : 0;
                        const bool ok = t < ntv && i + giv < nw &&
                                        (MP <= 8 ? col / GPA < M : true);
                        uint32_t val = 0;
                        if (ok) {
                            const size_t gidx =
                                (size_t)(pa + warp + (i + giv) * W) * p.N +
                                (size_t)(T0 + t) * 16 + R + 8 * (v >> 1);
                            val = (uint32_t)__ldg(p.s + gidx) | ((uint32_t)__ldg(p.z + gidx) << 16);
                        }
                        sz[t][v] = val;
                    }
                }
            }

            // B fragments of this group: x' for lanes whose column belongs to it, else zeros.
            uint32_t B[NH][8][2];
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                const int b = bl + 8 * h;
                const bool act = gil == gi && b < M;
                const uint4* src = act ? xs + (size_t)(b * GP + gl) * 16 : zblk;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint4 v = src[q * 4 + c];
                    B[h][2 * q][0] = v.x;
                    B[h][2 * q][1] = v.y;
                    B[h][2 * q + 1][0] = v.z;
                    B[h][2 * q + 1][1] = v.w;
                }
            }

            const uint8_t* slot = ring_w + (size_t)(i % S) * NT * F::kBytes;
#pragma unroll
            for (int t = 0; t < NT; ++t) {
                if (t < ntv) {
                    uint32_t wd[WPL];
                    const uint4 c0 = *reinterpret_cast<const uint4*>(slot + t * F::kBytes +
                                                                     lane * 16);
                    wd[0] = c0.x; wd[1] = c0.y; wd[2] = c0.z; wd[3] = c0.w;
                    if constexpr (BITS == 4) {
                        const uint4 c1 = *reinterpret_cast<const uint4*>(
                            slot + t * F::kBytes + 512 + lane * 16);
                        wd[4] = c1.x; wd[5] = c1.y; wd[6] = c1.z; wd[7] = c1.w;
                    } else {
                        const uint2 c1 = *reinterpret_cast<const uint2*>(
                            slot + t * F::kBytes + 512 + lane * 8);
                        wd[4] = c1.x; wd[5] = c1.y;
                    }
                    uint32_t a[8][4];
                    extract<BITS>(wd, a);
#pragma unroll
                    for (int j = 0; j < 8; ++j)
#pragma unroll
                        for (int h = 0; h < NH; ++h)
                            mma16816(D[t][h], a[j][0], a[j][1], a[j][2], a[j][3], B[h][j][0],
                                     B[h][j][1]);
                }
            }

            if (gi == GPA - 1 || i == nw - 1) {
                // Group epilogue (Eq. (1)): y += s * (D - 1024 S' - z S) per (group, column, row).
                const int ib = i - gi;
#pragma unroll
                for (int t = 0; t < NT; ++t) {
#pragma unroll
                    for (int h = 0; h < NH; ++h) {
#pragma unroll
                        for (int v = 0; v < 4; ++v) {
                            const int col = 2 * c + (v & 1);
                            const int b = MP <= 8 ? col / GPA : 8 * h + col;
                            const int giv = MP <= 8 ? col % GPA : 0;
                            if (t < ntv && b < M && ib + giv < nw) {
                                const int lg = warp + (ib + giv) * W;
                                const uint32_t e = sz[t][v];
                                const float sv = __half2float(__ushort_as_half((uint16_t)e));
                                const float zv = (float)(e >> 16);
                                const float corr = fmaf(zv, ssum[b * GP + lg], psum[b * GP + lg]);
                                yacc[t][h][v] = fmaf(sv, D[t][h][v] - corr, yacc[t][h][v]);
                            }
                        }
                    }
                }
            }
        }
        asm volatile("cp.async.wait_all;\n" ::: "memory");
    }
    if (!waited) {
        pdl_wait();
        pdl_launch_dependents();
    }

    // ---- reduction: group columns (shuffles) -> warps (shared) -> cluster CTAs (DSMEM) ----
    __syncthreads();  // the ring is free: reuse it for the per-warp partial sums
    float* red = reinterpret_cast<float*>(smem);
    const int E = NT * M * 16;
#pragma unroll
    for (int t = 0; t < NT; ++t) {
        float* rw = red + (size_t)warp * E + t * M * 16;
        if (MP <= 8 && GPA >= 2) {
            float y0 = yacc[t][0][0] + yacc[t][0][1];
            float y1 = yacc[t][0][2] + yacc[t][0][3];
            if (GPA >= 4) {
                y0 += __shfl_xor_sync(0xffffffffu, y0, 1);
                y1 += __shfl_xor_sync(0xffffffffu, y1, 1);
            }
            if (GPA >= 8) {
                y0 += __shfl_xor_sync(0xffffffffu, y0, 2);
                y1 += __shfl_xor_sync(0xffffffffu, y1, 2);
            }
            const int b = (2 * c) / GPA;
            if ((2 * c) % GPA == 0 && b < M) {
                rw[b * 16 + R] = y0;
                rw[b * 16 + R + 8] = y1;
            }
        } else {
#pragma unroll
            for (int h = 0; h < NH; ++h)
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    const int b = 8 * h + 2 * c + (v & 1);
                    if (b < M) rw[b * 16 + R + 8 * (v >> 1)] = yacc[t][h][v];
                }
        }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < E; e += blockDim.x) {
        float acc = 0.f;
        for (int w = 0; w < W; ++w) acc += red[(size_t)w * E + e];
        part[e] = acc;
    }

    auto store = [&](int e, float acc) {
        const int t = e / (M * 16), b = (e / 16) % M, row = e % 16;
        if (t < ntv) {
            const __half hv = __float2half_rn(acc);
            p.Y[(size_t)b * p.N + (size_t)(T0 + t) * 16 + row] = __half_as_ushort(hv);
        }
    };
    if (C == 1) {
        __syncthreads();
        for (int e = threadIdx.x; e < E; e += blockDim.x) store(e, part[e]);
    } else {
        cg::cluster_group cluster = cg::this_cluster();
        cluster.sync();  // every CTA's partial sums are complete
        for (int e = rank + threadIdx.x * C; e < E; e += blockDim.x * C) {
            float acc = 0.f;
            for (int q = 0; q < C; ++q) acc += cluster.map_shared_rank(part, q)[e];
            store(e, acc);
        }
        cluster.sync();  // peers have finished reading this CTA's shared memory
    }
}

using KernelFn = void (*)(Params);

template <int BITS, int MP>
KernelFn pick_nt(int nt) {
    switch (nt) {
        case 1: return gemm_kernel<BITS, MP, 1>;
        case 2: return gemm_kernel<BITS, MP, 2>;
        default: return gemm_kernel<BITS, MP, 4>;
    }
}

template <int BITS>
KernelFn pick_mp(int mp, int nt) {
    switch (mp) {
        case 1: return pick_nt<BITS, 1>(nt);
        case 2: return pick_nt<BITS, 2>(nt);
        case 4: return pick_nt<BITS, 4>(nt);
        case 8: return pick_nt<BITS, 8>(nt);
        default: return pick_nt<BITS, 16>(nt);
    }
}

int mp_class(int M) { return M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : M <= 8 ? 8 : 16; }
int mp_index(int mp) { return mp == 1 ? 0 : mp == 2 ? 1 : mp == 4 ? 2 : mp == 8 ? 3 : 4; }
int nt_index(int nt) { return nt == 1 ? 0 : nt == 2 ? 1 : 2; }

std::atomic<size_t> g_attr_limit[2][5][3];  // max dynamic smem already granted per kernel

constexpr size_t kXsBudget = 48 * 1024;  // shared memory for staged X per phase

}  // namespace

size_t gemm_smem_bytes(const GemmLaunch& L, int* groups_per_phase) {
    const size_t rec = L.bits == 4 ? 1024 : 768;
    const size_t ring = (size_t)L.warps * L.stages * L.tiles_per_cta * rec;
    const int G = L.K / 128;
    const int gc = (G + L.cluster - 1) / L.cluster;
    const size_t per_group = (size_t)L.M * (256 + 8);
    int gpp = (int)(kXsBudget / per_group);
    if (gpp > gc) gpp = gc;
    if (gpp < 1) gpp = 1;
    if (groups_per_phase) *groups_per_phase = gpp;
    return ring + 256 + (size_t)gpp * per_group + (size_t)L.tiles_per_cta * L.M * 16 * 4;
}

cudaError_t launch_gemm(const GemmLaunch& L, size_t smem_limit, cudaStream_t stream) {
    int gpp = 1;
    const size_t smem = gemm_smem_bytes(L, &gpp);
    if (smem > smem_limit) return cudaErrorInvalidConfiguration;
    const int mp = mp_class(L.M);
    const KernelFn fn = L.bits == 4 ? pick_mp<4>(mp, L.tiles_per_cta)
                                    : pick_mp<3>(mp, L.tiles_per_cta);
    std::atomic<size_t>& granted = g_attr_limit[L.bits == 4][mp_index(mp)][nt_index(L.tiles_per_cta)];
    if (granted.load() < smem) {
        const cudaError_t e = cudaFuncSetAttribute(
            (const void*)fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_limit);
        if (e != cudaSuccess) return e;
        granted.store(smem_limit);
    }
    Params prm;
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
    const cudaError_t e = cudaLaunchKernelExC(&cfg, (const void*)fn, args);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace laq
