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
//  * Dequantization is folded into a tensor-core contraction.  A code q at mantissa bit p of
//    an fp16 whose exponent field is 25 - p has the exact value 2^(10-p) + q, so one LOP3
//    (mask | exponent) turns two codes of a 32-bit word into A-fragment values c + q with a
//    per-field offset c = 2^(10-p).  The m16n8k16 MMA (fp16 in, fp32 accumulate) of these
//    against raw x gives, per group g and MMA column, D = sum_k c_k x_k + sum_k q_k x_k.  While
//    X is staged, the 16 lanes that load a group's 256 bytes sum P_g = sum_k c_k x_k and
//    S_g = sum_k x_k (shuffles), so the group epilogue applies Eq. (1) directly:
//    y_n += s_gn * (D - P_g - z_gn * S_g)  (= sum_k x_k s (q - z)).
//    The unpack costs about 0.7 integer ops per weight; nothing else touches a weight.
//
//  * Inside a record, lane c's rows are k = 32c + 4j + 2h + e, so its B fragments for the 8 k16
//    steps are the 32 consecutive x values x[32c .. 32c+31] of the group: four 16-byte shared
//    loads from a plain cp.async copy of X, with no pre-scaling or permutation pass.
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

#include "laq_device.cuh"
#include "laq_internal.cuh"

namespace cg = cooperative_groups;

// Compile-time trace points (start, PDL wait done, X staged, K loop done, reduction done, end).
// Empty in the library build; a tracing build defines LAQ_TRACE to timestamp them.
#ifndef LAQ_TRACE
#define LAQ_TRACE(point) \
    do {                 \
    } while (0)
#endif
#ifndef LAQ_TRACE_LOOP
#define LAQ_TRACE_LOOP(point, iter) \
    do {                            \
    } while (0)
#endif

namespace laq {

namespace {

constexpr int kMaxWarps = 8;

struct Params {
    const uint16_t* X;
    const uint8_t* packed;
    const uint16_t* s;
    const uint8_t* z;
    uint16_t* Y;
    int M, K, N, G, T;
    int stages;  // cp.async ring depth per warp
    int gpp;     // groups of X staged in shared memory per phase
    int gc;      // most groups a CTA owns: ceil(G / cluster)
    Exps exps;   // exponent fields of the A-fragment extraction
};

template <int BITS, int MP, int NT>
__global__ void __launch_bounds__(kMaxWarps * 32, 2) gemm_kernel(const Params p) {
    using F = RecordFmt<BITS>;
    constexpr int WPL = BITS == 4 ? 8 : 6;
    constexpr int GPA = MP >= 8 ? 1 : 8 / MP;  // groups sharing one accumulator (columns)
    constexpr int NH = MP > 8 ? 2 : 1;          // MMAs per step (batch rows 0-7, 8-15)

    // Let the next kernel on the stream start launching now: it only prefetches constant
    // weights before its own griddepcontrol.wait, which returns once this grid has finished.
    pdl_launch_dependents();
    // Cluster K split: arrive once now; the matching wait before the partial sums are pushed
    // into peers' shared memory guarantees that every CTA of the cluster has started.
    if (gridDim.y > 1) asm volatile("barrier.cluster.arrive.relaxed.aligned;\n" ::: "memory");
    LAQ_TRACE(0);

    extern __shared__ __align__(128) uint8_t smem[];
    const int W = blockDim.x >> 5;
    const int WT = W / NT;                     // warps per tile
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tile = warp % NT, team = warp / NT;
    const int c = lane & 3, R = lane >> 2;
    const int M = p.M, GP = p.gpp, S = p.stages;
    const int T0 = blockIdx.x * NT;
    const int ntv = min(NT, p.T - T0);
    const bool tile_ok = tile < ntv;
    const int C = gridDim.y, rank = blockIdx.y;
    const int g0 = (int)((long long)p.G * rank / C);
    const int g1 = (int)((long long)p.G * (rank + 1) / C);

    // shared memory: ring [W][S][record] | x [M][GP][128] fp16 | zero block (64 B)
    //                | s [gc][NT][16] fp16 | z [gc][NT][16] u8 | (S, P) [M][GP] float2
    //                | part [NT][MP][16] fp32
    uint8_t* ring = smem;
    uint4* xs = reinterpret_cast<uint4*>(smem + (size_t)W * S * F::kBytes);
    uint4* zblk = xs + (size_t)M * GP * 16;
    uint16_t* s_sm = reinterpret_cast<uint16_t*>(zblk + 4);
    uint8_t* z_sm = reinterpret_cast<uint8_t*>(s_sm + (size_t)p.gc * NT * 16);
    float2* ps = reinterpret_cast<float2*>(z_sm + (size_t)p.gc * NT * 16);
    float* part = reinterpret_cast<float*>(ps + (size_t)M * GP);
    if (threadIdx.x < 4) zblk[threadIdx.x] = make_uint4(0u, 0u, 0u, 0u);

    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(ring) +
                            (uint32_t)(warp * S * F::kBytes);
    const uint8_t* ring_w = ring + (size_t)warp * S * F::kBytes;

    float yacc[NH][4];
#pragma unroll
    for (int h = 0; h < NH; ++h)
#pragma unroll
        for (int v = 0; v < 4; ++v) yacc[h][v] = 0.f;

    bool first = true;
    for (int pa = g0; pa < g1; pa += GP) {
        const int pb = min(g1, pa + GP);
        const int ng = pb - pa;
        // groups of this warp: pa + team + i * WT, i < nw (none for a tile past the edge)
        const int nw = tile_ok ? (ng - team + WT - 1) / WT : 0;

        // Copy the warp's i-th record into the next ring slot (16 + 8 or 16 + 16 bytes per lane).
        const uint8_t* wsrc = p.packed + ((size_t)(T0 + tile) * p.G + pa + team) * F::kBytes;
        const size_t wstep = (size_t)WT * F::kBytes;
        int islot = 0;
        auto issue = [&](int i) {
            if (i < nw) {
                const uint8_t* src = wsrc + (size_t)i * wstep;
                const uint32_t dst = ring_s + (uint32_t)(islot * F::kBytes);
                cp_async16(dst + lane * 16, src + lane * 16);
                if (F::kChunk1 == 16)
                    cp_async16(dst + 512 + lane * 16, src + 512 + lane * 16);
                else
                    cp_async8(dst + 512 + lane * 8, src + 512 + lane * 8);
            }
            cp_async_commit();
            islot = islot + 1 == S ? 0 : islot + 1;
        };

        for (int i = 0; i < S - 1; ++i) issue(i);

        if (first) {
            // Scales and zeros of every group and tile of this CTA (32 + 16 bytes per (group,
            // tile)), in flight together with the weight records: warp per group, lane per
            // (tile, 16-byte piece).
            const uint32_t ss = (uint32_t)__cvta_generic_to_shared(s_sm);
            const uint32_t zs = (uint32_t)__cvta_generic_to_shared(z_sm);
            const int t = lane >> 2, piece = lane & 3;
            if (t < ntv && piece < 3) {
                for (int gl = warp; gl < g1 - g0; gl += W) {
                    const size_t goff = (size_t)(g0 + gl) * p.N + (size_t)(T0 + t) * 16;
                    const uint32_t slot = (uint32_t)(gl * NT + t);
                    if (piece < 2)
                        cp_async16(ss + slot * 32 + piece * 16, p.s + goff + piece * 8);
                    else
                        cp_async16(zs + slot * 16, p.z + goff);
                }
            }
            cp_async_commit();
            // X (and Y) belong to the preceding kernel on the stream until it completes.
            pdl_wait();
            LAQ_TRACE(1);
            first = false;
        } else {
            __syncthreads();  // every warp is done reading the previous phase's X, S and P
        }

        // Raw X of the phase (row b's groups pa..pb-1 are 256 * ng contiguous bytes), through
        // L2 into registers, then shared memory.  16-byte chunk q of a group holds x[8q .. 8q+7],
        // i.e. pairs 4 (q % 4) + w for its four 32-bit words w.  Unit u = (b, group, h), h < 8,
        // loads chunks h and h + 8 of the group, whose pairs have the same offsets c_k; the 8
        // aligned lanes of a group sum S_g = sum_k x_k and P_g = sum_k c_k x_k by shuffles.
        {
            const int per_row = ng * 8;     // units per batch row (a multiple of 8)
            const int nu = M * per_row;     // < 2^16
            // u / per_row = umulhi(u, inv) exactly for u, per_row < 2^16
            const uint32_t inv = 0xffffffffu / (uint32_t)per_row + 1u;
            for (int u0 = 0; u0 < nu; u0 += 2 * (int)blockDim.x) {
                uint4 v[2][2];
                int xo[2];  // offset of the unit's first chunk in xs (uint4), -1 past the end
                int po[2];  // its group's (S, P) slot [b][group]
#pragma unroll
                for (int r = 0; r < 2; ++r) {
                    const int u = u0 + r * (int)blockDim.x + (int)threadIdx.x;
                    if (u < nu) {
                        const int b = (int)__umulhi((uint32_t)u, inv);
                        const int uu = u - b * per_row;
                        const int q = (uu >> 3) * 16 + (uu & 7);  // chunk in the row
                        const uint16_t* src = p.X + (size_t)b * p.K + (size_t)pa * 128 + q * 8;
                        v[r][0] = ld_cg16(src);
                        v[r][1] = ld_cg16(src + 64);
                        xo[r] = b * GP * 16 + q;
                        po[r] = b * GP + (uu >> 3);
                    } else {
                        v[r][0] = v[r][1] = make_uint4(0u, 0u, 0u, 0u);
                        xo[r] = -1;
                        po[r] = 0;
                    }
                }
#pragma unroll
                for (int r = 0; r < 2; ++r) {
                    // (warp-uniform) nothing of this batch for this warp
                    if (u0 + r * (int)blockDim.x + warp * 32 >= nu) break;
                    const uint32_t w0[4] = {v[r][0].x, v[r][0].y, v[r][0].z, v[r][0].w};
                    const uint32_t w1[4] = {v[r][1].x, v[r][1].y, v[r][1].z, v[r][1].w};
                    float sx = 0.f, px = 0.f;
#pragma unroll
                    for (int w = 0; w < 4; ++w) {
                        const float2 f0 = __half22float2(*reinterpret_cast<const __half2*>(&w0[w]));
                        const float2 f1 = __half22float2(*reinterpret_cast<const __half2*>(&w1[w]));
                        const float pair = (f0.x + f0.y) + (f1.x + f1.y);
                        sx += pair;
                        px = fmaf(row_offset<BITS>((lane & 3) * 4 + w), pair, px);
                    }
#pragma unroll
                    for (int o = 1; o < 8; o <<= 1) {
                        sx += __shfl_xor_sync(0xffffffffu, sx, o);
                        px += __shfl_xor_sync(0xffffffffu, px, o);
                    }
                    if (xo[r] >= 0) {
                        xs[xo[r]] = v[r][0];
                        xs[xo[r] + 8] = v[r][1];
                        if ((lane & 7) == 0) ps[po[r]] = make_float2(sx, px);  // unit h = 0
                    }
                }
            }
            // the weights issued so far and the scales and zeros have landed
            asm volatile("cp.async.wait_all;\n" ::: "memory");
            __syncthreads();
            LAQ_TRACE(6);
            LAQ_TRACE(7);
            LAQ_TRACE(2);
        }

        // Batch row and group column of this lane's B fragment (MMA column R).
        const int bl = MP <= 8 ? R / GPA : R;
        const int gil = MP <= 8 ? R % GPA : 0;
        // X of the lane's B column for the warp's record i: uint4 offset xo0[h] + i * xstep.
        const int xstep = WT * 16;
        int xo0[NH];
#pragma unroll
        for (int h = 0; h < NH; ++h) xo0[h] = ((bl + 8 * h) * GP + team) * 16 + c * 4;

        int rslot = 0;
        float D[2][NH][4];  // two independent accumulator chains (even / odd k16 steps)

        // One record: B fragments, the packed words, extraction and the 8 k16-step MMAs.  A
        // lane's B column belongs to the block's record gil, so only that record reads X (from
        // xm); the others take zeros.
        auto record = [&](const int i, const int gi, const uint4* const* xm, const bool kStream) {
            LAQ_TRACE_LOOP(0, i);
            if (kStream) {
                issue(i + S - 1);
                cp_async_wait(S - 1);
            }
            LAQ_TRACE_LOOP(1, i);
            uint32_t B[NH][8][2];
#pragma unroll
            for (int h = 0; h < NH; ++h) {
                const uint4* src = gil == gi && bl + 8 * h < M ? xm[h] : zblk;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint4 v = src[q];
                    B[h][2 * q][0] = v.x;
                    B[h][2 * q][1] = v.y;
                    B[h][2 * q + 1][0] = v.z;
                    B[h][2 * q + 1][1] = v.w;
                }
            }
            LAQ_TRACE_LOOP(2, i);
            const uint8_t* slot = ring_w + (size_t)(kStream ? rslot : i) * F::kBytes;
            uint32_t wd[WPL];
            const uint4 c0 = *reinterpret_cast<const uint4*>(slot + lane * 16);
            wd[0] = c0.x; wd[1] = c0.y; wd[2] = c0.z; wd[3] = c0.w;
            if constexpr (BITS == 4) {
                const uint4 c1 = *reinterpret_cast<const uint4*>(slot + 512 + lane * 16);
                wd[4] = c1.x; wd[5] = c1.y; wd[6] = c1.z; wd[7] = c1.w;
            } else {
                const uint2 c1 = *reinterpret_cast<const uint2*>(slot + 512 + lane * 8);
                wd[4] = c1.x; wd[5] = c1.y;
            }
            uint32_t a[8][4];
            extract<BITS>(wd, p.exps, a);
#pragma unroll
            for (int j = 0; j < 8; ++j)
#pragma unroll
                for (int h = 0; h < NH; ++h)
                    mma16816(D[j & 1][h], a[j][0], a[j][1], a[j][2], a[j][3], B[h][j][0],
                             B[h][j][1]);
            if (kStream) rslot = rslot + 1 == S ? 0 : rslot + 1;
            LAQ_TRACE_LOOP(3, i);
        };

        // A block of GPA records (the groups sharing one accumulator) from record i0, then its
        // epilogue.  Without streaming (the usual case) the position in the block is a
        // compile-time constant, so slot and X offsets fold into immediates; the streaming
        // form keeps the loop rolled (one copy of the record code, less instruction cache).
        // (Called with a constant flag, folded once the lambda is inlined.)
        auto block = [&](const int i0, const bool stream) {
#pragma unroll
            for (int a = 0; a < 2; ++a)
#pragma unroll
                for (int h = 0; h < NH; ++h)
#pragma unroll
                    for (int v = 0; v < 4; ++v) D[a][h][v] = 0.f;
            const uint4* xm[NH];
#pragma unroll
            for (int h = 0; h < NH; ++h) xm[h] = xs + xo0[h] + (i0 + gil) * xstep;
            if (stream) {
#pragma unroll 1
                for (int gi = 0; gi < GPA; ++gi) {
                    if (i0 + gi >= nw) break;  // warp-uniform
                    record(i0 + gi, gi, xm, true);
                }
            } else {
#pragma unroll
                for (int gi = 0; gi < GPA; ++gi) {
                    if (i0 + gi >= nw) break;  // warp-uniform
                    record(i0 + gi, gi, xm, false);
                }
            }

            // Block epilogue (Eq. (1)): y += s * (D - P - z S) per (group, column, row).
            // Value v of the lane is MMA column 2c + (v & 1): batch row col / GPA and the
            // block's record col % GPA (MP <= 8), or batch row 8h + col (MP = 16).
#pragma unroll
            for (int h = 0; h < NH; ++h) {
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    const int col = 2 * c + (v & 1);
                    const int b = MP <= 8 ? col / GPA : 8 * h + col;
                    const int giv = MP <= 8 ? col % GPA : 0;
                    if (b < M && i0 + giv < nw) {
                        const int lg = team + (i0 + giv) * WT;        // in the phase
                        const int e = ((pa - g0 + lg) * NT + tile) * 16 + R + 8 * (v >> 1);
                        const float sv = __half2float(__ushort_as_half(s_sm[e]));
                        const float zv = (float)z_sm[e];
                        const float2 sp = ps[b * GP + lg];  // (S, P) of the group
                        const float d = D[0][h][v] + D[1][h][v] - sp.y;
                        yacc[h][v] = fmaf(sv, fmaf(-zv, sp.x, d), yacc[h][v]);
                    }
                }
            }
            LAQ_TRACE_LOOP(4, i0);
        };

        // With S - 1 >= nw every record of the warp was copied in the prologue and has landed;
        // record i then sits in slot i.
        if (S - 1 < nw) {
            for (int i0 = 0; i0 < nw; i0 += GPA) block(i0, true);
        } else {
            for (int i0 = 0; i0 < nw; i0 += GPA) block(i0, false);
        }
        asm volatile("cp.async.wait_all;\n" ::: "memory");
    }
    if (first) pdl_wait();  // a CTA without groups still writes Y after the previous kernel
    LAQ_TRACE(3);

    // ---- reduction: group columns (shuffles) -> warps of a tile (shared) -> cluster (DSMEM) ----
    // Per-warp partials live in the (now idle) ring as red[W][MP][16]; b >= M is unused.
    __syncthreads();
    float* red = reinterpret_cast<float*>(smem);
    {
        float* rw = red + (size_t)warp * MP * 16;
        if (MP <= 8 && GPA >= 2) {
            float y0 = yacc[0][0] + yacc[0][1];
            float y1 = yacc[0][2] + yacc[0][3];
            if (GPA >= 4) {
                y0 += __shfl_xor_sync(0xffffffffu, y0, 1);
                y1 += __shfl_xor_sync(0xffffffffu, y1, 1);
            }
            if (GPA >= 8) {
                y0 += __shfl_xor_sync(0xffffffffu, y0, 2);
                y1 += __shfl_xor_sync(0xffffffffu, y1, 2);
            }
            const int b = (2 * c) / GPA;
            if ((2 * c) % GPA == 0) {
                rw[b * 16 + R] = y0;
                rw[b * 16 + R + 8] = y1;
            }
        } else {
#pragma unroll
            for (int h = 0; h < NH; ++h)
#pragma unroll
                for (int v = 0; v < 4; ++v)
                    rw[(8 * h + 2 * c + (v & 1)) * 16 + R + 8 * (v >> 1)] = yacc[h][v];
        }
    }
    __syncthreads();
    constexpr int E = NT * MP * 16;
    // this CTA's sum of element e over its warps of the tile
    auto local = [&](int e) {
        const int t = e / (MP * 16), r = e % (MP * 16);
        float acc = 0.f;
        for (int u = 0; u < WT; ++u) acc += red[(size_t)(u * NT + t) * MP * 16 + r];
        return acc;
    };

    auto store = [&](int e, float acc) {
        const int t = e / (MP * 16), b = (e / 16) % MP, row = e % 16;
        if (t < ntv && b < M) {
            const __half hv = __float2half_rn(acc);
            p.Y[(size_t)b * p.N + (size_t)(T0 + t) * 16 + row] = __half_as_ushort(hv);
        }
    };
    if (C == 1) {
        for (int e = threadIdx.x; e < E; e += blockDim.x) store(e, local(e));
        LAQ_TRACE(4);
        LAQ_TRACE(5);
    } else {
        // Element e belongs to CTA e % C of the cluster: each CTA pushes its partial into the
        // owner's part[rank][e / C] (distributed shared memory), one cluster barrier, then the
        // owner sums the C partials in rank order.  Nothing reads another CTA's shared memory
        // after the barrier, so each CTA may finish at once.
        cg::cluster_group cluster = cg::this_cluster();
        const int EL = E / C;  // E is a multiple of 16, C divides 16
        asm volatile("barrier.cluster.wait.aligned;\n" ::: "memory");
        for (int e = threadIdx.x; e < E; e += blockDim.x)
            cluster.map_shared_rank(part, e % C)[rank * EL + e / C] = local(e);
        LAQ_TRACE(4);
        cluster.sync();  // every partial has arrived at its owner
        for (int el = threadIdx.x; el < EL; el += blockDim.x) {
            float acc = 0.f;
            for (int q = 0; q < C; ++q) acc += part[q * EL + el];
            store(el * C + rank, acc);
        }
        LAQ_TRACE(5);
    }
}

using KernelFn = void (*)(Params);

template <int BITS, int MP>
KernelFn pick_nt(int nt) {
    switch (nt) {
        case 1: return gemm_kernel<BITS, MP, 1>;
        case 2: return gemm_kernel<BITS, MP, 2>;
        case 4: return gemm_kernel<BITS, MP, 4>;
        default: return gemm_kernel<BITS, MP, 8>;
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
int nt_index(int nt) { return nt == 1 ? 0 : nt == 2 ? 1 : nt == 4 ? 2 : 3; }

std::atomic<size_t> g_attr_limit[2][5][4];  // max dynamic smem already granted per kernel

constexpr size_t kXsBudget = 64 * 1024;  // shared memory for staged X (and its tables) per phase

}  // namespace

size_t gemm_smem_bytes(const GemmLaunch& L, int* groups_per_phase) {
    const size_t rec = L.bits == 4 ? 1024 : 768;
    const size_t ring = (size_t)L.warps * L.stages * rec;
    const int G = L.K / 128;
    const int gc = (G + L.cluster - 1) / L.cluster;
    // raw X and (S, P) of one group
    const size_t per_group = (size_t)L.M * (256 + 8);
    int gpp = (int)(kXsBudget / per_group);
    if (gpp > gc) gpp = gc;
    if (gpp < 1) gpp = 1;
    if (groups_per_phase) *groups_per_phase = gpp;
    const int mp = mp_class(L.M);
    const size_t sz = (size_t)(gc > 0 ? gc : 1) * L.tiles_per_cta * 48;  // s (32 B) + z (16 B)
    return ring + (size_t)gpp * per_group + 64 + sz + (size_t)L.tiles_per_cta * mp * 16 * 4;
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
        // Every instance asks for the largest shared-memory carveout, so kernels of different
        // shapes following each other in a decode step never reconfigure L1 / shared memory.
        cudaError_t e = cudaFuncSetAttribute(
            (const void*)fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_limit);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute((const void*)fn,
                                 cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
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
    const cudaError_t e = cudaLaunchKernelExC(&cfg, (const void*)fn, args);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace laq
