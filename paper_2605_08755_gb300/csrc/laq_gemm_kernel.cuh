// laq_gemm_kernel.cuh -- the dequantize-fused GEMM kernel template, included by the two
// translation units that instantiate it: laq_gemm.cu (plain X) and laq_gemm_prologue.cu (X made
// by a fused RMSNorm or SiLU * up prologue).  Keeping the prologue a template parameter leaves
// the plain kernel without a trace of it.
//
// Y[M][N] = X[M][K] * W_hat[K][N] with W_hat = s * (q - z) per group of 128 rows
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
#pragma once
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

// Warps per CTA: up to 8 for M <= 2 (two CTAs per SM), up to 16 from M = 3, where a CTA
// shares staged X over 4 or 8 tiles and two warps per tile hide the MMA and shared-memory
// latency that one CTA per SM leaves exposed.
__host__ __device__ constexpr int max_warps(int mp) { return mp >= 4 ? 16 : 8; }

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
    // X prologue: kProRmsNorm (input = fp16(fp16(X + R) / rms * w), rms over each row's K) or
    // kProSiluMul (X rows hold gate | up, 2K wide; input = fp16(silu(gate) * up))
    int pro;
    float eps;
    const uint16_t* R;
    uint16_t* R_out;
    const uint16_t* w;
};

// h = fp16(x + r) of 8 elements (r may be all zero), as floats
__device__ __forceinline__ void residual8(const uint4 x, const uint4 r, float (&h)[8]) {
    const uint32_t xa[4] = {x.x, x.y, x.z, x.w}, ra[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&xa[i]));
        const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&ra[i]));
        const __half2 s = __floats2half2_rn(a.x + b.x, a.y + b.y);
        const float2 f = __half22float2(s);
        h[2 * i] = f.x;
        h[2 * i + 1] = f.y;
    }
}

__device__ __forceinline__ uint4 pack8f(const float (&f)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const __half2 h = __floats2half2_rn(f[2 * i], f[2 * i + 1]);
        w[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// The prologue's transform of the 8 input elements at column k of row b.
__device__ __forceinline__ uint4 prologue8(const Params& p, int b, size_t k, float inv_rms) {
    if (p.pro == kProRmsNorm) {
        const uint4 x = ld_cg16(p.X + (size_t)b * p.K + k);
        const uint4 r = p.R ? ld_cg16(p.R + (size_t)b * p.K + k) : make_uint4(0u, 0u, 0u, 0u);
        const uint4 wv = *reinterpret_cast<const uint4*>(p.w + k);
        float h[8], y[8];
        residual8(x, r, h);
        const uint32_t wa[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&wa[i]));
            y[2 * i] = h[2 * i] * inv_rms * f.x;
            y[2 * i + 1] = h[2 * i + 1] * inv_rms * f.y;
        }
        return pack8f(y);
    }
    const uint4 g = ld_cg16(p.X + (size_t)b * 2 * p.K + k);
    const uint4 u = ld_cg16(p.X + (size_t)b * 2 * p.K + p.K + k);
    const uint32_t ga[4] = {g.x, g.y, g.z, g.w}, ua[4] = {u.x, u.y, u.z, u.w};
    // Every CTA of the GEMM recomputes its K range, on the path to the first MMA: the
    // hardware exponential and reciprocal (about 2^-21 relative error, far inside fp16's
    // rounding) cost two special-function operations per element instead of ~40 instructions.
    // g very negative: e^-g = inf, g / inf = -0, the limit of silu.
    float y[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&ga[i]));
        const float2 c = __half22float2(*reinterpret_cast<const __half2*>(&ua[i]));
        y[2 * i] = __fdividef(a.x, 1.f + __expf(-a.x)) * c.x;
        y[2 * i + 1] = __fdividef(a.y, 1.f + __expf(-a.y)) * c.y;
    }
    return pack8f(y);
}

// RMSNorm prologue: the inverse RMS of each row of h = fp16(X + R) over its K elements, into
// inv_rms[b] (the same code, so the same bits, in every CTA); CTA (0, 0) also stores h to R_out.
// M = 1: all warps share the row, each thread's chunks loaded together, the warps' sums added
// in warp order.  M > 1: warp b % W takes row b, eight chunks of loads in flight per lane.
__device__ __forceinline__ void rms_chunk(const Params& p, int b, int i, bool writer,
                                          const uint4 x, const uint4 r, float& ss) {
    float h[8];
    residual8(x, r, h);
#pragma unroll
    for (int e = 0; e < 8; ++e) ss = fmaf(h[e], h[e], ss);
    if (writer) *reinterpret_cast<uint4*>(p.R_out + (size_t)b * p.K + 8 * i) = pack8f(h);
}

__device__ void rms_rows(const Params& p, float* inv_rms) {
    const int W = blockDim.x >> 5, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool writer = p.R_out && blockIdx.x == 0 && blockIdx.y == 0;
    const int nch = p.K / 8;
    const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
    if (p.M == 1) {
        float ss = 0.f;
        for (int i0 = threadIdx.x; i0 < nch; i0 += 4 * (int)blockDim.x) {
            uint4 x[4], r[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = i0 + u * (int)blockDim.x;
                x[u] = i < nch ? ld_cg16(p.X + 8 * i) : zero;
                r[u] = i < nch && p.R ? ld_cg16(p.R + 8 * i) : zero;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (i0 + u * (int)blockDim.x < nch)
                    rms_chunk(p, 0, i0 + u * (int)blockDim.x, writer, x[u], r[u], ss);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) inv_rms[16 + warp] = ss;  // (W <= 16)
        __syncthreads();
        if (threadIdx.x == 0) {
            float tot = 0.f;
            for (int k = 0; k < W; ++k) tot += inv_rms[16 + k];
            inv_rms[0] = rsqrtf(tot / (float)p.K + p.eps);
        }
        __syncthreads();
        return;
    }
    for (int b = warp; b < p.M; b += W) {
        float ss = 0.f;
        for (int i0 = lane; i0 < nch; i0 += 8 * 32) {
            uint4 x[8], r[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int i = i0 + 32 * u;
                x[u] = i < nch ? ld_cg16(p.X + (size_t)b * p.K + 8 * i) : zero;
                r[u] = i < nch && p.R ? ld_cg16(p.R + (size_t)b * p.K + 8 * i) : zero;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (i0 + 32 * u < nch) rms_chunk(p, b, i0 + 32 * u, writer, x[u], r[u], ss);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) inv_rms[b] = rsqrtf(ss / (float)p.K + p.eps);
    }
    __syncthreads();
}

template <int BITS, int MP, int NT, bool PRO>
__global__ void __launch_bounds__(max_warps(MP) * 32, 16 / max_warps(MP))
gemm_kernel(const Params p) {
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

    // shared memory: ring [W][S][record] | x [M][xs_row_chunks(GP, MP)] 16-byte chunks
    //                | zero block (64 B, MP <= 2) | s [gc][NT][16] fp16 | z [gc][NT][16] u8
    //                | (S, P) [M][GP] float2
    //                | part [NT][MP][16] fp32 | inv_rms [16] fp32
    uint8_t* ring = smem;
    uint4* xs = reinterpret_cast<uint4*>(smem + (size_t)W * S * F::kBytes);
    constexpr bool kPad = xs_padded(MP);
    constexpr int GC = xs_group_chunks(MP);     // chunks per group of staged X
    const int RS = xs_row_chunks(GP, MP);       // chunks per batch row of staged X
    uint4* zblk = xs + (size_t)M * RS;          // zeros for B columns of other records
    uint16_t* s_sm = reinterpret_cast<uint16_t*>(zblk + (kPad ? 0 : 4));
    uint8_t* z_sm = reinterpret_cast<uint8_t*>(s_sm + (size_t)p.gc * NT * 16);
    float2* ps = reinterpret_cast<float2*>(z_sm + (size_t)p.gc * NT * 16);
    float* part = reinterpret_cast<float*>(ps + (size_t)M * GP);
    float* inv_rms = part + NT * MP * 16;  // RMSNorm prologue: 1 / rms per row, warp sums
    if (!kPad && threadIdx.x < 4) zblk[threadIdx.x] = make_uint4(0u, 0u, 0u, 0u);

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
            if (PRO && p.pro == kProRmsNorm) rms_rows(p, inv_rms);
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
                        if (PRO) {
                            const size_t k = (size_t)pa * 128 + q * 8;
                            const float ir = p.pro == kProRmsNorm ? inv_rms[b] : 0.f;
                            v[r][0] = prologue8(p, b, k, ir);
                            v[r][1] = prologue8(p, b, k + 64, ir);
                        } else {
                            const uint16_t* src = p.X + (size_t)b * p.K + (size_t)pa * 128 + q * 8;
                            v[r][0] = ld_cg16(src);
                            v[r][1] = ld_cg16(src + 64);
                        }
                        xo[r] = b * RS + (uu >> 3) * GC + (uu & 7);
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
                        xs[xo[r] + (kPad ? 9 : 8)] = v[r][1];  // chunk h + 8 (past the pad)
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
        // X of the lane's B column for the warp's record i: uint4 offset xo0[h] + i * xstep
        // (chunks 4c .. 4c+3 of the group; rows past M are never read, and clamped anyway).
        const int xstep = WT * GC;
        int xo0[NH];
#pragma unroll
        for (int h = 0; h < NH; ++h)
            xo0[h] = min(bl + 8 * h, M - 1) * RS + team * GC + c * 4 + (kPad ? c >> 1 : 0);

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
                uint4 v[4];
                if (!kPad) {  // every lane loads: X of its record, or the zero block
                    const uint4* src = gil == gi && bl + 8 * h < M ? xm[h] : zblk;
#pragma unroll
                    for (int q = 0; q < 4; ++q) v[q] = src[q];
                } else if (gil == gi && bl + 8 * h < M) {  // others take zeros, reading nothing
#pragma unroll
                    for (int q = 0; q < 4; ++q) v[q] = xm[h][q];
                } else {
#pragma unroll
                    for (int q = 0; q < 4; ++q) v[q] = make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    B[h][2 * q][0] = v[q].x;
                    B[h][2 * q][1] = v[q].y;
                    B[h][2 * q + 1][0] = v[q].z;
                    B[h][2 * q + 1][1] = v[q].w;
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

// The kernel instance for (BITS, MP, NT, PRO), as the address cudaLaunchKernelExC takes.
template <int BITS, int MP, bool PRO>
const void* pick_nt(int nt) {
    switch (nt) {
        case 1: return (const void*)gemm_kernel<BITS, MP, 1, PRO>;
        case 2: return (const void*)gemm_kernel<BITS, MP, 2, PRO>;
        case 4: return (const void*)gemm_kernel<BITS, MP, 4, PRO>;
        default: return (const void*)gemm_kernel<BITS, MP, 8, PRO>;
    }
}

template <int BITS, bool PRO>
const void* pick_mp(int mp, int nt) {
    switch (mp) {
        case 1: return pick_nt<BITS, 1, PRO>(nt);
        case 2: return pick_nt<BITS, 2, PRO>(nt);
        case 4: return pick_nt<BITS, 4, PRO>(nt);
        case 8: return pick_nt<BITS, 8, PRO>(nt);
        default: return pick_nt<BITS, 16, PRO>(nt);
    }
}

}  // namespace

// The prologue instances (defined in laq_gemm_prologue.cu).
const void* gemm_prologue_kernel(int bits, int mp, int nt);

}  // namespace laq
