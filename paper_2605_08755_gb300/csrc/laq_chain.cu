// laq_chain.cu -- a chain of WbG128 GEMVs (Eq. (1) weights, M = 1..4) in one persistent launch.
//
// A decode step multiplies the step's activations by every projection of every layer, in an
// order fixed by the model: q, k and v read the same input; o reads the attention output; gate
// and up read the same input; down reads their product.  Launched one kernel per projection,
// every GEMV pays a launch, a prologue that waits for its input, and a drain at the end, and
// the weight stream stops at each boundary.  This kernel runs the whole chain instead:
//
//  * One CTA of 16 warps per SM, all resident at once (cooperative launch).  The chain is cut
//    into stages at the entries that wait for their predecessors.  The units (16-column tiles)
//    of a stage are split into equal contiguous ranges, one per CTA, and the CTA's records
//    (tile x group of 128 rows) into 16 contiguous shares that differ by at most one record.
//
//  * Each warp streams its records, across all stages, through a private cp.async ring of
//    `stages` slots (the packed codes plus the record's 16 scales and zeros).  Weights never
//    depend on activations, so the ring runs ahead across stage boundaries: while a stage
//    waits for its input, the next stages' weights are landing.
//
//  * Stage boundary: every CTA bumps the stage's arrival counter in global memory after its Y
//    stores (release); a CTA with work in the next stage waits until the counter reaches the
//    grid size (acquire), then stages X in shared memory and runs its records.  Waits are
//    bounded: after about a second the kernel records LAQ_ERR_TIMEOUT in the workspace and
//    every CTA returns.
//
//  * The record arithmetic is that of laq_gemm.cu: one LOP3 per pair of codes gives the fp16
//    values c + q, an m16n8k16 MMA contracts them with raw x into D.  While X is staged, the
//    16 lanes that load a group's 256 bytes also sum P_g = sum_k c_k x_k and S_g = sum_k x_k,
//    and the epilogue of each block of groups that share the accumulator applies Eq. (1) as
//    y += s * (D - P - z S), with the block's scales and zeros copied aside from the ring.  A
//    tile whose groups are split between warps is summed in shared memory at the end of the
//    stage in warp order (deterministic, no atomics on Y).
//
//  * The last CTA to finish resets the counters, so the workspace is zero again for the next
//    call on the stream.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <memory>

#include "laq.h"
#include "laq_device.cuh"
#include "laq_internal.cuh"

// Compile-time trace points of thread 0 per stage (empty in the library build; a tracing build
// defines LAQ_CHAIN_TRACE(stage, point) to timestamp them).
#ifndef LAQ_CHAIN_TRACE
#define LAQ_CHAIN_TRACE(stage, point) \
    do {                              \
    } while (0)
#endif

namespace laq {

namespace {

constexpr int kChainWarps = 16;
constexpr int kChainThreads = kChainWarps * 32;
constexpr int kSzBytes = 48;                          // 16 fp16 scales + 16 u8 zeros
constexpr unsigned long long kWaitNs = 1000000000ull; // stage wait limit (1 s)
constexpr int kWaitSpins = 1 << 24;                   // and an iteration limit besides

// Chain workspace (uint32 words): [0] status, [1] finished CTAs, [2 + s] CTAs done with stage
// s, then at word flags_at(count): one flag per CTA (the last stage + 1 whose shared-tile part
// it has published), then at word parts_at(count): one part [MP][16] fp32 per CTA (64 words).
constexpr int kMaxGrid = 256;
__host__ __device__ constexpr int flags_at(int count) { return (2 + count + 3) / 4 * 4; }
__host__ __device__ constexpr int parts_at(int count) { return flags_at(count) + kMaxGrid; }

struct ChainEntryDev {
    const uint16_t* X;
    const uint8_t* packed;
    const uint16_t* s;
    const uint8_t* z;
    uint16_t* Y;
    int K, N;
    int xoff;   // offset of this entry's X in the stage's shared X area (16-byte units)
    int psoff;  // offset of its (S, P) pairs in the stage's table (one per row and group)
};

struct ChainStageDev {
    int e0, ne;   // entries [e0, e0 + ne)
    int records;  // (tile, group) records of the stage, entry by entry, tile-major
    int split;    // 1: CTA shares are equal record ranges (tiles may straddle CTAs); 0: whole
                  // tiles, split evenly by tile count
};

struct ChainParams {
    ChainEntryDev e[kChainMax];
    ChainStageDev st[kChainMax];
    uint32_t* ws;  // see chain workspace layout below
    int count, nstages, M, xs_bytes;
    Exps exps;
};
static_assert(sizeof(ChainParams) <= 32000, "kernel parameters must stay below 32 KB");

// The entry and stage descriptors as the kernel reads them: copied from the (large) parameter
// block into shared memory once, so stage set-up and cursor moves never wait on a
// constant-cache miss.
struct Tables {
    const ChainEntryDev* e;
    const ChainStageDev* st;
    int nstages;
};

template <int BITS>
struct Slot {
    static constexpr int kRec = RecordFmt<BITS>::kBytes;
    static constexpr int kBytes = kRec + kSzBytes;  // 816 (b = 3) or 1072 (b = 4), 16-aligned
    // Ring slots per warp.  One record is consumed while the others are in flight: 16 warps x
    // 7 x 816 B (b = 3) or 5 x 1072 B (b = 4) ~ 90 KB per SM, above the ~64 KB that HBM's
    // bandwidth x latency needs per SM.  A compile-time depth keeps cp.async.wait_group an
    // immediate (a runtime count costs an indirect branch per record).
    static constexpr int kRing = BITS == 3 ? 8 : 6;
};

// Ring slots per warp of the chain kernel at `bits` (host side).
constexpr int chain_ring(int bits) { return bits == 3 ? Slot<3>::kRing : Slot<4>::kRing; }

__device__ __forceinline__ unsigned long long globaltimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t ld_relaxed(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void red_release_add(uint32_t* p, uint32_t v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ float ld_cg_f32(const float* p) {
    float v;
    asm volatile("ld.global.cg.f32 %0, [%1];" : "=f"(v) : "l"(p) : "memory");
    return v;
}

// Wait until *cnt >= target.  Returns false when an error is already recorded in the status
// word (read together with the first poll, so a recorded error stops every later stage; while
// waiting it is re-read every 32 polls, so that each poll is one L2 round trip), or when the
// wait runs out (after recording LAQ_ERR_TIMEOUT).
__device__ bool wait_count(const uint32_t* cnt, uint32_t target, uint32_t* status) {
    const unsigned long long t0 = globaltimer();
    const uint32_t st0 = ld_relaxed(status);
    const uint32_t c0 = ld_acquire(cnt);
    if (st0 != 0u) return false;
    if (c0 >= target) return true;
    for (int spin = 0; spin < kWaitSpins; ++spin) {
        if (ld_acquire(cnt) >= target) return true;
        if ((spin & 31) == 31) {
            if (ld_relaxed(status) != 0u) return false;
            if (globaltimer() - t0 > kWaitNs) break;
        }
    }
    atomicCAS(status, 0u, (uint32_t)LAQ_ERR_TIMEOUT);
    return false;
}

// Wait until *flag == value (a CTA's published part of stage value - 1), with the limits and
// the status checks of wait_count.
__device__ bool wait_flag(const uint32_t* flag, uint32_t value, uint32_t* status) {
    const unsigned long long t0 = globaltimer();
    const uint32_t st0 = ld_relaxed(status);
    const uint32_t f0 = ld_acquire(flag);
    if (st0 != 0u) return false;
    if (f0 == value) return true;
    for (int spin = 0; spin < kWaitSpins; ++spin) {
        if (ld_acquire(flag) == value) return true;
        if ((spin & 31) == 31) {
            if (ld_relaxed(status) != 0u) return false;
            if (globaltimer() - t0 > kWaitNs) break;
        }
    }
    atomicCAS(status, 0u, (uint32_t)LAQ_ERR_TIMEOUT);
    return false;
}

// The end of CTA b's contiguous share of a stage's `records` records (64-bit products).
__device__ __forceinline__ int cta_end(int records, int b) {
    return (int)((long long)records * (b + 1) / gridDim.x);
}

// A warp's position in its record stream: stage s, entry e, tile (16-column block of the entry)
// and group g.  A stage's records are its entries' (tile, group) records in order, tile-major;
// CTA b takes the contiguous share [R b / P, R (b + 1) / P) of the stage's R records (a tile
// may straddle two CTAs), and warp w the contiguous share [n w / 16, n (w + 1) / 16) of the
// CTA's n records, so CTAs differ by at most one record, and so do the warps of a CTA.
struct Cursor {
    int s;     // stage
    int left;  // records of the share from the current one to its end
    int e;     // entry
    int tile;  // tile within the entry
    int g;     // group within the tile
    int G, T;  // groups and tiles of the entry
};

// Place the cursor at the first record of warp w's share of stage c.s; false if it is empty.
__device__ bool cursor_begin(Cursor& c, const Tables& p, const int4* range, int w) {
    const int4 rg = range[c.s];  // CTA's first record, end record, record count
    const int a = (rg.z * w) >> 4, b = (rg.z * (w + 1)) >> 4;
    c.left = b - a;
    if (c.left <= 0) return false;
    int r = rg.x + a;
    const ChainStageDev st = p.st[c.s];
    for (int q = 0; q < st.ne; ++q) {
        const int e = st.e0 + q;
        const int T = p.e[e].N >> 4, G = p.e[e].K >> 7;
        if (r < T * G) {
            const int t = r / G;
            c.e = e;
            c.G = G;
            c.T = T;
            c.tile = t;
            c.g = r - t * G;
            return true;
        }
        r -= T * G;
    }
    c.left = 0;  // not reached: the share lies inside the stage
    return false;
}

// Move to the first group of the next tile of the share (the caller has checked that records
// remain): true if the entry changed.
__device__ bool cursor_next_tile(Cursor& c, const Tables& p) {
    c.g = 0;
    if (++c.tile < c.T) return false;
    ++c.e;
    c.tile = 0;
    c.G = p.e[c.e].K >> 7;
    c.T = p.e[c.e].N >> 4;
    return true;
}

// Step to the next record of the share (the caller has checked left > 1): 0 within the tile,
// 1 to the first group of the next tile of the entry, 2 to the first record of a new entry.
__device__ int cursor_step(Cursor& c, const Tables& p) {
    --c.left;
    if (++c.g < c.G) return 0;
    return cursor_next_tile(c, p) ? 2 : 1;
}

// The warp's record stream on the copy side of the ring (the compute side walks the same
// shares).  A slot holds the record's packed words followed by its 16 scales and 16 zeros;
// each lane copies 16-byte pieces of it from per-lane source pointers:
//   b = 3: piece l (record bytes 16 l), then piece 32 + l for l < 19 (record bytes 512 + 16 l
//          for l < 16, the scales for l = 16, 17, the zeros for l = 18);
//   b = 4: pieces l and 32 + l (record bytes 16 l and 512 + 16 l), then for l < 3 the scales
//          (l = 0, 1) or the zeros (l = 2).
template <int BITS>
struct RecordStream {
    static constexpr int REC = RecordFmt<BITS>::kBytes;
    Cursor c;
    bool live;
    const uint8_t* p1;
    const uint8_t* p2;
    const uint8_t* p3;
    long long st2, st3;  // bytes to the next group's piece (p1 always moves by REC)

    __device__ void point(const Tables& p, int lane) {
        const ChainEntryDev& E = p.e[c.e];
        const uint8_t* rec = E.packed + ((size_t)c.tile * c.G + c.g) * REC;
        const size_t gz = (size_t)c.g * E.N + (size_t)c.tile * 16;  // (group, column)
        const uint8_t* sp = reinterpret_cast<const uint8_t*>(E.s + gz);
        const uint8_t* zp = E.z + gz;
        p1 = rec + lane * 16;
        if (BITS == 3) {
            p2 = lane < 16 ? rec + 512 + lane * 16 : lane < 18 ? sp + (lane - 16) * 16 : zp;
            st2 = lane < 16 ? REC : lane < 18 ? 2LL * E.N : (long long)E.N;
            p3 = p2;
            st3 = 0;
        } else {
            p2 = rec + 512 + lane * 16;
            st2 = REC;
            p3 = lane < 2 ? sp + lane * 16 : zp;
            st3 = lane < 2 ? 2LL * E.N : (long long)E.N;
        }
    }
    __device__ void seek(const Tables& p, const int4* range, int w, int lane) {
        while (c.s < p.nstages && !cursor_begin(c, p, range, w)) ++c.s;
        live = c.s < p.nstages;
        if (live) point(p, lane);
    }
    __device__ void advance(const Tables& p, const int4* range, int w, int lane) {
        if (c.left > 1) {
            if (cursor_step(c, p) == 0) {
                p1 += REC;
                p2 += st2;
                p3 += st3;
            } else {
                point(p, lane);
            }
        } else {
            ++c.s;
            seek(p, range, w, lane);
        }
    }
};

template <int BITS, int MP>
__global__ void __launch_bounds__(kChainThreads, 1) chain_kernel(const __grid_constant__ ChainParams p) {
    using F = RecordFmt<BITS>;
    constexpr int SLOT = Slot<BITS>::kBytes;
    constexpr int WPL = BITS == 4 ? 8 : 6;
    constexpr int GPA = 8 / MP;  // groups sharing one accumulator (MMA columns), MP <= 4

    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = lane & 3, R = lane >> 2;
    const int M = p.M;
    constexpr int S = Slot<BITS>::kRing;
    uint32_t* status = p.ws;

    // shared memory: ring [16][S][slot] | X [xs_bytes] | zero block (64 B)
    //                | (S, P) per (entry, row, group) [xs_bytes / 256] float2
    //                | scales and zeros of each warp's current block [16][GPA][48 B]
    //                | split-tile partial sums [32][MP][16] fp32 | their tile keys [32]
    //                | this CTA's (first unit, end unit, records) per stage [nstages] int4
    //                | entry descriptors [count] | stage descriptors [nstages] | flag
    uint8_t* ring = smem;
    uint4* xs = reinterpret_cast<uint4*>(smem + (size_t)kChainWarps * S * SLOT);
    uint4* zblk = xs + p.xs_bytes / 16;
    float2* ps = reinterpret_cast<float2*>(zblk + 4);
    uint4* sbuf_all = reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(ps) +
                                               ((p.xs_bytes / 256 * 8 + 15) & ~15));
    float* red = reinterpret_cast<float*>(sbuf_all + kChainWarps * GPA * 3);
    int* keys = reinterpret_cast<int*>(red + (2 * kChainWarps + 1) * MP * 16);
    int4* range = reinterpret_cast<int4*>(keys + 2 * kChainWarps);
    ChainEntryDev* ent = reinterpret_cast<ChainEntryDev*>(range + p.nstages);
    ChainStageDev* stg = reinterpret_cast<ChainStageDev*>(ent + p.count);
    int* flag = reinterpret_cast<int*>(stg + p.nstages);
    if (threadIdx.x < 4) zblk[threadIdx.x] = make_uint4(0u, 0u, 0u, 0u);
    for (int i = threadIdx.x; i < p.count; i += kChainThreads) ent[i] = p.e[i];
    for (int i = threadIdx.x; i < p.nstages; i += kChainThreads) stg[i] = p.st[i];
    __syncthreads();
    const Tables tb{ent, stg, p.nstages};
    for (int s = threadIdx.x; s < p.nstages; s += kChainThreads) {
        const ChainStageDev st = stg[s];
        int r0, r1;
        if (st.split) {
            r0 = blockIdx.x == 0 ? 0 : cta_end(st.records, blockIdx.x - 1);
            r1 = cta_end(st.records, blockIdx.x);
        } else {
            // whole tiles: units [u0, u1) of the stage, as records
            int units = 0;
            for (int q = 0; q < st.ne; ++q) units += ent[st.e0 + q].N >> 4;
            const int u0 = blockIdx.x == 0 ? 0 : cta_end(units, blockIdx.x - 1);
            const int u1 = cta_end(units, blockIdx.x);
            r0 = r1 = 0;
            int ubase = 0, rbase = 0;
            for (int q = 0; q < st.ne; ++q) {
                const int T = ent[st.e0 + q].N >> 4, G = ent[st.e0 + q].K >> 7;
                if (u0 >= ubase && u0 < ubase + T) r0 = rbase + (u0 - ubase) * G;
                if (u1 >= ubase && u1 <= ubase + T) r1 = rbase + (u1 - ubase) * G;
                ubase += T;
                rbase += T * G;
            }
            if (u1 <= u0) r1 = r0;
        }
        range[s] = make_int4(r0, r1, r1 - r0, 0);
    }
    __syncthreads();

    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(ring) +
                            (uint32_t)(warp * S * SLOT);
    const uint8_t* ring_w = ring + (size_t)warp * S * SLOT;
    uint4* sbuf = sbuf_all + warp * GPA * 3;  // [GPA][3] 16-byte pieces: scales x 2, zeros
    // lanes that copied a scale / zero piece of each slot, and which piece
    const int szp = BITS == 3 ? lane - 16 : lane;
    const bool sz_lane = szp >= 0 && szp < 3;

    // Copy side of the ring: the next record of the warp's stream into the next slot (an
    // empty group once the stream is exhausted, so group counting stays uniform).
    RecordStream<BITS> is;
    is.c.s = 0;
    is.seek(tb, range, warp, lane);
    int islot = 0;
    auto issue = [&]() {
        if (is.live) {
            const uint32_t dst = ring_s + (uint32_t)(islot * SLOT) + lane * 16;
            cp_async16(dst, is.p1);
            if (BITS == 3) {
                if (lane < 19) cp_async16(dst + 512, is.p2);
            } else {
                cp_async16(dst + 512, is.p2);
                if (lane < 3) cp_async16(dst + 1024, is.p3);
            }
            is.advance(tb, range, warp, lane);
        }
        cp_async_commit();
        islot = islot + 1 == S ? 0 : islot + 1;
    };
    // Records in flight ahead of the one being consumed.
    constexpr int ahead = S - 1;
    for (int q = 0; q < ahead; ++q) issue();
    int rslot = 0;

    const int bl = R / GPA;   // batch row of this lane's B column
    const int gil = R % GPA;  // group position of this lane's B column
    bool ok = true;

    for (int s = 0; s < p.nstages; ++s) {
        const ChainStageDev st = stg[s];
        const int r0 = range[s].x, r1 = range[s].y;
        if (r1 <= r0) {
            // Nothing of this stage here: report it done at once.
            if (threadIdx.x == 0) red_release_add(p.ws + 2 + s, 1u);
            continue;
        }
        LAQ_CHAIN_TRACE(s, 0);
        if (threadIdx.x == 0) {
            bool good = true;
            if (s > 0) good = wait_count(p.ws + 2 + (s - 1), gridDim.x, status);
            *flag = good ? 1 : 0;
        }
        if (threadIdx.x < 2 * kChainWarps) keys[threadIdx.x] = -1;
        __syncthreads();  // the wait is over; every warp is done with the previous stage's X
        LAQ_CHAIN_TRACE(s, 1);
        if (*flag == 0) {
            ok = false;
            break;
        }

        // X of every entry of the stage that has a record here (M rows of K fp16, contiguous),
        // through L2 (ld.global.cg: written by other SMs during this kernel).
        {
            int rbase = 0;
            for (int q = 0; q < st.ne; ++q) {
                const ChainEntryDev& E = ent[st.e0 + q];
                const int nrec = (E.N >> 4) * (E.K >> 7);
                if (rbase < r1 && rbase + nrec > r0) {
                    // 16-byte chunk uu holds x[8 uu .. 8 uu + 7] of the [M][K] rows: chunk
                    // uu % 16 of group uu / 16 (row b, group g), rows 8 (uu % 16) + e of the
                    // group, i.e. pairs 4 (uu % 4) + w for its four 32-bit words w.  The 16
                    // chunks of a group sit in 16 consecutive lanes, which sum
                    // S_g = sum_k x_k and P_g = sum_k c_k x_k by shuffles.
                    const int n16 = M * E.K / 8;  // a multiple of 16
                    const uint8_t* src = reinterpret_cast<const uint8_t*>(E.X);
                    uint4* dst = xs + E.xoff;
                    for (int u = 0; u < n16; u += 4 * kChainThreads) {
                        uint4 v[4];
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            const int uu = u + r * kChainThreads + (int)threadIdx.x;
                            v[r] = uu < n16 ? ld_cg16(src + (size_t)uu * 16)
                                            : make_uint4(0u, 0u, 0u, 0u);
                        }
                        // a group's 16 chunks are 16 aligned lanes: n16 is a multiple of 16, so
                        // a warp's lanes are either all past n16 or share one boundary at a
                        // 16-lane half
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            // (warp-uniform) nothing of this batch for this warp
                            if (u + r * kChainThreads + warp * 32 >= n16) break;
                            const int uu = u + r * kChainThreads + (int)threadIdx.x;
                            const uint32_t w4[4] = {v[r].x, v[r].y, v[r].z, v[r].w};
                            float sx = 0.f, px = 0.f;
#pragma unroll
                            for (int w = 0; w < 4; ++w) {
                                const float2 f =
                                    __half22float2(*reinterpret_cast<const __half2*>(&w4[w]));
                                const float pair = f.x + f.y;
                                sx += pair;
                                px = fmaf(row_offset<BITS>((uu & 3) * 4 + w), pair, px);
                            }
#pragma unroll
                            for (int o = 1; o < 16; o <<= 1) {
                                sx += __shfl_xor_sync(0xffffffffu, sx, o);
                                px += __shfl_xor_sync(0xffffffffu, px, o);
                            }
                            if (uu < n16) {
                                dst[uu] = v[r];
                                if ((uu & 15) == 0) ps[E.psoff + (uu >> 4)] = make_float2(sx, px);
                            }
                        }
                    }
                }
                rbase += nrec;
            }
        }
        __syncthreads();
        LAQ_CHAIN_TRACE(s, 2);
        LAQ_CHAIN_TRACE(s, 3);

        // This warp's share of the stage, a block of up to GPA records (consecutive groups of
        // one tile, sharing the accumulator columns) at a time.
        Cursor cc;
        cc.s = s;
        if (cursor_begin(cc, tb, range, warp)) {
            int xoff = ent[cc.e].xoff, pso = ent[cc.e].psoff, G = cc.G;
            int piece_g0 = cc.g;  // first group of the current piece (run of one tile)
            bool first_piece = true;
            float yacc[4] = {0.f, 0.f, 0.f, 0.f};
            for (;;) {
                const int gb = cc.g;  // first group of the block
                const int nb = min(GPA, min(G - gb, cc.left));
                const int rs0 = rslot;
                float D[2][4];
#pragma unroll
                for (int a = 0; a < 2; ++a)
#pragma unroll
                    for (int v = 0; v < 4; ++v) D[a][v] = 0.f;
#pragma unroll
                for (int gi = 0; gi < GPA; ++gi) {
                    if (gi < nb) {
                        __syncwarp();  // every lane is done with the slot the next copy overwrites
                        issue();
                        asm volatile("cp.async.wait_group %0;\n" ::"n"(ahead) : "memory");
                        uint32_t B[8][2];
                        {
                            const bool act = gil == gi && bl < M;
                            const uint4* src =
                                act ? xs + xoff + (size_t)(bl * G + gb + gi) * 16 + c * 4 : zblk;
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const uint4 v = src[q];
                                B[2 * q][0] = v.x;
                                B[2 * q][1] = v.y;
                                B[2 * q + 1][0] = v.z;
                                B[2 * q + 1][1] = v.w;
                            }
                        }
                        const uint8_t* slot = ring_w + (size_t)rslot * SLOT;
                        // this lane's scale / zero piece of the record, for the block epilogue
                        if (sz_lane)
                            sbuf[gi * 3 + szp] =
                                *reinterpret_cast<const uint4*>(slot + F::kBytes + szp * 16);
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
                            mma16816(D[j & 1], a[j][0], a[j][1], a[j][2], a[j][3], B[j][0],
                                     B[j][1]);
                        rslot = rslot + 1 == S ? 0 : rslot + 1;
                    }
                }
                __syncwarp();  // the scales and zeros of the block's slots came from other lanes

                // Eq. (1) per block column (a group of one batch row): y += s (D - P - z S).
                // Value v of the lane is row R + 8 (v >> 1), column 2c + (v & 1), i.e. record
                // (column % GPA) of the block and batch row column / GPA.
#pragma unroll
                for (int v1 = 0; v1 < 2; ++v1) {
                    const int col = 2 * c + v1;
                    const int b = col / GPA, rec = col % GPA;
                    if (b < M && rec < nb) {
                        const uint8_t* sz = reinterpret_cast<const uint8_t*>(sbuf + rec * 3);
                        const uint16_t* ssl = reinterpret_cast<const uint16_t*>(sz);
                        const float s0 = __half2float(__ushort_as_half(ssl[R]));
                        const float s1 = __half2float(__ushort_as_half(ssl[R + 8]));
                        const float z0 = (float)sz[32 + R], z1 = (float)sz[32 + R + 8];
                        const float2 sp = ps[pso + b * G + gb + rec];  // (S, P)
                        const float d0 = D[0][v1] + D[1][v1] - sp.y;
                        const float d1 = D[0][v1 + 2] + D[1][v1 + 2] - sp.y;
                        yacc[v1] = fmaf(s0, fmaf(-z0, sp.x, d0), yacc[v1]);
                        yacc[v1 + 2] = fmaf(s1, fmaf(-z1, sp.x, d1), yacc[v1 + 2]);
                    }
                }

                cc.g += nb;
                cc.left -= nb;
                if (cc.g == G || cc.left == 0) {
                    // End of a piece.  Columns of one batch row -> one value per (row, column).
                    float y0 = yacc[0] + yacc[1];
                    float y1 = yacc[2] + yacc[3];
                    if (GPA >= 4) {
                        y0 += __shfl_xor_sync(0xffffffffu, y0, 1);
                        y1 += __shfl_xor_sync(0xffffffffu, y1, 1);
                    }
                    if (GPA >= 8) {
                        y0 += __shfl_xor_sync(0xffffffffu, y0, 2);
                        y1 += __shfl_xor_sync(0xffffffffu, y1, 2);
                    }
                    const int b = (2 * c) / GPA;
                    const bool writer = (2 * c) % GPA == 0 && b < M;
                    if (piece_g0 == 0 && cc.g == G) {
                        // the whole tile: store
                        if (writer) {
                            const ChainEntryDev& E = ent[cc.e];
                            uint16_t* y = E.Y + (size_t)b * E.N + (size_t)cc.tile * 16;
                            y[R] = __half_as_ushort(__float2half_rn(y0));
                            y[R + 8] = __half_as_ushort(__float2half_rn(y1));
                        }
                    } else {
                        // part of a tile shared with neighbouring warps: summed at stage end
                        const int sl = 2 * warp + (first_piece ? 0 : 1);
                        if (writer) {
                            float* rw = red + (size_t)sl * MP * 16;
                            rw[b * 16 + R] = y0;
                            rw[b * 16 + R + 8] = y1;
                        }
                        if (lane == 0) keys[sl] = (cc.e << 20) | cc.tile;
                    }
#pragma unroll
                    for (int v = 0; v < 4; ++v) yacc[v] = 0.f;
                    first_piece = false;
                    if (cc.left == 0) break;
                    if (cursor_next_tile(cc, tb)) {
                        xoff = ent[cc.e].xoff;
                        pso = ent[cc.e].psoff;
                        G = cc.G;
                    }
                    piece_g0 = 0;
                }
            }
        }
        LAQ_CHAIN_TRACE(s, 4);
        __syncthreads();  // partial sums of shared tiles are in red
        LAQ_CHAIN_TRACE(s, 5);

        // Tiles shared by several warps: sum their parts in slot (= warp) order.  Every warp
        // sees the 32 slot keys, one per lane; slots with equal keys are one tile's parts.  A
        // tile inside this CTA's records is stored; the CTA's last tile, if it runs past the
        // CTA's records, is published for the CTA that owns its end; the CTA's first tile, if
        // it began in earlier CTAs, is finished here with their published parts.
        float* pub = reinterpret_cast<float*>(p.ws + parts_at(p.count));  // [P][MP][16]
        uint32_t* pflag = p.ws + flags_at(p.count);                       // [P]
        {
            const int kl = keys[lane];
            const unsigned same = __match_any_sync(0xffffffffu, kl);
            const int firstl = kl >= 0 && (same & ((1u << lane) - 1u)) == 0u;
            for (int idx = threadIdx.x; idx < 2 * kChainWarps * M * 16; idx += kChainThreads) {
                const int sl = idx / (M * 16), r = idx - sl * (M * 16);
                const int key = __shfl_sync(0xffffffffu, kl, sl);
                const int first = __shfl_sync(0xffffffffu, firstl, sl);
                const unsigned m = __shfl_sync(0xffffffffu, same, sl);
                if (first) {
                    // all 32 slots loaded independently (the parts of a tile are the slots
                    // in m), then summed in slot order
                    float part[2 * kChainWarps];
#pragma unroll
                    for (int j = 0; j < 2 * kChainWarps; ++j)
                        part[j] = (m >> j) & 1u ? red[(size_t)j * MP * 16 + r] : 0.f;
                    float acc = 0.f;
#pragma unroll
                    for (int j = 0; j < 2 * kChainWarps; ++j) acc += part[j];
                    const int e = key >> 20, tile = key & 0xfffff;
                    int rbase = 0;  // first record of entry e in the stage
                    for (int q = st.e0; q < e; ++q) rbase += (ent[q].N >> 4) * (ent[q].K >> 7);
                    const int G = ent[e].K >> 7;
                    const int tfirst = rbase + tile * G, tend = tfirst + G;
                    if (tend > r1) {
                        pub[(size_t)blockIdx.x * MP * 16 + r] = acc;  // published below
                    } else if (tfirst < r0) {
                        red[(size_t)(2 * kChainWarps) * MP * 16 + r] = acc;  // finished below
                    } else {
                        const ChainEntryDev& E = ent[e];
                        const int bb = r >> 4, n = r & 15;
                        E.Y[(size_t)bb * E.N + (size_t)tile * 16 + n] =
                            __half_as_ushort(__float2half_rn(acc));
                    }
                }
            }
        }
        if (st.split) {
        __syncthreads();  // this CTA's published part is written
        // Publish at once (every CTA, every split stage), before waiting on anyone: owners wait
        // only for parts, never for each other's owned tiles.
        if (threadIdx.x == 0) st_release(pflag + blockIdx.x, (uint32_t)(s + 1));
        {
            // The CTA's first record starts a tile that began in earlier CTAs?
            int rbase = 0, q = 0;
            for (; q < st.ne; ++q) {
                const int nrec = (ent[st.e0 + q].N >> 4) * (ent[st.e0 + q].K >> 7);
                if (r0 < rbase + nrec) break;
                rbase += nrec;
            }
            const ChainEntryDev& E = ent[st.e0 + q];
            const int G = E.K >> 7, tile = (r0 - rbase) / G;
            const int tfirst = rbase + tile * G, tend = tfirst + G;
            if (tfirst < r0 && tend <= r1 && threadIdx.x < M * 16) {
                const int r = threadIdx.x;
                // parts of the CTAs before this one whose records reach into the tile,
                // in CTA order
                int b0 = blockIdx.x - 1;
                while (b0 > 0 && cta_end(st.records, b0 - 1) > tfirst) --b0;
                float acc = 0.f;
                bool good = true;
                for (int b = b0; b < (int)blockIdx.x && good; ++b) {
                    const int bs = b == 0 ? 0 : cta_end(st.records, b - 1);
                    if (cta_end(st.records, b) == bs) continue;  // no records: nothing published
                    good = wait_flag(pflag + b, (uint32_t)(s + 1), status);
                    if (good) acc += ld_cg_f32(pub + (size_t)b * MP * 16 + r);
                }
                acc += red[(size_t)(2 * kChainWarps) * MP * 16 + r];
                if (good) {
                    const int bb = r >> 4, n = r & 15;
                    E.Y[(size_t)bb * E.N + (size_t)tile * 16 + n] =
                        __half_as_ushort(__float2half_rn(acc));
                }
            }
        }
        }
        __syncthreads();  // every Y value finished by this CTA is stored
        LAQ_CHAIN_TRACE(s, 7);
        // Release: the CTA's Y stores (ordered before by the barrier) become visible before
        // the arrival does.
        if (threadIdx.x == 0) red_release_add(p.ws + 2 + s, 1u);
        LAQ_CHAIN_TRACE(s, 6);
    }

    asm volatile("cp.async.wait_all;\n" ::: "memory");
    if (!ok) return;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const uint32_t prev = atomicAdd(p.ws + 1, 1u);
        if (prev == gridDim.x - 1) {
            // Every CTA is past its last wait: leave the counters at zero for the next call.
            for (int s = 0; s < p.nstages; ++s) p.ws[2 + s] = 0u;
            for (int b = 0; b < (int)gridDim.x; ++b) p.ws[flags_at(p.count) + b] = 0u;
            p.ws[1] = 0u;
            __threadfence();
        }
    }
}

using ChainFn = void (*)(ChainParams);

template <int BITS>
ChainFn pick_chain(int mp) {
    switch (mp) {
        case 1: return chain_kernel<BITS, 1>;
        case 2: return chain_kernel<BITS, 2>;
        default: return chain_kernel<BITS, 4>;
    }
}

std::atomic<size_t> g_chain_attr[2][3];  // dynamic shared memory already granted per instance

}  // namespace

size_t chain_workspace_bytes(int count) {
    return ((size_t)parts_at(count) + (size_t)kMaxGrid * 4 * 16) * 4;
}
size_t chain_workspace_zeroed_bytes(int count) { return (size_t)parts_at(count) * 4; }

size_t chain_smem_bytes(int bits, int M, int xs_bytes, int nstages, int count) {
    const int stages = chain_ring(bits);
    const int mp = M <= 1 ? 1 : M <= 2 ? 2 : 4;
    const size_t slot = (size_t)(bits == 4 ? 1024 : 768) + kSzBytes;
    return (size_t)kChainWarps * stages * slot + (size_t)xs_bytes + 64 +
           ((size_t)xs_bytes / 256 * 8 + 15) / 16 * 16 + (size_t)kChainWarps * (8 / mp) * 48 +
           (size_t)(2 * kChainWarps + 1) * mp * 16 * 4 + (size_t)2 * kChainWarps * 4 +
           (size_t)nstages * 16 + (size_t)count * sizeof(ChainEntryDev) +
           (size_t)nstages * sizeof(ChainStageDev) + 16;
}

cudaError_t launch_chain(const ChainLaunch& L, int num_sms, cudaStream_t stream) {
    // The parameter block is large (about 26 KB): built on the heap, copied by the launch.
    std::unique_ptr<ChainParams> holder(new ChainParams());
    ChainParams& P = *holder;
    for (int i = 0; i < L.count; ++i) {
        const ChainEntry& E = L.e[i];
        P.e[i] = ChainEntryDev{E.X, E.packed, E.s, E.z, E.Y, E.K, E.N, E.xoff, E.psoff};
    }
    for (int s = 0; s < L.nstages; ++s) P.st[s] = ChainStageDev{L.st[s].e0, L.st[s].ne, L.st[s].records, L.st[s].split};
    P.ws = L.ws;
    P.count = L.count;
    P.nstages = L.nstages;
    P.M = L.M;
    P.xs_bytes = L.xs_bytes;
    P.exps = exps_for(L.bits);

    const int mp = L.M <= 1 ? 1 : L.M <= 2 ? 2 : 4;
    const ChainFn fn = L.bits == 4 ? pick_chain<4>(mp) : pick_chain<3>(mp);
    const size_t smem = chain_smem_bytes(L.bits, L.M, L.xs_bytes, L.nstages, L.count);
    std::atomic<size_t>& granted = g_chain_attr[L.bits == 4][mp == 1 ? 0 : mp == 2 ? 1 : 2];
    cudaError_t err = cudaSuccess;
    if (granted.load() < smem) {
        err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        granted.store(smem);
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)num_sms);
    cfg.blockDim = dim3(kChainThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    void* args[] = {&P};
    return cudaLaunchKernelExC(&cfg, (const void*)fn, args);
}

}  // namespace laq
