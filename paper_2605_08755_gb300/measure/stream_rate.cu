// stream_rate.cu -- the W3 record loop fed from HBM by two copy schemes, one CTA per SM.
//
// Each SM streams its own contiguous range of 816-byte W3 records (768 bytes of codes + 48 of
// scales and zeros, as in the planned pass's streams; 4.2 GB in all, far beyond L2) and runs the
// record loop on them (the mask-and-or extraction and 8 mma.sync per record).  Two schemes:
//   A. per-warp cp.async rings (the form of laq_gemm_wxg128): every warp copies its own next
//      records (a lane's 16 + 8 bytes of codes) into a private ring of shared memory and waits
//      with cp.async.wait_group;
//   B. one producer warp issuing cp.async.bulk copies of 16-record rounds (13 KB) into an
//      mbarrier ring (the form of laq_pass_run): each of 16 consumer warps takes one record of
//      every round, in blocks of 8 rounds per wait.
// Reported: the bytes streamed over the kernel's time (CUDA events), TB/s.  Every wait is
// bounded.
//
//   nvcc -gencode arch=compute_103a,code=sm_103a -O3 -o /tmp/stream_rate \
//       paper_2605_08755_gb300/measure/stream_rate.cu && /tmp/stream_rate
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>

namespace {

constexpr int kRB = 816;       // record bytes
constexpr int kCodes = 768;    // of which codes
constexpr int kWarps = 16;

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// The record's 32 A registers from a lane's 6 code words (plain shifts), then its 8 MMAs.
__device__ __forceinline__ void record(const uint32_t (&wd)[6], float (&D)[4][4], uint32_t b0,
                                       uint32_t b1) {
    const uint32_t e1 = 0x60006000u, e4 = 0x54005400u, e7 = 0x48004800u;
    uint32_t rp[16][2];
#pragma unroll
    for (int w = 0; w < 6; ++w) {
        const uint32_t u = wd[w] >> 9;
        rp[w][0] = (wd[w] & 0x000e000eu) | e1;
        rp[6 + w][0] = (wd[w] & 0x00700070u) | e4;
        rp[w][1] = (u & 0x000e000eu) | e1;
        rp[6 + w][1] = (u & 0x00700070u) | e4;
    }
#pragma unroll
    for (int q = 0; q < 3; ++q) {
        rp[12 + q][0] = (wd[2 * q] & 0x03800380u) | e7;
        rp[12 + q][1] = (wd[2 * q + 1] & 0x03800380u) | e7;
    }
    rp[15][0] = ((wd[0] << 4) & 0x00100010u) | ((wd[1] << 5) & 0x00200020u) |
                ((wd[2] << 6) & 0x00400040u) | e4;
    rp[15][1] = ((wd[3] << 4) & 0x00100010u) | ((wd[4] << 5) & 0x00200020u) |
                ((wd[5] << 6) & 0x00400040u) | e4;
#pragma unroll
    for (int j = 0; j < 8; ++j)
        mma16816(D[j & 3], rp[2 * j][0], rp[2 * j][1], rp[2 * j + 1][0], rp[2 * j + 1][1], b0, b1);
}

__device__ __forceinline__ void load_words(const uint8_t* rec, int lane, uint32_t (&wd)[6]) {
    const uint4 c0 = *reinterpret_cast<const uint4*>(rec + lane * 16);
    const uint2 c1 = *reinterpret_cast<const uint2*>(rec + 512 + lane * 8);
    wd[0] = c0.x; wd[1] = c0.y; wd[2] = c0.z; wd[3] = c0.w; wd[4] = c1.x; wd[5] = c1.y;
}

// A. Per-warp cp.async rings of S records.
template <int S>
__global__ void __launch_bounds__(kWarps * 32, 1) per_warp(const uint8_t* buf, int64_t per_sm,
                                                           float* sink) {
    extern __shared__ __align__(128) uint8_t sm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t per_warp_recs = per_sm / kWarps;
    const uint8_t* src = buf + ((int64_t)blockIdx.x * per_sm + warp * per_warp_recs) * kRB;
    uint8_t* ring = sm + warp * S * kCodes;
    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(ring);
    auto issue = [&](int64_t i) {
        const uint8_t* r = src + i * kRB;
        const uint32_t d = ring_s + (uint32_t)((i % S) * kCodes);
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d + lane * 16),
                     "l"(r + lane * 16) : "memory");
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(d + 512 + lane * 8),
                     "l"(r + 512 + lane * 8) : "memory");
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    float D[4][4] = {};
    const uint32_t b0 = 0x3c003c00u, b1 = 0x3c003c00u ^ (uint32_t)lane;
    for (int i = 0; i < S - 1; ++i) issue(i);
    for (int64_t i = 0; i < per_warp_recs; ++i) {
        if (i + S - 1 < per_warp_recs) issue(i + S - 1);
        else asm volatile("cp.async.commit_group;" ::: "memory");  // keep the group count
        asm volatile("cp.async.wait_group %0;" ::"n"(S - 1) : "memory");
        __syncwarp();
        uint32_t wd[6];
        load_words(ring + (i % S) * kCodes, lane, wd);
        record(wd, D, b0, b1);
        __syncwarp();
    }
    float s = 0.f;
    for (int c = 0; c < 4; ++c) s += D[c][0] + D[c][1] + D[c][2] + D[c][3];
    if (s == 12345.f) sink[0] = s;
}

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    for (int sp = 0; sp < (1 << 22); ++sp) {
        uint32_t ok;
        asm volatile("{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
                     "selp.u32 %0, 1, 0, p;\n}\n"
                     : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
        if (ok) return true;
    }
    return false;
}

// B. One producer warp, cp.async.bulk rounds of 16 records into NS slots; 16 consumer warps take
// record `warp` of each round, waiting for 8 rounds at a time.
template <int NS>
__global__ void __launch_bounds__((kWarps + 1) * 32, 1) bulk_ring(const uint8_t* buf,
                                                                  int64_t per_sm, float* sink,
                                                                  int* status) {
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ __align__(8) uint64_t full[NS], empty[NS];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int SLOT = kWarps * kRB;
    const int64_t rounds = per_sm / kWarps;
    if (threadIdx.x == 0) {
        for (int i = 0; i < NS; ++i) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(
                (uint32_t)__cvta_generic_to_shared(&full[i])));
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(
                (uint32_t)__cvta_generic_to_shared(&empty[i])), "r"(kWarps));
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(sm);
    const uint8_t* src = buf + (int64_t)blockIdx.x * per_sm * kRB;
    bool ok = true;
    if (warp == kWarps) {
        if (lane == 0) {
            for (int64_t r = 0; r < rounds && ok; ++r) {
                const int slot = (int)(r % NS);
                const uint32_t fb = (uint32_t)__cvta_generic_to_shared(&full[slot]);
                const uint32_t eb = (uint32_t)__cvta_generic_to_shared(&empty[slot]);
                if (r >= NS) ok = mbar_wait(eb, (uint32_t)(((r / NS) - 1) & 1));
                if (!ok) break;
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb),
                             "r"((uint32_t)SLOT) : "memory");
                asm volatile(
                    "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], "
                    "[%1], %2, [%3];" ::"r"(ring_s + (uint32_t)(slot * SLOT)),
                    "l"(src + r * SLOT), "r"((uint32_t)SLOT), "r"(fb)
                    : "memory");
            }
            // no copy may land after the CTA exits: the last round of each slot
            for (int64_t r = rounds > NS ? rounds - NS : 0; r < rounds; ++r)
                mbar_wait((uint32_t)__cvta_generic_to_shared(&full[r % NS]),
                          (uint32_t)((r / NS) & 1));
        }
    } else {
        float D[4][4] = {};
        const uint32_t b0 = 0x3c003c00u, b1 = 0x3c003c00u ^ (uint32_t)lane;
        for (int64_t r0 = 0; r0 < rounds && ok; r0 += 8) {
            const int n = rounds - r0 < 8 ? (int)(rounds - r0) : 8;
            for (int i = 0; i < n && ok; ++i)
                ok = mbar_wait((uint32_t)__cvta_generic_to_shared(&full[(r0 + i) % NS]),
                               (uint32_t)(((r0 + i) / NS) & 1));
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                if (i < n) {
                    uint32_t wd[6];
                    load_words(sm + ((r0 + i) % NS) * SLOT + warp * kRB, lane, wd);
                    record(wd, D, b0, b1);
                }
            }
            __syncwarp();
            if (lane == 0)
                for (int i = 0; i < n; ++i)
                    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(
                        (uint32_t)__cvta_generic_to_shared(&empty[(r0 + i) % NS])) : "memory");
        }
        float s = 0.f;
        for (int c = 0; c < 4; ++c) s += D[c][0] + D[c][1] + D[c][2] + D[c][3];
        if (s == 12345.f) sink[0] = s;
    }
    if (!ok) atomicExch(status, 1);
}

}  // namespace

int main() {
    int dev = 0, P = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&P, cudaDevAttrMultiProcessorCount, dev);
    const int64_t per_sm = 34048;  // records per SM (a multiple of 16 * 8); 4.2 GB in all
    const size_t bytes = (size_t)P * per_sm * kRB;
    uint8_t* buf = nullptr;
    float* sink = nullptr;
    int* status = nullptr;
    if (cudaMalloc(&buf, bytes) || cudaMalloc(&sink, 64) || cudaMalloc(&status, 4)) {
        printf("allocation failed\n");
        return 1;
    }
    cudaMemset(buf, 0x5a, bytes);
    cudaMemset(status, 0, 4);
    cudaEvent_t e0, e1;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    auto time = [&](auto launch, const char* name) {
        launch();  // warm-up
        cudaEventRecord(e0);
        for (int i = 0; i < 3; ++i) launch();
        cudaEventRecord(e1);
        if (cudaEventSynchronize(e1) != cudaSuccess) { printf("error in %s\n", name); return; }
        float ms = 0.f;
        cudaEventElapsedTime(&ms, e0, e1);
        int st = 0;
        cudaMemcpy(&st, status, 4, cudaMemcpyDeviceToHost);
        printf("%-58s %6.2f TB/s%s\n", name, 3.0 * bytes / (ms * 1e-3) / 1e12,
               st ? "  [a wait gave up]" : "");
    };
    printf("%d SMs, %.2f GB streamed per run\n", P, bytes / 1e9);
    const int smA = kWarps * 8 * kCodes;
    cudaFuncSetAttribute(per_warp<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, smA);
    time([&] { per_warp<8><<<P, kWarps * 32, smA>>>(buf, per_sm, sink); },
         "A. per-warp cp.async rings, 8 records per warp");
    const int smB16 = 16 * kWarps * kRB, smB8 = 8 * kWarps * kRB;
    cudaFuncSetAttribute(bulk_ring<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, smB16);
    cudaFuncSetAttribute(bulk_ring<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, smB8);
    time([&] { bulk_ring<16><<<P, (kWarps + 1) * 32, smB16>>>(buf, per_sm, sink, status); },
         "B. cp.async.bulk rounds of 16 records, 16-slot ring");
    time([&] { bulk_ring<8><<<P, (kWarps + 1) * 32, smB8>>>(buf, per_sm, sink, status); },
         "B. cp.async.bulk rounds of 16 records, 8-slot ring");
    return 0;
}
