// sync_latency.cu -- what a GPU-wide stage hand-over costs on this device.
//
// A decode-step weight pass is a chain of dependent stages (q|k|v -> o -> gate|up -> down per
// layer); a persistent kernel hands each stage over to the next through global memory.  This
// program measures the pieces of such a hand-over, one CTA per SM:
//   1. the cost of a gpu-scope acquire-release fence, a release store and L2 loads, measured by
//      one thread while (optionally) its SM has bulk copies from HBM in flight;
//   2. the cost of one poll of 152 per-CTA flags in the forms a poller can use;
//   3. four stage-barrier protocols with every CTA arriving at about the same time (as at the
//      end of a balanced stage): the delay from the last arrival until each CTA sees it.
// Every wait is bounded; the barrier runs as a cooperative launch (all CTAs resident).
//
//   nvcc -gencode arch=compute_103a,code=sm_103a -O3 -o /tmp/sync_latency \
//       paper_2605_08755_gb300/measure/sync_latency.cu && /tmp/sync_latency
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>

#include <algorithm>
#include <vector>

namespace {

__device__ __forceinline__ unsigned long long clk() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%clock64;" : "=l"(t));
    return t;
}
__device__ __forceinline__ unsigned long long gt() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ uint32_t ld_acq(const void* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t ld_rlx(const void* p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint4 ld_acq4(const void* p) {
    uint4 v;
    asm volatile("ld.acquire.gpu.global.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint4 ld_rlx4(const void* p) {
    uint4 v;
    asm volatile("ld.relaxed.gpu.global.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void fence_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile("{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
                 "selp.u32 %0, 1, 0, p;\n}\n"
                 : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
    return ok != 0u;
}

constexpr int kCopy = 16384;  // bytes per bulk copy
constexpr int kSlots = 8;

// Part 1.  Warp 1 keeps kSlots bulk copies of kCopy bytes in flight from a large buffer (when
// `stream`), warp 0's lane 0 times the operations (cycles, averaged over iterations).
__global__ void __launch_bounds__(64, 1) op_costs(uint32_t* flags, const uint8_t* big,
                                                  size_t big_bytes, int stream, int iters,
                                                  unsigned long long* out) {
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ __align__(8) uint64_t bar[kSlots];
    __shared__ volatile int stop;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kSlots; ++i)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(
                (uint32_t)__cvta_generic_to_shared(&bar[i])));
        stop = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    if (warp == 1) {
        if (stream && lane == 0) {
            uint32_t phase[kSlots] = {};
            size_t off = (size_t)blockIdx.x * kCopy * 64;
            int k = 0;
            for (; k < 1000000 && !stop; ++k) {
                const int s = k % kSlots;
                const uint32_t b = (uint32_t)__cvta_generic_to_shared(&bar[s]);
                if (k >= kSlots) {  // the copy that used this slot has landed
                    bool ok = false;
                    for (int sp = 0; sp < (1 << 22) && !ok; ++sp) ok = mbar_try(b, phase[s]);
                    phase[s] ^= 1u;
                }
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(b),
                             "r"((uint32_t)kCopy) : "memory");
                asm volatile(
                    "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], "
                    "%2, [%3];" ::"r"((uint32_t)__cvta_generic_to_shared(sm + s * kCopy)),
                    "l"(big + off % (big_bytes - kCopy)), "r"((uint32_t)kCopy), "r"(b)
                    : "memory");
                off += (size_t)kCopy * gridDim.x;
            }
            for (int s = 0; s < kSlots && s < k; ++s) {  // drain: the last copy of each slot
                const int last = k - 1 - ((k - 1 - s) % kSlots);
                const uint32_t b = (uint32_t)__cvta_generic_to_shared(&bar[last % kSlots]);
                bool ok = false;
                for (int sp = 0; sp < (1 << 22) && !ok; ++sp) ok = mbar_try(b, phase[last % kSlots]);
            }
        }
        return;
    }
    if (lane != 0) return;
    const unsigned long long t0 = gt();
    while (gt() - t0 < 20000) {}  // let the copies get going
    uint32_t* mine = flags + blockIdx.x * 32;
    const uint32_t* other = flags + ((blockIdx.x + gridDim.x / 2) % gridDim.x) * 32;
    unsigned long long t_fence = 0, t_rel = 0, t_ld = 0;
    uint32_t acc = 0;
    for (int i = 0; i < iters; ++i) {
        unsigned long long a = clk();
        fence_gpu();
        t_fence += clk() - a;
        a = clk();
        asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(mine), "r"((uint32_t)i) : "memory");
        t_rel += clk() - a;
        a = clk();
        acc += ld_acq(other + (i & 3));
        if (acc == 0xdeadbeefu) out[0] = 1;  // keep the load
        t_ld += clk() - a;
    }
    stop = 1;
    unsigned long long* o = out + blockIdx.x * 4;
    o[0] = t_fence / iters;
    o[1] = t_rel / iters;
    o[2] = t_ld / iters;
}

// Part 2.  One warp per SM polls 152 flags (4 bytes each, or 2 bytes for the vector forms):
// mode 0: 5 acquire loads per lane; 1: 5 relaxed loads per lane; 2: one 16-byte acquire load per
// lane (16-bit flags); 3: one 16-byte relaxed load per lane + an acquire fence.  Cycles per poll.
__global__ void __launch_bounds__(32, 1) poll_costs(const uint32_t* f, int mode, int iters,
                                                    unsigned long long* out) {
    const int lane = threadIdx.x;
    const unsigned long long t0 = gt();
    while (gt() - t0 < 5000) {}
    unsigned long long tot = 0;
    uint32_t acc = 0;
    for (int it = 0; it < iters; ++it) {
        const unsigned long long a = clk();
        uint32_t s = 0;
        if (mode <= 1) {
            uint32_t v[5];
#pragma unroll
            for (int u = 0; u < 5; ++u) {
                const int j = lane + 32 * u;
                v[u] = j < 152 ? (mode == 0 ? ld_acq(f + j) : ld_rlx(f + j)) : 0u;
            }
#pragma unroll
            for (int u = 0; u < 5; ++u) s += v[u];
        } else {
            uint4 v = make_uint4(0u, 0u, 0u, 0u);
            if (lane < 19) v = mode == 2 ? ld_acq4(f + 4 * lane) : ld_rlx4(f + 4 * lane);
            if (mode == 3) fence_gpu();
            s = v.x + v.y + v.z + v.w;
        }
        acc += __reduce_add_sync(0xffffffffu, s);
        tot += clk() - a;
    }
    if (lane == 0) {
        out[blockIdx.x * 2] = tot / iters;
        out[blockIdx.x * 2 + 1] = acc;
    }
}

// Part 3.  Stage barriers: every CTA spins for ~2-3.3 us (a stage's work, with some spread),
// stores 64 bytes of "Y", arrives, and its warp 0 waits until all have arrived.
//   mode 0: a 16-bit flag per CTA packed into three lines, one 16-byte acquire poll per lane;
//   mode 1: a 32-bit flag per CTA in a 128-byte line of its own, relaxed polls + acquire fence;
//   mode 2: one counter per stage (red.release.gpu.add by each CTA), lane 0 polls it (acquire);
//   mode 3: 32-bit flags packed into five lines, relaxed polls + acquire fence.
__global__ void __launch_bounds__(256, 1) stage_barrier(uint8_t* ws, uint16_t* Y, int mode,
                                                        int stages, unsigned long long* t_arr,
                                                        unsigned long long* t_seen) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int P = gridDim.x;
    for (int s = 1; s <= stages; ++s) {
        const unsigned long long t0 = gt();
        const unsigned long long work = 2000 + ((blockIdx.x * 37 + s * 101) % 13) * 100;
        while (gt() - t0 < work) {}
        if (tid < 32) Y[(size_t)s * P * 32 + blockIdx.x * 32 + tid] = (uint16_t)s;
        __syncthreads();
        if (tid == 0) {
            t_arr[(size_t)s * P + blockIdx.x] = gt();
            if (mode == 0)
                asm volatile("st.release.gpu.global.u16 [%0], %1;" ::"l"(ws + 16 + 2 * blockIdx.x),
                             "h"((uint16_t)s) : "memory");
            else if (mode == 1)
                asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(ws + 128 * blockIdx.x),
                             "r"((uint32_t)s) : "memory");
            else if (mode == 2)
                asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ws + 128 * (s & 7))
                             : "memory");
            else
                asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(ws + 16 + 4 * blockIdx.x),
                             "r"((uint32_t)s) : "memory");
        }
        if (warp == 0) {
            bool done = false;
            const unsigned long long tw = gt();
            while (!done && gt() - tw < 1000000000ull) {
                bool ok = true;
                if (mode == 0) {
                    if (lane < 19) {
                        const uint4 v = ld_acq4(ws + 16 + 16 * lane);
                        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
                        for (int i = 0; i < 8; ++i)
                            ok &= ((w[i >> 1] >> (16 * (i & 1))) & 0xffffu) >= (uint32_t)s;
                    }
                } else if (mode == 1 || mode == 3) {
                    uint32_t v[5];
                    for (int u = 0; u < 5; ++u) {
                        const int j = lane + 32 * u;
                        v[u] = j < P ? ld_rlx(ws + (mode == 1 ? 128 * j : 16 + 4 * j)) : ~0u;
                    }
                    for (int u = 0; u < 5; ++u) ok &= v[u] >= (uint32_t)s;
                } else {
                    const uint32_t want = (uint32_t)P * (uint32_t)((s + 7) / 8);
                    ok = lane != 0 || ld_acq(ws + 128 * (s & 7)) >= want;
                }
                done = __all_sync(0xffffffffu, ok);
            }
            if (mode == 1 || mode == 3) fence_gpu();
            if (lane == 0) t_seen[(size_t)s * P + blockIdx.x] = gt();
        }
        __syncthreads();
    }
}

template <class T>
T median(std::vector<T> v) {
    std::sort(v.begin(), v.end());
    return v[v.size() / 2];
}

}  // namespace

int main() {
    int dev = 0, P = 0, mhz = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&P, cudaDevAttrMultiProcessorCount, dev);
    cudaDeviceGetAttribute(&mhz, cudaDevAttrClockRate, dev);
    printf("SMs %d, max SM clock %d MHz\n", P, mhz / 1000);
    uint32_t* flags = nullptr;
    uint8_t* big = nullptr;
    uint8_t* ws = nullptr;
    uint16_t* Y = nullptr;
    unsigned long long *out = nullptr, *ta = nullptr, *tn = nullptr;
    const size_t big_bytes = (size_t)4 << 30;
    const int S = 40;
    if (cudaMalloc(&flags, 65536) || cudaMalloc(&big, big_bytes) || cudaMalloc(&out, 65536) ||
        cudaMalloc(&ws, 65536) || cudaMalloc(&Y, (size_t)(S + 1) * P * 64) ||
        cudaMalloc(&ta, (size_t)(S + 1) * P * 8) || cudaMalloc(&tn, (size_t)(S + 1) * P * 8)) {
        printf("allocation failed\n");
        return 1;
    }
    cudaMemset(flags, 0, 65536);
    cudaMemset(big, 1, big_bytes);
    cudaFuncSetAttribute(op_costs, cudaFuncAttributeMaxDynamicSharedMemorySize, kSlots * kCopy);

    printf("\n1. one thread's operation costs, cycles (median / max over the %d SMs)\n", P);
    for (int stream = 0; stream < 2; ++stream) {
        cudaMemset(out, 0, 65536);
        op_costs<<<P, 64, kSlots * kCopy>>>(flags, big, big_bytes, stream, 200, out);
        if (cudaDeviceSynchronize() != cudaSuccess) { printf("error\n"); return 1; }
        std::vector<unsigned long long> h((size_t)P * 4);
        cudaMemcpy(h.data(), out, h.size() * 8, cudaMemcpyDeviceToHost);
        const char* names[3] = {"fence.acq_rel.gpu", "st.release.gpu", "ld.acquire.gpu (L2 hit)"};
        printf("   %s\n", stream ? "with 8 bulk copies of 16 KB in flight on every SM"
                                 : "no other traffic");
        for (int k = 0; k < 3; ++k) {
            std::vector<unsigned long long> v;
            for (int j = 0; j < P; ++j) v.push_back(h[(size_t)j * 4 + k]);
            printf("     %-26s %6llu %6llu\n", names[k], median(v), *std::max_element(v.begin(), v.end()));
        }
    }

    printf("\n2. one poll of %d flags by one warp, cycles (median over SMs)\n", P);
    const char* pnames[4] = {"5 x ld.acquire.u32 per lane", "5 x ld.relaxed.u32 per lane",
                             "1 x ld.acquire.v4 per lane", "1 x ld.relaxed.v4 + fence"};
    for (int mode = 0; mode < 4; ++mode) {
        poll_costs<<<P, 32>>>(flags, mode, 400, out);
        if (cudaDeviceSynchronize() != cudaSuccess) { printf("error\n"); return 1; }
        std::vector<unsigned long long> h((size_t)P * 2), v;
        cudaMemcpy(h.data(), out, h.size() * 8, cudaMemcpyDeviceToHost);
        for (int j = 0; j < P; ++j) v.push_back(h[(size_t)j * 2]);
        printf("     %-30s %6llu\n", pnames[mode], median(v));
    }

    printf("\n3. stage barrier, all %d CTAs arriving together: last arrival -> seen (ns)\n", P);
    const char* bnames[4] = {"16-bit flags packed in 3 lines", "32-bit flag per line",
                             "one counter per stage", "32-bit flags packed in 5 lines"};
    for (int mode = 0; mode < 4; ++mode) {
        cudaMemset(ws, 0, 65536);
        int m = mode, st = S;
        void* args[] = {&ws, &Y, &m, &st, &ta, &tn};
        if (cudaLaunchCooperativeKernel((void*)stage_barrier, P, 256, args, 0) != cudaSuccess ||
            cudaDeviceSynchronize() != cudaSuccess) {
            printf("error\n");
            return 1;
        }
        std::vector<unsigned long long> ha((size_t)(S + 1) * P), hn((size_t)(S + 1) * P);
        cudaMemcpy(ha.data(), ta, ha.size() * 8, cudaMemcpyDeviceToHost);
        cudaMemcpy(hn.data(), tn, hn.size() * 8, cudaMemcpyDeviceToHost);
        std::vector<long long> d;
        for (int s = 3; s <= S; ++s) {
            unsigned long long last = 0;
            for (int j = 0; j < P; ++j) last = std::max(last, ha[(size_t)s * P + j]);
            for (int j = 0; j < P; ++j) d.push_back((long long)hn[(size_t)s * P + j] - (long long)last);
        }
        std::sort(d.begin(), d.end());
        printf("     %-32s p10 %5lld  p50 %5lld  p90 %5lld  max %5lld\n", bnames[mode],
               d[d.size() / 10], d[d.size() / 2], d[d.size() * 9 / 10], d.back());
    }
    return 0;
}
