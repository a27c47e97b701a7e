// laq_device.cuh -- device helpers shared by the GEMV kernels (not installed): record format,
// cp.async and griddepcontrol wrappers, the m16n8k16 MMA, and the A-fragment extraction that
// turns packed codes into fp16 values 2^(10-p) + q (see laq_gemm.cu for the scheme).
#pragma once
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace laq {
namespace {

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


__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async8(uint32_t dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;\n" ::: "memory");
}
// Wait until at most n of this thread's committed cp.async groups are pending (n = 0..15).
__device__ __forceinline__ void cp_async_wait(int n) {
    switch (n) {
        case 0: asm volatile("cp.async.wait_group 0;\n" ::: "memory"); break;
        case 1: asm volatile("cp.async.wait_group 1;\n" ::: "memory"); break;
        case 2: asm volatile("cp.async.wait_group 2;\n" ::: "memory"); break;
        case 3: asm volatile("cp.async.wait_group 3;\n" ::: "memory"); break;
        case 4: asm volatile("cp.async.wait_group 4;\n" ::: "memory"); break;
        case 5: asm volatile("cp.async.wait_group 5;\n" ::: "memory"); break;
        case 6: asm volatile("cp.async.wait_group 6;\n" ::: "memory"); break;
        case 7: asm volatile("cp.async.wait_group 7;\n" ::: "memory"); break;
        case 8: asm volatile("cp.async.wait_group 8;\n" ::: "memory"); break;
        case 9: asm volatile("cp.async.wait_group 9;\n" ::: "memory"); break;
        case 10: asm volatile("cp.async.wait_group 10;\n" ::: "memory"); break;
        case 11: asm volatile("cp.async.wait_group 11;\n" ::: "memory"); break;
        case 12: asm volatile("cp.async.wait_group 12;\n" ::: "memory"); break;
        case 13: asm volatile("cp.async.wait_group 13;\n" ::: "memory"); break;
        case 14: asm volatile("cp.async.wait_group 14;\n" ::: "memory"); break;
        default: asm volatile("cp.async.wait_group 15;\n" ::: "memory"); break;
    }
}

// 16-byte load through L2 only (the data may have been written by other SMs).
__device__ __forceinline__ uint4 ld_cg16(const void* p) {
    uint4 v;
    asm volatile("ld.global.cg.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p)
                 : "memory");
    return v;
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

// Exponent fields that turn a code at mantissa bit p into the exact fp16 value 2^(10-p) + q:
// exponent 25 - p, in both halves of a 32-bit register.
constexpr uint32_t kExpP0 = 0x64006400u;  // p = 0: 1024 + q
constexpr uint32_t kExpP1 = 0x60006000u;  // p = 1:  512 + q
constexpr uint32_t kExpP4 = 0x54005400u;  // p = 4:   64 + q
constexpr uint32_t kExpP7 = 0x48004800u;  // p = 7:    8 + q

// The exponent fields a kernel instance ORs into its A fragments: b = 3 uses p = 1, 4, 7;
// b = 4 uses p = 0, 4.  They arrive as kernel parameters so that they stay in registers and
// each extraction is a single mask-and-or.
struct Exps {
    uint32_t e[3];
};
inline Exps exps_for(int bits) {
    Exps x;
    if (bits == 4) {
        x.e[0] = kExpP0; x.e[1] = kExpP4; x.e[2] = 0u;
    } else {
        x.e[0] = kExpP1; x.e[1] = kExpP4; x.e[2] = kExpP7;
    }
    return x;
}

// Extract the A fragments of one record (one lane's words) into a[j][0..3] for the 8 k16 steps:
// a0 = (row r, pair (j,0)), a1 = (row r+8, pair (j,0)), a2 = (row r, pair (j,1)),
// a3 = (row r+8, pair (j,1)); each register holds 2^(10-p) + q for its two codes.  Shifts are
// plain shifts: on GB300 a shift issues at the mask-and-or rate (two warp instructions per SM
// cycle), a multiply-high only at one, and the legacy MMA leaves half of the integer work's
// issue slots unhidden, so the record loop from shared memory costs 42.2 SM cycles per W3
// record with shifts against 45.8 with multiply-high shifts.
template <int BITS>
__device__ __forceinline__ void extract(const uint32_t (&wd)[BITS == 4 ? 8 : 6],
                                        const Exps& x, uint32_t (&a)[8][4]) {
    if constexpr (BITS == 4) {
        const uint32_t e0 = x.e[0], e4 = x.e[1];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const uint32_t w = wd[j], t = w >> 8;
            a[j][0] = (w & 0x000f000fu) | e0;  // pair (j, 0, r)      p = 0
            a[j][2] = (w & 0x00f000f0u) | e4;  // pair (j, 1, r)      p = 4
            a[j][1] = (t & 0x000f000fu) | e0;  // pair (j, 0, r + 8)  p = 0
            a[j][3] = (t & 0x00f000f0u) | e4;  // pair (j, 1, r + 8)  p = 4
        }
    } else {
        const uint32_t e1 = x.e[0], e4 = x.e[1], e7 = x.e[2];
        uint32_t rp[16][2];
#pragma unroll
        for (int w = 0; w < 6; ++w) {
            const uint32_t u = wd[w] >> 9;
            rp[w][0] = (wd[w] & 0x000e000eu) | e1;              // bits 1-3    p = 1
            rp[6 + w][0] = (wd[w] & 0x00700070u) | e4;          // bits 4-6    p = 4
            rp[w][1] = (u & 0x000e000eu) | e1;                  // bits 10-12  p = 1
            rp[6 + w][1] = (u & 0x00700070u) | e4;              // bits 13-15  p = 4
        }
#pragma unroll
        for (int q = 0; q < 3; ++q) {
            rp[12 + q][0] = (wd[2 * q] & 0x03800380u) | e7;      // bits 7-9   p = 7
            rp[12 + q][1] = (wd[2 * q + 1] & 0x03800380u) | e7;
        }
        // pair 15: bit 0 of words 0,1,2 (row r) / 3,4,5 (row r+8) -> code bits 0,1,2 at p = 4
        rp[15][0] = ((wd[0] << 4) & 0x00100010u) | ((wd[1] << 5) & 0x00200020u) |
                    ((wd[2] << 6) & 0x00400040u) | e4;
        rp[15][1] = ((wd[3] << 4) & 0x00100010u) | ((wd[4] << 5) & 0x00200020u) |
                    ((wd[5] << 6) & 0x00400040u) | e4;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            a[j][0] = rp[2 * j][0];
            a[j][1] = rp[2 * j][1];
            a[j][2] = rp[2 * j + 1][0];
            a[j][3] = rp[2 * j + 1][1];
        }
    }
}

// Offset c_k = 2^(10-p) of row k of a group (k = 32c + 4j + 2h + e, pair index i = (k % 32) / 2).
template <int BITS>
__device__ __forceinline__ float row_offset(int i) {
    if (BITS == 4) return (i & 1) ? 64.f : 1024.f;
    return i < 6 ? 512.f : (i < 12 ? 64.f : (i < 15 ? 8.f : 64.f));
}

}  // namespace
}  // namespace laq
