// laq_quant.cu -- offline model-preparation kernels: the RTN group quantizer of Eq. (1) and the
// packer / unpacker of the library's record layout (both run once per weight, not per token).
//
// The quantizer works in fp64 so that it makes exactly the decisions the rule in laq.h
// describes: every quotient of two fp16 values is correctly rounded in fp64, and a quotient
// that is not exactly a tie (or exactly an fp16 value) is never rounded onto one, so rint() and
// the fp16 round-up see the same side as with exact arithmetic.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "laq_internal.cuh"

namespace laq {

namespace {

constexpr int kGroup = 128;

__device__ __forceinline__ double half_value(uint16_t h) {
    return (double)__half2float(__ushort_as_half(h));  // fp16 -> fp32 -> fp64 is exact
}

// Smallest fp16 >= v for 0 < v <= 65504: the nearest fp16, moved by one ulp if it lies on the
// wrong side (positive fp16 bit patterns are ordered like their values).
__device__ uint16_t half_round_up(double v) {
    uint16_t h = __half_as_ushort(__double2half(v));
    if (half_value(h) < v) {
        h = (uint16_t)(h + 1);
    } else if (h > 0 && half_value((uint16_t)(h - 1)) >= v) {
        h = (uint16_t)(h - 1);
    }
    return h;
}

// One thread per (group g, column n).  Reads of W are coalesced across n.
template <int BITS>
__global__ void quantize_rtn_kernel(const uint16_t* __restrict__ W, int64_t N,
                                    uint8_t* __restrict__ codes, uint16_t* __restrict__ s,
                                    uint8_t* __restrict__ z) {
    const int64_t n = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t g = blockIdx.y;
    if (n >= N) return;
    constexpr int qmax = (1 << BITS) - 1;
    const uint16_t* col = W + g * kGroup * N + n;
    double lo = half_value(col[0]), hi = lo;
    for (int k = 1; k < kGroup; ++k) {
        const double w = half_value(col[(int64_t)k * N]);
        lo = w < lo ? w : lo;
        hi = w > hi ? w : hi;
    }
    uint16_t sh;
    int zz;
    if (lo == hi) {
        // constant group c: s = |c| (1 when c == 0), z = 1 for c < 0, so w_hat == c exactly
        if (lo != 0.0) {
            sh = (uint16_t)(col[0] & 0x7fffu);
            zz = lo < 0.0 ? 1 : 0;
        } else {
            sh = 0x3c00u;
            zz = 0;
        }
    } else {
        const double lo0 = lo < 0.0 ? lo : 0.0;  // range widened to contain 0
        const double hi0 = hi > 0.0 ? hi : 0.0;
        sh = half_round_up((hi0 - lo0) / (double)qmax);
        if (sh < 0x0400u) sh = 0x0400u;           // smallest normal fp16
        zz = (int)rint(-lo0 / half_value(sh));
    }
    const double sv = half_value(sh);
    s[g * N + n] = sh;
    z[g * N + n] = (uint8_t)zz;
    uint8_t* out = codes + g * kGroup * N + n;
    for (int k = 0; k < kGroup; ++k) {
        int q = (int)rint(half_value(col[(int64_t)k * N]) / sv) + zz;  // round, then add z
        q = q < 0 ? 0 : (q > qmax ? qmax : q);
        out[(int64_t)k * N] = (uint8_t)q;
    }
}

// ---- record layout (see laq.h): lane l = 4r + c owns columns r, r+8 and rows 32c+4j+2h+e ----

// Code at (row-in-record kk, column-in-tile nn) of record (t, g).
__device__ __forceinline__ uint32_t code_at(const uint8_t* __restrict__ codes, int64_t N,
                                            int64_t t, int64_t g, int kk, int nn) {
    return codes[(g * kGroup + kk) * N + t * 16 + nn];
}

template <int BITS>
__global__ void pack_kernel(const uint8_t* __restrict__ codes, int64_t N, int64_t G,
                            int64_t records, uint32_t* __restrict__ packed) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= records * 32) return;
    const int64_t rec = idx >> 5;
    const int lane = (int)(idx & 31);
    const int64_t t = rec / G, g = rec % G;
    const int c = lane & 3, r = lane >> 2;
    if (BITS == 4) {
        uint32_t* out = packed + rec * 256;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            uint32_t word = 0;
#pragma unroll
            for (int e = 0; e < 2; ++e)
#pragma unroll
                for (int f = 0; f < 4; ++f) {
                    const int h = f & 1, row = f >> 1;
                    const uint32_t q =
                        code_at(codes, N, t, g, 32 * c + 4 * j + 2 * h + e, r + 8 * row) & 15u;
                    word |= q << (16 * e + 4 * f);
                }
            out[(j >> 2) * 128 + 4 * lane + (j & 3)] = word;
        }
    } else {
        uint32_t* out = packed + rec * 192;
        // pair i = 2j + h of row (r or r+8) -> the 3-bit code at element e
        auto pair_code = [&](int i, int row, int e) -> uint32_t {
            return code_at(codes, N, t, g, 32 * c + 4 * (i >> 1) + 2 * (i & 1) + e,
                           r + 8 * row) & 7u;
        };
#pragma unroll
        for (int w = 0; w < 6; ++w) {
            uint32_t word = 0;
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                uint32_t half = (pair_code(15, w >= 3 ? 1 : 0, e) >> (w % 3)) & 1u;  // bit 0
                half |= pair_code(w, 0, e) << 1                          // bits 1-3
                      | pair_code(6 + w, 0, e) << 4                      // bits 4-6
                      | pair_code(12 + (w >> 1), w & 1, e) << 7          // bits 7-9
                      | pair_code(w, 1, e) << 10                         // bits 10-12
                      | pair_code(6 + w, 1, e) << 13;                    // bits 13-15
                word |= half << (16 * e);
            }
            out[w < 4 ? 4 * lane + w : 128 + 2 * lane + (w - 4)] = word;
        }
    }
}

template <int BITS>
__global__ void unpack_kernel(const uint32_t* __restrict__ packed, int64_t N, int64_t G,
                              int64_t records, uint8_t* __restrict__ codes) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= records * 32) return;
    const int64_t rec = idx >> 5;
    const int lane = (int)(idx & 31);
    const int64_t t = rec / G, g = rec % G;
    const int c = lane & 3, r = lane >> 2;
    auto put = [&](int kk, int nn, uint32_t q) {
        codes[(g * kGroup + kk) * N + t * 16 + nn] = (uint8_t)q;
    };
    if (BITS == 4) {
        const uint32_t* in = packed + rec * 256;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const uint32_t word = in[(j >> 2) * 128 + 4 * lane + (j & 3)];
#pragma unroll
            for (int e = 0; e < 2; ++e)
#pragma unroll
                for (int f = 0; f < 4; ++f)
                    put(32 * c + 4 * j + 2 * (f & 1) + e, r + 8 * (f >> 1),
                        (word >> (16 * e + 4 * f)) & 15u);
        }
    } else {
        const uint32_t* in = packed + rec * 192;
        uint32_t words[6];
#pragma unroll
        for (int w = 0; w < 6; ++w) words[w] = in[w < 4 ? 4 * lane + w : 128 + 2 * lane + (w - 4)];
        auto put_pair = [&](int i, int row, int e, uint32_t q) {
            put(32 * c + 4 * (i >> 1) + 2 * (i & 1) + e, r + 8 * row, q);
        };
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            uint32_t spare[2] = {0, 0};
#pragma unroll
            for (int w = 0; w < 6; ++w) {
                const uint32_t half = (words[w] >> (16 * e)) & 0xffffu;
                spare[w >= 3 ? 1 : 0] |= (half & 1u) << (w % 3);
                put_pair(w, 0, e, (half >> 1) & 7u);
                put_pair(6 + w, 0, e, (half >> 4) & 7u);
                put_pair(12 + (w >> 1), w & 1, e, (half >> 7) & 7u);
                put_pair(w, 1, e, (half >> 10) & 7u);
                put_pair(6 + w, 1, e, (half >> 13) & 7u);
            }
            put_pair(15, 0, e, spare[0]);
            put_pair(15, 1, e, spare[1]);
        }
    }
}

}  // namespace

cudaError_t launch_quantize_rtn(const uint16_t* W, int64_t K, int64_t N, int bits,
                                uint8_t* codes, uint16_t* s, uint8_t* z, cudaStream_t stream) {
    const int64_t G = K / kGroup;
    const dim3 block(128);
    const dim3 grid((unsigned)((N + 127) / 128), (unsigned)G);
    if (bits == 3)
        quantize_rtn_kernel<3><<<grid, block, 0, stream>>>(W, N, codes, s, z);
    else
        quantize_rtn_kernel<4><<<grid, block, 0, stream>>>(W, N, codes, s, z);
    return cudaGetLastError();
}

cudaError_t launch_pack(const uint8_t* codes, int64_t K, int64_t N, int bits, uint32_t* packed,
                        cudaStream_t stream) {
    const int64_t G = K / kGroup, records = G * (N / 16);
    const int64_t threads = records * 32;
    const dim3 block(256), grid((unsigned)((threads + 255) / 256));
    if (bits == 3)
        pack_kernel<3><<<grid, block, 0, stream>>>(codes, N, G, records, packed);
    else
        pack_kernel<4><<<grid, block, 0, stream>>>(codes, N, G, records, packed);
    return cudaGetLastError();
}

cudaError_t launch_unpack(const uint32_t* packed, int64_t K, int64_t N, int bits, uint8_t* codes,
                          cudaStream_t stream) {
    const int64_t G = K / kGroup, records = G * (N / 16);
    const int64_t threads = records * 32;
    const dim3 block(256), grid((unsigned)((threads + 255) / 256));
    if (bits == 3)
        unpack_kernel<3><<<grid, block, 0, stream>>>(packed, N, G, records, codes);
    else
        unpack_kernel<4><<<grid, block, 0, stream>>>(packed, N, G, records, codes);
    return cudaGetLastError();
}

}  // namespace laq
