// laq_rotate.cu -- the online pairwise rotation that rotation-based weight quantizers run on the
// input of every projection at every forward pass (the step LAQuant removes; Sec. 1, Sec. 2 and
// the decode-speed comparison of Sec. 5.2), built here to measure its per-token cost beside the
// GEMV.  Per 128-channel group: v = x * alpha, then `rounds` rounds of Givens rotations, round r
// turning each of its 64 disjoint channel pairs (i, j) by its angle t:
// (v_i, v_j) -> (v_i cos t - v_j sin t, v_i sin t + v_j cos t); fp16 out, rounded once.
//
// One warp per (row, group).  The group's tables (the pairs and the (cos, sin) of every round,
// 640 bytes a round) are constant parameters, so the warp copies them to shared memory with
// cp.async before griddepcontrol.wait, under the tail of the kernel before it.  After the wait
// it loads its 128 inputs (four per lane), scales them into a shared fp32 vector, runs the
// rounds (two pairs per lane; a round's pairs are disjoint, so no two lanes touch one channel,
// and __syncwarp orders the rounds) and stores fp16 once.  Pair indices are masked to 0..127,
// so tables that are not matchings give wrong values but never an access outside the group.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "laq.h"
#include "laq_device.cuh"

namespace laq {
namespace {

constexpr int kRotMaxRounds = 16;
constexpr int kRotWarps = 4;  // groups per CTA

struct RotSmem {
    float x[128];
    uint16_t ij[kRotMaxRounds][64];    // pair p of round r: i | j << 8
    float2 cs[kRotMaxRounds][64];      // (cos t, sin t)
};

__global__ void __launch_bounds__(kRotWarps * 32)
rotate_kernel(const __half* X /* may equal Y */, int64_t K, int G,
              const __half* __restrict__ alpha,
              const uint16_t* __restrict__ pairs, const float2* __restrict__ cs, int rounds,
              __half* Y) {
    pdl_launch_dependents();
    __shared__ __align__(16) RotSmem sm[kRotWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = blockIdx.x * kRotWarps + warp;
    if (g >= G) return;  // no block-wide barrier follows
    RotSmem& s = sm[warp];
    const int64_t m = blockIdx.y;

    // the group's tables: rounds * 128 bytes of pairs, rounds * 512 bytes of (cos, sin)
    {
        const char* src_ij = reinterpret_cast<const char*>(pairs + (size_t)g * rounds * 64);
        const char* src_cs = reinterpret_cast<const char*>(cs + (size_t)g * rounds * 64);
        const uint32_t dst_ij = (uint32_t)__cvta_generic_to_shared(&s.ij[0][0]);
        const uint32_t dst_cs = (uint32_t)__cvta_generic_to_shared(&s.cs[0][0]);
        for (int c = lane; c < rounds * 8; c += 32) cp_async16(dst_ij + 16 * c, src_ij + 16 * c);
        for (int c = lane; c < rounds * 32; c += 32) cp_async16(dst_cs + 16 * c, src_cs + 16 * c);
        cp_async_commit();
    }
    float a[4] = {1.f, 1.f, 1.f, 1.f};
    if (alpha) {
        const uint2 av = *reinterpret_cast<const uint2*>(alpha + (size_t)g * 128 + 4 * lane);
        const float2 a01 = __half22float2(*reinterpret_cast<const __half2*>(&av.x));
        const float2 a23 = __half22float2(*reinterpret_cast<const __half2*>(&av.y));
        a[0] = a01.x, a[1] = a01.y, a[2] = a23.x, a[3] = a23.y;
    }

    pdl_wait();  // X belongs to the kernel before this one until it completes
    const size_t off = (size_t)m * K + (size_t)g * 128 + 4 * lane;
    const uint2 xv = __ldcg(reinterpret_cast<const uint2*>(X + off));  // through L2: fresh
    const float2 x01 = __half22float2(*reinterpret_cast<const __half2*>(&xv.x));
    const float2 x23 = __half22float2(*reinterpret_cast<const __half2*>(&xv.y));
    s.x[4 * lane + 0] = x01.x * a[0];
    s.x[4 * lane + 1] = x01.y * a[1];
    s.x[4 * lane + 2] = x23.x * a[2];
    s.x[4 * lane + 3] = x23.y * a[3];
    cp_async_wait(0);
    __syncwarp();

    for (int r = 0; r < rounds; ++r) {
        const uint32_t p0 = s.ij[r][lane], p1 = s.ij[r][lane + 32];
        const float2 t0 = s.cs[r][lane], t1 = s.cs[r][lane + 32];
        const int i0 = p0 & 127, j0 = (p0 >> 8) & 127, i1 = p1 & 127, j1 = (p1 >> 8) & 127;
        const float u0 = s.x[i0], v0 = s.x[j0], u1 = s.x[i1], v1 = s.x[j1];
        s.x[i0] = u0 * t0.x - v0 * t0.y;
        s.x[j0] = u0 * t0.y + v0 * t0.x;
        s.x[i1] = u1 * t1.x - v1 * t1.y;
        s.x[j1] = u1 * t1.y + v1 * t1.x;
        __syncwarp();
    }

    const __half2 y01 = __floats2half2_rn(s.x[4 * lane + 0], s.x[4 * lane + 1]);
    const __half2 y23 = __floats2half2_rn(s.x[4 * lane + 2], s.x[4 * lane + 3]);
    uint2 yv;
    yv.x = *reinterpret_cast<const uint32_t*>(&y01);
    yv.y = *reinterpret_cast<const uint32_t*>(&y23);
    *reinterpret_cast<uint2*>(Y + off) = yv;
}

__global__ void __launch_bounds__(256) rotation_tables_kernel(const float* __restrict__ theta,
                                                              int64_t n, float2* cs) {
    const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= n) return;
    float sn, c;
    sincosf(theta[k], &sn, &c);
    cs[k] = make_float2(c, sn);
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace
}  // namespace laq

using namespace laq;

extern "C" {

laq_status laq_rotation_tables(const float* theta, int64_t n, void* cs, void* stream) {
    if (n == 0) return LAQ_OK;
    if (!theta || !cs) return LAQ_ERR_NULL;
    if (n < 0 || n > ((int64_t)1 << 31)) return LAQ_ERR_SHAPE;  // grid.x limit x 256 threads
    if (((uintptr_t)theta & 3u) || ((uintptr_t)cs & 7u)) return LAQ_ERR_ALIGN;
    rotation_tables_kernel<<<(unsigned)((n + 255) / 256), 256, 0,
                             static_cast<cudaStream_t>(stream)>>>(theta, n,
                                                                  static_cast<float2*>(cs));
    return cudaGetLastError() == cudaSuccess ? LAQ_OK : LAQ_ERR_CUDA;
}

laq_status laq_pairwise_rotate(const void* X, int64_t M, int64_t K, const void* alpha,
                               const uint8_t* pairs, const void* cs, int32_t rounds, void* Y,
                               void* stream) {
    if (M == 0) return LAQ_OK;
    if (!X || !Y || (rounds > 0 && (!pairs || !cs))) return LAQ_ERR_NULL;
    if (M < 0 || M > 65535 || K < 128 || K % 128 || K > ((int64_t)1 << 31) || rounds < 0 ||
        rounds > kRotMaxRounds)
        return LAQ_ERR_SHAPE;
    if (!aligned16(X) || !aligned16(Y) || !aligned16(pairs) || !aligned16(cs) ||
        (alpha && !aligned16(alpha)))
        return LAQ_ERR_ALIGN;
    const int G = (int)(K / 128);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((G + kRotWarps - 1) / kRotWarps), (unsigned)M, 1);
    cfg.blockDim = dim3(kRotWarps * 32, 1, 1);
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(
        &cfg, rotate_kernel, static_cast<const __half*>(X), K, G,
        static_cast<const __half*>(alpha), reinterpret_cast<const uint16_t*>(pairs),
        static_cast<const float2*>(cs), (int)rounds, static_cast<__half*>(Y));
    return e == cudaSuccess ? LAQ_OK : LAQ_ERR_CUDA;
}

}  // extern "C"
