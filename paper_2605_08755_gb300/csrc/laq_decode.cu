// laq_decode.cu -- the decoder operations around the quantized projections of one decode step
// of a Qwen3-style model (the models whose decoding speed Sec. 5.2 reports): RMSNorm with the
// residual add, per-head q/k RMSNorm with rotary position embedding and the KV-cache append,
// grouped-query attention of the new token over its cache (flash-decoding: per-chunk partial
// softmax, then a combine in chunk order), SiLU(gate) * up, the embedding gather and the greedy
// argmax.  The paper defines none of them; they follow the standard decoder definitions, with
// fp32 arithmetic and one fp16 rounding per stored tensor.
//
// Every kernel lets its successor launch at once (griddepcontrol.launch_dependents) and waits
// for its predecessor (griddepcontrol.wait) before touching memory, so inside a CUDA graph of
// programmatically dependent launches each one's launch and set-up overlap the previous one.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "laq.h"
#include "laq_device.cuh"

namespace laq {
namespace {

constexpr int kHeadDim = 128;    // D: the only head size the attention kernels are built for
constexpr int kMaxGroup = 8;     // most q heads per kv head
constexpr int kChunk = 64;       // tokens per attention partial
constexpr int kPartial = kHeadDim + 2;  // floats per (row, q head, chunk): acc[D], max, sum

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ void unpack8(const uint4 u, float (&f)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 t = __half22float2(*reinterpret_cast<const __half2*>(&w[i]));
        f[2 * i] = t.x;
        f[2 * i + 1] = t.y;
    }
}

__device__ __forceinline__ uint4 pack8(const float (&f)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const __half2 h = __floats2half2_rn(f[2 * i], f[2 * i + 1]);
        w[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}


// RMSNorm over a head (lane l holds elements 4l .. 4l+3 of the warp's head), times the norm
// weights, then the rotate-half rotation at position p; every lane of the warp takes part.
// The rotation angles of lane l's elements 4l .. 4l+3 at position p: cos and sin of
// p * theta^(-2i/D), i = the element's index mod D/2 (the same for every head).
__device__ __forceinline__ void rope_angles(int lane, int64_t p, float log2_theta,
                                            float (&cs)[4], float (&sn)[4]) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const int i = (4 * lane + e) & (kHeadDim / 2 - 1);  // frequency index
        const float inv_freq = exp2f(-(2.f * (float)i / (float)kHeadDim) * log2_theta);
        sincosf((float)p * inv_freq, &sn[e], &cs[e]);
    }
}

__device__ __forceinline__ void norm_rope4(const float (&x)[4], const __half* __restrict__ wn,
                                           int lane, const float (&cs)[4], const float (&sn)[4],
                                           float eps, float (&o)[4]) {
    float ss = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) ss = fmaf(x[e], x[e], ss);
    ss = warp_sum(ss);
    const float inv = rsqrtf(ss / (float)kHeadDim + eps);
    float y[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) y[e] = x[e] * inv * __half2float(wn[4 * lane + e]);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float partner = __shfl_xor_sync(0xffffffffu, y[e], 16);
        o[e] = lane < 16 ? y[e] * cs[e] - partner * sn[e] : y[e] * cs[e] + partner * sn[e];
    }
}

__device__ __forceinline__ void load4(const __half* src, float (&x)[4]) {
    const uint2 raw = *reinterpret_cast<const uint2*>(src);
    const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&raw.x));
    const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&raw.y));
    x[0] = a.x; x[1] = a.y; x[2] = b.x; x[3] = b.y;
}

__device__ __forceinline__ uint2 round4(const float (&o)[4]) {
    const __half2 lo = __floats2half2_rn(o[0], o[1]), hi = __floats2half2_rn(o[2], o[3]);
    uint2 w;
    w.x = *reinterpret_cast<const uint32_t*>(&lo);
    w.y = *reinterpret_cast<const uint32_t*>(&hi);
    return w;
}

// ---- RMSNorm with the residual add ----
// Row m: h = X + R (rounded to fp16; h = X without R), R_out = h, Y = h / sqrt(mean(h^2) + eps)
// * w.  One CTA per row; each thread keeps up to kRmsChunks 8-element chunks in registers.
constexpr int kRmsThreads = 256;
constexpr int kRmsChunks = 4;  // H <= 8 * 256 * 4 = 8192

__global__ void __launch_bounds__(kRmsThreads) rmsnorm_kernel(const __half* __restrict__ X,
                                                              const __half* __restrict__ R,
                                                              __half* R_out,
                                                              const __half* __restrict__ w,
                                                              int H, float eps, __half* Y) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ float red[kRmsThreads / 32];
    const size_t row = (size_t)blockIdx.x * H;
    float h[kRmsChunks][8];
    float ss = 0.f;
#pragma unroll
    for (int c = 0; c < kRmsChunks; ++c) {
        const int i = (int)threadIdx.x + c * kRmsThreads;  // chunk index
        if (8 * i < H) {
            unpack8(*reinterpret_cast<const uint4*>(X + row + 8 * i), h[c]);
            if (R) {
                float r[8];
                unpack8(*reinterpret_cast<const uint4*>(R + row + 8 * i), r);
#pragma unroll
                for (int e = 0; e < 8; ++e) h[c][e] = __half2float(__float2half_rn(h[c][e] + r[e]));
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) ss = fmaf(h[c][e], h[c][e], ss);
        }
    }
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int k = 0; k < kRmsThreads / 32; ++k) tot += red[k];  // same order in every thread
    const float inv = rsqrtf(tot / (float)H + eps);
#pragma unroll
    for (int c = 0; c < kRmsChunks; ++c) {
        const int i = (int)threadIdx.x + c * kRmsThreads;
        if (8 * i < H) {
            if (R_out) *reinterpret_cast<uint4*>(R_out + row + 8 * i) = pack8(h[c]);
            float wv[8], y[8];
            unpack8(*reinterpret_cast<const uint4*>(w + 8 * i), wv);
#pragma unroll
            for (int e = 0; e < 8; ++e) y[e] = h[c][e] * inv * wv[e];
            *reinterpret_cast<uint4*>(Y + row + 8 * i) = pack8(y);
        }
    }
}

// ---- q/k RMSNorm + rotary embedding + KV-cache append ----
// One warp per head of qkv row m (q heads, then k heads, then v heads); lane l holds elements
// 4l .. 4l+3, so element d and its rotation partner d +- D/2 sit in lanes l and l ^ 16.
// Rotation (the rotate-half form): for i < D/2, angle a_i = pos * theta^(-2i/D),
//   out[i] = x[i] cos a_i - x[i + D/2] sin a_i,   out[i + D/2] = x[i + D/2] cos a_i + x[i] sin a_i.
__global__ void __launch_bounds__(128) qk_norm_rope_kernel(
    const __half* __restrict__ qkv, const __half* __restrict__ qw,
    const __half* __restrict__ kw, const int32_t* __restrict__ pos, int Hq, int Hkv,
    float log2_theta, float eps, __half* q_out, __half* k_cache, __half* v_cache,
    int64_t L_max) {
    pdl_launch_dependents();
    pdl_wait();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int head = blockIdx.x * 4 + warp, m = blockIdx.y;
    const int nh = Hq + 2 * Hkv;
    if (head >= nh) return;
    const int64_t p = pos[m];
    const bool in_cache = p >= 0 && p < L_max;  // a position outside the cache is not stored
    const __half* src = qkv + ((size_t)m * nh + head) * kHeadDim + 4 * lane;
    const uint2 raw = *reinterpret_cast<const uint2*>(src);
    if (head >= Hq + Hkv) {  // v: appended as is
        const int g = head - Hq - Hkv;
        if (in_cache)
            *reinterpret_cast<uint2*>(v_cache + (((size_t)m * Hkv + g) * L_max + p) * kHeadDim +
                                      4 * lane) = raw;
        return;
    }
    float x[4];
    {
        const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&raw.x));
        const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&raw.y));
        x[0] = a.x; x[1] = a.y; x[2] = b.x; x[3] = b.y;
    }
    float cs[4], sn[4], o[4];
    rope_angles(lane, p, log2_theta, cs, sn);
    norm_rope4(x, head < Hq ? qw : kw, lane, cs, sn, eps, o);
    const __half2 lo = __floats2half2_rn(o[0], o[1]), hi = __floats2half2_rn(o[2], o[3]);
    uint2 outw;
    outw.x = *reinterpret_cast<const uint32_t*>(&lo);
    outw.y = *reinterpret_cast<const uint32_t*>(&hi);
    if (head < Hq) {
        *reinterpret_cast<uint2*>(q_out + ((size_t)m * Hq + head) * kHeadDim + 4 * lane) = outw;
    } else if (in_cache) {
        const int g = head - Hq;
        *reinterpret_cast<uint2*>(k_cache + (((size_t)m * Hkv + g) * L_max + p) * kHeadDim +
                                  4 * lane) = outw;
    }
}

// The attention of one 64-token chunk whose K and V rows are staged in shared memory, for the
// G q heads of a kv head (qs: [G][D] fp32, already scaled), written to the partial slots
// part[j * nchunk * kPartial] (acc[D], max, sum) of head j.  Scores: a half-warp per token
// (lane l & 15 holds q and k elements 8 (l & 15) .. +7; q in registers); probabilities stored
// token-major (sc [kChunk][kMaxGroup]) so that one broadcast load gives every head's value of a
// token; weighted V sum: warp w takes tokens w, w + 4, ..., lane l dimensions 4l .. 4l+3, then
// the four warps' sums are added in warp order (red aliases the K rows, no longer needed).
// Every thread of the CTA must call it.
__device__ __forceinline__ void chunk_core(const __half (*ks)[kHeadDim],
                                           const __half (*vs)[kHeadDim], const float* qs,
                                           float* sc, float* mxs, float* sms, int nt, int G,
                                           float* part, int nchunk) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, hl = lane & 15;
    float qr[kMaxGroup][8];
#pragma unroll
    for (int j = 0; j < kMaxGroup; ++j)
#pragma unroll
        for (int e = 0; e < 8; ++e) qr[j][e] = j < G ? qs[j * kHeadDim + 8 * hl + e] : 0.f;
    for (int base = 0; base < nt; base += 8) {
        const int tt = base + 2 * warp + (lane >> 4);
        float kv[8];
        if (tt < nt) {
            unpack8(*reinterpret_cast<const uint4*>(&ks[tt][8 * hl]), kv);
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) kv[e] = 0.f;
        }
#pragma unroll
        for (int j = 0; j < kMaxGroup; ++j) {
            if (j >= G) break;  // uniform
            float s = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) s = fmaf(qr[j][e], kv[e], s);
#pragma unroll
            for (int o = 8; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
            if (hl == 0 && tt < nt) sc[tt * kMaxGroup + j] = s;
        }
    }
    __syncthreads();
    for (int j = warp; j < G; j += 4) {
        const float a = lane < nt ? sc[lane * kMaxGroup + j] : -INFINITY;
        const float b = lane + 32 < nt ? sc[(lane + 32) * kMaxGroup + j] : -INFINITY;
        float v = fmaxf(a, b);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
        const float pa = lane < nt ? expf(a - v) : 0.f;
        const float pb = lane + 32 < nt ? expf(b - v) : 0.f;
        if (lane < nt) sc[lane * kMaxGroup + j] = pa;
        if (lane + 32 < nt) sc[(lane + 32) * kMaxGroup + j] = pb;
        const float s = warp_sum(pa + pb);
        if (lane == 0) {
            mxs[j] = v;
            sms[j] = s;
        }
    }
    __syncthreads();
    float acc[kMaxGroup][4];
#pragma unroll
    for (int j = 0; j < kMaxGroup; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[j][e] = 0.f;
    for (int tt = warp; tt < nt; tt += 4) {
        float vv[4];
        load4(&vs[tt][4 * lane], vv);
        const float4 p0 = *reinterpret_cast<const float4*>(sc + tt * kMaxGroup);
        const float4 p1 = *reinterpret_cast<const float4*>(sc + tt * kMaxGroup + 4);
        const float pj[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
#pragma unroll
        for (int j = 0; j < kMaxGroup; ++j)
            if (j < G)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[j][e] = fmaf(pj[j], vv[e], acc[j][e]);
    }
    float* red = reinterpret_cast<float*>(const_cast<__half*>(&ks[0][0]));  // [4][G][D]
#pragma unroll
    for (int j = 0; j < kMaxGroup; ++j)
        if (j < G)
            *reinterpret_cast<float4*>(red + ((size_t)warp * G + j) * kHeadDim + 4 * lane) =
                make_float4(acc[j][0], acc[j][1], acc[j][2], acc[j][3]);
    __syncthreads();
    const int d = threadIdx.x;
    for (int j = 0; j < G; ++j) {
        float a = 0.f;
#pragma unroll
        for (int w = 0; w < 4; ++w) a += red[((size_t)w * G + j) * kHeadDim + d];
        float* pp = part + (size_t)j * nchunk * kPartial;
        pp[d] = a;
        if (d == 0) {
            pp[kHeadDim] = mxs[j];
            pp[kHeadDim + 1] = sms[j];
        }
    }
}

// ---- attention: per-chunk partials ----
// CTA (chunk c, kv head g, row m) over tokens [64c, 64c + 64) of the row's cached tokens, for
// the G = Hq / Hkv q heads of g at once (their K and V rows are read once): the chunk's K and V
// rows (2 x 16 KB) are copied to shared memory with every copy in flight at once, then scores
// s = scale * q . k, the chunk max, p = exp(s - max), sum p and acc = sum p v, written as
// partial [m][h][c] = (acc[D], max, sum).  Chunks at or past the row's length write nothing.
__global__ void __launch_bounds__(128) attn_partial_kernel(
    const __half* __restrict__ q, const __half* __restrict__ k_cache,
    const __half* __restrict__ v_cache, const int32_t* __restrict__ len, int Hq, int Hkv,
    int64_t L_max, float scale, float* part, int nchunk) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ __align__(16) __half ks[kChunk][kHeadDim];
    __shared__ __align__(16) __half vs[kChunk][kHeadDim];
    __shared__ __align__(16) float qs[kMaxGroup * kHeadDim];
    __shared__ __align__(16) float sc[kChunk * kMaxGroup];
    __shared__ float mx[kMaxGroup], sm[kMaxGroup];
    const int c = blockIdx.x, g = blockIdx.y, m = blockIdx.z;
    const int G = Hq / Hkv;
    const int L = (int)min((int64_t)max(len[m], 0), L_max);  // cached tokens of row m
    const int t0 = c * kChunk;
    if (t0 >= L) return;
    const int nt = min(kChunk, L - t0);
    const size_t kv0 = ((size_t)m * Hkv + g) * L_max + t0;  // row of token t0
    {
        const uint32_t kss = (uint32_t)__cvta_generic_to_shared(&ks[0][0]);
        const uint32_t vss = (uint32_t)__cvta_generic_to_shared(&vs[0][0]);
        for (int u = threadIdx.x; u < nt * (kHeadDim / 8); u += blockDim.x) {  // 16-byte pieces
            cp_async16(kss + 16 * u, k_cache + kv0 * kHeadDim + 8 * u);
            cp_async16(vss + 16 * u, v_cache + kv0 * kHeadDim + 8 * u);
        }
        cp_async_commit();
    }
    for (int i = threadIdx.x; i < G * kHeadDim; i += blockDim.x)
        qs[i] = scale * __half2float(q[((size_t)m * Hq + g * G) * kHeadDim + i]);
    asm volatile("cp.async.wait_all;\n" ::: "memory");
    __syncthreads();
    chunk_core(ks, vs, qs, sc, mx, sm, nt, G,
               part + (((size_t)m * Hq + g * G) * nchunk + c) * kPartial, nchunk);
}

// ---- attention: combine the chunk partials ----
// out[m][h][d] = sum_c e^(max_c - M) acc_c[d] / sum_c e^(max_c - M) sum_c, M = max_c max_c.
// 512 threads: each chunk's (max, sum) is read once, by one thread, into shared memory; the
// four 128-thread groups q take the chunks c = q mod 4 (8 independent loads in flight per
// thread) and their sums are added in group order; the denominator by warp 0.  Fixed orders:
// the result is deterministic.
constexpr int kCombineMax = 2048;  // chunks held in shared memory per pass
constexpr int kCombineThreads = 512;
__global__ void __launch_bounds__(kCombineThreads) attn_combine_kernel(
    const float* __restrict__ part, const int32_t* __restrict__ len, int len_is_pos, int Hq,
    int nchunk, __half* out) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ float fs[kCombineMax], ss[kCombineMax];
    __shared__ float red[kCombineThreads / 32];
    __shared__ float nums[4][kHeadDim];
    __shared__ float den_s;
    const int h = blockIdx.x, m = blockIdx.y, tid = threadIdx.x;
    const int d = tid & (kHeadDim - 1), q = tid >> 7;
    const int64_t n = (int64_t)len[m] + (len_is_pos ? 1 : 0);
    const int nc = (int)((min(max(n, (int64_t)0), (int64_t)nchunk * kChunk) + kChunk - 1) /
                         kChunk);
    __half* o = out + ((size_t)m * Hq + h) * kHeadDim;
    if (nc == 0) {  // no cached token: zeros
        if (q == 0) o[d] = __float2half_rn(0.f);
        return;
    }
    const float* pp = part + ((size_t)m * Hq + h) * nchunk * kPartial;
    // M = max over all chunks (order-independent); the first pass's (max, sum) stay in smem
    const int n0 = min(kCombineMax, nc);
    float lm = -INFINITY;
    for (int cc = tid; cc < nc; cc += kCombineThreads) {
        const float mc = pp[(size_t)cc * kPartial + kHeadDim];
        lm = fmaxf(lm, mc);
        if (cc < n0) {
            fs[cc] = mc;
            ss[cc] = pp[(size_t)cc * kPartial + kHeadDim + 1];
        }
    }
#pragma unroll
    for (int w = 16; w > 0; w >>= 1) lm = fmaxf(lm, __shfl_xor_sync(0xffffffffu, lm, w));
    if ((tid & 31) == 0) red[tid >> 5] = lm;
    __syncthreads();
    float M = red[0];
#pragma unroll
    for (int k = 1; k < kCombineThreads / 32; ++k) M = fmaxf(M, red[k]);
    float num = 0.f, dl = 0.f;  // dl: warp 0's share of the denominator
    for (int c0 = 0; c0 < nc; c0 += kCombineMax) {
        const int cnt = min(kCombineMax, nc - c0);
        if (c0 > 0) {
            __syncthreads();  // the previous pass is done with fs / ss
            for (int cc = tid; cc < cnt; cc += kCombineThreads) {
                fs[cc] = pp[(size_t)(c0 + cc) * kPartial + kHeadDim];
                ss[cc] = pp[(size_t)(c0 + cc) * kPartial + kHeadDim + 1];
            }
        }
        __syncthreads();
        for (int cc = tid; cc < cnt; cc += kCombineThreads) fs[cc] = expf(fs[cc] - M);
        __syncthreads();
        if (tid < 32)
            for (int cc = tid; cc < cnt; cc += 32) dl = fmaf(fs[cc], ss[cc], dl);
        int cc = q;
        for (; cc + 28 < cnt; cc += 32) {  // 8 chunks of this group per round
            float a[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) a[u] = pp[(size_t)(c0 + cc + 4 * u) * kPartial + d];
#pragma unroll
            for (int u = 0; u < 8; ++u) num = fmaf(fs[cc + 4 * u], a[u], num);
        }
        for (; cc < cnt; cc += 4) num = fmaf(fs[cc], pp[(size_t)(c0 + cc) * kPartial + d], num);
    }
    if (tid < 32) {
        dl = warp_sum(dl);
        if (tid == 0) den_s = dl;
    }
    nums[q][d] = num;
    __syncthreads();
    if (q == 0)
        o[d] = __float2half_rn((nums[0][d] + nums[1][d] + nums[2][d] + nums[3][d]) / den_s);
}

// ---- attention partials with the q/k norm, rotation and cache append folded in ----
// CTA (chunk c, kv head g, row m), n = clamp(pos[m] + 1, 0, L_max) tokens: the CTA normalises
// and rotates its G q heads (warp j: head g G + j), stages its chunk's cached K and V, and if
// the chunk holds position pos[m] (< L_max) computes the new k (norm, rotation) and v, stores
// them in the caches and uses them in place of the staged row.  Then the chunk partial as in
// attn_partial_kernel, combined by attn_combine_kernel with len = n.
__global__ void __launch_bounds__(128) attn_qkv_kernel(
    const __half* __restrict__ qkv, const __half* __restrict__ qw, const __half* __restrict__ kw,
    const int32_t* __restrict__ pos, int Hq, int Hkv, float log2_theta, float eps,
    __half* k_cache, __half* v_cache, int64_t L_max, float scale, float* part, int nchunk) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ __align__(16) __half ks[kChunk][kHeadDim];
    __shared__ __align__(16) __half vs[kChunk][kHeadDim];
    __shared__ __align__(16) float qs[kMaxGroup * kHeadDim];
    __shared__ __align__(16) float sc[kChunk * kMaxGroup];
    __shared__ float mx[kMaxGroup], sm[kMaxGroup];
    const int c = blockIdx.x, g = blockIdx.y, m = blockIdx.z;
    const int G = Hq / Hkv, nh = Hq + 2 * Hkv;
    const int64_t p = pos[m];
    const int n = (int)min(max(p + 1, (int64_t)0), L_max);  // tokens attended
    const int t0 = c * kChunk;
    if (t0 >= n) return;
    const int nt = min(kChunk, n - t0);
    const bool holds_new = p >= t0 && p < t0 + nt;  // (then p < L_max)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const size_t kv0 = ((size_t)m * Hkv + g) * L_max + t0;
    {
        const uint32_t kss = (uint32_t)__cvta_generic_to_shared(&ks[0][0]);
        const uint32_t vss = (uint32_t)__cvta_generic_to_shared(&vs[0][0]);
        for (int u = threadIdx.x; u < nt * (kHeadDim / 8); u += blockDim.x) {
            cp_async16(kss + 16 * u, k_cache + kv0 * kHeadDim + 8 * u);
            cp_async16(vss + 16 * u, v_cache + kv0 * kHeadDim + 8 * u);
        }
        cp_async_commit();
    }
    float cs[4], sn[4];
    rope_angles(lane, p, log2_theta, cs, sn);
    const __half* row = qkv + (size_t)m * nh * kHeadDim;
    for (int j = warp; j < G; j += 4) {
        float x[4], o[4];
        load4(row + (size_t)(g * G + j) * kHeadDim + 4 * lane, x);
        norm_rope4(x, qw, lane, cs, sn, eps, o);
        const uint2 rq = round4(o);  // the fp16 q of the separate path
        const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&rq.x));
        const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&rq.y));
        *reinterpret_cast<float4*>(qs + j * kHeadDim + 4 * lane) =
            make_float4(scale * a.x, scale * a.y, scale * b.x, scale * b.y);
    }
    uint2 knew = make_uint2(0u, 0u), vnew = make_uint2(0u, 0u);
    if (holds_new && warp < 2) {
        if (warp == 0) {
            float x[4], o[4];
            load4(row + (size_t)(Hq + g) * kHeadDim + 4 * lane, x);
            norm_rope4(x, kw, lane, cs, sn, eps, o);
            knew = round4(o);
        } else {
            vnew = *reinterpret_cast<const uint2*>(row + (size_t)(Hq + Hkv + g) * kHeadDim +
                                                   4 * lane);
        }
    }
    asm volatile("cp.async.wait_all;\n" ::: "memory");
    __syncthreads();
    if (holds_new && warp < 2) {  // the new token replaces the staged (stale) row
        const int tt = (int)(p - t0);
        __half* cache = warp == 0 ? k_cache : v_cache;
        const uint2 w = warp == 0 ? knew : vnew;
        *reinterpret_cast<uint2*>(warp == 0 ? &ks[tt][4 * lane] : &vs[tt][4 * lane]) = w;
        *reinterpret_cast<uint2*>(cache + (kv0 + tt) * kHeadDim + 4 * lane) = w;
    }
    __syncthreads();
    chunk_core(ks, vs, qs, sc, mx, sm, nt, G,
               part + (((size_t)m * Hq + g * G) * nchunk + c) * kPartial, nchunk);
}

// ---- SiLU(gate) * up ----
__global__ void __launch_bounds__(256) silu_mul_kernel(const __half* __restrict__ gu, int64_t I,
                                                       int64_t chunks, __half* hout) {
    pdl_launch_dependents();
    pdl_wait();
    const int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;  // 8-element chunk
    if (u >= chunks) return;
    const int64_t per_row = I / 8;
    const int64_t m = u / per_row, i = (u - m * per_row) * 8;
    float g[8], up[8], y[8];
    unpack8(*reinterpret_cast<const uint4*>(gu + m * 2 * I + i), g);
    unpack8(*reinterpret_cast<const uint4*>(gu + m * 2 * I + I + i), up);
#pragma unroll
    for (int e = 0; e < 8; ++e) y[e] = g[e] / (1.f + expf(-g[e])) * up[e];
    *reinterpret_cast<uint4*>(hout + m * I + i) = pack8(y);
}

// ---- embedding gather ----
__global__ void __launch_bounds__(256) embed_kernel(const __half* __restrict__ E,
                                                    const int32_t* __restrict__ tokens, int64_t V,
                                                    int64_t H, __half* X) {
    pdl_launch_dependents();
    pdl_wait();
    const int m = blockIdx.x;
    const int64_t t = tokens[m];
    const bool ok = t >= 0 && t < V;
    for (int64_t i = threadIdx.x; i < H / 8; i += blockDim.x) {
        const uint4 v = ok ? *reinterpret_cast<const uint4*>(E + t * H + 8 * i)
                           : make_uint4(0u, 0u, 0u, 0u);
        *reinterpret_cast<uint4*>(X + (size_t)m * H + 8 * i) = v;
    }
}

// ---- greedy argmax (ties: the smallest index; NaN never wins) ----
constexpr int kArgThreads = 1024;
// (bv, bi) starts at (-inf, none); a value must beat it strictly, ties between real candidates
// go to the smaller index, so -inf and NaN never win.
constexpr int kNone = 0x7fffffff;
__device__ __forceinline__ void better(float& bv, int& bi, float v, int i) {
    if (v > bv || (v == bv && bi != kNone && i < bi)) {
        bv = v;
        bi = i;
    }
}
__global__ void __launch_bounds__(kArgThreads) argmax_kernel(const __half* __restrict__ logits,
                                                             int64_t V, int32_t* out) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ float bvs[kArgThreads / 32];
    __shared__ int bis[kArgThreads / 32];
    const int m = blockIdx.x;
    const __half* row = logits + (size_t)m * V;
    float bv = -INFINITY;
    int bi = kNone;
    if (((uintptr_t)row & 15u) == 0 && V % 8 == 0) {
        // 16-byte loads, four in flight per thread
        const int64_t n8 = V / 8;
        for (int64_t b = threadIdx.x; b < n8; b += 4 * kArgThreads) {
            uint4 u[4];
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int64_t i8 = b + r * kArgThreads;
                u[r] = i8 < n8 ? *reinterpret_cast<const uint4*>(row + 8 * i8)
                               : make_uint4(0xfc00fc00u, 0xfc00fc00u, 0xfc00fc00u, 0xfc00fc00u);
            }
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                float f[8];
                unpack8(u[r], f);
                const int i0 = (int)(8 * (b + r * kArgThreads));
#pragma unroll
                for (int e = 0; e < 8; ++e) better(bv, bi, f[e], i0 + e);
            }
        }
    } else {
        for (int64_t i = threadIdx.x; i < V; i += kArgThreads)
            better(bv, bi, __half2float(row[i]), (int)i);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float v = __shfl_xor_sync(0xffffffffu, bv, o);
        const int i = __shfl_xor_sync(0xffffffffu, bi, o);
        better(bv, bi, v, i);
    }
    if ((threadIdx.x & 31) == 0) {
        bvs[threadIdx.x >> 5] = bv;
        bis[threadIdx.x >> 5] = bi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float v = bvs[0];
        int i = bis[0];
        for (int k = 1; k < kArgThreads / 32; ++k) better(v, i, bvs[k], bis[k]);
        out[m] = i == kNone ? 0 : i;  // no value above -inf: index 0
    }
}

// Launch with programmatic stream serialization (the kernel may start while its predecessor
// finishes; it waits for it with griddepcontrol.wait).
template <typename... KArgs, typename... Args>
laq_status launch_pdl(void (*fn)(KArgs...), dim3 grid, dim3 block, cudaStream_t stream,
                      Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, fn, args...);
    return e == cudaSuccess ? LAQ_OK : LAQ_ERR_CUDA;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace
}  // namespace laq

using namespace laq;

extern "C" {

laq_status laq_rmsnorm(const void* X, const void* R, void* R_out, const void* w, int64_t M,
                       int64_t H, float eps, void* Y, void* stream) {
    if (!X || !w || !Y) return LAQ_ERR_NULL;
    if (M < 1 || M > 65535 || H < 8 || H % 8 || H > 8 * kRmsThreads * kRmsChunks)
        return LAQ_ERR_SHAPE;
    if (!(eps >= 0.f)) return LAQ_ERR_SHAPE;
    if (!aligned16(X) || !aligned16(w) || !aligned16(Y) || (R && !aligned16(R)) ||
        (R_out && !aligned16(R_out)))
        return LAQ_ERR_ALIGN;
    return launch_pdl(rmsnorm_kernel, dim3((unsigned)M), dim3(kRmsThreads),
                      static_cast<cudaStream_t>(stream), static_cast<const __half*>(X),
                      static_cast<const __half*>(R), static_cast<__half*>(R_out),
                      static_cast<const __half*>(w), (int)H, eps, static_cast<__half*>(Y));
}

laq_status laq_qk_norm_rope(const void* qkv, const void* q_norm_w, const void* k_norm_w,
                            const int32_t* pos, int64_t M, int32_t Hq, int32_t Hkv, int32_t D,
                            float theta, float eps, void* q_out, void* k_cache, void* v_cache,
                            int64_t L_max, void* stream) {
    if (!qkv || !q_norm_w || !k_norm_w || !pos || !q_out || !k_cache || !v_cache)
        return LAQ_ERR_NULL;
    if (D != kHeadDim || M < 1 || M > 65535 || Hq < 1 || Hkv < 1 || Hq % Hkv ||
        Hq / Hkv > kMaxGroup || L_max < 1 || !(theta > 1.f) || !(eps >= 0.f))
        return LAQ_ERR_SHAPE;
    if (((uintptr_t)qkv & 7u) || ((uintptr_t)q_out & 7u) || ((uintptr_t)k_cache & 7u) ||
        ((uintptr_t)v_cache & 7u))
        return LAQ_ERR_ALIGN;
    const int nh = Hq + 2 * Hkv;
    return launch_pdl(qk_norm_rope_kernel, dim3((unsigned)((nh + 3) / 4), (unsigned)M), dim3(128),
                      static_cast<cudaStream_t>(stream), static_cast<const __half*>(qkv),
                      static_cast<const __half*>(q_norm_w), static_cast<const __half*>(k_norm_w),
                      pos, (int)Hq, (int)Hkv, log2f(theta), eps, static_cast<__half*>(q_out),
                      static_cast<__half*>(k_cache), static_cast<__half*>(v_cache), L_max);
}

size_t laq_attention_workspace_bytes(int64_t M, int32_t Hq, int64_t L_max) {
    if (M < 1 || Hq < 1 || L_max < 1) return 0;
    const int64_t nchunk = (L_max + kChunk - 1) / kChunk;
    return (size_t)M * Hq * nchunk * kPartial * sizeof(float);
}

laq_status laq_attention_decode(const void* q, const void* k_cache, const void* v_cache,
                                const int32_t* len, int64_t M, int32_t Hq, int32_t Hkv,
                                int32_t D, int64_t L_max, float scale, void* out,
                                void* workspace, size_t workspace_bytes, void* stream) {
    if (!q || !k_cache || !v_cache || !len || !out || !workspace) return LAQ_ERR_NULL;
    if (D != kHeadDim || M < 1 || M > 65535 || Hq < 1 || Hkv < 1 || Hq % Hkv ||
        Hq / Hkv > kMaxGroup || Hkv > 65535 || L_max < 1 || !(scale > 0.f))
        return LAQ_ERR_SHAPE;
    if (!aligned16(k_cache) || !aligned16(v_cache) || ((uintptr_t)q & 1u) ||
        ((uintptr_t)out & 1u) || ((uintptr_t)workspace & 3u))
        return LAQ_ERR_ALIGN;
    if (workspace_bytes < laq_attention_workspace_bytes(M, Hq, L_max)) return LAQ_ERR_WORKSPACE;
    const int64_t nchunk = (L_max + kChunk - 1) / kChunk;
    if (nchunk > 0x7fffffff) return LAQ_ERR_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    laq_status st = launch_pdl(attn_partial_kernel, dim3((unsigned)nchunk, (unsigned)Hkv,
                                                         (unsigned)M),
                               dim3(128), s, static_cast<const __half*>(q),
                               static_cast<const __half*>(k_cache),
                               static_cast<const __half*>(v_cache), len, (int)Hq, (int)Hkv, L_max,
                               scale, static_cast<float*>(workspace), (int)nchunk);
    if (st != LAQ_OK) return st;
    return launch_pdl(attn_combine_kernel, dim3((unsigned)Hq, (unsigned)M),
                      dim3(kCombineThreads), s, static_cast<const float*>(workspace), len, 0,
                      (int)Hq, (int)nchunk, static_cast<__half*>(out));
}

size_t laq_attention_qkv_workspace_bytes(int64_t M, int32_t Hq, int32_t Hkv, int64_t L_max) {
    if (M < 1 || Hq < 1 || Hkv < 1 || L_max < 1) return 0;
    return laq_attention_workspace_bytes(M, Hq, L_max);
}

laq_status laq_attention_qkv(const void* qkv, const void* q_norm_w, const void* k_norm_w,
                             const int32_t* pos, int64_t M, int32_t Hq, int32_t Hkv, int32_t D,
                             float theta, float eps, void* k_cache, void* v_cache, int64_t L_max,
                             float scale, void* out, void* workspace, size_t workspace_bytes,
                             void* stream) {
    if (!qkv || !q_norm_w || !k_norm_w || !pos || !k_cache || !v_cache || !out || !workspace)
        return LAQ_ERR_NULL;
    if (D != kHeadDim || M < 1 || M > 65535 || Hq < 1 || Hkv < 1 || Hq % Hkv ||
        Hq / Hkv > kMaxGroup || Hkv > 65535 || L_max < 1 || !(theta > 1.f) || !(eps >= 0.f) ||
        !(scale > 0.f))
        return LAQ_ERR_SHAPE;
    if (((uintptr_t)qkv & 7u) || !aligned16(k_cache) || !aligned16(v_cache) ||
        ((uintptr_t)out & 1u) || !aligned16(workspace))
        return LAQ_ERR_ALIGN;
    if (workspace_bytes < laq_attention_qkv_workspace_bytes(M, Hq, Hkv, L_max))
        return LAQ_ERR_WORKSPACE;
    const int64_t nchunk = (L_max + kChunk - 1) / kChunk;
    if (nchunk > 0x7fffffff) return LAQ_ERR_SHAPE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    laq_status st = launch_pdl(attn_qkv_kernel, dim3((unsigned)nchunk, (unsigned)Hkv, (unsigned)M),
                               dim3(128), s, static_cast<const __half*>(qkv),
                               static_cast<const __half*>(q_norm_w),
                               static_cast<const __half*>(k_norm_w), pos, (int)Hq, (int)Hkv,
                               log2f(theta), eps, static_cast<__half*>(k_cache),
                               static_cast<__half*>(v_cache), L_max, scale,
                               static_cast<float*>(workspace), (int)nchunk);
    if (st != LAQ_OK) return st;
    return launch_pdl(attn_combine_kernel, dim3((unsigned)Hq, (unsigned)M),
                      dim3(kCombineThreads), s, static_cast<const float*>(workspace), pos, 1,
                      (int)Hq, (int)nchunk, static_cast<__half*>(out));
}

laq_status laq_silu_mul(const void* gate_up, int64_t M, int64_t I, void* h, void* stream) {
    if (!gate_up || !h) return LAQ_ERR_NULL;
    if (M < 1 || I < 8 || I % 8) return LAQ_ERR_SHAPE;
    if (!aligned16(gate_up) || !aligned16(h)) return LAQ_ERR_ALIGN;
    const int64_t chunks = M * I / 8;
    return launch_pdl(silu_mul_kernel, dim3((unsigned)((chunks + 255) / 256)), dim3(256),
                      static_cast<cudaStream_t>(stream), static_cast<const __half*>(gate_up), I,
                      chunks, static_cast<__half*>(h));
}

laq_status laq_embed(const void* E, const int32_t* tokens, int64_t M, int64_t V, int64_t H,
                     void* X, void* stream) {
    if (!E || !tokens || !X) return LAQ_ERR_NULL;
    if (M < 1 || M > 65535 || V < 1 || H < 8 || H % 8) return LAQ_ERR_SHAPE;
    if (!aligned16(E) || !aligned16(X)) return LAQ_ERR_ALIGN;
    return launch_pdl(embed_kernel, dim3((unsigned)M), dim3(256),
                      static_cast<cudaStream_t>(stream), static_cast<const __half*>(E), tokens, V,
                      H, static_cast<__half*>(X));
}

laq_status laq_argmax(const void* logits, int64_t M, int64_t V, int32_t* out, void* stream) {
    if (!logits || !out) return LAQ_ERR_NULL;
    if (M < 1 || M > 65535 || V < 1 || V > 0x7ffffffe) return LAQ_ERR_SHAPE;
    if ((uintptr_t)logits & 1u) return LAQ_ERR_ALIGN;
    return launch_pdl(argmax_kernel, dim3((unsigned)M), dim3(kArgThreads),
                      static_cast<cudaStream_t>(stream), static_cast<const __half*>(logits), V,
                      out);
}

}  // extern "C"
