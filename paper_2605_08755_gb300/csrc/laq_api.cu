// laq_api.cu -- the C ABI of include/laq.h: argument validation, launch planning and dispatch.
// Validation happens before any CUDA call, so invalid arguments are reported without a device.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "laq.h"
#include "laq_internal.cuh"

namespace {

constexpr int64_t kGroup = 128;
constexpr int64_t kMaxK = 65535 * kGroup;  // group index fits a grid dimension
constexpr int64_t kMaxN = int64_t(1) << 24;

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

laq_status check_bits(int bits) { return (bits == 3 || bits == 4) ? LAQ_OK : LAQ_ERR_BITS; }

laq_status check_kn(int64_t K, int64_t N, bool need_tiles) {
    if (K < 0 || N < 0 || K > kMaxK || N > kMaxN) return LAQ_ERR_SHAPE;
    if (K % kGroup) return LAQ_ERR_SHAPE;
    if (need_tiles && N % 16) return LAQ_ERR_SHAPE;
    return LAQ_OK;
}

laq_status from_cuda(cudaError_t e) {
    if (e == cudaSuccess) return LAQ_OK;
    if (e == cudaErrorInvalidConfiguration) return LAQ_ERR_CONFIG;
    return LAQ_ERR_CUDA;
}

// Per-device facts the planner and launcher need, cached on first use.
struct DeviceFacts {
    int sms;
    size_t smem_optin;
};
constexpr int kMaxDevices = 64;
std::atomic<int> g_sms[kMaxDevices];
std::atomic<long long> g_smem[kMaxDevices];

laq_status device_facts(DeviceFacts* f) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return LAQ_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return LAQ_ERR_CUDA;
    int sms = g_sms[dev].load();
    long long smem = g_smem[dev].load();
    if (sms <= 0 || smem <= 0) {
        int a = 0, b = 0;
        if (cudaDeviceGetAttribute(&a, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            return LAQ_ERR_CUDA;
        if (cudaDeviceGetAttribute(&b, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess)
            return LAQ_ERR_CUDA;
        sms = a;
        smem = b;
        g_sms[dev].store(sms);
        g_smem[dev].store(smem);
    }
    f->sms = sms;
    f->smem_optin = (size_t)smem;
    return LAQ_OK;
}

laq_status check_gemm_args(const void* X, int64_t M, int64_t K, int64_t N, const void* packed,
                           const void* s, const uint8_t* z, int bits, void* Y) {
    laq_status st = check_bits(bits);
    if (st != LAQ_OK) return st;
    if (M < 0 || M > 16) return LAQ_ERR_M_RANGE;
    st = check_kn(K, N, true);
    if (st != LAQ_OK) return st;
    if (M == 0 || N == 0) return LAQ_OK;
    if (!Y) return LAQ_ERR_NULL;
    if (!aligned(Y, 16)) return LAQ_ERR_ALIGN;
    if (K == 0) return LAQ_OK;
    if (!X || !packed || !s || !z) return LAQ_ERR_NULL;
    if (!aligned(X, 16) || !aligned(packed, 16) || !aligned(s, 2)) return LAQ_ERR_ALIGN;
    return LAQ_OK;
}

laq_status check_config(const laq_gemm_config* c) {
    if (!c) return LAQ_ERR_NULL;
    if (c->tiles_per_cta != 1 && c->tiles_per_cta != 2 && c->tiles_per_cta != 4)
        return LAQ_ERR_CONFIG;
    if (c->warps < 1 || c->warps > 8) return LAQ_ERR_CONFIG;
    if (c->cluster != 1 && c->cluster != 2 && c->cluster != 4 && c->cluster != 8)
        return LAQ_ERR_CONFIG;
    if (c->stages < 2 || c->stages > 8) return LAQ_ERR_CONFIG;
    if (c->pdl != 0 && c->pdl != 1) return LAQ_ERR_CONFIG;
    return LAQ_OK;
}

int ceil_div(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }

// Launch-shape heuristic.  The kernel is HBM-bound; the plan aims for one wave of CTAs that
// splits the records (16 columns x 128 rows of K) evenly over the SMs with enough copies in
// flight per SM.  Estimated time in units of "records streamed by one SM":
//   max(perfect balance, busiest SM's load at ~2.5x its fair-share rate) + per-wave latency,
// plus a small cost for cluster reductions.
void plan(int64_t M, int64_t K, int64_t N, int bits, int sms, laq_gemm_config* out) {
    const int64_t T = N / 16, G = K / kGroup;
    const int mp = M <= 1 ? 1 : M <= 2 ? 2 : M <= 4 ? 4 : M <= 8 ? 8 : 16;
    double best = 1e300;
    laq_gemm_config bestc = {1, 8, 1, 4, 0, {0, 0, 0}};
    const int nts[3] = {1, 2, 4};
    const int cls[4] = {1, 2, 4, 8};
    const int wps[2] = {4, 8};
    for (int a = 0; a < 3; ++a) {
        const int nt = nts[a];
        if (mp == 16 && nt == 4) continue;  // register pressure: two MMA column halves
        for (int b = 0; b < 4; ++b) {
            const int cl = cls[b];
            if (cl > 1 && cl > G) continue;
            for (int d = 0; d < 2; ++d) {
                const int w = wps[d];
                const int64_t ctas = (int64_t)ceil_div(T, nt) * cl;
                const int64_t gc = (G + cl - 1) / cl;
                const int64_t iters = (gc + w - 1) / w;
                const double cta_rec = (double)nt * iters * w;
                laq::GemmLaunch L = {};
                L.M = (int)M; L.K = (int)K; L.N = (int)N; L.bits = bits;
                L.tiles_per_cta = nt; L.warps = w; L.cluster = cl; L.stages = 4;
                const size_t smem = laq::gemm_smem_bytes(L, nullptr);
                int occ = (int)((228 * 1024) / (smem + 1024));
                const int occ_thr = 16 / w;  // 2 CTAs of 8 warps per SM (launch bounds)
                if (occ > occ_thr) occ = occ_thr;
                if (occ < 1) continue;
                const int64_t slots = (int64_t)sms * occ;
                const int64_t busiest = (ctas + sms - 1) / sms;
                const int64_t waves = (ctas + slots - 1) / slots;
                const double t_bw = (double)T * G / sms;
                const double t_sm = (double)busiest * cta_rec / 2.5;
                double est = (t_bw > t_sm ? t_bw : t_sm) + 12.0 * waves;
                if (cl > 1) est += 2.0;
                if (ctas < sms) est += 0.5 * (double)(sms - ctas) / sms * t_bw;
                if (est < best - 1e-9) {
                    best = est;
                    bestc.tiles_per_cta = nt;
                    bestc.warps = w;
                    bestc.cluster = cl;
                    bestc.stages = 4;
                    bestc.pdl = 0;
                }
            }
        }
    }
    *out = bestc;
}

laq_status run_gemm(const void* X, int64_t M, int64_t K, int64_t N, const void* packed,
                    const void* s, const uint8_t* z, int bits, void* Y,
                    const laq_gemm_config* cfg, void* stream) {
    laq_status st = check_gemm_args(X, M, K, N, packed, s, z, bits, Y);
    if (st != LAQ_OK) return st;
    if (cfg) {
        st = check_config(cfg);
        if (st != LAQ_OK) return st;
    }
    if (M == 0 || N == 0) return LAQ_OK;
    cudaStream_t strm = static_cast<cudaStream_t>(stream);
    if (K == 0) return from_cuda(cudaMemsetAsync(Y, 0, (size_t)M * N * 2, strm));
    DeviceFacts f;
    st = device_facts(&f);
    if (st != LAQ_OK) return st;
    laq_gemm_config c;
    if (cfg) {
        c = *cfg;
    } else {
        plan(M, K, N, bits, f.sms, &c);
    }
    laq::GemmLaunch L;
    L.X = static_cast<const uint16_t*>(X);
    L.packed = static_cast<const uint8_t*>(packed);
    L.s = static_cast<const uint16_t*>(s);
    L.z = z;
    L.Y = static_cast<uint16_t*>(Y);
    L.M = (int)M;
    L.K = (int)K;
    L.N = (int)N;
    L.bits = bits;
    L.tiles_per_cta = c.tiles_per_cta;
    L.warps = c.warps;
    L.cluster = c.cluster;
    L.stages = c.stages;
    L.pdl = c.pdl;
    return from_cuda(laq::launch_gemm(L, f.smem_optin, strm));
}

}  // namespace

extern "C" {

const char* laq_status_str(int status) {
    switch (status) {
        case LAQ_OK: return "LAQ_OK";
        case LAQ_ERR_NULL: return "LAQ_ERR_NULL: a required pointer is NULL";
        case LAQ_ERR_BITS: return "LAQ_ERR_BITS: bits must be 3 or 4";
        case LAQ_ERR_GROUP: return "LAQ_ERR_GROUP: group size must be 128";
        case LAQ_ERR_SHAPE: return "LAQ_ERR_SHAPE: unsupported K or N";
        case LAQ_ERR_ALIGN: return "LAQ_ERR_ALIGN: misaligned pointer";
        case LAQ_ERR_M_RANGE: return "LAQ_ERR_M_RANGE: M must be in 0..16";
        case LAQ_ERR_CUDA: return "LAQ_ERR_CUDA: CUDA runtime error";
        case LAQ_ERR_TIMEOUT: return "LAQ_ERR_TIMEOUT: a device-side wait gave up";
        case LAQ_ERR_CONFIG: return "LAQ_ERR_CONFIG: unsupported launch configuration";
        default: return "unknown laq status";
    }
}

int laq_version(void) { return 1; }

size_t laq_packed_bytes(int64_t K, int64_t N, int bits) {
    if (check_bits(bits) != LAQ_OK || check_kn(K, N, false) != LAQ_OK) return 0;
    return (size_t)(K * N * bits / 8);
}

laq_status laq_quantize_rtn(const void* W, int64_t K, int64_t N, int bits, int group,
                            uint8_t* codes, void* s, uint8_t* z, void* stream) {
    laq_status st = check_bits(bits);
    if (st != LAQ_OK) return st;
    if (group != kGroup) return LAQ_ERR_GROUP;
    st = check_kn(K, N, false);
    if (st != LAQ_OK) return st;
    if (K == 0 || N == 0) return LAQ_OK;
    if (!W || !codes || !s || !z) return LAQ_ERR_NULL;
    if (!aligned(W, 2) || !aligned(s, 2)) return LAQ_ERR_ALIGN;
    return from_cuda(laq::launch_quantize_rtn(static_cast<const uint16_t*>(W), K, N, bits, codes,
                                              static_cast<uint16_t*>(s), z,
                                              static_cast<cudaStream_t>(stream)));
}

laq_status laq_pack(const uint8_t* codes, int64_t K, int64_t N, int bits, void* packed,
                    void* stream) {
    laq_status st = check_bits(bits);
    if (st != LAQ_OK) return st;
    st = check_kn(K, N, true);
    if (st != LAQ_OK) return st;
    if (K == 0 || N == 0) return LAQ_OK;
    if (!codes || !packed) return LAQ_ERR_NULL;
    if (!aligned(packed, 16)) return LAQ_ERR_ALIGN;
    return from_cuda(laq::launch_pack(codes, K, N, bits, static_cast<uint32_t*>(packed),
                                      static_cast<cudaStream_t>(stream)));
}

laq_status laq_unpack(const void* packed, int64_t K, int64_t N, int bits, uint8_t* codes,
                      void* stream) {
    laq_status st = check_bits(bits);
    if (st != LAQ_OK) return st;
    st = check_kn(K, N, true);
    if (st != LAQ_OK) return st;
    if (K == 0 || N == 0) return LAQ_OK;
    if (!codes || !packed) return LAQ_ERR_NULL;
    if (!aligned(packed, 16)) return LAQ_ERR_ALIGN;
    return from_cuda(laq::launch_unpack(static_cast<const uint32_t*>(packed), K, N, bits, codes,
                                        static_cast<cudaStream_t>(stream)));
}

laq_status laq_gemm_plan(int64_t M, int64_t K, int64_t N, int bits, int num_sms,
                         laq_gemm_config* out) {
    if (!out) return LAQ_ERR_NULL;
    laq_status st = check_bits(bits);
    if (st != LAQ_OK) return st;
    if (M < 0 || M > 16) return LAQ_ERR_M_RANGE;
    st = check_kn(K, N, true);
    if (st != LAQ_OK) return st;
    if (num_sms < 1) return LAQ_ERR_CONFIG;
    plan(M < 1 ? 1 : M, K, N, bits, num_sms, out);
    return LAQ_OK;
}

laq_status laq_gemm_wxg128(const void* X, int64_t M, int64_t K, int64_t N, const void* packed,
                           const void* s, const uint8_t* z, int bits, void* Y, void* stream) {
    return run_gemm(X, M, K, N, packed, s, z, bits, Y, nullptr, stream);
}

laq_status laq_gemm_wxg128_config(const void* X, int64_t M, int64_t K, int64_t N,
                                  const void* packed, const void* s, const uint8_t* z, int bits,
                                  void* Y, const laq_gemm_config* cfg, void* stream) {
    if (!cfg) return LAQ_ERR_NULL;
    return run_gemm(X, M, K, N, packed, s, z, bits, Y, cfg, stream);
}

}  // extern "C"
