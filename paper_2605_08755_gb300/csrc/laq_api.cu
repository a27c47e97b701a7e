// laq_api.cu -- the C ABI of include/laq.h: argument validation, launch planning and dispatch.
// Validation happens before any CUDA call, so invalid arguments are reported without a device.
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <climits>
#include <mutex>
#include <vector>

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
    if (!aligned(X, 16) || !aligned(packed, 16) || !aligned(s, 16) || !aligned(z, 16))
        return LAQ_ERR_ALIGN;
    return LAQ_OK;
}

laq_status check_config(const laq_gemm_config* c) {
    if (!c) return LAQ_ERR_NULL;
    if (c->tiles_per_cta != 1 && c->tiles_per_cta != 2 && c->tiles_per_cta != 4 &&
        c->tiles_per_cta != 8)
        return LAQ_ERR_CONFIG;
    if (c->warps < 1 || c->warps > 16) return LAQ_ERR_CONFIG;
    if (c->warps % c->tiles_per_cta) return LAQ_ERR_CONFIG;  // whole warps per tile
    if (c->cluster != 1 && c->cluster != 2 && c->cluster != 4 && c->cluster != 8)
        return LAQ_ERR_CONFIG;
    if (c->stages < 2 || c->stages > 16) return LAQ_ERR_CONFIG;
    if (c->pdl != 0 && c->pdl != 1) return LAQ_ERR_CONFIG;
    return LAQ_OK;
}

int ceil_div(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }

// Launch-shape plan: tiles per CTA (NT), K split over a cluster (C), warps and ring depth.
//  * M = 1, 2: the cheapest split by estimated SM time -- records per warp plus a start cost of
//    two records' time per wave of CTAs, x the waves (two 8-warp CTAs per SM at a time), x 1.3
//    when two CTAs share an SM (16 warps retire a record in ~0.65x the time of 8; measured on
//    GB300), x 1.02 for a cluster's reduction -- over NT, C in {1, 2, 4, 8}.  Several waves win
//    for wide outputs: a single wave of 8-tile CTAs leaves the Qwen3-8B gate|up (1536 tiles)
//    with 1.26 CTAs per SM, the SMs holding two doing twice the work (measured on GB300, fused
//    Qwen3-8B pass: 1624 -> 1262 us with 2-tile CTAs in three waves).
//  * M > 2: every CTA reads X for its whole K range, M rows of it -- at M = 16 with one tile per
//    CTA that is 5x the CTA's weight bytes (b = 3).  So X is shared across 4 (M <= 4) or 8 tiles
//    per CTA and K is split over a cluster (which also splits X) until there is about one CTA
//    per SM.  Measured on GB300, fused Qwen3-4B pass, against the rule above: W3 M = 4 887 vs
//    915 us, W4 M = 3 856 vs 889, M = 5 1160 vs 1235, M = 8 1183 vs 1586, M = 16 1791 vs 2574;
//    at M = 2 the rule above is the faster one (W3 810 vs 868 us).
//  * M <= 4 with fewer than 1.5 tiles per SM (N < 24 x SMs) and a long K, where the first plan
//    leaves a warp more than 5 records (the 2560 x 9728 down projection: 160 tiles on 152 SMs,
//    ~10 records per warp): 4-warp CTAs of 2 tiles instead, K split over a cluster that
//    doubles until a warp holds at most 5 records and the grid covers every SM (down: 640
//    CTAs, 5 records per warp; measured on GB300 in the Qwen3-4B pass, W3 and W4: 1.6 us less
//    per down launch).  Shorter K (o, q, k, v) measured best with the rule above.
//  * M > 4: 16 warps per CTA where the plan above leaves one 8-warp CTA per SM (wide outputs;
//    the long-K down projection at M > 8, with half the cluster).
//  * Eight warps otherwise (fewer when a CTA owns fewer groups), and a cp.async ring deep
//    enough to hold all of a warp's records (at most 16) within 100 KB.
// Shared memory of one SM of sm_100 / sm_103 and what the hardware reserves per CTA.
constexpr size_t kSmemPerSm = 228 * 1024, kSmemPerCta = 1024;

void plan(int64_t M, int64_t K, int64_t N, int bits, int sms, laq_gemm_config* out);

// X of a long K, or of 3-4 rows, beside the ring can leave a CTA just too large for two to share
// an SM; where the grid needs two per SM, the ring loses stages until two fit (measured on
// GB300, W4 M = 4 fused Qwen3-4B pass: gate|up 11 -> 10 stages, 1032 -> 940 us).
void fit_two_ctas(int64_t M, int64_t K, int64_t N, int bits, int sms, laq_gemm_config* c) {
    const int64_t ctas = (int64_t)ceil_div(N / 16, c->tiles_per_cta) * c->cluster;
    if (ctas <= sms) return;
    laq::GemmLaunch L;
    L.M = (int)M;
    L.K = (int)K;
    L.N = (int)N;
    L.bits = bits;
    L.tiles_per_cta = c->tiles_per_cta;
    L.warps = c->warps;
    L.cluster = c->cluster;
    L.pdl = 0;
    for (; c->stages > 2; --c->stages) {
        L.stages = c->stages;
        if (2 * (laq::gemm_smem_bytes(L, nullptr) + kSmemPerCta) <= kSmemPerSm) break;
    }
}

// Warps and ring depth of a shape (nt tiles per CTA, K over a cluster of cl): at most
// warps_max warps, whole warps per tile, a ring deep enough for every record of a warp (at most
// 16 slots) within 100 KB.
void shape(int64_t G, int64_t rec, int nt, int cl, int64_t warps_max, laq_gemm_config* out) {
    const int64_t gc = (G + cl - 1) / cl;
    const int64_t wt_max = warps_max / nt;  // warps per tile
    const int64_t wt = gc < wt_max ? (gc < 1 ? 1 : gc) : wt_max;
    const int w = (int)(wt * nt);
    const int64_t iters = (gc + wt - 1) / wt;
    int st = (int)(iters + 1 > 16 ? 16 : (iters + 1 < 2 ? 2 : iters + 1));
    while (st > 2 && (int64_t)w * st * rec > 100 * 1024) --st;
    out->tiles_per_cta = nt;
    out->warps = w;
    out->cluster = cl;
    out->stages = st;
    out->pdl = 0;
    out->reserved[0] = out->reserved[1] = out->reserved[2] = 0;
}

void plan(int64_t M, int64_t K, int64_t N, int bits, int sms, laq_gemm_config* out) {
    const int64_t T = N / 16, G = K / kGroup;
    const int64_t rec = bits == 4 ? 1024 : 768;
    int best_nt = 8, best_cl = 1;
    int64_t warps_max = 8;
    // M = 3, 4 take the first rule's down shape (below) where it applies, else the batch rule
    bool batch = M > 4;
    if (M > 2 && M <= 4) {
        laq_gemm_config one;
        plan(1, K, N, bits, sms, &one);
        batch = !(one.warps == 4 && one.tiles_per_cta == 2 && one.cluster > 1);
        if (!batch) {
            *out = one;
            fit_two_ctas(M, K, N, bits, sms, out);
            return;
        }
    }
    if (batch) {
        int nt = M <= 4 ? 4 : 8;
        while (nt > 1 && ceil_div(T, nt) < sms / 8) nt /= 2;
        int cl = 1;
        while (cl < 8 && cl * 2 <= G && (int64_t)ceil_div(T, nt) * cl < sms) cl *= 2;
        best_nt = nt;
        best_cl = cl;
        // M > 4: one 8-warp CTA per SM leaves each scheduler two warps, too few to hide the
        // MMA and shared-memory latency of the wider batch.  16-warp CTAs (two warps per tile)
        // where the output alone fills the SMs, and for the long K of the down projection at
        // M > 8 with half the cluster (measured on GB300, Qwen3-4B W3 pass: gate|up -140 us at
        // M = 8 and -196 us at M = 16, down -266 us at M = 16; q|k|v, o and M <= 4 within 2%).
        if (M > 8 && G >= 64 && best_cl >= 2) {
            warps_max = 16;
            best_cl /= 2;
        } else if (M > 4 && M <= 8 && G >= 64 && 2 * T < 3 * (int64_t)sms &&
                   (bits == 4 || M >= 7)) {
            // M = 5..8 (W3: 7, 8), a long K and fewer than 1.5 tiles per SM (the down
            // projection): 4-tile CTAs of 4 warps, one per tile, K over a cluster of 8 -- small
            // CTAs, two or more per SM.  Measured on GB300, fused Qwen3-4B pass, against 8-tile
            // 8-warp CTAs with a cluster of 8: W4 M = 5 1135 -> 1104 us, M = 8 1350 -> 1130 (one
            // such CTA per SM fits there; with a shallower ring, 1202), W3 M = 8 1186 -> 1166;
            // but W3 M = 5, 6 1162 -> 1184, 1173 -> 1195, so W3 keeps the 8-warp shape there.
            best_nt = 4;
            best_cl = 8;
            warps_max = 4;
        } else if (M > 4 && best_cl == 1 && (int64_t)ceil_div(T, best_nt) >= sms) {
            warps_max = 16;
            // one 16-warp CTA per SM at a time: a grid between one and two CTAs per SM leaves
            // some SMs two in turn, so K goes over a cluster of 2 (measured on GB300, Qwen3-8B
            // W3 M = 16 gate|up, 192 -> 384 CTAs: pass 3183 -> 3099 us)
            const int64_t ctas = ceil_div(T, best_nt);
            if (ctas > sms && ctas < 2 * (int64_t)sms && G >= 2) best_cl = 2;
        }
    } else {
        double best_cost = 1e300;
        int64_t best_ctas = INT64_MAX;
        for (int cl = 1; cl <= 8; cl *= 2) {
            if (cl > 1 && cl > G) break;
            for (int nt = 1; nt <= 8; nt *= 2) {
                const int64_t ctas = (int64_t)ceil_div(T, nt) * cl;
                if (ctas > 16 * (int64_t)sms) continue;
                const int64_t gc = (G + cl - 1) / cl;
                const int64_t per_warp = (gc + (8 / nt) - 1) / (8 / nt);
                const int64_t waves = (ctas + 2 * sms - 1) / (2 * sms);
                const double cost = (double)(per_warp + 2) * (double)waves *
                                    (ctas > sms ? 1.3 : 1.0) * (cl > 1 ? 1.02 : 1.0);
                if (cost < best_cost - 1e-9 || (cost < best_cost + 1e-9 && ctas < best_ctas)) {
                    best_cost = cost;
                    best_ctas = ctas;
                    best_nt = nt;
                    best_cl = cl;
                }
            }
        }
        const int64_t gc8 = (G + best_cl - 1) / best_cl;
        const int64_t wt8 = gc8 < 8 / best_nt ? gc8 : 8 / best_nt;
        if (T >= 2 && 2 * T < 3 * (int64_t)sms && (gc8 + wt8 - 1) / wt8 > 5) {
            best_nt = 2;
            best_cl = 1;
            warps_max = 4;
            while (best_cl < 8 && 2 * best_cl <= G &&
                   ((int64_t)best_nt * ((G + best_cl - 1) / best_cl) > 5 * warps_max ||
                    (int64_t)ceil_div(T, best_nt) * best_cl < sms))
                best_cl *= 2;
        }
    }
    shape(G, rec, best_nt, best_cl, warps_max, out);
    const int full = out->stages;
    if (M <= 4 || out->warps <= 8) fit_two_ctas(M, K, N, bits, sms, out);
    // M = 3, 4: where two 4-tile CTAs share an SM only with a shallower ring, 8 tiles per CTA
    // over twice the cluster halve each CTA's X instead (measured on GB300, W4 M = 4 fused
    // Qwen3-4B pass, gate|up: 942 -> 921 us)
    if (batch && M > 2 && M <= 4 && best_nt == 4 && out->stages < full && 2 * best_cl <= 8 &&
        2 * best_cl <= G) {
        laq_gemm_config alt;
        shape(G, rec, 8, 2 * best_cl, warps_max, &alt);
        const int alt_full = alt.stages;
        fit_two_ctas(M, K, N, bits, sms, &alt);
        if (alt.stages == alt_full) *out = alt;
    }
}

laq_status run_gemm(const void* X, int64_t M, int64_t K, int64_t N, const void* packed,
                    const void* s, const uint8_t* z, int bits, void* Y,
                    const laq_gemm_config* cfg, void* stream,
                    const laq_gemm_prologue* pro = nullptr) {
    laq_status st = check_gemm_args(X, M, K, N, packed, s, z, bits, Y);
    if (st != LAQ_OK) return st;
    const int kind = pro ? pro->kind : LAQ_PROLOGUE_NONE;
    if (kind != LAQ_PROLOGUE_NONE && kind != LAQ_PROLOGUE_RMSNORM && kind != LAQ_PROLOGUE_SILU_MUL)
        return LAQ_ERR_CONFIG;
    if (kind == LAQ_PROLOGUE_RMSNORM) {
        if (!pro->w) return LAQ_ERR_NULL;
        if (!(pro->eps >= 0.f)) return LAQ_ERR_SHAPE;
        if (pro->R_out && (pro->R_out == X || pro->R_out == pro->R)) return LAQ_ERR_SHAPE;
        if (((uintptr_t)pro->w & 15u) || ((uintptr_t)pro->R & 15u) ||
            ((uintptr_t)pro->R_out & 15u))
            return LAQ_ERR_ALIGN;
    }
    if (kind != LAQ_PROLOGUE_NONE && ((uintptr_t)X & 15u)) return LAQ_ERR_ALIGN;
    if (cfg) {
        st = check_config(cfg);
        if (st != LAQ_OK) return st;
        if (cfg->warps > 8 && M < 3) return LAQ_ERR_CONFIG;  // 16-warp CTAs from M = 3
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
    L.pro = kind == LAQ_PROLOGUE_RMSNORM ? laq::kProRmsNorm
            : kind == LAQ_PROLOGUE_SILU_MUL ? laq::kProSiluMul : laq::kProNone;
    if (kind == LAQ_PROLOGUE_RMSNORM) {
        L.eps = pro->eps;
        L.R = static_cast<const uint16_t*>(pro->R);
        L.R_out = static_cast<uint16_t*>(pro->R_out);
        L.w = static_cast<const uint16_t*>(pro->w);
    }
    return from_cuda(laq::launch_gemm(L, f.smem_optin, strm));
}


// ---- laq_gemm_chain -------------------------------------------------------------------------

constexpr int kChainMaxM = 4;

size_t chain_ws_bytes(int32_t count) {
    return (laq::chain_workspace_bytes(count) + 255) / 256 * 256;
}

laq_status static_scratch(void** out, size_t* bytes);

// With use_static, the workspace is the library's static scratch (laq_gemm_chain_static): its
// address is looked up, and the counters and flags it must start with at zero are cleared on
// the stream, only once every argument has passed its checks, just before the launch.
laq_status run_chain(const laq_gemv* g, int32_t count, void* workspace, size_t workspace_bytes,
                     void* stream, bool use_static = false) {
    if (count < 0 || count > LAQ_CHAIN_MAX) return LAQ_ERR_SHAPE;
    if (count == 0) return LAQ_OK;
    if (!g) return LAQ_ERR_NULL;
    if (!use_static &&
        (!workspace || !aligned(workspace, 16) || workspace_bytes < chain_ws_bytes(count)))
        return LAQ_ERR_WORKSPACE;
    const int bits = g[0].bits;
    laq_status st = check_bits(bits);
    if (st != LAQ_OK) return st;
    const int64_t M = g[0].M;
    if (M < 1 || M > kChainMaxM) return LAQ_ERR_M_RANGE;
    std::vector<laq::ChainEntry> ents((size_t)count);
    std::vector<laq::ChainStage> stages((size_t)count);
    int nst = 0;
    int64_t xs_need = 0, stage_x = 0, stage_records = 0;
    for (int32_t i = 0; i < count; ++i) {
        const laq_gemv& e = g[i];
        if (e.bits != bits) return LAQ_ERR_BITS;
        if (e.M != M) return LAQ_ERR_M_RANGE;
        st = check_kn(e.K, e.N, true);
        if (st != LAQ_OK) return st;
        if (e.K == 0 || e.N == 0) return LAQ_ERR_SHAPE;
        if (e.K * M * 2 > (int64_t)1 << 30 || e.N / 16 > (int64_t)1 << 24) return LAQ_ERR_SHAPE;
        if (!e.X || !e.packed || !e.s || !e.z || !e.Y) return LAQ_ERR_NULL;
        if (!aligned(e.X, 16) || !aligned(e.packed, 16) || !aligned(e.s, 16) ||
            !aligned(e.z, 16) || !aligned(e.Y, 16))
            return LAQ_ERR_ALIGN;
        if (i == 0 || e.wait_prev != 0) {
            if (i > 0) stages[nst - 1].records = (int)stage_records;
            stages[nst] = laq::ChainStage{i, 0, 0, 0};
            ++nst;
            stage_x = 0;
            stage_records = 0;
        }
        laq::ChainStage& cs = stages[nst - 1];
        laq::ChainEntry& ce = ents[i];
        ce.X = static_cast<const uint16_t*>(e.X);
        ce.packed = static_cast<const uint8_t*>(e.packed);
        ce.s = static_cast<const uint16_t*>(e.s);
        ce.z = e.z;
        ce.Y = static_cast<uint16_t*>(e.Y);
        ce.K = (int)e.K;
        ce.N = (int)e.N;
        ce.xoff = (int)(stage_x / 16);
        ce.psoff = (int)(stage_x / 256);  // one (S, P) pair per 128 fp16 of X
        stage_x += M * e.K * 2;
        stage_records += (e.N / 16) * (e.K / 128);  // records
        if (stage_records > ((int64_t)1 << 26)) return LAQ_ERR_SHAPE;
        ++cs.ne;
        if (stage_x > xs_need) xs_need = stage_x;
    }
    stages[nst - 1].records = (int)stage_records;

    if (use_static) {
        st = static_scratch(&workspace, &workspace_bytes);
        if (st != LAQ_OK) return st;
        if (workspace_bytes < chain_ws_bytes(count)) return LAQ_ERR_WORKSPACE;
    }
    DeviceFacts f;
    st = device_facts(&f);
    if (st != LAQ_OK) return st;
    if (f.sms > 256) return LAQ_ERR_SHAPE;  // one published part per CTA in the workspace
    // Split a stage's tiles across CTAs (record shares, with a cross-CTA fix-up of the tiles
    // that straddle two CTAs, about 1.5 us) only where whole-tile shares leave the busiest CTA
    // far above the mean: at least 48 records (3 per warp) more.
    for (int k = 0; k < nst; ++k) {
        laq::ChainStage& cs = stages[k];
        int64_t units = 0, maxrec = 0;
        for (int q = 0; q < cs.ne; ++q) units += ents[cs.e0 + q].N / 16;
        for (int b = 0; b < f.sms; ++b) {
            // records of CTA b under whole-tile shares
            const int64_t u0 = units * b / f.sms, u1 = units * (b + 1) / f.sms;
            int64_t rec = 0, ubase = 0;
            for (int q = 0; q < cs.ne; ++q) {
                const int64_t T = ents[cs.e0 + q].N / 16, G = ents[cs.e0 + q].K / 128;
                const int64_t lo = u0 > ubase ? u0 : ubase;
                const int64_t hi = u1 < ubase + T ? u1 : ubase + T;
                if (hi > lo) rec += (hi - lo) * G;
                ubase += T;
            }
            if (rec > maxrec) maxrec = rec;
        }
        const int64_t even = (cs.records + f.sms - 1) / f.sms;
        cs.split = maxrec - even >= 48 ? 1 : 0;
    }
    if (laq::chain_smem_bytes(bits, (int)M, (int)xs_need, nst, count) > f.smem_optin)
        return LAQ_ERR_SHAPE;  // the stage's X does not fit beside the weight ring

    laq::ChainLaunch L;
    L.e = ents.data();
    L.st = stages.data();
    L.count = count;
    L.nstages = nst;
    L.M = (int)M;
    L.bits = bits;
    L.xs_bytes = (int)xs_need;
    L.ws = static_cast<uint32_t*>(workspace);
    if (use_static && cudaMemsetAsync(workspace, 0, laq::chain_workspace_zeroed_bytes(count),
                                      static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return LAQ_ERR_CUDA;
    return from_cuda(laq::launch_chain(L, f.sms, static_cast<cudaStream_t>(stream)));
}


// ---- laq_gemm_chain_static: the chain with library-owned scratch ----------------------------

// The chain's workspace for calls that pass none: status, finished CTAs, one arrival counter
// per stage and one flag and published partial tile per CTA, for up to LAQ_CHAIN_MAX entries
// and 256 CTAs (68,352 bytes).  Every GPU that loads the library keeps it until the process
// exits.
constexpr size_t kStaticScratchBytes = 68352;
static __device__ __align__(256) uint32_t g_chain_scratch[kStaticScratchBytes / 4];

// Device address of g_chain_scratch per device (the array's name is only a host-side stand-in
// for it), looked up with the device current on the first call in each CUDA context: after
// cudaDeviceReset the device's next context holds the array at another address, so the cached
// address is tied to the unique id of the context it was looked up in.
struct ScratchAddr {
    unsigned long long ctx_id;
    void* ptr;
};
ScratchAddr g_scratch_addr[kMaxDevices];
std::mutex g_scratch_mu;

// The unique id of the calling thread's current context.  The two driver calls are reached
// through the runtime's entry-point query, so the library does not link the driver library
// itself (it still loads where no driver is installed, for its host-only entry points).
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

laq_status current_ctx_id(unsigned long long* id) {
    static CtxGetCurrentFn get_current = nullptr;
    static CtxGetIdFn get_id = nullptr;
    if (!get_current || !get_id) {
        void* f0 = nullptr;
        void* f1 = nullptr;
        cudaDriverEntryPointQueryResult q0, q1;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f0, 12000, cudaEnableDefault,
                                             &q0) != cudaSuccess ||
            q0 != cudaDriverEntryPointSuccess ||
            cudaGetDriverEntryPointByVersion("cuCtxGetId", &f1, 12000, cudaEnableDefault,
                                             &q1) != cudaSuccess ||
            q1 != cudaDriverEntryPointSuccess || !f0 || !f1)
            return LAQ_ERR_CUDA;
        get_current = reinterpret_cast<CtxGetCurrentFn>(f0);
        get_id = reinterpret_cast<CtxGetIdFn>(f1);
    }
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return LAQ_ERR_CUDA;
    return get_id(ctx, id) == CUDA_SUCCESS ? LAQ_OK : LAQ_ERR_CUDA;
}

laq_status static_scratch(void** out, size_t* bytes) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return LAQ_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return LAQ_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    unsigned long long id = 0;
    const bool have_ctx = current_ctx_id(&id) == LAQ_OK;  // none yet: the lookup makes one
    ScratchAddr& a = g_scratch_addr[dev];
    if (!have_ctx || !a.ptr || a.ctx_id != id) {
        void* ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_chain_scratch) != cudaSuccess || !ptr)
            return LAQ_ERR_CUDA;
        if (current_ctx_id(&id) != LAQ_OK) return LAQ_ERR_CUDA;
        a.ptr = ptr;
        a.ctx_id = id;
    }
    *out = a.ptr;
    *bytes = kStaticScratchBytes;
    return LAQ_OK;
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
        case LAQ_ERR_M_RANGE: return "LAQ_ERR_M_RANGE: M outside the supported range";
        case LAQ_ERR_CUDA: return "LAQ_ERR_CUDA: CUDA runtime error";
        case LAQ_ERR_TIMEOUT: return "LAQ_ERR_TIMEOUT: a device-side wait gave up";
        case LAQ_ERR_CONFIG: return "LAQ_ERR_CONFIG: unsupported launch configuration";
        case LAQ_ERR_WORKSPACE: return "LAQ_ERR_WORKSPACE: workspace missing, misaligned or too small";
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

laq_status laq_gemm_wxg128_prologue(const void* X, int64_t M, int64_t K, int64_t N,
                                    const void* packed, const void* s, const uint8_t* z, int bits,
                                    void* Y, const laq_gemm_prologue* pro,
                                    const laq_gemm_config* cfg, void* stream) {
    return run_gemm(X, M, K, N, packed, s, z, bits, Y, cfg, stream, pro);
}

size_t laq_chain_workspace_bytes(int32_t count) {
    if (count < 0 || count > LAQ_CHAIN_MAX) return 0;
    return chain_ws_bytes(count);
}

laq_status laq_gemm_chain(const laq_gemv* gemvs, int32_t count, void* workspace,
                          size_t workspace_bytes, void* stream) {
    return run_chain(gemvs, count, workspace, workspace_bytes, stream);
}

laq_status laq_gemm_chain_static(const laq_gemv* gemvs, int32_t count, void* stream) {
    if (count > LAQ_CHAIN_MAX) return LAQ_ERR_WORKSPACE;  // beyond the scratch
    // Counters and flags must start at zero (a previous call that gave up may have left them
    // set; the published parts need no clearing): run_chain clears them only once every
    // argument has passed its checks, right before the launch.
    return run_chain(gemvs, count, nullptr, 0, stream, true);
}

}  // extern "C"
