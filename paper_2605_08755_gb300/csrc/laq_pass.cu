// laq_pass.cu -- the decode-step weight pass (Sec. 5.2, "Inference": every projection's
// weights streamed once per token) as a planned persistent launch over per-SM weight streams.
//
// laq_gemm_chain runs the same chain of WbG128 GEMVs (Eq. (1) weights) in one launch, but each
// of its warps walks the packed weights, scales and zeros of its shares itself (a cursor over
// entries, tiles and groups, and three source arrays per record).  Here that walk happens once,
// on the host, when the chain is planned:
//
//  * Plan (host only).  The chain is cut into stages at the entries that wait for their
//    predecessors.  Each stage's 16-column tiles are dealt in order, as whole tiles, to shares
//    balanced by records (tile x group of 128 rows), and the shares rotated over the SMs from
//    stage to stage, so no output tile is split between SMs, no cross-SM reduction sits on the
//    critical path, and every SM streams an equal part of the pass.  An SM's records of a stage are cut into
//    16 contiguous warp shares that differ by at most one record.  The SM's records, all
//    stages in order, form its stream, laid out in rounds: round r holds the r-th record of
//    every warp that has one, warp w's at position w.
//
//  * Prepare (once).  A gather kernel writes every SM's stream into one device buffer: each
//    record's packed codes followed by its 16 scales and 16 zeros (as pairs of output rows
//    r, r + 8, the two rows one lane of the MMA holds), so an SM's whole pass is one contiguous
//    byte range.
//
//  * Run.  One cooperative CTA per SM: 16 consumer warps and one producer warp.  The producer
//    copies the SM's stream round by round with cp.async.bulk into a ring of shared-memory
//    slots (one mbarrier pair per slot), with no knowledge of stages: weights never depend on
//    activations, so the ring runs ahead across stage boundaries while the consumers wait for
//    a stage's input.  Per stage the consumers wait for every SM to have finished the previous
//    stage (a release flag per CTA in the workspace: the stages it has completed), stage the
//    stage's X in shared memory with the group sums S_g = sum_k x_k and P_g = sum_k c_k x_k,
//    take their records from the ring (one per round and warp), and reduce their partial tiles
//    in warp order (deterministic, no atomics on Y).
//
//  * The record arithmetic is that of laq_gemm_wxg128 at M = 1: one mask-and-or per pair of
//    codes gives fp16 values c + q, the m16n8k16 MMA contracts them with raw x, the eight groups
//    of a block share one accumulator (one MMA column each), and the block epilogue applies
//    Eq. (1) as y += s * (D - P - z S).
//
//  * Every wait is bounded (about a second): a timed-out wait records LAQ_ERR_TIMEOUT in the
//    workspace, the CTA's warps leave together (barrier reductions decide it), the producer
//    first waits for its copies in flight, and the call's results are undefined.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <climits>
#include <cstring>
#include <vector>

#include "laq.h"
#include "laq_device.cuh"

namespace laq {
namespace {

constexpr uint32_t kPassMagic = 0x5051414cu;  // "LAQP"
constexpr int32_t kPassVersion = 1;
constexpr int kPW = 16;                        // consumer warps
constexpr int kPThreads = (kPW + 1) * 32;      // and the producer warp
constexpr int kPRec = 16;                      // records per round (one per consumer warp)
constexpr int kSZ = 48;                        // a record's 16 fp16 scales and 16 uint8 zeros
constexpr int kMaxSegs = 255;                  // warp segments per (SM, stage)
constexpr int kMaxXsBytes = 104 * 1024;        // staged X per (SM, stage), all M rows
constexpr int kMaxM = 4;                       // batch rows
constexpr int kMaxRing = 16;                   // ring slots
// Rounds a producer keeps in flight.  About four rounds per SM (50-70 KB, 8-10 MB over the GPU)
// already sustain the full HBM rate; many more queue so deep in the memory system that the
// latency-critical loads of a stage change (the completed-stage flags, the stage's X) wait
// behind them: with the whole ring refilled at once after a large stage, a single flag poll
// took 5 us.
constexpr int kInflight = 4;
// Stages the producer may run ahead of the consumers: it copies the rounds of stage s only once
// the consumers have seen stage s - kLead's dependency met.  Copies issued while the stages hand
// over (every SM's release store, the flag polls and the next stage's X loads) queue those
// latency-critical accesses behind HBM reads: after a large stage, with every SM refilling its
// ring at once, the 152 release stores took up to 5 us to become visible.
constexpr int kLead = 1;
constexpr int kMaxSms = 1024;
constexpr unsigned long long kWaitNs = 1000000000ull;  // wait limit (1 s)
constexpr int kWaitSpins = 1 << 24;                    // and an iteration limit besides

// ---- plan tables: the same bytes in the host plan and in the device buffer -------------------

struct SmDesc {        // one per SM
    int64_t rec0;      // the SM's first record in the stream buffer (records, all of rb bytes)
    int32_t round0;    // its first entry of the round table
    int32_t nrounds;
};
struct StageDesc {     // one per (SM, stage), SM-major
    int32_t n;         // records of the SM in the stage
    int32_t nr;        // rounds: ceil(n / 16)
    int32_t seg0;      // first segment (index into the segment table)
    int32_t tile0;     // first local tile
    int32_t x0;        // first staged X
    int16_t nseg, nt, nx, pad;
    uint8_t wseg[kPW + 1];  // warp w's segments: [seg0 + wseg[w], seg0 + wseg[w + 1])
    uint8_t pad2[3];
};
struct Seg {           // groups [g0, g0 + ng) of tile t of entry e, as one warp runs them
    int32_t e, t;
    int16_t g0, ng;
    int16_t xg;        // the entry's first group in the stage's X area
    int16_t lt;        // local tile (index into the stage's local tiles)
};
struct LTile {         // a tile of the SM's stage share: its 16 outputs, its segments' slots
    uint16_t* y;       // Y + 16 t of its entry (row 0)
    int32_t slot0, nslot;
    int32_t ldy;       // the entry's N: the distance between Y rows
    int32_t pad;
};
struct XItem {         // one entry's X staged for the SM's stage share
    const uint16_t* x;
    int32_t K;
    int32_t xg;        // first group in the X area (a group is 256 bytes of X)
};
struct PrepEntry {     // what the gather kernel reads of an entry
    const uint8_t* packed;
    const uint16_t* s;
    const uint8_t* z;
    int32_t N, G;
};
struct GatherRec {     // stream record i is record rid = t * G + g of entry e
    int32_t e, rid;
};
static_assert(sizeof(SmDesc) == 16 && sizeof(StageDesc) == 48 && sizeof(Seg) == 16 &&
                  sizeof(LTile) == 24 && sizeof(XItem) == 16 && sizeof(PrepEntry) == 32 &&
                  sizeof(GatherRec) == 8,
              "plan table layout");

struct PlanHeader {
    uint32_t magic;
    int32_t version;
    int32_t count, nstages, sms, bits;
    int32_t rb;        // stream bytes of a record (packed codes + scales + zeros)
    int32_t M;         // batch rows of every entry
    int32_t xg_row;    // groups of one staged X row: the most any (SM, stage) stages
    int32_t xs_bytes;  // the X area: M rows of xg_row groups (256 bytes each)
    int32_t max_segs;  // most segments of an (SM, stage)
    int32_t max_nx;    // most staged X items of an (SM, stage)
    int64_t records, rounds, segs, ltiles, xitems;
    int64_t tables_h;      // offset of the table region in the plan buffer
    int64_t tables_bytes;  // its size (the same region follows the streams on the device)
    int64_t stream_bytes;  // bytes of the streams at the start of the device buffer
    // offsets of the tables within the table region
    int64_t o_sm, o_rounds, o_stage, o_seg, o_tile, o_x, o_prep, o_gather;
    int64_t plan_bytes, device_bytes;
};
static_assert(sizeof(PlanHeader) <= 256, "plan header");

constexpr int64_t align_up(int64_t v, int64_t a) { return (v + a - 1) / a * a; }

int record_bytes(int bits) { return (bits == 4 ? 1024 : 768) + kSZ; }

// ---- host planner ------------------------------------------------------------------------------

struct HostPlan {
    int count = 0, nstages = 0, sms = 0, bits = 3, M = 1;
    int xg_row = 0, max_segs = 0, max_nx = 0;
    std::vector<SmDesc> sm;
    std::vector<uint8_t> rounds;
    std::vector<StageDesc> stage;
    std::vector<Seg> seg;
    std::vector<LTile> tile;
    std::vector<XItem> xi;
    std::vector<PrepEntry> prep;
    std::vector<GatherRec> gather;
};

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

laq_status plan_pass(const laq_gemv* g, int32_t count, int32_t P, HostPlan& H) {
    if (count < 0 || count > LAQ_CHAIN_MAX) return LAQ_ERR_SHAPE;
    if (P < 1 || P > kMaxSms) return LAQ_ERR_SHAPE;
    if (count > 0 && !g) return LAQ_ERR_NULL;
    H = HostPlan();
    H.count = count;
    H.sms = P;
    std::vector<int> start;  // first entry of each stage
    for (int i = 0; i < count; ++i) {
        const laq_gemv& e = g[i];
        if (e.bits != 3 && e.bits != 4) return LAQ_ERR_BITS;
        if (i == 0) H.bits = e.bits;
        if (e.bits != H.bits) return LAQ_ERR_BITS;
        if (e.M < 1 || e.M > kMaxM) return LAQ_ERR_M_RANGE;
        if (i == 0) H.M = (int)e.M;
        if (e.M != H.M) return LAQ_ERR_M_RANGE;
        if (e.K <= 0 || e.N <= 0 || e.K % 128 != 0 || e.N % 16 != 0) return LAQ_ERR_SHAPE;
        if (e.K * 2 * e.M > kMaxXsBytes || e.N / 16 > ((int64_t)1 << 24)) return LAQ_ERR_SHAPE;
        // a record's id t * G + g (GatherRec::rid) is a 32-bit int
        if ((e.N / 16) * (e.K / 128) > (int64_t)INT_MAX) return LAQ_ERR_SHAPE;
        if (!e.X || !e.packed || !e.s || !e.z || !e.Y) return LAQ_ERR_NULL;
        if (!aligned16(e.X) || !aligned16(e.packed) || !aligned16(e.s) || !aligned16(e.z) ||
            !aligned16(e.Y))
            return LAQ_ERR_ALIGN;
        if (i == 0 || e.wait_prev != 0) start.push_back(i);
        H.prep.push_back(PrepEntry{static_cast<const uint8_t*>(e.packed),
                                   static_cast<const uint16_t*>(e.s), e.z, (int32_t)e.N,
                                   (int32_t)(e.K / 128)});
    }
    const int S = (int)start.size();
    H.nstages = S;
    start.push_back(count);

    // Whole tiles to shares, in order: a tile goes to the share whose equal part of the stage's
    // records holds the tile's middle record, so shares are contiguous tile ranges and differ
    // from the mean by less than one tile.  first[s][v] = share v's first stage tile.  SM j
    // takes share (j + 41 s) mod P of stage s: the shares that hold one tile more than the
    // others fall on other SMs from stage to stage, so no SM streams more than its part of the
    // whole pass.
    std::vector<std::vector<int64_t>> first(S);
    for (int s = 0; s < S; ++s) {
        int64_t tiles = 0, W = 0;
        for (int e = start[s]; e < start[s + 1]; ++e) {
            tiles += g[e].N / 16;
            W += (g[e].N / 16) * (g[e].K / 128);
        }
        std::vector<int64_t>& f = first[s];
        f.assign((size_t)P + 1, tiles);
        int64_t c = 0, tix = 0;
        int jp = -1;
        for (int e = start[s]; e < start[s + 1]; ++e) {
            const int64_t T = g[e].N / 16, G = g[e].K / 128;
            for (int64_t t = 0; t < T; ++t, ++tix, c += G) {
                int64_t j = (2 * c + G) * P / (2 * W);
                if (j > P - 1) j = P - 1;
                while (jp < j) f[(size_t)(++jp)] = tix;
            }
        }
        while (jp < P) f[(size_t)(++jp)] = tiles;
    }

    struct TileRef {
        int e;
        int64_t t;
        int G;
    };
    for (int j = 0; j < P; ++j) {
        SmDesc sd;
        sd.rec0 = (int64_t)H.gather.size();
        sd.round0 = (int32_t)H.rounds.size();
        for (int s = 0; s < S; ++s) {
            // the SM's tiles of the stage
            std::vector<TileRef> tl;
            {
                const size_t v = (size_t)(((int64_t)j + 41 * (int64_t)s) % P);
                int64_t ta = first[s][v], tb = first[s][v + 1], base = 0;
                for (int e = start[s]; e < start[s + 1] && ta < tb; ++e) {
                    const int64_t T = g[e].N / 16;
                    for (; ta < tb && ta < base + T; ++ta)
                        tl.push_back(TileRef{e, ta - base, (int)(g[e].K / 128)});
                    base += T;
                }
            }
            StageDesc d;
            std::memset(&d, 0, sizeof(d));
            d.seg0 = (int32_t)H.seg.size();
            d.tile0 = (int32_t)H.tile.size();
            d.x0 = (int32_t)H.xi.size();
            int64_t n = 0;
            for (const TileRef& r : tl) n += r.G;
            if (n > INT_MAX / 2) return LAQ_ERR_SHAPE;
            d.n = (int32_t)n;
            d.nr = (int32_t)((n + kPRec - 1) / kPRec);
            if (n == 0) {
                H.stage.push_back(d);
                continue;
            }
            if ((int64_t)tl.size() > kMaxSegs) return LAQ_ERR_SHAPE;
            // X of every entry the share touches, one after another, whole groups
            std::vector<int> xg_of(tl.size());
            int xg = 0, last_e = -1;
            for (size_t k = 0; k < tl.size(); ++k) {
                if (tl[k].e != last_e) {
                    last_e = tl[k].e;
                    H.xi.push_back(XItem{static_cast<const uint16_t*>(g[last_e].X),
                                         (int32_t)g[last_e].K, (int32_t)xg});
                    xg += (int)(g[last_e].K / 128);
                    ++d.nx;
                }
                xg_of[k] = H.xi.back().xg;
            }
            if ((int64_t)xg * 256 * H.M > kMaxXsBytes) return LAQ_ERR_SHAPE;
            if (xg > H.xg_row) H.xg_row = xg;
            if (d.nx > H.max_nx) H.max_nx = d.nx;
            // record offset of each local tile
            std::vector<int64_t> toff(tl.size() + 1, 0);
            for (size_t k = 0; k < tl.size(); ++k) toff[k + 1] = toff[k] + tl[k].G;
            // warp shares and their segments
            const int64_t q = n / kPW, rem = n % kPW;
            size_t lt = 0;
            int nseg = 0;
            for (int w = 0; w < kPW; ++w) {
                int64_t a = w * q + (w < rem ? w : rem);
                const int64_t b = a + q + (w < rem ? 1 : 0);
                if (nseg > kMaxSegs) return LAQ_ERR_SHAPE;
                d.wseg[w] = (uint8_t)nseg;
                while (a < b) {
                    while (toff[lt + 1] <= a) ++lt;
                    const int64_t end = b < toff[lt + 1] ? b : toff[lt + 1];
                    H.seg.push_back(Seg{tl[lt].e, (int32_t)tl[lt].t, (int16_t)(a - toff[lt]),
                                        (int16_t)(end - a), (int16_t)xg_of[lt], (int16_t)lt});
                    ++nseg;
                    a = end;
                }
            }
            if (nseg > kMaxSegs) return LAQ_ERR_SHAPE;
            d.wseg[kPW] = (uint8_t)nseg;
            d.nseg = (int16_t)nseg;
            d.nt = (int16_t)tl.size();
            if (nseg > H.max_segs) H.max_segs = nseg;
            // local tiles: the consecutive segments that cover each
            for (size_t k = 0; k < tl.size(); ++k) {
                LTile t;
                t.y = static_cast<uint16_t*>(g[tl[k].e].Y) + tl[k].t * 16;
                t.slot0 = -1;
                t.nslot = 0;
                t.ldy = (int32_t)g[tl[k].e].N;
                t.pad = 0;
                H.tile.push_back(t);
            }
            for (int k = 0; k < nseg; ++k) {
                LTile& t = H.tile[(size_t)d.tile0 + (size_t)H.seg[(size_t)d.seg0 + k].lt];
                if (t.slot0 < 0) t.slot0 = k;
                ++t.nslot;
            }
            // rounds, and the stream records in round order
            int cur_k[kPW], cur_i[kPW];
            for (int w = 0; w < kPW; ++w) {
                cur_k[w] = d.wseg[w];
                cur_i[w] = 0;
            }
            for (int64_t r = 0; r < d.nr; ++r) {
                const int cnt = r < q ? kPRec : (int)rem;
                H.rounds.push_back((uint8_t)cnt);
                for (int w = 0; w < cnt; ++w) {
                    const Seg& sg = H.seg[(size_t)d.seg0 + cur_k[w]];
                    const int64_t G = g[sg.e].K / 128;
                    H.gather.push_back(GatherRec{sg.e, (int32_t)(sg.t * G + sg.g0 + cur_i[w])});
                    if (++cur_i[w] == sg.ng) {
                        ++cur_k[w];
                        cur_i[w] = 0;
                    }
                }
            }
            H.stage.push_back(d);
        }
        const int64_t nr = (int64_t)H.rounds.size() - sd.round0;
        if ((int64_t)H.rounds.size() > INT_MAX / 2) return LAQ_ERR_SHAPE;
        sd.nrounds = (int32_t)nr;
        H.sm.push_back(sd);
    }
    return LAQ_OK;
}

// Layout of the serialized plan and of the device buffer.
void layout(const HostPlan& H, PlanHeader& h) {
    std::memset(&h, 0, sizeof(h));
    h.magic = kPassMagic;
    h.version = kPassVersion;
    h.count = H.count;
    h.nstages = H.nstages;
    h.sms = H.sms;
    h.bits = H.bits;
    h.rb = record_bytes(H.bits);
    h.M = H.M;
    h.xg_row = H.xg_row;
    h.xs_bytes = H.xg_row * 256 * H.M;
    h.max_segs = H.max_segs;
    h.max_nx = H.max_nx;
    h.records = (int64_t)H.gather.size();
    h.rounds = (int64_t)H.rounds.size();
    h.segs = (int64_t)H.seg.size();
    h.ltiles = (int64_t)H.tile.size();
    h.xitems = (int64_t)H.xi.size();
    int64_t o = 0;
    h.o_sm = o;      o = align_up(o + (int64_t)H.sm.size() * (int64_t)sizeof(SmDesc), 256);
    h.o_rounds = o;  o = align_up(o + (int64_t)H.rounds.size(), 256);
    h.o_stage = o;   o = align_up(o + (int64_t)H.stage.size() * (int64_t)sizeof(StageDesc), 256);
    h.o_seg = o;     o = align_up(o + (int64_t)H.seg.size() * (int64_t)sizeof(Seg), 256);
    h.o_tile = o;    o = align_up(o + (int64_t)H.tile.size() * (int64_t)sizeof(LTile), 256);
    h.o_x = o;       o = align_up(o + (int64_t)H.xi.size() * (int64_t)sizeof(XItem), 256);
    h.o_prep = o;    o = align_up(o + (int64_t)H.prep.size() * (int64_t)sizeof(PrepEntry), 256);
    h.o_gather = o;  o = align_up(o + (int64_t)H.gather.size() * (int64_t)sizeof(GatherRec), 256);
    h.tables_bytes = o;
    h.tables_h = align_up(256 + (int64_t)H.count * (int64_t)sizeof(laq_gemv), 256);
    h.plan_bytes = h.tables_h + h.tables_bytes;
    h.stream_bytes = align_up(h.records * h.rb, 256);
    h.device_bytes = h.stream_bytes + h.tables_bytes;
}

template <class T>
void put(uint8_t* region, int64_t off, const std::vector<T>& v) {
    if (!v.empty()) std::memcpy(region + off, v.data(), v.size() * sizeof(T));
}

// A plan buffer from laq_pass_plan_build, or nullptr.
const PlanHeader* as_plan(const void* plan) {
    if (!plan) return nullptr;
    const PlanHeader* h = static_cast<const PlanHeader*>(plan);
    if (h->magic != kPassMagic || h->version != kPassVersion) return nullptr;
    if (h->sms < 1 || h->sms > kMaxSms || h->nstages < 0 || h->nstages > LAQ_CHAIN_MAX ||
        (h->bits != 3 && h->bits != 4) || h->rb != record_bytes(h->bits) ||
        h->M < 1 || h->M > kMaxM || h->xg_row < 0 || h->xs_bytes != h->xg_row * 256 * h->M ||
        h->xs_bytes > kMaxXsBytes || h->max_segs < 0 ||
        h->max_segs > kMaxSegs || h->max_nx < 0 || h->max_nx > kMaxSegs)
        return nullptr;
    return h;
}

// Workspace: uint32 [0] status, [1] finished CTAs; then kCounters stage counters, each in a
// 128-byte line of its own: every CTA adds 1 to counter s % kCounters when it has completed
// stage s, so stage s is complete once that counter reaches P (s / kCounters + 1).  (Measured on
// GB300 with all 152 CTAs arriving at once: the last arrival is seen 0.96 us later, against
// 2.1 us for per-CTA 16-bit flags packed into three lines and 1.5 us for per-CTA flags in lines
// of their own: many writers into the lines every CTA polls are what costs.)
constexpr int kCounters = 8;
constexpr int kCounterStride = 32;  // uint32 words: one 128-byte line
size_t pass_workspace(const PlanHeader&) {
    return (size_t)align_up(4 * kCounterStride * (1 + kCounters), 256);
}

// ---- shared memory layout of the pass kernel (host and device) -------------------------------

struct PassSmem {
    int xs, sp, seg, tile, xi, slot, zero, bar, flag, total;
};
// Regions: the ring (ns slots of 16 records), the X area (xs_bytes) and its (S, P) pair per
// group, the stage's segments, local tiles and staged X items, the segment partials (mp rows of
// 16 outputs per segment), a zero block, the ring's mbarriers and the abort flag.
__host__ __device__ inline PassSmem pass_smem(int rb, int ns, int xs_bytes, int max_segs,
                                              int max_nx, int mp) {
    auto a16 = [](int v) { return (v + 15) / 16 * 16; };
    PassSmem m;
    m.xs = (ns * kPRec * rb + 127) / 128 * 128;
    m.sp = m.xs + xs_bytes;
    m.seg = a16(m.sp + xs_bytes / 256 * 8);
    m.tile = a16(m.seg + max_segs * (int)sizeof(Seg));
    m.xi = a16(m.tile + max_segs * (int)sizeof(LTile));
    m.slot = a16(m.xi + max_nx * (int)sizeof(XItem));
    m.zero = a16(m.slot + max_segs * mp * 16 * 4);
    m.bar = m.zero + 64;
    m.flag = m.bar + 2 * kMaxRing * 8;
    m.total = m.flag + 16;
    return m;
}

// ---- device helpers ----------------------------------------------------------------------------

__device__ __forceinline__ unsigned long long gtimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ uint32_t ld_acq(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint32_t ld_rlx(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void red_rel_add(uint32_t* p, uint32_t v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t atom_acq_rel_add(uint32_t* p, uint32_t v) {
    uint32_t old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;"
                 : "=r"(old)
                 : "l"(p), "r"(v)
                 : "memory");
    return old;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n"
        ".reg .pred p;\n"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        "selp.u32 %0, 1, 0, p;\n"
        "}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0u;
}
// An L2 policy that evicts first what it tags: the weight stream is read exactly once per pass,
// so it should not push X, Y and the plan's tables out of L2.
__device__ __forceinline__ uint64_t evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
// Copy `bytes` (a multiple of 16) from global memory into this CTA's shared memory under L2
// policy `pol`; the copy counts its bytes against the transaction count of mbarrier `bar`.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint32_t bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;"
        ::"r"(dst), "l"(src), "r"(bytes), "r"(bar), "l"(pol)
        : "memory");
}

// Named barrier of the 16 consumer warps, returning whether any of them passed `v` true (the
// same answer in every thread, so decisions taken on it keep the warps together).
__device__ __forceinline__ bool cbar_any(bool v) {
    uint32_t r;
    asm volatile(
        "{\n"
        ".reg .pred p, q;\n"
        "setp.ne.u32 q, %1, 0;\n"
        "bar.red.or.pred p, 1, 512, q;\n"
        "selp.u32 %0, 1, 0, p;\n"
        "}\n"
        : "=r"(r)
        : "r"((uint32_t)v)
        : "memory");
    return r != 0u;
}
__device__ __forceinline__ void cbar() { asm volatile("bar.sync 1, 512;" ::: "memory"); }

// Record a device-side timeout in the workspace status word (the first error stays).
__device__ __forceinline__ void record_timeout(uint32_t* status) {
    atomicCAS(status, 0u, (uint32_t)LAQ_ERR_TIMEOUT);
}

// Wait for phase `parity` of mbarrier `bar`.  False when the CTA is aborting (the flag is read
// every 64 polls) or after about a second (then the flag and the status word are set).
__device__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                          uint32_t* status) {
    if (mbar_try(bar, parity)) return true;
    const unsigned long long t0 = gtimer();
    for (int spin = 0; spin < kWaitSpins; ++spin) {
        if (mbar_try(bar, parity)) return true;
        if ((spin & 63) == 63) {
            if (abort_flag && *abort_flag) return false;
            if (gtimer() - t0 > kWaitNs) break;
        }
    }
    if (abort_flag) {
        *abort_flag = 1;
        record_timeout(status);
    }
    return false;
}

// One warp waits until stage `stage` is complete: its counter has reached the number of CTAs
// times the count of stages so far that share the counter.  Lane 0 polls with acquire loads;
// the answer is warp-wide: false when the status word holds an error (checked every 16th poll),
// or after about a second (then LAQ_ERR_TIMEOUT is recorded).
__device__ bool wait_stage_done(const uint32_t* ws, int stage, uint32_t ctas, uint32_t* status,
                                int lane) {
    const uint32_t* cnt = ws + kCounterStride * (1 + stage % kCounters);
    const uint32_t target = ctas * (uint32_t)(stage / kCounters + 1);
    const unsigned long long t0 = gtimer();
    for (int spin = 0; spin < kWaitSpins; ++spin) {
        const int ok = lane == 0 ? (int)(ld_acq(cnt) >= target) : 0;
        if (__shfl_sync(0xffffffffu, ok, 0)) return true;
        if ((spin & 15) == 15) {
            const uint32_t st = lane == 0 ? ld_rlx(status) : 0u;
            if (__shfl_sync(0xffffffffu, st, 0) != 0u) return false;
            const bool late = lane == 0 && gtimer() - t0 > kWaitNs;
            if (__shfl_sync(0xffffffffu, (int)late, 0)) break;
        }
    }
    if (lane == 0) record_timeout(status);
    return false;
}

struct PassParams {
    const uint8_t* stream;
    const SmDesc* sm;
    const uint8_t* rounds;
    const StageDesc* stage;
    const Seg* seg;
    const LTile* tile;
    const XItem* xi;
    uint32_t* ws;  // [0] status, [1] finished CTAs, then the stage counters
    int nstages, ns, xs_bytes, max_segs, max_nx;
    int M;       // batch rows (1..4)
    int xg_row;  // groups of one staged X row
    Exps exps;
};

// ---- the producer warp -------------------------------------------------------------------------

// Lane 0 waits until the consumers have met the dependency of stage `target` (*cur_stage, set by
// the consumers, is at least target); the answer is warp-wide.  False when the CTA aborts or
// after about a second (then the abort flag and LAQ_ERR_TIMEOUT are set).
__device__ bool wait_stage(volatile int* cur_stage, int target, volatile int* abort_flag,
                           uint32_t* status, int lane) {
    int ok = 1;
    if (lane == 0 && *cur_stage < target) {
        ok = 0;
        const unsigned long long t0 = gtimer();
        for (int spin = 0; spin < kWaitSpins; ++spin) {
            if (*cur_stage >= target) {
                ok = 1;
                break;
            }
            if (*abort_flag) break;
            __nanosleep(64);
            if ((spin & 63) == 63 && gtimer() - t0 > kWaitNs) {
                *abort_flag = 1;
                record_timeout(status);
                break;
            }
        }
    }
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

template <int BITS>
__device__ void pass_producer(const PassParams& p, const SmDesc& sd, uint32_t ring_s,
                              uint32_t full_s, uint32_t empty_s, volatile int* abort_flag,
                              volatile int* cur_stage, int lane) {
    constexpr int RB = RecordFmt<BITS>::kBytes + kSZ;
    constexpr uint32_t SLOT = (uint32_t)(kPRec * RB);
    const int NS = p.ns, NR = sd.nrounds;
    const uint8_t* src = p.stream + sd.rec0 * RB;
    const uint8_t* rt = p.rounds + sd.round0;
    const uint64_t pol = evict_first_policy();
    int issued = 0;
    bool ok = true;
    // the stage of round r: rounds [stage_end - nr(stage), stage_end)
    const StageDesc* sdp = p.stage + (size_t)blockIdx.x * p.nstages;
    int stage = -1, stage_end = 0;
    for (int r0 = 0; r0 < NR && ok; r0 += 32) {
        const int mine = r0 + lane < NR ? (int)rt[r0 + lane] : 0;
        const int lim = NR - r0 < 32 ? NR - r0 : 32;
        for (int i = 0; i < lim; ++i) {
            const int cnt = __shfl_sync(0xffffffffu, mine, i);
            const int r = r0 + i, slot = r % NS, k = r / NS;
            if (r == stage_end) {
                do {
                    ++stage;
                    stage_end += sdp[stage].nr;
                } while (r == stage_end);
                // the consumers have met stage (stage - kLead)'s dependency
                if (stage - kLead > 0 && !wait_stage(cur_stage, stage - kLead, abort_flag, p.ws, lane)) {
                    ok = false;
                    break;
                }
            }
            // slot reuse: every consumer warp has released the round that used it last
            if (k > 0 && !__all_sync(0xffffffffu,
                                     mbar_wait(empty_s + 8u * slot, (uint32_t)((k - 1) & 1),
                                               abort_flag, p.ws))) {
                ok = false;
                break;
            }
            // at most kInflight rounds in flight: round r - kInflight has landed
            if (r >= kInflight) {
                const int ro = r - kInflight;
                if (!__all_sync(0xffffffffu, mbar_wait(full_s + 8u * (ro % NS),
                                                       (uint32_t)((ro / NS) & 1), abort_flag,
                                                       p.ws))) {
                    ok = false;
                    break;
                }
            }
            if (lane == 0) {
                const uint32_t bytes = (uint32_t)(cnt * RB);
                mbar_expect_tx(full_s + 8u * slot, bytes);
                bulk_g2s(ring_s + SLOT * (uint32_t)slot, src, bytes, full_s + 8u * slot, pol);
            }
            __syncwarp();
            src += (size_t)cnt * RB;
            issued = r + 1;
        }
    }
    // No copy may still be landing in shared memory when the CTA exits: wait for the last
    // round issued into each slot (immediate when the consumers took every round).
    for (int r = issued > NS ? issued - NS : 0; r < issued; ++r)
        mbar_wait(full_s + 8u * (r % NS), (uint32_t)((r / NS) & 1), nullptr, p.ws);
}

// ---- the consumer warps ------------------------------------------------------------------------

// Stage one entry's X (M rows of K fp16) in the X area, whose rows are xg_row groups apart:
// 16-byte chunk cr of row b lands at xs[16 (b xg_row + xg) + cr]; the 16 lanes holding a
// group's chunks sum S = sum_k x_k and P = sum_k c_k x_k into sp[b xg_row + xg + group].  K / 8
// is a multiple of 16, so the 16 lanes of a group are a half-warp of one row, and a thread's
// chunks all sit at the same position q % 4 of their group (q = tid % 4): chunk q holds pairs
// 4 q + w, w < 4, of the record layout, whose offsets c_k the thread keeps in off[w].
__device__ void pass_stage_x(const XItem& X, int M, int xg_row, uint4* xs, float2* sp, int tid,
                             const float (&off)[4]) {
    const int nch = X.K >> 3;  // chunks per row
    const int total = M * nch;
    for (int c0 = 0; c0 < total; c0 += 4 * 512) {
        uint4 v[4];
        int bb[4], cc[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int ci = c0 + u * 512 + tid;
            const int b = (ci >= nch) + (ci >= 2 * nch) + (ci >= 3 * nch);  // M <= 4 rows
            bb[u] = b;
            cc[u] = ci - b * nch;
            v[u] = ci < total ? ld_cg16(X.x + (size_t)b * X.K + 8 * (size_t)cc[u])
                              : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (c0 + u * 512 + (tid & ~31) >= total) break;  // warp-uniform
            const int ci = c0 + u * 512 + tid;
            const uint32_t w4[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
            float sx = 0.f, px = 0.f;
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w4[w]));
                const float pair = f.x + f.y;
                sx += pair;
                px = fmaf(off[w], pair, px);
            }
#pragma unroll
            for (int o = 1; o < 16; o <<= 1) {
                sx += __shfl_xor_sync(0xffffffffu, sx, o);
                px += __shfl_xor_sync(0xffffffffu, px, o);
            }
            if (ci < total) {
                const int b = bb[u], cr = cc[u];
                xs[16 * (b * xg_row + X.xg) + cr] = v[u];
                if ((cr & 15) == 0) sp[b * xg_row + X.xg + (cr >> 4)] = make_float2(sx, px);
            }
        }
    }
}

// MP: the batch rows M rounded up to 1, 2 or 4.  The MMA's 8 columns hold GPA = 8 / MP groups
// of each of MP batch rows: column col is batch row col / GPA and record col % GPA of a block of
// GPA records (at M = 1 the 8 columns are 8 groups of the one row).

// A position in the ring: the slot of a round and the phase parity of that slot's use.
struct RingPos {
    int slot;
    uint32_t par;
};
__device__ __forceinline__ void ring_next(RingPos& q, int NS) {
    if (++q.slot == NS) {
        q.slot = 0;
        q.par ^= 1u;
    }
}

// Wait for the n rounds from ring position q on (every lane polls; the answer is warp-wide).
// False when the CTA is aborting or a wait gave up.
__device__ __forceinline__ bool wait_rounds(uint32_t full_s, RingPos q, int n, int NS,
                                            volatile int* abort_flag, uint32_t* status) {
    bool ok = true;
    for (int i = 0; i < n && ok; ++i) {
        ok = mbar_wait(full_s + 8u * q.slot, q.par, abort_flag, status);
        ring_next(q, NS);
    }
    return __all_sync(0xffffffffu, ok);
}

// This warp is done with the n rounds from ring position q on: one arrival each on their slots'
// empty barriers (after every lane's reads), and q moves past them.
__device__ __forceinline__ void release_rounds(uint32_t empty_s, RingPos& q, int n, int NS,
                                               int lane) {
    __syncwarp();
    for (int i = 0; i < n; ++i) {
        if (lane == 0) mbar_arrive(empty_s + 8u * q.slot);
        ring_next(q, NS);
    }
}

// One record: its packed codes (this lane's words at rec), the B fragments at xsrc (this lane's
// x values, or the zero block), the mask-and-or extraction and the 8 MMAs of the 8 k16 steps of
// the group, accumulated on four chains (steps j and j + 4 share chain j % 4).
template <int BITS>
__device__ __forceinline__ void pass_record(const uint8_t* rec, const uint4* xsrc,
                                            const Exps& ex, float (&D)[4][4], int lane) {
    constexpr int WPL = BITS == 4 ? 8 : 6;
    uint32_t B[8][2];
#pragma unroll
    for (int qq = 0; qq < 4; ++qq) {
        const uint4 v = xsrc[qq];
        B[2 * qq][0] = v.x;
        B[2 * qq][1] = v.y;
        B[2 * qq + 1][0] = v.z;
        B[2 * qq + 1][1] = v.w;
    }
    uint32_t wd[WPL];
    const uint4 c0 = *reinterpret_cast<const uint4*>(rec + lane * 16);
    wd[0] = c0.x;
    wd[1] = c0.y;
    wd[2] = c0.z;
    wd[3] = c0.w;
    if constexpr (BITS == 4) {
        const uint4 c1 = *reinterpret_cast<const uint4*>(rec + 512 + lane * 16);
        wd[4] = c1.x;
        wd[5] = c1.y;
        wd[6] = c1.z;
        wd[7] = c1.w;
    } else {
        const uint2 c1 = *reinterpret_cast<const uint2*>(rec + 512 + lane * 8);
        wd[4] = c1.x;
        wd[5] = c1.y;
    }
    uint32_t a[8][4];
    extract<BITS>(wd, ex, a);
#pragma unroll
    for (int j = 0; j < 8; ++j)
        mma16816(D[j & 3], a[j][0], a[j][1], a[j][2], a[j][3], B[j][0], B[j][1]);
}

// The block epilogue (Eq. (1)) of a block of len records whose first record is at ring slot
// slot0: accumulator value v of this lane is output row R + 8 (v >> 1) and MMA column
// col = 2c + (v & 1), i.e. batch row col / GPA and block record col % GPA; it adds
// s (D - P - z S) with the record's scale and zero (read from the record's ring slot, which the
// warp still holds) and the group's (S, P) sums (spb: the block's first group, row 0).
template <int BITS, int MP>
__device__ __forceinline__ void pass_epilogue(const uint8_t* ring, int slot0, int NS, int warp,
                                              int lane, int len, int M, int XR,
                                              const float2* spb, const float (&D)[4][4],
                                              float (&y)[4]) {
    constexpr int RBC = RecordFmt<BITS>::kBytes;
    constexpr int RB = RBC + kSZ;
    constexpr int SLOT = kPRec * RB;
    constexpr int GPA = 8 / MP;
    const int c = lane & 3, R = lane >> 2;
#pragma unroll
    for (int h = 0; h < 2; ++h) {  // the lane's two MMA columns
        const int col = 2 * c + h;
        const int b = col / GPA, giv = col % GPA;
        if (giv < len && b < M) {
            int sl = slot0 + giv;
            if (sl >= NS) sl -= NS;
            const uint8_t* sz = ring + (size_t)sl * SLOT + (size_t)warp * RB + RBC;
            const uint32_t sw = reinterpret_cast<const uint32_t*>(sz)[R];   // s of rows R, R + 8
            const uint32_t zw = reinterpret_cast<const uint16_t*>(sz + 32)[R];  // z of R, R + 8
            const float2 spv = spb[b * XR + giv];                             // (S, P)
#pragma unroll
            for (int hi = 0; hi < 2; ++hi) {
                const int v = 2 * hi + h;
                const float dv = (D[0][v] + D[1][v]) + (D[2][v] + D[3][v]);
                const float sc = __half2float(__ushort_as_half((uint16_t)(sw >> (16 * hi))));
                const float zc = (float)((zw >> (8 * hi)) & 0xffu);
                y[v] = fmaf(sc, dv - spv.y - zc * spv.x, y[v]);
            }
        }
    }
}

template <int BITS, int MP>
__device__ void pass_consumer(const PassParams& p, uint8_t* smem, const PassSmem& L,
                              uint32_t full_s, uint32_t empty_s, volatile int* abort_flag,
                              volatile int* cur_stage, int warp, int lane) {
    constexpr int RBC = RecordFmt<BITS>::kBytes;
    constexpr int RB = RBC + kSZ;
    constexpr int SLOT = kPRec * RB;
    constexpr int GPA = 8 / MP;  // records per block: groups sharing one accumulator
    constexpr int LPB = 4 / MP;  // lanes of one output row that hold one batch row's columns
    const int tid = warp * 32 + lane;
    const int c = lane & 3, R = lane >> 2;
    const int bl = R / GPA, gil = R % GPA;  // batch row and block record of MMA column R
    const int NS = p.ns, M = p.M, XR = p.xg_row;
    uint4* xs = reinterpret_cast<uint4*>(smem + L.xs);
    float2* sp = reinterpret_cast<float2*>(smem + L.sp);
    Seg* segs = reinterpret_cast<Seg*>(smem + L.seg);
    LTile* tiles = reinterpret_cast<LTile*>(smem + L.tile);
    XItem* xitems = reinterpret_cast<XItem*>(smem + L.xi);
    float* slots = reinterpret_cast<float*>(smem + L.slot);
    const uint4* zblk = reinterpret_cast<const uint4*>(smem + L.zero);
    const uint8_t* ring = smem;
    float off[4];        // offsets c_k of this thread's pairs of X (see pass_stage_x)
#pragma unroll
    for (int w = 0; w < 4; ++w) off[w] = row_offset<BITS>((tid & 3) * 4 + w);
    RingPos pos{0, 0u};  // ring position of the SM's next round

    for (int s = 0; s < p.nstages; ++s) {
        const StageDesc* dp = p.stage + (size_t)blockIdx.x * p.nstages + s;
        // Stage s reads what earlier stages wrote: warp 0 waits until every CTA has completed
        // stage s - 1 (hence all before it), at once, so that the wait is not queued behind a
        // table load; a CTA without work in the stage waits too, long before the stage as a
        // whole can finish.  Meanwhile warps 1-15 copy the stage's tables (constants) into
        // shared memory: every consumer has passed the previous stage's last barrier, so
        // nothing reads the old ones any more.
        bool bad = false;
        if (warp == 0 && s > 0) bad = !wait_stage_done(p.ws, s - 1, gridDim.x, p.ws, lane);
        if (tid == 0 && bad) *abort_flag = 1;
        if (warp > 0) {
            const int nseg = dp->nseg, nt = dp->nt, nx = dp->nx;
            for (int i = tid - 32; i < nseg; i += 480) segs[i] = p.seg[dp->seg0 + i];
            for (int i = tid - 32; i < nt; i += 480) tiles[i] = p.tile[dp->tile0 + i];
            for (int i = tid - 32; i < nx; i += 480) xitems[i] = p.xi[dp->x0 + i];
        }
        if (cbar_any(bad || *abort_flag)) return;
        if (tid == 0) *cur_stage = s;  // the producer may copy the stage's rounds
        const int n = dp->n, nr = dp->nr, nt = dp->nt, nx = dp->nx;
        const int k0 = dp->wseg[warp], k1 = dp->wseg[warp + 1];
        if (n > 0) {
            for (int i = 0; i < nx; ++i) pass_stage_x(xitems[i], M, XR, xs, sp, tid, off);
            cbar();

            // This warp's records are the first len rounds of the stage (position `warp` of
            // each round's slot); walked segment by segment, in blocks of up to GPA records.
            const int len = (n >> 4) + (warp < (n & 15) ? 1 : 0);
            RingPos q = pos;
            bool aborted = false;
            for (int k = k0; k < k1 && !aborted; ++k) {
                const Seg sg = segs[k];
                float y[4] = {0.f, 0.f, 0.f, 0.f};
                for (int i = 0; i < sg.ng; i += GPA) {
                    const int bn = sg.ng - i < GPA ? sg.ng - i : GPA;
                    if (!wait_rounds(full_s, q, bn, NS, abort_flag, p.ws)) {
                        aborted = true;
                        break;
                    }
                    const int gb = sg.xg + sg.g0 + i;  // the block's first group in the X area
                    // B fragments of this lane: x of batch row bl of block record gil (rows
                    // 32c .. 32c + 31 of its group) when that record exists, else zeros
                    const uint4* xrow =
                        gil < bn && bl < M ? xs + 16 * (bl * XR + gb + gil) + 4 * c : zblk;
                    float D[4][4];
#pragma unroll
                    for (int v = 0; v < 4; ++v) D[0][v] = D[1][v] = D[2][v] = D[3][v] = 0.f;
                    if (bn == GPA) {
                        int sl = q.slot;
#pragma unroll
                        for (int gi = 0; gi < GPA; ++gi) {
                            pass_record<BITS>(ring + (size_t)sl * SLOT + (size_t)warp * RB,
                                              gil == gi ? xrow : zblk, p.exps, D, lane);
                            if (++sl == NS) sl = 0;
                        }
                    } else {
                        int sl = q.slot;
                        for (int gi = 0; gi < bn; ++gi) {
                            pass_record<BITS>(ring + (size_t)sl * SLOT + (size_t)warp * RB,
                                              gil == gi ? xrow : zblk, p.exps, D, lane);
                            if (++sl == NS) sl = 0;
                        }
                    }
                    pass_epilogue<BITS, MP>(ring, q.slot, NS, warp, lane, bn, M, XR, sp + gb, D,
                                            y);
                    release_rounds(empty_s, q, bn, NS, lane);
                }
                if (aborted) break;
                // Segment end: a lane's two columns belong to one batch row (c / LPB); its LPB
                // lanes of the output row add up, and slot (k, b) gets the 16 outputs of batch
                // row b.
                float lo = y[0] + y[1], hi = y[2] + y[3];
#pragma unroll
                for (int o = 1; o < LPB; o <<= 1) {
                    lo += __shfl_xor_sync(0xffffffffu, lo, o);
                    hi += __shfl_xor_sync(0xffffffffu, hi, o);
                }
                const int b = c / LPB;
                if (c % LPB == 0 && b < M) {
                    slots[16 * (k * MP + b) + R] = lo;
                    slots[16 * (k * MP + b) + R + 8] = hi;
                }
            }
            // the stage's last round, when it holds no record of this warp
            if (!aborted && len < nr) {
                if (wait_rounds(full_s, q, 1, NS, abort_flag, p.ws))
                    release_rounds(empty_s, q, 1, NS, lane);
                else
                    aborted = true;
            }
            pos = q;
            if (cbar_any(aborted || *abort_flag)) return;

            // The SM's tiles of the stage: each output is its segments' slots summed in order.
            for (int b = 0; b < M; ++b) {
                for (int idx = tid; idx < nt * 16; idx += 512) {
                    const int lt = idx >> 4, col = idx & 15;
                    const LTile t = tiles[lt];
                    float acc = 0.f;
                    for (int qq = 0; qq < t.nslot; ++qq)
                        acc += slots[16 * ((t.slot0 + qq) * MP + b) + col];
                    t.y[(size_t)b * t.ldy + col] = __half_as_ushort(__float2half_rn(acc));
                }
            }
            cbar();
        }
        // the stage is complete here once its Y stores are (release: ordered after them)
        if (tid == 0) red_rel_add(p.ws + kCounterStride * (1 + s % kCounters), 1u);
    }
}

template <int BITS, int MP>
__global__ void __launch_bounds__(kPThreads, 1) pass_kernel(const PassParams p) {
    extern __shared__ __align__(128) uint8_t smem[];
    constexpr int RB = RecordFmt<BITS>::kBytes + kSZ;
    const PassSmem L = pass_smem(RB, p.ns, p.xs_bytes, p.max_segs, p.max_nx, MP);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(smem);
    const uint32_t full_s = base + (uint32_t)L.bar;
    const uint32_t empty_s = full_s + 8u * kMaxRing;
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L.flag);
    volatile int* cur_stage = abort_flag + 1;  // the last stage whose dependency is met

    if (threadIdx.x == 0) {
        for (int i = 0; i < p.ns; ++i) {
            mbar_init(full_s + 8u * i, 1u);
            mbar_init(empty_s + 8u * i, (uint32_t)kPW);
        }
        // an error recorded by an earlier call: the call does nothing
        *abort_flag = ld_rlx(p.ws) != 0u ? 1 : 0;
        *cur_stage = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (threadIdx.x < 4)
        reinterpret_cast<uint4*>(smem + L.zero)[threadIdx.x] = make_uint4(0u, 0u, 0u, 0u);
    __syncthreads();

    const SmDesc sd = p.sm[blockIdx.x];
    if (*abort_flag) {
        // no copy is issued, no stage runs, and the workspace stays as it is
    } else if (warp == kPW)
        pass_producer<BITS>(p, sd, base, full_s, empty_s, abort_flag, cur_stage, lane);
    else
        pass_consumer<BITS, MP>(p, smem, L, full_s, empty_s, abort_flag, cur_stage, warp, lane);
    __syncthreads();

    // The last CTA to finish (every other one has made its last counter read) zeroes the
    // counters for the next call on the stream.
    if (threadIdx.x == 0 && *abort_flag == 0) {
        const uint32_t done = atom_acq_rel_add(p.ws + 1, 1u);
        if (done == gridDim.x - 1) {
            for (int j = 0; j < kCounters; ++j) p.ws[kCounterStride * (1 + j)] = 0u;
            p.ws[1] = 0u;
        }
    }
}

// ---- the gather kernel of laq_pass_prepare -----------------------------------------------------

// One warp per stream record: its packed codes (rbc bytes), then the scales and zeros of its
// (group, tile) as row pairs: 32-bit word r (r < 8) holds the fp16 scales of tile columns r
// (low half) and r + 8 (high half), then 16-bit word r the zeros of columns r (low byte) and
// r + 8, so the lane of output rows r and r + 8 reads one word and one half-word.
__global__ void pass_gather_kernel(const GatherRec* __restrict__ gt,
                                   const PrepEntry* __restrict__ pe, uint8_t* __restrict__ out,
                                   int64_t records, int rbc, int rb) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < records;
         i += nw) {
        const GatherRec g = gt[i];
        const PrepEntry E = pe[g.e];
        const int t = g.rid / E.G, grp = g.rid - t * E.G;
        const uint4* src = reinterpret_cast<const uint4*>(E.packed + (int64_t)g.rid * rbc);
        uint4* dst = reinterpret_cast<uint4*>(out + i * rb);
        for (int ch = lane; ch < rbc / 16; ch += 32) dst[ch] = src[ch];
        const size_t so = (size_t)grp * (size_t)E.N + (size_t)t * 16;
        if (lane < 8) {
            uint8_t* sz = out + i * rb + rbc;
            reinterpret_cast<uint32_t*>(sz)[lane] =
                (uint32_t)E.s[so + lane] | ((uint32_t)E.s[so + lane + 8] << 16);
            reinterpret_cast<uint16_t*>(sz + 32)[lane] =
                (uint16_t)((uint32_t)E.z[so + lane] | ((uint32_t)E.z[so + lane + 8] << 8));
        }
    }
}

std::atomic<int> g_pass_attr[2][3];  // shared memory granted to pass_kernel<bits, 1 | 2 | 4>

template <int BITS>
const void* pick_pass(int mp) {
    return mp == 1 ? (const void*)pass_kernel<BITS, 1>
                   : mp == 2 ? (const void*)pass_kernel<BITS, 2> : (const void*)pass_kernel<BITS, 4>;
}

int device_sms(int* sms, int* smem_optin) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return -1;
    if (cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return -1;
    if (cudaDeviceGetAttribute(smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
        cudaSuccess)
        return -1;
    return 0;
}

}  // namespace
}  // namespace laq

using namespace laq;

extern "C" {

laq_status laq_pass_plan_sizes(const laq_gemv* gemvs, int32_t count, int32_t num_sms,
                               size_t* plan_bytes, size_t* device_bytes) {
    if (!plan_bytes || !device_bytes) return LAQ_ERR_NULL;
    HostPlan H;
    const laq_status st = plan_pass(gemvs, count, num_sms, H);
    if (st != LAQ_OK) return st;
    PlanHeader h;
    layout(H, h);
    *plan_bytes = (size_t)h.plan_bytes;
    *device_bytes = (size_t)h.device_bytes;
    return LAQ_OK;
}

laq_status laq_pass_plan_build(const laq_gemv* gemvs, int32_t count, int32_t num_sms,
                               void* plan, size_t plan_bytes) {
    if (!plan) return LAQ_ERR_NULL;
    HostPlan H;
    const laq_status st = plan_pass(gemvs, count, num_sms, H);
    if (st != LAQ_OK) return st;
    PlanHeader h;
    layout(H, h);
    if (plan_bytes < (size_t)h.plan_bytes) return LAQ_ERR_WORKSPACE;
    uint8_t* out = static_cast<uint8_t*>(plan);
    std::memset(out, 0, (size_t)h.plan_bytes);
    std::memcpy(out, &h, sizeof(h));
    if (count > 0) std::memcpy(out + 256, gemvs, (size_t)count * sizeof(laq_gemv));
    uint8_t* t = out + h.tables_h;
    put(t, h.o_sm, H.sm);
    put(t, h.o_rounds, H.rounds);
    put(t, h.o_stage, H.stage);
    put(t, h.o_seg, H.seg);
    put(t, h.o_tile, H.tile);
    put(t, h.o_x, H.xi);
    put(t, h.o_prep, H.prep);
    put(t, h.o_gather, H.gather);
    return LAQ_OK;
}

size_t laq_pass_workspace_bytes(const void* plan) {
    const PlanHeader* h = as_plan(plan);
    return h ? pass_workspace(*h) : 0;
}

laq_status laq_pass_prepare(const void* plan, void* device, size_t device_bytes, void* stream) {
    const PlanHeader* h = as_plan(plan);
    if (!h) return LAQ_ERR_CONFIG;
    if (!device) return LAQ_ERR_NULL;
    if (reinterpret_cast<uintptr_t>(device) & 255u) return LAQ_ERR_ALIGN;
    if (device_bytes < (size_t)h->device_bytes) return LAQ_ERR_WORKSPACE;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* dev = static_cast<uint8_t*>(device);
    const uint8_t* host = static_cast<const uint8_t*>(plan);
    if (h->tables_bytes > 0 &&
        cudaMemcpyAsync(dev + h->stream_bytes, host + h->tables_h, (size_t)h->tables_bytes,
                        cudaMemcpyHostToDevice, st) != cudaSuccess)
        return LAQ_ERR_CUDA;
    if (h->records == 0) return LAQ_OK;
    const uint8_t* tables = dev + h->stream_bytes;
    const int64_t blocks64 = (h->records + 7) / 8;
    const unsigned blocks = (unsigned)(blocks64 < 8192 ? blocks64 : 8192);
    pass_gather_kernel<<<blocks, 256, 0, st>>>(
        reinterpret_cast<const GatherRec*>(tables + h->o_gather),
        reinterpret_cast<const PrepEntry*>(tables + h->o_prep), dev, h->records,
        h->rb - kSZ, h->rb);
    return cudaGetLastError() == cudaSuccess ? LAQ_OK : LAQ_ERR_CUDA;
}

laq_status laq_pass_run(const void* plan, const void* device, void* workspace,
                        size_t workspace_bytes, void* stream) {
    const PlanHeader* h = as_plan(plan);
    if (!h) return LAQ_ERR_CONFIG;
    if (!device || !workspace) return LAQ_ERR_NULL;
    if (reinterpret_cast<uintptr_t>(device) & 255u) return LAQ_ERR_ALIGN;
    if ((reinterpret_cast<uintptr_t>(workspace) & 15u) || workspace_bytes < pass_workspace(*h))
        return LAQ_ERR_WORKSPACE;
    if (h->nstages == 0) return LAQ_OK;
    int sms = 0, optin = 0;
    if (device_sms(&sms, &optin) != 0) return LAQ_ERR_CUDA;
    if (sms != h->sms) return LAQ_ERR_CONFIG;  // planned for another SM count
    // ring depth: as many 16-record slots as the shared memory left over holds
    const int mp = h->M == 1 ? 1 : h->M == 2 ? 2 : 4;
    int ns = kMaxRing;
    while (ns >= 2 &&
           pass_smem(h->rb, ns, h->xs_bytes, h->max_segs, h->max_nx, mp).total > optin)
        --ns;
    // a warp holds the rounds of one block (8 / MP records) at once, in distinct slots
    if (ns < 8 / mp) return LAQ_ERR_SHAPE;
    const PassSmem L = pass_smem(h->rb, ns, h->xs_bytes, h->max_segs, h->max_nx, mp);

    const uint8_t* dev = static_cast<const uint8_t*>(device);
    const uint8_t* t = dev + h->stream_bytes;
    PassParams P;
    P.stream = dev;
    P.sm = reinterpret_cast<const SmDesc*>(t + h->o_sm);
    P.rounds = t + h->o_rounds;
    P.stage = reinterpret_cast<const StageDesc*>(t + h->o_stage);
    P.seg = reinterpret_cast<const Seg*>(t + h->o_seg);
    P.tile = reinterpret_cast<const LTile*>(t + h->o_tile);
    P.xi = reinterpret_cast<const XItem*>(t + h->o_x);
    P.ws = static_cast<uint32_t*>(workspace);
    P.nstages = h->nstages;
    P.ns = ns;
    P.xs_bytes = h->xs_bytes;
    P.max_segs = h->max_segs;
    P.max_nx = h->max_nx;
    P.M = h->M;
    P.xg_row = h->xg_row;
    P.exps = exps_for(h->bits);

    const void* fn = h->bits == 4 ? pick_pass<4>(mp) : pick_pass<3>(mp);
    // First call with this much shared memory (before any stream capture): raise the kernel's
    // limit and check that a CTA fits an SM, as the cooperative launch requires.
    std::atomic<int>& granted = g_pass_attr[h->bits == 4][mp == 1 ? 0 : mp == 2 ? 1 : 2];
    if (granted.load() < L.total) {
        if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, L.total) !=
            cudaSuccess)
            return LAQ_ERR_CUDA;
        int per_sm = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kPThreads, L.total) !=
                cudaSuccess ||
            per_sm < 1)
            return LAQ_ERR_CONFIG;
        granted.store(L.total);
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)h->sms);
    cfg.blockDim = dim3(kPThreads);
    cfg.dynamicSmemBytes = (size_t)L.total;
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    void* args[] = {&P};
    const cudaError_t err = cudaLaunchKernelExC(&cfg, fn, args);
    if (err == cudaErrorInvalidConfiguration || err == cudaErrorCooperativeLaunchTooLarge)
        return LAQ_ERR_CONFIG;
    return err == cudaSuccess ? LAQ_OK : LAQ_ERR_CUDA;
}

}  // extern "C"
