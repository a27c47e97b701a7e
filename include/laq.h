/*
 * laq.h -- C ABI of the weight-only WbG128 (b = 3 or 4) quantized linear layer for NVIDIA GB300
 * (sm_103a): RTN group quantizer, bit packing, and the dequantize-fused GEMV / skinny GEMM
 * Y[M,N] = X[M,K] * W_hat[K,N] for M = 1..16 (LAQuant, arXiv 2605.08755).
 *
 * Quantization format (Eq. (1) and Sec. 2 "Grouped quantization"): every weight w is a b-bit
 * code q in [0, 2^b - 1] with a scale s and a zero z shared by a group of g = 128 consecutive
 * elements of a weight row, and w_hat = s * (q - z).  With the weight stored as W[K][N]
 * (K = in_features, N = out_features) a group is 128 consecutive k of one column n, and the
 * scales and zeros form (num_groups, out_features) tensors as in App. H ("Group-wise
 * quantization").  No online transform is applied to X (Sec. 3, "Runtime-overhead-free
 * quantization").
 *
 * Conventions shared by every entry point:
 *   - Pointers are caller-owned DEVICE memory unless stated otherwise.  The library never
 *     allocates, frees or synchronizes, and never reads device memory on the host.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Work is enqueued
 *     asynchronously on it; results are ready when the stream says so.
 *   - Arguments are validated on the host first.  An invalid call returns its status and
 *     enqueues nothing.  A launch failure returns LAQ_ERR_CUDA.
 *   - Matrices are dense row-major with no padding: X[M][K] and Y[M][N] fp16, W[K][N] fp16,
 *     codes[K][N] uint8, s[K/128][N] fp16, z[K/128][N] uint8.
 *   - Empty shapes are legal: a call with M, K or N equal to 0 writes only the (possibly
 *     empty) outputs it defines (a GEMM with K = 0 sets Y to zero).
 *   - Every entry point that takes a stream may be captured into a CUDA graph, provided the
 *     first call for each (bits, M-class) variant happens before capture begins (that first
 *     call sets the kernel's shared-memory limit and caches the device's SM count).
 */
#ifndef LAQ_H
#define LAQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    LAQ_OK = 0,
    LAQ_ERR_NULL = 1,     /* a required pointer is NULL                                  */
    LAQ_ERR_BITS = 2,     /* bits is not 3 or 4                                          */
    LAQ_ERR_GROUP = 3,    /* group size is not 128                                       */
    LAQ_ERR_SHAPE = 4,    /* negative size, K % 128 != 0, N % 16 != 0, or a size too big */
    LAQ_ERR_ALIGN = 5,    /* a pointer breaks its alignment requirement                  */
    LAQ_ERR_M_RANGE = 6,  /* M outside 0..16 (1..4 for laq_gemm_chain)                   */
    LAQ_ERR_CUDA = 7,     /* the CUDA runtime reported an error for the launch           */
    LAQ_ERR_TIMEOUT = 8,  /* a bounded device-side wait gave up (laq_gemm_chain status)  */
    LAQ_ERR_CONFIG = 9,   /* an explicit launch configuration is not supported           */
    LAQ_ERR_WORKSPACE = 10 /* workspace missing, misaligned or smaller than required      */
} laq_status;

/* Human-readable name of a status code (static storage, never NULL). */
const char *laq_status_str(int status);

/* ABI version of this header: 1. */
int laq_version(void);

/* Bytes of packed codes for a K x N weight at `bits` per code: K * N * bits / 8 exactly (no
 * padding).  Returns 0 for invalid arguments. */
size_t laq_packed_bytes(int64_t K, int64_t N, int bits);

/*
 * laq_quantize_rtn -- min-max round-to-nearest group quantizer of Eq. (1).
 *
 *   W      [K][N] fp16, finite values.                                  (in,  2-byte aligned)
 *   codes  [K][N] uint8, q = clip(rint(w / s) + z, 0, 2^b - 1).          (out)
 *   s      [K/128][N] fp16 group scales.                                 (out, 2-byte aligned)
 *   z      [K/128][N] uint8 group zeros in [0, 2^b - 1].                 (out)
 *   bits   3 or 4;  group must be 128;  K % 128 == 0.
 *
 * Eq. (1) fixes q and w_hat given s and z; the paper learns s and z by QAT.  This initializer
 * fixes them per (group, column) from lo = min w, hi = max w, in fp64:
 *   - constant group (lo == hi == c): s = |c| (1.0 if c == 0), z = 1 if c < 0 else 0, so
 *     w_hat == c exactly;
 *   - otherwise lo' = min(lo, 0), hi' = max(hi, 0), s = the smallest fp16 >= (hi' - lo') /
 *     (2^b - 1), raised to 2^-14 if below it, and z = rint(-lo' / s);
 *   - rint is round-half-to-even and is applied to w / s before z is added, as Eq. (1) reads.
 * Consequences: 0 <= z <= 2^b - 1 and |w - w_hat| <= s / 2 for every element.  Results are
 * deterministic and bit-identical to a plain fp64 implementation of the rule above.
 * Non-finite inputs give unspecified codes.
 */
laq_status laq_quantize_rtn(const void *W, int64_t K, int64_t N, int bits, int group,
                            uint8_t *codes, void *s, uint8_t *z, void *stream);

/*
 * laq_pack -- codes[K][N] (values < 2^bits) -> packed words, the layout laq_gemm_wxg128 reads.
 * App. H keeps the INT3 kernel's "32 weights in three 32-bit words" packing; this library uses
 * its own layout with the same density (K * N * bits / 8 bytes), built around the tensor-core
 * fragment that consumes it.  Requires K % 128 == 0, N % 16 == 0, packed 16-byte aligned.
 *
 * Layout.  Codes are grouped into records of 16 columns x 128 rows: record (t, g) covers
 * columns n = 16t..16t+15 and rows k = 128g..128g+127 and is stored at record index
 * t * (K/128) + g (tile-major).  A record is 32 * bits 32-bit words (1024 bytes at b = 4, 768
 * at b = 3) and is split among 32 lanes; lane l (c = l % 4, r = l / 4) owns the 64 codes at
 * columns r and r + 8 of the tile and rows k = 128g + 32c + 4j + 2h + e (j = 0..7,
 * h, e = 0..1), so a lane's rows are 32 consecutive rows of the group.  A "pair" (j, h, row) is
 * the two codes with e = 0 (bits 0..15 of a word) and e = 1 (the same position in bits
 * 16..31).  Fields below are positions within each 16-bit half, least significant code bit
 * first:
 *   b = 4: 8 words per lane; word j: bits 0-3 pair (j,0,r), 4-7 (j,1,r), 8-11 (j,0,r+8),
 *          12-15 (j,1,r+8).  Word w of lane l is record word (w/4)*128 + 4l + (w%4).
 *   b = 3: 6 words per lane; with pair index i = 2j + h, word w holds: bit 0 = bit (w % 3)
 *          of pair (i = 15, r if w < 3 else r+8), bits 1-3 pair (i = w, r), 4-6 (i = 6+w, r),
 *          7-9 (i = 12 + w/2, r if w even else r+8), 10-12 (i = w, r+8), 13-15 (i = 6+w, r+8).
 *          Word w of lane l is record word 4l + w (w < 4) or 128 + 2l + (w - 4) (w >= 4).
 */
laq_status laq_pack(const uint8_t *codes, int64_t K, int64_t N, int bits, void *packed,
                    void *stream);

/* laq_unpack -- the inverse of laq_pack (a test and inspection aid).  Same requirements. */
laq_status laq_unpack(const void *packed, int64_t K, int64_t N, int bits, uint8_t *codes,
                      void *stream);

/*
 * laq_gemm_wxg128 -- Y[M][N] = X[M][K] * W_hat[K][N], W_hat = s * (q - z) per Eq. (1), the
 * quantized linear layer of the decode step (Sec. 5.2 "Inference", Table 3; App. H).
 *
 *   X       [M][K] fp16 activations.                                (in, 16-byte aligned)
 *   packed  laq_pack output for the K x N codes at `bits`.          (in, 16-byte aligned)
 *   s, z    [K/128][N] fp16 scales and uint8 zeros.                 (in, 16-byte aligned)
 *   Y       [M][N] fp16, must not overlap any input.                (out, 16-byte aligned)
 *   0 <= M <= 16, K % 128 == 0, N % 16 == 0, bits 3 or 4.
 *
 * Arithmetic: products and sums in fp32 (tensor-core accumulation), one fp16 rounding of each
 * output.  |Y - Y_exact| stays within 5e-3 * max|Y_exact| + 1e-3 for the weight and activation
 * distributions of the paper's workloads.  Deterministic: no atomics; a given launch
 * configuration always sums in the same order.
 */
laq_status laq_gemm_wxg128(const void *X, int64_t M, int64_t K, int64_t N, const void *packed,
                           const void *s, const uint8_t *z, int bits, void *Y, void *stream);

/*
 * Launch configuration of laq_gemm_wxg128 (a tuning interface; the library picks one itself).
 *   tiles_per_cta  16-column tiles per CTA: 1, 2, 4 or 8.
 *   warps          warps per CTA, 1..16 (1..8 for M <= 2), a multiple of tiles_per_cta;
 *                  each tile gets warps / tiles_per_cta warps, which split the CTA's K range.
 *   cluster        CTAs per thread-block cluster, 1, 2, 4 or 8; the CTAs of a cluster split
 *                  K and reduce their partial sums through distributed shared memory.
 *   stages         depth of each warp's cp.async ring of weight records, 2..16; with
 *                  stages > the warp's record count the whole slice is copied up front.
 *   pdl            1: launch with programmatic dependent launch, so the kernel may start and
 *                  prefetch weights while the previous kernel on the stream finishes; X is
 *                  read and Y written only after that kernel completes.  Only valid when the
 *                  immediately preceding work on the stream does not write packed, s or z.
 */
typedef struct {
    int32_t tiles_per_cta;
    int32_t warps;
    int32_t cluster;
    int32_t stages;
    int32_t pdl;
    int32_t reserved[3];
} laq_gemm_config;

/* The configuration laq_gemm_wxg128 uses for this shape on a GPU with `num_sms` SMs (host-only
 * computation; no device access; the shared memory of an SM is taken as sm_100 / sm_103's
 * 228 KB, so that two CTAs fit one SM where the grid needs it).  Returns the same argument
 * statuses as laq_gemm_wxg128. */
laq_status laq_gemm_plan(int64_t M, int64_t K, int64_t N, int bits, int num_sms,
                         laq_gemm_config *out);

/* laq_gemm_wxg128 with an explicit configuration.  Same contract; LAQ_ERR_CONFIG if a field is
 * outside its range or the shared memory it needs exceeds the device limit. */
laq_status laq_gemm_wxg128_config(const void *X, int64_t M, int64_t K, int64_t N,
                                  const void *packed, const void *s, const uint8_t *z, int bits,
                                  void *Y, const laq_gemm_config *cfg, void *stream);

/*
 * One GEMV of a chain (laq_gemm_chain): Y[M][N] = X[M][K] * W_hat[K][N], with the operands and
 * rules of laq_gemm_wxg128.  `wait_prev` != 0 marks an entry that reads results of earlier
 * entries (its X is the output of, or computed from, an earlier Y): it starts only after every
 * earlier entry has completed.  Entries with wait_prev == 0 join the run of entries since the
 * last marked one (a "stage") and may execute alongside it, as q, k and v, or gate and up, of a
 * decoder layer do.  Entry 0's flag is ignored.
 */
typedef struct laq_gemv {
    const void *X;       /* fp16 [M][K], 16-byte aligned                 */
    const void *packed;  /* laq_pack layout, 16-byte aligned             */
    const void *s;       /* fp16 [K/128][N], 16-byte aligned             */
    const uint8_t *z;    /* uint8 [K/128][N], 16-byte aligned            */
    void *Y;             /* fp16 [M][N], 16-byte aligned, no overlap     */
    int64_t M, K, N;
    int32_t bits;
    int32_t wait_prev;
} laq_gemv;

/* Most entries one laq_gemm_chain call takes. */
#define LAQ_CHAIN_MAX 384

/* Workspace bytes laq_gemm_chain needs for `count` entries (0 if count is out of range). */
size_t laq_chain_workspace_bytes(int32_t count);

/*
 * Run `count` GEMVs in one persistent kernel launch on `stream`, with the results of issuing
 * laq_gemm_wxg128 for each entry in order on that stream: the decode-step weight pass of a
 * decoder (Sec. 5.2, "Inference": decoding streams every projection's weights once per token)
 * without a kernel boundary between projections.  Each entry's Y is the fp32 sum of its
 * dequantized products (Eq. (1)) rounded once to fp16, like laq_gemm_wxg128's; the two agree
 * to fp32 rounding (their summation orders differ).
 *
 *   gemvs      HOST array of `count` entries (read during the call only).  All entries share
 *              `bits` (3 or 4) and M (1..4).  K % 128 == 0, N % 16 == 0, K, N > 0.
 *   count      0..LAQ_CHAIN_MAX (0: nothing is enqueued).
 *   workspace  DEVICE buffer of at least laq_chain_workspace_bytes(count) bytes (about 67 KB:
 *              stage counters, and a flag and a 256-byte partial tile for each of up to 256
 *              CTAs), 16-byte aligned, ZERO-FILLED before its first use.  A call that
 *              completes normally leaves its counters and flags zero again.  Word 0 (uint32)
 *              is the device-side status: 0, or
 *              LAQ_ERR_TIMEOUT if a wait between stages gave up (after about a second); the
 *              call's Y values are then undefined and the caller must zero the workspace
 *              before the next call.  Calls sharing one workspace must not overlap in time.
 *
 * Restrictions: the packed codes, scales and zeros of every entry are read ahead of the chain
 * order, so no entry may write them; an entry may not read a Y written by an entry of its own
 * stage; the X of one stage (M * K * 2 bytes summed over its entries) must fit the kernel's
 * shared memory beside its weight ring and descriptors (LAQ_ERR_SHAPE otherwise; on GB300
 * about 95 KB for a 252-entry chain, a little more for shorter ones).  Uses every SM of
 * the device with one cooperative CTA each, so concurrent kernels on other streams wait.
 * Returns LAQ_ERR_M_RANGE for M outside 1..4, LAQ_ERR_BITS for mixed or invalid bits,
 * LAQ_ERR_WORKSPACE for a bad workspace, and the per-entry statuses of laq_gemm_wxg128.
 */
laq_status laq_gemm_chain(const laq_gemv *gemvs, int32_t count, void *workspace,
                          size_t workspace_bytes, void *stream);

/*
 * laq_gemm_chain without a caller-provided workspace, for callers that cannot allocate device
 * memory: a plug-in or custom operator whose host framework owns every device allocation and
 * offers no scratch, or a decode loop that must not call cudaMalloc once it runs (cudaMalloc
 * may synchronize the device and stalls every stream).  The paper has no counterpart; this is
 * a deployment convenience of this library.
 *
 * Same entries, results and restrictions as laq_gemm_chain.  The workspace lives in a scratch
 * array inside the library (a static device array of 68,352 bytes, enough for LAQ_CHAIN_MAX
 * entries), held by every GPU that loads the library until the process exits.  Nothing is
 * allocated: once every argument has passed its checks, each call clears the counters and
 * flags it uses (cudaMemsetAsync on `stream`) and launches; a call rejected by a check
 * enqueues nothing.
 *   count < 0              -> LAQ_ERR_SHAPE (as laq_gemm_chain)
 *   count > LAQ_CHAIN_MAX  -> LAQ_ERR_WORKSPACE (the scratch holds no more).
 * The first call on each device looks up the scratch array's device address (and, like every
 * first call of a kernel variant, sets its shared-memory limit): make it before any stream
 * capture.  The address belongs to the CUDA context it was looked up in; after
 * cudaDeviceReset the next call looks it up again in the new context (that call, too, should
 * come before any capture).  All calls share the one array, so calls whose executions overlap on the GPU (other
 * streams, or other host threads) race and give undefined results; serialize them.  A
 * device-side timeout is not reported here (laq_gemm_chain's workspace status word is the way
 * to observe one).
 */
laq_status laq_gemm_chain_static(const laq_gemv *gemvs, int32_t count, void *stream);

/*
 * ======================================================================================
 * The planned pass: the chain of laq_gemm_chain (same laq_gemv entries and stage rules), with
 * the walk over its weights done once on the host.  A plan deals each stage's 16-column tiles
 * to the SMs as whole tiles (balanced by records of 16 columns x 128 rows), cuts every SM's
 * records into 16 warp shares, and orders them into one contiguous stream per SM, each record's
 * 16 scales and 16 zeros beside its packed codes.  laq_pass_prepare writes those streams into a
 * caller-owned device buffer once; laq_pass_run then streams them with bulk copies into a ring
 * of shared memory that runs ahead across the stage boundaries (the weights never depend on the
 * activations), while the stages wait for their inputs.  It serves the decode-step weight pass
 * (Sec. 5.2, "Inference": a decode step streams every projection's weights once), and each
 * entry's Y is that of laq_gemm_wxg128 (fp32 sums of Eq. (1) products, one fp16 rounding; the
 * summation orders differ).  M = 1..4, the same for every entry.
 *
 * Usage: laq_pass_plan_sizes -> allocate the host plan (plan_bytes) and the device buffer
 * (device_bytes, 256-byte aligned) -> laq_pass_plan_build -> laq_pass_prepare -> a zeroed
 * workspace of laq_pass_workspace_bytes -> laq_pass_run, any number of times.
 * ====================================================================================== */

/* Host bytes of the plan and device bytes of the streams and tables for `count` entries
 * (HOST array, read during the call) on a device with `num_sms` SMs.  Host work only (no CUDA
 * call).  Entries as laq_gemm_chain's, with one M (1..4) and one `bits` for all, M * K * 2 <=
 * 106496 bytes (an entry's X must fit the kernel's staging area), N % 16 == 0, K, N > 0.  The device buffer holds every
 * packed record once more (K * N * bits / 8 + 3 * N * K / 128 bytes per entry) plus tables.
 * Errors: LAQ_ERR_NULL, LAQ_ERR_BITS (invalid or mixed bits), LAQ_ERR_M_RANGE (M outside 1..4
 * or mixed), LAQ_ERR_SHAPE (count outside 0..LAQ_CHAIN_MAX, num_sms outside 1..1024, a bad K or
 * N, an SM's share of one stage above 255 warp segments, or the X it stages above 106496 bytes), LAQ_ERR_ALIGN (a pointer not 16-byte
 * aligned). */
laq_status laq_pass_plan_sizes(const laq_gemv *gemvs, int32_t count, int32_t num_sms,
                               size_t *plan_bytes, size_t *device_bytes);

/* Write the plan into the HOST buffer `plan` (plan_bytes from laq_pass_plan_sizes; smaller:
 * LAQ_ERR_WORKSPACE).  Host work only.  The plan records the entries' X and Y addresses, which
 * every laq_pass_run uses; packed, s and z are read only by laq_pass_prepare. */
laq_status laq_pass_plan_build(const laq_gemv *gemvs, int32_t count, int32_t num_sms,
                               void *plan, size_t plan_bytes);

/* Workspace bytes laq_pass_run needs for this plan (status word, a finished-CTA count and one
 * completed-stage flag per SM; 0 if `plan` is not a plan). */
size_t laq_pass_workspace_bytes(const void *plan);

/* Lay the plan's weights out in the DEVICE buffer `device` (256-byte aligned, device_bytes from
 * laq_pass_plan_sizes): copies the plan's tables (a host-to-device copy from pageable memory,
 * which waits for the stream's earlier work; not for stream capture) and enqueues the gather
 * kernel on `stream`.  The entries' packed codes, scales and zeros must stay valid until that
 * kernel has run; afterwards the pass reads only `device`.  Errors: LAQ_ERR_CONFIG (not a
 * plan), LAQ_ERR_NULL, LAQ_ERR_ALIGN, LAQ_ERR_WORKSPACE (device buffer too small),
 * LAQ_ERR_CUDA. */
laq_status laq_pass_prepare(const void *plan, void *device, size_t device_bytes, void *stream);

/* Run the planned pass on `stream`: one cooperative launch of one CTA per SM.  `plan` is the
 * HOST plan, `device` the prepared buffer, `workspace` a DEVICE buffer of at least
 * laq_pass_workspace_bytes(plan) bytes, 16-byte aligned, zero before its first use (a completed
 * call leaves it zero again); word 0 (uint32) is the device-side status: 0, or LAQ_ERR_TIMEOUT
 * if a wait gave up after about a second (Y undefined; zero the workspace before the next
 * call).  Calls sharing one workspace must not overlap in time.  The device must have the SM
 * count the plan was built for (LAQ_ERR_CONFIG otherwise).  The first call for each bit width
 * and shared-memory size sets the kernel's limit: make it before any stream capture, which may
 * then record later calls.  Errors: LAQ_ERR_CONFIG (not a plan,
 * another SM count, the launch does not fit), LAQ_ERR_NULL, LAQ_ERR_ALIGN (device buffer),
 * LAQ_ERR_WORKSPACE, LAQ_ERR_SHAPE (the staging area and a ring of two slots exceed shared
 * memory), LAQ_ERR_CUDA. */
laq_status laq_pass_run(const void *plan, const void *device, void *workspace,
                        size_t workspace_bytes, void *stream);

/*
 * A prologue applied to X while laq_gemm_wxg128_prologue stages it, so that the operation
 * before a projection costs no launch of its own.  The paper has no counterpart: this fuses two
 * of the decoder operations declared below (laq_rmsnorm, laq_silu_mul) into the GEMV.
 *   LAQ_PROLOGUE_RMSNORM: the GEMV's input is laq_rmsnorm's Y of (X [M][K], R, w, eps):
 *     h = fp16(X + R) (h = X when R is NULL), input = fp16(h / sqrt(mean_k h^2 + eps) * w),
 *     and when R_out is not NULL, R_out = h [M][K].  R_out must not alias X or R (CTAs read the
 *     whole rows of X and R while one of them writes R_out): LAQ_ERR_SHAPE otherwise.
 *   LAQ_PROLOGUE_SILU_MUL: X holds [M][2K] (gate | up); input = fp16(silu(gate) * up), as
 *     laq_silu_mul.
 * X, R, R_out and w 16-byte aligned.
 */
#define LAQ_PROLOGUE_NONE 0
#define LAQ_PROLOGUE_RMSNORM 1
#define LAQ_PROLOGUE_SILU_MUL 2
typedef struct laq_gemm_prologue {
    int32_t kind;
    float eps;          /* RMSNORM */
    const void *R;      /* RMSNORM: residual [M][K] or NULL */
    void *R_out;        /* RMSNORM: receives fp16(X + R) [M][K], or NULL */
    const void *w;      /* RMSNORM: weights [K] */
} laq_gemm_prologue;

/* laq_gemm_wxg128 with a prologue on X (pro NULL or kind NONE: plain) and an optional explicit
 * configuration (cfg NULL: planned; laq_gemm_wxg128_config's rules otherwise).  All pointers are
 * device pointers owned by the caller; Y [M][N] is overwritten.  Results equal those of the
 * unfused sequence within fp16 rounding: the row's sum of squares is added in another order, and
 * SILU_MUL uses the hardware exponential and reciprocal (relative error ~2^-21).  Errors: as
 * laq_gemm_wxg128, plus LAQ_ERR_CONFIG for an unknown kind, LAQ_ERR_NULL for RMSNORM without
 * w, LAQ_ERR_SHAPE for eps < 0 (or NaN) or R_out equal to X or R, LAQ_ERR_ALIGN for a
 * misaligned X, R, R_out or w. */
laq_status laq_gemm_wxg128_prologue(const void *X, int64_t M, int64_t K, int64_t N,
                                    const void *packed, const void *s, const uint8_t *z, int bits,
                                    void *Y, const laq_gemm_prologue *pro,
                                    const laq_gemm_config *cfg, void *stream);

/* ======================================================================================
 * Decoder operations around the projections: the rest of one decode step of a Qwen3-style
 * model (the models whose decoding speed Sec. 5.2 reports).  The paper defines none of them;
 * each follows the standard decoder definition stated below, computes in fp32 and rounds each
 * stored tensor to fp16 once.  All tensors are caller-owned device memory, row-major, fp16
 * unless stated; sizes are validated on the host (LAQ_ERR_SHAPE / LAQ_ERR_ALIGN /
 * LAQ_ERR_NULL, nothing launched); values read from device memory (positions, lengths,
 * tokens) are clamped in the kernels as stated and never index outside the given buffers.
 * Each kernel may start while its predecessor on the stream finishes (programmatic dependent
 * launch) and waits for it before touching memory.
 * ====================================================================================== */

/*
 * RMSNorm with the residual add, one row per m < M (1 <= M <= 65535, H % 8 == 0, 8 <= H <=
 * 8192; X, R, R_out, w, Y 16-byte aligned):
 *   h = fp16(X + R)            (h = X when R is NULL)
 *   R_out = h                  (skipped when R_out is NULL; R_out may equal R)
 *   Y = fp16(h / sqrt(mean_k h_k^2 + eps) * w)     w: [H] weights.
 */
laq_status laq_rmsnorm(const void *X, const void *R, void *R_out, const void *w, int64_t M,
                       int64_t H, float eps, void *Y, void *stream);

/*
 * Per-head RMSNorm of q and k, rotary position embedding, and the KV-cache append, for the
 * fused q|k|v projection output qkv [M][(Hq + 2 Hkv) * D] (q heads, then k heads, then v heads).
 * D must be 128; Hq % Hkv == 0 and Hq / Hkv <= 8.  For row m at position p = pos[m] (device):
 *   q_h = rope(rmsnorm(q_h) * q_norm_w)  -> q_out [M][Hq][D]
 *   k_g = rope(rmsnorm(k_g) * k_norm_w)  -> k_cache [M][Hkv][L_max][D] at [m][g][p]
 *   v_g                                  -> v_cache (same layout) at [m][g][p]
 * rmsnorm(x) = x / sqrt(mean(x^2) + eps); rope rotates pairs (i, i + D/2) by the angle
 * p * theta^(-2i/D):  (x_i, x_{i+D/2}) -> (x_i cos - x_{i+D/2} sin, x_{i+D/2} cos + x_i sin).
 * A position outside [0, L_max) still produces q but stores nothing in the caches.  qkv, q_out
 * and the caches must be 8-byte aligned.
 */
laq_status laq_qk_norm_rope(const void *qkv, const void *q_norm_w, const void *k_norm_w,
                            const int32_t *pos, int64_t M, int32_t Hq, int32_t Hkv, int32_t D,
                            float theta, float eps, void *q_out, void *k_cache, void *v_cache,
                            int64_t L_max, void *stream);

/* Bytes of workspace laq_attention_decode needs (fp32 partials of 64-token chunks); 0 for
 * invalid sizes. */
size_t laq_attention_workspace_bytes(int64_t M, int32_t Hq, int64_t L_max);

/*
 * Grouped-query attention of each row's new token over its cache (decode):
 *   out[m][h] = sum_{t < n} softmax_t(scale * q[m][h] . K[m][g][t]) V[m][g][t],  g = h / (Hq/Hkv),
 * n = len[m] (device) clamped to [0, L_max]; a row with n = 0 gets zeros.  q, out [M][Hq][D],
 * caches [M][Hkv][L_max][D], D = 128, Hq / Hkv <= 8.  Two launches: 64-token chunk partials
 * (max, sum of exponentials, weighted V sum) into `workspace`, then their combination in chunk
 * order (deterministic).  workspace_bytes >= laq_attention_workspace_bytes(M, Hq, L_max)
 * (LAQ_ERR_WORKSPACE otherwise; 4-byte aligned).  Both caches 16-byte aligned.
 */
laq_status laq_attention_decode(const void *q, const void *k_cache, const void *v_cache,
                                const int32_t *len, int64_t M, int32_t Hq, int32_t Hkv,
                                int32_t D, int64_t L_max, float scale, void *out,
                                void *workspace, size_t workspace_bytes, void *stream);

/* Bytes of workspace laq_attention_qkv needs (the chunk partials, as for
 * laq_attention_decode); 0 for invalid sizes. */
size_t laq_attention_qkv_workspace_bytes(int64_t M, int32_t Hq, int32_t Hkv, int64_t L_max);

/*
 * laq_qk_norm_rope followed by laq_attention_decode with len[m] = pos[m] + 1, in two launches
 * instead of three (same inputs, outputs and results): each attention CTA (64-token chunk, kv
 * head, row) normalises and rotates its q heads itself, and the CTA whose chunk holds pos[m]
 * computes the new k and v, stores them in the caches and uses them in place of the cached
 * row; the chunk partials are then combined in chunk order.  Workspace 16-byte aligned and
 * >= laq_attention_qkv_workspace_bytes (LAQ_ERR_WORKSPACE otherwise).
 */
laq_status laq_attention_qkv(const void *qkv, const void *q_norm_w, const void *k_norm_w,
                             const int32_t *pos, int64_t M, int32_t Hq, int32_t Hkv, int32_t D,
                             float theta, float eps, void *k_cache, void *v_cache, int64_t L_max,
                             float scale, void *out, void *workspace, size_t workspace_bytes,
                             void *stream);

/* h[m][i] = fp16(silu(g) * u), g = gate_up[m][i], u = gate_up[m][I + i], silu(x) = x / (1 +
 * e^-x): the fused gate|up projection output [M][2I] -> [M][I].  I % 8 == 0, 16-byte aligned. */
laq_status laq_silu_mul(const void *gate_up, int64_t M, int64_t I, void *h, void *stream);

/* X[m] = E[tokens[m]] for the embedding table E [V][H]; a token outside [0, V) gives a zero
 * row.  H % 8 == 0, E and X 16-byte aligned. */
laq_status laq_embed(const void *E, const int32_t *tokens, int64_t M, int64_t V, int64_t H,
                     void *X, void *stream);

/* out[m] = argmax_v logits[m][v] over fp16 logits [M][V] (ties: the smallest index; NaN never
 * wins; a row of NaN or -inf gives 0). */
laq_status laq_argmax(const void *logits, int64_t M, int64_t V, int32_t *out, void *stream);

/* ======================================================================================
 * The online pairwise rotation of rotation-based quantizers (the comparison of Sec. 5.2):
 * ParoQuant-style methods turn each projection's input by a transform that cannot be folded
 * into the weights and so runs before every projection at every token (Sec. 1, Sec. 2).  LAQuant
 * has no such step; these two calls exist to measure what it costs beside the GEMV.  The paper
 * does not define the transform; the one computed here:
 *
 *   per group of 128 channels (the quantization groups), v = x * alpha (per channel), then for
 *   r = 0 .. rounds-1 and each of round r's 64 pairs (i, j) with angle t, in any order (a round's
 *   pairs are disjoint): (v_i, v_j) <- (v_i cos t - v_j sin t, v_i sin t + v_j cos t);
 *   Y = fp16(v), rounded once (fp32 arithmetic).
 * ====================================================================================== */

/* cs[2k] = cos(theta[k]), cs[2k + 1] = sin(theta[k]) for k < n (fp32; theta 4-byte aligned, cs
 * 8-byte aligned, device pointers; 0 <= n <= 2^31, LAQ_ERR_SHAPE otherwise).  Run once per set of
 * angles: the angles are parameters. */
laq_status laq_rotation_tables(const float *theta, int64_t n, void *cs, void *stream);

/* Y [M][K] fp16 = the rotation of X [M][K] fp16.
 *   alpha  fp16 [K] channel scales, or NULL for none;
 *   pairs  uint8 [K/128][rounds][64][2]: pair p of round r of group g is
 *          (pairs[g][r][p][0], pairs[g][r][p][1]), channels within the group; each round's 64
 *          pairs must partition 0..127 (not checked: indices are masked to 0..127, so other
 *          tables give wrong values but no access outside the group);
 *   cs     float [K/128][rounds][64][2] (cos, sin) of each pair's angle (laq_rotation_tables);
 *   rounds 0..16 (0: the scales alone; pairs and cs may then be NULL).
 * Device pointers, all 16-byte aligned (alpha too, when given); Y may equal X (in place).
 * M = 0: nothing.  Errors: LAQ_ERR_NULL, LAQ_ERR_SHAPE (M > 65535, K not a positive multiple of
 * 128, rounds outside 0..16), LAQ_ERR_ALIGN, LAQ_ERR_CUDA.  Launched with programmatic dependent
 * launch: the tables are read before the preceding kernel on the stream has finished. */
laq_status laq_pairwise_rotate(const void *X, int64_t M, int64_t K, const void *alpha,
                               const uint8_t *pairs, const void *cs, int32_t rounds, void *Y,
                               void *stream);

#ifdef __cplusplus
}
#endif

#endif /* LAQ_H */
