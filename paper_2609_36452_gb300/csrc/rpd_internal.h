// rpd_internal.h - shared between the host entry points and the kernels' translation
// units: scratch layout, launch parameters and launcher declarations.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/rpd.h"

namespace rpd {

// Head-statistics tiles (tcgen05 cta_group::2: a cluster of two CTAs, one per SM, M = 256).
// Pair tiles: 256 rows x 256 vocabulary columns per pair; each CTA stages its own 128 rows of
// u and 128 rows of W per K-step of 64 (32 KB), 7 stages deep.
constexpr int kTileM = 128;   // rows of u per CTA (TMEM lanes) and the row padding unit of scratch
constexpr int kTileN = 256;   // vocabulary entries per tile
constexpr int kTileK = 64;
constexpr int kPairTileM = 256;
constexpr int kPairStages = 7;
constexpr int kPairHalfRows = 128;
constexpr int kPairStageBytesA = kPairHalfRows * kTileK * 2;
constexpr int kPairStageBytesB = kPairHalfRows * kTileK * 2;
// "Rows on N" tiles: a pair multiplies 256 vocabulary entries (128 per CTA, the MMA's M side)
// by a group of up to 512 projected rows (the N side, in steps of 32), so rows are padded to a
// multiple of 32 instead of a multiple of 256.  Each CTA stages its 128 head rows (16 KB) and
// half of the group's rows per K-step; the accumulators of groups of at most 256 rows are
// double-buffered in TMEM, groups of 288-320 rows go round a ring of 32-column TMEM chunks, and
// larger groups use columns [0, G) in turn.
constexpr int kSwapMaxRows = 512;
constexpr int kSwapRowStep = 32;  // N of the M = 256 MMA: a multiple of 32, at least 32
// At most 8 operand stages per CTA: small groups would fit 12, but with 12 the HBM-bound
// head streamed 2 % slower (20 rows: 0.158 against 0.153 ms) - the extra copies in flight
// bought nothing; 6 was slower again.  The barrier arrays are sized by this, so it must also
// cover the pair tiling's stages.
constexpr int kSwapMaxStages = 8;
constexpr int kSwapStageBytesA = kPairHalfRows * kTileK * 2;

constexpr int kSwapEpiWarps = 8;   // two per TMEM sub-partition, alternating its chunks
constexpr int kSwapXposeStride = 33;                             // floats per padded row
constexpr int kSwapXposeBytes = kSwapEpiWarps * 32 * kSwapXposeStride * 4;  // 32 x 32 fp32 per warp
// rows on N: running statistics [sub-partition][row of the group], 4 * ng float4
constexpr int kUBoxRows = 16;  // granularity of a half group's rows (the TMA box heights)
// Roles: warp 0 TMA, warp 1 MMA + TMEM owner, warps 2-9 epilogue (pair tiles use warps 2-5).
// At 128 registers a thread the CTA holds 40 K of an SM's 64 K registers, which leaves room for
// a CTA of the next kernel in the stream (launched early, waiting on this grid).
constexpr int kHeadKernelThreads = 64 + 32 * kSwapEpiWarps;
constexpr int kHeadBarrierBytes = 512;
// The pair tiles' operand ring, or the rows-on-N ring, transpose blocks and statistics (the
// ring takes what the other two leave): the 7-stage pair ring, 224 KB.
constexpr int kHeadRegionBytes = 224 * 1024;
static_assert(kPairStages <= kSwapMaxStages, "the stage barriers are shared by both tilings");
static_assert(kPairStages * (kPairStageBytesA + kPairStageBytesB) <= kHeadRegionBytes,
              "the pair tiles' operand ring fits the region");
static_assert(kHeadRegionBytes - kSwapXposeBytes - 4 * kSwapMaxRows * 16 >=
                  3 * (kSwapStageBytesA + (kSwapMaxRows / 2) * kTileK * 2),
              "a 512-row group still gets three stages");
// 1024-byte alignment slack + that region + barriers
constexpr int kHeadKernelSmemBytes = 1024 + kHeadRegionBytes + kHeadBarrierBytes;
static_assert(kHeadKernelSmemBytes <= 232448, "dynamic shared memory per CTA");
// Values of meta[kMetaHeadMode].
constexpr int kHeadModePair = 2;
constexpr int kHeadModeRowsN = 3;
constexpr int kMaxBatch = 128;
constexpr int kMaxCanvas = 8192;
constexpr int kScoreThreads = 1024;
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // bounded mbarrier waits: 2 s
constexpr long long kBandBytes = 32ll << 20;       // u tiles a band of head work units re-reads

// Indices into the per-step device metadata words.
enum MetaIndex : int {
    kMetaMasked = 0,   // total masked positions over all canvases (NMT)
    kMetaRows = 1,     // projected rows R = K * NMT
    kMetaStatus = 2,   // RPD_OK or RPD_ERR_TIMEOUT, latched by kernels
    kMetaSplits = 3,   // vocabulary splits G chosen for the head kernel
    kMetaHeadMode = 4, // kHeadModePair or kHeadModeRowsN: the pass's head tiling
    kMetaSel = 5,      // positions projected by the current pass
    kMetaLayer0 = 6,   // first window layer of the current pass (rows are layer-major)
    kMetaRowsTotal = 7,// rows projected by all passes of this step
    kMetaLazy = 8,     // 1 when this step projects lazily (two passes)
    kMetaUnitNext = 9, // next head work unit to claim (zeroed before each projection pass)
    kMetaMergeDone = 10, // CTAs that finished the fused merge-and-score (zeroed per step)
    kMetaSwapRows = 11,  // rows per row group of the "rows on N" tiling (mode 3)
    kMetaWords = 16
};

// Tiling plan of a projection pass (head_plan.h): which tiling the head kernel runs, with how
// many vocabulary splits.
struct HeadPlan {
    int mode;       // kHeadModePair or kHeadModeRowsN
    int splits;     // partials per row the merge reads (vocabulary splits; twice that for rows on N)
    int swap_rows;  // rows per group of the rows-on-N tiling (0 for pair tiles)
    float est;      // estimated time, in 128 x 256-tile units
};
struct HeadPlanInputs {
    int num_n;        // vocabulary tiles of 256
    int max_splits;   // partials per row the scratch holds
    int pair_slots;   // CTA pairs of the head kernel
    float hbm_tiles;  // time to stream the head once, in tile units
    int force;        // RPD_TILING_*
};
// Rows up to which a context tabulates the plan (larger passes evaluate it on the device).
constexpr int kPlanRows = 16384;

struct CompactParams {
    const uint8_t *mask;  // [B*N]
    int32_t *q_of_pos;    // [B*N] compact index or -1
    int32_t *pos_of_q;    // [B*N] flat position b*N+i of compact index q
    int32_t *canvas_off;  // [B+1]
    int32_t *meta;        // [kMetaWords]
    int B, N, K;
    HeadPlanInputs plan_in;
    const HeadPlan *plan; // [plan_rows + 1] plans by row count, or null
    int plan_rows;
    int block;            // 0: every masked position; > 0: only each canvas's active block
    int lazy;             // 0: all window layers; 1: lazy; 2: lazy when it is estimated cheaper
    int keep_status;      // 1: leave the status word as the previous call of the step left it
};

// Band fraction assumed when the device weighs lazy against full projection before the
// first pass (the real band is known only after it).
constexpr float kLazyBandGuess = 0.25f;

// Second pass of lazy projection: selects the positions whose final confidence lies in the
// stability band theta_c <= c < tau of their canvas and sets up the pass over their earlier
// window layers (tiling, split count, row mapping).
// Where merged per-row statistics go: split partials (log2 units) in, argmax / max
// probability / entropy per (layer, compact position) out, at layer * NMT + q.
struct MergeArgs {
    const float4 *partials;  // [rows][max_splits]
    int max_splits;
    int32_t *row_arg;
    float *row_pmax;
    float *row_H;
    // Vocabulary-sharded steps: when shard_out is set, each row's merged statistics themselves
    // (max, sum, tsum, argmax + v_offset) go to shard_out[layer * shard_stride + position]
    // instead of the derived outputs above.
    float4 *shard_out;
    const int32_t *pos_of_q;
    int shard_stride;
    int v_offset;
};

// Merge of the statistics of P vocabulary shards (rpd_step_shard_finish): per (layer k, masked
// position) the P records gathered[(p * K + k) * N + position], p = 0..P-1 in order, give the
// row's argmax, probability and entropy at k * NMT + q.
struct ShardMergeParams {
    const float4 *gathered;   // [P][K][B*N]
    int P, K, BN;
    const int32_t *pos_of_q;  // [NMT]
    const int32_t *meta;
    int32_t *row_arg;
    float *row_pmax;
    float *row_H;
};

struct BandParams {
    int32_t *meta;
    MergeArgs mg;              // merged first-pass statistics (final-layer confidences)
    const int32_t *pos_of_q;   // [NMT] flat position b*N+i of compact index q
    const int32_t *canvas_off; // [B+1] first compact index of each canvas
    int32_t *sel_q;            // out: compact indices of the band positions
    int32_t *band_off;         // out: [B+1] first band entry of each canvas
    int B, N, K;
    float theta_c;
    HeadPlanInputs plan_in;
    const HeadPlan *plan;
    int plan_rows;
    float tau[kMaxBatch];
};

// Costs of the tiling choice are in units of one 128-row x 256-entry tile's MMA work on one SM
// at the nominal rate below (24.4 us).  The per-tile costs are measured ones (LLaDA head,
// d = 4096, GB300, head time / tiles per pair, both tilings forced at 20 to 1024 rows):
//   pair tile (256 rows x 256 entries per pair): 22.3 us, 0.914 units;
//   rows-on-N tile (256 entries x a group of ng rows): 20.5 + 0.025 ng us (0.840 + 0.00102 ng
//   units) for ng <= 256, whose accumulators are double-buffered, and 4.9 + 0.0888 ng us
//   (0.201 + 0.00364 ng units) for larger groups (288 rows: 30.5 us, 416: 42.8 us, 512: 50.4 us).
// When streaming the head bounds a pass, pair tiles - half of whose staged bytes are rows of u -
// stream it about 4 % slower than rows-on-N tiles (20 rows: 0.159 against 0.153 ms).
constexpr float kPairTileCost = 0.914f;
constexpr float kSwapTileBase = 0.840f;
constexpr float kSwapTilePerRow = 0.00102f;
constexpr float kSwapWideTileBase = 0.201f;
constexpr float kSwapWideTilePerRow = 0.00364f;
constexpr float kPairStreamFactor = 1.04f;
// Per-SM MMA rate of the unit tile and the sustained HBM read rate used by the tiling choice
// (GB300 measurements; only their ratio matters).
constexpr double kSingleTileFlopsPerSm = 1.1e13;
constexpr double kHeadStreamBytesPerSec = 6.5e12;

// Row r of a projection pass: layer k = meta[kMetaLayer0] + r / S and position
// q = sel[r % S] (sel = the pass's list of compact indices, or the identity when null),
// S = meta[kMetaSel]; its merged statistics land at k * NMT + q.
struct NormParams {
    const __nv_bfloat16 *hidden;  // [K][B*N][d]
    const __nv_bfloat16 *gain;    // [d]
    const int32_t *pos_of_q;
    const int32_t *sel_list;      // null: every compact position
    const int32_t *meta;
    __nv_bfloat16 *u;             // [rows][d] compact head operand bf16(g*h)
    float *inv_rms;               // [rows]
    int BN, d;
    float eps;
};

struct HeadParams {
    const float *inv_rms;  // [rows]
    float4 *partials;      // [rows][max_splits]: (max, sum, tsum, argmax bits), log2 units
    int32_t *meta;
    int V, d, max_splits;
    uint64_t wait_limit_ns;  // bound on every mbarrier wait
    int stall;               // diagnostics: issue no loads (the waits run out)
    int w_tiled;             // W is the context's tiled copy (rpd_set_head_layout), else row-major
};

// Time to stream the head once, in units of one 128 x 256 tile's MMA time on one SM.
inline float head_stream_in_tiles(int V, int d, int num_sms) {
    (void)num_sms;
    const double t_hbm = 2.0 * V * static_cast<double>(d) / kHeadStreamBytesPerSec;
    const double t_tile = 2.0 * kTileM * kTileN * static_cast<double>(d) / kSingleTileFlopsPerSm;
    return static_cast<float>(t_hbm / t_tile);
}

struct ScoreParams {
    uint8_t *mask;              // [B][N] in/out
    const int32_t *q_of_pos;    // [B*N]
    const int32_t *canvas_off;  // [B+1]
    const int32_t *meta;
    const int32_t *row_arg;
    const float *row_pmax;
    const float *row_H;
    uint8_t *out_commit;        // [B][N]
    int32_t *out_token;         // [B][N]
    rpd_stats *out_stats;       // [B]
    rpd_debug dbg;
    int B, N, K;
    float theta_c, theta_s, w;
    int k_max, window;
    int block;                  // 0: full RPD; > 0: RPD-block (no budget, in-block fallback)
    int lazy;                   // 1: earlier window layers exist only for band positions
    float tau[kMaxBatch];
    float budget[kMaxBatch];
};

// Launch with programmatic stream serialisation, so that the kernel's prologue overlaps the
// tail of its predecessor in the stream (the kernel itself waits with griddepcontrol.wait
// before it reads what the predecessor wrote).
// Set on a host thread while it records launches that may not carry programmatic dependencies
// (a graph body that refuses them): the launches are then plainly stream-ordered, and the
// kernels' griddepcontrol instructions have nothing to wait for.
inline thread_local bool t_no_pdl = false;

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = t_no_pdl ? 0 : 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

// Bounds checks of the checked build (compiled with -DRPD_CHECKS): a failed check latches
// RPD_ERR_CHECK in the step's status word (`status`, device memory) and the guarded access is
// skipped; without RPD_CHECKS every check is `true` and compiles away.
#ifdef RPD_CHECKS
__device__ __forceinline__ bool rpd_check(bool ok, const int32_t *status) {
    if (!ok) atomicCAS(const_cast<int32_t *>(status), RPD_OK, RPD_ERR_CHECK);
    return ok;
}
#else
__device__ __forceinline__ bool rpd_check(bool, const int32_t *) { return true; }
#endif

// Record the message returned by rpd_last_error() on this host thread.
void set_last_error(const char *msg);

// ------------------------------------------------------------------ argument checks
// Shared by every entry point, so that they accept and refuse the same arguments.  Each
// returns nullptr when the argument is acceptable, else the message to report.

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Rule parameters (Table 4): theta_c, w finite and >= 0, theta_s not NaN, k_max, window >= 1,
// block >= 0.
inline const char *rule_error(const rpd_rule &r) {
    if (!(r.theta_c >= 0.f) || !(r.theta_c <= 3.402823466e38f)) return "theta_c must be finite and >= 0";
    if (r.theta_s != r.theta_s) return "theta_s is NaN";
    if (!(r.w >= 0.f) || !(r.w <= 3.402823466e38f)) return "w must be finite and >= 0";
    if (r.k_max < 1) return "k_max must be >= 1";
    if (r.window < 1) return "window must be >= 1";
    if (r.block < 0) return "block must be >= 0";
    return nullptr;
}

// Per-call thresholds: 0 < tau <= 1, theta_c < tau (Eq. 5 needs theta_c < theta_h), budget >= 0.
inline const char *call_error(const rpd_rule &r, float tau, float budget) {
    if (!(tau > 0.f && tau <= 1.f)) return "tau must be in (0, 1]";
    if (!(r.theta_c < tau)) return "theta_c must be below tau";
    if (!(budget >= 0.f)) return "budget must be >= 0";
    return nullptr;
}

// Memory the kernels read with TMA (the head, the gain) must be device or managed memory of
// `device`; memory the gather kernel reads with plain loads (hidden states) may also be
// page-locked host memory mapped into the device's address space.  Any other pointer - pageable
// host memory, another device's memory - would make the kernels fault, so it is refused.
inline bool pointer_usable(const void *p, int device, bool host_mapped_ok) {
    cudaPointerAttributes a{};
    const bool ok = cudaPointerGetAttributes(&a, p) == cudaSuccess &&
                    (((a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) &&
                      a.device == device) ||
                     (host_mapped_ok && a.type == cudaMemoryTypeHost && a.devicePointer == p));
    cudaGetLastError();  // clear the (non-sticky) error the query may have recorded
    return ok;
}

cudaError_t launch_compact(const CompactParams &p, cudaStream_t s);
cudaError_t launch_gather_norm(const NormParams &p, int grid, cudaStream_t s);
// Tensor maps of the head kernel's operands (128-byte swizzling, K boxes of 64): u in boxes of
// 128 rows (pair tiles) and, for the rows-on-N tiles, in boxes of 16, 32, ..., 128 rows (one
// per half-group height, so that a stage copies each MMA's share of u with one instruction:
// the TMA unit's time per copy, not its bytes, bounded a stage built from 16-row boxes); W in
// boxes of 128 rows.
constexpr int kUMaps = (kSwapMaxRows / 2) / kUBoxRows;  // box heights kUBoxRows * (1 .. kUMaps)
struct HeadMaps {
    CUtensorMap u;                // box 64 x 128 rows
    CUtensorMap w128;             // box 64 x 128 rows of W
    CUtensorMap u_rows[kUMaps];   // u_rows[j]: box 64 x kUBoxRows*(j+1) rows
};
// The head kernel (every tiling; the pass's choice is read from the meta words), launched as
// `grid` CTAs in clusters of two, one per SM.
cudaError_t launch_head(const HeadMaps &maps, const HeadParams &p, int grid, cudaStream_t s);
// Copy W [V][d] (d % 64 == 0) into blocks of 128 rows x 64 columns, block (t, k) at element
// ((t * (d / 64) + k) * 128) * 64, rows past V zero; Wt holds ceil(V/128)*128*d elements.
cudaError_t launch_tile_head(const void *W, void *Wt, int V, int d, cudaStream_t s);
// Largest number of clusters of the head kernel that can be resident at once.
int head_max_clusters();
cudaError_t launch_merge(const MergeArgs &mg, const int32_t *meta, const int32_t *sel_list,
                         int grid, cudaStream_t s);
cudaError_t launch_band(const BandParams &p, cudaStream_t s);
cudaError_t launch_score_commit(const ScoreParams &p, cudaStream_t s);
// Stop test of the decoding loop: counts the step and sets the loop's condition (one thread).
cudaError_t launch_loop_test(cudaGraphConditionalHandle handle, const rpd_stats *stats, int B, int N,
                             float stop_frac, int max_steps, int32_t *steps, cudaStream_t s);
cudaError_t launch_merge_shards(const ShardMergeParams &p, int grid, cudaStream_t s);
// The step's last merge fused with the scoring of its canvas (one canvas of at most
// kFuseScoreMaxN positions); the separate score launch is then skipped.
constexpr int kFuseScoreMaxN = 2048;
cudaError_t launch_merge_score(const MergeArgs &mg, int32_t *meta, const int32_t *sel_list,
                               int grid, const ScoreParams &p, cudaStream_t s);

}  // namespace rpd
