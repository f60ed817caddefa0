// rpd_internal.h - shared between the host entry points and the kernels' translation
// units: scratch layout, launch parameters and launcher declarations.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/rpd.h"

namespace rpd {

// Head-statistics tile: 128 rows (TMEM lanes) x 256 vocabulary columns, K-step 64.
constexpr int kTileM = 128;
constexpr int kTileN = 256;
constexpr int kTileK = 64;
constexpr int kStages = 4;
constexpr int kHeadThreads = 192;  // warp 0 TMA, warp 1 MMA + TMEM owner, warps 2-5 epilogue
constexpr int kStageBytesA = kTileM * kTileK * 2;
constexpr int kStageBytesB = kTileN * kTileK * 2;
constexpr int kHeadSmemBytes = kStages * (kStageBytesA + kStageBytesB) + 1024 + 256;
constexpr int kMaxBatch = 128;
constexpr int kMaxCanvas = 8192;
constexpr int kScoreThreads = 1024;
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // bounded mbarrier waits: 2 s

// Indices into the per-step device metadata words.
enum MetaIndex : int {
    kMetaMasked = 0,   // total masked positions over all canvases (NMT)
    kMetaRows = 1,     // projected rows R = K * NMT
    kMetaStatus = 2,   // RPD_OK or RPD_ERR_TIMEOUT, latched by kernels
    kMetaSplits = 3,   // vocabulary splits G chosen for the head kernel
    kMetaWords = 8
};

struct CompactParams {
    const uint8_t *mask;  // [B*N]
    int32_t *q_of_pos;    // [B*N] compact index or -1
    int32_t *pos_of_q;    // [B*N] flat position b*N+i of compact index q
    int32_t *canvas_off;  // [B+1]
    int32_t *meta;        // [kMetaWords]
    int B, N, K;
    int num_n_tiles;      // ceil(V / kTileN)
    int grid_ctas;        // CTAs of the head kernel
    int max_splits;       // capacity of the partial-statistics buffer per row
};

struct NormParams {
    const __nv_bfloat16 *hidden;  // [K][B*N][d]
    const __nv_bfloat16 *gain;    // [d]
    const int32_t *pos_of_q;
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
};

struct MergeParams {
    const float4 *partials;
    const int32_t *meta;
    int32_t *row_arg;   // [rows]
    float *row_pmax;    // [rows]
    float *row_H;       // [rows]
    int max_splits;
};

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
    float tau[kMaxBatch];
    float budget[kMaxBatch];
};

// Record the message returned by rpd_last_error() on this host thread.
void set_last_error(const char *msg);

cudaError_t launch_compact(const CompactParams &p, cudaStream_t s);
cudaError_t launch_gather_norm(const NormParams &p, int grid, cudaStream_t s);
cudaError_t launch_head_stats(const CUtensorMap &tmU, const CUtensorMap &tmW, const HeadParams &p,
                              int grid, cudaStream_t s);
cudaError_t launch_merge(const MergeParams &p, int grid, cudaStream_t s);
cudaError_t launch_score_commit(const ScoreParams &p, cudaStream_t s);

}  // namespace rpd
