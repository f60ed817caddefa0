// step_common.cuh - device routines shared by the step's small kernels: block scans, the
// head-tiling choice and the merge of per-split softmax statistics.
#pragma once

#include "rpd_internal.h"

namespace rpd {
namespace {

__device__ __forceinline__ int warp_inclusive_scan(int v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int t = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += t;
    }
    return v;
}

// Smallest time over vocabulary split counts g = 1..gmax of `row_tiles` x g work units on
// `slots` persistent CTAs (or pairs): waves x tiles-per-unit x `tile_cost`, the smallest g on
// ties.  Called by every thread of the CTA; the result is valid in every thread.
__device__ float best_split_count(float tile_cost, long long row_tiles, int slots, int num_n,
                                  int gmax, int &g_best) {
    __shared__ unsigned long long best;
    if (threadIdx.x == 0) best = ~0ull;
    __syncthreads();
    unsigned long long key = ~0ull;
    for (int g = threadIdx.x + 1; g <= gmax; g += blockDim.x) {
        const long long per = (num_n + g - 1) / g;
        const long long waves = (row_tiles * g + slots - 1) / slots;
        const float cost = static_cast<float>(waves * per) * tile_cost;
        const unsigned long long k = (static_cast<unsigned long long>(__float_as_uint(cost)) << 20) | g;
        key = k < key ? k : key;
    }
    atomicMin(&best, key);
    __syncthreads();
    const unsigned long long b = best;
    __syncthreads();  // `best` may be reused by the next call
    g_best = static_cast<int>(b & 0xFFFFFull);
    return __uint_as_float(static_cast<unsigned>(b >> 20));
}

// Time of one "rows on N" tile (256 vocabulary entries x a group of `ng` rows on a CTA pair)
// in units of a 128 x 256 tile's MMA work on one SM: the MMA work (ng/256 of a CTA-pair tile, plus the exposed epilogue
// when a group over 256 rows fills TMEM and cannot be double-buffered), or the operand bytes
// an SM receives per tile, (128 + ng/2) rows against the 384 of a 128 x 256 tile, whichever
// is larger.
__device__ __forceinline__ float swap_tile_cost(int ng) {
    const float mma = kPairTileCost * static_cast<float>(ng) / kPairTileM *
                      (ng > kPairTileM ? kSwapSingleBufferCost : 1.0f);
    const float feed = kSwapFeedCost * (kPairHalfRows + 0.5f * ng) / (kTileM + kTileN);
    return fmaxf(mma, feed);
}

__device__ __forceinline__ int swap_group_rows(long long rows, int groups) {
    const long long per = (rows + groups - 1) / groups;
    return static_cast<int>((per + kSwapRowStep - 1) / kSwapRowStep * kSwapRowStep);
}

// Head tiling for a pass of `rows` projected rows, chosen on the device (no host round-trip).
// Candidates, both on `pair_slots` CTA pairs: pair tiles of 256 rows; "rows on N" tiles with
// the rows in ceil(rows/512) equal groups (a group over 256 rows is single-buffered).  For each the split count comes from best_split_count, and the
// estimate is the larger of that MMA time and the head streaming time scaled by the vocabulary
// share of the largest split.  The cheapest candidate wins, or the one `force` names
// (RPD_TILING_*).  Called by every thread of the CTA; the results are valid in every thread.
// `mode` is kHeadModePair or kHeadModeRowsN; `splits` is the number of partials per row the
// merge reads: the vocabulary split count, twice it for rows on N (one per CTA of the pair);
// `swap_rows` is the rows-on-N group size (0 for pair tiles).
__device__ float choose_head_tiling(long long rows, int num_n, int max_splits, int pair_slots,
                                    float hbm_tiles, int force, int &mode, int &splits,
                                    int &swap_rows) {
    mode = kHeadModePair;
    splits = 1;
    swap_rows = 0;
    if (rows <= 0 || pair_slots <= 0) return 0.f;
    auto est_of = [&](float t, int g) {
        const float per = static_cast<float>((num_n + g - 1) / g);
        return fmaxf(t, hbm_tiles * per * g / num_n);
    };
    int g2;
    const float t2 = best_split_count(kPairTileCost, (rows + kPairTileM - 1) / kPairTileM, pair_slots,
                                      num_n, min(num_n, max_splits), g2);
    const float e2 = est_of(t2, g2);
    const int gmax3 = min(num_n, max_splits / 2);
    float e3 = 0.f, t3b = 0.f;
    int g3 = 0, ng3 = 0;
    if (gmax3 > 0) {
        // As few groups as possible: every group streams the whole head through its SMs, and
        // measured on GB300, groups of 256 rows or fewer (double-buffered, but carrying more
        // head bytes per MMA) never beat pair tiles, while larger groups do where pair tiles
        // pad heavily.
        const int groups = static_cast<int>((rows + kSwapMaxRows - 1) / kSwapMaxRows);
        const int ng = swap_group_rows(rows, groups);
        const float t = best_split_count(swap_tile_cost(ng), groups, pair_slots, num_n, gmax3, g3);
        e3 = est_of(t, g3);
        t3b = t;
        ng3 = ng;
    }
    // Equal estimates (both bound by streaming the head) go to the tiling with less MMA work.
    const bool rows_n = ng3 > 0 && force != RPD_TILING_PAIR &&
                        (force == RPD_TILING_ROWS_N || e3 < e2 || (e3 == e2 && t3b < t2));
    mode = rows_n ? kHeadModeRowsN : kHeadModePair;
    splits = rows_n ? 2 * g3 : g2;
    swap_rows = rows_n ? ng3 : 0;
    return rows_n ? e3 : e2;
}

// Running softmax statistics of one row over part of the vocabulary, in log2 units:
// m = max x, s = sum 2^(x-m), t = sum 2^(x-m) (x-m), a = argmax (lowest index).
struct Stat {
    float m, s, t;
    int a;
};

// Combine two partials: m = max, alpha = 2^(m_j - m), s = sum alpha s_j,
// t = sum alpha (t_j + (m_j - m) s_j); the argmax is the lowest index attaining m.
__device__ __forceinline__ Stat merge2(const Stat &x, const Stat &y) {
    if (y.s <= 0.f) return x;
    if (x.s <= 0.f) return y;
    Stat r;
    r.m = fmaxf(x.m, y.m);
    const float dx = x.m - r.m, dy = y.m - r.m;
    const float ax = exp2f(dx), ay = exp2f(dy);
    r.s = ax * x.s + ay * y.s;
    r.t = ax * fmaf(dx, x.s, x.t) + ay * fmaf(dy, y.s, y.t);
    r.a = (x.m > y.m) ? x.a : (y.m > x.m) ? y.a : min(x.a, y.a);
    return r;
}

constexpr float kLn2 = 0.6931471805599453f;

// Merge the split partials of the current projection pass's rows whose position index lies
// in [s_begin, s_end) of the pass's list, and store each row's argmax, its probability 1/s
// and the entropy H = ln s - ln2 * t / s (Eq. 1) at layer * NMT + q.  Rows are handled by
// groups of gs lanes, gs the smallest power of two keeping <= 8 partials per lane (at most
// a warp), so that every lane's loads are issued together; this CTA's groups take row
// slots first_group, first_group + group_stride, ... (in units of groups).  Returns how many
// of the cta_slots CTAs have rows to merge (the same value in every CTA).
__device__ int merge_pass_rows(const MergeArgs &mg, const int32_t *meta, const int32_t *sel_list,
                               int s_begin, int s_end, int cta_slot, int cta_slots) {
    const int rows = meta[kMetaRows];
    const int sel = meta[kMetaSel];
    if (rows <= 0 || sel <= 0 || s_end <= s_begin) return 0;
    const int layers = rows / sel;
    const int layer0 = meta[kMetaLayer0];
    const int nmt = meta[kMetaMasked];
    const int splits = meta[kMetaSplits];
    const int span = s_end - s_begin;
    const int total = layers * span;
    int gs = 1;
    while (gs < 32 && gs * 8 < splits) gs <<= 1;
    const int groups = blockDim.x / gs;
    const int gid = threadIdx.x / gs, gl = threadIdx.x % gs;
    for (int base = cta_slot * groups; base < total; base += cta_slots * groups) {  // uniform trips
        const int idx = base + gid;
        const bool valid = idx < total;
        Stat acc{-INFINITY, 0.f, 0.f, 0x7fffffff};
        int kr = 0, s = 0;
        if (valid) {
            kr = idx / span;
            s = s_begin + (idx - kr * span);
            const float4 *row = mg.partials + static_cast<size_t>(kr * sel + s) * mg.max_splits;
            for (int g0 = gl; g0 < splits; g0 += 8 * gs) {
                float4 v[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const int g = g0 + j * gs;
                    if (g < splits) v[j] = row[g];
                }
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const int g = g0 + j * gs;
                    if (g < splits) acc = merge2(acc, Stat{v[j].x, v[j].y, v[j].z, __float_as_int(v[j].w)});
                }
            }
        }
        for (int o = gs >> 1; o > 0; o >>= 1) {
            Stat other;
            other.m = __shfl_xor_sync(0xffffffffu, acc.m, o, gs);
            other.s = __shfl_xor_sync(0xffffffffu, acc.s, o, gs);
            other.t = __shfl_xor_sync(0xffffffffu, acc.t, o, gs);
            other.a = __shfl_xor_sync(0xffffffffu, acc.a, o, gs);
            acc = (gl & o) ? merge2(other, acc) : merge2(acc, other);  // fixed operand order
        }
        if (valid && gl == 0) {
            const size_t out = static_cast<size_t>(layer0 + kr) * nmt + (sel_list ? sel_list[s] : s);
            mg.row_arg[out] = acc.a;
            mg.row_pmax[out] = 1.0f / acc.s;
            mg.row_H[out] = fmaxf(logf(acc.s) - kLn2 * (acc.t / acc.s), 0.f);
        }
    }
    return min(cta_slots, (total + groups - 1) / groups);
}

}  // namespace
}  // namespace rpd
