// head_plan.h - the choice of the head kernel's tiling and vocabulary split count for a
// projection pass of `rows` rows (host and device).  It changes no computed quantity, only
// how the contraction is laid out on the GPU.
//
// A context evaluates it on the host for every row count up to kPlanRows when it sizes its
// scratch and keeps the results in a device table, so that the step's compaction kernel - on
// the critical path of every step - only looks its row count up.  Passes with more rows (and
// the allocation-free entry point, which keeps no table) evaluate it on the device with one
// warp.
#pragma once

#include <cstring>

#include "rpd_internal.h"

namespace rpd {

static_assert(sizeof(HeadPlan) == 16, "a plan is one 16-byte table entry");

__host__ __device__ inline unsigned float_bits(float x) {
#ifdef __CUDA_ARCH__
    return __float_as_uint(x);
#else
    unsigned u;
    std::memcpy(&u, &x, sizeof(u));
    return u;
#endif
}

__host__ __device__ inline float bits_float(unsigned u) {
#ifdef __CUDA_ARCH__
    return __uint_as_float(u);
#else
    float x;
    std::memcpy(&x, &u, sizeof(x));
    return x;
#endif
}

// Smallest (time, g) over split counts g = g0, g0 + step, ... <= gmax of `tiles` x g work
// units on `slots` persistent pairs: waves x tiles-per-unit x tile_cost, packed so that the
// smaller key is the smaller time, then the smaller g.
__host__ __device__ inline unsigned long long best_split_key(float tile_cost, int tiles, int slots,
                                                             int num_n, int gmax, int g0, int step) {
    unsigned long long key = ~0ull;
    for (int g = g0; g <= gmax; g += step) {
        const int per = (num_n + g - 1) / g;
        const int waves = (tiles * g + slots - 1) / slots;
        const float cost = static_cast<float>(waves) * static_cast<float>(per) * tile_cost;
        const unsigned long long k = (static_cast<unsigned long long>(float_bits(cost)) << 20) |
                                     static_cast<unsigned>(g);
        key = k < key ? k : key;
    }
    return key;
}

// Time of one "rows on N" tile (256 vocabulary entries x a group of `ng` rows on a CTA pair)
// in tile units (the measured calibration of rpd_internal.h).
__host__ __device__ inline float swap_tile_cost(int ng) {
    return ng <= kPairTileM ? kSwapTileBase + kSwapTilePerRow * static_cast<float>(ng)
                            : kSwapWideTileBase + kSwapWideTilePerRow * static_cast<float>(ng);
}

// Rows-on-N groups of a pass: as few as possible (every group streams the whole head through
// its SMs; measured on GB300, groups of 256 rows or fewer never beat pair tiles), equal,
// padded to a multiple of kSwapRowStep.
__host__ __device__ inline int swap_groups(long long rows) {
    return static_cast<int>((rows + kSwapMaxRows - 1) / kSwapMaxRows);
}
__host__ __device__ inline int swap_group_rows(long long rows, int groups) {
    const long long per = (rows + groups - 1) / groups;
    return static_cast<int>((per + kSwapRowStep - 1) / kSwapRowStep * kSwapRowStep);
}

// The plan from the best keys of both tilings: each estimate is the larger of its MMA time and
// the head streaming time scaled by the vocabulary share of its largest split (and, for pair
// tiles, by their slower streaming); the cheaper wins (equal estimates go to the one with less
// MMA work), or the one `force` names.
__host__ __device__ inline HeadPlan plan_from_keys(const HeadPlanInputs &in, unsigned long long key2,
                                                   unsigned long long key3, int ng3) {
    auto est_of = [&](float t, int g, float stream) {
        const float per = static_cast<float>((in.num_n + g - 1) / g);
        const float hbm = stream * in.hbm_tiles * per * static_cast<float>(g) / static_cast<float>(in.num_n);
        return t > hbm ? t : hbm;
    };
    const int g2 = static_cast<int>(key2 & 0xFFFFFull);
    const float t2 = bits_float(static_cast<unsigned>(key2 >> 20));
    const float e2 = est_of(t2, g2, kPairStreamFactor);
    HeadPlan pair{kHeadModePair, g2, 0, e2};
    if (key3 == ~0ull || in.force == RPD_TILING_PAIR) return pair;
    const int g3 = static_cast<int>(key3 & 0xFFFFFull);
    const float t3 = bits_float(static_cast<unsigned>(key3 >> 20));
    const float e3 = est_of(t3, g3, 1.f);
    const bool rows_n = in.force == RPD_TILING_ROWS_N || e3 < e2 || (e3 == e2 && t3 < t2);
    return rows_n ? HeadPlan{kHeadModeRowsN, 2 * g3, ng3, e3} : pair;
}

// Host evaluation (and the device's, in one thread).
__host__ __device__ inline HeadPlan plan_head(long long rows, const HeadPlanInputs &in) {
    if (rows <= 0 || in.pair_slots <= 0) return HeadPlan{kHeadModePair, 1, 0, 0.f};
    const int tiles2 = static_cast<int>((rows + kPairTileM - 1) / kPairTileM);
    const int gmax2 = in.num_n < in.max_splits ? in.num_n : in.max_splits;
    const unsigned long long key2 =
        best_split_key(kPairTileCost, tiles2, in.pair_slots, in.num_n, gmax2, 1, 1);
    const int gmax3 = in.num_n < in.max_splits / 2 ? in.num_n : in.max_splits / 2;
    const int groups = swap_groups(rows);
    const int ng = swap_group_rows(rows, groups);
    const unsigned long long key3 =
        gmax3 > 0 ? best_split_key(swap_tile_cost(ng), groups, in.pair_slots, in.num_n, gmax3, 1, 1)
                  : ~0ull;
    return plan_from_keys(in, key2, key3, ng);
}

#ifdef __CUDACC__
// Device evaluation by one full warp (lanes share the split search); valid in every lane.
__device__ inline HeadPlan plan_head_warp(long long rows, const HeadPlanInputs &in) {
    if (rows <= 0 || in.pair_slots <= 0) return HeadPlan{kHeadModePair, 1, 0, 0.f};
    const int lane = threadIdx.x & 31;
    const int tiles2 = static_cast<int>((rows + kPairTileM - 1) / kPairTileM);
    const int gmax2 = in.num_n < in.max_splits ? in.num_n : in.max_splits;
    unsigned long long key2 =
        best_split_key(kPairTileCost, tiles2, in.pair_slots, in.num_n, gmax2, lane + 1, 32);
    const int gmax3 = in.num_n < in.max_splits / 2 ? in.num_n : in.max_splits / 2;
    const int groups = swap_groups(rows);
    const int ng = swap_group_rows(rows, groups);
    unsigned long long key3 =
        gmax3 > 0 ? best_split_key(swap_tile_cost(ng), groups, in.pair_slots, in.num_n, gmax3, lane + 1, 32)
                  : ~0ull;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long a = __shfl_xor_sync(0xffffffffu, key2, o);
        const unsigned long long b = __shfl_xor_sync(0xffffffffu, key3, o);
        key2 = a < key2 ? a : key2;
        key3 = b < key3 ? b : key3;
    }
    return plan_from_keys(in, key2, gmax3 > 0 ? key3 : ~0ull, ng);
}

// The plan of a pass: the context's table when it covers `rows`, else one warp evaluates it.
// Called by the first warp of the CTA.
__device__ inline HeadPlan lookup_plan(long long rows, const HeadPlan *table, int table_rows,
                                       const HeadPlanInputs &in) {
    if (table && rows <= table_rows) return table[rows];
    return plan_head_warp(rows, in);
}
#endif

}  // namespace rpd
