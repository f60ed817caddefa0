// k_head_stats.cu - the layerwise projection's contraction with online softmax statistics
// (logit lens of §2.2 / App. A.2 through the LM head; Eq. 1 needs only the final layer's
// entropy, Eq. 2-3 only each layer's argmax and its probability).
//
//   z[r][v] = inv_rms[r] * sum_d u[r][d] * W[v][d]
//
// is computed tile by tile on the 5th-generation tensor cores (tcgen05.mma kind::f16,
// bf16 operands staged in shared memory by TMA with 128-byte swizzling, fp32 accumulators
// in TMEM) and reduced in the epilogue straight out of TMEM into per-row running
// statistics in base-2 units (x = z * log2 e):
//   m = max x,  s = sum 2^(x-m),  t = sum 2^(x-m) (x-m),  a = argmax (lowest index).
// Logits never reach global memory.  Each work unit is (row tile, contiguous range of
// 256-wide vocabulary tiles); its statistics are written once per row as one partial
// (float4) that the merge kernel combines.
//
// One persistent kernel, launched as clusters of two CTAs (one per SM), serves two tilings;
// the compaction kernel picks one per projection pass on the device and the kernel reads it
// from the step's meta words.  Both run on CTA pairs (tcgen05 cta_group::2, M = 256):
//   pair tiles:  256 rows (M, 128 per CTA) x 256 vocabulary entries (N);
//   rows on N:   256 vocabulary entries (M, 128 per CTA) x a group of up to 512 rows (N,
//                padded to a multiple of 32), so that a pass whose row count is not a multiple
//                of 256 pads by at most 31 rows per group.
// Roles: warp 0 TMA producer (one thread), warp 1 TMEM owner (512 columns) and MMA issuer
// (the whole warp in the even CTA, one elected lane issuing), warps 2-9 epilogue (pair tiles
// use warps 2-5).  Every wait is
// bounded; a timeout latches RPD_ERR_TIMEOUT in the step's status word and the CTA drains and
// exits.
#include <atomic>

#include "ptx.cuh"
#include "rpd_internal.h"

namespace rpd {
namespace {

constexpr uint32_t kTmemCols = 2 * kTileN;
constexpr float kLog2e = 1.4426950408889634f;

// Work units (row tile m, vocabulary split g) in the order the persistent CTAs take them:
// row tiles are grouped into bands of `band` tiles; inside a band m runs fastest, then g.
// The units running at the same time therefore share W tiles (each streamed from HBM once
// per band) and re-read at most `band` u tiles (kept in L2 while the band runs).  With few
// row tiles there is a single band and the order is plain (m fastest).
struct TileWalk {
    int num_m, num_n, splits, units, band;
    __device__ __forceinline__ void init(int rows, int tile_rows, int V, int d, int g) {
        num_m = (rows + tile_rows - 1) / tile_rows;
        num_n = (V + kTileN - 1) / kTileN;
        splits = g;
        units = num_m * splits;
        const long long tile_bytes = static_cast<long long>(tile_rows) * d * 2;
        band = static_cast<int>(kBandBytes / tile_bytes);
        band = max(1, min(num_m, band));
    }
    __device__ __forceinline__ void unit(int u, int &m, int &g, int &n0, int &n1) const {
        const int per_band = band * splits;
        const int b = u / per_band;
        const int r = u - b * per_band;
        const int m0 = b * band;
        const int in_band = min(band, num_m - m0);
        m = m0 + r % in_band;
        g = r / in_band;
        n0 = static_cast<int>((static_cast<long long>(g) * num_n) / splits);
        n1 = static_cast<int>((static_cast<long long>(g + 1) * num_n) / splits);
    }
};

// Work units are claimed at run time from a per-pass counter (meta[kMetaUnitNext]) by the
// TMA producer, in the walk's order, so the units in flight are always a window of
// consecutive indices however the CTAs' speeds differ.  The producer passes each claimed
// index to the MMA issuer and the epilogue warps through a small ring in shared memory
// (-1: no unit left).
constexpr int kUnitRing = 4;

struct UnitCursor {
    int slot = 0;
    uint32_t phase = 0;
    __device__ __forceinline__ void advance() {
        if (++slot == kUnitRing) {
            slot = 0;
            phase ^= 1u;
        }
    }
};

// Fold one 32-entry chunk of logits, column col0 + i in v[i], into the running statistics
// (v is scaled to log2 units in place).
template <bool kFull>
__device__ __forceinline__ void fold_chunk(float (&x)[32], float scale, int col0, int V,
                                           float &run_m, float &run_s, float &run_t,
                                           int &run_a) {
    float cmax = -INFINITY;
    int carg = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        x[i] *= scale;
        if (!kFull && col0 + i >= V) x[i] = -INFINITY;
        if (x[i] > cmax) {
            cmax = x[i];
            carg = i;
        }
    }
    if (cmax > run_m) {
        if (run_s > 0.f) {
            const float dm = run_m - cmax;
            const float alpha = exp2f(dm);
            run_t = alpha * fmaf(dm, run_s, run_t);
            run_s = alpha * run_s;
        }
        run_m = cmax;
        run_a = col0 + carg;
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        if (kFull || col0 + i < V) {
            const float dl = x[i] - run_m;
            const float e = exp2f(dl);
            run_s += e;
            run_t = fmaf(e, dl, run_t);
        }
    }
}

// Combine two partial statistics (same rule as the merge kernel's): m = max, alpha =
// 2^(m_j - m), s = sum alpha s_j, t = sum alpha (t_j + (m_j - m) s_j), argmax the lowest index
// attaining m.
__device__ __forceinline__ float4 merge_stat(float4 x, float4 y) {
    if (y.y <= 0.f) return x;
    if (x.y <= 0.f) return y;
    const float m = fmaxf(x.x, y.x);
    const float dx = x.x - m, dy = y.x - m;
    const float ax = exp2f(dx), ay = exp2f(dy);
    const int a = (x.x > y.x) ? __float_as_int(x.w)
                : (y.x > x.x) ? __float_as_int(y.w) : min(__float_as_int(x.w), __float_as_int(y.w));
    return make_float4(m, ax * x.y + ay * y.y, ax * fmaf(dx, x.y, x.z) + ay * fmaf(dy, y.y, y.z),
                       __int_as_float(a));
}

// Shared memory of the head kernel: the operand ring (and for rows on N the transpose blocks
// and running statistics), then the barriers.
struct HeadSmem {
    uint8_t *ring;            // 1024-byte aligned

    uint64_t *full;           // [kSwapMaxStages] TMA -> MMA (in the even CTA for pair tilings)
    uint64_t *empty;          // [kSwapMaxStages] MMA -> TMA
    uint64_t *acc_full;       // [2] MMA -> epilogue
    uint64_t *acc_empty;      // [2] epilogue -> MMA (in the even CTA for pair tilings)
    uint64_t *drain;          // [1] MMA completion at exit
    uint64_t *unit_full;      // [kUnitRing] producer -> MMA, epilogue
    uint64_t *unit_empty;     // [kUnitRing] MMA, epilogue -> producer
    uint64_t *epi;            // [1] rows-on-N tiling: barrier of the epilogue warps
    uint64_t *chunk_free;     // [16] rows-on-N tiling: TMEM chunk read (in the even CTA)
    uint32_t *tmem_slot;
    volatile int *abort_flag;
    volatile int *unit_ring;  // [kUnitRing] claimed unit indices
};

__device__ __forceinline__ HeadSmem carve_smem(uint8_t *raw) {
    HeadSmem s;
    uint8_t *base = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(raw) + 1023) & ~static_cast<uintptr_t>(1023));
    s.ring = base;  // the rows-on-N tiles place their transpose blocks and statistics after their ring
    uint64_t *bars = reinterpret_cast<uint64_t *>(base + kHeadRegionBytes);
    s.full = bars;
    s.empty = bars + kSwapMaxStages;
    s.acc_full = bars + 2 * kSwapMaxStages;
    s.acc_empty = s.acc_full + 2;
    s.drain = s.acc_empty + 2;
    s.unit_full = s.drain + 1;
    s.unit_empty = s.unit_full + kUnitRing;
    s.epi = s.unit_empty + kUnitRing;
    s.chunk_free = s.epi + 1;
    s.tmem_slot = reinterpret_cast<uint32_t *>(s.chunk_free + kTmemCols / 32);
    s.abort_flag = reinterpret_cast<volatile int *>(s.tmem_slot + 1);
    s.unit_ring = s.abort_flag + 1;
    return s;
}

static_assert((2 * kSwapMaxStages + 6 + 2 * kUnitRing + kTmemCols / 32) * 8 + 8 + 4 * kUnitRing <=
                  kHeadBarrierBytes,
              "barrier region");

// ------------------------------------------------------------------------------------------
// Tiling 1: CTA pairs, rows on M (tcgen05 cta_group::2).  A pair (cluster of 2 CTAs) computes a tile of
// 256 rows x 256 vocabulary columns: CTA r of the pair stages rows [128r, 128r+128) of the row
// tile and W rows [128r, 128r+128) of the vocabulary tile; the even CTA issues
// tcgen05.mma.cta_group::2 with M=256, N=256, which reads both CTAs' shared memory and
// accumulates rows [128r, 128r+128) x all 256 columns into CTA r's TMEM.  Per SM and K-step
// that is 32 KB of operands for the MMA work a single CTA's 128 x 256 tile would need 48 KB for.
//
// Barriers: full[s] lives in the even CTA and receives both CTAs' TMA completions (tx bytes
// 64 KB per stage); empty[s], acc_full[a] and drain receive multicast commits from the MMA
// thread in both CTAs; acc_empty[a] lives in the even CTA and counts the 4 epilogue warps
// of both CTAs (8 arrivals).
__device__ __forceinline__ void head_pair(const CUtensorMap *tmU, const CUtensorMap *tmW,
                                          const HeadParams &p, const HeadSmem &sm, int rows,
                                          int splits) {
    constexpr int kStageBytes = kPairStageBytesA + kPairStageBytesB;
    uint64_t *full = sm.full, *empty = sm.empty, *acc_full = sm.acc_full,
             *acc_empty = sm.acc_empty, *unit_full = sm.unit_full, *unit_empty = sm.unit_empty;
    volatile int *abort_flag = sm.abort_flag;
    volatile int *unit_ring = sm.unit_ring;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();  // 0 = even CTA (issues the MMAs), 1 = odd

    if (threadIdx.x == 0) {
        for (int i = 0; i < kPairStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 8);
        }
        for (int i = 0; i < kUnitRing; ++i) {
            mbar_init(&unit_full[i], 1);
            // even CTA: its MMA issuer and 4 epilogue warps, the odd producer and 4 epilogue warps
            mbar_init(&unit_empty[i], 10);
        }
        mbar_init(sm.drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(tmU);
        tma_prefetch_desc(tmW);
    }
    if (warp == 1) tmem_alloc_pair(sm.tmem_slot, kTmemCols);
    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();  // both CTAs' barriers initialised before any cross-CTA signal
    tc_fence_after_sync();
    const uint32_t tmem_base = *sm.tmem_slot;

    TileWalk tw;
    tw.init(rows, kPairTileM, p.V, p.d, splits);
    const int num_kb = (p.d + kTileK - 1) / kTileK;

    if (warp == 0) {
        if (lane == 0 && !p.stall) {
            // ------------------------------------------------------- TMA producer (both CTAs)
            const uint32_t full0 = mapa_shared(smem_u32(&full[0]), 0);
            const uint32_t unit_full1 = mapa_shared(smem_u32(&unit_full[0]), 1);
            const uint32_t unit_ring1 = mapa_shared(smem_u32(const_cast<int *>(&unit_ring[0])), 1);
            const uint32_t unit_empty0 = mapa_shared(smem_u32(&unit_empty[0]), 0);
            int stage = 0;
            uint32_t phase = 0;
            long long fills = 0;
            bool ok = true;
            UnitCursor uc;
            while (ok) {
                int u;
                if (rank == 0) {
                    // claim the next unit and hand it to both CTAs
                    if (!mbar_wait_bounded_cluster(&unit_empty[uc.slot], uc.phase ^ 1u, abort_flag,
                                                   p.wait_limit_ns))
                        break;
                    const int claimed = atomicAdd(&p.meta[kMetaUnitNext], 1);
                    u = claimed < tw.units ? claimed : -1;
                    unit_ring[uc.slot] = u;
                    st_shared_cluster(unit_ring1 + static_cast<uint32_t>(uc.slot * sizeof(int)), u);
                    mbar_arrive(&unit_full[uc.slot]);
                    mbar_arrive_cluster(unit_full1 + static_cast<uint32_t>(uc.slot * sizeof(uint64_t)));
                } else {
                    if (!mbar_wait_bounded_cluster(&unit_full[uc.slot], uc.phase, abort_flag,
                                                   p.wait_limit_ns))
                        break;
                    u = unit_ring[uc.slot];
                    mbar_arrive_cluster(unit_empty0 + static_cast<uint32_t>(uc.slot * sizeof(uint64_t)));
                }
                uc.advance();
                if (u < 0) break;
                int m, g, n0, n1;
                tw.unit(u, m, g, n0, n1);
                for (int n = n0; ok && n < n1; ++n) {
                    for (int kb = 0; kb < num_kb; ++kb) {
                        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_flag, p.wait_limit_ns)) {
                            ok = false;
                            break;
                        }
                        if (rank == 0) mbar_arrive_expect_tx(&full[stage], 2 * kStageBytes);
                        const uint32_t fb = full0 + static_cast<uint32_t>(stage * sizeof(uint64_t));
                        uint8_t *st = sm.ring + stage * kStageBytes;
                        tma_load_2d_pair(st, tmU, fb, kb * kTileK,
                                         m * kPairTileM + static_cast<int>(rank) * kPairHalfRows);
                        if (p.w_tiled)  // block (2n + rank, kb): 128 contiguous rows of 64
                            tma_load_2d_pair(st + kPairStageBytesA, tmW, fb, 0,
                                             ((2 * n + static_cast<int>(rank)) * num_kb + kb) * kPairHalfRows);
                        else
                            tma_load_2d_pair(st + kPairStageBytesA, tmW, fb, kb * kTileK,
                                             n * kTileN + static_cast<int>(rank) * kPairHalfRows);
                        ++fills;
                        if (++stage == kPairStages) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                }
            }
            // Drain: a stage's copy has landed once the MMAs that read it have completed, which
            // the multicast commit on empty[s] reports in this CTA.
            for (int s = 0; s < kPairStages; ++s) {
                const long long n_s = fills / kPairStages + (s < fills % kPairStages ? 1 : 0);
                if (n_s > 0)
                    mbar_wait_drain(&empty[s], static_cast<uint32_t>((n_s - 1) & 1), p.wait_limit_ns / 8);
            }
        }
    } else if (warp == 1) {
        if (rank == 0) {
            // -------------------------------------------- MMA issuer (even CTA only): the whole
            // warp runs the loop, one elected lane issues (every branch below is warp-uniform)
            constexpr uint32_t idesc = idesc_bf16_f32(kPairTileM, kTileN);
            int stage = 0;
            uint32_t phase = 0;
            uint32_t tile_iter = 0;
            bool ok = true;
            UnitCursor uc;
            while (ok) {
                if (!mbar_wait_bounded_warp(&unit_full[uc.slot], uc.phase, abort_flag, p.wait_limit_ns))
                    break;
                const int u = unit_ring[uc.slot];
                __syncwarp();
                if (lane == 0) mbar_arrive(&unit_empty[uc.slot]);
                uc.advance();
                if (u < 0) break;
                int m, g, n0, n1;
                tw.unit(u, m, g, n0, n1);
                for (int n = n0; ok && n < n1; ++n, ++tile_iter) {
                    const uint32_t acc = tile_iter & 1u;
                    const uint32_t acc_phase = (tile_iter >> 1) & 1u;
                    if (!mbar_wait_bounded_warp(&acc_empty[acc], acc_phase ^ 1u, abort_flag,
                                                p.wait_limit_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t d_tmem = tmem_base + acc * kTileN;
                    for (int kb = 0; kb < num_kb; ++kb) {
                        if (!mbar_wait_bounded_warp(&full[stage], phase, abort_flag, p.wait_limit_ns)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after_sync();
                        const uint32_t a0 = smem_u32(sm.ring + stage * kStageBytes);
                        const uint32_t b0 = a0 + kPairStageBytesA;
#pragma unroll
                        for (int kk = 0; kk < kTileK / 16; ++kk) {
                            umma_bf16_pair_warp(d_tmem, smem_desc_sw128(a0 + kk * 32),
                                                smem_desc_sw128(b0 + kk * 32), idesc,
                                                (kb > 0 || kk > 0) ? 1u : 0u);
                        }
                        umma_commit_pair_multicast_warp(&empty[stage], 0x3);
                        if (++stage == kPairStages) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                    if (!ok) break;
                    umma_commit_pair_multicast_warp(&acc_full[acc], 0x3);
                }
            }
            umma_commit_pair_multicast_warp(sm.drain, 0x3);
        }
        // Both CTAs: every MMA writing this CTA's TMEM has completed before it is freed.
        if (lane == 0) mbar_wait_drain(sm.drain, 0, p.wait_limit_ns);
        __syncwarp();
    } else if (warp < 6) {
        // ---------------------------------------------------------- epilogue (both CTAs)
        const int sub = warp & 3;
        const int row_in_tile = static_cast<int>(rank) * kPairHalfRows + sub * 32 + lane;
        const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(sub * 32) << 16);
        const uint32_t acc_empty0 = mapa_shared(smem_u32(&acc_empty[0]), 0);
        const uint32_t unit_empty0 = mapa_shared(smem_u32(&unit_empty[0]), 0);
        uint32_t tile_iter = 0;
        bool ok = true;
        UnitCursor uc;
        while (ok) {
            if (!mbar_wait_bounded_cluster(&unit_full[uc.slot], uc.phase, abort_flag, p.wait_limit_ns))
                break;
            const int u = unit_ring[uc.slot];
            __syncwarp();
            if (lane == 0)
                mbar_arrive_cluster(unit_empty0 + static_cast<uint32_t>(uc.slot * sizeof(uint64_t)));
            uc.advance();
            if (u < 0) break;
            int m, g, n0, n1;
            tw.unit(u, m, g, n0, n1);
            const int r = m * kPairTileM + row_in_tile;
            const bool valid = r < rows;
            const float scale = valid ? p.inv_rms[r] * kLog2e : 0.f;
            float run_m = -INFINITY, run_s = 0.f, run_t = 0.f;
            int run_a = 0;
            for (int n = n0; n < n1; ++n, ++tile_iter) {
                const uint32_t acc = tile_iter & 1u;
                const uint32_t acc_phase = (tile_iter >> 1) & 1u;
                if (!mbar_wait_bounded(&acc_full[acc], acc_phase, abort_flag, p.wait_limit_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                const int col_base = n * kTileN;
                const bool full_tile = col_base + kTileN <= p.V;
#pragma unroll 1
                for (int c = 0; c < kTileN / 32; ++c) {
                    float v[32];
                    tmem_ld_32x32b_x32(lane_base + acc * kTileN + c * 32, v);
                    if (full_tile)
                        fold_chunk<true>(v, scale, col_base + c * 32, p.V, run_m, run_s, run_t, run_a);
                    else
                        fold_chunk<false>(v, scale, col_base + c * 32, p.V, run_m, run_s, run_t, run_a);
                }
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(acc_empty0 + acc * static_cast<uint32_t>(sizeof(uint64_t)));
            }
            if (!ok) break;
            if (valid && rpd_check(g < p.max_splits, p.meta + kMetaStatus)) {
                p.partials[static_cast<size_t>(r) * p.max_splits + g] =
                    make_float4(run_m, run_s, run_t, __int_as_float(run_a));
            }
        }
    }

    __syncwarp();
    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();  // no signal may still be in flight to a CTA that is about to exit
    tc_fence_after_sync();
    if (*abort_flag && threadIdx.x == 0) atomicExch(&p.meta[kMetaStatus], RPD_ERR_TIMEOUT);
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc_pair(tmem_base, kTmemCols);
    }
}

// Barrier of the rows-on-N epilogue's threads: every thread arrives (release) and waits
// for the phase (acquire), bounded like every other wait.  Returns false if it gave up.
__device__ __forceinline__ bool epi_sync(uint64_t *bar, uint32_t &phase, volatile int *abort,
                                         uint64_t limit_ns) {
    mbar_arrive(bar);
    const bool ok = mbar_wait_bounded(bar, phase, abort, limit_ns);
    phase ^= 1u;
    return ok;
}

// ------------------------------------------------------------------------------------------
// Tiling 2: "rows on N" CTA pairs.  The pair's MMA (cta_group::2, M = 256) takes the head as
// its A operand - CTA r stages vocabulary rows [256n + 128r, +128) of tile n, 16 KB per
// K-step - and a group of G rows of u as its B operand (N = G, a multiple of 32 up to 512).
// So CTA r's TMEM holds logits for 128 vocabulary entries (lanes) x the group's rows
// (columns): per row the softmax statistics reduce across lanes.
//
// Operands: each CTA stages its half of the group (rows [r G/2, +G/2)) as one TMA copy per
// stage, from the tensor map whose box has that height (16 to 256 rows; a stage with a second,
// small copy measured far slower).
//
// TMEM: 16 chunks of 32 columns.  A tile of at most 256 columns alternates between the two
// halves (double buffering); a tile of 288 or 320 columns follows its predecessor around the
// ring of chunks, so that it waits only for the chunks it overwrites (with 288 columns, the
// first two of its predecessor's nine) instead of for the whole epilogue of its predecessor;
// larger tiles use columns [0, G) in turn.  A tile's columns are issued as one MMA per
// contiguous segment of at most 256 columns per 16-wide K-step, and the MMA for columns
// [c, c + N) of segment j takes the first N/2 of them from rows [o_j, o_j + N/2) of the even
// CTA's half and the rest from the same rows of the odd CTA's half, o_j being half the columns
// of the tile before segment j; the epilogue maps each column back to its row.
//
// Epilogue: 8 warps, two per TMEM sub-partition, alternating its chunks.  A warp loads a
// 32 x 32 block, releases the chunk (ring tiles), transposes the block through shared memory
// so that each thread holds one row's 32 vocabulary entries, and folds them into that row's
// running statistics (per sub-partition, in shared memory).  At the end of a work unit the
// four sub-partitions' statistics of each row are combined and each CTA writes one partial
// per row (the merge sees 2 partials per split).
// The K-steps of one rows-on-N tile issued as kSegs MMAs per 16-wide step (one per column
// segment), run by the whole issuing warp.  A separate loop per segment count keeps the loop
// free of branches: with the segment tests inside it a tile measured 60 % slower.
template <int kSegs>
__device__ __forceinline__ bool swap_tile_mmas(const HeadSmem &sm, int num_kb, int stages,
                                               int stage_bytes, int &stage, uint32_t &phase,
                                               uint32_t d0, uint32_t d1, uint32_t d2, uint32_t id0,
                                               uint32_t id1, uint32_t id2, uint32_t bo1,
                                               uint32_t bo2, volatile int *abort_flag,
                                               uint64_t limit) {
    for (int kb = 0; kb < num_kb; ++kb) {
        if (!mbar_wait_bounded_warp(&sm.full[stage], phase, abort_flag, limit)) return false;
        tc_fence_after_sync();
        const uint32_t a0 = smem_u32(sm.ring + stage * stage_bytes);
        const uint32_t b0 = a0 + kSwapStageBytesA;
#pragma unroll
        for (int kk = 0; kk < kTileK / 16; ++kk) {
            const uint32_t accum = (kb > 0 || kk > 0) ? 1u : 0u;
            umma_bf16_pair_warp(d0, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(b0 + kk * 32), id0, accum);
            if (kSegs > 1)
                umma_bf16_pair_warp(d1, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(b0 + bo1 + kk * 32),
                                    id1, accum);
            if (kSegs > 2)
                umma_bf16_pair_warp(d2, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(b0 + bo2 + kk * 32),
                                    id2, accum);
        }
        umma_commit_pair_multicast_warp(&sm.empty[stage], 0x3);
        if (++stage == stages) {
            stage = 0;
            phase ^= 1u;
        }
    }
    return true;
}

// Column segments of a rows-on-N tile placed at TMEM chunk c0: up to three contiguous column
// ranges, each within [0, 512) and at most 256 wide (the MMA's N).
struct SwapSegs {
    int col0, col1, col2;  // first TMEM column of each
    int n0, n1, n2;        // widths (0: unused)
};
__device__ __forceinline__ SwapSegs swap_segments(int c0, int ng) {
    SwapSegs g;
    g.col0 = c0 * 32;
    g.n0 = min(min(ng, kTmemCols - g.col0), kPairTileM);
    g.col1 = (g.col0 + g.n0) % kTmemCols;
    g.n1 = min(min(ng - g.n0, kTmemCols - g.col1), kPairTileM);
    g.col2 = (g.col1 + g.n1) % kTmemCols;
    g.n2 = ng - g.n0 - g.n1;
    return g;
}

__device__ __forceinline__ void head_swap(const CUtensorMap *tmUrows /* [kUMaps] */,
                                          const CUtensorMap *tmW,
                                          const HeadParams &p, const HeadSmem &sm, int rows,
                                          int splits, int ng) {
    uint64_t *full = sm.full, *empty = sm.empty, *acc_full = sm.acc_full,
             *acc_empty = sm.acc_empty, *unit_full = sm.unit_full, *unit_empty = sm.unit_empty,
             *chunk_free = sm.chunk_free;
    volatile int *abort_flag = sm.abort_flag;
    volatile int *unit_ring = sm.unit_ring;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    // TMEM placement: tiles of at most 256 columns alternate between the two halves; tiles of
    // 288 to 320 columns follow one another around a ring of 16 chunks of 32 columns; larger
    // tiles use all of TMEM in turn (with 11 or more chunks a tile would wait for nearly all of
    // its predecessor's chunks anyway, and the ring's column splits measured slower there)
    constexpr uint32_t kChunks = kTmemCols / 32;
    constexpr uint32_t kRingMaxChunks = 10;
    const uint32_t nch = static_cast<uint32_t>(ng / 32);
    const bool single = nch > kRingMaxChunks;
    const bool ring = 2 * nch > kChunks && !single;
    const int stage_b = (ng / 2) * kTileK * 2;
    const int stage_bytes = kSwapStageBytesA + stage_b;
    // region: operand ring (as many stages as fit), transpose blocks, statistics [4][ng]
    int stages = (kHeadRegionBytes - kSwapXposeBytes - 4 * ng * 16) / stage_bytes;
    stages = stages < kSwapMaxStages ? stages : kSwapMaxStages;
    float *xpose = reinterpret_cast<float *>(sm.ring + stages * stage_bytes);
    float4 *stats = reinterpret_cast<float4 *>(sm.ring + stages * stage_bytes + kSwapXposeBytes);
    constexpr int kEpiThreads = 32 * kSwapEpiWarps;

    if (threadIdx.x == 0) {
        for (int i = 0; i < stages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 2 * kSwapEpiWarps);
        }
        for (int i = 0; i < kUnitRing; ++i) {
            mbar_init(&unit_full[i], 1);
            // even CTA: its MMA issuer and epilogue warps; odd CTA: its producer and epilogue warps
            mbar_init(&unit_empty[i], 2 + 2 * kSwapEpiWarps);
        }
        // ring tiles: a chunk is read by one warp per TMEM sub-partition in each CTA
        for (uint32_t i = 0; i < kChunks; ++i) mbar_init(&chunk_free[i], 8);
        mbar_init(sm.epi, kEpiThreads);
        mbar_init(sm.drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tmUrows[(ng / 2) / kUBoxRows - 1]);
        tma_prefetch_desc(tmW);
    }
    if (warp == 1) tmem_alloc_pair(sm.tmem_slot, kTmemCols);
    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();
    tc_fence_after_sync();
    const uint32_t tmem_base = *sm.tmem_slot;

    TileWalk tw;
    tw.init(rows, ng, p.V, p.d, splits);
    const int num_kb = (p.d + kTileK - 1) / kTileK;

    if (warp == 0) {
        if (lane == 0 && !p.stall) {
            // ------------------------------------------------------- TMA producer (both CTAs)
            const uint32_t full0 = mapa_shared(smem_u32(&full[0]), 0);
            const uint32_t unit_full1 = mapa_shared(smem_u32(&unit_full[0]), 1);
            const uint32_t unit_ring1 = mapa_shared(smem_u32(const_cast<int *>(&unit_ring[0])), 1);
            const uint32_t unit_empty0 = mapa_shared(smem_u32(&unit_empty[0]), 0);
            // this CTA's half of the group's rows, one copy: the map whose box is that many rows
            // high (rows [rank * half, +half) of the group; see the epilogue's row order)
            const int half = ng / 2;
            const CUtensorMap *umap = &tmUrows[half / kUBoxRows - 1];
            int stage = 0;
            uint32_t phase = 0;
            long long fills = 0;
            bool ok = true;
            UnitCursor uc;
            while (ok) {
                int u;
                if (rank == 0) {
                    if (!mbar_wait_bounded_cluster(&unit_empty[uc.slot], uc.phase ^ 1u, abort_flag,
                                                   p.wait_limit_ns))
                        break;
                    const int claimed = atomicAdd(&p.meta[kMetaUnitNext], 1);
                    u = claimed < tw.units ? claimed : -1;
                    unit_ring[uc.slot] = u;
                    st_shared_cluster(unit_ring1 + static_cast<uint32_t>(uc.slot * sizeof(int)), u);
                    mbar_arrive(&unit_full[uc.slot]);
                    mbar_arrive_cluster(unit_full1 + static_cast<uint32_t>(uc.slot * sizeof(uint64_t)));
                } else {
                    if (!mbar_wait_bounded_cluster(&unit_full[uc.slot], uc.phase, abort_flag,
                                                   p.wait_limit_ns))
                        break;
                    u = unit_ring[uc.slot];
                    mbar_arrive_cluster(unit_empty0 + static_cast<uint32_t>(uc.slot * sizeof(uint64_t)));
                }
                uc.advance();
                if (u < 0) break;
                int m, g, v0, v1;
                tw.unit(u, m, g, v0, v1);
                const int urow = m * ng + static_cast<int>(rank) * half;
                const int w_off = static_cast<int>(rank) * kPairHalfRows;
                for (int n = v0; ok && n < v1; ++n) {
                    for (int kb = 0; kb < num_kb; ++kb) {
                        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_flag, p.wait_limit_ns)) {
                            ok = false;
                            break;
                        }
                        if (rank == 0) mbar_arrive_expect_tx(&full[stage], 2 * stage_bytes);
                        const uint32_t fb = full0 + static_cast<uint32_t>(stage * sizeof(uint64_t));
                        uint8_t *st = sm.ring + stage * stage_bytes;
                        const int x = kb * kTileK;
                        if (p.w_tiled)  // block (2n + rank, kb): 128 contiguous rows of 64
                            tma_load_2d_pair(st, tmW, fb, 0,
                                             ((2 * n + static_cast<int>(rank)) * num_kb + kb) * kPairHalfRows);
                        else
                            tma_load_2d_pair(st, tmW, fb, x, n * kTileN + w_off);
                        tma_load_2d_pair(st + kSwapStageBytesA, umap, fb, x, urow);
                        ++fills;
                        if (++stage == stages) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                }
            }
            for (int s = 0; s < stages; ++s) {
                const long long n_s = fills / stages + (s < fills % stages ? 1 : 0);
                if (n_s > 0)
                    mbar_wait_drain(&empty[s], static_cast<uint32_t>((n_s - 1) & 1), p.wait_limit_ns / 8);
            }
        }
    } else if (warp == 1) {
        if (rank == 0) {
            // -------------------------------------------- MMA issuer (even CTA only): the whole
            // warp runs the loop, one elected lane issues (every branch below is warp-uniform)
            int stage = 0;
            uint32_t phase = 0;
            uint32_t tile_iter = 0;
            bool ok = true;
            UnitCursor uc;
            while (ok) {
                if (!mbar_wait_bounded_warp(&unit_full[uc.slot], uc.phase, abort_flag, p.wait_limit_ns))
                    break;
                const int u = unit_ring[uc.slot];
                __syncwarp();
                if (lane == 0) mbar_arrive(&unit_empty[uc.slot]);
                uc.advance();
                if (u < 0) break;
                int m, g, v0, v1;
                tw.unit(u, m, g, v0, v1);
                for (int n = v0; ok && n < v1; ++n, ++tile_iter) {
                    // tile t-2 read (its accumulator barrier is reused), or tile t-1 for tiles
                    // that use all of TMEM ...
                    const uint32_t acc = single ? 0u : (tile_iter & 1u);
                    const uint32_t acc_phase = (single ? tile_iter : (tile_iter >> 1)) & 1u;
                    if (!mbar_wait_bounded_warp(&acc_empty[acc], acc_phase ^ 1u, abort_flag,
                                                p.wait_limit_ns)) {
                        ok = false;
                        break;
                    }
                    // ... and, on the ring, the chunks of tile t-1 this tile overwrites
                    const uint32_t a0 = tile_iter * nch;
                    if (ring && tile_iter > 0) {
                        for (uint32_t c = kChunks - nch; ok && c < nch; ++c) {
                            const uint32_t a = a0 + c;  // previous use: a - 16, in tile t-1
                            if (!mbar_wait_bounded_warp(&chunk_free[a % kChunks], ((a / kChunks) & 1u) ^ 1u,
                                                        abort_flag, p.wait_limit_ns))
                                ok = false;
                        }
                        if (!ok) break;
                    }
                    tc_fence_after_sync();
                    const SwapSegs sg = swap_segments(static_cast<int>(ring ? a0 % kChunks : acc * 8u), ng);
                    // (single: acc = 0, the tile starts at column 0)
                    const uint32_t d0 = tmem_base + sg.col0, d1 = tmem_base + sg.col1,
                                   d2 = tmem_base + sg.col2;
                    const uint32_t id0 = idesc_bf16_f32(kPairTileM, sg.n0);
                    const uint32_t id1 = idesc_bf16_f32(kPairTileM, sg.n1 > 0 ? sg.n1 : 32);
                    const uint32_t id2 = idesc_bf16_f32(kPairTileM, sg.n2 > 0 ? sg.n2 : 32);
                    // segment j's rows of u start at row (columns before it) / 2 of each CTA's half
                    const uint32_t bo1 = static_cast<uint32_t>((sg.n0 / 2) * kTileK * 2);
                    const uint32_t bo2 = static_cast<uint32_t>(((sg.n0 + sg.n1) / 2) * kTileK * 2);
                    ok = sg.n2 > 0 ? swap_tile_mmas<3>(sm, num_kb, stages, stage_bytes, stage, phase, d0, d1,
                                                       d2, id0, id1, id2, bo1, bo2, abort_flag,
                                                       p.wait_limit_ns)
                       : sg.n1 > 0 ? swap_tile_mmas<2>(sm, num_kb, stages, stage_bytes, stage, phase, d0,
                                                       d1, d2, id0, id1, id2, bo1, bo2, abort_flag,
                                                       p.wait_limit_ns)
                                   : swap_tile_mmas<1>(sm, num_kb, stages, stage_bytes, stage, phase, d0,
                                                       d1, d2, id0, id1, id2, bo1, bo2, abort_flag,
                                                       p.wait_limit_ns);
                    if (!ok) break;
                    umma_commit_pair_multicast_warp(&acc_full[acc], 0x3);
                }
            }
            umma_commit_pair_multicast_warp(sm.drain, 0x3);
        }
        if (lane == 0) mbar_wait_drain(sm.drain, 0, p.wait_limit_ns);
        __syncwarp();
    } else {
        // ---------------------------------------------------------- epilogue (both CTAs)
        const int sub = warp & 3;                 // TMEM sub-partition (lanes 32*sub..+31)
        const int etid = (warp - 2) * 32 + lane;  // 0 .. kEpiThreads-1
        const int chunk0 = (warp - 2) / 4;        // the two warps of a sub-partition alternate chunks
        constexpr int kChunkStep = kSwapEpiWarps / 4;
        const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(sub * 32) << 16);
        const uint32_t acc_empty0 = mapa_shared(smem_u32(&acc_empty[0]), 0);
        const uint32_t chunk_free0 = mapa_shared(smem_u32(&chunk_free[0]), 0);
        const uint32_t unit_empty0 = mapa_shared(smem_u32(&unit_empty[0]), 0);
        float *xp = xpose + (warp - 2) * 32 * kSwapXposeStride;
        const float4 kEmpty = make_float4(-INFINITY, 0.f, 0.f, __int_as_float(0));
        for (int i = etid; i < 4 * ng; i += kEpiThreads) stats[i] = kEmpty;
        uint32_t epi_phase = 0;
        uint32_t tile_iter = 0;
        bool ok = epi_sync(sm.epi, epi_phase, abort_flag, p.wait_limit_ns);
        UnitCursor uc;
        while (ok) {
            if (!mbar_wait_bounded_cluster(&unit_full[uc.slot], uc.phase, abort_flag, p.wait_limit_ns))
                break;
            const int u = unit_ring[uc.slot];
            __syncwarp();
            if (lane == 0)
                mbar_arrive_cluster(unit_empty0 + static_cast<uint32_t>(uc.slot * sizeof(uint64_t)));
            uc.advance();
            if (u < 0) break;
            int m, g, v0, v1;
            tw.unit(u, m, g, v0, v1);
            for (int n = v0; n < v1; ++n, ++tile_iter) {
                const uint32_t acc = single ? 0u : (tile_iter & 1u);
                const uint32_t acc_phase = (single ? tile_iter : (tile_iter >> 1)) & 1u;
                if (!mbar_wait_bounded(&acc_full[acc], acc_phase, abort_flag, p.wait_limit_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                const uint32_t c0 = ring ? (tile_iter * nch) % kChunks : acc * 8u;
                const SwapSegs sg = swap_segments(static_cast<int>(c0), ng);
                const int x1 = sg.n0, x2 = sg.n0 + sg.n1;
                // the 32 vocabulary entries of this warp's sub-partition
                const int vbase = n * kTileN + static_cast<int>(rank) * kPairHalfRows + sub * 32;
                const bool full_tile = vbase + 32 <= p.V;
#pragma unroll 1
                for (int c = chunk0; c < static_cast<int>(nch); c += kChunkStep) {
                    float v[32];
                    const uint32_t slot = (c0 + static_cast<uint32_t>(c)) % kChunks;
                    tmem_ld_32x32b_x32(lane_base + slot * 32, v);
                    if (ring) {  // the chunk's columns may be overwritten by the next tile now
                        tc_fence_before_sync();
                        __syncwarp();
                        if (lane == 0) mbar_arrive_cluster(chunk_free0 + slot * static_cast<uint32_t>(sizeof(uint64_t)));
                    }
                    // thread `lane` holds vocabulary entry vbase + lane for rows c*32 + i; write
                    // it as row `lane` of a block padded to 33 floats a row (bank lane + i: no
                    // conflict) and read back column `lane` (bank i + lane: no conflict)
#pragma unroll
                    for (int i = 0; i < 32; ++i) xp[lane * kSwapXposeStride + i] = v[i];
                    __syncwarp();
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = xp[i * kSwapXposeStride + lane];
                    __syncwarp();
                    // now v[i] = logit of vocabulary entry vbase + i for TMEM column c*32 + lane,
                    // i.e. for row rl of the group: MMA j takes its first N_j/2 columns from the
                    // even CTA's rows [o_j, o_j + N_j/2) and the rest from the odd CTA's, and CTA r
                    // holds the group's rows [r * ng/2, +ng/2) (o_0 = 0, o_1 = n0/2)
                    const int col = c * 32 + lane;  // column of the tile
                    const int xj = col < x1 ? 0 : (col < x2 ? x1 : x2);
                    const int nj = col < x1 ? sg.n0 : (col < x2 ? sg.n1 : sg.n2);
                    const int x = col - xj;
                    const int rl = xj / 2 + (x < nj / 2 ? x : ng / 2 + (x - nj / 2));
                    const int r = m * ng + rl;
                    const float scale = r < rows ? __ldg(p.inv_rms + r) * kLog2e : 0.f;
                    float4 st = stats[sub * ng + rl];
                    int a = __float_as_int(st.w);
                    if (full_tile)
                        fold_chunk<true>(v, scale, vbase, p.V, st.x, st.y, st.z, a);
                    else
                        fold_chunk<false>(v, scale, vbase, p.V, st.x, st.y, st.z, a);
                    st.w = __int_as_float(a);
                    stats[sub * ng + rl] = st;
                }
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(acc_empty0 + acc * static_cast<uint32_t>(sizeof(uint64_t)));
            }
            if (!ok) break;
            // Combine the four sub-partitions' statistics of each row of the group, write this
            // CTA's partial and reset the entries for the next unit.  The epilogue warps meet at
            // an mbarrier rather than a named barrier, so that a wait that runs out (or another
            // role's abort) can never leave a warp blocked.
            if (!epi_sync(sm.epi, epi_phase, abort_flag, p.wait_limit_ns)) break;
            for (int rl = etid; rl < ng; rl += kEpiThreads) {
                const int r = m * ng + rl;
                float4 acc4 = stats[rl];
                stats[rl] = kEmpty;
#pragma unroll
                for (int s4 = 1; s4 < 4; ++s4) {
                    acc4 = merge_stat(acc4, stats[s4 * ng + rl]);
                    stats[s4 * ng + rl] = kEmpty;
                }
                if (r < rows && rpd_check(2 * g + static_cast<int>(rank) < p.max_splits, p.meta + kMetaStatus))
                    p.partials[static_cast<size_t>(r) * p.max_splits + 2 * g + static_cast<int>(rank)] = acc4;
            }
            if (!epi_sync(sm.epi, epi_phase, abort_flag, p.wait_limit_ns)) break;
        }
    }

    __syncwarp();
    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();
    tc_fence_after_sync();
    if (*abort_flag && threadIdx.x == 0) atomicExch(&p.meta[kMetaStatus], RPD_ERR_TIMEOUT);
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc_pair(tmem_base, kTmemCols);
    }
}

// The head kernel: one launch per projection pass, clusters of two CTAs, one CTA per SM.
__global__ void __launch_bounds__(kHeadKernelThreads, 1)
    k_head(const __grid_constant__ HeadMaps maps, HeadParams p) {
    pdl_trigger();  // successors may launch now; they wait for this grid before reading
    pdl_wait();     // row count, tiling, u and inv_rms come from the preceding kernels
    const int rows = p.meta[kMetaRows];
    if (rows == 0) return;  // uniform over the grid: no cluster-wide barrier is left waiting
    const int mode = p.meta[kMetaHeadMode];
    const int splits = p.meta[kMetaSplits];
    extern __shared__ uint8_t smem_raw[];
    const HeadSmem sm = carve_smem(smem_raw);
    if (mode == kHeadModePair)
        head_pair(&maps.u, &maps.w128, p, sm, rows, splits);
    else if (mode == kHeadModeRowsN)
        head_swap(maps.u_rows, &maps.w128, p, sm, rows, splits / 2, p.meta[kMetaSwapRows]);
}

// The tiled copy of the head: thread i writes 16-byte vector i of Wt, which is vector k8 of
// row r of block blk = t * (d / 64) + k, i.e. W[128 t + r][64 k + 8 k8 ...].
__global__ void k_tile_head(const uint4 *__restrict__ W, uint4 *__restrict__ Wt, int V, int d) {
    const int nkb = d / 64;
    const long long total = static_cast<long long>((V + 127) / 128) * nkb * 128 * 8;
    for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int k8 = static_cast<int>(i & 7);
        const long long rest = i >> 3;
        const int r = static_cast<int>(rest & 127);
        const long long blk = rest >> 7;
        const int k = static_cast<int>(blk % nkb);
        const int row = static_cast<int>(blk / nkb) * 128 + r;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (row < V) v = W[(static_cast<long long>(row) * d + k * 64) / 8 + k8];
        Wt[i] = v;
    }
}

// Per-device one-time settings (the dynamic shared-memory opt-in is a property of the
// kernel on each device).
constexpr int kMaxDevices = 64;
std::atomic<int> g_head_ready[kMaxDevices];
std::atomic<int> g_head_clusters[kMaxDevices];  // resident pairs + 1 (0: not queried yet)

int current_device() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return -1;
    return dev;
}

cudaError_t opt_in_smem() {
    const int dev = current_device();
    if (dev < 0) return cudaErrorInvalidDevice;
    if (g_head_ready[dev].load(std::memory_order_acquire)) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(k_head, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kHeadKernelSmemBytes);
    if (e == cudaSuccess) g_head_ready[dev].store(1, std::memory_order_release);
    return e;
}

}  // namespace

int head_max_clusters() {
    const int dev = current_device();
    if (dev < 0) return 0;
    const int cached = g_head_clusters[dev].load(std::memory_order_acquire);
    if (cached > 0) return cached - 1;
    if (opt_in_smem() != cudaSuccess) return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2);
    cfg.blockDim = dim3(kHeadKernelThreads);
    cfg.dynamicSmemBytes = kHeadKernelSmemBytes;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k_head, &cfg) != cudaSuccess) n = 0;
    g_head_clusters[dev].store(n + 1, std::memory_order_release);
    return n;
}

cudaError_t launch_tile_head(const void *W, void *Wt, int V, int d, cudaStream_t s) {
    k_tile_head<<<1024, 256, 0, s>>>(static_cast<const uint4 *>(W), static_cast<uint4 *>(Wt), V, d);
    return cudaGetLastError();
}

cudaError_t launch_head(const HeadMaps &maps, const HeadParams &p, int grid, cudaStream_t s) {
    cudaError_t e = opt_in_smem();
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kHeadKernelThreads);
    cfg.dynamicSmemBytes = kHeadKernelSmemBytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = t_no_pdl ? 1 : 2;
    return cudaLaunchKernelEx(&cfg, k_head, maps, p);
}

}  // namespace rpd
