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
// Logits never reach global memory.  Each work unit is (128-row tile, contiguous range of
// 256-wide vocabulary tiles); its statistics are written once per row as one partial
// (float4) that the merge kernel combines.
//
// Persistent CTA, 6 warps:
//   warp 0      TMA producer (one thread): u tile 128x64 and W tile 256x64 per stage
//   warp 1      TMEM owner (alloc/dealloc 512 columns) and MMA issuer (one thread)
//   warps 2..5  epilogue: warp w reads TMEM lanes 32*(w%4)..+31, one row per thread
// Two 256-column fp32 accumulators (512 TMEM columns) let the epilogue of one tile run
// under the MMAs of the next.  Every wait is bounded; a timeout latches RPD_ERR_TIMEOUT
// in the step's status word and the CTA drains and exits.
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

// Fold one 32-column chunk (already scaled to log2 units) into the running statistics.
template <bool kFull>
__device__ __forceinline__ void fold_chunk(const float (&v)[32], float scale, int col0, int V,
                                           float &run_m, float &run_s, float &run_t,
                                           int &run_a) {
    float x[32];
    float cmax = -INFINITY;
    int carg = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        x[i] = v[i] * scale;
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

__global__ void __launch_bounds__(kHeadThreads, 1)
    k_head_stats(const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmW,
                 HeadParams p) {
    pdl_trigger();  // successors may launch now; they wait for this grid before reading
    pdl_wait();     // row count, tiling, u and inv_rms come from the preceding kernels
    if (p.meta[kMetaHeadMode] != 1 || p.meta[kMetaRows] == 0) return;  // pair tiling, or nothing to do
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t *sA = smem;
    uint8_t *sB = smem + kStages * kStageBytesA;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kStages * (kStageBytesA + kStageBytesB));
    uint64_t *full = bars;                  // [kStages] TMA -> MMA
    uint64_t *empty = bars + kStages;       // [kStages] MMA -> TMA
    uint64_t *acc_full = bars + 2 * kStages;      // [2] MMA -> epilogue
    uint64_t *acc_empty = bars + 2 * kStages + 2; // [2] epilogue -> MMA
    uint64_t *drain = bars + 2 * kStages + 4;     // [1] MMA completion at exit
    uint64_t *unit_full = bars + 2 * kStages + 5; // [kUnitRing] producer -> MMA, epilogue
    uint64_t *unit_empty = unit_full + kUnitRing; // [kUnitRing] MMA, epilogue -> producer
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(unit_empty + kUnitRing);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
    volatile int *unit_ring = abort_flag + 1;     // [kUnitRing] claimed unit indices

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 4);
        }
        for (int i = 0; i < kUnitRing; ++i) {
            mbar_init(&unit_full[i], 1);
            mbar_init(&unit_empty[i], 1 + 4);  // MMA issuer + 4 epilogue warps
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tmU);
        tma_prefetch_desc(&tmW);
    }
    if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;

    const int rows = p.meta[kMetaRows];
    TileWalk tw;
    tw.init(rows, kTileM, p.V, p.d, p.meta[kMetaSplits]);
    const int num_kb = (p.d + kTileK - 1) / kTileK;

    if (warp == 0) {
        if (lane == 0 && !p.stall) {
            // ---------------------------------------------------------------- TMA producer
            int stage = 0;
            uint32_t phase = 0;
            long long fills = 0;
            bool ok = true;
            UnitCursor uc;
            while (ok) {
                if (!mbar_wait_bounded(&unit_empty[uc.slot], uc.phase ^ 1u, abort_flag, p.wait_limit_ns))
                    break;
                const int claimed = atomicAdd(&p.meta[kMetaUnitNext], 1);
                const int u = claimed < tw.units ? claimed : -1;
                unit_ring[uc.slot] = u;
                mbar_arrive(&unit_full[uc.slot]);
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
                        mbar_arrive_expect_tx(&full[stage], kStageBytesA + kStageBytesB);
                        tma_load_2d(sA + stage * kStageBytesA, &tmU, &full[stage], kb * kTileK,
                                    m * kTileM);
                        tma_load_2d(sB + stage * kStageBytesB, &tmW, &full[stage], kb * kTileK,
                                    n * kTileN);
                        ++fills;
                        if (++stage == kStages) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                }
            }
            // Drain: every issued copy must have landed before the CTA may exit (on the
            // normal path they all have, since the MMA consumed them).
            for (int s = 0; s < kStages; ++s) {
                const long long n_s = fills / kStages + (s < fills % kStages ? 1 : 0);
                if (n_s > 0) mbar_wait_drain(&full[s], static_cast<uint32_t>((n_s - 1) & 1), p.wait_limit_ns);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------------------------------------------------------- MMA issuer
            constexpr uint32_t idesc = idesc_bf16_f32(kTileM, kTileN);
            int stage = 0;
            uint32_t phase = 0;
            uint32_t tile_iter = 0;
            bool ok = true;
            UnitCursor uc;
            while (ok) {
                if (!mbar_wait_bounded(&unit_full[uc.slot], uc.phase, abort_flag, p.wait_limit_ns)) break;
                const int u = unit_ring[uc.slot];
                mbar_arrive(&unit_empty[uc.slot]);
                uc.advance();
                if (u < 0) break;
                int m, g, n0, n1;
                tw.unit(u, m, g, n0, n1);
                for (int n = n0; ok && n < n1; ++n, ++tile_iter) {
                    const uint32_t acc = tile_iter & 1u;
                    const uint32_t acc_phase = (tile_iter >> 1) & 1u;
                    if (!mbar_wait_bounded(&acc_empty[acc], acc_phase ^ 1u, abort_flag,
                                           p.wait_limit_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t d_tmem = tmem_base + acc * kTileN;
                    for (int kb = 0; kb < num_kb; ++kb) {
                        if (!mbar_wait_bounded(&full[stage], phase, abort_flag, p.wait_limit_ns)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after_sync();
                        const uint32_t a0 = smem_u32(sA + stage * kStageBytesA);
                        const uint32_t b0 = smem_u32(sB + stage * kStageBytesB);
#pragma unroll
                        for (int kk = 0; kk < kTileK / 16; ++kk) {
                            umma_bf16(d_tmem, smem_desc_sw128(a0 + kk * 32),
                                      smem_desc_sw128(b0 + kk * 32), idesc,
                                      (kb > 0 || kk > 0) ? 1u : 0u);
                        }
                        umma_commit(&empty[stage]);
                        if (++stage == kStages) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                    if (!ok) break;
                    umma_commit(&acc_full[acc]);
                }
            }
            // Drain: wait until every MMA this thread issued has completed.
            umma_commit(drain);
            mbar_wait_drain(drain, 0, p.wait_limit_ns);
        }
    } else {
        // -------------------------------------------------------------------- epilogue
        const int sub = warp & 3;  // TMEM sub-partition this warp may access
        const int row_in_tile = sub * 32 + lane;
        const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(sub * 32) << 16);
        uint32_t tile_iter = 0;
        bool ok = true;
        UnitCursor uc;
        while (ok) {
            if (!mbar_wait_bounded(&unit_full[uc.slot], uc.phase, abort_flag, p.wait_limit_ns)) break;
            const int u = unit_ring[uc.slot];
            __syncwarp();
            if (lane == 0) mbar_arrive(&unit_empty[uc.slot]);
            uc.advance();
            if (u < 0) break;
            int m, g, n0, n1;
            tw.unit(u, m, g, n0, n1);
            const int r = m * kTileM + row_in_tile;
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
                if (lane == 0) mbar_arrive(&acc_empty[acc]);
            }
            if (!ok) break;
            if (valid) {
                p.partials[static_cast<size_t>(r) * p.max_splits + g] =
                    make_float4(run_m, run_s, run_t, __int_as_float(run_a));
            }
        }
    }

    __syncwarp();
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    if (*abort_flag && threadIdx.x == 0) atomicExch(&p.meta[kMetaStatus], RPD_ERR_TIMEOUT);
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc(tmem_base, kTmemCols);
    }
}


// ------------------------------------------------------------------------------------------
// CTA-pair form (tcgen05 cta_group::2).  A pair (cluster of 2 CTAs) computes a tile of 256
// rows x 256 vocabulary columns: CTA r of the pair stages rows [128r, 128r+128) of the row
// tile and W rows [128r, 128r+128) of the vocabulary tile; the even CTA issues
// tcgen05.mma.cta_group::2 with M=256, N=256, which reads both CTAs' shared memory and
// accumulates rows [128r, 128r+128) x all 256 columns into CTA r's TMEM.  Per SM and K-step
// that is 32 KB of operands for the same MMA work the single-CTA tile does with 48 KB.
//
// Barriers: full[s] lives in the even CTA and receives both CTAs' TMA completions (tx bytes
// 64 KB per stage); empty[s], acc_full[a] and drain receive multicast commits from the MMA
// thread in both CTAs; acc_empty[a] lives in the even CTA and counts the 4 epilogue warps
// of both CTAs (8 arrivals).
__global__ void __launch_bounds__(kHeadThreads, 1)
    k_head_stats_pair(const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmW,
                      HeadParams p) {
    pdl_trigger();  // successors may launch now; they wait for this grid before reading
    pdl_wait();     // row count, tiling, u and inv_rms come from the preceding kernels
    if (p.meta[kMetaHeadMode] != 2 || p.meta[kMetaRows] == 0) return;  // single tiling, or nothing
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t *sA = smem;
    uint8_t *sB = smem + kPairStages * kPairStageBytesA;
    uint64_t *bars =
        reinterpret_cast<uint64_t *>(smem + kPairStages * (kPairStageBytesA + kPairStageBytesB));
    uint64_t *full = bars;                            // [kPairStages] (used in the even CTA)
    uint64_t *empty = bars + kPairStages;             // [kPairStages]
    uint64_t *acc_full = bars + 2 * kPairStages;      // [2]
    uint64_t *acc_empty = bars + 2 * kPairStages + 2; // [2] (used in the even CTA)
    uint64_t *drain = bars + 2 * kPairStages + 4;     // [1]
    uint64_t *unit_full = bars + 2 * kPairStages + 5; // [kUnitRing] even producer -> all others
    uint64_t *unit_empty = unit_full + kUnitRing;     // [kUnitRing] (used in the even CTA)
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(unit_empty + kUnitRing);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
    volatile int *unit_ring = abort_flag + 1;         // [kUnitRing] claimed unit indices

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
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tmU);
        tma_prefetch_desc(&tmW);
    }
    if (warp == 1) tmem_alloc_pair(tmem_slot, kTmemCols);
    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();  // both CTAs' barriers initialised before any cross-CTA signal
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;

    const int rows = p.meta[kMetaRows];
    TileWalk tw;
    tw.init(rows, kPairTileM, p.V, p.d, p.meta[kMetaSplits]);
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
                        if (rank == 0)
                            mbar_arrive_expect_tx(&full[stage], 2 * (kPairStageBytesA + kPairStageBytesB));
                        const uint32_t fb = full0 + static_cast<uint32_t>(stage * sizeof(uint64_t));
                        tma_load_2d_pair(sA + stage * kPairStageBytesA, &tmU, fb, kb * kTileK,
                                         m * kPairTileM + static_cast<int>(rank) * kPairHalfRows);
                        tma_load_2d_pair(sB + stage * kPairStageBytesB, &tmW, fb, kb * kTileK,
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
        if (lane == 0) {
            if (rank == 0) {
                // ------------------------------------------------ MMA issuer (even CTA only)
                constexpr uint32_t idesc = idesc_bf16_f32(kPairTileM, kTileN);
                int stage = 0;
                uint32_t phase = 0;
                uint32_t tile_iter = 0;
                bool ok = true;
                UnitCursor uc;
                while (ok) {
                    if (!mbar_wait_bounded(&unit_full[uc.slot], uc.phase, abort_flag, p.wait_limit_ns))
                        break;
                    const int u = unit_ring[uc.slot];
                    mbar_arrive(&unit_empty[uc.slot]);
                    uc.advance();
                    if (u < 0) break;
                    int m, g, n0, n1;
                    tw.unit(u, m, g, n0, n1);
                    for (int n = n0; ok && n < n1; ++n, ++tile_iter) {
                        const uint32_t acc = tile_iter & 1u;
                        const uint32_t acc_phase = (tile_iter >> 1) & 1u;
                        if (!mbar_wait_bounded(&acc_empty[acc], acc_phase ^ 1u, abort_flag,
                                               p.wait_limit_ns)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after_sync();
                        const uint32_t d_tmem = tmem_base + acc * kTileN;
                        for (int kb = 0; kb < num_kb; ++kb) {
                            if (!mbar_wait_bounded(&full[stage], phase, abort_flag, p.wait_limit_ns)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after_sync();
                            const uint32_t a0 = smem_u32(sA + stage * kPairStageBytesA);
                            const uint32_t b0 = smem_u32(sB + stage * kPairStageBytesB);
#pragma unroll
                            for (int kk = 0; kk < kTileK / 16; ++kk) {
                                umma_bf16_pair(d_tmem, smem_desc_sw128(a0 + kk * 32),
                                               smem_desc_sw128(b0 + kk * 32), idesc,
                                               (kb > 0 || kk > 0) ? 1u : 0u);
                            }
                            umma_commit_pair_multicast(&empty[stage], 0x3);
                            if (++stage == kPairStages) {
                                stage = 0;
                                phase ^= 1u;
                            }
                        }
                        if (!ok) break;
                        umma_commit_pair_multicast(&acc_full[acc], 0x3);
                    }
                }
                umma_commit_pair_multicast(drain, 0x3);
            }
            // Both CTAs: every MMA writing this CTA's TMEM has completed before it is freed.
            mbar_wait_drain(drain, 0, p.wait_limit_ns);
        }
    } else {
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
            if (valid) {
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

// Per-device one-time settings (the dynamic shared-memory opt-in is a property of the
// kernel on each device).
constexpr int kMaxDevices = 64;
std::atomic<int> g_single_ready[kMaxDevices];
std::atomic<int> g_pair_ready[kMaxDevices];
std::atomic<int> g_pair_clusters[kMaxDevices];  // resident pairs + 1 (0: not queried yet)

int current_device() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return -1;
    return dev;
}

cudaError_t opt_in_smem(const void *kernel, int bytes, std::atomic<int> *ready) {
    const int dev = current_device();
    if (dev < 0) return cudaErrorInvalidDevice;
    if (ready[dev].load(std::memory_order_acquire)) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) ready[dev].store(1, std::memory_order_release);
    return e;
}

}  // namespace

cudaError_t launch_head_stats(const CUtensorMap &tmU, const CUtensorMap &tmW, const HeadParams &p,
                              int grid, cudaStream_t s) {
    cudaError_t e = opt_in_smem(reinterpret_cast<const void *>(k_head_stats), kHeadSmemBytes,
                                g_single_ready);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_head_stats, dim3(grid), dim3(kHeadThreads), kHeadSmemBytes, s, tmU, tmW, p);
}

}  // namespace rpd

namespace rpd {

int head_stats_pair_max_clusters() {
    const int dev = current_device();
    if (dev < 0) return 0;
    const int cached = g_pair_clusters[dev].load(std::memory_order_acquire);
    if (cached > 0) return cached - 1;
    if (opt_in_smem(reinterpret_cast<const void *>(k_head_stats_pair), kPairSmemBytes,
                    g_pair_ready) != cudaSuccess)
        return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2);
    cfg.blockDim = dim3(kHeadThreads);
    cfg.dynamicSmemBytes = kPairSmemBytes;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k_head_stats_pair, &cfg) != cudaSuccess) n = 0;
    g_pair_clusters[dev].store(n + 1, std::memory_order_release);
    return n;
}

cudaError_t launch_head_stats_pair(const CUtensorMap &tmU, const CUtensorMap &tmW,
                                   const HeadParams &p, int grid, cudaStream_t s) {
    cudaError_t e = opt_in_smem(reinterpret_cast<const void *>(k_head_stats_pair), kPairSmemBytes,
                                g_pair_ready);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kHeadThreads);
    cfg.dynamicSmemBytes = kPairSmemBytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, k_head_stats_pair, tmU, tmW, p);
}

}  // namespace rpd
