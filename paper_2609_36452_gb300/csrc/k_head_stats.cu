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
#include "ptx.cuh"
#include "rpd_internal.h"

namespace rpd {
namespace {

constexpr uint32_t kTmemCols = 2 * kTileN;
constexpr float kLog2e = 1.4426950408889634f;

struct TileWalk {
    int num_m, num_n, splits, units;
    __device__ __forceinline__ void unit(int u, int &m, int &n0, int &n1) const {
        m = u % num_m;
        const int g = u / num_m;
        n0 = static_cast<int>((static_cast<long long>(g) * num_n) / splits);
        n1 = static_cast<int>((static_cast<long long>(g + 1) * num_n) / splits);
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
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 2 * kStages + 5);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    const int rows = p.meta[kMetaRows];
    TileWalk tw;
    tw.num_m = (rows + kTileM - 1) / kTileM;
    tw.num_n = (p.V + kTileN - 1) / kTileN;
    tw.splits = p.meta[kMetaSplits];
    tw.units = tw.num_m * tw.splits;
    const int num_kb = (p.d + kTileK - 1) / kTileK;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 4);
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

    if (warp == 0) {
        if (lane == 0) {
            // ---------------------------------------------------------------- TMA producer
            int stage = 0;
            uint32_t phase = 0;
            long long fills = 0;
            bool ok = true;
            for (int u = blockIdx.x; ok && u < tw.units; u += gridDim.x) {
                int m, n0, n1;
                tw.unit(u, m, n0, n1);
                for (int n = n0; ok && n < n1; ++n) {
                    for (int kb = 0; kb < num_kb; ++kb) {
                        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_flag, kWaitLimitNs)) {
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
                if (n_s > 0) mbar_wait_drain(&full[s], static_cast<uint32_t>((n_s - 1) & 1), kWaitLimitNs);
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
            for (int u = blockIdx.x; ok && u < tw.units; u += gridDim.x) {
                int m, n0, n1;
                tw.unit(u, m, n0, n1);
                for (int n = n0; ok && n < n1; ++n, ++tile_iter) {
                    const uint32_t acc = tile_iter & 1u;
                    const uint32_t acc_phase = (tile_iter >> 1) & 1u;
                    if (!mbar_wait_bounded(&acc_empty[acc], acc_phase ^ 1u, abort_flag,
                                           kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t d_tmem = tmem_base + acc * kTileN;
                    for (int kb = 0; kb < num_kb; ++kb) {
                        if (!mbar_wait_bounded(&full[stage], phase, abort_flag, kWaitLimitNs)) {
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
            mbar_wait_drain(drain, 0, kWaitLimitNs);
        }
    } else {
        // -------------------------------------------------------------------- epilogue
        const int sub = warp & 3;  // TMEM sub-partition this warp may access
        const int row_in_tile = sub * 32 + lane;
        const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(sub * 32) << 16);
        uint32_t tile_iter = 0;
        bool ok = true;
        for (int u = blockIdx.x; ok && u < tw.units; u += gridDim.x) {
            int m, n0, n1;
            tw.unit(u, m, n0, n1);
            const int r = m * kTileM + row_in_tile;
            const bool valid = r < rows;
            const float scale = valid ? p.inv_rms[r] * kLog2e : 0.f;
            float run_m = -INFINITY, run_s = 0.f, run_t = 0.f;
            int run_a = 0;
            for (int n = n0; n < n1; ++n, ++tile_iter) {
                const uint32_t acc = tile_iter & 1u;
                const uint32_t acc_phase = (tile_iter >> 1) & 1u;
                if (!mbar_wait_bounded(&acc_full[acc], acc_phase, abort_flag, kWaitLimitNs)) {
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
                const int g = u / tw.num_m;
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

}  // namespace

cudaError_t launch_head_stats(const CUtensorMap &tmU, const CUtensorMap &tmW, const HeadParams &p,
                              int grid, cudaStream_t s) {
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(k_head_stats, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kHeadSmemBytes);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    k_head_stats<<<grid, kHeadThreads, kHeadSmemBytes, s>>>(tmU, tmW, p);
    return cudaGetLastError();
}

}  // namespace rpd
