// k_merge_commit.cu - merge of the per-split softmax statistics, the lazy projection's band
// selection, and the scoring, candidate flags, entropy prefix scan and commitment of §3.
//
// k_merge (grid): combines each row's split partials of a projection pass into the row's
//   argmax, its probability and its entropy (merge rule in step_common.cuh).
//
// k_band (one CTA; lazy projection only): selects the positions whose final confidence lies
//   in their canvas's stability band theta_c <= c < tau (Eq. 5 reads S_i only there) and sets
//   up the second pass over their earlier window layers.
//
// k_score_commit (one CTA per canvas, positions in blocked order across threads):
//   y_i = argmax of the final layer, c_i its probability, H_i its entropy;
//   K_i = window layers, counted back from the final one, whose argmax is y_i (Eq. 2,
//         stopping at the first disagreement, App. A.2);
//   r_i = max over those layers of p(y_i) - c_i (Eq. 3; inside the suffix the layer argmax
//         is y_i, so p(y_i) is that layer's maximum probability);
//   S_i = min(K_i, K_max) - w r_i (Eq. 4);  cand_i per Eq. 5;
//   Q_i = sum over j < i of H_j for masked non-candidates (block-wide exclusive scan);
//   accept the candidates before the first candidate with Q > beta.  This equals the
//   sequential rule of §3.2: H >= 0, accepted candidates are excluded from E_i, so while
//   every earlier candidate was accepted E_i = Q_i, and after the first rejection every
//   later candidate sees at least that much entropy.
//   If nothing is accepted and something is masked, commit the most confident of the
//   first W masked positions (leftmost on ties, §3.2).  Then write the outputs, clear the
//   committed mask bits and the per-canvas counters.  RPD-block skips the budget and takes
//   the fallback over the active block.
//
// k_merge_score (grid; a single canvas of at most kFuseScoreMaxN positions): the step's last
//   merge, after which the CTA that finishes last (a device counter) scores and commits the
//   canvas exactly as k_score_commit does, saving a launch.
#include "ptx.cuh"
#include "rpd_internal.h"
#include "step_common.cuh"

namespace rpd {
namespace {

constexpr int kMergeThreads = 256;

// Grid-wide merge of the current projection pass (every row of every canvas).
__global__ void __launch_bounds__(kMergeThreads) k_merge(MergeArgs mg, const int32_t *meta,
                                                         const int32_t *sel_list) {
    pdl_trigger();  // successors may launch now; they wait for this grid before reading
    pdl_wait();
    merge_pass_rows(mg, meta, sel_list, 0, meta[kMetaSel], blockIdx.x, gridDim.x);
}

// Merge of P vocabulary shards' statistics per (layer, masked position), shards in order.
__global__ void __launch_bounds__(kMergeThreads) k_merge_shards(ShardMergeParams p) {
    pdl_trigger();
    pdl_wait();
    const int nmt = p.meta[kMetaMasked];
    const long long total = static_cast<long long>(p.K) * nmt;
    for (long long r = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; r < total;
         r += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int k = static_cast<int>(r / nmt);
        const int q = static_cast<int>(r - static_cast<long long>(k) * nmt);
        const int pos = p.pos_of_q[q];
        Stat acc{-INFINITY, 0.f, 0.f, 0x7fffffff};
        for (int sh = 0; sh < p.P; ++sh) {
            const float4 v = p.gathered[(static_cast<size_t>(sh) * p.K + k) * p.BN + pos];
            acc = merge2(acc, Stat{v.x, v.y, v.z, __float_as_int(v.w)});
        }
        p.row_arg[r] = acc.a;
        p.row_pmax[r] = 1.0f / acc.s;
        p.row_H[r] = fmaxf(logf(acc.s) - kLn2 * (acc.t / acc.s), 0.f);
    }
}

constexpr int kBandThreads = 1024;
constexpr int kBandItems = 4;

__global__ void __launch_bounds__(kBandThreads, 1) k_band(BandParams p) {
    __shared__ int warp_sum[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    pdl_trigger();  // successors may launch now; they wait for this grid before reading
    pdl_wait();
    const int nmt = p.meta[kMetaMasked];
    const bool lazy_on = p.meta[kMetaLazy] != 0;  // else the first pass covered every layer
    // 1. band positions, in compact order (the first pass was merged by k_merge)
    const float *final_p = p.mg.row_pmax + static_cast<size_t>(p.K - 1) * nmt;
    int carry = 0;
    for (int base = 0; lazy_on && base < nmt; base += kBandThreads * kBandItems) {
        const int q0 = base + tid * kBandItems;
        int f[kBandItems];
        int cnt = 0;
#pragma unroll
        for (int j = 0; j < kBandItems; ++j) {
            const int q = q0 + j;
            f[j] = 0;
            if (q < nmt && p.K > 1) {
                const float c = final_p[q];
                const int b = p.pos_of_q[q] / p.N;
                f[j] = (c >= p.theta_c && c < p.tau[b]) ? 1 : 0;
            }
            cnt += f[j];
        }
        const int incl = warp_inclusive_scan(cnt, lane);
        if (lane == 31) warp_sum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            const int v = warp_sum[lane];
            const int vi = warp_inclusive_scan(v, lane);
            warp_sum[lane] = vi - v;
        }
        __syncthreads();
        int excl = carry + warp_sum[warp] + incl - cnt;
#pragma unroll
        for (int j = 0; j < kBandItems; ++j) {
            if (f[j]) p.sel_q[excl] = q0 + j;
            excl += f[j];
        }
        __syncthreads();
        if (tid == kBandThreads - 1) warp_sum[0] = excl;
        __syncthreads();
        carry = warp_sum[0];
        __syncthreads();
    }
    // 2. each canvas's range in the band list (the list is sorted, canvases are contiguous)
    for (int b = tid; b <= p.B; b += kBandThreads) {
        const int key = p.canvas_off[b];
        int lo = 0, hi = carry;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (p.sel_q[mid] < key) lo = mid + 1; else hi = mid;
        }
        p.band_off[b] = lo;
    }
    // 3. the second pass: the K-1 earlier window layers of the band positions
    const long long rows = static_cast<long long>(p.K - 1) * carry;
    if (warp == 0) {
        const HeadPlan hp = lookup_plan(rows, p.plan, p.plan_rows, p.plan_in);
        if (lane == 0) {
            p.meta[kMetaSwapRows] = hp.swap_rows;
            p.meta[kMetaSplits] = hp.splits;
            p.meta[kMetaHeadMode] = hp.mode;
        }
    }
    if (tid == 0) {
        p.meta[kMetaRows] = static_cast<int>(rows);
        p.meta[kMetaSel] = carry;
        p.meta[kMetaLayer0] = 0;
        p.meta[kMetaRowsTotal] += static_cast<int>(rows);
        p.meta[kMetaUnitNext] = 0;
    }
}

// ------------------------------------------------------------------ block-wide helpers

struct ScanPair {
    float q;  // entropy of masked non-candidates
    int m;    // masked positions
};

// Exclusive scan of (q, m) in thread order over the block, plus the block totals.
__device__ __forceinline__ ScanPair block_scan_pair(ScanPair v, ScanPair *sh, ScanPair &total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nwarps = (blockDim.x + 31) >> 5;
    ScanPair incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float tq = __shfl_up_sync(0xffffffffu, incl.q, o);
        const int tm = __shfl_up_sync(0xffffffffu, incl.m, o);
        if (lane >= o) {
            incl.q += tq;
            incl.m += tm;
        }
    }
    if (lane == 31) sh[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        ScanPair w = lane < nwarps ? sh[lane] : ScanPair{0.f, 0};
        ScanPair wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float tq = __shfl_up_sync(0xffffffffu, wi.q, o);
            const int tm = __shfl_up_sync(0xffffffffu, wi.m, o);
            if (lane >= o) {
                wi.q += tq;
                wi.m += tm;
            }
        }
        sh[lane] = ScanPair{wi.q - w.q, wi.m - w.m};
        if (lane == 31) sh[32] = wi;
    }
    __syncthreads();
    total = sh[32];
    const ScanPair base = sh[warp];
    return ScanPair{base.q + incl.q - v.q, base.m + incl.m - v.m};
}

// Block-wide sums of four counters.
__device__ __forceinline__ int4 block_sum4(int4 v, int4 *sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nwarps = (blockDim.x + 31) >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        v.x += __shfl_xor_sync(0xffffffffu, v.x, o);
        v.y += __shfl_xor_sync(0xffffffffu, v.y, o);
        v.z += __shfl_xor_sync(0xffffffffu, v.z, o);
        v.w += __shfl_xor_sync(0xffffffffu, v.w, o);
    }
    if (lane == 0) sh[warp] = v;
    __syncthreads();
    int4 t = make_int4(0, 0, 0, 0);
    for (int w = 0; w < nwarps; ++w) {
        t.x += sh[w].x;
        t.y += sh[w].y;
        t.z += sh[w].z;
        t.w += sh[w].w;
    }
    return t;
}

constexpr int kLayerBatch = 8;  // window layers whose statistics are loaded together

// Scores and commits canvas b with the whole CTA.  kMaxItems positions per thread at most
// (N <= kMaxItems * blockDim.x); instantiated for 1, 2, 4 and 8 so that short canvases carry
// no unused per-item state.  The merged row statistics are read through L2 (ld.cg): in the
// fused merge-and-score kernel other CTAs of the same grid wrote them.
template <int kMaxItems>
__device__ __forceinline__ void score_canvas(const ScoreParams &p, const int b) {
    __shared__ ScanPair sh_scan[33];
    __shared__ int4 sh_sum[32];
    __shared__ int first_reject;
    __shared__ unsigned long long best_fb;

    const int N = p.N;
    const int nmt = p.meta[kMetaMasked];
    const int K = p.K;
    const float tau = p.tau[b], beta = p.budget[b];
    const int items = (N + blockDim.x - 1) / blockDim.x;
    const int i0 = threadIdx.x * items;
    uint8_t *mask = p.mask + static_cast<size_t>(b) * N;
    const bool dbg_layers = p.dbg.layer_argmax || p.dbg.layer_pmax;
    const bool lazy_on = p.meta[kMetaLazy] != 0;  // earlier layers exist only in the band

    bool masked[kMaxItems], cand[kMaxItems], high[kMaxItems];
    int y[kMaxItems];
    float conf[kMaxItems], H[kMaxItems];

    ScanPair local{0.f, 0};  // (entropy of scored non-candidates, scored positions)
    int n_cand = 0, n_masked_all = 0;
#pragma unroll
    for (int j = 0; j < kMaxItems; ++j) {
        masked[j] = cand[j] = high[j] = false;
        y[j] = -1;
        conf[j] = H[j] = 0.f;
        const int i = i0 + j;
        if (j >= items || i >= N) continue;
        const size_t pos = static_cast<size_t>(b) * N + i;
        // both loads issued together (q_of_pos is -1 wherever the mask is 0)
        const int q_raw = p.q_of_pos[pos];
        const bool is_masked = mask[i] != 0;
        n_masked_all += is_masked;
        // Scored positions: every masked one, or (RPD-block) the active block's masked ones,
        // which are exactly those the compaction kept.
        const int q = is_masked ? q_raw : -1;
        masked[j] = q >= 0;
        int ki = 0;
        float r = 0.f, s = 0.f;
        if (masked[j]) {
            // Backward over the window, a batch of layers at a time (loads issued together).
            float peak = 0.f;
            bool run = true;
            bool projected = true;  // lazy projection: earlier layers exist only in the band
            for (int k_hi = K; k_hi > 0; k_hi -= kLayerBatch) {
                if (!run && !dbg_layers) break;  // persistence settled; debug wants every layer
                int a_b[kLayerBatch];
                float p_b[kLayerBatch];
#pragma unroll
                for (int t = 0; t < kLayerBatch; ++t) {
                    const int k = k_hi - 1 - t;
                    if (k >= 0) {
                        const size_t rk = static_cast<size_t>(k) * nmt + q;
                        a_b[t] = __ldcg(p.row_arg + rk);
                        p_b[t] = __ldcg(p.row_pmax + rk);
                    }
                }
#pragma unroll
                for (int t = 0; t < kLayerBatch; ++t) {
                    const int k = k_hi - 1 - t;
                    if (k < 0) break;
                    if (k == K - 1) {
                        y[j] = a_b[t];
                        conf[j] = p_b[t];
                        peak = p_b[t];
                        ki = 1;
                        if (lazy_on && !(conf[j] >= p.theta_c && conf[j] < tau)) {
                            projected = false;  // outside the band: K_i, r_i not needed
                            run = false;
                        }
                    } else if (!projected) {
                        a_b[t] = -1;
                        p_b[t] = 0.f;
                    } else if (run) {
                        if (a_b[t] != y[j]) {
                            run = false;
                        } else {
                            ++ki;
                            peak = fmaxf(peak, p_b[t]);
                        }
                    }
                    if (dbg_layers) {
                        const size_t o = (static_cast<size_t>(k) * p.B) * N + pos;
                        if (p.dbg.layer_argmax) p.dbg.layer_argmax[o] = a_b[t];
                        if (p.dbg.layer_pmax) p.dbg.layer_pmax[o] = p_b[t];
                    }
                }
            }
            H[j] = __ldcg(p.row_H + static_cast<size_t>(K - 1) * nmt + q);
            r = peak - conf[j];
            s = static_cast<float>(min(ki, p.k_max)) - p.w * r;
            high[j] = conf[j] >= tau;
            cand[j] = high[j] || (conf[j] >= p.theta_c && conf[j] < tau && s >= p.theta_s);
            if (!projected) {  // reported as not evaluated
                ki = 0;
                r = 0.f;
                s = 0.f;
            }
            ++local.m;
            n_cand += cand[j];
            if (!cand[j]) local.q += H[j];
        } else if (dbg_layers) {
            for (int k = 0; k < K; ++k) {
                const size_t o = (static_cast<size_t>(k) * p.B) * N + pos;
                if (p.dbg.layer_argmax) p.dbg.layer_argmax[o] = -1;
                if (p.dbg.layer_pmax) p.dbg.layer_pmax[o] = 0.f;
            }
        }
        if (p.dbg.conf) p.dbg.conf[pos] = masked[j] ? conf[j] : 0.f;
        if (p.dbg.entropy) p.dbg.entropy[pos] = masked[j] ? H[j] : 0.f;
        if (p.dbg.persist) p.dbg.persist[pos] = ki;
        if (p.dbg.drop) p.dbg.drop[pos] = r;
        if (p.dbg.stability) p.dbg.stability[pos] = masked[j] ? s : 0.f;
        if (p.dbg.candidate) p.dbg.candidate[pos] = cand[j];
    }

    // ------------------------------ entropy of masked non-candidates and masked ranks, scanned
    if (threadIdx.x == 0) {
        first_reject = N;
        best_fb = 0ull;
    }
    ScanPair total;
    const ScanPair pre = block_scan_pair(local, sh_scan, total);  // synchronises the block
    float q = pre.q;
#pragma unroll
    for (int j = 0; j < kMaxItems; ++j) {
        if (p.block > 0) break;  // RPD-block: no entropy budget
        if (j >= items || i0 + j >= N) break;
        if (cand[j] && q > beta) {
            atomicMin(&first_reject, i0 + j);
            break;
        }
        if (masked[j] && !cand[j]) q += H[j];
    }
    __syncthreads();
    const int reject_at = first_reject;

    // accepted, accepted through c >= tau, candidates, masked positions of the canvas
    int4 cnt = make_int4(0, 0, n_cand, n_masked_all);
#pragma unroll
    for (int j = 0; j < kMaxItems; ++j) {
        const bool acc = cand[j] && (i0 + j) < reject_at;
        cnt.x += acc;
        cnt.y += acc && high[j];
    }
    const int4 tot = block_sum4(cnt, sh_sum);
    const int total_masked = tot.w;
    const int fallback_window = p.block > 0 ? p.block : p.window;

    // ------------------------------------------------------------------------ fallback
    int fb_pos = -1;
    if (tot.x == 0 && total.m > 0) {  // uniform across the block
        int rank = pre.m;
        unsigned long long mine = 0ull;
#pragma unroll
        for (int j = 0; j < kMaxItems; ++j) {
            if (!masked[j]) continue;
            if (rank < fallback_window) {
                // c >= 0: its bit pattern orders like the value; ties -> lowest position
                const unsigned long long key =
                    (static_cast<unsigned long long>(__float_as_uint(conf[j])) << 32) |
                    static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<unsigned>(i0 + j));
                mine = key > mine ? key : mine;
            }
            ++rank;
        }
        if (mine) atomicMax(&best_fb, mine);
        __syncthreads();
        fb_pos = static_cast<int>(0xFFFFFFFFu - static_cast<unsigned>(best_fb & 0xFFFFFFFFull));
    }

    // ------------------------------------------------------------------------- outputs
#pragma unroll
    for (int j = 0; j < kMaxItems; ++j) {
        const int i = i0 + j;
        if (j >= items || i >= N) break;
        const size_t pos = static_cast<size_t>(b) * N + i;
        const bool commit = (cand[j] && i < reject_at) || i == fb_pos;
        p.out_commit[pos] = commit ? 1 : 0;
        if (commit) {
            p.out_token[pos] = y[j];
            mask[i] = 0;
        }
    }
    if (threadIdx.x == 0) {
        rpd_stats st;
        st.n_masked = total_masked;
        st.n_candidates = tot.z;
        st.n_high_conf = tot.y;
        st.n_stability = tot.x - tot.y;
        st.n_committed = tot.x + (fb_pos >= 0 ? 1 : 0);
        st.fallback_used = fb_pos >= 0 ? 1 : 0;
        st.fallback_pos = fb_pos;
        st.status = p.meta[kMetaStatus];
        st.n_rows = p.meta[kMetaRowsTotal];
        p.out_stats[b] = st;
    }
}

template <int kMaxItems>
__global__ void __launch_bounds__(kScoreThreads, 1) k_score_commit(ScoreParams p) {
    pdl_trigger();  // successors may launch now; they wait for this grid before reading
    pdl_wait();
    score_canvas<kMaxItems>(p, blockIdx.x);
}

// The step's last merge and the scoring of its single canvas in one grid: the CTAs merge
// their rows; the one that finishes last (a device counter, zeroed by the compaction)
// scores the canvas.  No CTA waits for another.  With no rows to merge, CTA 0 scores.
template <int kMaxItems>
__global__ void __launch_bounds__(kMergeThreads) k_merge_score(MergeArgs mg, int32_t *meta,
                                                                const int32_t *sel_list,
                                                                ScoreParams p) {
    __shared__ int last;
    pdl_trigger();
    pdl_wait();
    const int working = merge_pass_rows(mg, meta, sel_list, 0, meta[kMetaSel], blockIdx.x, gridDim.x);
    if (working == 0) {
        if (blockIdx.x != 0) return;
    } else {
        if (static_cast<int>(blockIdx.x) >= working) return;
        __threadfence();  // this CTA's merged rows are visible before it is counted
        __syncthreads();
        if (threadIdx.x == 0) last = atomicAdd(&meta[kMetaMergeDone], 1) == working - 1;
        __syncthreads();
        if (!last) return;
        __threadfence();
    }
    score_canvas<kMaxItems>(p, 0);
}

}  // namespace

cudaError_t launch_merge(const MergeArgs &mg, const int32_t *meta, const int32_t *sel_list,
                         int grid, cudaStream_t s) {
    return launch_pdl(k_merge, dim3(grid), dim3(kMergeThreads), 0, s, mg, meta, sel_list);
}

cudaError_t launch_merge_score(const MergeArgs &mg, int32_t *meta, const int32_t *sel_list,
                               int grid, const ScoreParams &p, cudaStream_t s) {
    if (p.B != 1 || p.N > kFuseScoreMaxN) return cudaErrorInvalidValue;
    const int items = (p.N + kMergeThreads - 1) / kMergeThreads;
    const dim3 g(grid), t(kMergeThreads);
    if (items <= 1) return launch_pdl(k_merge_score<1>, g, t, 0, s, mg, meta, sel_list, p);
    if (items <= 2) return launch_pdl(k_merge_score<2>, g, t, 0, s, mg, meta, sel_list, p);
    if (items <= 4) return launch_pdl(k_merge_score<4>, g, t, 0, s, mg, meta, sel_list, p);
    return launch_pdl(k_merge_score<8>, g, t, 0, s, mg, meta, sel_list, p);
}

namespace {
// The stop test of the decoding loop: one thread counts the step and keeps the loop going
// while some canvas has more than floor(stop_frac * N) positions masked, fewer than max_steps
// steps have run and every canvas's step succeeded.
__global__ void k_loop_test(cudaGraphConditionalHandle handle, const rpd_stats *stats, int B, int N,
                            float stop_frac, int max_steps, int32_t *steps) {
    const int n = *steps + 1;
    *steps = n;
    const int limit = static_cast<int>(floorf(stop_frac * static_cast<float>(N)));
    bool ok = true, open = false;
    for (int b = 0; b < B; ++b) {
        ok = ok && stats[b].status == RPD_OK;
        open = open || stats[b].n_masked - stats[b].n_committed > limit;
    }
    cudaGraphSetConditional(handle, ok && open && n < max_steps ? 1u : 0u);
}
}  // namespace

cudaError_t launch_loop_test(cudaGraphConditionalHandle handle, const rpd_stats *stats, int B, int N,
                             float stop_frac, int max_steps, int32_t *steps, cudaStream_t s) {
    // a plain launch: it must see the finished step's statistics
    k_loop_test<<<1, 1, 0, s>>>(handle, stats, B, N, stop_frac, max_steps, steps);
    return cudaGetLastError();
}

cudaError_t launch_merge_shards(const ShardMergeParams &p, int grid, cudaStream_t s) {
    return launch_pdl(k_merge_shards, dim3(grid), dim3(kMergeThreads), 0, s, p);
}

cudaError_t launch_band(const BandParams &p, cudaStream_t s) {
    return launch_pdl(k_band, dim3(1), dim3(kBandThreads), 0, s, p);
}

cudaError_t launch_score_commit(const ScoreParams &p, cudaStream_t s) {
    const int threads = p.N >= kScoreThreads ? kScoreThreads : ((p.N + 31) / 32) * 32;
    const int items = (p.N + threads - 1) / threads;
    if (items <= 1) return launch_pdl(k_score_commit<1>, dim3(p.B), dim3(threads), 0, s, p);
    if (items <= 2) return launch_pdl(k_score_commit<2>, dim3(p.B), dim3(threads), 0, s, p);
    if (items <= 4) return launch_pdl(k_score_commit<4>, dim3(p.B), dim3(threads), 0, s, p);
    return launch_pdl(k_score_commit<kMaxCanvas / kScoreThreads>, dim3(p.B), dim3(threads), 0, s, p);
}

}  // namespace rpd
