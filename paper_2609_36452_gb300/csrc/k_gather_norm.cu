// k_gather_norm.cu - device-side compaction of the masked positions and the RMSNorm
// prologue of the layerwise projection (App. A.6: only masked positions are projected;
// App. A.2: the model's final normalisation is applied to every window layer).
//
// k_compact (one CTA): order-preserving compaction of mask[B][N] into compact indices
//   q = 0..NMT-1 (canvas-major, then position), per-canvas offsets, the projected row
//   count R = K*NMT and the vocabulary split count the head kernel will use.  Nothing
//   goes back to the host: later kernels read these words from device memory.
// k_gather_norm (grid-stride, one warp per row): row r of a projection pass (layer k and
//   compact position q from the pass's meta words) reads hidden[k][pos(q)], writes the head
//   operand u[r] = bf16_rne(g * h) (exact product, one rounding) and
//   inv_rms[r] = (mean(h^2) + eps)^(-1/2); the RMS factor is applied after the contraction.
#include "ptx.cuh"
#include "rpd_internal.h"
#include "step_common.cuh"

namespace rpd {
namespace {

constexpr int kCompactThreads = 1024;
constexpr int kCompactItems = 4;

// At most 48 registers a thread: the CTA then needs 48 K of an SM's 64 K registers, so it can
// start (launched early, waiting on its predecessor) beside one CTA of the previous step's merge
// instead of waiting for an SM to empty.
__global__ void __maxnreg__(48) k_compact(CompactParams p) {
    __shared__ int warp_sum[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ int block_lo[kMaxBatch];  // RPD-block: first position of each canvas's active block
    pdl_trigger();  // successors may launch now; they wait for this grid before reading
    pdl_wait();
    const int total = p.B * p.N;
    if (p.block > 0) {
        for (int b = tid; b < p.B; b += kCompactThreads) block_lo[b] = p.N;
        __syncthreads();
        for (int i = tid; i < total; i += kCompactThreads)
            if (p.mask[i]) atomicMin(&block_lo[i / p.N], i % p.N);
        __syncthreads();
        for (int b = tid; b < p.B; b += kCompactThreads)
            block_lo[b] = block_lo[b] < p.N ? (block_lo[b] / p.block) * p.block : p.N;
        __syncthreads();
    }
    int carry = 0;
    for (int base = 0; base < total; base += kCompactThreads * kCompactItems) {
        const int i0 = base + tid * kCompactItems;
        int f[kCompactItems];
        int cnt = 0;
#pragma unroll
        for (int j = 0; j < kCompactItems; ++j) {
            const int i = i0 + j;
            f[j] = (i < total) ? (p.mask[i] != 0) : 0;
            if (f[j] && p.block > 0) {
                const int lo = block_lo[i / p.N], pos = i % p.N;
                f[j] = pos >= lo && pos < lo + p.block;
            }
            cnt += f[j];
        }
        const int incl = warp_inclusive_scan(cnt, lane);
        if (lane == 31) warp_sum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            const int v = warp_sum[lane];
            const int vi = warp_inclusive_scan(v, lane);
            warp_sum[lane] = vi - v;  // exclusive prefix of warp totals
        }
        __syncthreads();
        int excl = carry + warp_sum[warp] + incl - cnt;
#pragma unroll
        for (int j = 0; j < kCompactItems; ++j) {
            const int i = i0 + j;
            if (i < total) {
                if (i % p.N == 0) p.canvas_off[i / p.N] = excl;
                p.q_of_pos[i] = f[j] ? excl : -1;
                if (f[j]) p.pos_of_q[excl] = i;
                excl += f[j];
            }
        }
        // chunk total = exclusive prefix of the last warp + its inclusive total
        __syncthreads();
        if (tid == kCompactThreads - 1) warp_sum[0] = excl;  // running count after the chunk
        __syncthreads();
        carry = warp_sum[0];
        __syncthreads();
    }

    // First pass: every window layer of the scored positions, or only the final layer (lazy).
    // Automatic choice: lazy when its two passes (the final layer of every position, then
    // the earlier layers of an assumed band fraction) are estimated cheaper than one pass
    // over all layers.
    __shared__ int lazy_on;
    __shared__ HeadPlan plan;
    const long long all_rows = static_cast<long long>(p.K) * carry;
    if (warp == 0) {
        int lz = (p.lazy == 1 && p.K > 1) ? 1 : 0;
        if (p.lazy == 2 && p.K > 1) {
            const long long guess = static_cast<long long>(kLazyBandGuess * (p.K - 1) * carry);
            const float e_all = lookup_plan(all_rows, p.plan, p.plan_rows, p.plan_in).est;
            const float e_fin = lookup_plan(carry, p.plan, p.plan_rows, p.plan_in).est;
            const float e_band = lookup_plan(guess, p.plan, p.plan_rows, p.plan_in).est;
            lz = (e_fin + e_band < e_all) ? 1 : 0;
        }
        const HeadPlan hp = lookup_plan(lz ? static_cast<long long>(carry) : all_rows, p.plan,
                                        p.plan_rows, p.plan_in);
        if (lane == 0) {
            lazy_on = lz;
            plan = hp;
        }
    }
    __syncthreads();
    const long long rows = lazy_on ? static_cast<long long>(carry) : all_rows;
    const int mode = plan.mode, splits = plan.splits, swap_rows = plan.swap_rows;
    if (tid == 0) {
        p.canvas_off[p.B] = carry;
        p.meta[kMetaSwapRows] = swap_rows;
        p.meta[kMetaMasked] = carry;
        p.meta[kMetaRows] = static_cast<int>(rows);
        if (!p.keep_status) p.meta[kMetaStatus] = RPD_OK;
        p.meta[kMetaSplits] = splits;
        p.meta[kMetaHeadMode] = mode;
        p.meta[kMetaSel] = carry;
        p.meta[kMetaLayer0] = lazy_on ? p.K - 1 : 0;
        p.meta[kMetaRowsTotal] = static_cast<int>(rows);
        p.meta[kMetaLazy] = lazy_on;
        p.meta[kMetaUnitNext] = 0;
        p.meta[kMetaMergeDone] = 0;
    }
}

// One warp per row; the gain is staged once per CTA in shared memory and each lane keeps up
// to kVecPerLane 16-byte loads of its row in flight before using any of them.
constexpr int kNormThreads = 256;
constexpr int kVecPerLane = 16;  // 32 lanes x 16 x 8 bf16 = 4096 elements per pass

__global__ void __launch_bounds__(kNormThreads) k_gather_norm(NormParams p) {
    extern __shared__ uint4 g_smem[];
    const int lane = threadIdx.x & 31;
    const int warps_per_cta = blockDim.x >> 5;
    const int nvec = p.d >> 3;  // 8 bf16 per 16-byte vector
    const uint4 *__restrict__ gvec = reinterpret_cast<const uint4 *>(p.gain);
    pdl_trigger();  // successors may launch now; they wait for this grid before reading
    pdl_wait();
    const int rows = p.meta[kMetaRows];
    if (static_cast<long long>(blockIdx.x) * warps_per_cta >= rows) return;  // no row here
    for (int v = threadIdx.x; v < nvec; v += blockDim.x) g_smem[v] = __ldg(gvec + v);
    __syncthreads();
    const int sel = p.meta[kMetaSel];
    const int layer0 = p.meta[kMetaLayer0];
    for (int r = blockIdx.x * warps_per_cta + (threadIdx.x >> 5); r < rows;
         r += gridDim.x * warps_per_cta) {
        const int kr = r / sel;
        const int sr = r - kr * sel;
        const int k = layer0 + kr;
        const int q = p.sel_list ? p.sel_list[sr] : sr;
        if (!rpd_check(q >= 0 && q < p.BN, p.meta + kMetaStatus)) continue;  // warp-uniform
        const int pos = p.pos_of_q[q];
        if (!rpd_check(pos >= 0 && pos < p.BN, p.meta + kMetaStatus)) continue;
        const uint4 *__restrict__ src =
            reinterpret_cast<const uint4 *>(p.hidden + (static_cast<size_t>(k) * p.BN + pos) * p.d);
        uint4 *__restrict__ dst = reinterpret_cast<uint4 *>(p.u + static_cast<size_t>(r) * p.d);
        float ss = 0.f;
        for (int v0 = lane; v0 < nvec; v0 += 32 * kVecPerLane) {
            uint4 hv[kVecPerLane];
#pragma unroll
            for (int j = 0; j < kVecPerLane; ++j) {
                const int v = v0 + 32 * j;
                if (v < nvec) hv[j] = __ldcs(src + v);
            }
#pragma unroll
            for (int j = 0; j < kVecPerLane; ++j) {
                const int v = v0 + 32 * j;
                if (v >= nvec) break;
                const uint4 gv = g_smem[v];
                const __nv_bfloat162 *h2 = reinterpret_cast<const __nv_bfloat162 *>(&hv[j]);
                const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gv);
                uint4 out;
                __nv_bfloat162 *o2 = reinterpret_cast<__nv_bfloat162 *>(&out);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 h = __bfloat1622float2(h2[e]);
                    const float2 g = __bfloat1622float2(g2[e]);
                    ss = fmaf(h.x, h.x, ss);
                    ss = fmaf(h.y, h.y, ss);
                    // g*h of two bf16 values is exact in fp32; one RNE to bf16 (reading D1)
                    o2[e] = __float22bfloat162_rn(make_float2(g.x * h.x, g.y * h.y));
                }
                dst[v] = out;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) p.inv_rms[r] = 1.0f / sqrtf(ss / static_cast<float>(p.d) + p.eps);
    }
}

}  // namespace

cudaError_t launch_compact(const CompactParams &p, cudaStream_t s) {
    return launch_pdl(k_compact, dim3(1), dim3(kCompactThreads), 0, s, p);
}

cudaError_t launch_gather_norm(const NormParams &p, int grid, cudaStream_t s) {
    const size_t smem = static_cast<size_t>(p.d) * 2;  // the gain, staged once per CTA
    if (smem > 48 * 1024) {  // set on the current device before every such launch
        cudaError_t e = cudaFuncSetAttribute(k_gather_norm, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    return launch_pdl(k_gather_norm, dim3(grid), dim3(kNormThreads), smem, s, p);
}

}  // namespace rpd
