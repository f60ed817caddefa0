// k_gather_norm.cu - device-side compaction of the masked positions and the RMSNorm
// prologue of the layerwise projection (App. A.6: only masked positions are projected;
// App. A.2: the model's final normalisation is applied to every window layer).
//
// k_compact (one CTA): order-preserving compaction of mask[B][N] into compact indices
//   q = 0..NMT-1 (canvas-major, then position), per-canvas offsets, the projected row
//   count R = K*NMT and the vocabulary split count the head kernel will use.  Nothing
//   goes back to the host: later kernels read these words from device memory.
// k_gather_norm (grid-stride, one warp per row): row r = k*NMT + q reads hidden[k][pos(q)],
//   writes the head operand u[r] = bf16_rne(g * h) (exact product, one rounding) and
//   inv_rms[r] = (mean(h^2) + eps)^(-1/2); the RMS factor is applied after the contraction.
#include "rpd_internal.h"

namespace rpd {
namespace {

constexpr int kCompactThreads = 1024;
constexpr int kCompactItems = 4;

__device__ __forceinline__ int warp_inclusive_scan(int v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int t = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += t;
    }
    return v;
}

__global__ void __launch_bounds__(kCompactThreads, 1) k_compact(CompactParams p) {
    __shared__ int warp_sum[32];
    __shared__ unsigned long long best_split;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int total = p.B * p.N;
    int carry = 0;
    for (int base = 0; base < total; base += kCompactThreads * kCompactItems) {
        const int i0 = base + tid * kCompactItems;
        int f[kCompactItems];
        int cnt = 0;
#pragma unroll
        for (int j = 0; j < kCompactItems; ++j) {
            const int i = i0 + j;
            f[j] = (i < total) ? (p.mask[i] != 0) : 0;
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

    // Vocabulary split count G for the head kernel: units (m-tile, split) are dealt to the
    // grid round-robin; minimise waves * n-tiles-per-unit, smallest G on ties.
    const long long nm_rows = static_cast<long long>(p.K) * carry;
    const long long num_m = (nm_rows + kTileM - 1) / kTileM;
    if (tid == 0) best_split = ~0ull;
    __syncthreads();
    const int gmax = min(p.num_n_tiles, p.max_splits);
    unsigned long long mine = ~0ull;
    if (num_m > 0) {
        for (int g = tid + 1; g <= gmax; g += kCompactThreads) {
            const long long units = num_m * g;
            const long long waves = (units + p.grid_ctas - 1) / p.grid_ctas;
            const long long per = (p.num_n_tiles + g - 1) / g;
            const unsigned long long key =
                (static_cast<unsigned long long>(waves * per) << 20) | static_cast<unsigned>(g);
            mine = key < mine ? key : mine;
        }
        atomicMin(&best_split, mine);
    }
    __syncthreads();
    if (tid == 0) {
        p.canvas_off[p.B] = carry;
        p.meta[kMetaMasked] = carry;
        p.meta[kMetaRows] = static_cast<int>(nm_rows);
        p.meta[kMetaStatus] = RPD_OK;
        p.meta[kMetaSplits] = num_m > 0 ? static_cast<int>(best_split & 0xFFFFFull) : 1;
    }
}

__global__ void __launch_bounds__(256) k_gather_norm(NormParams p) {
    const int nmt = p.meta[kMetaMasked];
    const int rows = p.meta[kMetaRows];
    const int lane = threadIdx.x & 31;
    const int warps_per_cta = blockDim.x >> 5;
    const int nvec = p.d >> 3;  // 8 bf16 per 16-byte vector
    const uint4 *gvec = reinterpret_cast<const uint4 *>(p.gain);
    for (int r = blockIdx.x * warps_per_cta + (threadIdx.x >> 5); r < rows;
         r += gridDim.x * warps_per_cta) {
        const int k = r / nmt;
        const int q = r - k * nmt;
        const int pos = p.pos_of_q[q];
        const uint4 *src =
            reinterpret_cast<const uint4 *>(p.hidden + (static_cast<size_t>(k) * p.BN + pos) * p.d);
        uint4 *dst = reinterpret_cast<uint4 *>(p.u + static_cast<size_t>(r) * p.d);
        float ss = 0.f;
        for (int v = lane; v < nvec; v += 32) {
            const uint4 hv = __ldcs(src + v);
            const uint4 gv = __ldg(gvec + v);
            const __nv_bfloat162 *h2 = reinterpret_cast<const __nv_bfloat162 *>(&hv);
            const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gv);
            uint4 out;
            __nv_bfloat162 *o2 = reinterpret_cast<__nv_bfloat162 *>(&out);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 h = __bfloat1622float2(h2[j]);
                const float2 g = __bfloat1622float2(g2[j]);
                ss = fmaf(h.x, h.x, ss);
                ss = fmaf(h.y, h.y, ss);
                // g*h of two bf16 values is exact in fp32; one RNE to bf16 (reading D1)
                o2[j] = __float22bfloat162_rn(make_float2(g.x * h.x, g.y * h.y));
            }
            dst[v] = out;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (lane == 0) p.inv_rms[r] = 1.0f / sqrtf(ss / static_cast<float>(p.d) + p.eps);
    }
}

}  // namespace

cudaError_t launch_compact(const CompactParams &p, cudaStream_t s) {
    k_compact<<<1, kCompactThreads, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_gather_norm(const NormParams &p, int grid, cudaStream_t s) {
    k_gather_norm<<<grid, 256, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace rpd
