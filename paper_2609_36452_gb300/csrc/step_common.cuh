// step_common.cuh - device routines shared by the step's small kernels: block scans and the
// merge of per-split softmax statistics (the head-tiling plan is in head_plan.h).
#pragma once

#include "head_plan.h"
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
        const bool valid = idx < total &&
                           rpd_check(splits <= mg.max_splits && (idx / span) * sel + s_begin +
                                     (idx - (idx / span) * span) < rows, meta + kMetaStatus);
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
            const int q = sel_list ? sel_list[s] : s;
            if (mg.shard_out) {
                mg.shard_out[static_cast<size_t>(layer0 + kr) * mg.shard_stride + mg.pos_of_q[q]] =
                    make_float4(acc.m, acc.s, acc.t, __int_as_float(acc.a + mg.v_offset));
            } else {
                const size_t out = static_cast<size_t>(layer0 + kr) * nmt + q;
                mg.row_arg[out] = acc.a;
                mg.row_pmax[out] = 1.0f / acc.s;
                mg.row_H[out] = fmaxf(logf(acc.s) - kLn2 * (acc.t / acc.s), 0.f);
            }
        }
    }
    return min(cta_slots, (total + groups - 1) / groups);
}

}  // namespace
}  // namespace rpd
