// rpd_host.cu - the C ABI of include/rpd.h: context, argument checks, scratch, TMA
// descriptors and the launch sequence of one commit step.
//
// Step = k_compact -> k_gather_norm -> k_head_stats -> k_merge -> k_score_commit, all on
// the context's stream, sized from device-resident counts (nothing is read back
// mid-step).  Scratch is owned by the context and sized for the largest B*N seen.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "head_plan.h"
#include "rpd_internal.h"

using namespace rpd;

namespace {

thread_local std::string g_last_error;

int fail(int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return code;
}

int cuda_fail(cudaError_t e, const char *what) {
    return fail(e == cudaErrorMemoryAllocation ? RPD_ERR_OUT_OF_MEMORY : RPD_ERR_CUDA, "%s: %s",
                what, cudaGetErrorString(e));
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static const EncodeTiledFn fn = [] {  // initialised once, thread-safely
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<EncodeTiledFn>(ptr);
        return static_cast<EncodeTiledFn>(nullptr);
    }();
    return fn;
}

// Entry points that touch the GPU run with the context's device current and its primary
// context bound to the calling thread - cudaSetDevice does both; a host thread that has not
// used the CUDA runtime yet has no context, and the driver's tensor-map encoder then fails -
// and give the thread its previous device back when they return.
struct DeviceGuard {
    int prev = -1;
    cudaError_t err = cudaSuccess;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        err = cudaSetDevice(dev);
    }
    ~DeviceGuard() {
        int now = -1;
        if (prev >= 0 && cudaGetDevice(&now) == cudaSuccess && now != prev) cudaSetDevice(prev);
    }
    DeviceGuard(const DeviceGuard &) = delete;
    DeviceGuard &operator=(const DeviceGuard &) = delete;
};

// Row-major bf16 matrix [rows][cols] -> 2-D tensor map with a (64 x box_rows) box and
// 128-byte swizzling; out-of-range elements read as zero.
int encode_bf16_2d(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols,
                   uint32_t box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(RPD_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(kTileK), box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(RPD_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return RPD_OK;
}

}  // namespace

struct rpd_ctx {
    int d = 0, V = 0, K = 0;
    float eps = 0.f;
    int device = 0, num_sms = 0;
    const void *W = nullptr, *g = nullptr;
    int head_layout = RPD_HEAD_TILED;
    void *W_tiled = nullptr;  // the tiled copy of the head (RPD_HEAD_TILED), else null
    rpd_rule rule{0.6f, 3.5f, 15.0f, 6, 32, 0};
    cudaStream_t stream = nullptr;
    rpd_debug dbg{};

    // scratch, sized for cap_bn = B*N positions
    int cap_bn = 0, cap_b = 0, cap_rows = 0, max_splits = 0;
    __nv_bfloat16 *u = nullptr;
    float *inv_rms = nullptr;
    float4 *partials = nullptr;
    int32_t *row_arg = nullptr;
    float *row_pmax = nullptr, *row_H = nullptr;
    int32_t *q_of_pos = nullptr, *pos_of_q = nullptr, *canvas_off = nullptr, *meta = nullptr;
    HeadPlan *plan = nullptr;  // head-tiling plans by pass row count, rows 0..plan_rows
    int plan_rows = 0;
    int32_t *sel_q = nullptr;  // lazy projection: compact indices of the band positions
    int32_t *band_off = nullptr;  // lazy projection: [B+1] each canvas's first band entry
    int v_offset = 0, V_total = 0;  // vocabulary shard: rows of the head are entries
                                    // [v_offset, v_offset + V) of a V_total vocabulary
    int projection = RPD_PROJECT_ALL;
    int tiling = RPD_TILING_AUTO;
    uint64_t wait_limit_ns = kWaitLimitNs;
    bool stall_next = false;  // diagnostics: the next step's head kernels issue no loads
    HeadMaps maps{};     // u (scratch) and W tensor maps of the head kernel
    int head_grid = 0;   // CTAs of the head kernel: 2 x resident clusters of two, <= SMs

    // host-buffer entry point staging: device buffer, and a pinned host copy of its small
    // part (mask, commit, tokens, stats) so that those move in one copy each way
    size_t stage_bytes = 0;
    uint8_t *stage = nullptr;
    size_t stage_host_bytes = 0;
    uint8_t *stage_host = nullptr;

    // profiling
    bool profile = false;
    std::vector<cudaEvent_t> ev_pool;

    // decoding loops built on this context, with the generation of the buffers they were
    // recorded against; the generation moves whenever scratch is reallocated or the head
    // replaced, and a loop recorded against an older one is refused at launch
    uint64_t buffers_gen = 0;
    std::vector<std::pair<cudaGraphExec_t, uint64_t>> loops;
    std::vector<std::pair<int, std::pair<cudaEvent_t, cudaEvent_t>>> ev_rec;
    size_t ev_next = 0;

    void free_scratch() {
        void *ptrs[] = {u, inv_rms, partials, row_arg, row_pmax, row_H, q_of_pos, pos_of_q,
                        canvas_off, meta, sel_q, band_off, plan};
        for (void *p : ptrs)
            if (p) cudaFree(p);
        u = nullptr;
        inv_rms = nullptr;
        partials = nullptr;
        row_arg = nullptr;
        row_pmax = row_H = nullptr;
        q_of_pos = pos_of_q = canvas_off = meta = sel_q = band_off = nullptr;
        plan = nullptr;
        cap_bn = cap_b = cap_rows = plan_rows = 0;
    }
};

namespace {

HeadPlanInputs plan_inputs(const rpd_ctx *c) {
    HeadPlanInputs in;
    in.num_n = (c->V + kTileN - 1) / kTileN;
    in.max_splits = c->max_splits;
    in.pair_slots = c->head_grid / 2;
    in.hbm_tiles = head_stream_in_tiles(c->V, c->d, c->num_sms);
    in.force = c->tiling;
    return in;
}

// The head-tiling plan of every pass row count up to min(scratch rows, kPlanRows), evaluated
// here (memoised by the quantities the plan depends on: the pair tile count, and the rows-on-N
// group count and size) and uploaded to the device table the step's kernels look up.  The
// stream must be idle (no step may be reading the table).
int build_plan(rpd_ctx *c) {
    const int n = std::min(c->cap_rows, kPlanRows);
    if (!c->plan || n < 0) return RPD_OK;
    const HeadPlanInputs in = plan_inputs(c);
    const int gmax2 = std::min(in.num_n, in.max_splits);
    const int gmax3 = std::min(in.num_n, in.max_splits / 2);
    std::vector<HeadPlan> table(static_cast<size_t>(n) + 1);
    std::vector<unsigned long long> key2((n + kPairTileM - 1) / kPairTileM + 1, 0ull);
    std::vector<std::vector<unsigned long long>> key3;  // [groups][ng / step]
    for (int r = 0; r <= n; ++r) {
        if (r == 0 || in.pair_slots <= 0) {
            table[r] = plan_head(r, in);
            continue;
        }
        const int tiles2 = (r + kPairTileM - 1) / kPairTileM;
        if (!key2[tiles2]) key2[tiles2] = best_split_key(kPairTileCost, tiles2, in.pair_slots, in.num_n, gmax2, 1, 1);
        const int groups = swap_groups(r);
        const int ng = swap_group_rows(r, groups);
        unsigned long long k3 = ~0ull;
        if (gmax3 > 0) {
            if (static_cast<int>(key3.size()) <= groups) key3.resize(groups + 1);
            std::vector<unsigned long long> &row = key3[groups];
            const int slot = ng / kSwapRowStep;
            if (static_cast<int>(row.size()) <= slot) row.resize(slot + 1, 0ull);
            if (!row[slot]) row[slot] = best_split_key(swap_tile_cost(ng), groups, in.pair_slots, in.num_n, gmax3, 1, 1);
            k3 = row[slot];
        }
        table[r] = plan_from_keys(in, key2[tiles2], k3, ng);
    }
    cudaError_t e = cudaMemcpy(c->plan, table.data(), table.size() * sizeof(HeadPlan), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy(plan table)");
    c->plan_rows = n;
    return RPD_OK;
}

int ensure_scratch(rpd_ctx *c, int B, int N) {
    const long long bn = static_cast<long long>(B) * N;
    if (bn <= c->cap_bn && B <= c->cap_b) return RPD_OK;
    const int new_bn = static_cast<int>(std::max<long long>(bn, c->cap_bn));
    const int new_b = std::max(B, c->cap_b);
    // padded to whole pair tiles, so that every u box (at most 256 rows) fits in the tensor
    long long rows = static_cast<long long>(c->K) * new_bn;
    rows = ((rows + kPairTileM - 1) / kPairTileM) * kPairTileM;
    if (rows < kPairTileM) rows = kPairTileM;
    if (rows > (1ll << 30)) return fail(RPD_ERR_UNSUPPORTED, "too many projected rows (%lld)", rows);
    cudaError_t e = cudaStreamSynchronize(c->stream);  // no step may still use old scratch
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    c->free_scratch();
    const int num_n = (c->V + kTileN - 1) / kTileN;
    // partials per row: a vocabulary split each (pair tiles), two per split (rows on N)
    c->max_splits = std::min(2 * num_n, 2 * c->num_sms);
    struct {
        void **p;
        size_t bytes;
    } allocs[] = {
        {reinterpret_cast<void **>(&c->u), static_cast<size_t>(rows) * c->d * 2},
        {reinterpret_cast<void **>(&c->inv_rms), static_cast<size_t>(rows) * 4},
        {reinterpret_cast<void **>(&c->partials), static_cast<size_t>(rows) * c->max_splits * 16},
        {reinterpret_cast<void **>(&c->row_arg), static_cast<size_t>(rows) * 4},
        {reinterpret_cast<void **>(&c->row_pmax), static_cast<size_t>(rows) * 4},
        {reinterpret_cast<void **>(&c->row_H), static_cast<size_t>(rows) * 4},
        {reinterpret_cast<void **>(&c->q_of_pos), static_cast<size_t>(new_bn) * 4},
        {reinterpret_cast<void **>(&c->pos_of_q), static_cast<size_t>(new_bn) * 4},
        {reinterpret_cast<void **>(&c->sel_q), static_cast<size_t>(new_bn) * 4},
        {reinterpret_cast<void **>(&c->canvas_off), static_cast<size_t>(new_b + 1) * 4},
        {reinterpret_cast<void **>(&c->band_off), static_cast<size_t>(new_b + 1) * 4},
        {reinterpret_cast<void **>(&c->meta), kMetaWords * 4},
        {reinterpret_cast<void **>(&c->plan),
         (static_cast<size_t>(std::min<long long>(rows, kPlanRows)) + 1) * sizeof(HeadPlan)},
    };
    for (auto &a : allocs) {
        e = cudaMalloc(a.p, a.bytes);
        if (e != cudaSuccess) {
            c->free_scratch();
            return cuda_fail(e, "cudaMalloc(scratch)");
        }
    }
    // the head operand rows past the live count are read by the last tile: keep them finite
    e = cudaMemsetAsync(c->u, 0, static_cast<size_t>(rows) * c->d * 2, c->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(c->meta, 0, kMetaWords * 4, c->stream);
    if (e != cudaSuccess) {
        c->free_scratch();
        return cuda_fail(e, "cudaMemsetAsync(scratch)");
    }
    ++c->buffers_gen;
    c->cap_bn = new_bn;
    c->cap_b = new_b;
    c->cap_rows = static_cast<int>(rows);
    int rc = encode_bf16_2d(&c->maps.u, c->u, static_cast<uint64_t>(rows), c->d, kTileM);
    for (int j = 0; rc == RPD_OK && j < kUMaps; ++j)
        rc = encode_bf16_2d(&c->maps.u_rows[j], c->u, static_cast<uint64_t>(rows), c->d,
                            static_cast<uint32_t>(kUBoxRows * (j + 1)));
    if (rc == RPD_OK) {
        e = cudaStreamSynchronize(c->stream);  // the memsets above precede the table upload
        rc = e == cudaSuccess ? build_plan(c) : cuda_fail(e, "cudaStreamSynchronize");
    }
    return rc;
}

cudaEvent_t take_event(rpd_ctx *c) {
    if (c->ev_next == c->ev_pool.size()) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        c->ev_pool.push_back(e);
    }
    return c->ev_pool[c->ev_next++];
}

struct KernelTimer {
    rpd_ctx *c;
    int kernel;
    cudaEvent_t a = nullptr, b = nullptr;
    KernelTimer(rpd_ctx *ctx, int k) : c(ctx), kernel(k) {
        if (c->profile) {
            a = take_event(c);
            b = take_event(c);
            if (a && b) cudaEventRecord(a, c->stream);
        }
    }
    ~KernelTimer() {
        if (a && b) {
            cudaEventRecord(b, c->stream);
            c->ev_rec.push_back({kernel, {a, b}});
        }
    }
};

int check_rule(const rpd_rule &r) {
    const char *msg = rule_error(r);
    return msg ? fail(RPD_ERR_INVALID_ARGUMENT, "%s", msg) : RPD_OK;
}

int check_call(const rpd_ctx *c, float tau, float budget) {
    const char *msg = call_error(c->rule, tau, budget);
    if (msg)
        return fail(RPD_ERR_INVALID_ARGUMENT, "%s (theta_c %g, tau %g, budget %g)", msg,
                    (double)c->rule.theta_c, (double)tau, (double)budget);
    return RPD_OK;
}

ScoreParams score_params(const rpd_ctx *c, uint8_t *mask, int B, int N, const float *tau,
                         const float *budget, uint8_t *out_commit, int32_t *out_token,
                         rpd_stats *out_stats, bool lazy) {
    ScoreParams sp{};
    sp.mask = mask;
    sp.q_of_pos = c->q_of_pos;
    sp.canvas_off = c->canvas_off;
    sp.meta = c->meta;
    sp.row_arg = c->row_arg;
    sp.row_pmax = c->row_pmax;
    sp.row_H = c->row_H;
    sp.out_commit = out_commit;
    sp.out_token = out_token;
    sp.out_stats = out_stats;
    sp.dbg = c->dbg;
    sp.B = B;
    sp.N = N;
    sp.K = c->K;
    sp.theta_c = c->rule.theta_c;
    sp.theta_s = c->rule.theta_s;
    sp.w = c->rule.w;
    sp.k_max = c->rule.k_max;
    sp.window = c->rule.window;
    sp.block = c->rule.block;
    sp.lazy = lazy ? 1 : 0;
    for (int b = 0; b < B; ++b) {
        sp.tau[b] = tau[b];
        sp.budget[b] = budget[b];
    }
    return sp;
}

// Arguments every single-canvas step checks before it touches the GPU.
int check_canvas(const rpd_ctx *c, const void *hidden, const void *mask, int N) {
    if (!c->W || !c->g) return fail(RPD_ERR_NO_HEAD, "rpd_set_head has not been called");
    if (N < 0) return fail(RPD_ERR_INVALID_ARGUMENT, "N must be >= 0");
    if (N > kMaxCanvas) return fail(RPD_ERR_UNSUPPORTED, "N must be <= %d", kMaxCanvas);
    if (N > 0 && (!hidden || !mask)) return fail(RPD_ERR_INVALID_ARGUMENT, "null buffer");
    if (hidden && !aligned16(hidden))
        return fail(RPD_ERR_INVALID_ARGUMENT, "hidden must be 16-byte aligned");
    if (hidden && !pointer_usable(hidden, c->device, true))
        return fail(RPD_ERR_INVALID_ARGUMENT,
                    "hidden must be device memory of the context's device or mapped page-locked host memory");
    return RPD_OK;
}

int run_step(rpd_ctx *c, const void *hidden, uint8_t *mask, int B, int N, const float *tau,
             const float *budget, uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    if (!c->W || !c->g) return fail(RPD_ERR_NO_HEAD, "rpd_set_head has not been called");
    if (B < 1) return fail(RPD_ERR_INVALID_ARGUMENT, "B must be >= 1");
    if (B > kMaxBatch) return fail(RPD_ERR_UNSUPPORTED, "B must be <= %d", kMaxBatch);
    if (N < 0) return fail(RPD_ERR_INVALID_ARGUMENT, "N must be >= 0");
    if (N > kMaxCanvas) return fail(RPD_ERR_UNSUPPORTED, "N must be <= %d", kMaxCanvas);
    if (!tau || !budget) return fail(RPD_ERR_INVALID_ARGUMENT, "null tau/budget");
    for (int b = 0; b < B; ++b) {
        int rc = check_call(c, tau[b], budget[b]);
        if (rc) return rc;
    }
    if (N == 0) return RPD_OK;
    if (!hidden || !mask || !out_commit || !out_token || !out_stats)
        return fail(RPD_ERR_INVALID_ARGUMENT, "null buffer");
    if (!aligned16(hidden)) return fail(RPD_ERR_INVALID_ARGUMENT, "hidden must be 16-byte aligned");
    if (!pointer_usable(hidden, c->device, true))
        return fail(RPD_ERR_INVALID_ARGUMENT,
                    "hidden must be device memory of the context's device or mapped page-locked host memory");
    int rc = ensure_scratch(c, B, N);
    if (rc) return rc;

    const int bn = B * N;
    const int num_n = (c->V + kTileN - 1) / kTileN;
    const HeadPlanInputs plan_in = plan_inputs(c);
    // Lazy projection (forced, or chosen on the device per step): a second pass over the band.
    // It is not launched when even the largest possible row count keeps a single pass cheaper.
    const bool lazy = c->projection == RPD_PROJECT_LAZY ||
                      (c->projection == RPD_PROJECT_AUTO && c->K > 1 &&
                       static_cast<long long>(c->K) * bn > 2LL * kTileM);
    cudaError_t e;
    {
        KernelTimer t(c, 0);
        CompactParams cp{mask, c->q_of_pos, c->pos_of_q, c->canvas_off, c->meta, B, N, c->K,
                         plan_in, c->plan, c->plan_rows, c->rule.block,
                         c->projection == RPD_PROJECT_LAZY ? 1 : (lazy ? 2 : 0)};
        e = launch_compact(cp, c->stream);
    }
    if (e != cudaSuccess) return cuda_fail(e, "compaction launch");

    // Scoring, scan and commit of every canvas (k_score_commit, or the last merge's grid).
    const ScoreParams sp = score_params(c, mask, B, N, tau, budget, out_commit, out_token,
                                        out_stats, lazy);
    const bool fuse_score = B == 1 && N <= kFuseScoreMaxN;

    // One projection pass: gather + RMSNorm prologue, head statistics, merge.  Rows, layers
    // and positions of the pass come from the device-side meta words.
    const MergeArgs mg{c->partials, c->max_splits, c->row_arg, c->row_pmax, c->row_H};
    auto pass = [&](const int32_t *sel_list, bool last) -> cudaError_t {
        cudaError_t err;
        {
            KernelTimer t(c, 0);
            NormParams np{static_cast<const __nv_bfloat16 *>(hidden),
                          static_cast<const __nv_bfloat16 *>(c->g), c->pos_of_q, sel_list, c->meta,
                          c->u, c->inv_rms, bn, c->d, c->eps};
            // one warp per row: no more CTAs than the largest possible row count needs
            const long long max_rows = static_cast<long long>(c->K) * bn;
            const int grid = static_cast<int>(std::min<long long>(c->num_sms * 8, (max_rows + 7) / 8));
            err = launch_gather_norm(np, grid, c->stream);
        }
        if (err != cudaSuccess) return err;
        {
            KernelTimer t(c, 1);
            HeadParams hp{c->inv_rms, c->partials, c->meta, c->V, c->d, c->max_splits,
                          c->wait_limit_ns, c->stall_next ? 1 : 0, c->W_tiled != nullptr ? 1 : 0};
            // One launch: the kernel reads the tiling chosen on the device for this pass.
            err = launch_head(c->maps, hp, c->head_grid, c->stream);
        }
        if (err != cudaSuccess) return err;
        KernelTimer t(c, 2);
        if (last && fuse_score)
            return launch_merge_score(mg, c->meta, sel_list, c->num_sms * 4, sp, c->stream);
        return launch_merge(mg, c->meta, sel_list, c->num_sms * 4, c->stream);
    };
    e = pass(nullptr, !lazy);
    if (e == cudaSuccess && lazy) {
        {
            KernelTimer t(c, 2);
            BandParams bp{};
            bp.meta = c->meta;
            bp.mg = mg;
            bp.pos_of_q = c->pos_of_q;
            bp.canvas_off = c->canvas_off;
            bp.sel_q = c->sel_q;
            bp.band_off = c->band_off;
            bp.B = B;
            bp.N = N;
            bp.K = c->K;
            bp.theta_c = c->rule.theta_c;
            bp.plan_in = plan_in;
            bp.plan = c->plan;
            bp.plan_rows = c->plan_rows;
            for (int b = 0; b < B; ++b) bp.tau[b] = tau[b];
            e = launch_band(bp, c->stream);
        }
        if (e == cudaSuccess) e = pass(c->sel_q, true);
    }
    c->stall_next = false;
    if (e != cudaSuccess) return cuda_fail(e, "projection launch");
    // The step's last merge also scores the canvas when there is a single canvas of at most
    // kFuseScoreMaxN positions (one launch fewer); otherwise score/commit is its own launch.
    if (fuse_score) return RPD_OK;
    {
        KernelTimer t(c, 3);
        e = launch_score_commit(sp, c->stream);
    }
    if (e != cudaSuccess) return cuda_fail(e, "score/commit launch");
    return RPD_OK;
}

}  // namespace

void rpd::set_last_error(const char *msg) { g_last_error = msg ? msg : ""; }

extern "C" {

const char *rpd_last_error(void) { return g_last_error.c_str(); }

const char *rpd_version(void) { return "rpd-gb300 0.1 (sm_103a, tcgen05 head statistics)"; }

rpd_ctx *rpd_create(int d, int V, int K, float eps) {
    if (d < 64 || d % 8 != 0) {
        fail(RPD_ERR_INVALID_ARGUMENT, "d must be a multiple of 8 and >= 64 (got %d)", d);
        return nullptr;
    }
    if (V < kTileN) {
        fail(RPD_ERR_UNSUPPORTED, "V must be >= %d (got %d)", kTileN, V);
        return nullptr;
    }
    if (K < 1 || K > 64) {
        fail(RPD_ERR_INVALID_ARGUMENT, "K must be in [1, 64] (got %d)", K);
        return nullptr;
    }
    if (!(eps >= 0.f) || !std::isfinite(eps)) {
        fail(RPD_ERR_INVALID_ARGUMENT, "eps must be finite and >= 0");
        return nullptr;
    }
    rpd_ctx *c = new rpd_ctx();
    c->d = d;
    c->V = V;
    c->K = K;
    c->eps = eps;
    cudaError_t e = cudaGetDevice(&c->device);
    if (e == cudaSuccess) e = cudaSetDevice(c->device);  // binds the primary context to this thread
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess) {
        cuda_fail(e, "device query");
        delete c;
        return nullptr;
    }
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, c->device);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, c->device);
    if (major != 10 || minor != 3) {
        fail(RPD_ERR_UNSUPPORTED, "device is sm_%d%d; this library is built for sm_103a", major, minor);
        delete c;
        return nullptr;
    }
    const int clusters = std::min(head_max_clusters(), c->num_sms / 2);
    if (clusters < 1) {
        fail(RPD_ERR_UNSUPPORTED, "the head kernel (clusters of two CTAs) cannot be resident on this device");
        delete c;
        return nullptr;
    }
    c->head_grid = 2 * clusters;
    return c;
}

int rpd_set_head(rpd_ctx *c, const void *W_head, const void *g_norm) {
    if (!c || !W_head || !g_norm) return fail(RPD_ERR_INVALID_ARGUMENT, "null argument");
    if (!aligned16(W_head) || !aligned16(g_norm))
        return fail(RPD_ERR_INVALID_ARGUMENT, "W_head and g_norm must be 16-byte aligned");
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    // The head is read by TMA: it must be device memory of this context's device.
    if (!pointer_usable(W_head, c->device, false) || !pointer_usable(g_norm, c->device, false))
        return fail(RPD_ERR_INVALID_ARGUMENT,
                    "W_head and g_norm must be device memory on the context's device");
    // No step may still read the previous head (or its tiled copy) once it is replaced.
    cudaError_t e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    if (c->W_tiled) cudaFree(c->W_tiled);
    c->W_tiled = nullptr;
    c->W = nullptr;
    ++c->buffers_gen;
    CUtensorMap m2;
    int rc;
    if (c->head_layout == RPD_HEAD_TILED && c->d % 64 == 0) {
        // rows as 2-D tensor map rows of 64 columns: block (t, k) is map rows
        // [128 (t (d/64) + k), +128)
        const uint64_t vpad = (static_cast<uint64_t>(c->V) + 127) / 128 * 128;
        void *wt = nullptr;
        e = cudaMalloc(&wt, vpad * static_cast<uint64_t>(c->d) * 2);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(tiled head)");
        e = launch_tile_head(W_head, wt, c->V, c->d, c->stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
        if (e != cudaSuccess) {
            cudaFree(wt);
            return cuda_fail(e, "tiled copy of the head");
        }
        rc = encode_bf16_2d(&m2, wt, vpad * static_cast<uint64_t>(c->d) / 64, 64, kPairHalfRows);
        if (rc) {
            cudaFree(wt);
            return rc;
        }
        c->W_tiled = wt;
    } else {
        rc = encode_bf16_2d(&m2, W_head, static_cast<uint64_t>(c->V), c->d, kPairHalfRows);
        if (rc) return rc;
    }
    c->maps.w128 = m2;
    ++c->buffers_gen;
    c->W = W_head;
    c->g = g_norm;
    return RPD_OK;
}

int rpd_set_rule(rpd_ctx *c, const rpd_rule *r) {
    if (!c || !r) return fail(RPD_ERR_INVALID_ARGUMENT, "null argument");
    int rc = check_rule(*r);
    if (rc) return rc;
    c->rule = *r;
    return RPD_OK;
}

int rpd_get_rule(const rpd_ctx *c, rpd_rule *r) {
    if (!c || !r) return fail(RPD_ERR_INVALID_ARGUMENT, "null argument");
    *r = c->rule;
    return RPD_OK;
}

int rpd_set_stream(rpd_ctx *c, void *stream) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    c->stream = static_cast<cudaStream_t>(stream);
    return RPD_OK;
}

int rpd_reserve(rpd_ctx *c, int B, int N) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    if (B < 1 || N < 1) return fail(RPD_ERR_INVALID_ARGUMENT, "reserve: B and N must be >= 1");
    if (B > kMaxBatch || N > kMaxCanvas)
        return fail(RPD_ERR_UNSUPPORTED, "reserve: B <= %d, N <= %d", kMaxBatch, kMaxCanvas);
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    return ensure_scratch(c, B, N);
}

int rpd_set_projection(rpd_ctx *c, int mode) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    if (mode != RPD_PROJECT_ALL && mode != RPD_PROJECT_LAZY && mode != RPD_PROJECT_AUTO)
        return fail(RPD_ERR_INVALID_ARGUMENT, "unknown projection mode %d", mode);
    c->projection = mode;
    return RPD_OK;
}

int rpd_set_head_layout(rpd_ctx *c, int layout) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    if (layout != RPD_HEAD_TILED && layout != RPD_HEAD_BORROWED)
        return fail(RPD_ERR_INVALID_ARGUMENT, "unknown head layout %d", layout);
    c->head_layout = layout;
    return RPD_OK;
}

int rpd_set_head_tiling(rpd_ctx *c, int tiling) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    if (tiling < RPD_TILING_AUTO || tiling > RPD_TILING_ROWS_N)
        return fail(RPD_ERR_INVALID_ARGUMENT, "unknown head tiling %d", tiling);
    if (tiling == c->tiling) return RPD_OK;
    c->tiling = tiling;
    if (!c->plan) return RPD_OK;
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    cudaError_t e = cudaStreamSynchronize(c->stream);  // no step may still read the plan table
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    return build_plan(c);
}

int rpd_set_wait_limit(rpd_ctx *c, int64_t microseconds) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    if (microseconds < 1000) return fail(RPD_ERR_INVALID_ARGUMENT, "wait limit must be >= 1000 us");
    c->wait_limit_ns = static_cast<uint64_t>(microseconds) * 1000ull;
    return RPD_OK;
}

int rpd_inject_stall(rpd_ctx *c) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    c->stall_next = true;
    return RPD_OK;
}

int rpd_set_debug(rpd_ctx *c, const rpd_debug *dbg) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    if (dbg)
        c->dbg = *dbg;
    else
        c->dbg = rpd_debug{};
    return RPD_OK;
}

int rpd_step(rpd_ctx *c, const void *hidden, uint8_t *mask, int N, float tau, float budget,
             uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats) {
    return run_step(c, hidden, mask, 1, N, &tau, &budget, out_commit, out_token, out_stats);
}

namespace {

// One attempt at the decoding-loop graph (see rpd_build_decode_loop); `no_pdl` records the
// step's launches without programmatic dependencies.
int build_decode_loop_once(rpd_ctx *c, cudaGraph_t forward, const void *hidden, uint8_t *mask,
                           int B, int N, const float *tau, const float *budget, uint8_t *out_commit,
                           int32_t *out_token, rpd_stats *out_stats, float stop_frac, int max_steps,
                           int32_t *steps, bool no_pdl, cudaGraphExec_t *out_exec) {
    cudaStream_t cs = nullptr;
    cudaGraph_t g = nullptr;
    cudaError_t e = cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaGraphCreate(&g, 0);
    cudaGraphConditionalHandle handle = 0;
    // the condition is 1 at the start of every launch: the body runs at least once
    if (e == cudaSuccess) e = cudaGraphConditionalHandleCreate(&handle, g, 1, cudaGraphCondAssignDefault);
    // steps = 0, then while (condition) { forward; step; stop test }
    cudaGraphNode_t zero = nullptr, loop = nullptr;
    if (e == cudaSuccess) {
        cudaMemsetParams ms = {};
        ms.dst = steps;
        ms.value = 0;
        ms.elementSize = 4;
        ms.width = 1;
        ms.height = 1;
        e = cudaGraphAddMemsetNode(&zero, g, nullptr, 0, &ms);
    }
    cudaGraph_t body = nullptr;
    if (e == cudaSuccess) {
        cudaGraphNodeParams cp = {};
        cp.type = cudaGraphNodeTypeConditional;
        cp.conditional.handle = handle;
        cp.conditional.type = cudaGraphCondTypeWhile;
        cp.conditional.size = 1;
        e = cudaGraphAddNode(&loop, g, &zero, nullptr, 1, &cp);
        if (e == cudaSuccess) body = cp.conditional.phGraph_out[0];
    }
    cudaGraphNode_t fwd = nullptr;
    if (e == cudaSuccess && forward) e = cudaGraphAddChildGraphNode(&fwd, body, nullptr, 0, forward);
    int rc = RPD_OK;
    if (e == cudaSuccess) {
        e = cudaStreamBeginCaptureToGraph(cs, body, fwd ? &fwd : nullptr, nullptr, fwd ? 1 : 0,
                                          cudaStreamCaptureModeThreadLocal);
        if (e == cudaSuccess) {
            cudaStream_t saved = c->stream;
            const bool saved_profile = c->profile;
            c->stream = cs;
            c->profile = false;
            t_no_pdl = no_pdl;
            rc = run_step(c, hidden, mask, B, N, tau, budget, out_commit, out_token, out_stats);
            cudaError_t el = rc == RPD_OK ? launch_loop_test(handle, out_stats, B, N, stop_frac,
                                                             max_steps, steps, cs)
                                          : cudaSuccess;
            t_no_pdl = false;
            c->stream = saved;
            c->profile = saved_profile;
            cudaGraph_t captured = nullptr;
            e = cudaStreamEndCapture(cs, &captured);
            if (e == cudaSuccess) e = el;
        }
    }
    cudaGraphExec_t exec = nullptr;
    if (rc == RPD_OK && e == cudaSuccess) e = cudaGraphInstantiate(&exec, g, 0);
    if (g) cudaGraphDestroy(g);
    if (cs) cudaStreamDestroy(cs);
    if (rc != RPD_OK) return rc;
    if (e != cudaSuccess) {
        cudaGetLastError();
        return cuda_fail(e, "decoding-loop graph");
    }
    *out_exec = exec;
    return RPD_OK;
}

}  // namespace

namespace {

int build_decode_loop(rpd_ctx *c, void *forward, const void *hidden, uint8_t *mask, int B, int N,
                      const float *tau, const float *budget, uint8_t *out_commit, int32_t *out_token,
                      rpd_stats *out_stats, float stop_frac, int max_steps, int32_t *steps,
                      void **out_exec) {
    if (!c || !out_exec || !steps || !hidden || !mask || !out_commit || !out_token || !out_stats ||
        !tau || !budget)
        return fail(RPD_ERR_INVALID_ARGUMENT, "null argument");
    *out_exec = nullptr;
    if (B < 1 || B > kMaxBatch) return fail(RPD_ERR_INVALID_ARGUMENT, "B must be in [1, %d]", kMaxBatch);
    if (N < 1 || N > kMaxCanvas) return fail(RPD_ERR_INVALID_ARGUMENT, "N must be in [1, %d]", kMaxCanvas);
    if (!(stop_frac >= 0.f && stop_frac <= 1.f))
        return fail(RPD_ERR_INVALID_ARGUMENT, "stop_frac must be in [0, 1]");
    if (max_steps < 1) return fail(RPD_ERR_INVALID_ARGUMENT, "max_steps must be >= 1");
    if (c->V_total > 0) return fail(RPD_ERR_UNSUPPORTED, "a vocabulary slice has no decoding loop");
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    if (!pointer_usable(steps, c->device, false) || !pointer_usable(mask, c->device, false) ||
        !pointer_usable(hidden, c->device, false))
        return fail(RPD_ERR_INVALID_ARGUMENT, "hidden, mask and steps must be device memory");
    for (int b = 0; b < B; ++b) {
        int rc = check_call(c, tau[b], budget[b]);
        if (rc) return rc;
    }
    int rc = ensure_scratch(c, B, N);  // nothing may allocate while the step is recorded
    if (rc) return rc;
    cudaGraphExec_t exec = nullptr;
    rc = build_decode_loop_once(c, static_cast<cudaGraph_t>(forward), hidden, mask, B, N, tau, budget,
                                out_commit, out_token, out_stats, stop_frac, max_steps, steps, false,
                                &exec);
    if (rc == RPD_ERR_CUDA)  // a loop body may refuse programmatic dependencies: plain order
        rc = build_decode_loop_once(c, static_cast<cudaGraph_t>(forward), hidden, mask, B, N, tau,
                                    budget, out_commit, out_token, out_stats, stop_frac, max_steps,
                                    steps, true, &exec);
    if (rc) return rc;
    c->loops.push_back({exec, c->buffers_gen});
    *out_exec = exec;
    return RPD_OK;
}

}  // namespace

int rpd_build_decode_loop(rpd_ctx *c, void *forward, const void *hidden, uint8_t *mask, int N,
                          float tau, float budget, uint8_t *out_commit, int32_t *out_token,
                          rpd_stats *out_stats, float stop_frac, int max_steps, int32_t *steps,
                          void **out_exec) {
    return build_decode_loop(c, forward, hidden, mask, 1, N, &tau, &budget, out_commit, out_token,
                             out_stats, stop_frac, max_steps, steps, out_exec);
}

int rpd_build_decode_loop_batched(rpd_ctx *c, void *forward, const void *hidden, uint8_t *mask,
                                  int B, int N, const float *tau, const float *budget,
                                  uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats,
                                  float stop_frac, int max_steps, int32_t *steps, void **out_exec) {
    return build_decode_loop(c, forward, hidden, mask, B, N, tau, budget, out_commit, out_token,
                             out_stats, stop_frac, max_steps, steps, out_exec);
}

int rpd_decode_loop_launch(rpd_ctx *c, void *exec, void *stream) {
    if (!c || !exec) return fail(RPD_ERR_INVALID_ARGUMENT, "null argument");
    for (const auto &l : c->loops) {
        if (l.first != static_cast<cudaGraphExec_t>(exec)) continue;
        if (l.second != c->buffers_gen)
            return fail(RPD_ERR_INVALID_ARGUMENT,
                        "the context's scratch or head changed after the loop was built: rebuild it");
        DeviceGuard dg(c->device);
        if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
        cudaError_t e = cudaGraphLaunch(l.first, static_cast<cudaStream_t>(stream));
        return e == cudaSuccess ? RPD_OK : cuda_fail(e, "cudaGraphLaunch");
    }
    return fail(RPD_ERR_INVALID_ARGUMENT, "not a decoding loop of this context");
}

void rpd_decode_loop_destroy(rpd_ctx *c, void *exec) {
    if (!c || !exec) return;
    for (size_t i = 0; i < c->loops.size(); ++i) {
        if (c->loops[i].first != static_cast<cudaGraphExec_t>(exec)) continue;
        DeviceGuard dg(c->device);
        cudaGraphExecDestroy(c->loops[i].first);
        c->loops.erase(c->loops.begin() + static_cast<long>(i));
        return;
    }
}

int rpd_step_batched(rpd_ctx *c, const void *hidden, uint8_t *mask, int B, int N, const float *tau,
                     const float *budget, uint8_t *out_commit, int32_t *out_token,
                     rpd_stats *out_stats) {
    return run_step(c, hidden, mask, B, N, tau, budget, out_commit, out_token, out_stats);
}

int rpd_step_host(rpd_ctx *c, const void *hidden, uint8_t *mask, int N, float tau, float budget,
                  uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    if (N < 0) return fail(RPD_ERR_INVALID_ARGUMENT, "N must be >= 0");
    if (N > kMaxCanvas) return fail(RPD_ERR_UNSUPPORTED, "N must be <= %d", kMaxCanvas);
    if (N == 0) return run_step(c, nullptr, nullptr, 1, 0, &tau, &budget, nullptr, nullptr, nullptr);
    if (!hidden || !mask || !out_commit || !out_token || !out_stats)
        return fail(RPD_ERR_INVALID_ARGUMENT, "null buffer");
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    // Pinned (page-locked, mapped) host memory is read in place by the gather kernel over the
    // host link: only the masked positions' rows cross it, and no copy precedes the step.
    // Any other host memory is copied to the device first.
    const void *in_place = nullptr;
    {
        cudaPointerAttributes a{};
        if (cudaPointerGetAttributes(&a, hidden) == cudaSuccess && a.type == cudaMemoryTypeHost)
            in_place = a.devicePointer;
        cudaGetLastError();  // clear the (non-sticky) error the query may have recorded
    }
    const size_t hid = in_place ? 0 : static_cast<size_t>(c->K) * N * c->d * 2;
    const size_t off_mask = (hid + 255) & ~size_t(255);
    const size_t off_commit = off_mask + ((N + 255) & ~255);
    const size_t off_token = off_commit + ((N + 255) & ~255);
    const size_t off_stats = off_token + ((static_cast<size_t>(N) * 4 + 255) & ~size_t(255));
    const size_t need = off_stats + 256;
    if (need > c->stage_bytes) {
        cudaError_t e = cudaStreamSynchronize(c->stream);
        if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
        if (c->stage) cudaFree(c->stage);
        c->stage = nullptr;
        c->stage_bytes = 0;
        e = cudaMalloc(&c->stage, need);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(staging)");
        c->stage_bytes = need;
    }
    const size_t small = need - off_mask;  // mask, commit, tokens, stats (with padding)
    if (small > c->stage_host_bytes) {
        if (c->stage_host) cudaFreeHost(c->stage_host);
        c->stage_host = nullptr;
        c->stage_host_bytes = 0;
        cudaError_t e = cudaMallocHost(&c->stage_host, small);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMallocHost(staging)");
        c->stage_host_bytes = small;
    }
    const void *d_hidden = in_place ? in_place : c->stage;
    uint8_t *d_mask = c->stage + off_mask;
    uint8_t *d_commit = c->stage + off_commit;
    int32_t *d_token = reinterpret_cast<int32_t *>(c->stage + off_token);
    rpd_stats *d_stats = reinterpret_cast<rpd_stats *>(c->stage + off_stats);
    uint8_t *h = c->stage_host;  // same layout as the device region from off_mask on
    // tokens are written only where committed: the step starts from the caller's canvas
    std::memcpy(h, mask, static_cast<size_t>(N));
    std::memcpy(h + (off_token - off_mask), out_token, static_cast<size_t>(N) * 4);
    cudaError_t e = cudaSuccess;
    if (!in_place) e = cudaMemcpyAsync(c->stage, hidden, hid, cudaMemcpyHostToDevice, c->stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(d_mask, h, off_stats - off_mask, cudaMemcpyHostToDevice, c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "host->device copy");
    int rc = run_step(c, d_hidden, d_mask, 1, N, &tau, &budget, d_commit, d_token, d_stats);
    if (rc) return rc;
    e = cudaMemcpyAsync(h, d_mask, small, cudaMemcpyDeviceToHost, c->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "device->host copy");
    std::memcpy(mask, h, static_cast<size_t>(N));
    std::memcpy(out_commit, h + (off_commit - off_mask), static_cast<size_t>(N));
    std::memcpy(out_token, h + (off_token - off_mask), static_cast<size_t>(N) * 4);
    std::memcpy(out_stats, h + (off_stats - off_mask), sizeof(rpd_stats));
    return RPD_OK;
}

int rpd_set_vocab_shard(rpd_ctx *c, int v_offset, int V_total) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    if (v_offset < 0 || V_total < c->V || v_offset > V_total - c->V)
        return fail(RPD_ERR_INVALID_ARGUMENT,
                    "shard [%d, %d + %d) must lie inside a vocabulary of %d entries", v_offset,
                    v_offset, c->V, V_total);
    c->v_offset = v_offset;
    c->V_total = V_total;
    return RPD_OK;
}

int rpd_step_shard_partials(rpd_ctx *c, const void *hidden, const uint8_t *mask, int N,
                            float *out_partials) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    int rc = check_canvas(c, hidden, mask, N);
    if (rc) return rc;
    if (c->projection != RPD_PROJECT_ALL)
        return fail(RPD_ERR_UNSUPPORTED,
                    "vocabulary-sharded steps project every window layer (RPD_PROJECT_ALL)");
    if (N == 0) return RPD_OK;
    if (!out_partials || !aligned16(out_partials))
        return fail(RPD_ERR_INVALID_ARGUMENT, "out_partials must be 16-byte aligned device memory");
    rc = ensure_scratch(c, 1, N);
    if (rc) return rc;
    const HeadPlanInputs plan_in = plan_inputs(c);
    CompactParams cp{mask, c->q_of_pos, c->pos_of_q, c->canvas_off, c->meta, 1, N, c->K,
                     plan_in, c->plan, c->plan_rows, c->rule.block, 0};
    cudaError_t e = launch_compact(cp, c->stream);
    if (e == cudaSuccess) {
        NormParams np{static_cast<const __nv_bfloat16 *>(hidden),
                      static_cast<const __nv_bfloat16 *>(c->g), c->pos_of_q, nullptr, c->meta,
                      c->u, c->inv_rms, N, c->d, c->eps};
        const long long max_rows = static_cast<long long>(c->K) * N;
        e = launch_gather_norm(np, static_cast<int>(std::min<long long>(c->num_sms * 8, (max_rows + 7) / 8)),
                               c->stream);
    }
    if (e == cudaSuccess) {
        HeadParams hp{c->inv_rms, c->partials, c->meta, c->V, c->d, c->max_splits, c->wait_limit_ns,
                      c->stall_next ? 1 : 0, c->W_tiled != nullptr ? 1 : 0};
        e = launch_head(c->maps, hp, c->head_grid, c->stream);
        c->stall_next = false;
    }
    if (e == cudaSuccess) {
        MergeArgs mg{c->partials, c->max_splits, c->row_arg, c->row_pmax, c->row_H,
                     reinterpret_cast<float4 *>(out_partials), c->pos_of_q, N, c->v_offset};
        e = launch_merge(mg, c->meta, nullptr, c->num_sms * 4, c->stream);
    }
    if (e != cudaSuccess) return cuda_fail(e, "sharded projection launch");
    return RPD_OK;
}

int rpd_step_shard_finish(rpd_ctx *c, const float *gathered, int P, uint8_t *mask, int N, float tau,
                          float budget, uint8_t *out_commit, int32_t *out_token,
                          rpd_stats *out_stats) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    if (P < 1 || P > 4096) return fail(RPD_ERR_INVALID_ARGUMENT, "P must be in [1, 4096]");
    int rc = check_call(c, tau, budget);
    if (rc) return rc;
    if (N < 0) return fail(RPD_ERR_INVALID_ARGUMENT, "N must be >= 0");
    if (N > kMaxCanvas) return fail(RPD_ERR_UNSUPPORTED, "N must be <= %d", kMaxCanvas);
    if (N == 0) return RPD_OK;
    if (!gathered || !mask || !out_commit || !out_token || !out_stats)
        return fail(RPD_ERR_INVALID_ARGUMENT, "null buffer");
    if (!aligned16(gathered)) return fail(RPD_ERR_INVALID_ARGUMENT, "gathered must be 16-byte aligned");
    rc = ensure_scratch(c, 1, N);
    if (rc) return rc;
    const HeadPlanInputs plan_in = plan_inputs(c);
    CompactParams cp{mask, c->q_of_pos, c->pos_of_q, c->canvas_off, c->meta, 1, N, c->K,
                     plan_in, c->plan, c->plan_rows, c->rule.block, 0,
                     1 /* keep the partials call's status (a timed-out wait) */};
    cudaError_t e = launch_compact(cp, c->stream);
    if (e == cudaSuccess) {
        ShardMergeParams mp{reinterpret_cast<const float4 *>(gathered), P, c->K, N, c->pos_of_q,
                            c->meta, c->row_arg, c->row_pmax, c->row_H};
        e = launch_merge_shards(mp, c->num_sms * 2, c->stream);
    }
    if (e == cudaSuccess) {
        const ScoreParams sp = score_params(c, mask, 1, N, &tau, &budget, out_commit, out_token,
                                            out_stats, false);
        e = launch_score_commit(sp, c->stream);
    }
    if (e != cudaSuccess) return cuda_fail(e, "shard merge / score launch");
    return RPD_OK;
}

int rpd_profile_enable(rpd_ctx *c, int enable) {
    if (!c) return fail(RPD_ERR_INVALID_ARGUMENT, "null context");
    c->profile = enable != 0;
    return RPD_OK;
}

int rpd_kernel_times(rpd_ctx *c, double *ms, int64_t *launches, int reset) {
    if (!c || !ms || !launches) return fail(RPD_ERR_INVALID_ARGUMENT, "null argument");
    DeviceGuard dg(c->device);
    if (dg.err != cudaSuccess) return cuda_fail(dg.err, "cudaSetDevice");
    for (int k = 0; k < RPD_NUM_KERNELS; ++k) {
        ms[k] = 0.0;
        launches[k] = 0;
    }
    for (auto &r : c->ev_rec) {
        cudaError_t e = cudaEventSynchronize(r.second.second);
        if (e != cudaSuccess) return cuda_fail(e, "cudaEventSynchronize");
        float t = 0.f;
        e = cudaEventElapsedTime(&t, r.second.first, r.second.second);
        if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
        ms[r.first] += t;
        launches[r.first] += 1;
    }
    if (reset) {
        c->ev_rec.clear();
        c->ev_next = 0;
    }
    return RPD_OK;
}

void rpd_destroy(rpd_ctx *c) {
    if (!c) return;
    DeviceGuard dg(c->device);
    cudaStreamSynchronize(c->stream);
    for (auto &l : c->loops) cudaGraphExecDestroy(l.first);
    c->free_scratch();
    if (c->W_tiled) cudaFree(c->W_tiled);
    if (c->stage) cudaFree(c->stage);
    if (c->stage_host) cudaFreeHost(c->stage_host);
    for (cudaEvent_t e : c->ev_pool) cudaEventDestroy(e);
    delete c;
}

}  // extern "C"
