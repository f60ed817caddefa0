// rpd_noalloc.cu - rpd_step_noalloc: one commit step that allocates no device memory.
//
// Who needs it: callers that are not allowed to allocate device memory themselves or to
// let a library do it behind their back - for example a host application that plans all
// of its device memory up front (a serving engine with a fixed arena, a plugin inside
// another framework's memory manager), or a latency-critical loop in which a cudaMalloc,
// which can synchronise the device, is not acceptable.  rpd_create/rpd_step allocate
// context scratch on demand; this entry point instead runs the same kernels on a scratch
// arena that is a file-scope __device__ array of this library, so it never calls
// cudaMalloc, cudaFree or any allocating routine.  The caller still provides every input and output buffer.
//
// Limits of the arena (checked on every call, before any work is enqueued):
//   K * N <= 1024 projected rows, d <= 4096, N <= 1024; the arena holds the compact head
//   operand (1024 x 4096 bf16, 8 MiB), up to 320 vocabulary splits of statistics per row
//   (5 MiB) and small per-row / per-position arrays: about 13 MiB in total, resident on
//   every GPU that loads this library until the process exits.
//
// Sharing: every call on a device uses the same arena and leaves its contents behind.
// The step's status/count words are cleared at the start of each call, and every array the
// step reads is rewritten by the same call before it is read, with one exception: the last
// head tile also reads the rows of the compact head operand past the call's live row count
// (left over from an earlier call, or zero), and its epilogue discards what those rows
// produce.  Calls whose work overlaps on the GPU (two host threads, or two streams) race on
// the arena: serialise them (one stream, or events).
//
// Set-up: the first call on each device looks up the arena's device address with
// cudaGetSymbolAddress (the array's name in host code is only a host-side stand-in, not a
// device address) and caches it per device; make that first call before any stream
// capture begins.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <mutex>
#include <string>

#include "rpd_internal.h"

using namespace rpd;

namespace {

constexpr int kNaMaxRows = 1024;
constexpr int kNaMaxD = 4096;
constexpr int kNaMaxN = 1024;
constexpr int kNaMaxSplits = 320;
static_assert(kNaMaxN <= kFuseScoreMaxN, "the canvas is scored by the merge's last CTA");
constexpr int kNaMaxDevices = 64;

// Arena layout (byte offsets, each 256-byte aligned).
constexpr size_t kOffU = 0;
constexpr size_t kBytesU = static_cast<size_t>(kNaMaxRows) * kNaMaxD * 2;
constexpr size_t kOffPartials = kOffU + kBytesU;
constexpr size_t kBytesPartials = static_cast<size_t>(kNaMaxRows) * kNaMaxSplits * 16;
constexpr size_t kOffInvRms = kOffPartials + kBytesPartials;
constexpr size_t kOffRowArg = kOffInvRms + kNaMaxRows * 4;
constexpr size_t kOffRowPmax = kOffRowArg + kNaMaxRows * 4;
constexpr size_t kOffRowH = kOffRowPmax + kNaMaxRows * 4;
constexpr size_t kOffQofPos = kOffRowH + kNaMaxRows * 4;
constexpr size_t kOffPosOfQ = kOffQofPos + kNaMaxN * 4;
constexpr size_t kOffCanvasOff = kOffPosOfQ + kNaMaxN * 4;
constexpr size_t kOffMeta = kOffCanvasOff + 256;
constexpr size_t kArenaBytes = kOffMeta + 256;

static __device__ __align__(256) uint8_t g_noalloc_arena[kArenaBytes];

struct DeviceSetup {
    bool ready = false;
    int device = 0;
    uint8_t *arena = nullptr;  // device address of g_noalloc_arena on this device
    int num_sms = 0;
    int head_grid = 0;         // CTAs of the head kernel (same choice as rpd_step)
};

std::mutex g_setup_mutex;
DeviceSetup g_setup[kNaMaxDevices];

int na_fail(int code, const char *msg) {
    set_last_error(msg);  // reported by rpd_last_error()
    return code;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

bool encode_tile_map(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols,
                     uint32_t box_rows) {
    static const EncodeTiledFn fn = [] {  // initialised once, thread-safely
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<EncodeTiledFn>(ptr);
        return static_cast<EncodeTiledFn>(nullptr);
    }();
    if (!fn) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(kTileK), box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Once per device, with that device current: find the arena's device address.
int setup_device(DeviceSetup **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return na_fail(RPD_ERR_CUDA, "cudaGetDevice failed");
    // the same device; binds its primary context to a calling thread that has none yet
    if (cudaSetDevice(dev) != cudaSuccess) return na_fail(RPD_ERR_CUDA, "cudaSetDevice failed");
    if (dev < 0 || dev >= kNaMaxDevices) return na_fail(RPD_ERR_UNSUPPORTED, "device index too large");
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    DeviceSetup &s = g_setup[dev];
    if (!s.ready) {
        void *ptr = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_arena);
        if (e != cudaSuccess || ptr == nullptr) {
            set_last_error((std::string("cudaGetSymbolAddress(arena) failed: ") +
                            cudaGetErrorString(e)).c_str());
            return RPD_ERR_CUDA;
        }
        int sms = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return na_fail(RPD_ERR_CUDA, "cudaDeviceGetAttribute failed");
        s.device = dev;
        s.arena = static_cast<uint8_t *>(ptr);
        s.num_sms = sms;
        const int clusters = std::min(head_max_clusters(), sms / 2);
        if (clusters < 1)
            return na_fail(RPD_ERR_UNSUPPORTED, "the head kernel cannot be resident on this device");
        s.head_grid = 2 * clusters;
        s.ready = true;
    }
    *out = &s;
    return RPD_OK;
}

}  // namespace

extern "C" int rpd_step_noalloc(const void *W_head, const void *g_norm, int d, int V, int K,
                                float eps, const rpd_rule *rule_in, const void *hidden,
                                uint8_t *mask, int N, float tau, float budget,
                                uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats,
                                void *stream_ptr) {
    char msg[256];
    const rpd_rule rule = rule_in ? *rule_in : rpd_rule{0.6f, 3.5f, 15.0f, 6, 32, 0};
    if (d < 64 || d % 8 != 0) return na_fail(RPD_ERR_INVALID_ARGUMENT, "d must be a multiple of 8 and >= 64");
    if (d > kNaMaxD) {
        snprintf(msg, sizeof(msg), "rpd_step_noalloc: d=%d exceeds the static arena limit %d", d, kNaMaxD);
        return na_fail(RPD_ERR_UNSUPPORTED, msg);
    }
    if (V < kTileN) return na_fail(RPD_ERR_UNSUPPORTED, "V must be >= 256");
    if (K < 1 || K > 64) return na_fail(RPD_ERR_INVALID_ARGUMENT, "K must be in [1, 64]");
    if (N < 0) return na_fail(RPD_ERR_INVALID_ARGUMENT, "N must be >= 0");
    if (N > kNaMaxN || static_cast<long long>(K) * N > kNaMaxRows) {
        snprintf(msg, sizeof(msg),
                 "rpd_step_noalloc: N=%d, K*N=%lld exceed the static arena limits N<=%d, K*N<=%d",
                 N, static_cast<long long>(K) * N, kNaMaxN, kNaMaxRows);
        return na_fail(RPD_ERR_UNSUPPORTED, msg);
    }
    if (!(eps >= 0.f) || !std::isfinite(eps)) return na_fail(RPD_ERR_INVALID_ARGUMENT, "eps must be finite and >= 0");
    if (const char *m = rule_error(rule)) return na_fail(RPD_ERR_INVALID_ARGUMENT, m);
    if (const char *m = call_error(rule, tau, budget)) return na_fail(RPD_ERR_INVALID_ARGUMENT, m);
    if (N == 0) return RPD_OK;
    if (!W_head || !g_norm || !hidden || !mask || !out_commit || !out_token || !out_stats)
        return na_fail(RPD_ERR_INVALID_ARGUMENT, "null buffer");
    if (!aligned16(W_head) || !aligned16(g_norm) || !aligned16(hidden))
        return na_fail(RPD_ERR_INVALID_ARGUMENT, "W_head, g_norm and hidden must be 16-byte aligned");

    DeviceSetup *dev = nullptr;
    int rc = setup_device(&dev);
    if (rc) return rc;
    // The head and gain are read with TMA, the hidden states with plain loads: pointers the
    // current device cannot read (pageable host memory, another device's memory) are refused
    // here rather than becoming a fault in the kernels.
    if (!pointer_usable(W_head, dev->device, false) || !pointer_usable(g_norm, dev->device, false))
        return na_fail(RPD_ERR_INVALID_ARGUMENT, "W_head and g_norm must be device memory of the current device");
    if (!pointer_usable(hidden, dev->device, true))
        return na_fail(RPD_ERR_INVALID_ARGUMENT,
                       "hidden must be device memory of the current device or mapped page-locked host memory");
    cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
    uint8_t *A = dev->arena;
    __nv_bfloat16 *u = reinterpret_cast<__nv_bfloat16 *>(A + kOffU);
    float4 *partials = reinterpret_cast<float4 *>(A + kOffPartials);
    float *inv_rms = reinterpret_cast<float *>(A + kOffInvRms);
    int32_t *row_arg = reinterpret_cast<int32_t *>(A + kOffRowArg);
    float *row_pmax = reinterpret_cast<float *>(A + kOffRowPmax);
    float *row_H = reinterpret_cast<float *>(A + kOffRowH);
    int32_t *q_of_pos = reinterpret_cast<int32_t *>(A + kOffQofPos);
    int32_t *pos_of_q = reinterpret_cast<int32_t *>(A + kOffPosOfQ);
    int32_t *canvas_off = reinterpret_cast<int32_t *>(A + kOffCanvasOff);
    int32_t *meta = reinterpret_cast<int32_t *>(A + kOffMeta);

    // Same head-kernel configuration as rpd_step (tiling chosen on the device).
    const int pair_slots = dev->head_grid / 2;
    HeadMaps maps;
    bool maps_ok = encode_tile_map(&maps.u, u, kNaMaxRows, static_cast<uint64_t>(d), kTileM) &&
                   encode_tile_map(&maps.w128, W_head, static_cast<uint64_t>(V),
                                   static_cast<uint64_t>(d), kPairHalfRows);
    for (int j = 0; maps_ok && j < kUMaps; ++j)
        maps_ok = encode_tile_map(&maps.u_rows[j], u, kNaMaxRows, static_cast<uint64_t>(d),
                                  static_cast<uint32_t>(kUBoxRows * (j + 1)));
    if (!maps_ok) return na_fail(RPD_ERR_CUDA, "cuTensorMapEncodeTiled failed");

    const int num_n = (V + kTileN - 1) / kTileN;
    int splits = 2 * num_n < 2 * dev->num_sms ? 2 * num_n : 2 * dev->num_sms;
    if (splits > kNaMaxSplits) splits = kNaMaxSplits;

    // The per-step count/status words must start from zero on every call.
    cudaError_t e = cudaMemsetAsync(meta, 0, kMetaWords * 4, stream);
    if (e == cudaSuccess) {
        // no plan table (it would have to be allocated): the compaction kernel evaluates the
        // head-tiling plan itself
        const HeadPlanInputs plan_in{num_n, splits, pair_slots,
                                     head_stream_in_tiles(V, d, dev->num_sms), RPD_TILING_AUTO};
        CompactParams cp{mask, q_of_pos, pos_of_q, canvas_off, meta, 1, N, K, plan_in, nullptr, 0,
                         rule.block, 0};
        e = launch_compact(cp, stream);
    }
    if (e == cudaSuccess) {
        NormParams np{static_cast<const __nv_bfloat16 *>(hidden),
                      static_cast<const __nv_bfloat16 *>(g_norm), pos_of_q, nullptr, meta, u,
                      inv_rms, N, d, eps};
        e = launch_gather_norm(np, std::min(dev->num_sms * 8, (K * N + 7) / 8), stream);
    }
    if (e == cudaSuccess) {
        HeadParams hp{inv_rms, partials, meta, V, d, splits, kWaitLimitNs, 0};
        e = launch_head(maps, hp, dev->head_grid, stream);
    }
    if (e == cudaSuccess) {
        // the merge's last CTA scores the canvas (N <= kNaMaxN <= kFuseScoreMaxN), as rpd_step does
        ScoreParams sp{};
        sp.mask = mask;
        sp.q_of_pos = q_of_pos;
        sp.canvas_off = canvas_off;
        sp.meta = meta;
        sp.row_arg = row_arg;
        sp.row_pmax = row_pmax;
        sp.row_H = row_H;
        sp.out_commit = out_commit;
        sp.out_token = out_token;
        sp.out_stats = out_stats;
        sp.B = 1;
        sp.N = N;
        sp.K = K;
        sp.theta_c = rule.theta_c;
        sp.theta_s = rule.theta_s;
        sp.w = rule.w;
        sp.k_max = rule.k_max;
        sp.window = rule.window;
        sp.block = rule.block;
        sp.tau[0] = tau;
        sp.budget[0] = budget;
        e = launch_merge_score(MergeArgs{partials, splits, row_arg, row_pmax, row_H}, meta, nullptr,
                               dev->num_sms * 4, sp, stream);
    }
    if (e != cudaSuccess) {
        set_last_error((std::string("rpd_step_noalloc launch failed: ") + cudaGetErrorString(e)).c_str());
        return RPD_ERR_CUDA;
    }
    return RPD_OK;
}
