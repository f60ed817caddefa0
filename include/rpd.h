/*
 * rpd.h - C ABI of the Reliable Parallel Decoding (RPD) commit step on one GPU.
 *
 * One call of rpd_step() performs one decoding iteration's commitment decision for a
 * masked diffusion LM (paper §3): for every masked canvas position it projects the
 * hidden states of the last K layers through the final RMSNorm and the LM head (the
 * logit-lens readout of §2.2 and App. A.2, restricted to masked positions as App. A.6
 * states), reads each layer's argmax and its probability and the final layer's
 * confidence and entropy (Eq. 1), scores layerwise stability (Eq. 2-4), forms the
 * candidate set (Eq. 5), and commits the candidates whose preceding masked positions
 * hold at most `budget` nats of entropy (§3.2, E_i and A_t), falling back to the most
 * confident of the first W masked positions when none qualifies (§3.2).
 *
 * Conventions for every entry point:
 *  - Pointers named "device" are CUDA device pointers on the context's device; pointers
 *    named "host" are host memory (pinned memory makes the copies asynchronous).
 *  - bf16 arrays hold IEEE bfloat16 bit patterns (2 bytes per element).
 *  - All device work is enqueued on the context's stream (rpd_set_stream) and is
 *    asynchronous unless stated otherwise; nothing is read back to the host mid-step.
 *  - Every int-returning function returns RPD_OK (0) or one of the RPD_ERR_* codes and
 *    records a message for rpd_last_error() (per host thread).  On an error return no
 *    output has been written unless the code is RPD_ERR_CUDA.
 *  - A context is not thread safe; use one context per host thread or serialise calls.  A
 *    context may be used from any host thread: each call that touches the GPU makes the
 *    context's device (and its primary context) current for its duration and gives the
 *    thread its previous device back.
 *  - Inputs must be finite; with eps = 0 an all-zero hidden row has no defined RMS factor.
 *    Sums of squares, logits and softmax statistics are fp32 (h^2 must not overflow fp32).
 */
#ifndef RPD_H_
#define RPD_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RPD_OK 0
#define RPD_ERR_INVALID_ARGUMENT 1 /* bad size, pointer, threshold or alignment */
#define RPD_ERR_NO_HEAD 2          /* rpd_step before rpd_set_head */
#define RPD_ERR_CUDA 3             /* a CUDA runtime/driver call failed */
#define RPD_ERR_OUT_OF_MEMORY 4    /* scratch allocation failed */
#define RPD_ERR_TIMEOUT 5          /* a kernel's bounded wait ran out (latched in rpd_stats.status) */
#define RPD_ERR_UNSUPPORTED 6      /* shape outside what the kernels handle */
#define RPD_ERR_CHECK 7            /* a device-side bounds check failed (only in a library built
                                      with RPD_CHECKS; latched in rpd_stats.status) */

typedef struct rpd_ctx rpd_ctx; /* opaque, owned by the library */

/* Rule parameters other than theta_h (= tau) and beta (= budget); Table 4 (App. A.6).
 * rpd_create installs the LLaDA profile: theta_c 0.6, theta_s 3.5, w 15, k_max 6, window 32,
 * block 0.
 * The Dream profile is theta_s 2.5, w 20 with the rest unchanged. */
typedef struct rpd_rule {
    float theta_c;  /* minimum confidence for admission through stability (Eq. 5) */
    float theta_s;  /* stability threshold (Eq. 5) */
    float w;        /* weight of the confidence-drop penalty (Eq. 4), >= 0 */
    int32_t k_max;  /* cap on prediction persistence (Eq. 4), >= 1 */
    int32_t window; /* fallback window W: first W masked positions (§3.2), >= 1 */
    int32_t block;  /* 0: full RPD (§3.2).  > 0: RPD-block (the variant of §3.2, App. A.6):
                       only the active block - the first run of `block` positions (32 in
                       the paper) that still holds a masked position - is projected and
                       scored; every candidate in it is committed (no entropy budget;
                       `budget` is ignored) and, if there is none, its most confident
                       masked position.  Debug outputs outside the active block read as
                       unmasked; rpd_stats.n_masked still counts the whole canvas. */
} rpd_rule;

/* Per-canvas step summary, written to DEVICE memory by rpd_step / rpd_step_batched. */
typedef struct rpd_stats {
    int32_t n_masked;     /* |M_t| before the step */
    int32_t n_candidates; /* |C_t| (Eq. 5) */
    int32_t n_high_conf;  /* commits admitted through c >= theta_h */
    int32_t n_stability;  /* commits admitted through theta_c <= c < theta_h and S >= theta_s */
    int32_t n_committed;  /* positions committed this step, fallback included */
    int32_t fallback_used;/* 1 if A_t was empty and the fallback commit was made */
    int32_t fallback_pos; /* canvas index of the fallback commit, -1 if none */
    int32_t status;       /* RPD_OK, or RPD_ERR_TIMEOUT if a kernel's bounded wait ran out */
    int32_t n_rows;       /* hidden-state rows projected through the head by this call (all
                             canvases): K x scored positions, or with lazy projection the
                             final layer of every scored position plus the earlier window
                             layers of the band positions */
} rpd_stats;

/* Optional per-position outputs (DEVICE pointers; any may be NULL).  Layouts use the
 * step's B and N: "[B][N]" arrays are indexed b*N+i, "[K][B][N]" arrays (k*B+b)*N+i with
 * k = 0 the earliest window layer and k = K-1 the final layer.  Unmasked positions get
 * conf/entropy/drop/stability 0, persist 0, candidate 0, layer_argmax -1, layer_pmax 0. */
typedef struct rpd_debug {
    float *conf;          /* [B][N] c_i = p^(L)(y_i) */
    float *entropy;       /* [B][N] H(p^(L)_i), nats */
    int32_t *persist;     /* [B][N] K_i (Eq. 2) */
    float *drop;          /* [B][N] r_i (Eq. 3) */
    float *stability;     /* [B][N] S_i (Eq. 4) */
    uint8_t *candidate;   /* [B][N] 1 if i in C_t */
    int32_t *layer_argmax;/* [K][B][N] argmax token of each window layer */
    float *layer_pmax;    /* [K][B][N] probability of that argmax */
} rpd_debug;

/* Create a context for hidden size d, vocabulary V, window K (the last K layers; the
 * paper's l0 = L-K+1) and RMSNorm epsilon eps, on the current CUDA device.
 * Requires d % 8 == 0 and d >= 64, V >= 256, 1 <= K <= 64, eps >= 0.
 * Returns NULL on failure (see rpd_last_error()). */
rpd_ctx *rpd_create(int d, int V, int K, float eps);

/* Set the LM head W_head ([V][d] bf16, row v = token v's output embedding, device, 16-byte
 * aligned) and the final-norm gain g_norm ([d] bf16, device, 16-byte aligned).  g_norm is
 * borrowed: it must stay valid until the context is destroyed or the head is replaced.
 * W_head is copied into the context's tiled layout and not read after the call returns, or
 * borrowed in the same way as g_norm (see rpd_set_head_layout).  The copy runs on the
 * context's stream and the call waits for it.  Host memory, or memory of another device, is
 * refused with RPD_ERR_INVALID_ARGUMENT.  App. A.2: the model's own final normalisation and
 * head. */
int rpd_set_head(rpd_ctx *ctx, const void *W_head, const void *g_norm);

/* Layout in which the head kernel reads W (no counterpart in the paper; the results are
 * bitwise the same in both).
 *   RPD_HEAD_TILED (default): rpd_set_head copies W into context-owned device memory as
 *     contiguous blocks of 128 rows x 64 columns (16 KB; block (t, k) holds rows
 *     [128t, 128t + 128) and columns [64k, 64k + 64), blocks ordered by t, then k, rows past V
 *     zero), so that every block the head kernel stages is one contiguous read.  It costs
 *     ceil(V/128)*128*d*2 bytes of device memory (1.04 GB at the LLaDA-8B head) and one copy
 *     per rpd_set_head.  Needs d % 64 == 0; with other d the context borrows W_head.
 *   RPD_HEAD_BORROWED: the head kernel reads W_head in place; W_head must stay valid like
 *     g_norm, and nothing is copied.
 * Takes effect at the next rpd_set_head.  Other values: RPD_ERR_INVALID_ARGUMENT. */
#define RPD_HEAD_TILED 0
#define RPD_HEAD_BORROWED 1
int rpd_set_head_layout(rpd_ctx *ctx, int layout);

/* Replace the rule parameters (Table 4).  Requires 0 <= theta_c, w >= 0, k_max >= 1,
 * window >= 1, block >= 0.  theta_c < tau is checked per step (Eq. 5 requires theta_c < theta_h). */
int rpd_set_rule(rpd_ctx *ctx, const rpd_rule *rule);
int rpd_get_rule(const rpd_ctx *ctx, rpd_rule *rule);

/* Run every later step on `stream` (a cudaStream_t; NULL = legacy default stream). */
int rpd_set_stream(rpd_ctx *ctx, void *stream);

/* Pre-size scratch for B canvases of N positions, so that later steps of that size
 * allocate nothing.  Steps grow scratch on demand otherwise (synchronising the device).
 * Requires B >= 1 and N >= 1; B > 128 or N > 8192: RPD_ERR_UNSUPPORTED. */
int rpd_reserve(rpd_ctx *ctx, int B, int N);

/* How the window layers are projected (App. A.6, the layerwise projection).
 *   RPD_PROJECT_ALL (default): every window layer of every scored position, in one pass over
 *     the head.
 *   RPD_PROJECT_LAZY: a first pass projects the final layer of every scored position; a second
 *     pass projects the earlier window layers only of the positions whose final confidence lies
 *     in the stability band theta_c <= c < tau - the only positions whose candidacy depends on
 *     K_i and r_i (Eq. 5).  Commits, tokens, confidences and entropies are the same as with
 *     RPD_PROJECT_ALL; the head is streamed twice when the band is not empty.  Debug outputs
 *     of positions outside the band report persist 0, drop 0, stability 0 and, for layers
 *     below the final one, layer_argmax -1 and layer_pmax 0. */
#define RPD_PROJECT_ALL 0
#define RPD_PROJECT_LAZY 1
/*   RPD_PROJECT_AUTO: per step, on the device, lazy when its two passes are estimated cheaper
 *     than one pass over every layer (many scored positions: the contraction is bound by the
 *     tensor cores), otherwise every layer (few positions: bound by streaming the head). */
#define RPD_PROJECT_AUTO 2
int rpd_set_projection(rpd_ctx *ctx, int mode);

/* Tiling of the head contraction (no counterpart in the paper; it changes neither the
 * computed quantities nor, beyond fp32 summation order, their values).  Both tilings run on
 * pairs of CTAs (tcgen05 cta_group::2).  By default (RPD_TILING_AUTO) the step picks, on the
 * device and per projection pass, the cheaper of:
 *   RPD_TILING_PAIR    tiles of 256 rows x 256 vocabulary entries (rows padded to 256);
 *   RPD_TILING_ROWS_N  tiles of 256 vocabulary entries x a group of up to 512 rows, the rows
 *                      on the MMA's N side (each group padded to a multiple of 32 rows).
 * Forcing one is for tests and measurements. */
#define RPD_TILING_AUTO 0
#define RPD_TILING_PAIR 1
#define RPD_TILING_ROWS_N 2
int rpd_set_head_tiling(rpd_ctx *ctx, int tiling);

/* Decoding loop with device-side stopping.  The paper's decoder alternates the model's forward
 * pass with the commit step until the canvas is complete (§3; App. A.6).  This builds a CUDA
 * graph whose one launch repeats on the device, without returning to the host:
 *   1. `forward`, a cudaGraph_t the caller built (for instance by stream capture): the
 *      backbone's forward pass, which writes the next step's hidden states into `hidden` from
 *      the canvas as it stands (NULL: the hidden states are not refreshed, for tests and
 *      measurements);
 *   2. one rpd_step(hidden, mask, N, tau, budget, out_commit, out_token, out_stats) on the
 *      context, with its rule, projection and head tiling as they are at build time;
 *   3. a stop test: the loop ends once at most floor(stop_frac * N) positions remain masked,
 *      after max_steps steps, or when the step's status is not RPD_OK;
 * and runs steps 1-3 at least once per launch.  steps (device int32) receives the number of
 * steps run, out_stats the last step's statistics, out_commit and out_token the last step's
 * commits (mask holds the canvas's remaining masked positions).  The graph is instantiated
 * into *out_exec (a cudaGraphExec_t owned by the context): launch it with
 * rpd_decode_loop_launch on any stream and free it with rpd_decode_loop_destroy; `forward` is
 * copied into it and stays the caller's.  Scratch is reserved for one canvas of N positions while
 * building.  hidden and mask are device memory (hidden 16-byte aligned).
 * Requires 1 <= N <= 8192, 0 <= stop_frac <= 1, max_steps >= 1; a context holding a vocabulary
 * slice is refused with RPD_ERR_UNSUPPORTED.  Errors from building the graph: RPD_ERR_CUDA. */
int rpd_build_decode_loop(rpd_ctx *ctx, void *forward, const void *hidden, uint8_t *mask, int N,
                          float tau, float budget, uint8_t *out_commit, int32_t *out_token,
                          rpd_stats *out_stats, float stop_frac, int max_steps, int32_t *steps,
                          void **out_exec);
/* The decoding loop over B canvases of N positions (the rpd_step_batched layout: hidden
 * [K][B][N][d], mask / out_commit / out_token [B][N], out_stats [B]; tau[B] and budget[B] are
 * host arrays read at build time).  The loop runs while some canvas has more than
 * floor(stop_frac * N) positions masked, fewer than max_steps steps have run and every
 * canvas's step succeeded.  Requires 1 <= B <= 128; otherwise as rpd_build_decode_loop. */
int rpd_build_decode_loop_batched(rpd_ctx *ctx, void *forward, const void *hidden, uint8_t *mask,
                                  int B, int N, const float *tau, const float *budget,
                                  uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats,
                                  float stop_frac, int max_steps, int32_t *steps, void **out_exec);

/* Launch a decoding loop built by rpd_build_decode_loop(_batched) on this context on `stream` (a
 * cudaStream_t, NULL = legacy default stream), asynchronously.  The loop records the context's
 * scratch and head: once either has been reallocated or replaced (a step on a larger canvas,
 * rpd_reserve growing scratch, rpd_set_head), the launch is refused with
 * RPD_ERR_INVALID_ARGUMENT and the loop must be rebuilt.  rpd_decode_loop_destroy frees a loop
 * once no launch of it is in flight (NULL or unknown handles are ignored); rpd_destroy frees the
 * context's remaining loops.  The debug buffers set before building (rpd_set_debug) must stay
 * valid while the loop is used. */
int rpd_decode_loop_launch(rpd_ctx *ctx, void *exec, void *stream);
void rpd_decode_loop_destroy(rpd_ctx *ctx, void *exec);

/* Diagnostics.  Every wait inside the step's kernels (mbarrier waits of the head kernels) is
 * bounded; when one runs out the kernel stops, drains what it has in flight, frees its
 * tensor memory and latches RPD_ERR_TIMEOUT in rpd_stats.status (the other outputs of that
 * step are then meaningless); the context stays usable.
 *   rpd_set_wait_limit: the bound, in microseconds (default 2 000 000), >= 1000.
 *   rpd_inject_stall:  the next step's head kernels issue no loads at all, so their waits run
 *                      out and the step reports RPD_ERR_TIMEOUT; used to test the path. */
int rpd_set_wait_limit(rpd_ctx *ctx, int64_t microseconds);
int rpd_inject_stall(rpd_ctx *ctx);

/* Install (or with NULL, clear) the optional per-position outputs. */
int rpd_set_debug(rpd_ctx *ctx, const rpd_debug *debug);

/* One commit step for one canvas (§3).
 *   hidden     [K][N][d] bf16, device (or mapped page-locked host memory; anything else is
 *              refused with RPD_ERR_INVALID_ARGUMENT): pre-norm hidden state of each window
 *              layer at each canvas position (the final layer last).  Rows of unmasked
 *              positions are never read.
 *   mask       [N] uint8, device, in/out: 1 = masked.  Committed positions are set to 0.
 *   N          canvas length, 0 <= N <= 8192 (N = 0 is a no-op; N > 8192:
 *              RPD_ERR_UNSUPPORTED).
 *   tau        theta_h, 0 < tau <= 1 and tau > theta_c.
 *   budget     beta in nats, >= 0 (may be +inf).
 *   out_commit [N] uint8, device: 1 where committed this step, 0 elsewhere.
 *   out_token  [N] int32, device: y_i written ONLY at committed positions, so it may be
 *              the canvas itself.
 *   out_stats  one rpd_stats, device.
 * With N_m > 0 masked positions at least one position is committed. */
int rpd_step(rpd_ctx *ctx, const void *hidden, uint8_t *mask, int N, float tau, float budget,
             uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats);

/* B independent canvases of N positions in one step; the head is read once for all.
 *   hidden [K][B][N][d] bf16 device; mask, out_commit, out_token [B][N] device;
 *   tau, budget [B] HOST arrays (per-canvas theta_h and beta); out_stats [B] device.
 * Requires 1 <= B <= 128 (B > 128 or N > 8192: RPD_ERR_UNSUPPORTED).  Canvases of
 * different lengths are padded to a common N with mask 0: unmasked positions are never
 * projected, scored, counted in E_i or committed, so each canvas's result is that of its
 * unpadded length. */
int rpd_step_batched(rpd_ctx *ctx, const void *hidden, uint8_t *mask, int B, int N,
                     const float *tau, const float *budget, uint8_t *out_commit,
                     int32_t *out_token, rpd_stats *out_stats);

/* rpd_step with HOST buffers: copies hidden, mask and out_token in, runs the step, copies
 * mask, out_commit, out_token and out_stats back, and returns after the stream has finished.
 * mask and out_token are in/out: out_token (the canvas) changes only at committed positions.
 * hidden in pinned (page-locked) host memory is read in place by the step's gather kernel,
 * so only the masked positions' rows cross the host link; hidden in other host memory is
 * copied to the device first.  mask, out_token and the results travel through a pinned
 * staging buffer, one copy each way.
 * Staging buffers are owned by the context (grown on demand; the first call of a larger size
 * allocates). */
int rpd_step_host(rpd_ctx *ctx, const void *hidden, uint8_t *mask, int N, float tau,
                  float budget, uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats);

/* Vocabulary-parallel step over P devices (no counterpart in the paper: the same step as
 * rpd_step, with the LM head's rows divided among devices).  Each device holds a contiguous
 * slice of the head - rows [v_offset, v_offset + V) of a V_total-entry vocabulary, with V the
 * context's vocabulary size - and runs, on the same hidden states and mask:
 *   1. rpd_step_shard_partials: compaction, RMSNorm prologue and the head contraction over its
 *      slice; writes, for every window layer k and masked position i, the softmax statistics
 *      of the slice in base-2 units - (max, sum of 2^(x - max), sum of 2^(x - max)(x - max),
 *      argmax as a global token index), x = logit * log2(e) - to out_partials[k][i] (float4,
 *      [K][N][4] floats, device, 16-byte aligned; 16 bytes per projected row).  Entries of
 *      positions that are not projected are left as they were.
 *   2. the caller gathers every device's out_partials, in increasing v_offset order, into
 *      [P][K][N][4] (one all-gather, e.g. NCCL), and
 *   3. rpd_step_shard_finish: merges the P records of every projected row (in order; ties of
 *      the argmax go to the lower token index, as in rpd_step), then scores, scans and commits
 *      the canvas exactly as rpd_step does.  mask/out_* and tau/budget as in rpd_step; the mask
 *      must be the one given to rpd_step_shard_partials, on the same context, with no other
 *      step of the context in between.  out_stats->status reports this device's head waits.
 * Every device then holds the same commits.  The projection must be RPD_PROJECT_ALL (lazy
 * projection would need an exchange between its passes: RPD_ERR_UNSUPPORTED); RPD-block rules
 * work unchanged.  rpd_set_vocab_shard: 0 <= v_offset and v_offset + V <= V_total. */
int rpd_set_vocab_shard(rpd_ctx *ctx, int v_offset, int V_total);
int rpd_step_shard_partials(rpd_ctx *ctx, const void *hidden, const uint8_t *mask, int N,
                            float *out_partials);
int rpd_step_shard_finish(rpd_ctx *ctx, const float *gathered, int P, uint8_t *mask, int N,
                          float tau, float budget, uint8_t *out_commit, int32_t *out_token,
                          rpd_stats *out_stats);

/* Per-kernel timing with CUDA events recorded on the context's stream around every
 * launch while enabled.  rpd_kernel_times synchronises the recorded events and returns,
 * for each of the RPD_NUM_KERNELS kernels (gather/norm, head statistics, merge,
 * score/commit; the compaction kernel is counted with gather/norm, and for a single canvas
 * of at most 2048 positions score/commit runs inside the step's last merge and is counted
 * with it), the summed milliseconds and the launch count since the last reset; reset
 * clears them. */
#define RPD_NUM_KERNELS 4
int rpd_profile_enable(rpd_ctx *ctx, int enable);
int rpd_kernel_times(rpd_ctx *ctx, double *ms /*[RPD_NUM_KERNELS]*/,
                     int64_t *launches /*[RPD_NUM_KERNELS]*/, int reset);

/* rpd_step for callers that cannot allocate device memory.  (The paper has no counterpart:
 * this is a deployment variant of rpd_step.)  Some callers own every byte of device memory
 * themselves - a serving engine that plans one fixed arena, a plugin running inside another
 * framework's memory manager, a latency-critical loop in which a cudaMalloc (which can
 * synchronise the device) is not acceptable - so a library that calls cudaMalloc on their
 * behalf is not an option.  This entry point takes
 * no context and allocates nothing: it runs the same kernels as rpd_step with its scratch in
 * a static device array of this library (about 13 MiB, held on every GPU that loads the
 * library until the process exits).  The caller passes every input and output.
 *   W_head [V][d], g_norm [d], hidden [K][N][d]: bf16 device, 16-byte aligned;
 *   rule: NULL for theta_c 0.6, theta_s 3.5, w 15, k_max 6, window 32, block 0 (the values
 *   rpd_create installs); mask/out_commit/out_token/out_stats and tau/budget as in rpd_step,
 *   with the same checks of the rule and thresholds; stream: a cudaStream_t (NULL = legacy
 *   default stream).  W_head, g_norm and hidden that the current device cannot read (pageable
 *   host memory, another device's memory) are refused with RPD_ERR_INVALID_ARGUMENT; hidden
 *   may be mapped page-locked host memory.
 * Limits: K*N <= 1024, N <= 1024, d <= 4096 (plus rpd_create's shape rules); larger sizes
 * return RPD_ERR_UNSUPPORTED with a message naming the limit, before any work is enqueued.
 * All calls on a device share the one scratch array, which keeps the previous call's
 * contents (the step's count/status words are cleared at the start of every call): calls
 * whose GPU work overlaps - concurrent host threads or different streams - race on it, so
 * order them on one stream.  The first call on each device finds the array's device address
 * (cudaGetSymbolAddress) and caches it; make that first call before any stream capture. */
int rpd_step_noalloc(const void *W_head, const void *g_norm, int d, int V, int K, float eps,
                     const rpd_rule *rule, const void *hidden, uint8_t *mask, int N, float tau,
                     float budget, uint8_t *out_commit, int32_t *out_token, rpd_stats *out_stats,
                     void *stream);

/* Free the context, its scratch and its copy of the head (not the caller's buffers).  NULL
 * is ignored. */
void rpd_destroy(rpd_ctx *ctx);

/* Message of the last failing call on this host thread ("" if none). */
const char *rpd_last_error(void);

/* Library version string. */
const char *rpd_version(void);

#ifdef __cplusplus
}
#endif

#endif /* RPD_H_ */
