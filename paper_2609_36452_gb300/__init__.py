"""RPD commit step on GB300 (sm_103a): Python binding of the C ABI in ``include/rpd.h``.

The functions below carry the C names and only marshal arguments (ctypes); every step of
the computation runs in the library's CUDA kernels.  PyTorch is used by callers for
device memory and streams; the ``Rpd`` helper accepts torch tensors and passes their
device pointers.  There is no CPU fallback: if ``librpd.so`` is missing or fails to
load, importing the binding raises.
"""
from __future__ import annotations

import ctypes
import os

__all__ = [
    "RPD_OK", "RPD_ERR_INVALID_ARGUMENT", "RPD_ERR_NO_HEAD", "RPD_ERR_CUDA",
    "RPD_ERR_OUT_OF_MEMORY", "RPD_ERR_TIMEOUT", "RPD_ERR_UNSUPPORTED", "RPD_ERR_CHECK", "RpdRule", "RpdStats",
    "RpdDebug", "RpdError", "lib", "lib_path", "rpd_create", "rpd_set_head", "rpd_set_rule",
    "rpd_get_rule", "rpd_set_stream", "rpd_reserve", "rpd_set_debug", "rpd_set_projection", "rpd_set_head_tiling", "rpd_set_head_layout", "rpd_set_wait_limit", "rpd_inject_stall", "rpd_step",
    "rpd_step_batched", "rpd_step_host", "rpd_step_noalloc", "rpd_set_vocab_shard",
    "rpd_step_shard_partials", "rpd_step_shard_finish", "rpd_profile_enable", "rpd_kernel_times",
    "rpd_build_decode_loop", "rpd_build_decode_loop_batched", "rpd_decode_loop_launch", "rpd_decode_loop_destroy", "DecodeLoop",
    "rpd_destroy", "rpd_last_error", "rpd_version", "Rpd", "RULE_PROFILES", "KERNEL_NAMES",
]

RPD_OK = 0
RPD_ERR_INVALID_ARGUMENT = 1
RPD_ERR_NO_HEAD = 2
RPD_ERR_CUDA = 3
RPD_ERR_OUT_OF_MEMORY = 4
RPD_ERR_TIMEOUT = 5
RPD_ERR_UNSUPPORTED = 6
RPD_ERR_CHECK = 7
RPD_NUM_KERNELS = 4
KERNEL_NAMES = ("gather_norm", "head_stats", "merge", "score_commit")

# Table 4 (App. A.6) rule profiles: theta_c, theta_s, w, k_max, window, block (0 = full RPD;
# 32 = the paper's RPD-block variant).
RULE_PROFILES = {
    "llada": (0.6, 3.5, 15.0, 6, 32, 0),
    "dream": (0.6, 2.5, 20.0, 6, 32, 0),
    "llada_block": (0.6, 3.5, 15.0, 6, 32, 32),
    "dream_block": (0.6, 2.5, 20.0, 6, 32, 32),
}

# RPD_LIBRARY names another build of the library (the tests' checked build, librpd_checked.so)
lib_path = os.environ.get("RPD_LIBRARY") or os.path.join(os.path.dirname(os.path.abspath(__file__)),
                                                          "librpd.so")


class RpdRule(ctypes.Structure):
    _fields_ = [("theta_c", ctypes.c_float), ("theta_s", ctypes.c_float), ("w", ctypes.c_float),
                ("k_max", ctypes.c_int32), ("window", ctypes.c_int32), ("block", ctypes.c_int32)]


class RpdStats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "n_masked", "n_candidates", "n_high_conf", "n_stability", "n_committed",
        "fallback_used", "fallback_pos", "status", "n_rows")]


class RpdDebug(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in (
        "conf", "entropy", "persist", "drop", "stability", "candidate", "layer_argmax",
        "layer_pmax")]


STATS_FIELDS = [f[0] for f in RpdStats._fields_]
STATS_WORDS = len(STATS_FIELDS)  # int32 words of one rpd_stats
RPD_PROJECT_ALL = 0
RPD_PROJECT_LAZY = 1
RPD_PROJECT_AUTO = 2
PROJECTION_MODES = {"all": RPD_PROJECT_ALL, "lazy": RPD_PROJECT_LAZY, "auto": RPD_PROJECT_AUTO}
RPD_TILING_AUTO = 0
RPD_TILING_PAIR = 1
RPD_TILING_ROWS_N = 2
HEAD_TILINGS = {"auto": RPD_TILING_AUTO, "pair": RPD_TILING_PAIR, "rows_n": RPD_TILING_ROWS_N}
RPD_HEAD_TILED = 0
RPD_HEAD_BORROWED = 1
HEAD_LAYOUTS = {"tiled": RPD_HEAD_TILED, "borrowed": RPD_HEAD_BORROWED}


class RpdError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"rpd error {code}: {msg}")
        self.code = code


def _load():
    if not os.path.exists(lib_path):
        raise ImportError(
            f"{lib_path} is missing: build it with `python -c \"import __graft_entry__ as g; "
            f"g.build()\"` (nvcc, sm_103a)")
    L = ctypes.CDLL(lib_path)
    vp, i32, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    sig = {
        "rpd_create": (vp, [i32, i32, i32, f32]),
        "rpd_set_head": (i32, [vp, vp, vp]),
        "rpd_set_rule": (i32, [vp, ctypes.POINTER(RpdRule)]),
        "rpd_get_rule": (i32, [vp, ctypes.POINTER(RpdRule)]),
        "rpd_set_stream": (i32, [vp, vp]),
        "rpd_reserve": (i32, [vp, i32, i32]),
        "rpd_set_debug": (i32, [vp, ctypes.POINTER(RpdDebug)]),
        "rpd_set_projection": (i32, [vp, i32]),
        "rpd_set_head_tiling": (i32, [vp, i32]),
        "rpd_set_head_layout": (i32, [vp, i32]),
        "rpd_set_wait_limit": (i32, [vp, ctypes.c_int64]),
        "rpd_inject_stall": (i32, [vp]),
        "rpd_step": (i32, [vp, vp, vp, i32, f32, f32, vp, vp, vp]),
        "rpd_step_batched": (i32, [vp, vp, vp, i32, i32, vp, vp, vp, vp, vp]),
        "rpd_step_host": (i32, [vp, vp, vp, i32, f32, f32, vp, vp, vp]),
        "rpd_step_noalloc": (i32, [vp, vp, i32, i32, i32, f32, ctypes.POINTER(RpdRule), vp, vp,
                                   i32, f32, f32, vp, vp, vp, vp]),
        "rpd_set_vocab_shard": (i32, [vp, i32, i32]),
        "rpd_step_shard_partials": (i32, [vp, vp, vp, i32, vp]),
        "rpd_step_shard_finish": (i32, [vp, vp, i32, vp, i32, f32, f32, vp, vp, vp]),
        "rpd_build_decode_loop": (i32, [vp, vp, vp, vp, i32, f32, f32, vp, vp, vp, f32, i32, vp,
                                        ctypes.POINTER(vp)]),
        "rpd_build_decode_loop_batched": (i32, [vp, vp, vp, vp, i32, i32, vp, vp, vp, vp, vp, f32, i32,
                                                vp, ctypes.POINTER(vp)]),
        "rpd_decode_loop_launch": (i32, [vp, vp, vp]),
        "rpd_decode_loop_destroy": (None, [vp, vp]),
        "rpd_profile_enable": (i32, [vp, i32]),
        "rpd_kernel_times": (i32, [vp, ctypes.POINTER(ctypes.c_double),
                                   ctypes.POINTER(ctypes.c_int64), i32]),
        "rpd_destroy": (None, [vp]),
        "rpd_last_error": (ctypes.c_char_p, []),
        "rpd_version": (ctypes.c_char_p, []),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    return L


lib = _load()

rpd_create = lib.rpd_create
rpd_set_head = lib.rpd_set_head
rpd_set_rule = lib.rpd_set_rule
rpd_get_rule = lib.rpd_get_rule
rpd_set_stream = lib.rpd_set_stream
rpd_reserve = lib.rpd_reserve
rpd_set_debug = lib.rpd_set_debug
rpd_set_projection = lib.rpd_set_projection
rpd_set_head_tiling = lib.rpd_set_head_tiling
rpd_build_decode_loop = lib.rpd_build_decode_loop
rpd_build_decode_loop_batched = lib.rpd_build_decode_loop_batched
rpd_decode_loop_launch = lib.rpd_decode_loop_launch
rpd_decode_loop_destroy = lib.rpd_decode_loop_destroy
rpd_set_head_layout = lib.rpd_set_head_layout
rpd_set_wait_limit = lib.rpd_set_wait_limit
rpd_inject_stall = lib.rpd_inject_stall
rpd_step = lib.rpd_step
rpd_step_batched = lib.rpd_step_batched
rpd_step_host = lib.rpd_step_host
rpd_step_noalloc = lib.rpd_step_noalloc
rpd_set_vocab_shard = lib.rpd_set_vocab_shard
rpd_step_shard_partials = lib.rpd_step_shard_partials
rpd_step_shard_finish = lib.rpd_step_shard_finish
rpd_profile_enable = lib.rpd_profile_enable
rpd_kernel_times = lib.rpd_kernel_times
rpd_destroy = lib.rpd_destroy
rpd_last_error = lib.rpd_last_error
rpd_version = lib.rpd_version


def _check(code: int):
    if code != RPD_OK:
        raise RpdError(code, rpd_last_error().decode())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _arg(t, name: str, dtype: str, numel: int = None, cuda: bool = True):
    """Refuse, before any GPU work, a tensor the C ABI would misread: on the wrong side
    (host/device), of the wrong element type, not contiguous, or of the wrong size."""
    if t is None or not hasattr(t, "data_ptr"):
        raise RpdError(RPD_ERR_INVALID_ARGUMENT, f"{name}: a tensor is required")
    if bool(t.is_cuda) != cuda:
        raise RpdError(RPD_ERR_INVALID_ARGUMENT,
                       f"{name}: must be a {'CUDA' if cuda else 'host (CPU)'} tensor")
    if str(t.dtype) != "torch." + dtype:
        raise RpdError(RPD_ERR_INVALID_ARGUMENT, f"{name}: dtype must be {dtype}, not {t.dtype}")
    if not t.is_contiguous():
        raise RpdError(RPD_ERR_INVALID_ARGUMENT, f"{name}: must be contiguous")
    if numel is not None and t.numel() != numel:
        raise RpdError(RPD_ERR_INVALID_ARGUMENT, f"{name}: {t.numel()} elements, expected {numel}")
    return _ptr(t)


_DEBUG_DTYPES = {"conf": "float32", "entropy": "float32", "persist": "int32", "drop": "float32",
                 "stability": "float32", "candidate": "uint8", "layer_argmax": "int32",
                 "layer_pmax": "float32"}


class DecodeLoop:
    """An instantiated decoding-loop graph (rpd_build_decode_loop): ``launch(stream)`` runs the
    whole loop asynchronously on ``stream`` (a torch.cuda.Stream, or None for the current one)."""

    def __init__(self, ctx, handle):
        self.ctx, self.handle = ctx, handle

    def launch(self, stream=None):
        import torch
        s = stream if stream is not None else torch.cuda.current_stream()
        _check(rpd_decode_loop_launch(self.ctx.handle, self.handle, ctypes.c_void_p(s.cuda_stream)))

    def close(self):
        if getattr(self, "handle", None) and getattr(self.ctx, "handle", None):
            rpd_decode_loop_destroy(self.ctx.handle, self.handle)
        self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Rpd:
    """A context bound to torch tensors.  ``W`` ([V][d]) and ``g`` ([d]) are bf16 CUDA
    tensors; this object keeps references to both, so they outlive the context (the library
    borrows ``g``, and ``W`` too under the "borrowed" head layout)."""

    def __init__(self, d: int, V: int, K: int, eps: float = 1e-6):
        self.d, self.V, self.K, self.eps = d, V, K, eps
        h = rpd_create(d, V, K, ctypes.c_float(eps))
        if not h:
            raise RpdError(RPD_ERR_INVALID_ARGUMENT, rpd_last_error().decode())
        self.handle = ctypes.c_void_p(h)
        self._keep = []

    def close(self):
        if getattr(self, "handle", None):
            rpd_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_head(self, W, g):
        pw = _arg(W, "W", "bfloat16", self.V * self.d)
        pg = _arg(g, "g", "bfloat16", self.d)
        self._keep = [W, g]
        _check(rpd_set_head(self.handle, pw, pg))

    def set_rule(self, theta_c, theta_s, w, k_max, window, block=0):
        _check(rpd_set_rule(self.handle,
                            ctypes.byref(RpdRule(theta_c, theta_s, w, k_max, window, block))))

    def set_profile(self, name: str):
        self.set_rule(*RULE_PROFILES[name])

    def get_rule(self) -> dict:
        r = RpdRule()
        _check(rpd_get_rule(self.handle, ctypes.byref(r)))
        return dict(theta_c=r.theta_c, theta_s=r.theta_s, w=r.w, k_max=r.k_max, window=r.window,
                    block=r.block)

    def set_stream(self, stream):
        """``stream``: a torch.cuda.Stream, a raw cudaStream_t int, or None (legacy)."""
        raw = getattr(stream, "cuda_stream", stream)
        _check(rpd_set_stream(self.handle, ctypes.c_void_p(raw) if raw else None))

    def set_projection(self, mode):
        """Projection of the window layers (App. A.6): "all", "lazy" (two passes) or "auto"
        (chosen per step on the device); True/False mean "lazy"/"all"."""
        if isinstance(mode, bool):
            mode = "lazy" if mode else "all"
        _check(rpd_set_projection(self.handle, PROJECTION_MODES[mode]))

    def set_head_layout(self, layout):
        """How the head kernel reads W: "tiled" (default: set_head copies W into contiguous
        128 x 64 blocks owned by the context) or "borrowed" (W read in place, kept alive by
        this object).  Takes effect at the next set_head."""
        _check(rpd_set_head_layout(self.handle, HEAD_LAYOUTS[layout]))

    def set_head_tiling(self, tiling):
        """Tiling of the head contraction: "auto" (default, chosen per pass on the device),
        "pair" (256-row x 256-entry tiles on CTA pairs) or "rows_n" (256 entries x row groups
        of up to 512 rows, padded to 32); for tests and measurements."""
        _check(rpd_set_head_tiling(self.handle, HEAD_TILINGS[tiling]))

    def set_wait_limit(self, microseconds: int):
        _check(rpd_set_wait_limit(self.handle, int(microseconds)))

    def inject_stall(self):
        """Diagnostics: the next step's head kernel issues no loads; the step reports
        RPD_ERR_TIMEOUT once its bounded waits run out."""
        _check(rpd_inject_stall(self.handle))

    def reserve(self, B: int, N: int):
        _check(rpd_reserve(self.handle, B, N))

    def set_debug(self, **tensors):
        """Keyword tensors named like the rpd_debug fields (CUDA, contiguous); None clears."""
        if not tensors:
            _check(rpd_set_debug(self.handle, None))
            return
        for f in tensors:
            if f not in _DEBUG_DTYPES:
                raise RpdError(RPD_ERR_INVALID_ARGUMENT, f"unknown debug output {f}")
        dbg = RpdDebug(*[_arg(tensors[f], f, _DEBUG_DTYPES[f]) if tensors.get(f) is not None else None
                         for f, _ in RpdDebug._fields_])
        self._dbg_keep = tensors
        _check(rpd_set_debug(self.handle, ctypes.byref(dbg)))

    def step(self, hidden, mask, tau, budget, out_commit, out_token, out_stats):
        """One canvas: hidden [K][N][d] bf16, mask [N] uint8 (in/out), out_commit [N] uint8,
        out_token [N] int32, out_stats int32 tensor of STATS_WORDS (an rpd_stats), all CUDA."""
        N = mask.numel()
        args = (_arg(hidden, "hidden", "bfloat16", self.K * N * self.d), _arg(mask, "mask", "uint8"),
                _arg(out_commit, "out_commit", "uint8", N), _arg(out_token, "out_token", "int32", N),
                _arg(out_stats, "out_stats", "int32", STATS_WORDS))
        _check(rpd_step(self.handle, args[0], args[1], N, ctypes.c_float(tau),
                        ctypes.c_float(budget), *args[2:]))

    def build_decode_loop(self, hidden, mask, tau, budget, out_commit, out_token, out_stats,
                          steps, stop_frac=0.02, max_steps=64, forward=None):
        """A CUDA graph that repeats [forward; step; stop test] on the device until at most
        floor(stop_frac * N) positions remain masked (or max_steps steps, or an error status).
        ``forward``: None, a torch.cuda.CUDAGraph built with keep_graph=True (the backbone's
        forward pass writing ``hidden`` from the canvas), or a raw cudaGraph_t handle.
        ``steps``: a CUDA int32 tensor of one element (steps run).  Returns a DecodeLoop."""
        N = mask.numel()
        fwd = None
        if forward is not None:
            fwd = forward.raw_cuda_graph() if hasattr(forward, "raw_cuda_graph") else int(forward)
        exe = ctypes.c_void_p()
        _check(rpd_build_decode_loop(
            self.handle, fwd, _arg(hidden, "hidden", "bfloat16", self.K * N * self.d),
            _arg(mask, "mask", "uint8", N), N, ctypes.c_float(tau), ctypes.c_float(budget),
            _arg(out_commit, "out_commit", "uint8", N), _arg(out_token, "out_token", "int32", N),
            _arg(out_stats, "out_stats", "int32", STATS_WORDS), ctypes.c_float(stop_frac),
            int(max_steps), _arg(steps, "steps", "int32", 1), ctypes.byref(exe)))
        loop = DecodeLoop(self, exe.value)
        loop._keep = [hidden, mask, out_commit, out_token, out_stats, steps, forward]
        return loop

    def build_decode_loop_batched(self, hidden, mask, tau, budget, out_commit, out_token,
                                  out_stats, steps, stop_frac=0.02, max_steps=64, forward=None):
        """build_decode_loop over B canvases: hidden [K][B][N][d], mask / out_commit / out_token
        [B][N], out_stats [B][STATS_WORDS]; tau and budget are length-B host sequences."""
        B, N = mask.shape
        fwd = None
        if forward is not None:
            fwd = forward.raw_cuda_graph() if hasattr(forward, "raw_cuda_graph") else int(forward)
        taus = (ctypes.c_float * B)(*[float(x) for x in tau])
        budgets = (ctypes.c_float * B)(*[float(x) for x in budget])
        exe = ctypes.c_void_p()
        _check(rpd_build_decode_loop_batched(
            self.handle, fwd, _arg(hidden, "hidden", "bfloat16", self.K * B * N * self.d),
            _arg(mask, "mask", "uint8", B * N), B, N, taus, budgets,
            _arg(out_commit, "out_commit", "uint8", B * N), _arg(out_token, "out_token", "int32", B * N),
            _arg(out_stats, "out_stats", "int32", B * STATS_WORDS), ctypes.c_float(stop_frac),
            int(max_steps), _arg(steps, "steps", "int32", 1), ctypes.byref(exe)))
        loop = DecodeLoop(self, exe.value)
        loop._keep = [hidden, mask, out_commit, out_token, out_stats, steps, forward]
        return loop

    def step_batched(self, hidden, mask, tau, budget, out_commit, out_token, out_stats):
        """B canvases: hidden [K][B][N][d], mask/out_commit/out_token [B][N], out_stats
        [B][STATS_WORDS];
        tau and budget are length-B host sequences."""
        B, N = mask.shape
        if len(tau) != B or len(budget) != B:
            raise RpdError(RPD_ERR_INVALID_ARGUMENT, "tau and budget need one value per canvas")
        args = (_arg(hidden, "hidden", "bfloat16", self.K * B * N * self.d),
                _arg(mask, "mask", "uint8"), _arg(out_commit, "out_commit", "uint8", B * N),
                _arg(out_token, "out_token", "int32", B * N),
                _arg(out_stats, "out_stats", "int32", B * STATS_WORDS))
        ta = (ctypes.c_float * B)(*[float(x) for x in tau])
        bu = (ctypes.c_float * B)(*[float(x) for x in budget])
        _check(rpd_step_batched(self.handle, args[0], args[1], B, N,
                                ctypes.cast(ta, ctypes.c_void_p), ctypes.cast(bu, ctypes.c_void_p),
                                *args[2:]))

    def step_host(self, hidden, mask, tau, budget, out_commit, out_token, out_stats):
        """Host (CPU, ideally pinned) tensors; returns after the results are back."""
        N = mask.numel()
        args = (_arg(hidden, "hidden", "bfloat16", self.K * N * self.d, cuda=False),
                _arg(mask, "mask", "uint8", cuda=False),
                _arg(out_commit, "out_commit", "uint8", N, cuda=False),
                _arg(out_token, "out_token", "int32", N, cuda=False),
                _arg(out_stats, "out_stats", "int32", STATS_WORDS, cuda=False))
        _check(rpd_step_host(self.handle, args[0], args[1], N, ctypes.c_float(tau),
                             ctypes.c_float(budget), *args[2:]))

    def set_vocab_shard(self, v_offset: int, V_total: int):
        """This context's head rows are vocabulary entries [v_offset, v_offset + V) of V_total."""
        _check(rpd_set_vocab_shard(self.handle, int(v_offset), int(V_total)))

    def step_shard_partials(self, hidden, mask, out_partials):
        """Vocabulary-sharded step, part 1: hidden [K][N][d] bf16, mask [N] uint8 (read only),
        out_partials [K][N][4] float32 (the slice's softmax statistics per projected row)."""
        N = mask.numel()
        args = (_arg(hidden, "hidden", "bfloat16", self.K * N * self.d), _arg(mask, "mask", "uint8"),
                _arg(out_partials, "out_partials", "float32", self.K * N * 4))
        _check(rpd_step_shard_partials(self.handle, args[0], args[1], N, args[2]))

    def step_shard_finish(self, gathered, mask, tau, budget, out_commit, out_token, out_stats):
        """Part 3: gathered [P][K][N][4] float32 (every slice's statistics, slices in vocabulary
        order), then mask/out_* as in step()."""
        N = mask.numel()
        P = gathered.shape[0]
        args = (_arg(gathered, "gathered", "float32", P * self.K * N * 4), _arg(mask, "mask", "uint8"),
                _arg(out_commit, "out_commit", "uint8", N), _arg(out_token, "out_token", "int32", N),
                _arg(out_stats, "out_stats", "int32", STATS_WORDS))
        _check(rpd_step_shard_finish(self.handle, args[0], P, args[1], N, ctypes.c_float(tau),
                                     ctypes.c_float(budget), *args[2:]))

    def profile(self, enable: bool):
        _check(rpd_profile_enable(self.handle, 1 if enable else 0))

    def kernel_times(self, reset: bool = True):
        ms = (ctypes.c_double * RPD_NUM_KERNELS)()
        n = (ctypes.c_int64 * RPD_NUM_KERNELS)()
        _check(rpd_kernel_times(self.handle, ms, n, 1 if reset else 0))
        return {KERNEL_NAMES[i]: (ms[i], n[i]) for i in range(RPD_NUM_KERNELS)}


def stats_dict(t) -> dict:
    """Decode one rpd_stats (an int32 tensor/array of STATS_WORDS) into a dict."""
    vals = [int(x) for x in (t.tolist() if hasattr(t, "tolist") else t)]
    return dict(zip(STATS_FIELDS, vals))
