"""rpd_step_noalloc: the entry point for callers that cannot allocate device memory.

Such callers (a serving engine that owns one pre-planned arena, a plugin inside another
framework's memory manager, a latency-critical loop where a device-synchronising cudaMalloc
is not acceptable) cannot let the library call cudaMalloc, so this entry point runs the step on a static
device array inside the library.  These tests call it through the C ABI and check that
its outputs equal those of rpd_step (the context-based entry point) on the same inputs,
for consecutive calls that leave different amounts of stale data in the shared array,
and that sizes beyond the array's limits are refused before any work is done.

The file is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

import workloads as WL

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, never run there
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2609_36452_gb300 as rpd  # noqa: E402

DEV = torch.device("cuda:0")


def make_case(seed, K, N, d, V, mask_frac):
    W, g = WL.make_head(V, d, seed, w_std=0.08)
    b = WL.u_profile(N, 0.5, 3.0)
    cv = WL.make_hidden(W, K, N, seed + 1000, b, WL.calibrated_sigma(V, d, 0.08, 3.0),
                        flip_frac=0.1)
    mask = torch.ones(N, dtype=torch.uint8) if mask_frac >= 1.0 else \
        WL.uniform_fraction_mask(N, mask_frac, seed + 5)
    return dict(W=W.to(DEV), g=g.to(DEV), hidden=cv.hidden.to(DEV), mask=mask.to(DEV),
                K=K, N=N, d=d, V=V)


def outputs(N):
    return (torch.full((N,), 7, dtype=torch.uint8, device=DEV),
            torch.full((N,), -5, dtype=torch.int32, device=DEV),
            torch.full((rpd.STATS_WORDS,), -9, dtype=torch.int32, device=DEV))


def run_context(case, tau, budget):
    ctx = rpd.Rpd(case["d"], case["V"], case["K"], 1e-6)
    ctx.set_head(case["W"], case["g"])
    ctx.set_stream(torch.cuda.current_stream(DEV))
    mask = case["mask"].clone()
    commit, token, stats = outputs(case["N"])
    ctx.step(case["hidden"], mask, tau, budget, commit, token, stats)
    torch.cuda.synchronize(DEV)
    ctx.close()
    return mask.cpu(), commit.cpu(), token.cpu(), stats.cpu()


def run_noalloc(case, tau, budget):
    mask = case["mask"].clone()
    commit, token, stats = outputs(case["N"])
    rule = rpd.RpdRule(*rpd.RULE_PROFILES["llada"])
    p = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
    rc = rpd.rpd_step_noalloc(p(case["W"]), p(case["g"]), case["d"], case["V"], case["K"],
                              ctypes.c_float(1e-6), ctypes.byref(rule), p(case["hidden"]), p(mask),
                              case["N"], ctypes.c_float(tau), ctypes.c_float(budget), p(commit),
                              p(token), p(stats),
                              ctypes.c_void_p(torch.cuda.current_stream(DEV).cuda_stream))
    assert rc == rpd.RPD_OK, rpd.rpd_last_error()
    torch.cuda.synchronize(DEV)
    return mask.cpu(), commit.cpu(), token.cpu(), stats.cpu()


def assert_same(a, b):
    mask_a, commit_a, token_a, stats_a = a
    mask_b, commit_b, token_b, stats_b = b
    assert torch.equal(commit_a, commit_b)
    assert torch.equal(mask_a, mask_b)
    sel = commit_a == 1
    assert torch.equal(token_a[sel], token_b[sel])
    assert torch.all(token_b[~sel] == -5)  # tokens are written only where committed
    assert torch.equal(stats_a, stats_b)
    assert int(stats_b[7]) == rpd.RPD_OK and int(stats_b[4]) >= 1


def test_noalloc_matches_context_step_on_consecutive_calls():
    big = make_case(81, K=4, N=256, d=1024, V=8192, mask_frac=1.0)     # 1024 rows: the limit
    small = make_case(82, K=3, N=100, d=256, V=4100, mask_frac=0.6)    # fewer rows, other d, ragged V
    for case, tau, budget in [(big, 0.9, 1.0), (small, 0.85, 2.0), (big, 0.9, 1.0)]:
        assert_same(run_context(case, tau, budget), run_noalloc(case, tau, budget))


def call_noalloc(case, W, g, hidden, K=None, d=None, N=None, stream=None):
    """One rpd_step_noalloc call with fresh, recognisable outputs; returns (rc, outputs)."""
    N = case["N"] if N is None else N
    mask = case["mask"].clone()
    commit, token, stats = outputs(case["N"])
    p = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
    rc = rpd.rpd_step_noalloc(p(W), p(g), case["d"] if d is None else d, case["V"],
                              case["K"] if K is None else K, ctypes.c_float(1e-6), None, p(hidden),
                              p(mask), N, ctypes.c_float(0.9), ctypes.c_float(1.0), p(commit),
                              p(token), p(stats), stream)
    torch.cuda.synchronize(DEV)
    return rc, (mask, commit, token, stats)


def assert_untouched(case, outs):
    mask, commit, token, stats = outs
    assert torch.all(commit == 7) and torch.all(token == -5) and torch.all(stats == -9)
    assert torch.equal(mask, case["mask"])


@pytest.mark.parametrize("K,N,d,limit", [
    (5, 256, 256, b"1024"),    # K*N = 1280 rows > 1024
    (1, 1025, 256, b"1024"),   # N = 1025 > 1024
    (1, 64, 4104, b"4096"),    # d = 4104 > 4096
])
def test_noalloc_refuses_sizes_beyond_the_static_array(K, N, d, limit):
    case = make_case(83, K=K, N=N, d=d, V=4096, mask_frac=1.0)
    rc, outs = call_noalloc(case, case["W"], case["g"], case["hidden"])
    assert rc == rpd.RPD_ERR_UNSUPPORTED
    assert limit in rpd.rpd_last_error()
    assert_untouched(case, outs)


def test_noalloc_refuses_memory_the_device_cannot_read():
    """A head in ordinary (pageable) host memory would be a TMA source the GPU cannot read:
    the call refuses it before any work is enqueued."""
    case = make_case(84, K=2, N=64, d=256, V=4096, mask_frac=1.0)
    W_host, g_host, h_host = case["W"].cpu(), case["g"].cpu(), case["hidden"].cpu()
    for W, g, h in [(W_host, case["g"], case["hidden"]), (case["W"], g_host, case["hidden"]),
                    (case["W"], case["g"], h_host)]:
        rc, outs = call_noalloc(case, W, g, h)
        assert rc == rpd.RPD_ERR_INVALID_ARGUMENT, rpd.rpd_last_error()
        assert_untouched(case, outs)


def test_noalloc_allocates_no_device_memory():
    """After calls that have loaded every kernel the step uses, further calls with other
    shapes leave the device's free memory unchanged (the scratch is the static array)."""
    warm = [make_case(85, K=4, N=256, d=512, V=4096, mask_frac=1.0),
            make_case(86, K=2, N=300, d=256, V=8192, mask_frac=0.7)]
    fresh = [make_case(87, K=3, N=200, d=1024, V=5000, mask_frac=0.9),
             make_case(88, K=1, N=400, d=768, V=4096, mask_frac=0.5)]
    bufs = []
    for case in warm + fresh:  # every output buffer exists before the measurement
        bufs.append((case, outputs(case["N"]), case["mask"].clone()))
    for case in warm:
        rc, _ = call_noalloc(case, case["W"], case["g"], case["hidden"])
        assert rc == rpd.RPD_OK, rpd.rpd_last_error()
    torch.cuda.synchronize(DEV)
    free0, _ = torch.cuda.mem_get_info(DEV)
    p = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
    for case, (commit, token, stats), mask in bufs[len(warm):]:
        rc = rpd.rpd_step_noalloc(p(case["W"]), p(case["g"]), case["d"], case["V"], case["K"],
                                  ctypes.c_float(1e-6), None, p(case["hidden"]), p(mask), case["N"],
                                  ctypes.c_float(0.9), ctypes.c_float(1.0), p(commit), p(token),
                                  p(stats), None)
        assert rc == rpd.RPD_OK, rpd.rpd_last_error()
    torch.cuda.synchronize(DEV)
    free1, _ = torch.cuda.mem_get_info(DEV)
    assert free1 == free0, (free0, free1)
    for case, (commit, token, stats), mask in bufs[len(warm):]:
        assert int(stats[7]) == rpd.RPD_OK and int(stats[4]) >= 1
