"""The decoding loop with device-side stopping (rpd_build_decode_loop): one graph launch runs
[forward; step; stop test] until at most floor(stop_frac * N) positions remain masked.  The
loop must reach exactly the state a host loop of rpd_step reaches with the same forward pass:
the same number of steps, the same remaining mask and the same last step's commits, tokens
and statistics."""
import ctypes

import numpy as np
import pytest
import torch

from tests.test_gpu_parity import small_case

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, never run there
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2609_36452_gb300 as rpd  # noqa: E402

DEV = torch.device("cuda:0")


def context(case, projection="all", profile=None):
    c = rpd.Rpd(case["d"], case["V"], case["K"], case["eps"])
    c.set_stream(torch.cuda.current_stream(DEV))
    c.set_head(case["W"].to(DEV), case["g"].to(DEV))
    c.set_profile(profile or case["rule"])
    c.set_projection(projection)
    c.reserve(1, case["N"])
    return c


def outputs(N):
    return dict(commit=torch.zeros(N, dtype=torch.uint8, device=DEV),
                token=torch.full((N,), -1, dtype=torch.int32, device=DEV),
                stats=torch.zeros(rpd.STATS_WORDS, dtype=torch.int32, device=DEV))


def host_loop(ctx, case, hidden, mask, forward, stop_frac, max_steps):
    """The reference: rpd_step from the host, one forward pass before each step."""
    N = case["N"]
    out = outputs(N)
    limit = int(np.floor(stop_frac * N))
    steps = 0
    while True:
        forward()
        ctx.step(hidden, mask, case["tau"], case["budget"], out["commit"], out["token"], out["stats"])
        steps += 1
        st = rpd.stats_dict(out["stats"].cpu())
        if st["status"] != 0 or st["n_masked"] - st["n_committed"] <= limit or steps >= max_steps:
            break
    torch.cuda.synchronize(DEV)
    return steps, out


def device_loop(ctx, case, hidden, mask, stop_frac, max_steps, forward_graph=None):
    N = case["N"]
    out = outputs(N)
    steps = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    loop = ctx.build_decode_loop(hidden, mask, case["tau"], case["budget"], out["commit"],
                                 out["token"], out["stats"], steps, stop_frac=stop_frac,
                                 max_steps=max_steps, forward=forward_graph)
    try:
        loop.launch()
        torch.cuda.synchronize(DEV)
    finally:
        loop.close()
    return int(steps.item()), out


def same_state(a, b, mask_a, mask_b):
    (sa, oa), (sb, ob) = a, b
    assert sa == sb
    assert torch.equal(mask_a, mask_b)
    assert torch.equal(oa["commit"], ob["commit"]) and torch.equal(oa["token"], ob["token"])
    assert rpd.stats_dict(oa["stats"].cpu()) == rpd.stats_dict(ob["stats"].cpu())


@pytest.mark.parametrize("stop_frac,max_steps,projection,profile", [
    (0.0, 200, "all", None), (0.25, 200, "all", None), (0.0, 3, "all", None),
    (0.0, 200, "lazy", None),            # k_band and a second projection pass inside the loop
    (0.0, 200, "auto", None),
    (0.0, 200, "all", "llada_block"),    # RPD-block: the active block's positions only
])
def test_device_loop_matches_host_loop_without_forward(stop_frac, max_steps, projection, profile):
    """Fixed hidden states: every step commits at least one position, so the loop ends by the
    masked fraction or by max_steps."""
    case = small_case(2101, K=3, N=64, d=256, V=4100, w_std=0.08)
    ctx = context(case, projection, profile)
    try:
        hidden = case["hidden"].to(DEV).contiguous()
        m_host = case["mask"].to(DEV).clone()
        m_dev = case["mask"].to(DEV).clone()
        a = host_loop(ctx, case, hidden, m_host, lambda: None, stop_frac, max_steps)
        b = device_loop(ctx, case, hidden, m_dev, stop_frac, max_steps)
        same_state(a, b, m_host, m_dev)
        assert a[0] == min(max_steps, a[0]) and a[0] >= 1
        remaining = int(m_dev.sum())
        assert remaining <= int(np.floor(stop_frac * case["N"])) or a[0] == max_steps
    finally:
        ctx.close()


def test_device_loop_with_a_forward_graph():
    """The forward pass reads the canvas: hidden = bf16(base + (committed fraction) * drift),
    recomputed before every step; captured once as a CUDA graph for the device loop, run
    eagerly before every host step."""
    case = small_case(2102, K=3, N=96, d=256, V=4100, w_std=0.08, mask_frac=0.9)
    ctx = context(case)
    try:
        base = case["hidden"].to(DEV).float()
        drift = torch.randn(base.shape, generator=torch.Generator().manual_seed(5)).to(DEV)

        def make_forward(hidden, mask):
            def fwd():
                committed = 1.0 - mask.float().mean()
                hidden.copy_((base + 3.0 * committed * drift).to(torch.bfloat16))
            return fwd

        h_host = torch.empty_like(base, dtype=torch.bfloat16)
        m_host = case["mask"].to(DEV).clone()
        a = host_loop(ctx, case, h_host, m_host, make_forward(h_host, m_host), 0.0, 100)

        h_dev = torch.empty_like(base, dtype=torch.bfloat16)
        m_dev = case["mask"].to(DEV).clone()
        fwd = make_forward(h_dev, m_dev)
        try:
            graph = torch.cuda.CUDAGraph(keep_graph=True)
        except TypeError:
            pytest.skip("this PyTorch cannot hand out its captured graph")
        fwd()  # warm the ops up outside the capture
        m_dev.copy_(case["mask"].to(DEV))
        with torch.cuda.graph(graph):
            fwd()
        b = device_loop(ctx, case, h_dev, m_dev, 0.0, 100, forward_graph=graph)
        same_state(a, b, m_host, m_dev)
        assert torch.equal(h_host, h_dev)  # the last forward pass saw the same canvas
    finally:
        ctx.close()


def test_decode_loop_refusals():
    case = small_case(2103, K=2, N=32, d=256, V=4100, w_std=0.08)
    ctx = context(case)
    try:
        hidden = case["hidden"].to(DEV).contiguous()
        mask = case["mask"].to(DEV).clone()
        out = outputs(case["N"])
        steps = torch.zeros(1, dtype=torch.int32, device=DEV)
        for kw in (dict(stop_frac=1.5), dict(stop_frac=-0.1), dict(max_steps=0)):
            args = dict(stop_frac=0.0, max_steps=10)
            args.update(kw)
            with pytest.raises(rpd.RpdError) as e:
                ctx.build_decode_loop(hidden, mask, case["tau"], case["budget"], out["commit"],
                                      out["token"], out["stats"], steps, **args)
            assert e.value.code == rpd.RPD_ERR_INVALID_ARGUMENT
        exe = ctypes.c_void_p()
        host_steps = torch.zeros(1, dtype=torch.int32)
        rc = rpd.rpd_build_decode_loop(ctx.handle, None, hidden.data_ptr(), mask.data_ptr(), case["N"],
                                       ctypes.c_float(case["tau"]), ctypes.c_float(case["budget"]),
                                       out["commit"].data_ptr(), out["token"].data_ptr(),
                                       out["stats"].data_ptr(), ctypes.c_float(0.0), 10,
                                       host_steps.data_ptr(), ctypes.byref(exe))
        assert rc == rpd.RPD_ERR_INVALID_ARGUMENT and not exe.value  # host memory for steps
        assert rpd.rpd_decode_loop_launch(None, None, None) == rpd.RPD_ERR_INVALID_ARGUMENT
        assert rpd.rpd_decode_loop_launch(ctx.handle, ctypes.c_void_p(12345), None) == \
            rpd.RPD_ERR_INVALID_ARGUMENT  # not a loop of this context
    finally:
        ctx.close()
    shard = rpd.Rpd(case["d"], 2048, case["K"], case["eps"])
    try:
        shard.set_head(case["W"][:2048].to(DEV), case["g"].to(DEV))
        shard.set_vocab_shard(0, case["V"])
        with pytest.raises(rpd.RpdError) as e:
            shard.build_decode_loop(hidden, mask, case["tau"], case["budget"], out["commit"],
                                    out["token"], out["stats"], steps)
        assert e.value.code == rpd.RPD_ERR_UNSUPPORTED
    finally:
        shard.close()


def test_loop_is_refused_after_scratch_or_head_change():
    """A loop records the context's scratch and head: after scratch grows, or the head is
    replaced, launching it is refused (it would read freed memory); a rebuilt loop runs."""
    case = small_case(2104, K=2, N=32, d=256, V=4100, w_std=0.08)
    ctx = context(case)
    try:
        hidden = case["hidden"].to(DEV).contiguous()
        mask = case["mask"].to(DEV).clone()
        out = outputs(case["N"])
        steps = torch.zeros(1, dtype=torch.int32, device=DEV)

        def build():
            return ctx.build_decode_loop(hidden, mask, case["tau"], case["budget"], out["commit"],
                                         out["token"], out["stats"], steps, stop_frac=0.5,
                                         max_steps=4)
        loop = build()
        loop.launch()
        torch.cuda.synchronize(DEV)
        assert int(steps.item()) >= 1
        ctx.reserve(1, 4 * case["N"])  # scratch reallocated
        with pytest.raises(rpd.RpdError) as e:
            loop.launch()
        assert e.value.code == rpd.RPD_ERR_INVALID_ARGUMENT
        loop.close()
        loop = build()
        mask.copy_(case["mask"].to(DEV))
        loop.launch()
        torch.cuda.synchronize(DEV)
        ctx.set_head(case["W"].to(DEV), case["g"].to(DEV))  # head replaced
        with pytest.raises(rpd.RpdError):
            loop.launch()
        loop.close()
        kept = build()  # freed by the context's destruction
    finally:
        ctx.close()
    kept.close()  # after the context: a no-op


def test_batched_device_loop_matches_host_loop():
    """Three canvases of different masked fractions and thresholds: the loop runs until every
    canvas is down to floor(stop_frac * N) masked positions; the host loop of rpd_step_batched
    reaches the same state."""
    import workloads as WL
    B, N, K, d, V = 3, 48, 3, 256, 4100
    W, g = WL.make_head(V, d, 2105, w_std=0.08)
    b = WL.u_profile(N, 0.5, 3.0)
    sigma = WL.calibrated_sigma(V, d, 0.08, b_max=float(b.max()))
    hidden = torch.stack([WL.make_hidden(W, K, N, 3000 + i, b, sigma, flip_frac=0.1).hidden
                          for i in range(B)], dim=1).to(DEV).contiguous()
    mask0 = torch.stack([WL.uniform_fraction_mask(N, f, 40 + i)
                         for i, f in enumerate((1.0, 0.6, 0.8))]).to(DEV)
    taus, budgets = [0.9, 0.85, 0.95], [1.0, 2.0, 0.5]
    ctx = rpd.Rpd(d, V, K, 1e-6)
    ctx.set_stream(torch.cuda.current_stream(DEV))
    ctx.set_head(W.to(DEV), g.to(DEV))
    ctx.set_profile("llada")
    ctx.reserve(B, N)

    def outs():
        return dict(commit=torch.zeros(B, N, dtype=torch.uint8, device=DEV),
                    token=torch.full((B, N), -1, dtype=torch.int32, device=DEV),
                    stats=torch.zeros(B, rpd.STATS_WORDS, dtype=torch.int32, device=DEV))
    try:
        stop_frac, limit = 0.1, int(np.floor(0.1 * N))
        m_host, oh = mask0.clone(), outs()
        n = 0
        while True:
            ctx.step_batched(hidden, m_host, taus, budgets, oh["commit"], oh["token"], oh["stats"])
            n += 1
            st = [rpd.stats_dict(oh["stats"][i].cpu()) for i in range(B)]
            if any(x["status"] != 0 for x in st) or \
                    all(x["n_masked"] - x["n_committed"] <= limit for x in st) or n >= 100:
                break
        m_dev, od = mask0.clone(), outs()
        steps = torch.zeros(1, dtype=torch.int32, device=DEV)
        loop = ctx.build_decode_loop_batched(hidden, m_dev, taus, budgets, od["commit"], od["token"],
                                             od["stats"], steps, stop_frac=stop_frac, max_steps=100)
        loop.launch()
        torch.cuda.synchronize(DEV)
        loop.close()
        assert int(steps.item()) == n
        assert torch.equal(m_host, m_dev)
        assert torch.equal(oh["commit"], od["commit"]) and torch.equal(oh["token"], od["token"])
        assert torch.equal(oh["stats"], od["stats"])
        assert all(int(m_dev[i].sum()) <= limit for i in range(B))
    finally:
        ctx.close()
