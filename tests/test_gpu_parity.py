"""Parity of the CUDA commit step with the CPU oracle, through the C ABI, on cuda:0.

Tolerances and the near-threshold exemption are stated in ``tests/parity.py``.
Small cases compare every output element by element; the full-size LLaDA-8B and
Dream-7B head shapes run the oracle over every projected row (fp64 BLAS).
"""
import math

import numpy as np
import pytest
import torch

import workloads as WL
from oracle import rpd_oracle as O
from tests.gpu_util import DeviceRunner, bits
from tests.parity import compare_block_step, compare_step

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, never run there
    pytest.skip("needs a CUDA GPU", allow_module_level=True)


def rpd_mod():
    import paper_2609_36452_gb300 as rpd
    return rpd


def oracle_step(case, hidden=None, mask=None, tau=None, budget=None, rule=None):
    hidden = case["hidden"] if hidden is None else hidden
    mask = case["mask"] if mask is None else mask
    return O.rpd_step(bits(hidden), mask.numpy(), bits(case["g"]), bits(case["W"]), case["eps"],
                      case["tau"] if tau is None else tau,
                      case["budget"] if budget is None else budget,
                      case["rule"] if rule is None else rule)


def small_case(seed, K=3, N=64, d=256, V=4096, w_std=0.08, sigma=None, flip=0.1, a=None,
               mask_frac=1.0, tau=0.9, budget=1.0, rule="llada", b=None):
    """Calibrated small workload: U-shaped signal whose canvas ends are confident."""
    W, g = WL.make_head(V, d, seed, w_std=w_std)
    b = WL.u_profile(N, 0.5, 3.0) if b is None else b
    if sigma is None:
        sigma = WL.calibrated_sigma(V, d, w_std, b_max=float(b.max()))
    cv = WL.make_hidden(W, K, N, seed + 1000, b, sigma, flip_frac=flip, a=a)
    mask = torch.ones(N, dtype=torch.uint8) if mask_frac >= 1.0 else \
        WL.uniform_fraction_mask(N, mask_frac, seed + 5)
    return dict(W=W, g=g, hidden=cv.hidden, mask=mask, K=K, N=N, d=d, V=V, eps=1e-6, tau=tau,
                budget=budget, rule=rule)


def run_and_compare(case, rule=None, tau=None, budget=None, mask=None):
    runner = DeviceRunner(case["W"], case["g"], case["K"], case["eps"],
                          rule=case["rule"] if rule is None else rule)
    try:
        m = case["mask"] if mask is None else mask
        got = runner.step(case["hidden"], m, case["tau"] if tau is None else tau,
                          case["budget"] if budget is None else budget)
        ref = oracle_step(case, mask=m, tau=tau, budget=budget, rule=rule)
        rep = compare_step(ref, got)
        return ref, got, rep
    finally:
        runner.close()


# ------------------------------------------------------------------------- small cases

def test_tiny_literal_takes_fallback():
    """The literal tiny workload (N=64, K=3, d=256, V=4096): no confident position exists,
    so every step is the fallback commit of the most confident early position."""
    case = WL.tiny_step(seed=1, calibrated=False)
    ref, got, rep = run_and_compare(case)
    assert got["stats"]["fallback_used"] == 1 and got["stats"]["n_committed"] == 1
    assert np.nanmax(ref.conf) < 0.05
    print(rep)


@pytest.mark.parametrize("seed", [1, 2, 3, 4])
def test_tiny_calibrated(seed):
    case = WL.tiny_step(seed=seed, calibrated=True)
    ref, got, rep = run_and_compare(case)
    print(rep)


def test_paths_are_exercised():
    """Across a few calibrated seeds the budget holds candidates back, high-confidence and
    stability admissions both commit, and flipped positions have persistence 1."""
    held = high = stab = 0
    for seed in range(10, 16):
        case = small_case(seed, K=4, N=96, a=torch.ones(4), flip=0.15)
        ref, got, rep = run_and_compare(case, rule=dict(O.RULES["llada"], theta_s=2.0))
        held += int(ref.cand.sum() - len(ref.accepted))
        high += got["stats"]["n_high_conf"]
        stab += got["stats"]["n_stability"]
    assert held > 0 and high > 0 and stab > 0, (held, high, stab)


@pytest.mark.parametrize("d,V,K,N,frac", [
    (200, 1000, 2, 77, 0.7),     # ragged K-block (200 = 3*64+8) and vocabulary tile (1000)
    (128, 4100, 5, 300, 1.0),    # 1500 rows: 12 row tiles, last one ragged; V ragged
    (64, 256, 1, 33, 1.0),       # single vocabulary tile, K = 1
    (4096, 1280, 3, 50, 0.5),    # LLaDA hidden size, 64 K-blocks
])
def test_ragged_shapes(d, V, K, N, frac):
    case = small_case(7 + d + V, K=K, N=N, d=d, V=V, w_std=0.08, mask_frac=frac)
    ref, got, rep = run_and_compare(case)
    print(rep)


@pytest.mark.parametrize("tiling", ["pair", "rows_n"])
@pytest.mark.parametrize("d,V,K,N,frac", [
    (256, 4100, 3, 100, 1.0),    # 300 rows: ragged last tile / one 320-row group
    (4096, 1280, 3, 50, 1.0),    # 150 rows, 64 K-blocks
    (200, 1000, 2, 77, 0.7),     # ragged K-block and vocabulary tile, ~108 rows
    (128, 4100, 5, 300, 1.0),    # 1500 rows: 6 pair row tiles / 3 groups of 512
    (64, 512, 4, 128, 1.0),      # 512 rows: whole tiles / one full group
])
def test_head_tilings_match_oracle(tiling, d, V, K, N, frac):
    """Both head tilings, forced, on the same inputs; each is compared with the oracle
    element by element."""
    case = small_case(11 + d + V + K, K=K, N=N, d=d, V=V, w_std=0.08, mask_frac=frac)
    runner = DeviceRunner(case["W"], case["g"], K, case["eps"], rule=case["rule"])
    try:
        runner.ctx.set_head_tiling(tiling)
        got = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
    finally:
        runner.close()
    ref = oracle_step(case)
    print(compare_step(ref, got))


@pytest.mark.parametrize("tiling", ["pair", "rows_n"])
@pytest.mark.parametrize("d,V,K,N", [
    (256, 4100, 3, 100),    # ragged last vocabulary block (4100 = 32 x 128 + 4)
    (4096, 1280, 2, 150),   # 64 column blocks per row block
    (192, 2100, 4, 300),    # 1200 rows: several row tiles / two groups
])
def test_head_layouts_give_identical_outputs(tiling, d, V, K, N):
    """The context's tiled copy of the head and the caller's row-major head feed the MMAs the
    same operands in the same order, so every output is bitwise the same."""
    case = small_case(1300 + d + K, K=K, N=N, d=d, V=V, w_std=0.08)
    outs = {}
    for layout in ("tiled", "borrowed"):
        runner = DeviceRunner(case["W"], case["g"], K, case["eps"], rule=case["rule"], layout=layout)
        try:
            runner.ctx.set_head_tiling(tiling)
            outs[layout] = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
        finally:
            runner.close()
    a, b = outs["tiled"], outs["borrowed"]
    assert a["stats"] == b["stats"]
    for k in a:
        if k != "stats":
            assert np.array_equal(a[k], b[k]), k


def test_tiled_head_is_a_copy_and_borrowed_head_is_read_in_place():
    """After rpd_set_head the tiled layout no longer reads the caller's W (overwriting W leaves
    the outputs unchanged); the borrowed layout reads it at every step (the same overwrite
    changes them).  Unknown layouts are refused."""
    case = small_case(1401, K=2, N=48, d=256, V=4100, w_std=0.08)
    outs = {}
    for layout in ("tiled", "borrowed"):
        runner = DeviceRunner(case["W"], case["g"], 2, case["eps"], rule=case["rule"], layout=layout)
        try:
            before = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
            runner.W.copy_(torch.flip(runner.W, dims=[0]))  # the caller's buffer, rows reversed
            after = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
            outs[layout] = (before, after)
        finally:
            runner.close()
    b, a = outs["tiled"]
    assert np.array_equal(b["layer_argmax"], a["layer_argmax"]) and np.array_equal(b["conf"], a["conf"])
    b, a = outs["borrowed"]
    assert not np.array_equal(b["layer_argmax"], a["layer_argmax"])
    import paper_2609_36452_gb300 as rpd
    ctx = rpd.Rpd(256, 4100, 2, 1e-6)
    try:
        with pytest.raises(rpd.RpdError) as e:
            rpd._check(rpd.rpd_set_head_layout(ctx.handle, 7))
        assert e.value.code == rpd.RPD_ERR_INVALID_ARGUMENT
    finally:
        ctx.close()


@pytest.mark.parametrize("tiling", ["pair", "rows_n"])
@pytest.mark.parametrize("rows", [1, 64, 127, 128, 129, 257, 320, 383, 384, 385, 513, 769, 832,
                                  895, 896, 897, 1023, 1025])
def test_row_counts_around_tile_boundaries(tiling, rows):
    """Row counts 256q + {1, 64, 127, 128, 129} (and around the 512-row group of the rows-on-N
    tiling) on both tilings: one window layer, so the pass projects exactly `rows` rows; every
    output is compared with the oracle."""
    case = small_case(700 + rows, K=1, N=rows, d=192, V=2100, w_std=0.08)
    runner = DeviceRunner(case["W"], case["g"], 1, case["eps"], rule=case["rule"])
    try:
        runner.ctx.set_head_tiling(tiling)
        got = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
    finally:
        runner.close()
    assert got["stats"]["n_rows"] == rows
    print(compare_step(oracle_step(case), got))


@pytest.mark.parametrize("rows", [280, 300, 320, 416])
def test_rows_n_tmem_ring_with_several_tiles_per_pair(rows):
    """Rows-on-N groups of 288 and 320 columns go round the ring of TMEM chunks (the second
    tile of a CTA pair wraps at column 512 and waits for chunks of the first), 416 columns use
    all of TMEM in turn.  A vocabulary of 60000 entries (235 tiles) gives every pair about three
    tiles; every output is compared with the oracle."""
    case = small_case(1500 + rows, K=1, N=rows, d=256, V=60000, w_std=0.08)
    runner = DeviceRunner(case["W"], case["g"], 1, case["eps"], rule=case["rule"])
    try:
        runner.ctx.set_head_tiling("rows_n")
        got = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
    finally:
        runner.close()
    assert got["stats"]["n_rows"] == rows
    print(compare_step(oracle_step(case), got))


@pytest.mark.parametrize("K,N", [(4, 70), (4, 107), (4, 128), (2, 300)])
def test_rows_n_groups_with_window_layers(K, N):
    """The rows-on-N tiling with several window layers (rows are layer-major, so a group mixes
    layers and positions): 280, 428 (two groups of 224 or one of 448), 512 and 600 rows."""
    case = small_case(900 + K * N, K=K, N=N, d=256, V=4100, w_std=0.08)
    runner = DeviceRunner(case["W"], case["g"], K, case["eps"], rule=case["rule"])
    try:
        runner.ctx.set_head_tiling("rows_n")
        got = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
    finally:
        runner.close()
    print(compare_step(oracle_step(case), got))


def test_many_row_tiles_in_bands():
    """5100 rows at d = 4096: 20 CTA-pair row tiles (10 rows-on-N groups) of 2-4 MB of u each,
    more than the head kernels keep in one L2 band of work units, so every row of the second
    band comes from the band-ordered unit walk.  Every output is compared with the oracle."""
    case = small_case(301, K=5, N=1020, d=4096, V=4100, w_std=0.02)
    ref, got, rep = run_and_compare(case)
    assert got["stats"]["n_rows"] == 5 * 1020
    print(rep)


def test_stability_route_with_drops():
    """Flat layer ramp with explicit theta_s: persistence is long and drops small but
    nonzero, so the stability route admits and rejects on the drop penalty."""
    case = small_case(31, K=6, N=128, a=torch.tensor([1.0, 0.95, 1.05, 1.0, 0.97, 1.0]), flip=0.1)
    rule = dict(theta_c=0.6, theta_s=4.5, w=15.0, k_max=6, window=32)
    ref, got, rep = run_and_compare(case, rule=rule, budget=50.0)
    m = ref.masked
    assert np.any(ref.drop[m] > 0.001)
    print(rep, "stability commits", got["stats"]["n_stability"])


@pytest.mark.parametrize("tau,budget", [(0.9, 0.0), (0.9, math.inf), (1.0, 1.0), (0.61, 4.0)])
def test_threshold_extremes(tau, budget):
    case = small_case(41, K=3, N=80)
    run_and_compare(case, tau=tau, budget=budget)


def test_fallback_window_counts_masked_positions():
    case = small_case(43, K=3, N=100, mask_frac=0.4, w_std=0.02, sigma=1.0)
    rule = dict(O.RULES["llada"], window=3)
    ref, got, rep = run_and_compare(case, rule=rule)
    assert got["stats"]["fallback_used"] == 1
    first3 = np.nonzero(ref.masked)[0][:3]
    assert got["stats"]["fallback_pos"] in first3


def test_empty_and_single_masks():
    case = small_case(45, K=3, N=40)
    runner = DeviceRunner(case["W"], case["g"], 3)
    try:
        none = torch.zeros(40, dtype=torch.uint8)
        got = runner.step(case["hidden"], none, 0.9, 1.0)
        assert got["commit"].sum() == 0 and np.all(got["new_mask"] == 0)
        assert got["stats"]["n_masked"] == 0 and got["stats"]["n_committed"] == 0
        assert got["stats"]["fallback_pos"] == -1 and got["stats"]["status"] == 0
        assert np.all(got["token"] == -5)  # tokens untouched where nothing commits
        one = torch.zeros(40, dtype=torch.uint8)
        one[17] = 1
        got = runner.step(case["hidden"], one, 0.9, 1.0)
        ref = oracle_step(case, mask=one)
        compare_step(ref, got)
        assert got["commit"][17] == 1 and got["stats"]["n_committed"] == 1
        # N = 1
        h1 = case["hidden"][:, :1].contiguous()
        got = runner.step(h1, torch.ones(1, dtype=torch.uint8), 0.9, 1.0)
        assert got["commit"][0] == 1
    finally:
        runner.close()


def test_batched_matches_per_canvas_oracle():
    K, N, d, V, B = 3, 120, 256, 2048, 4
    W, g = WL.make_head(V, d, 51, w_std=0.08)
    hidden = torch.empty(K, B, N, d, dtype=torch.bfloat16)
    masks = torch.empty(B, N, dtype=torch.uint8)
    for b in range(B):
        cv = WL.make_hidden(W, K, N, 600 + b, WL.u_profile(N, 0.5, 3.0),
                              WL.calibrated_sigma(V, d, 0.08, 3.0), flip_frac=0.1)
        hidden[:, b] = cv.hidden
        masks[b] = WL.uniform_fraction_mask(N, [1.0, 0.5, 0.0, 0.9][b], 700 + b)
    taus, budgets = [0.9, 0.8, 0.9, 0.95], [1.0, 3.0, 1.0, 0.5]
    runner = DeviceRunner(W, g, K)
    try:
        outs = runner.step_batched(hidden, masks, taus, budgets)
    finally:
        runner.close()
    for b in range(B):
        ref = O.rpd_step(bits(hidden[:, b]), masks[b].numpy(), bits(g), bits(W), 1e-6, taus[b],
                         budgets[b], "llada")
        compare_step(ref, outs[b])
    assert outs[2]["stats"]["n_masked"] == 0


def test_largest_batch():
    """B = 128 canvases (the most one call accepts) of 24 positions, with masked counts from
    0 and 1 up to all 24 and per-canvas thresholds; every canvas against its own oracle
    step.  B = 129 is refused."""
    K, N, d, V, B = 2, 24, 128, 1024, 128
    W, g = WL.make_head(V, d, 57, w_std=0.3)
    hidden = torch.empty(K, B, N, d, dtype=torch.bfloat16)
    masks = torch.zeros(B, N, dtype=torch.uint8)
    gen = torch.Generator().manual_seed(5700)
    for b in range(B):
        cv = WL.make_hidden(W, K, N, 5800 + b, WL.u_profile(N, 0.5, 3.0),
                              WL.calibrated_sigma(V, d, 0.3, 3.0), flip_frac=0.1)
        hidden[:, b] = cv.hidden
        n_masked = b % (N + 1)                      # 0, 1, ..., N, 0, 1, ...
        masks[b, torch.randperm(N, generator=gen)[:n_masked]] = 1
    taus = [0.9 if b % 3 else 0.7 for b in range(B)]
    budgets = [float(b % 5) for b in range(B)]
    runner = DeviceRunner(W, g, K)
    try:
        outs = runner.step_batched(hidden, masks, taus, budgets)
        import paper_2609_36452_gb300 as rpd
        dev = torch.device("cuda:0")
        big = torch.ones(B + 1, N, dtype=torch.uint8, device=dev)
        h = torch.zeros(K, B + 1, N, d, dtype=torch.bfloat16, device=dev)
        c = torch.zeros(B + 1, N, dtype=torch.uint8, device=dev)
        t = torch.zeros(B + 1, N, dtype=torch.int32, device=dev)
        s = torch.zeros(B + 1, rpd.STATS_WORDS, dtype=torch.int32, device=dev)
        with pytest.raises(rpd.RpdError) as e:
            runner.ctx.step_batched(h, big, [0.9] * (B + 1), [1.0] * (B + 1), c, t, s)
        assert e.value.code == rpd.RPD_ERR_UNSUPPORTED
    finally:
        runner.close()
    for b in range(B):
        ref = O.rpd_step(bits(hidden[:, b]), masks[b].numpy(), bits(g), bits(W), 1e-6, taus[b],
                         budgets[b], "llada")
        compare_step(ref, outs[b])
        assert (outs[b]["stats"]["n_committed"] >= 1) == (b % (N + 1) > 0)


@pytest.mark.parametrize("projection", ["all", "lazy"])
@pytest.mark.parametrize("pinned_hidden", [True, False])
def test_host_entry_point_matches_device(pinned_hidden, projection):
    """rpd_step_host equals rpd_step: hidden in pinned memory is read in place (by both
    projection passes when lazy), hidden in pageable memory is copied to the device first."""
    case = small_case(61, K=3, N=64, mask_frac=0.7, a=torch.ones(3))
    runner = DeviceRunner(case["W"], case["g"], 3)
    runner.ctx.set_projection(projection)
    try:
        dev = runner.step(case["hidden"], case["mask"], 0.9, 1.0)
        hid = case["hidden"].contiguous()
        hid = hid.pin_memory() if pinned_hidden else hid.clone()
        mask = case["mask"].clone().pin_memory()
        commit = torch.zeros(64, dtype=torch.uint8).pin_memory()
        token = torch.full((64,), -5, dtype=torch.int32).pin_memory()
        stats = torch.zeros(rpd_mod().STATS_WORDS, dtype=torch.int32).pin_memory()
        runner.ctx.set_debug()
        runner.ctx.step_host(hid, mask, 0.9, 1.0, commit, token, stats)
        assert np.array_equal(commit.numpy(), dev["commit"])
        assert np.array_equal(mask.numpy(), dev["new_mask"])
        sel = dev["commit"] == 1
        assert np.array_equal(token.numpy()[sel], dev["token"][sel])
        assert np.all(token.numpy()[~sel] == -5)
        assert runner.rpd.stats_dict(stats) == dev["stats"]
    finally:
        runner.close()


def test_repeat_is_bit_identical():
    case = small_case(71, K=4, N=200, d=512, V=3000)
    runner = DeviceRunner(case["W"], case["g"], 4)
    try:
        a = runner.step(case["hidden"], case["mask"], 0.9, 1.0)
        b = runner.step(case["hidden"], case["mask"], 0.9, 1.0)
    finally:
        runner.close()
    for k in a:
        if k == "stats":
            assert a[k] == b[k]
        else:
            assert np.array_equal(a[k], b[k]), k


def test_invalid_arguments_on_gpu():
    import paper_2609_36452_gb300 as rpd
    ctx = rpd.Rpd(256, 4096, 3)
    dev = torch.device("cuda:0")
    h = torch.zeros(3, 8, 256, dtype=torch.bfloat16, device=dev)
    m = torch.ones(8, dtype=torch.uint8, device=dev)
    c = torch.zeros(8, dtype=torch.uint8, device=dev)
    t = torch.zeros(8, dtype=torch.int32, device=dev)
    s = torch.zeros(rpd.STATS_WORDS, dtype=torch.int32, device=dev)
    with pytest.raises(rpd.RpdError) as e:
        ctx.step(h, m, 0.9, 1.0, c, t, s)
    assert e.value.code == rpd.RPD_ERR_NO_HEAD
    W = torch.zeros(4096, 256, dtype=torch.bfloat16, device=dev)
    g = torch.ones(256, dtype=torch.bfloat16, device=dev)
    ctx.set_head(W, g)
    for tau, budget in [(0.5, 1.0), (0.0, 1.0), (1.5, 1.0), (0.9, -1.0), (0.9, float("nan"))]:
        with pytest.raises(rpd.RpdError) as e:
            ctx.step(h, m, tau, budget, c, t, s)
        assert e.value.code == rpd.RPD_ERR_INVALID_ARGUMENT
    with pytest.raises(rpd.RpdError) as e:
        ctx.set_rule(0.6, 3.5, 15.0, 0, 32)
    assert e.value.code == rpd.RPD_ERR_INVALID_ARGUMENT
    # TMA needs 16-byte aligned rows: a hidden tensor or head that starts 2 bytes off is
    # refused before any work (outputs untouched)
    flat = torch.zeros(3 * 8 * 256 + 1, dtype=torch.bfloat16, device=dev)
    c.fill_(7)
    with pytest.raises(rpd.RpdError) as e:
        ctx.step(flat[1:].view(3, 8, 256), m, 0.9, 1.0, c, t, s)
    assert e.value.code == rpd.RPD_ERR_INVALID_ARGUMENT
    torch.cuda.synchronize(dev)
    assert torch.all(c == 7) and torch.all(m == 1)
    Wflat = torch.zeros(4096 * 256 + 1, dtype=torch.bfloat16, device=dev)
    with pytest.raises(rpd.RpdError) as e:
        ctx.set_head(Wflat[1:].view(4096, 256), g)
    assert e.value.code == rpd.RPD_ERR_INVALID_ARGUMENT
    # a host head handed to the C ABI directly (past the binding's own checks) is refused
    import ctypes
    W_host = torch.zeros(4096, 256, dtype=torch.bfloat16)
    rc = rpd.rpd_set_head(ctx.handle, ctypes.c_void_p(W_host.data_ptr()), ctypes.c_void_p(g.data_ptr()))
    assert rc == rpd.RPD_ERR_INVALID_ARGUMENT and b"device memory" in rpd.rpd_last_error()
    ctx.set_head(W, g)  # still usable
    ctx.close()


# ------------------------------------------------------------------ full-size head shapes

@pytest.fixture(scope="module")
def llada_head():
    return WL.make_head(WL.LLADA_V, WL.LLADA_D, seed=2)


def test_llada_first_step_full(llada_head):
    """Batch 1, N=256 all masked, K=4, d=4096, V=126464 (1024 projected rows): every row
    checked against the oracle."""
    W, g = llada_head
    case = WL.llada_first_step(seed=2, W=W, g=g)
    ref, got, rep = run_and_compare(case)
    print(rep, got["stats"])
    assert got["stats"]["n_committed"] >= 1


def test_dream_mid_decode_full():
    """Batch 1, N=512, front-loaded 50% mask, K=4, d=3584, V=152064, tau 0.85, budget 2,
    Dream rule profile."""
    case = WL.dream_mid_decode(seed=3)
    ref, got, rep = run_and_compare(case)
    print(rep, got["stats"])


# ----------------------------------------------------------------------------- RPD-block

def block_rule(block, base="llada"):
    return dict(O.RULES[base], block=block)


@pytest.mark.parametrize("block,prefix", [(32, 0), (32, 40), (16, 70), (8, 3)])
def test_rpd_block_matches_oracle(block, prefix):
    """RPD-block on a calibrated canvas whose first ``prefix`` positions are committed: the
    active block is the first one still holding a masked position."""
    case = small_case(91 + block + prefix, K=4, N=128, a=torch.ones(4), flip=0.15)
    mask = case["mask"].clone()
    mask[:prefix] = 0
    rule = block_rule(block)
    runner = DeviceRunner(case["W"], case["g"], case["K"], case["eps"], rule=rule)
    try:
        got = runner.step(case["hidden"], mask, case["tau"], case["budget"])
    finally:
        runner.close()
    ref = O.rpd_block_step(bits(case["hidden"]), mask.numpy(), bits(case["g"]), bits(case["W"]),
                           case["eps"], case["tau"], rule, block=block)
    rep = compare_block_step(ref, got)
    print(rep, got["stats"])


def test_rpd_block_batched_canvases():
    K, N, d, V, B = 3, 96, 256, 2048, 3
    W, g = WL.make_head(V, d, 92, w_std=0.08)
    hidden = torch.empty(K, B, N, d, dtype=torch.bfloat16)
    masks = torch.ones(B, N, dtype=torch.uint8)
    for b in range(B):
        cv = WL.make_hidden(W, K, N, 800 + b, WL.u_profile(N, 0.5, 3.0),
                            WL.calibrated_sigma(V, d, 0.08, 3.0), flip_frac=0.1)
        hidden[:, b] = cv.hidden
    masks[1, :33] = 0   # canvas 1: active block starts at 32
    masks[2, :] = 0     # canvas 2: nothing masked
    rule = block_rule(32)
    runner = DeviceRunner(W, g, K, rule=rule)
    try:
        outs = runner.step_batched(hidden, masks, [0.9] * B, [1.0] * B)
    finally:
        runner.close()
    for b in range(B):
        ref = O.rpd_block_step(bits(hidden[:, b]), masks[b].numpy(), bits(g), bits(W), 1e-6, 0.9,
                               rule, block=32)
        compare_block_step(ref, outs[b])
    assert outs[2]["stats"]["n_committed"] == 0


def test_rpd_block_llada_first_step_full(llada_head):
    """RPD-block at the LLaDA-8B head shape: only the first 32 positions are projected."""
    W, g = llada_head
    case = WL.llada_first_step(seed=2, W=W, g=g)
    rule = block_rule(32)
    runner = DeviceRunner(W, g, case["K"], case["eps"], rule=rule)
    try:
        got = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
    finally:
        runner.close()
    ref = O.rpd_block_step(bits(case["hidden"]), case["mask"].numpy(), bits(g), bits(W),
                           case["eps"], case["tau"], rule, block=32)
    rep = compare_block_step(ref, got)
    print(rep, got["stats"])


# ----------------------------------------------------------------------------- lazy projection

def run_lazy_and_eager(case, rule=None, tau=None, budget=None):
    outs = {}
    for lazy in (False, True):
        runner = DeviceRunner(case["W"], case["g"], case["K"], case["eps"],
                              rule=case["rule"] if rule is None else rule)
        runner.ctx.set_projection(lazy)
        try:
            outs[lazy] = runner.step(case["hidden"], case["mask"], case["tau"] if tau is None else tau,
                                     case["budget"] if budget is None else budget)
        finally:
            runner.close()
    return outs[False], outs[True]


def check_lazy(case, eager, lazy, ref, K):
    rep = compare_step(ref, lazy, lazy=True)
    assert np.array_equal(lazy["commit"], eager["commit"])
    assert np.array_equal(lazy["new_mask"], eager["new_mask"])
    sel = lazy["commit"] == 1
    assert np.array_equal(lazy["token"][sel], eager["token"][sel])
    m = case["mask"].numpy().astype(bool)
    c = lazy["conf"]
    p = ref.params
    # the band test in the same precision as the kernel (fp32 confidences and thresholds)
    n_band = int(np.sum(m & (c >= np.float32(p["theta_c"])) & (c < np.float32(p["tau"]))))
    assert eager["stats"]["n_rows"] == K * int(m.sum())
    assert lazy["stats"]["n_rows"] == int(m.sum()) + (K - 1) * n_band
    return rep, n_band


@pytest.mark.parametrize("seed", [201, 202, 203])
def test_lazy_projection_small(seed):
    case = small_case(seed, K=5, N=160, a=torch.ones(5), flip=0.15, mask_frac=0.8)
    rule = dict(O.RULES["llada"], theta_s=3.0)
    eager, lazy = run_lazy_and_eager(case, rule=rule)
    ref = oracle_step(case, rule=rule)
    rep, n_band = check_lazy(case, eager, lazy, ref, case["K"])
    print(rep, "band", n_band, lazy["stats"])


def test_lazy_projection_empty_band():
    """No confidence in [theta_c, tau): the second pass has no rows and the head is streamed
    once."""
    case = small_case(205, K=4, N=64, w_std=0.02, sigma=1.0)   # every confidence ~ 1/V
    eager, lazy = run_lazy_and_eager(case)
    ref = oracle_step(case)
    rep, n_band = check_lazy(case, eager, lazy, ref, case["K"])
    assert n_band == 0 and lazy["stats"]["n_rows"] == 64


def test_lazy_projection_llada_full(llada_head):
    W, g = llada_head
    case = WL.llada_first_step(seed=2, W=W, g=g)
    eager, lazy = run_lazy_and_eager(case)
    ref = oracle_step(case)
    rep, n_band = check_lazy(case, eager, lazy, ref, case["K"])
    print(rep, "band", n_band, lazy["stats"])


@pytest.mark.parametrize("rule_name,block", [("llada", 0), ("dream", 0), ("llada", 32)])
def test_lazy_projection_batched(rule_name, block):
    """Lazy projection over several canvases with their own tau and budget (each canvas has
    its own stability band), for both Table 4 profiles and for RPD-block: commits, tokens and
    masks equal the all-layer step, every canvas matches its oracle step, and the rows
    projected are each canvas's scored positions plus the earlier layers of its band."""
    K, N, d, V, B = 4, 96, 256, 2048, 4
    W, g = WL.make_head(V, d, 77, w_std=0.08)
    hidden = torch.empty(K, B, N, d, dtype=torch.bfloat16)
    masks = torch.empty(B, N, dtype=torch.uint8)
    for b in range(B):
        cv = WL.make_hidden(W, K, N, 7700 + b, WL.u_profile(N, 0.5, 3.0),
                              WL.calibrated_sigma(V, d, 0.08, 3.0), flip_frac=0.15, a=torch.ones(K))
        hidden[:, b] = cv.hidden
        masks[b] = WL.uniform_fraction_mask(N, [1.0, 0.7, 0.4, 0.9][b], 7800 + b)
    taus, budgets = [0.9, 0.8, 0.95, 0.7], [1.0, 3.0, 0.5, 2.0]
    rule = dict(O.RULES[rule_name], theta_s=3.0, block=block)
    outs = {}
    for lazy in (False, True):
        runner = DeviceRunner(W, g, K, rule=rule)
        runner.ctx.set_projection(lazy)
        try:
            outs[lazy] = runner.step_batched(hidden, masks, taus, budgets)
        finally:
            runner.close()
    rows_lazy = 0
    for b in range(B):
        eager, lazy = outs[False][b], outs[True][b]
        assert np.array_equal(lazy["commit"], eager["commit"])
        assert np.array_equal(lazy["new_mask"], eager["new_mask"])
        sel = lazy["commit"] == 1
        assert np.array_equal(lazy["token"][sel], eager["token"][sel])
        if block:
            ref = O.rpd_block_step(bits(hidden[:, b]), masks[b].numpy(), bits(g), bits(W), 1e-6,
                                   taus[b], rule)
            compare_block_step(ref, lazy, lazy=True)
        else:
            ref = O.rpd_step(bits(hidden[:, b]), masks[b].numpy(), bits(g), bits(W), 1e-6, taus[b],
                             budgets[b], rule)
            compare_step(ref, lazy, lazy=True)
        scored = np.isfinite(ref.conf) & ref.masked
        c = lazy["conf"]
        band = scored & (c >= np.float32(rule["theta_c"])) & (c < np.float32(taus[b]))
        rows_lazy += int(scored.sum()) + (K - 1) * int(band.sum())
    # n_rows counts the rows of the whole call (all canvases)
    assert outs[True][0]["stats"]["n_rows"] == rows_lazy
    assert rows_lazy < outs[False][0]["stats"]["n_rows"]


def test_auto_projection_picks_per_step(llada_head):
    """Automatic projection: lazy at the LLaDA first step (1024 rows: bound by the tensor
    cores), every layer when 5 positions remain (bound by streaming the head); commits equal
    the all-layer step either way."""
    W, g = llada_head
    case = WL.llada_first_step(seed=2, W=W, g=g)
    tail = case["mask"].clone()
    tail[:-5] = 0
    for mask, expect_lazy in ((case["mask"], True), (tail, False)):
        outs = {}
        for mode in ("all", "auto"):
            runner = DeviceRunner(W, g, case["K"], case["eps"], rule="llada")
            runner.ctx.set_projection(mode)
            try:
                outs[mode] = runner.step(case["hidden"], mask, case["tau"], case["budget"])
            finally:
                runner.close()
        a, b = outs["all"], outs["auto"]
        assert np.array_equal(a["commit"], b["commit"]) and np.array_equal(a["new_mask"], b["new_mask"])
        sel = a["commit"] == 1
        assert np.array_equal(a["token"][sel], b["token"][sel])
        nm = int(mask.sum())
        assert a["stats"]["n_rows"] == case["K"] * nm
        if expect_lazy:
            assert b["stats"]["n_rows"] < case["K"] * nm
        else:
            assert b["stats"]["n_rows"] == case["K"] * nm


def test_batched_heterogeneous_lengths():
    """Canvases of different lengths in one batched step: each is padded to N with mask 0
    (padding is never projected, scored, counted in the budget or committed) and must equal
    the oracle on the unpadded canvas."""
    K, N, d, V = 3, 100, 256, 2048
    lengths = [100, 64, 37]
    B = len(lengths)
    W, g = WL.make_head(V, d, 93, w_std=0.08)
    hidden = torch.empty(K, B, N, d, dtype=torch.bfloat16)
    masks = torch.zeros(B, N, dtype=torch.uint8)
    for b, nb in enumerate(lengths):
        cv = WL.make_hidden(W, K, N, 900 + b, WL.u_profile(N, 0.5, 3.0),
                            WL.calibrated_sigma(V, d, 0.08, 3.0), flip_frac=0.1)
        hidden[:, b] = cv.hidden
        hidden[:, b, nb:] = 0          # padding rows carry nothing
        masks[b, :nb] = WL.uniform_fraction_mask(nb, 0.8, 950 + b)
    taus, budgets = [0.9, 0.85, 0.9], [1.0, 2.0, 0.5]
    runner = DeviceRunner(W, g, K)
    try:
        outs = runner.step_batched(hidden, masks, taus, budgets)
    finally:
        runner.close()
    for b, nb in enumerate(lengths):
        ref = O.rpd_step(bits(hidden[:, b, :nb]), masks[b, :nb].numpy(), bits(g), bits(W), 1e-6,
                         taus[b], budgets[b], "llada")
        got = {k: (v[:nb] if isinstance(v, np.ndarray) and v.ndim == 1 else
                   (v[:, :nb] if isinstance(v, np.ndarray) else v)) for k, v in outs[b].items()}
        compare_step(ref, got)
        assert np.all(outs[b]["commit"][nb:] == 0) and np.all(outs[b]["new_mask"][nb:] == 0)


# ----------------------------------------------------------------------------- failure detection

@pytest.mark.parametrize("N,K,tiling", [(256, 4, "pair"), (32, 2, "rows_n"), (150, 4, "rows_n")])
def test_stalled_head_reports_timeout_and_context_recovers(N, K, tiling):
    """A step whose head kernel issues no loads: its bounded waits run out, the step reports
    RPD_ERR_TIMEOUT in rpd_stats.status without faulting or hanging, and the next step on the
    same context is correct again (both tilings; 600 rows make one single-buffered rows-on-N
    group)."""
    import paper_2609_36452_gb300 as rpd
    case = small_case(301 + N, K=K, N=N)
    runner = DeviceRunner(case["W"], case["g"], K)
    try:
        runner.ctx.set_head_tiling(tiling)
        runner.ctx.set_wait_limit(20000)          # 20 ms
        runner.ctx.inject_stall()
        bad = runner.step(case["hidden"], case["mask"], 0.9, 1.0)
        assert bad["stats"]["status"] == rpd.RPD_ERR_TIMEOUT
        good = runner.step(case["hidden"], case["mask"], 0.9, 1.0)
    finally:
        runner.close()
    assert good["stats"]["status"] == 0
    compare_step(oracle_step(case), good)


def test_exact_argmax_tie_takes_lowest_token():
    """Two identical head rows give bitwise-equal logits; the argmax is the lower token index,
    on every layer, as the oracle's reading (first occurrence) requires."""
    K, N, d, V = 2, 8, 128, 2048
    W, g = WL.make_head(V, d, 99, w_std=0.08)
    lo, hi = 100, 1900          # different vocabulary tiles and splits
    W[hi] = W[lo]
    targets = torch.full((N,), lo, dtype=torch.long)
    cv = WL.make_hidden(W, K, N, 98, torch.full((N,), 3.0), WL.calibrated_sigma(V, d, 0.08, 3.0),
                        targets=targets)
    mask = torch.ones(N, dtype=torch.uint8)
    runner = DeviceRunner(W, g, K)
    try:
        got = runner.step(cv.hidden, mask, 0.9, 1.0)
    finally:
        runner.close()
    ref = O.rpd_step(bits(cv.hidden), mask.numpy(), bits(g), bits(W), 1e-6, 0.9, 1.0, "llada")
    assert np.all(ref.layer_argmax == lo) and np.all(ref.layer_gap == 0.0)
    assert np.all(got["layer_argmax"] == lo)
    assert np.all(got["token"][got["commit"] == 1] == lo)


def test_one_context_across_shapes_heads_and_rules():
    """One context through a sequence a serving loop produces: a short canvas, a batch that
    makes scratch grow, a short canvas again, a new head (same shape), and the Dream rule;
    every step against its own oracle."""
    K, d, V = 3, 256, 2048
    case_a = small_case(501, K=K, N=50, d=d, V=V)
    W2, g2 = WL.make_head(V, d, 502, w_std=0.08)
    runner = DeviceRunner(case_a["W"], case_a["g"], K)
    try:
        got = runner.step(case_a["hidden"], case_a["mask"], 0.9, 1.0)
        compare_step(oracle_step(case_a), got)
        # batch of 3 canvases of 300: scratch grows
        B, N = 3, 300
        hidden = torch.empty(K, B, N, d, dtype=torch.bfloat16)
        masks = torch.empty(B, N, dtype=torch.uint8)
        for b in range(B):
            cv = WL.make_hidden(case_a["W"], K, N, 510 + b, WL.u_profile(N, 0.5, 3.0),
                                  WL.calibrated_sigma(V, d, 0.08, 3.0), flip_frac=0.1)
            hidden[:, b] = cv.hidden
            masks[b] = WL.uniform_fraction_mask(N, [1.0, 0.6, 0.3][b], 520 + b)
        outs = runner.step_batched(hidden, masks, [0.9, 0.85, 0.9], [1.0, 2.0, 0.5])
        for b in range(B):
            ref = O.rpd_step(bits(hidden[:, b]), masks[b].numpy(), bits(case_a["g"]),
                             bits(case_a["W"]), 1e-6, [0.9, 0.85, 0.9][b], [1.0, 2.0, 0.5][b], "llada")
            compare_step(ref, outs[b])
        # short canvas again on the grown scratch
        got = runner.step(case_a["hidden"], case_a["mask"], 0.9, 1.0)
        compare_step(oracle_step(case_a), got)
        # a new head of the same shape, then the Dream rule
        W2d, g2d = W2.to(runner.dev).contiguous(), g2.to(runner.dev).contiguous()
        runner.ctx.set_head(W2d, g2d)
        cv = WL.make_hidden(W2, K, 50, 530, WL.u_profile(50, 0.5, 3.0),
                            WL.calibrated_sigma(V, d, 0.08, 3.0), flip_frac=0.1)
        case_b = dict(case_a, W=W2, g=g2, hidden=cv.hidden)
        got = runner.step(case_b["hidden"], case_b["mask"], 0.9, 1.0)
        compare_step(oracle_step(case_b), got)
        runner.set_rule("dream")
        got = runner.step(case_b["hidden"], case_b["mask"], 0.85, 2.0)
        compare_step(oracle_step(case_b, tau=0.85, budget=2.0, rule="dream"), got)
    finally:
        runner.close()


def test_two_contexts_on_two_host_threads():
    """Two contexts, each driven by its own host thread on its own stream, step concurrently
    (their kernels share the GPU); every step's outputs equal the same step run alone."""
    import threading
    import paper_2609_36452_gb300 as rpd
    dev = torch.device("cuda:0")
    cases = [small_case(91, K=4, N=256, d=1024, V=8192), small_case(92, K=3, N=200, d=512, V=6000)]

    def run(case, stream, out, reps):
        ctx = rpd.Rpd(case["d"], case["V"], case["K"])
        try:
            ctx.set_head(case["Wd"], case["gd"])
            ctx.set_profile("llada")
            ctx.set_stream(stream)
            ctx.reserve(1, case["N"])
            for _ in range(reps):
                with torch.cuda.stream(stream):
                    m = case["maskd"].clone()
                    c = torch.zeros(case["N"], dtype=torch.uint8, device=dev)
                    t = torch.full((case["N"],), -1, dtype=torch.int32, device=dev)
                    s = torch.zeros(rpd.STATS_WORDS, dtype=torch.int32, device=dev)
                ctx.step(case["hd"], m, 0.9, 1.0, c, t, s)
                stream.synchronize()
                out.append((m.cpu(), c.cpu(), t.cpu(), s.cpu()))
        finally:
            ctx.close()

    for case in cases:
        case["Wd"], case["gd"] = case["W"].to(dev), case["g"].to(dev)
        case["hd"], case["maskd"] = case["hidden"].to(dev), case["mask"].to(dev)
    alone = []
    for case in cases:
        res = []
        run(case, torch.cuda.Stream(dev), res, 1)
        alone.append(res[0])
    together = [[], []]
    threads = [threading.Thread(target=run, args=(cases[i], torch.cuda.Stream(dev), together[i], 6))
               for i in range(2)]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    for i in range(2):
        assert len(together[i]) == 6
        for res in together[i]:
            for a, b in zip(res, alone[i]):
                assert torch.equal(a, b)


def test_all_zero_hidden_rows_give_uniform_predictions():
    """A hidden row of zeros (eps > 0) normalises to zeros, so every logit is 0: the
    prediction is uniform - c = 1/V, H = ln V, argmax the lowest token (index 0) on every
    layer - and such positions are never candidates.  The other positions are unaffected."""
    K, N, d, V = 3, 40, 256, 4100
    case = small_case(71, K=K, N=N, d=d, V=V)
    zero = [0, 7, 8, 39]
    case["hidden"][:, zero] = 0
    ref, got, rep = run_and_compare(case)
    for i in zero:
        assert np.all(got["layer_argmax"][:, i] == 0)
        assert abs(got["conf"][i] - 1.0 / V) < 1e-7
        assert abs(got["entropy"][i] - math.log(V)) < 2e-3
        assert got["candidate"][i] == 0
    print(rep)


# ------------------------------------------------------------------ window and canvas limits

@pytest.mark.parametrize("K,N,rule", [(16, 96, "llada"), (14, 96, "dream"), (64, 40, "llada")])
def test_paper_windows_and_largest_window(K, N, rule):
    """The windows the paper projects (the last 16 layers of LLaDA, the last 14 of Dream;
    App. A.6) and the largest the library accepts (K = 64).  A flat layer ramp keeps the
    argmax through many layers, so persistence reaches k_max and stability admissions occur."""
    case = small_case(5 + K + N, K=K, N=N, d=256, V=1024, a=torch.ones(K), rule=rule)
    ref, got, rep = run_and_compare(case)
    assert np.max(got["persist"][ref.masked]) >= 6
    print(rep)


def test_largest_canvas():
    """One canvas of N = 8192 positions (the largest accepted), half of them masked: the
    widest instantiation of the score/commit kernel.  N = 8193 is refused before any work."""
    case = small_case(8201, K=2, N=8192, d=256, V=1024, mask_frac=0.5)
    ref, got, rep = run_and_compare(case)
    assert got["stats"]["n_masked"] == int(case["mask"].sum())
    print(rep)
    import paper_2609_36452_gb300 as rpd
    dev = torch.device("cuda:0")
    ctx = rpd.Rpd(256, 1024, 2)
    try:
        ctx.set_head(case["W"].to(dev), case["g"].to(dev))
        n = 8193
        h = torch.zeros(2, n, 256, dtype=torch.bfloat16, device=dev)
        m = torch.ones(n, dtype=torch.uint8, device=dev)
        c = torch.full((n,), 7, dtype=torch.uint8, device=dev)
        t = torch.zeros(n, dtype=torch.int32, device=dev)
        s = torch.zeros(rpd.STATS_WORDS, dtype=torch.int32, device=dev)
        with pytest.raises(rpd.RpdError) as e:
            ctx.step(h, m, 0.9, 1.0, c, t, s)
        assert e.value.code == rpd.RPD_ERR_UNSUPPORTED
        torch.cuda.synchronize(dev)
        assert torch.all(c == 7) and torch.all(m == 1)
    finally:
        ctx.close()
