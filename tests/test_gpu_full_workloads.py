"""Full-size workloads that the fp64 oracle cannot evaluate row for row in seconds.

* Batched serving: 8 canvases x 1024 positions, K = 6, LLaDA-8B head, 30-100% masked
  (~32k projected rows).  Two whole canvases (about 5k rows each) are compared with the whole
  oracle step, output by output; sampled positions of every canvas, and the positions of the
  rows on both sides of every L2-band boundary of the head kernel's work walk, are projected
  by the oracle and compared score by score; the commitment of every canvas is also checked
  by replaying the oracle's rule on the GPU's own scores.
* Decode trajectory at the LLaDA-8B head shape: at every step the invariants, the commit
  rule replayed on the GPU's scores, the same commits with the projection chosen per step on
  the device, and the whole oracle step (every projected row, the commit set) compared
  output by output.
"""

import numpy as np
import pytest
import torch

import workloads as WL
from oracle import rpd_oracle as O
from tests.gpu_util import DeviceRunner, bits
from tests.oracle_pool import oracle_steps
from tests.parity import DELTA, compare_rows, compare_step, replay_commit_rule

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, never run there
    pytest.skip("needs a CUDA GPU", allow_module_level=True)


def oracle_rows(hidden_rows, g, W, eps):
    """Oracle readout of several positions' K rows (``hidden_rows`` [P][K][d]): per position
    argmax, pmax, gap, p(y) per layer and the final entropy; one projection for all rows."""
    P_, K, d = hidden_rows.shape
    z = O.project_logits(bits(hidden_rows.reshape(P_ * K, d)), bits(g), bits(W), eps)
    out = []
    for j in range(P_):
        P, a, pm, gap = O.readout_rows(z[j * K:(j + 1) * K])
        y = int(a[-1])
        out.append((a, pm, gap, P[:, y], float(O.entropy(P[-1]))))
    return out


def test_batched_serving_full():
    case = WL.batched_serving(seed=5)
    K, B, N = case["K"], case["B"], case["N"]
    runner = DeviceRunner(case["W"], case["g"], K, case["eps"], rule="llada")
    try:
        outs = runner.step_batched(case["hidden"], case["mask"], case["tau"], case["budget"])
    finally:
        runner.close()
    rule = O.RULES["llada"]
    gen = np.random.default_rng(55)
    samples = {}
    for b in range(B):
        idx = np.nonzero(case["mask"][b].numpy())[0]
        samples[b] = [int(i) for i in gen.choice(idx, size=min(3, len(idx)), replace=False)]
    # Rows on both sides of every boundary between L2 bands of the head kernel's work walk
    # (rows are layer-major over the canvases' masked positions in order; a band covers
    # 16 tiles of 256 rows), and the positions they belong to.
    order = [(b, int(i)) for b in range(B) for i in np.nonzero(case["mask"][b].numpy())[0]]
    nmt = len(order)
    R = K * nmt
    for r in [x for j in range(1, R // 4096 + 1) for x in (4096 * j - 1, 4096 * j) if x < R]:
        b, i = order[r % nmt]
        if i not in samples[b]:
            samples[b].append(i)
    picks = [(b, i) for b in range(B) for i in samples[b]]
    rows = torch.stack([case["hidden"][:, b, i] for b, i in picks])    # [P][K][d]
    readouts = dict(zip(picks, oracle_rows(rows, case["g"], case["W"], case["eps"])))
    for b in range(B):
        got = outs[b]
        masked = case["mask"][b].numpy().astype(bool)
        st = got["stats"]
        assert st["status"] == 0 and st["n_masked"] == int(masked.sum())
        # commitment replayed on the GPU's own scores
        exp, cand, near = replay_commit_rule(got, masked, case["tau"][b], case["budget"][b], rule, K)
        gcand = got["candidate"].astype(bool)
        for i in np.nonzero(masked)[0]:
            if i not in near:
                assert gcand[i] == cand[i], (b, i)
        diff = np.nonzero(exp != got["commit"])[0]
        if near:
            # a decision within DELTA of its threshold may flip; everything before it may not
            assert np.all(diff >= min(near)), (b, diff[:10], sorted(near)[:5])
        else:
            assert len(diff) == 0, (b, diff[:10])
        assert np.array_equal(got["new_mask"], (masked & (got["commit"] == 0)).astype(np.uint8))
        assert st["n_committed"] == int(got["commit"].sum()) >= 1
        # sampled positions against the oracle
        ref_rows = {i: readouts[(b, i)] for i in samples[b]}
        compare_rows(ref_rows, got, samples[b], K)
    # Whole canvases against the whole oracle step: every projected row of the canvas and its
    # commit set (the canvases are independent, so the oracle runs each on its own).
    counts = [int(case["mask"][b].sum()) for b in range(B)]
    whole = sorted(range(B), key=lambda b: abs(counts[b] - 850))[:2]
    tasks = [(bits(case["hidden"][:, b]), case["mask"][b].numpy(), case["eps"], case["tau"][b],
              case["budget"][b], "llada") for b in whole]
    for b, ref in zip(whole, oracle_steps(case["V"], case["d"], 5, tasks)):
        rep = compare_step(ref, outs[b])
        print(f"canvas {b}: {K * counts[b]} rows against the whole oracle step: {rep}")


@pytest.fixture(scope="module")
def traj_head():
    return WL.make_head(WL.LLADA_V, WL.LLADA_D, seed=4)


def test_llada_trajectory(traj_head):
    W, g = traj_head
    K, N, V = 4, 256, WL.LLADA_V
    gen = torch.Generator().manual_seed(4004)
    targets = torch.randint(0, V, (N,), generator=gen)
    runner = DeviceRunner(W, g, K, 1e-6, rule="llada")
    auto = DeviceRunner(W, g, K, 1e-6, rule="llada")     # projection chosen per step
    auto.ctx.set_projection("auto")
    mask = torch.ones(N, dtype=torch.uint8)
    checked = []
    steps = []
    lazy_steps = 0
    try:
        for t in range(64):
            cv = WL.trajectory_hidden(W, K, N, seed=4, step=t, mask=mask, targets=targets)
            got = runner.step(cv.hidden, mask, 0.9, 1.0)
            a = auto.step(cv.hidden, mask, 0.9, 1.0)
            assert np.array_equal(a["commit"], got["commit"]) and np.array_equal(a["new_mask"], got["new_mask"])
            sel = got["commit"] == 1
            assert np.array_equal(a["token"][sel], got["token"][sel])
            lazy_steps += a["stats"]["n_rows"] < got["stats"]["n_rows"]
            m = mask.numpy().astype(bool)
            st = got["stats"]
            assert st["status"] == 0 and st["n_masked"] == int(m.sum())
            assert st["n_committed"] >= 1 and np.all(got["commit"][~m] == 0)
            assert np.array_equal(got["new_mask"], (m & (got["commit"] == 0)).astype(np.uint8))
            steps.append((cv, mask.clone(), got))
            mask = torch.from_numpy(got["new_mask"].copy())
            if int(mask.sum()) <= 0.02 * N:
                break
    finally:
        runner.close()
        auto.close()
    assert int(mask.sum()) <= 0.02 * N, "trajectory did not finish within 64 steps"
    assert 0 < lazy_steps < len(steps), (lazy_steps, len(steps))   # both choices were taken
    # every step: the commit rule replayed on the GPU's own scores, and two sampled masked
    # positions projected by the oracle (one fp64 projection for all sampled rows)
    rule = O.RULES["llada"]
    pick = np.random.default_rng(404)
    samples = []
    for t, (cv, m, got) in enumerate(steps):
        masked = m.numpy().astype(bool)
        exp, cand, near = replay_commit_rule(got, masked, 0.9, 1.0, rule, K)
        diff = np.nonzero(exp != got["commit"])[0]
        if near:
            assert np.all(diff >= min(near)), (t, diff[:10], sorted(near)[:5])
        else:
            assert len(diff) == 0, (t, diff[:10])
        idx = np.nonzero(masked)[0]
        samples += [(t, int(i)) for i in pick.choice(idx, size=min(2, len(idx)), replace=False)]
    rows = torch.stack([steps[t][0].hidden[:, i] for t, i in samples])     # [P][K][d]
    readouts = dict(zip(samples, oracle_rows(rows, g, W, 1e-6)))
    for t, (cv, m, got) in enumerate(steps):
        mine = [i for tt, i in samples if tt == t]
        compare_rows({i: readouts[(t, i)] for i in mine}, got, mine, K)
    # the whole oracle step at every step of the trajectory (worker processes; each draws the
    # same head from its seed)
    tasks = [(bits(cv.hidden), m.numpy(), 1e-6, 0.9, 1.0, "llada") for cv, m, got in steps]
    refs = oracle_steps(V, WL.LLADA_D, 4, tasks)
    for t, ((cv, m, got), ref) in enumerate(zip(steps, refs)):
        rep = compare_step(ref, got)
        checked.append((t, rep.n_masked, len(rep.near_threshold)))
    print("trajectory steps", len(steps), "oracle-checked (step, masked, near-threshold)", checked)
