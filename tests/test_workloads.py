"""The seeded input generators: deterministic, right shapes and the stated structure."""
import math

import torch

import workloads as WL


def test_head_deterministic_and_shaped():
    W1, g1 = WL.make_head(100, 32, seed=5)
    W2, g2 = WL.make_head(100, 32, seed=5)
    assert W1.shape == (100, 32) and g1.shape == (32,)
    assert W1.dtype == torch.bfloat16 and torch.equal(W1, W2) and torch.equal(g1, g2)
    assert abs(W1.float().std().item() - 0.02) < 0.002


def test_u_profile_ends_and_middle():
    b = WL.u_profile(256, 0.3, 4.0)
    assert abs(b[0].item() - 4.0) < 1e-6 and abs(b[-1].item() - 4.0) < 1e-6
    assert b.min().item() >= 0.3 - 1e-6 and b[127].item() < 0.31


def test_hidden_flip_count_and_layers():
    W, _ = WL.make_head(500, 64, seed=1)
    cv = WL.make_hidden(W, K=4, N=50, seed=2, b=WL.u_profile(50, 0.5, 3), sigma=8.0, flip_frac=0.1)
    assert cv.hidden.shape == (4, 50, 64)
    flipped = cv.flip_targets >= 0
    assert int(flipped.sum()) == 5
    assert torch.all(cv.flip_targets[flipped] != cv.targets[flipped])


def test_masks():
    m = WL.uniform_fraction_mask(1024, 0.3, seed=3)
    assert int(m.sum()) == round(0.3 * 1024)
    f = WL.front_loaded_mask(512, seed=4)
    # the back of the canvas is masked more often than the front
    assert f[:128].float().mean() < f[-128:].float().mean()


def test_trajectory_profile_rises_with_committed_prefix():
    base = torch.ones(8)
    mask = torch.tensor([0, 0, 0, 0, 1, 1, 1, 1], dtype=torch.uint8)
    b = WL.trajectory_profile(base, mask, b_hi=4.0, gamma=2.0)
    assert math.isclose(b[0].item(), 4.0)                      # nothing to its left
    assert math.isclose(b[4].item(), 4.0)                      # whole prefix committed
    assert math.isclose(b[7].item(), 1 + 3 * (4 / 7) ** 2, rel_tol=1e-6)
