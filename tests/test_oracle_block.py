"""Pins of the RPD-block oracle (the block variant of §3.2 and App. A.6)."""
import json
import math
import os

import numpy as np

from oracle import rpd_oracle as O
from tests.test_oracle_pins import _tiny_inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_block_variant_omits_the_budget_on_the_fig3_case():
    """Same hand-built Fig. 3 table: full RPD holds C back on the entropy budget; RPD-block
    (all six positions in one block) commits every candidate, A, B and C."""
    f = json.load(open(os.path.join(GOLDEN, "fig3_narrative.json")))
    commit, cand, fb = O.block_step_from_scores(f["mask"], f["layer_argmax"], f["layer_p_of_y"],
                                                f["tau"], f["rule"], block=8)
    assert list(cand.astype(int)) == f["expected"]["candidate"]
    assert list(commit.astype(int)) == [1, 0, 1, 0, 0, 1]
    assert fb == -1


def test_active_block_is_first_block_with_a_masked_position():
    m = np.zeros(100, dtype=bool)
    m[[40, 41, 63, 64, 90]] = True
    assert list(O.active_block(m, 32)) == [40, 41, 63]
    assert list(O.active_block(m, 10)) == [40, 41]
    assert len(O.active_block(np.zeros(5, dtype=bool), 32)) == 0


def test_block_fallback_is_most_confident_in_active_block():
    K, N = 2, 12
    masked = np.zeros(N, dtype=bool)
    masked[[5, 6, 7, 9]] = True
    argmax = np.zeros((K, N), dtype=int)
    p = np.full((K, N), 0.1)
    p[:, 7] = 0.3            # most confident inside the first block of 8 (positions 0-7)
    p[:, 9] = 0.5            # more confident, but in the next block
    commit, cand, fb = O.block_step_from_scores(masked, argmax, p, 0.9, "llada", block=8)
    assert fb == 7 and list(np.nonzero(commit)[0]) == [7]
    p[:, 6] = 0.3            # tie: leftmost wins
    commit, cand, fb = O.block_step_from_scores(masked, argmax, p, 0.9, "llada", block=8)
    assert fb == 6


def test_block_equals_full_rule_restricted_to_active_block_with_infinite_budget():
    """RPD-block = full RPD with beta = inf (every candidate passes) and a fallback window
    covering the block, applied to the canvas with everything outside the active block
    treated as unmasked."""
    for seed in range(8):
        h, mask, gain, W = _tiny_inputs(100 + seed, N=40)
        for block in (8, 16, 32):
            r_blk = O.rpd_block_step(h, mask, gain, W, 1e-6, 0.9, "llada", block=block)
            act = O.active_block(mask.astype(bool), block)
            restricted = np.zeros_like(mask)
            restricted[act] = 1
            rule = dict(O.RULES["llada"], window=block)
            r_full = O.rpd_step(h, restricted, gain, W, 1e-6, 0.9, math.inf, rule)
            assert np.array_equal(r_blk.commit, r_full.commit), (seed, block)
            assert np.all(r_blk.commit[~np.isin(np.arange(len(mask)), act)] == 0)
            if mask.any():
                assert r_blk.commit.sum() >= 1
