"""The process pool that runs whole oracle steps for the full-size parity tests gives exactly
what calling the oracle in this process gives (no GPU needed)."""
import numpy as np

import workloads as WL
from oracle import rpd_oracle as O
from tests.gpu_util import bits
from tests.oracle_pool import oracle_steps


def test_pool_matches_direct_calls():
    V, d, K, N, seed = 700, 64, 3, 40, 77
    W, g = WL.make_head(V, d, seed, w_std=0.08)
    tasks, direct = [], []
    for s in range(3):
        cv = WL.make_hidden(W, K, N, 500 + s, WL.u_profile(N, 0.5, 3.0),
                            WL.calibrated_sigma(V, d, 0.08, 3.0), flip_frac=0.1)
        mask = WL.uniform_fraction_mask(N, 0.4 + 0.3 * s, 600 + s).numpy()
        tasks.append((bits(cv.hidden), mask, 1e-6, 0.9, 1.0, "llada"))
        direct.append(O.rpd_step(bits(cv.hidden), mask, bits(g), bits(W), 1e-6, 0.9, 1.0, "llada"))
    pooled = oracle_steps(V, d, seed, tasks, workers=2, w_std=0.08)
    for a, b in zip(direct, pooled):
        assert np.array_equal(a.commit, b.commit) and np.array_equal(a.token, b.token)
        np.testing.assert_array_equal(a.conf, b.conf)
        np.testing.assert_array_equal(a.H, b.H)
        np.testing.assert_array_equal(a.layer_argmax, b.layer_argmax)
