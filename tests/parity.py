"""Comparison of one GPU commit step with the CPU oracle.

Tolerances (stated once, used by every parity test):
  * probabilities (layer max probability, confidence) and entropies: 2e-3 absolute;
  * tokens, per-layer argmaxes, persistence and commit masks: exact, except where an
    oracle quantity lies within DELTA = 1e-4 of the threshold that decides it:
      - a top-2 logit gap below DELTA at a window layer (the argmax is a near tie),
      - |c - tau|, |c - theta_c| or (inside the stability band) |S - theta_s| below DELTA,
      - |Q_i - beta| below DELTA for the budget comparison,
      - for the fallback, confidences within a relative 1e-4 of the window's best.
    Because a flipped candidate flag moves Q for every later position, the GPU commit
    vector must equal one of the oracle's outcomes under some choice of those
    near-threshold decisions (the admissible set); the number of such decisions is
    reported.
"""
from __future__ import annotations

import itertools
from dataclasses import dataclass, field

import numpy as np

from oracle import rpd_oracle as O

DELTA = 1e-4
PROB_TOL = 2e-3
FALLBACK_REL = 1e-4
MAX_FREE = 12


@dataclass
class ParityReport:
    n_masked: int = 0
    near_threshold: list = field(default_factory=list)
    argmax_exempt: int = 0
    max_dconf: float = 0.0
    max_dH: float = 0.0
    max_dpmax: float = 0.0
    admissible: int = 0

    def __str__(self):
        return (f"masked={self.n_masked} near_threshold={len(self.near_threshold)} "
                f"argmax_exempt={self.argmax_exempt} max|dc|={self.max_dconf:.2e} "
                f"max|dH|={self.max_dH:.2e} max|dpmax|={self.max_dpmax:.2e} "
                f"admissible_outcomes={self.admissible}")


def _accept_sets(masked, cand, H, beta):
    """All accepted sets reachable when budget comparisons within DELTA may go either way."""
    N = len(masked)
    q = 0.0
    first_definite = N
    ambiguous = []
    for i in range(N):
        if cand[i]:
            if q > beta + DELTA:
                first_definite = i
                break
            if abs(q - beta) <= DELTA:
                ambiguous.append(i)
        if masked[i] and not cand[i]:
            q += H[i]
    C = [i for i in range(N) if cand[i]]
    outs = set()
    for cut in ambiguous + [first_definite]:
        if cut > first_definite:
            continue
        outs.add(tuple(i for i in C if i < cut))
    # also the reading where every ambiguous comparison passes
    outs.add(tuple(i for i in C if i < first_definite))
    return outs


def admissible_commits(ref: O.StepResult, free_positions):
    """Set of commit vectors (as tuples of indices) the oracle admits."""
    p = ref.params
    masked = ref.masked
    N = len(masked)
    free = list(free_positions)
    if len(free) > MAX_FREE:
        raise AssertionError(f"{len(free)} near-threshold decisions: parity unpinned for this case")
    results = set()
    for flips in itertools.product([False, True], repeat=len(free)):
        cand = ref.cand.copy()
        for f, pos in zip(flips, free):
            if f:
                cand[pos] = not cand[pos]
        for acc in _accept_sets(masked, cand, ref.H, p["budget"]):
            if acc:
                results.add(tuple(sorted(acc)))
            elif masked.any():
                window = [i for i in range(N) if masked[i]][:p["window"]]
                cbest = max(ref.conf[i] for i in window)
                for i in window:
                    if ref.conf[i] >= cbest * (1 - FALLBACK_REL):
                        results.add((i,))
            else:
                results.add(())
    return results


def near_threshold_positions(ref: O.StepResult):
    p = ref.params
    out = []
    for i in np.nonzero(ref.masked & np.isfinite(ref.conf))[0]:   # scored positions
        c, s = ref.conf[i], ref.stab[i]
        near = abs(c - p["tau"]) < DELTA or abs(c - p["theta_c"]) < DELTA
        if p["theta_c"] - DELTA <= c < p["tau"] + DELTA and abs(s - p["theta_s"]) < DELTA:
            near = True
        if np.nanmin(ref.layer_gap[:, i]) < DELTA:
            near = True
        if near:
            out.append(int(i))
    return out


def lazy_band(ref: O.StepResult):
    """Positions whose earlier window layers a lazy step projects (theta_c <= c < tau), and
    those within DELTA of the band's edges (either side may be taken)."""
    p = ref.params
    c = ref.conf
    m = ref.masked & np.isfinite(c)
    band = m & (c >= p["theta_c"]) & (c < p["tau"])
    edge = m & ((np.abs(c - p["theta_c"]) < DELTA) | (np.abs(c - p["tau"]) < DELTA))
    return band, edge


def compare_step(ref: O.StepResult, got: dict, check_scores: bool = True,
                 lazy: bool = False) -> ParityReport:
    """``got`` holds numpy arrays for one canvas: commit, token (after the step; only
    committed positions are compared), new_mask, stats (dict) and optionally conf,
    entropy, persist, drop, candidate, layer_argmax [K][N], layer_pmax [K][N].
    ``lazy``: the step projected earlier window layers only for band positions, so those
    layers (and K_i, r_i) are compared there only."""
    rep = ParityReport()
    m = ref.masked
    rep.n_masked = int(m.sum())
    free = near_threshold_positions(ref)
    rep.near_threshold = free
    free_set = set(free)
    K = ref.layer_argmax.shape[0]
    band, edge = lazy_band(ref) if lazy else (np.ones_like(m), np.zeros_like(m))

    if check_scores and "conf" in got:
        idx = np.nonzero(m)[0]
        if len(idx):
            rep.max_dconf = float(np.max(np.abs(got["conf"][idx] - ref.conf[idx])))
            rep.max_dH = float(np.max(np.abs(got["entropy"][idx] - ref.H[idx])))
            assert rep.max_dconf < PROB_TOL, f"confidence off by {rep.max_dconf}"
            assert rep.max_dH < PROB_TOL, f"entropy off by {rep.max_dH}"
        if "layer_argmax" in got:
            la, lp = got["layer_argmax"], got["layer_pmax"]
            for i in idx:
                for k in range(K):
                    if k < K - 1 and (not band[i] or edge[i]):
                        continue  # lazy: not projected outside the band
                    if ref.layer_gap[k, i] < DELTA:
                        rep.argmax_exempt += 1
                        continue
                    assert la[k, i] == ref.layer_argmax[k, i], (k, i, la[k, i], ref.layer_argmax[k, i])
                    rep.max_dpmax = max(rep.max_dpmax, abs(lp[k, i] - ref.layer_pmax[k, i]))
            assert rep.max_dpmax < PROB_TOL, f"layer max probability off by {rep.max_dpmax}"
        if "persist" in got:
            for i in idx:
                if np.nanmin(ref.layer_gap[:, i]) < DELTA or not band[i] or edge[i]:
                    continue
                assert got["persist"][i] == ref.persist[i], (i, got["persist"][i], ref.persist[i])
                assert abs(got["drop"][i] - ref.drop[i]) < 2 * PROB_TOL, (i, got["drop"][i], ref.drop[i])
        if "candidate" in got:
            for i in idx:
                if i in free_set:
                    continue
                assert bool(got["candidate"][i]) == bool(ref.cand[i]), (
                    i, ref.conf[i], ref.stab[i], ref.persist[i])
        # unmasked positions are never candidates
        if "candidate" in got:
            assert not np.any(got["candidate"][~m])

    commit = np.asarray(got["commit"]).astype(np.uint8)
    assert np.all(commit[~m] == 0), "committed an unmasked position"
    cset = tuple(int(i) for i in np.nonzero(commit)[0])
    adm = admissible_commits(ref, free)
    rep.admissible = len(adm)
    assert cset in adm, (f"commit set {cset} not among {len(adm)} admissible outcomes; "
                         f"oracle {tuple(np.nonzero(ref.commit)[0])}")
    tok = np.asarray(got["token"])
    for i in cset:
        if ref.layer_gap[K - 1, i] < DELTA:
            continue
        assert tok[i] == ref.y[i], (i, tok[i], ref.y[i])
    new_mask = np.asarray(got["new_mask"]).astype(np.uint8)
    assert np.array_equal(new_mask, (m & (commit == 0)).astype(np.uint8))
    st = got["stats"]
    assert st["status"] == 0, st
    assert st["n_masked"] == rep.n_masked
    assert st["n_committed"] == len(cset)
    assert (st["fallback_used"] == 1) == (st["fallback_pos"] >= 0)
    if st["fallback_used"]:
        assert cset == (st["fallback_pos"],)
    assert st["n_high_conf"] + st["n_stability"] + st["fallback_used"] == st["n_committed"]
    if not free:
        assert st["n_candidates"] == int(ref.cand.sum())
    return rep


def replay_commit_rule(got: dict, masked, tau: float, budget: float, rule: dict, K: int):
    """Apply the oracle's rule steps (Eq. 5, the sequential E_i <= beta rule and the fallback)
    to the GPU's own per-position scores, in fp64, and return (expected commit vector, the
    positions whose decision is within DELTA of a threshold).  This checks the scan, the
    acceptance and the fallback at any size, independently of the projection."""
    masked = np.asarray(masked).astype(bool)
    N = masked.shape[0]
    c = got["conf"].astype(np.float64)
    S = got["stability"].astype(np.float64)
    H = got["entropy"].astype(np.float64)
    cand = np.zeros(N, dtype=bool)
    near = []
    for i in np.nonzero(masked)[0]:
        cand[i] = O.is_candidate(c[i], S[i], tau, rule["theta_c"], rule["theta_s"])
        if (abs(c[i] - tau) < DELTA or abs(c[i] - rule["theta_c"]) < DELTA or
                (rule["theta_c"] <= c[i] < tau and abs(S[i] - rule["theta_s"]) < DELTA)):
            near.append(int(i))
    A = O.commit_sequential(masked, cand, H, budget)
    fb = -1
    if not A and masked.any():
        fb = O.fallback_commit(masked, c, rule["window"])
    commit = np.zeros(N, dtype=np.uint8)
    commit[A] = 1
    if fb >= 0:
        commit[fb] = 1
    # budget comparisons within DELTA
    q = 0.0
    for i in range(N):
        if cand[i] and abs(q - budget) < DELTA:
            near.append(int(i))
        if masked[i] and not cand[i]:
            q += H[i]
    return commit, cand, near


def compare_rows(ref_rows: dict, got: dict, positions, K: int):
    """Per-position scores of sampled positions against the oracle's readout of their K rows.
    ``ref_rows[i]`` = (argmax[K], pmax[K], gap[K], p_of_y[K], H_final)."""
    worst = 0.0
    for i in positions:
        a, pm, gap, pyk, Hf = ref_rows[i]
        near = np.min(gap) < DELTA
        for k in range(K):
            if gap[k] >= DELTA:
                assert got["layer_argmax"][k, i] == a[k], (i, k, got["layer_argmax"][k, i], a[k])
                worst = max(worst, abs(got["layer_pmax"][k, i] - pm[k]))
        assert abs(got["conf"][i] - pyk[-1]) < PROB_TOL
        assert abs(got["entropy"][i] - Hf) < PROB_TOL
        if not near:
            k_i = O.persistence(a)
            assert got["persist"][i] == k_i
            assert abs(got["drop"][i] - O.confidence_drop(pyk, k_i)) < 2 * PROB_TOL
    assert worst < PROB_TOL
    return worst


def compare_block_step(ref: O.StepResult, got: dict, lazy: bool = False) -> ParityReport:
    """RPD-block: scores of the active block's positions, and the commit set against every
    outcome the oracle admits under its near-threshold decisions (same tolerances as
    compare_step; no budget is involved).  ``lazy`` as in compare_step."""
    rep = ParityReport()
    band, edge = lazy_band(ref) if lazy else (np.ones_like(ref.masked), np.zeros_like(ref.masked))
    scored = np.isfinite(ref.conf)
    idx = np.nonzero(scored)[0]
    rep.n_masked = int(ref.masked.sum())
    K = ref.layer_argmax.shape[0]
    p = ref.params
    free = [i for i in near_threshold_positions(ref) if scored[i]]
    rep.near_threshold = free
    if len(idx):
        rep.max_dconf = float(np.max(np.abs(got["conf"][idx] - ref.conf[idx])))
        rep.max_dH = float(np.max(np.abs(got["entropy"][idx] - ref.H[idx])))
        assert rep.max_dconf < PROB_TOL and rep.max_dH < PROB_TOL
        for i in idx:
            for k in range(K):
                if k < K - 1 and (not band[i] or edge[i]):
                    continue  # lazy: not projected outside the band
                if ref.layer_gap[k, i] >= DELTA:
                    assert got["layer_argmax"][k, i] == ref.layer_argmax[k, i], (k, i)
            if i not in free:
                assert bool(got["candidate"][i]) == bool(ref.cand[i]), i
    # positions outside the active block are not scored and never committed
    outside = ref.masked & ~scored
    assert np.all(got["candidate"][outside] == 0) and np.all(got["commit"][outside] == 0)
    if len(free) > MAX_FREE:
        raise AssertionError("too many near-threshold decisions: parity unpinned for this case")
    adm = set()
    for flips in itertools.product([False, True], repeat=len(free)):
        cand = ref.cand.copy()
        for f, pos in zip(flips, free):
            if f:
                cand[pos] = not cand[pos]
        A = tuple(int(i) for i in idx if cand[i])
        if A:
            adm.add(A)
        elif len(idx):
            cbest = max(ref.conf[i] for i in idx)
            for i in idx:
                if ref.conf[i] >= cbest * (1 - FALLBACK_REL):
                    adm.add((int(i),))
        else:
            adm.add(())
    rep.admissible = len(adm)
    commit = np.asarray(got["commit"]).astype(np.uint8)
    cset = tuple(int(i) for i in np.nonzero(commit)[0])
    assert cset in adm, (cset, sorted(adm)[:5])
    for i in cset:
        if ref.layer_gap[K - 1, i] >= DELTA:
            assert got["token"][i] == ref.y[i]
    assert np.array_equal(got["new_mask"], (ref.masked & (commit == 0)).astype(np.uint8))
    st = got["stats"]
    assert st["status"] == 0 and st["n_masked"] == rep.n_masked
    assert st["n_committed"] == len(cset)
    assert st["n_high_conf"] + st["n_stability"] + st["fallback_used"] == st["n_committed"]
    return rep
