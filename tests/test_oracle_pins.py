"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each test names what it is pinned to: a library routine, a closed form, an invariant the
paper states, the numbers Table 4 and App. A.6 print, a hand-built table realising the
Fig. 3 narrative, or brute force over every subset on tiny inputs.
"""
import itertools
import json
import math
import os

import numpy as np
import scipy.special
import scipy.stats
import torch
import torch.nn.functional as F

from oracle import rpd_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


# ----------------------------------------------------------------------------- bf16 storage

def test_bf16_decode_matches_torch():
    """bf16 bits -> value agrees with torch's own bf16 -> float64 conversion."""
    g = torch.Generator().manual_seed(0)
    t = (torch.randn(4096, generator=g) * 10).to(torch.bfloat16)
    ours = O.bf16_to_f64(bf16_bits(t))
    ref = t.to(torch.float64).numpy()
    assert np.array_equal(ours, ref)


def test_bf16_rne_matches_torch_on_products():
    """Rounding a product of two bf16 values agrees with torch's bf16 RNE conversion,
    including exact halfway cases (ties go to even)."""
    g = torch.Generator().manual_seed(1)
    a = (1 + 0.1 * torch.randn(20000, generator=g)).to(torch.bfloat16)
    b = torch.randn(20000, generator=g).to(torch.bfloat16)
    prod = a.to(torch.float64) * b.to(torch.float64)
    ours = O.f64_to_bf16_rne(prod.numpy())
    ref = bf16_bits(prod.to(torch.bfloat16))
    assert np.array_equal(ours, ref)
    # halfway cases: 1 + 2^-8 lies exactly between two bf16 neighbours (1 and 1 + 2^-7)
    halves = np.array([1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, -(1 + 2.0 ** -8)])
    ours = O.bf16_to_f64(O.f64_to_bf16_rne(halves))
    assert list(ours) == [1.0, 1 + 2 * 2.0 ** -7, -1.0]


# ----------------------------------------------------------------------------- projection

def _rand_head(V, d, seed, std=0.05):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(V, d, generator=g) * std).to(torch.bfloat16)


def test_projection_equals_torch_rmsnorm_linear_when_gain_is_exact():
    """With power-of-two gains, bf16(g*h) = g*h exactly, so reading D1 reduces to the
    textbook RMSNorm followed by the head: torch rms_norm + linear in fp64."""
    V, d, R = 97, 48, 7
    W = _rand_head(V, d, 2)
    gen = torch.Generator().manual_seed(3)
    h = (torch.randn(R, d, generator=gen) * 2).to(torch.bfloat16)
    gain = torch.tensor([0.5, 1.0, 2.0, 4.0] * (d // 4), dtype=torch.bfloat16)
    eps = 1e-6
    z = O.project_logits(bf16_bits(h), bf16_bits(gain), bf16_bits(W), eps)
    ref = F.linear(F.rms_norm(h.double(), (d,), gain.double(), eps), W.double()).numpy()
    np.testing.assert_allclose(z, ref, rtol=1e-12, atol=1e-12)


def test_unrounded_reading_equals_torch_rmsnorm_linear():
    """Reading D3 (diagnostic) is the textbook RMSNorm with a general gain followed by the
    head: torch rms_norm + linear in fp64.  With power-of-two gains it equals reading D1."""
    V, d, R = 89, 56, 6
    W = _rand_head(V, d, 12)
    gen = torch.Generator().manual_seed(13)
    h = (torch.randn(R, d, generator=gen) * 3).to(torch.bfloat16)
    gain = (1 + 0.1 * torch.randn(d, generator=gen)).to(torch.bfloat16)
    eps = 1e-5
    z3 = O.project_logits_exact(bf16_bits(h), bf16_bits(gain), bf16_bits(W), eps)
    ref = F.linear(F.rms_norm(h.double(), (d,), gain.double(), eps), W.double()).numpy()
    np.testing.assert_allclose(z3, ref, rtol=1e-12, atol=1e-12)
    exact = torch.tensor([0.5, 1.0, 2.0, 4.0] * (d // 4), dtype=torch.bfloat16)
    gap = O.reading_gap(bf16_bits(h), bf16_bits(exact), bf16_bits(W), eps)
    assert gap["max_abs_dp"] == 0.0 and gap["argmax_differs"] == 0
    gap = O.reading_gap(bf16_bits(h), bf16_bits(gain), bf16_bits(W), eps)
    assert 0.0 < gap["max_abs_dp"] < 1e-2 and gap["rows"] == R


def test_norm_operand_rounding_matches_torch():
    """For general gains the head operand is the bf16 RNE of g*h (torch's conversion)."""
    d, R = 64, 9
    gen = torch.Generator().manual_seed(4)
    h = torch.randn(R, d, generator=gen).to(torch.bfloat16)
    gain = (1 + 0.1 * torch.randn(d, generator=gen)).to(torch.bfloat16)
    u = O.norm_operand(bf16_bits(h), bf16_bits(gain))
    ref = bf16_bits((gain.double() * h.double()).to(torch.bfloat16))
    assert np.array_equal(u, ref)


def test_projection_row_orientation_brute_force():
    """Tiny case evaluated element by element with plain Python loops: z[r][v] sums over d
    the product of row r's operand and token v's head row, times row r's RMS factor."""
    V, d, R = 5, 8, 3
    W = _rand_head(V, d, 5, std=0.3)
    gen = torch.Generator().manual_seed(6)
    h = torch.randn(R, d, generator=gen).to(torch.bfloat16)
    gain = (1 + 0.2 * torch.randn(d, generator=gen)).to(torch.bfloat16)
    eps = 1e-5
    z = O.project_logits(bf16_bits(h), bf16_bits(gain), bf16_bits(W), eps)
    hv, gv, Wv = h.double().tolist(), gain.double().tolist(), W.double().tolist()
    for r in range(R):
        ms = sum(x * x for x in hv[r]) / d
        rho = 1.0 / math.sqrt(ms + eps)
        ur = [float(torch.tensor(gv[k] * hv[r][k], dtype=torch.float64).to(torch.bfloat16))
              for k in range(d)]
        for v in range(V):
            acc = sum(ur[k] * Wv[v][k] for k in range(d))
            assert abs(z[r, v] - rho * acc) <= 1e-12 * max(1.0, abs(rho * acc))


def test_projection_scale_invariance():
    """Scaling h by a power of two leaves the logits bit-identical when eps = 0 (RMSNorm is
    scale free); a wrong exponent on the RMS factor breaks this."""
    V, d, R = 33, 32, 4
    W = _rand_head(V, d, 7)
    gen = torch.Generator().manual_seed(8)
    h = torch.randn(R, d, generator=gen).to(torch.bfloat16)
    gain = (1 + 0.1 * torch.randn(d, generator=gen)).to(torch.bfloat16)
    z1 = O.project_logits(bf16_bits(h), bf16_bits(gain), bf16_bits(W), 0.0)
    z2 = O.project_logits(bf16_bits(h * 8), bf16_bits(gain), bf16_bits(W), 0.0)
    assert np.array_equal(z1, z2)


def test_zero_hidden_gives_uniform():
    """h = 0: the logits vanish, the distribution is uniform, H = ln V, c = 1/V, y = 0."""
    V, d = 50, 16
    W = _rand_head(V, d, 9)
    h = torch.zeros(1, d, dtype=torch.bfloat16)
    gain = torch.ones(d, dtype=torch.bfloat16)
    z = O.project_logits(bf16_bits(h), bf16_bits(gain), bf16_bits(W), 1e-6)
    P, a, pmax, gap = O.readout_rows(z)
    assert a[0] == 0 and gap[0] == 0.0
    assert abs(pmax[0] - 1.0 / V) < 1e-15
    assert abs(O.entropy(P[0]) - math.log(V)) < 1e-12


# ----------------------------------------------------------------------------- readout (Eq. 1)

def test_uniform_logits_closed_form():
    for V in (2, 7, 4096):
        z = np.full(V, 3.25)
        p = O.softmax(z)
        assert abs(O.entropy(p) - math.log(V)) < 1e-12
        assert O.argmax_lowest(z) == 0
        assert abs(p[0] - 1.0 / V) < 1e-15


def test_two_level_closed_form():
    """Logits {x at one token, 0 elsewhere}: p = e^x/(e^x+V-1) and
    H = ln(e^x + V - 1) - x e^x / (e^x + V - 1)."""
    for V, x, j in [(16, 2.0, 5), (4096, 9.5, 4095), (126464, 14.0, 77)]:
        z = np.zeros(V)
        z[j] = x
        p = O.softmax(z)
        Z = math.exp(x) + V - 1
        assert abs(p[j] - math.exp(x) / Z) < 1e-14
        H_closed = math.log(Z) - x * math.exp(x) / Z
        assert abs(O.entropy(p) - H_closed) < 1e-11
        assert O.argmax_lowest(z) == j
        assert abs(O.top2_gap(z) - x) < 1e-15


def test_readout_matches_scipy():
    rng = np.random.default_rng(10)
    for V in (3, 100, 5000):
        z = rng.normal(0, 3, size=(4, V))
        p = O.softmax(z)
        np.testing.assert_allclose(p, scipy.special.softmax(z, axis=-1), rtol=1e-12, atol=0)
        np.testing.assert_allclose(O.entropy(p), scipy.stats.entropy(p, axis=-1), rtol=1e-12)
        assert np.all(O.entropy(p) >= 0) and np.all(O.entropy(p) <= math.log(V) + 1e-12)


def test_argmax_ties_lowest_and_gap():
    z = np.array([1.0, 5.0, 2.0, 5.0, -1.0])
    assert O.argmax_lowest(z) == 1
    assert O.top2_gap(z) == 0.0
    assert O.top2_gap(np.array([0.0, 3.0, 2.5])) == 0.5


def test_one_hot_entropy_zero():
    z = np.array([0.0, 800.0, 0.0])  # exp underflows to exactly 0 for the others
    p = O.softmax(z)
    assert p[1] == 1.0 and O.entropy(p) == 0.0


# ----------------------------------------------------------------------------- Eq. 2-5

def test_persistence_backward_scan():
    assert O.persistence([4, 4, 4, 4]) == 4
    assert O.persistence([9, 4, 4, 4]) == 3
    # an earlier match separated by a disagreement is excluded (App. A.2)
    assert O.persistence([4, 9, 4, 4]) == 2
    assert O.persistence([4, 4, 4, 9]) == 1
    assert O.persistence([7]) == 1


def test_confidence_drop():
    p = [0.5, 0.9, 0.7, 0.6]
    assert abs(O.confidence_drop(p, 3) - 0.3) < 1e-15
    assert abs(O.confidence_drop(p, 2) - 0.1) < 1e-15
    assert O.confidence_drop(p, 1) == 0.0
    rng = np.random.default_rng(11)
    for _ in range(200):
        q = rng.random(6)
        k = int(rng.integers(1, 7))
        assert O.confidence_drop(q, k) >= 0.0


def test_table4_ceiling_matches_printed_values():
    """App. A.6: with K_max = 6 the stability route tolerates r <= (6 - theta_s)/w, printed as
    0.167 (LLaDA) and 0.175 (Dream).  The oracle's rule must admit just inside the ceiling
    and reject just outside it, for any persistence at or above the cap."""
    t4 = json.load(open(os.path.join(GOLDEN, "table4_hparams.json")))
    for name in ("llada", "dream"):
        rule = O.RULES[name]
        assert rule["theta_s"] == t4[name]["theta_s"] and rule["w"] == t4[name]["w"]
        assert rule["theta_c"] == t4["theta_c"] and rule["k_max"] == t4["k_max"]
        assert rule["window"] == t4["window"]
        ceiling = (rule["k_max"] - rule["theta_s"]) / rule["w"]
        assert round(ceiling, 3) == t4[name]["printed_ceiling"]
        for k_i in (6, 7, 16):
            for c in (0.6, 0.75, 0.899):
                s_in = O.stability(k_i, ceiling - 1e-9, rule["k_max"], rule["w"])
                s_out = O.stability(k_i, ceiling + 1e-9, rule["k_max"], rule["w"])
                assert O.is_candidate(c, s_in, t4["theta_h"], rule["theta_c"], rule["theta_s"])
                assert not O.is_candidate(c, s_out, t4["theta_h"], rule["theta_c"], rule["theta_s"])


def test_candidate_boundaries_and_ceiling_invariant():
    rule = O.RULES["llada"]
    th, tc, ts = 0.9, rule["theta_c"], rule["theta_s"]
    assert O.is_candidate(0.9, -100.0, th, tc, ts)        # c >= theta_h bypasses stability
    assert O.is_candidate(0.6, 3.5, th, tc, ts)           # both lower bounds inclusive
    assert not O.is_candidate(0.6 - 1e-12, 100.0, th, tc, ts)
    assert not O.is_candidate(0.7, 3.5 - 1e-12, th, tc, ts)
    rng = np.random.default_rng(12)
    for _ in range(2000):
        k_i = int(rng.integers(1, 17))
        r = float(rng.random() * 0.5)
        c = float(0.6 + 0.3 * rng.random())
        s = O.stability(k_i, r, rule["k_max"], rule["w"])
        if O.is_candidate(c, s, th, tc, ts):
            # stability-route admissions sit under (min(K_i,K_max) - theta_s)/w <= ceiling
            assert r <= (min(k_i, rule["k_max"]) - ts) / rule["w"] + 1e-12
            assert r <= (rule["k_max"] - ts) / rule["w"] + 1e-12 < 0.25


def test_fig3_narrative():
    """Hand-built realisation of Fig. 3: A, B, C are candidates; D (changing argmax) and E
    (large drop) are not; A and B commit together; C waits on the budget."""
    f = json.load(open(os.path.join(GOLDEN, "fig3_narrative.json")))
    A = np.array(f["layer_argmax"])
    P = np.array(f["layer_p_of_y"])
    ex = f["expected"]
    for i in range(A.shape[1]):
        k_i = O.persistence(A[:, i])
        assert k_i == ex["persistence"][i]
        assert abs(O.confidence_drop(P[:, i], k_i) - ex["drop"][i]) < 1e-12
    commit, cand, acc, fb = O.step_from_scores(f["mask"], A, P, f["H_final"], f["tau"],
                                               f["beta"], f["rule"])
    assert list(cand.astype(int)) == ex["candidate"]
    assert list(commit.astype(int)) == ex["commit"]
    assert fb == ex["fallback"]


# ----------------------------------------------------------------------------- §3.2 commitment

def _prefix_form(masked, cand, H, beta):
    """The closed form of the sequential rule: candidate i is committed iff the entropy of the
    masked non-candidates before it, Q_i, is <= beta (proof: H >= 0, so once one candidate
    is rejected every later one sees at least as much entropy)."""
    out = []
    q = 0.0
    for i in range(len(masked)):
        if cand[i] and q <= beta:
            out.append(i)
        if masked[i] and not cand[i]:
            q += H[i]
    return out


def test_sequential_equals_prefix_form_exhaustive():
    rng = np.random.default_rng(13)
    for n in range(0, 9):
        for mbits in itertools.product([0, 1], repeat=n):
            masked = np.array(mbits, dtype=bool)
            idx = np.nonzero(masked)[0]
            for cbits in itertools.product([0, 1], repeat=len(idx)):
                cand = np.zeros(n, dtype=bool)
                cand[idx[np.array(cbits, dtype=bool)]] = True
                H = rng.choice([0.0, 0.25, 0.5, 1.0, 3.0], size=n)
                for beta in (0.0, 0.5, 1.0, 2.0, math.inf):
                    seq = O.commit_sequential(masked, cand, H, beta)
                    assert seq == _prefix_form(masked, cand, H, beta)
                    assert seq == O.accepted_prefix(masked, cand, H, beta)


def test_commit_set_is_unique_fixed_point_brute_force():
    """Brute force over every subset S of C: S is the committed set iff each candidate i is in
    S exactly when the entropy of masked positions before i outside S is <= beta.  Exactly one
    subset satisfies this and it is the oracle's."""
    rng = np.random.default_rng(14)
    for trial in range(300):
        n = int(rng.integers(1, 9))
        masked = rng.random(n) < 0.8
        cand = masked & (rng.random(n) < 0.5)
        H = np.round(rng.random(n) * 2, 2)
        beta = float(rng.choice([0.0, 0.3, 1.0, 2.5]))
        C = list(np.nonzero(cand)[0])
        fixed = []
        for r in range(len(C) + 1):
            for S in itertools.combinations(C, r):
                S = set(S)
                ok = True
                for i in C:
                    e = sum(H[j] for j in range(i) if masked[j] and j not in S)
                    if (i in S) != (e <= beta):
                        ok = False
                        break
                if ok:
                    fixed.append(sorted(S))
        assert len(fixed) == 1
        assert [int(i) for i in fixed[0]] == [int(i) for i in O.commit_sequential(masked, cand, H, beta)]


def test_commit_special_cases():
    masked = np.array([1, 1, 0, 1, 1, 1], dtype=bool)
    cand = np.array([0, 1, 0, 0, 1, 1], dtype=bool)
    H = np.array([5.0, 1.0, 9.0, 0.0, 2.0, 1.0])
    assert O.commit_sequential(masked, cand, H, math.inf) == [1, 4, 5]     # beta = inf: A = C
    assert O.commit_sequential(masked, cand, H, 4.99) == []                 # position 0 blocks all
    assert O.commit_sequential(masked, cand, H, 5.0) == [1, 4, 5]           # E <= beta inclusive
    # unmasked entropy is never counted; accepted candidates are excluded from later sums
    m2 = np.array([0, 1, 1], dtype=bool)
    c2 = np.array([0, 1, 1], dtype=bool)
    assert O.commit_sequential(m2, c2, np.array([100.0, 50.0, 0.0]), 0.0) == [1, 2]


def test_fallback_rule():
    masked = np.array([0, 1, 1, 0, 1, 1], dtype=bool)
    c = np.array([0.99, 0.2, 0.5, 0.99, 0.5, 0.9])
    assert O.fallback_commit(masked, c, 32) == 5
    assert O.fallback_commit(masked, c, 3) == 2         # window = first 3 *masked* positions
    assert O.fallback_commit(masked, c, 1) == 1
    assert O.fallback_commit(np.zeros(4, dtype=bool), c[:4], 32) == -1


# ----------------------------------------------------------------------------- full step

def _tiny_inputs(seed, K=3, N=24, d=32, V=64, w_std=0.5, sig=4.0):
    gen = torch.Generator().manual_seed(seed)
    W = (torch.randn(V, d, generator=gen) * w_std).to(torch.bfloat16)
    gain = (1 + 0.1 * torch.randn(d, generator=gen)).to(torch.bfloat16)
    t = torch.randint(0, V, (N,), generator=gen)
    dirs = W[t].float()
    dirs = dirs / dirs.norm(dim=1, keepdim=True)
    b = torch.rand(N, generator=gen) * sig
    h = torch.stack([(0.6 + 0.4 * k / max(K - 1, 1)) * b[:, None] * dirs * math.sqrt(d)
                     + torch.randn(N, d, generator=gen) for k in range(K)]).to(torch.bfloat16)
    mask = (torch.rand(N, generator=gen) < 0.8).to(torch.uint8)
    return bf16_bits(h), mask.numpy(), bf16_bits(gain), bf16_bits(W)


def test_full_step_invariants():
    for seed in range(6):
        h, mask, gain, W = _tiny_inputs(seed)
        K, N, d = h.shape
        V = W.shape[0]
        r = O.rpd_step(h, mask, gain, W, 1e-6, 0.9, 1.0, "llada")
        m = mask.astype(bool)
        assert set(np.nonzero(r.commit)[0]) <= set(np.nonzero(r.cand)[0]) | {r.fallback_pos}
        assert set(r.accepted) <= set(np.nonzero(r.cand)[0])
        assert r.commit.sum() >= 1 if m.any() else r.commit.sum() == 0
        assert np.all(r.commit[~m] == 0)
        assert np.all((r.H[m] >= 0) & (r.H[m] <= math.log(V) + 1e-9))
        assert np.all((r.persist[m] >= 1) & (r.persist[m] <= K))
        assert np.all(r.drop[m] >= 0)
        assert np.all(r.token[r.commit == 1] == r.y[r.commit == 1])
        assert np.array_equal(r.new_mask, (m & (r.commit == 0)).astype(np.uint8))
        # p^(k)(y_i) at the suffix layers equals the layer max probability (App. A.2 argument)
        for i in np.nonzero(m)[0]:
            for k in range(K - r.persist[i], K):
                assert abs(r.p_of_y[k, i] - r.layer_pmax[k, i]) < 1e-15


def test_full_step_k1_window():
    """K = 1: persistence is 1 and the drop is 0 for every masked position."""
    h, mask, gain, W = _tiny_inputs(21, K=1)
    r = O.rpd_step(h, mask, gain, W, 1e-6, 0.9, 1.0, "llada")
    m = mask.astype(bool)
    assert np.all(r.persist[m] == 1) and np.all(r.drop[m] == 0)


def test_full_step_all_committed_when_thresholds_trivial():
    """theta_h below every confidence and beta = inf: every masked position commits."""
    h, mask, gain, W = _tiny_inputs(22)
    rule = dict(O.RULES["llada"])
    r = O.rpd_step(h, mask, gain, W, 1e-6, 1e-9, math.inf, rule)
    assert np.array_equal(r.commit, mask.astype(np.uint8))


def test_full_step_no_mask():
    h, mask, gain, W = _tiny_inputs(23)
    r = O.rpd_step(h, np.zeros_like(mask), gain, W, 1e-6, 0.9, 1.0, "llada")
    assert r.commit.sum() == 0 and r.fallback_pos == -1


def test_only_band_positions_need_earlier_layers():
    """Eq. 5: outside theta_c <= c < theta_h a position's candidacy does not depend on S_i,
    so the earlier window layers of such positions can be replaced by anything without
    changing the commit set (what lazy projection relies on, App. A.6)."""
    rng = np.random.default_rng(31)
    for seed in range(10):
        h, mask, gain, W = _tiny_inputs(200 + seed, K=4, N=30)
        r = O.rpd_step(h, mask, gain, W, 1e-6, 0.9, 1.0, "llada")
        band = r.masked & (r.conf >= 0.6) & (r.conf < 0.9)
        A = r.layer_argmax.copy()
        P = r.p_of_y.copy()
        for i in np.nonzero(r.masked & ~band)[0]:
            A[:-1, i] = rng.integers(0, 64, size=A.shape[0] - 1)
            P[:-1, i] = rng.random(A.shape[0] - 1)
        commit, cand, acc, fb = O.step_from_scores(r.masked, A, P, r.H, 0.9, 1.0, "llada")
        assert np.array_equal(commit, r.commit) and np.array_equal(cand, r.cand)
