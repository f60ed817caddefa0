"""CPU oracle for the Reliable Parallel Decoding (RPD) commit step.

TEST INFRASTRUCTURE ONLY.  This module is the plain, slow, fp64 statement of what
one RPD commit step computes.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (its cpu_baseline leg and its ``--impl reference`` arm) may import it.
The library in ``paper_2609_36452_gb300`` never calls it and shares no code with it.

What one step computes (paper §3, Eq. 2-7, with the layerwise readout of App. A.2
and A.6):

1. For every masked position i and every layer of the window (the last K layers,
   l0 = L-K+1 .. L), project the hidden state through the final RMSNorm and the LM
   head (the "logit lens", §2.2, App. A.2) and take the softmax over the whole
   vocabulary.
2. Final-layer prediction y_i, confidence c_i = p^(L)(y_i) and entropy
   H_i = -sum_v p(v) ln p(v) (Eq. 1, natural log).
3. Prediction persistence K_i (Eq. 2, counted backward from the final layer and
   stopping at the first disagreement, App. A.2), confidence drop r_i (Eq. 3) and
   stability score S_i = min(K_i, K_max) - w r_i (Eq. 4).
4. Candidate set C_t (Eq. 5).
5. Sequential entropy-budget commitment A_t (the unnumbered E_i equation and
   A_t = {i in C_t : E_i <= beta}, §3.2), with the fallback commit when A_t is
   empty (§3.2).

Readings taken where the paper is silent (each is listed with its reason in the
design notes of the repository):

* Rounding of the norm (reading D1): the LM-head operand is u = bf16_rne(g * h);
  the RMS factor rho = (mean_d h_d^2 + eps)^(-1/2) multiplies the contraction, so
  z_v = rho * sum_d u_d W[v, d].  Logits are kept in fp64 and never rounded.
* The window layer K-1 (the final layer) goes through the same norm and head, which
  is what the model's native logits are (App. A.2: the final layer's logits are not
  normalised twice).
* argmax ties go to the lowest token index; fallback ties go to the leftmost
  position; the fallback window is the first W *masked* positions in canvas order.
* Thresholds are inclusive exactly as printed: c >= theta_h; theta_c <= c < theta_h;
  S >= theta_s; E_i <= beta.

Parity pins live in ``tests/test_oracle_*.py``.  The projection and the softmax
readout are pinned against library routines (torch rms_norm/linear, scipy softmax
and entropy) and closed forms; the scoring and commitment rules against hand-built
tables, the Table 4 ceilings of App. A.6 and brute force over all subsets.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

# Table 4 (App. A.6): hyperparameters of RPD.  theta_h and beta are per-call
# arguments (the step's ``tau`` and ``budget``); the rest form the rule profile.
RULES = {
    "llada": dict(theta_c=0.6, theta_s=3.5, w=15.0, k_max=6, window=32),
    "dream": dict(theta_c=0.6, theta_s=2.5, w=20.0, k_max=6, window=32),
}


# ----------------------------------------------------------------------------------------
# bf16 storage helpers (inputs arrive as raw bf16 bit patterns, uint16)
# ----------------------------------------------------------------------------------------

def bf16_to_f64(bits) -> np.ndarray:
    """Exact value of each bf16 bit pattern, as fp64 (bf16 is the top half of an fp32)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def f64_to_bf16_rne(x) -> np.ndarray:
    """Round values to bf16, round-to-nearest-even, returning bit patterns.

    The oracle only rounds products of two bf16 numbers; such a product has at most
    16 significant bits, so it is exact in fp32 and a single RNE from fp32 to bf16 is
    the correctly rounded result.  Inputs that are not exact in fp32 are rejected.
    """
    x = np.asarray(x, dtype=np.float64)
    f = x.astype(np.float32)
    finite = np.isfinite(x)
    if not np.array_equal(f.astype(np.float64)[finite], x[finite]):
        raise ValueError("f64_to_bf16_rne: value not exactly representable in fp32")
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16).astype(np.uint16)
    nan = np.isnan(f)
    r[nan] = ((u[nan] >> 16) | 0x40).astype(np.uint16)
    return r


# ----------------------------------------------------------------------------------------
# Layerwise projection (§2.2 logit lens; App. A.2, the readout of intermediate layers; App.
# A.6, the projection as implemented: final normalisation + output head on masked positions only)
# ----------------------------------------------------------------------------------------

def rms_factor(h_bits, eps: float) -> np.ndarray:
    """rho_r = (mean_d h_{r,d}^2 + eps)^(-1/2) for each row, in fp64."""
    h = bf16_to_f64(h_bits)
    return 1.0 / np.sqrt(np.mean(h * h, axis=-1) + eps)


def norm_operand(h_bits, g_bits) -> np.ndarray:
    """Reading D1: the head operand u = bf16_rne(g * h), elementwise, as bf16 bits."""
    return f64_to_bf16_rne(bf16_to_f64(g_bits) * bf16_to_f64(h_bits))


def project_logits(h_bits, g_bits, W_bits, eps: float, v_chunk: int = 8192) -> np.ndarray:
    """Logits z[r, v] = rho_r * sum_d u[r, d] * W[v, d] for every row r and every token v.

    ``h_bits`` is ``[R][d]``, ``g_bits`` ``[d]``, ``W_bits`` ``[V][d]`` (row v is token v's
    output embedding).  The full ``[R][V]`` fp64 matrix is materialised; the head is
    converted to fp64 in slabs of ``v_chunk`` tokens only to bound memory.
    """
    h_bits = np.ascontiguousarray(h_bits, dtype=np.uint16)
    R, d = h_bits.shape
    V = W_bits.shape[0]
    rho = rms_factor(h_bits, eps)
    u = bf16_to_f64(norm_operand(h_bits, g_bits))
    z = np.empty((R, V), dtype=np.float64)
    for v0 in range(0, V, v_chunk):
        v1 = min(V, v0 + v_chunk)
        z[:, v0:v1] = u @ bf16_to_f64(W_bits[v0:v1]).T
    z *= rho[:, None]
    return z


def project_logits_exact(h_bits, g_bits, W_bits, eps: float, v_chunk: int = 8192) -> np.ndarray:
    """Reading D3, a diagnostic only: the same logits with no rounding anywhere,
    z[r, v] = rho_r * sum_d g_d h_{r,d} W[v, d] in fp64 (the textbook RMSNorm followed by the
    head).  Comparing it with ``project_logits`` measures what reading D1's single bf16
    rounding of g*h changes."""
    h_bits = np.ascontiguousarray(h_bits, dtype=np.uint16)
    R, d = h_bits.shape
    V = W_bits.shape[0]
    rho = rms_factor(h_bits, eps)
    x = bf16_to_f64(g_bits) * bf16_to_f64(h_bits)  # unrounded
    z = np.empty((R, V), dtype=np.float64)
    for v0 in range(0, V, v_chunk):
        v1 = min(V, v0 + v_chunk)
        z[:, v0:v1] = x @ bf16_to_f64(W_bits[v0:v1]).T
    z *= rho[:, None]
    return z


def reading_gap(h_bits, g_bits, W_bits, eps: float) -> dict:
    """Diagnostic: how far reading D1 lies from the unrounded reading D3 on the given rows -
    the largest |p_D1(v) - p_D3(v)| over rows and tokens, the largest entropy difference, and
    how many rows change their argmax."""
    z1 = project_logits(h_bits, g_bits, W_bits, eps)
    z3 = project_logits_exact(h_bits, g_bits, W_bits, eps)
    p1, p3 = softmax(z1), softmax(z3)
    return {
        "rows": int(z1.shape[0]),
        "max_abs_dp": float(np.max(np.abs(p1 - p3))),
        "max_abs_dH": float(np.max(np.abs(entropy(p1) - entropy(p3)))),
        "argmax_differs": int(np.sum(np.argmax(z1, axis=-1) != np.argmax(z3, axis=-1))),
    }


# ----------------------------------------------------------------------------------------
# Readout of one predictive distribution (Eq. 1)
# ----------------------------------------------------------------------------------------

def softmax(z) -> np.ndarray:
    """p(v) = exp(z_v) / sum_u exp(z_u), computed with the maximum subtracted, fp64."""
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - np.max(z, axis=-1, keepdims=True))
    return e / np.sum(e, axis=-1, keepdims=True)


def entropy(p) -> np.ndarray:
    """H(p) = -sum_v p(v) ln p(v) in nats, with 0 ln 0 = 0 (Eq. 1)."""
    p = np.asarray(p, dtype=np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        terms = np.where(p > 0, p * np.log(np.where(p > 0, p, 1.0)), 0.0)
    return -np.sum(terms, axis=-1)


def argmax_lowest(z) -> np.ndarray:
    """Index of the largest logit; the lowest index wins an exact tie."""
    return np.argmax(np.asarray(z), axis=-1)


def top2_gap(z) -> np.ndarray:
    """Largest minus second-largest logit (0 on an exact tie)."""
    z = np.asarray(z, dtype=np.float64)
    part = np.partition(z, -2, axis=-1)
    return part[..., -1] - part[..., -2]


# ----------------------------------------------------------------------------------------
# Layerwise stability (§2.2 Eq. 2-3 with App. A.2; §3.1 Eq. 4-5)
# ----------------------------------------------------------------------------------------

def persistence(layer_argmax) -> int:
    """K_i (Eq. 2): consecutive window layers, counted backward from the final layer, whose
    argmax equals the final prediction.  The count stops at the first disagreement, so
    earlier matches separated by a disagreement are excluded (App. A.2)."""
    a = list(layer_argmax)
    y = a[-1]
    k_i = 1
    for k in range(len(a) - 2, -1, -1):
        if a[k] != y:
            break
        k_i += 1
    return k_i


def confidence_drop(p_of_y, k_i: int) -> float:
    """r_i (Eq. 3): max over the consistent suffix [s_i, L] of p^(l)(y_i), minus p^(L)(y_i).

    ``p_of_y[k]`` is layer k's probability of the final prediction y_i (window order,
    last entry = final layer); the suffix is its last ``k_i`` entries (s_i = L - K_i + 1)."""
    p = list(p_of_y)
    suffix = p[len(p) - k_i:]
    return max(suffix) - p[-1]


def stability(k_i: int, r_i: float, k_max: int, w: float) -> float:
    """S_i = min(K_i, K_max) - w * r_i (Eq. 4)."""
    return min(k_i, k_max) - w * r_i


def is_candidate(c: float, s: float, theta_h: float, theta_c: float, theta_s: float) -> bool:
    """Membership in C_t (Eq. 5) for a masked position: c >= theta_h, or
    theta_c <= c < theta_h together with S >= theta_s."""
    return bool(c >= theta_h or (theta_c <= c < theta_h and s >= theta_s))


# ----------------------------------------------------------------------------------------
# Parallel commitment with cumulative entropy (§3.2)
# ----------------------------------------------------------------------------------------

def commit_sequential(masked, cand, H, beta: float) -> list:
    """A_t built left to right (§3.2): scanning candidates in canvas order, candidate i joins
    when E_i = sum of H_j over j < i, j masked and not already in A_{t,<i}, is <= beta.
    The sum runs over every earlier masked position (non-candidates and rejected
    candidates included) and skips the candidates already selected."""
    N = len(masked)
    A = []
    chosen = set()
    for i in range(N):
        if not cand[i]:
            continue
        E = 0.0
        for j in range(i):
            if masked[j] and j not in chosen:
                E += float(H[j])
        if E <= beta:
            A.append(i)
            chosen.add(i)
    return A


def accepted_prefix(masked, cand, H, beta: float) -> list:
    """Closed form of the §3.2 rule, used only to cross-check ``commit_sequential`` at every
    call: with Q_i the entropy of the masked non-candidates before i (a running sum in canvas
    order), A_t is the candidates before the first candidate with Q_i > beta.  While every
    earlier candidate was accepted E_i = Q_i term by term, and H >= 0 means that once one
    candidate is rejected every later one is too; the sums are therefore bit-identical."""
    A = []
    q = 0.0
    for i in range(len(masked)):
        if cand[i]:
            if q > beta:
                break
            A.append(i)
        elif masked[i]:
            q += float(H[i])
    return A


def fallback_commit(masked, c, window: int) -> int:
    """§3.2: when A_t is empty, commit the single prediction with the highest final
    confidence among the first ``window`` masked positions from the left (leftmost wins a
    tie).  Returns -1 when nothing is masked."""
    first = [i for i in range(len(masked)) if masked[i]][:window]
    if not first:
        return -1
    best = first[0]
    for i in first[1:]:
        if c[i] > c[best]:
            best = i
    return best


# ----------------------------------------------------------------------------------------
# One full step
# ----------------------------------------------------------------------------------------

@dataclass
class StepResult:
    commit: np.ndarray        # [N] uint8, 1 where committed this step
    token: np.ndarray         # [N] int64, y_i where committed, -1 elsewhere
    new_mask: np.ndarray      # [N] uint8
    masked: np.ndarray        # [N] bool (input mask)
    layer_argmax: np.ndarray  # [K][N] int64 (-1 at unmasked positions)
    layer_pmax: np.ndarray    # [K][N] p^(k)(argmax) (nan at unmasked)
    layer_gap: np.ndarray     # [K][N] top-2 logit gap (nan at unmasked)
    p_of_y: np.ndarray        # [K][N] p^(k)(y_i)
    y: np.ndarray             # [N] final prediction
    conf: np.ndarray          # [N] c_i
    H: np.ndarray             # [N] final-layer entropy
    persist: np.ndarray       # [N] K_i
    drop: np.ndarray          # [N] r_i
    stab: np.ndarray          # [N] S_i
    cand: np.ndarray          # [N] bool
    high_conf: np.ndarray     # [N] bool, candidate through c >= theta_h
    accepted: list            # A_t from the sequential rule (before fallback)
    fallback_pos: int         # -1 if no fallback was needed
    params: dict


def readout_rows(z_rows: np.ndarray):
    """Per-row readout for one position's window rows: the full distributions, the argmax,
    the probability at the argmax and the top-2 logit gap of every row."""
    P = softmax(z_rows)
    a = argmax_lowest(z_rows)
    pmax = P[np.arange(P.shape[0]), a]
    gap = top2_gap(z_rows)
    return P, a, pmax, gap


def score_positions(hidden_bits, positions, g_bits, W_bits, eps: float, tau: float, rule):
    """Steps 1-4 for the given masked positions: per-layer readout (App. A.2), y, c, H (Eq. 1),
    K_i, r_i, S_i (Eq. 2-4) and candidacy (Eq. 5).  Returns arrays over the canvas (entries
    outside ``positions`` keep their "not scored" values)."""
    hidden_bits = np.asarray(hidden_bits, dtype=np.uint16)
    K, N, d = hidden_bits.shape
    M = np.asarray(positions, dtype=np.int64)
    nm = len(M)
    out = dict(
        layer_argmax=np.full((K, N), -1, dtype=np.int64), layer_pmax=np.full((K, N), np.nan),
        layer_gap=np.full((K, N), np.nan), p_of_y=np.full((K, N), np.nan),
        y=np.full(N, -1, dtype=np.int64), conf=np.full(N, np.nan), H=np.zeros(N),
        persist=np.zeros(N, dtype=np.int64), drop=np.full(N, np.nan), stab=np.full(N, np.nan),
        cand=np.zeros(N, dtype=bool), high=np.zeros(N, dtype=bool))
    if nm == 0:
        return out
    rows = hidden_bits[:, M, :].reshape(K * nm, d)     # masked positions only (App. A.6)
    z = project_logits(rows, g_bits, W_bits, eps).reshape(K, nm, -1)
    for qi, i in enumerate(M):
        P, a, pmax, gap = readout_rows(z[:, qi, :])
        out["layer_argmax"][:, i] = a
        out["layer_pmax"][:, i] = pmax
        out["layer_gap"][:, i] = gap
        yi = int(a[-1])
        out["y"][i] = yi
        out["p_of_y"][:, i] = P[:, yi]
        out["conf"][i] = P[-1, yi]
        out["H"][i] = float(entropy(P[-1]))
        out["persist"][i] = persistence(a)
        out["drop"][i] = confidence_drop(P[:, yi], int(out["persist"][i]))
        out["stab"][i] = stability(int(out["persist"][i]), float(out["drop"][i]), rule["k_max"],
                                   rule["w"])
        out["cand"][i] = is_candidate(out["conf"][i], out["stab"][i], tau, rule["theta_c"],
                                      rule["theta_s"])
        out["high"][i] = bool(out["conf"][i] >= tau)
    return out


def _result(sc, masked, A, fb, params):
    N = masked.shape[0]
    commit = np.zeros(N, dtype=np.uint8)
    for i in A:
        commit[i] = 1
    if fb >= 0:
        commit[fb] = 1
    token = np.where(commit == 1, sc["y"], -1)
    new_mask = (masked & (commit == 0)).astype(np.uint8)
    return StepResult(commit=commit, token=token, new_mask=new_mask, masked=masked,
                      layer_argmax=sc["layer_argmax"], layer_pmax=sc["layer_pmax"],
                      layer_gap=sc["layer_gap"], p_of_y=sc["p_of_y"], y=sc["y"], conf=sc["conf"],
                      H=sc["H"], persist=sc["persist"], drop=sc["drop"], stab=sc["stab"],
                      cand=sc["cand"], high_conf=sc["high"], accepted=A, fallback_pos=fb,
                      params=params)


def rpd_step(hidden_bits, mask, g_bits, W_bits, eps: float, tau: float, budget: float,
             rule) -> StepResult:
    """One RPD commit step for one canvas.

    ``hidden_bits`` is ``[K][N][d]`` bf16 bits (window layers in depth order, the last one
    the final layer, each the pre-norm hidden state), ``mask`` ``[N]`` (1 = masked),
    ``g_bits`` ``[d]``, ``W_bits`` ``[V][d]``.  ``tau`` is theta_h, ``budget`` is beta and
    ``rule`` is a dict with theta_c, theta_s, w, k_max, window (or a Table 4 profile name).
    """
    if isinstance(rule, str):
        rule = RULES[rule]
    masked = np.asarray(mask).astype(bool)
    sc = score_positions(hidden_bits, np.nonzero(masked)[0], g_bits, W_bits, eps, tau, rule)
    A = commit_sequential(masked, sc["cand"], sc["H"], budget)
    assert A == accepted_prefix(masked, sc["cand"], sc["H"], budget)
    fb = -1
    if not A and masked.any():
        fb = fallback_commit(masked, sc["conf"], rule["window"])
    params = dict(rule)
    params.update(tau=tau, budget=budget)
    return _result(sc, masked, A, fb, params)


def active_block(masked, block: int):
    """RPD-block (App. A.6): the active block is the first fixed block of ``block`` positions
    that still holds a masked position; returns its masked positions (empty if none)."""
    masked = np.asarray(masked).astype(bool)
    idx = np.nonzero(masked)[0]
    if len(idx) == 0:
        return idx
    j = int(idx[0]) // block
    return idx[(idx >= j * block) & (idx < (j + 1) * block)]


def rpd_block_step(hidden_bits, mask, g_bits, W_bits, eps: float, tau: float, rule,
                   block: int = 32) -> StepResult:
    """RPD-block (the variant of §3.2, App. A.6): the candidate selection of Eq. 5 applied within
    the active block of ``block`` positions, no cumulative-entropy budget (every candidate of
    the block is committed), and, when no candidate passes, the most confident masked
    position of the active block (leftmost on ties)."""
    if isinstance(rule, str):
        rule = RULES[rule]
    masked = np.asarray(mask).astype(bool)
    act = active_block(masked, block)
    sc = score_positions(hidden_bits, act, g_bits, W_bits, eps, tau, rule)
    A = [int(i) for i in act if sc["cand"][i]]
    fb = -1
    if not A and len(act):
        fb = int(act[0])
        for i in act[1:]:
            if sc["conf"][i] > sc["conf"][fb]:
                fb = int(i)
    params = dict(rule)
    params.update(tau=tau, budget=math.inf, block=block)
    return _result(sc, masked, A, fb, params)


def rpd_step_batched(hidden_bits, masks, g_bits, W_bits, eps: float, taus, budgets, rule):
    """Independent canvases: ``hidden_bits`` ``[K][B][N][d]``, ``masks`` ``[B][N]``."""
    hidden_bits = np.asarray(hidden_bits, dtype=np.uint16)
    B = hidden_bits.shape[1]
    return [rpd_step(hidden_bits[:, b], masks[b], g_bits, W_bits, eps, taus[b], budgets[b], rule)
            for b in range(B)]


def step_from_scores(masked, layer_argmax, layer_p_of_y, H, tau, budget, rule):
    """Steps 3-5 applied to given per-layer argmaxes, per-layer p(y_i) and final entropies.

    Used to replay the commitment rule on score tables (hand-built cases); returns
    (commit[N] uint8, cand[N] bool, accepted list, fallback position)."""
    if isinstance(rule, str):
        rule = RULES[rule]
    masked = np.asarray(masked).astype(bool)
    layer_argmax = np.asarray(layer_argmax)
    layer_p_of_y = np.asarray(layer_p_of_y, dtype=np.float64)
    N = masked.shape[0]
    cand = np.zeros(N, dtype=bool)
    conf = np.full(N, np.nan)
    for i in range(N):
        if not masked[i]:
            continue
        k_i = persistence(layer_argmax[:, i])
        r_i = confidence_drop(layer_p_of_y[:, i], k_i)
        s_i = stability(k_i, r_i, rule["k_max"], rule["w"])
        conf[i] = layer_p_of_y[-1, i]
        cand[i] = is_candidate(conf[i], s_i, tau, rule["theta_c"], rule["theta_s"])
    A = commit_sequential(masked, cand, H, budget)
    assert A == accepted_prefix(masked, cand, H, budget)
    fb = -1
    if not A and masked.any():
        fb = fallback_commit(masked, conf, rule["window"])
    commit = np.zeros(N, dtype=np.uint8)
    commit[A] = 1
    if fb >= 0:
        commit[fb] = 1
    return commit, cand, A, fb


def block_step_from_scores(masked, layer_argmax, layer_p_of_y, tau, rule, block: int = 32):
    """RPD-block's rule applied to given per-layer argmaxes and p(y_i) tables (hand-built
    cases): returns (commit[N] uint8, cand[N] bool, fallback position)."""
    if isinstance(rule, str):
        rule = RULES[rule]
    masked = np.asarray(masked).astype(bool)
    layer_argmax = np.asarray(layer_argmax)
    layer_p_of_y = np.asarray(layer_p_of_y, dtype=np.float64)
    N = masked.shape[0]
    act = active_block(masked, block)
    cand = np.zeros(N, dtype=bool)
    conf = np.full(N, np.nan)
    for i in act:
        k_i = persistence(layer_argmax[:, i])
        r_i = confidence_drop(layer_p_of_y[:, i], k_i)
        conf[i] = layer_p_of_y[-1, i]
        cand[i] = is_candidate(conf[i], stability(k_i, r_i, rule["k_max"], rule["w"]), tau,
                               rule["theta_c"], rule["theta_s"])
    commit = np.zeros(N, dtype=np.uint8)
    A = [int(i) for i in act if cand[i]]
    fb = -1
    if not A and len(act):
        fb = int(act[0])
        for i in act[1:]:
            if conf[i] > conf[fb]:
                fb = int(i)
    commit[A] = 1
    if fb >= 0:
        commit[fb] = 1
    return commit, cand, fb
