"""Seeded synthetic inputs for the RPD commit step.

This module draws inputs only: LM heads, RMSNorm gains, per-layer hidden states
and canvas masks, with the shapes and structure of the workloads the method runs
on (LLaDA-8B head: d=4096, V=126464; Dream-7B head: d=3584, V=152064; a 256-token
generation canvas whose confidence profile is U-shaped along the canvas, §1 and
§4.1 of the paper).  It holds none of the step's arithmetic; both the CUDA path
and the CPU oracle consume what it returns.

Every tensor is a CPU torch tensor produced from an explicit ``torch.Generator``
seed, so the same call gives the same bits on any machine.  bf16 tensors are
returned as ``torch.bfloat16``.

Hidden-state recipe (one canvas, K window layers, N positions):

    h[k][p] = a_k * b_p * sigma * W[t_p] / ||W[t_p]||  +  n,   n ~ N(0, I_d)

with target tokens ``t_p`` uniform over the vocabulary, ``a_k`` rising linearly
from 0.6 to 1.0 over the window (the last entry is the final layer), ``b_p`` a
per-position signal profile, and ``sigma`` the signal scale.  ``sigma = 1`` is
the literal recipe; it leaves every final-layer confidence near 1/V on the large
heads, so the calibrated recipe uses ``sigma = kappa * sqrt(d)`` (kappa = 0.06
by default), which makes the canvas ends confident and its middle uncertain.
A seeded fraction of positions (``flip_frac``) reads a different target in the
penultimate window layer, which breaks their layerwise agreement.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

LLADA_D, LLADA_V = 4096, 126464
DREAM_D, DREAM_V = 3584, 152064

DEFAULT_KAPPA = 0.06


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return g


def make_head(V: int, d: int, seed: int, w_std: float = 0.02, g_std: float = 0.1):
    """LM head ``W[V][d] ~ N(0, w_std)`` and RMSNorm gain ``g[d] = 1 + N(0, g_std)``, both bf16."""
    gen = _gen(seed)
    W = torch.empty(V, d, dtype=torch.bfloat16)
    rows = max(1, (1 << 24) // max(d, 1))  # draw in slabs to bound fp32 temporaries
    for r0 in range(0, V, rows):
        r1 = min(V, r0 + rows)
        W[r0:r1] = (torch.randn(r1 - r0, d, generator=gen) * w_std).to(torch.bfloat16)
    g = (1.0 + g_std * torch.randn(d, generator=gen)).to(torch.bfloat16)
    return W, g


def u_profile(N: int, lo: float, hi: float) -> torch.Tensor:
    """U-shaped signal profile over canvas positions: ``lo`` mid-canvas, ``hi`` at both ends."""
    if N == 1:
        return torch.tensor([hi], dtype=torch.float32)
    x = (torch.arange(N, dtype=torch.float64) - (N - 1) / 2) / ((N - 1) / 2)
    return (lo + (hi - lo) * x * x).to(torch.float32)


def lognormal_profile(N: int, seed: int, sigma: float = 0.7) -> torch.Tensor:
    gen = _gen(seed)
    return torch.exp(sigma * torch.randn(N, generator=gen)).to(torch.float32)


def layer_ramp(K: int, lo: float = 0.6, hi: float = 1.0) -> torch.Tensor:
    if K == 1:
        return torch.tensor([hi], dtype=torch.float32)
    return torch.linspace(lo, hi, K, dtype=torch.float32)


@dataclass
class Canvas:
    """Hidden states ``[K][N][d]`` (bf16) plus the draw's bookkeeping."""
    hidden: torch.Tensor
    targets: torch.Tensor          # [N] int64
    flip_targets: torch.Tensor     # [N] int64, -1 where the position is not flipped
    b: torch.Tensor                # [N] float32
    a: torch.Tensor                # [K] float32
    sigma: float
    extra: dict = field(default_factory=dict)


def make_hidden(W: torch.Tensor, K: int, N: int, seed: int, b: torch.Tensor,
                sigma: float, flip_frac: float = 0.0, a: torch.Tensor | None = None,
                targets: torch.Tensor | None = None) -> Canvas:
    """Hidden states for one canvas following the module recipe."""
    V, d = W.shape
    gen = _gen(seed)
    if targets is None:
        targets = torch.randint(0, V, (N,), generator=gen)
    else:
        targets = targets.clone()
        torch.randint(0, V, (N,), generator=gen)  # keep the stream aligned
    if a is None:
        a = layer_ramp(K)
    flip = torch.full((N,), -1, dtype=torch.int64)
    n_flip = int(round(flip_frac * N))
    if n_flip > 0 and K >= 2:
        pos = torch.randperm(N, generator=gen)[:n_flip]
        alt = torch.randint(1, V, (n_flip,), generator=gen)
        flip[pos] = (targets[pos] + alt) % V
    else:
        torch.randperm(max(N, 1), generator=gen)
    wt = W[targets].to(torch.float32)
    wt = wt / wt.norm(dim=1, keepdim=True).clamp_min(1e-30)
    if (flip >= 0).any():
        wf = W[flip.clamp_min(0)].to(torch.float32)
        wf = wf / wf.norm(dim=1, keepdim=True).clamp_min(1e-30)
    hidden = torch.empty(K, N, d, dtype=torch.bfloat16)
    for k in range(K):
        dirs = wt
        if k == K - 2 and (flip >= 0).any():
            dirs = torch.where((flip >= 0)[:, None], wf, wt)
        sig = (float(a[k]) * sigma) * b[:, None] * dirs
        noise = torch.randn(N, d, generator=gen)
        hidden[k] = (sig + noise).to(torch.bfloat16)
    return Canvas(hidden=hidden, targets=targets, flip_targets=flip, b=b, a=a, sigma=sigma)


def front_loaded_mask(N: int, seed: int) -> torch.Tensor:
    """Mid-decode mask: position p is already committed with probability 1 - p/(N-1)."""
    gen = _gen(seed)
    p = torch.arange(N, dtype=torch.float64)
    prob_committed = 1.0 - p / max(N - 1, 1)
    u = torch.rand(N, generator=gen, dtype=torch.float64)
    return (u >= prob_committed).to(torch.uint8)


def uniform_fraction_mask(N: int, frac: float, seed: int) -> torch.Tensor:
    """Exactly ``round(frac*N)`` masked positions, uniformly placed."""
    gen = _gen(seed)
    m = torch.zeros(N, dtype=torch.uint8)
    n = int(round(frac * N))
    m[torch.randperm(N, generator=gen)[:n]] = 1
    return m


def calibrated_sigma(V: int, d: int, w_std: float, b_max: float, margin: float = 5.0) -> float:
    """Signal scale putting the final-layer target logit at ``b_max`` a ``margin`` (nats)
    above the log-partition of the noise logits.  With h = sigma*b*w_hat + n and
    W ~ N(0, w_std), the target logit is about sigma*b*w_std*sqrt(d) and the V noise
    logits are about N(0, (w_std*sqrt(d))^2), whose log-partition is
    ln V + (w_std*sqrt(d))^2 / 2."""
    s = w_std * math.sqrt(d)
    return (math.log(V) + 0.5 * s * s + margin) / (b_max * s)


# --------------------------------------------------------------------------------------
# Named workloads.  Each returns a dict with the head, the hidden states, the mask(s) and
# the per-call parameters; "rule" names the Table 4 profile (llada or dream).
# --------------------------------------------------------------------------------------

def tiny_step(seed: int = 1, calibrated: bool = False):
    """Batch 1, N=64 all masked, K=3, d=256, V=4096, tau 0.9, budget 1.0.

    ``calibrated=False`` is the literal recipe (W ~ N(0, 0.02), sigma = 1), whose
    confidences stay near 1/V so every step takes the fallback commit.
    ``calibrated=True`` widens the head to W ~ N(0, 0.08) and sets the signal so that the
    final-layer target logit at the canvas ends sits 5 nats above the noise partition
    (``calibrated_sigma``), so that candidates, budget waits and fallbacks all occur.
    """
    K, N, d, V = 3, 64, 256, 4096
    w_std = 0.08 if calibrated else 0.02
    W, g = make_head(V, d, seed, w_std=w_std)
    b = u_profile(N, 0.5, 3.0)
    sigma = calibrated_sigma(V, d, w_std, b_max=3.0) if calibrated else 1.0
    cv = make_hidden(W, K, N, seed + 1000, b, sigma, flip_frac=0.1 if calibrated else 0.0)
    mask = torch.ones(N, dtype=torch.uint8)
    return dict(name="tiny", W=W, g=g, hidden=cv.hidden, mask=mask, K=K, N=N, d=d, V=V,
                eps=1e-6, tau=0.9, budget=1.0, rule="llada", canvas=cv, seed=seed)


def llada_first_step(seed: int = 2, kappa: float = DEFAULT_KAPPA, W=None, g=None, K: int = 4):
    """Batch 1, N=256 all masked, K=4 (or another window), LLaDA-8B head (d=4096, V=126464),
    tau 0.9, budget 1.0.

    b_p is U-shaped from 0.3 (mid) to 4 (ends); 10% of positions flip their target in the
    penultimate window layer.
    """
    N, d, V = 256, LLADA_D, LLADA_V
    if W is None:
        W, g = make_head(V, d, seed)
    b = u_profile(N, 0.3, 4.0)
    cv = make_hidden(W, K, N, seed + 1000, b, kappa * math.sqrt(d), flip_frac=0.1)
    mask = torch.ones(N, dtype=torch.uint8)
    return dict(name="llada_first_step", W=W, g=g, hidden=cv.hidden, mask=mask, K=K, N=N,
                d=d, V=V, eps=1e-6, tau=0.9, budget=1.0, rule="llada", canvas=cv, seed=seed,
                kappa=kappa)


def dream_mid_decode(seed: int = 3, kappa: float = DEFAULT_KAPPA, W=None, g=None):
    """Batch 1, N=512, front-loaded 50% mask, K=4, Dream-7B head (d=3584, V=152064),
    tau 0.85, budget 2.0; b_p ~ LogNormal(0, 0.7) scaled to the calibrated signal."""
    K, N, d, V = 4, 512, DREAM_D, DREAM_V
    if W is None:
        W, g = make_head(V, d, seed)
    b = lognormal_profile(N, seed + 7) * 2.5
    cv = make_hidden(W, K, N, seed + 1000, b, kappa * math.sqrt(d), flip_frac=0.1)
    mask = front_loaded_mask(N, seed + 11)
    return dict(name="dream_mid_decode", W=W, g=g, hidden=cv.hidden, mask=mask, K=K, N=N,
                d=d, V=V, eps=1e-6, tau=0.85, budget=2.0, rule="dream", canvas=cv, seed=seed,
                kappa=kappa)


def batched_serving(seed: int = 5, kappa: float = DEFAULT_KAPPA, B: int = 8, N: int = 1024,
                    K: int = 6, d: int = LLADA_D, V: int = LLADA_V, W=None, g=None):
    """B independent canvases of N positions, each masked at a fraction drawn from U(0.3, 1),
    K=6, LLaDA head; per-canvas tau 0.9 and budget 1.5."""
    if W is None:
        W, g = make_head(V, d, seed)
    gen = _gen(seed + 17)
    fracs = 0.3 + 0.7 * torch.rand(B, generator=gen, dtype=torch.float64)
    hidden = torch.empty(K, B, N, d, dtype=torch.bfloat16)
    masks = torch.empty(B, N, dtype=torch.uint8)
    canvases = []
    for bi in range(B):
        b = u_profile(N, 0.3, 4.0)
        cv = make_hidden(W, K, N, seed + 1000 + bi, b, kappa * math.sqrt(d), flip_frac=0.1)
        hidden[:, bi] = cv.hidden
        masks[bi] = uniform_fraction_mask(N, float(fracs[bi]), seed + 2000 + bi)
        canvases.append(cv)
    return dict(name="batched_serving", W=W, g=g, hidden=hidden, mask=masks, K=K, B=B, N=N,
                d=d, V=V, eps=1e-6, tau=[0.9] * B, budget=[1.5] * B, rule="llada",
                canvases=canvases, seed=seed, kappa=kappa)


def trajectory_profile(base_b: torch.Tensor, mask: torch.Tensor, b_hi: float = 4.0,
                       gamma: float = 8.0) -> torch.Tensor:
    """Signal profile for a decode-trajectory step: ``b_p + (b_hi - b_p) * f_p**gamma`` where
    ``f_p`` is the committed fraction of the positions before p.  A position becomes as
    confident as the canvas ends once (nearly) all the context to its left has been
    committed, so the canvas resolves left to right (the progression of App. A.7); a larger
    ``gamma`` resolves fewer positions per step."""
    N = mask.numel()
    committed = (mask == 0).to(torch.float64)
    before = torch.cumsum(committed, 0) - committed
    denom = torch.arange(N, dtype=torch.float64).clamp_min(1)
    f = torch.where(torch.arange(N) > 0, before / denom, torch.ones(N, dtype=torch.float64))
    b = base_b.to(torch.float64)
    return (b + (b_hi - b).clamp_min(0) * f.pow(gamma)).to(torch.float32)


def trajectory_hidden(W: torch.Tensor, K: int, N: int, seed: int, step: int, mask: torch.Tensor,
                      kappa: float = DEFAULT_KAPPA, targets: torch.Tensor | None = None,
                      gamma: float = 8.0) -> Canvas:
    """Hidden states for step ``step`` of a decode trajectory at the current ``mask``."""
    d = W.shape[1]
    b = trajectory_profile(u_profile(N, 0.3, 4.0), mask, gamma=gamma)
    return make_hidden(W, K, N, seed * 1000 + step, b, kappa * math.sqrt(d), flip_frac=0.1,
                       targets=targets)
