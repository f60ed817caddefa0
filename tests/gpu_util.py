"""Helpers for GPU tests: run one step through the C ABI and fetch every output."""
from __future__ import annotations

import numpy as np
import torch


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> raw uint16 bit patterns (numpy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


class DeviceRunner:
    """Context + head on cuda:0; runs single or batched steps with every debug output."""

    def __init__(self, W: torch.Tensor, g: torch.Tensor, K: int, eps: float = 1e-6, rule="llada",
                 layout=None):
        import paper_2609_36452_gb300 as rpd
        self.rpd = rpd
        self.dev = torch.device("cuda:0")
        self.V, self.d = W.shape
        self.K = K
        self.W = W.to(self.dev).contiguous()
        self.g = g.to(self.dev).contiguous()
        self.ctx = rpd.Rpd(self.d, self.V, K, eps)
        if layout is not None:
            self.ctx.set_head_layout(layout)
        self.ctx.set_head(self.W, self.g)
        self.set_rule(rule)
        self.ctx.set_stream(torch.cuda.current_stream(self.dev))

    def set_rule(self, rule):
        if isinstance(rule, str):
            self.ctx.set_profile(rule)
        else:
            self.ctx.set_rule(rule["theta_c"], rule["theta_s"], rule["w"], rule["k_max"], rule["window"],
                              rule.get("block", 0))

    def _alloc(self, B, N):
        dev, K = self.dev, self.K
        out = dict(
            commit=torch.full((B, N), 7, dtype=torch.uint8, device=dev),
            token=torch.full((B, N), -5, dtype=torch.int32, device=dev),
            stats=torch.full((B, self.rpd.STATS_WORDS), -9, dtype=torch.int32, device=dev),
            conf=torch.full((B, N), -1.0, device=dev),
            entropy=torch.full((B, N), -1.0, device=dev),
            persist=torch.full((B, N), -1, dtype=torch.int32, device=dev),
            drop=torch.full((B, N), -1.0, device=dev),
            stability=torch.full((B, N), -1.0, device=dev),
            candidate=torch.full((B, N), 9, dtype=torch.uint8, device=dev),
            layer_argmax=torch.full((K, B, N), -7, dtype=torch.int32, device=dev),
            layer_pmax=torch.full((K, B, N), -1.0, device=dev),
        )
        self.ctx.set_debug(**{k: out[k] for k in ("conf", "entropy", "persist", "drop", "stability",
                                                   "candidate", "layer_argmax", "layer_pmax")})
        return out

    def _fetch(self, out, mask, B):
        torch.cuda.synchronize(self.dev)
        res = []
        for b in range(B):
            r = {k: v[b].cpu().numpy() for k, v in out.items() if k not in ("layer_argmax", "layer_pmax", "stats")}
            r["layer_argmax"] = out["layer_argmax"][:, b].cpu().numpy()
            r["layer_pmax"] = out["layer_pmax"][:, b].cpu().numpy()
            r["stats"] = self.rpd.stats_dict(out["stats"][b].cpu())
            # a library built with RPD_CHECKS latches a failed device-side bounds check here
            assert r["stats"]["status"] != self.rpd.RPD_ERR_CHECK, "device-side bounds check failed"
            r["new_mask"] = mask[b].cpu().numpy()
            res.append(r)
        return res

    def step(self, hidden: torch.Tensor, mask: torch.Tensor, tau: float, budget: float):
        """hidden [K][N][d] bf16 (CPU or CUDA), mask [N] uint8 -> dict of numpy outputs."""
        N = mask.numel()
        h = hidden.to(self.dev).contiguous()
        m = mask.to(self.dev).clone().reshape(1, N)
        out = self._alloc(1, N)
        self.ctx.step(h, m[0], tau, budget, out["commit"][0], out["token"][0], out["stats"][0])
        return self._fetch(out, m, 1)[0]

    def step_batched(self, hidden: torch.Tensor, mask: torch.Tensor, taus, budgets):
        """hidden [K][B][N][d], mask [B][N] -> list of per-canvas dicts."""
        B, N = mask.shape
        h = hidden.to(self.dev).contiguous()
        m = mask.to(self.dev).clone()
        out = self._alloc(B, N)
        self.ctx.step_batched(h, m, taus, budgets, out["commit"], out["token"], out["stats"])
        return self._fetch(out, m, B)

    def close(self):
        self.ctx.close()
