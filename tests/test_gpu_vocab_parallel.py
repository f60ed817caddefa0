"""Vocabulary-parallel step on one GPU: the head is split into contiguous slices, one context
per slice computes its statistics (rpd_step_shard_partials), the slices' records are stacked
as an all-gather would, and one context merges and commits (rpd_step_shard_finish).  Compared
with the oracle on the whole head, and with the unsharded step."""
import numpy as np
import pytest
import torch

import workloads as WL
from tests.gpu_util import DeviceRunner
from tests.parity import compare_step
from tests.test_gpu_parity import oracle_step, small_case

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # collected on CPU machines, never run there
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2609_36452_gb300 as rpd  # noqa: E402
from paper_2609_36452_gb300.vocab_parallel import shard_bounds  # noqa: E402

DEV = torch.device("cuda:0")


def sharded(case, P, rule="llada", stall_slice=None):
    """Run the sharded step with P slices; returns a DeviceRunner-style result dict."""
    K, N, d, V = case["K"], case["N"], case["d"], case["V"]
    W = case["W"].to(DEV)
    g = case["g"].to(DEV)
    hidden = case["hidden"].to(DEV).contiguous()
    mask = case["mask"].to(DEV).clone()
    ctxs, parts = [], []
    for r in range(P):
        v0, v1 = shard_bounds(V, P, r)
        c = rpd.Rpd(d, v1 - v0, K, case["eps"])
        c.set_head(W[v0:v1], g)
        c.set_vocab_shard(v0, V)
        c.set_profile(rule) if isinstance(rule, str) else c.set_rule(**rule)
        c.set_stream(torch.cuda.current_stream(DEV))
        if stall_slice == r:
            c.set_wait_limit(20000)
            c.inject_stall()
        part = torch.full((K, N, 4), float("nan"), device=DEV)
        c.step_shard_partials(hidden, mask, part)
        ctxs.append(c)
        parts.append(part)
    gathered = torch.stack(parts).contiguous()
    out = dict(commit=torch.full((N,), 7, dtype=torch.uint8, device=DEV),
               token=torch.full((N,), -5, dtype=torch.int32, device=DEV),
               stats=torch.full((rpd.STATS_WORDS,), -9, dtype=torch.int32, device=DEV),
               conf=torch.full((N,), -1.0, device=DEV), entropy=torch.full((N,), -1.0, device=DEV),
               persist=torch.full((N,), -1, dtype=torch.int32, device=DEV),
               drop=torch.full((N,), -1.0, device=DEV), stability=torch.full((N,), -1.0, device=DEV),
               candidate=torch.full((N,), 9, dtype=torch.uint8, device=DEV),
               layer_argmax=torch.full((K, N), -7, dtype=torch.int32, device=DEV),
               layer_pmax=torch.full((K, N), -1.0, device=DEV))
    fin = ctxs[stall_slice or 0]
    fin.set_debug(**{k: out[k] for k in ("conf", "entropy", "persist", "drop", "stability",
                                         "candidate", "layer_argmax", "layer_pmax")})
    fin.step_shard_finish(gathered, mask, case["tau"], case["budget"], out["commit"], out["token"],
                          out["stats"])
    torch.cuda.synchronize(DEV)
    res = {k: v.cpu().numpy() for k, v in out.items() if k != "stats"}
    res["stats"] = rpd.stats_dict(out["stats"].cpu())
    res["new_mask"] = mask.cpu().numpy()
    for c in ctxs:
        c.close()
    return res


@pytest.mark.parametrize("P", [2, 3])
@pytest.mark.parametrize("d,V,K,N,frac", [
    (256, 4100, 3, 100, 1.0),    # slices of 1280-1536 entries, ragged last one
    (192, 1000, 4, 77, 0.6),     # slices of 256-512 entries
])
def test_sharded_step_matches_oracle(P, d, V, K, N, frac):
    case = small_case(500 + d + V + K + P, K=K, N=N, d=d, V=V, w_std=0.08, mask_frac=frac)
    got = sharded(case, P)
    assert got["stats"]["status"] == rpd.RPD_OK
    print(compare_step(oracle_step(case), got))


def test_sharded_step_matches_unsharded_llada_first_step():
    """LLaDA-8B head split in two (63232 + 63232 entries) against the unsharded step on the
    same inputs: the same commits and tokens, confidences and entropies within 1e-4."""
    W, g = WL.make_head(WL.LLADA_V, WL.LLADA_D, seed=2)
    case = WL.llada_first_step(seed=2, W=W, g=g)
    got = sharded(case, 2)
    runner = DeviceRunner(case["W"], case["g"], case["K"], case["eps"], rule="llada")
    try:
        ref = runner.step(case["hidden"], case["mask"], case["tau"], case["budget"])
    finally:
        runner.close()
    assert got["stats"]["status"] == rpd.RPD_OK
    assert np.array_equal(got["commit"], ref["commit"]) and np.array_equal(got["new_mask"], ref["new_mask"])
    sel = got["commit"] == 1
    assert np.array_equal(got["token"][sel], ref["token"][sel])
    assert np.array_equal(got["layer_argmax"], ref["layer_argmax"])
    assert np.abs(got["conf"] - ref["conf"]).max() < 1e-4
    assert np.abs(got["entropy"] - ref["entropy"]).max() < 1e-4
    assert got["stats"]["n_committed"] == ref["stats"]["n_committed"] >= 1


def test_sharded_step_reports_a_slice_that_timed_out():
    """A slice whose head kernel issues no loads: its partials call's bounded waits run out and
    the finish on that slice's context reports RPD_ERR_TIMEOUT."""
    case = small_case(611, K=2, N=64, d=256, V=4100, w_std=0.08)
    got = sharded(case, 2, stall_slice=1)
    assert got["stats"]["status"] == rpd.RPD_ERR_TIMEOUT


def test_sharded_step_refuses_lazy_projection():
    case = small_case(612, K=2, N=32, d=256, V=4100, w_std=0.08)
    c = rpd.Rpd(case["d"], 2048, case["K"], case["eps"])
    W = case["W"].to(DEV)
    c.set_head(W[:2048], case["g"].to(DEV))
    c.set_vocab_shard(0, case["V"])
    c.set_projection("lazy")
    part = torch.zeros(case["K"], case["N"], 4, device=DEV)
    with pytest.raises(rpd.RpdError) as e:
        c.step_shard_partials(case["hidden"].to(DEV), case["mask"].to(DEV), part)
    assert e.value.code == rpd.RPD_ERR_UNSUPPORTED
    with pytest.raises(rpd.RpdError):
        c.set_vocab_shard(3000, case["V"])           # slice past the end of the vocabulary
    c.close()
