"""The vocabulary-parallel step's exchange on two gloo ranks (no GPU): the slices of the head,
the rank order of the gathered statistics, and that merging the slices' softmax statistics in
that order gives the statistics of the whole vocabulary (the rule the shard-merge kernel
applies, restated here in numpy)."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_36452_gb300.vocab_parallel import shard_bounds, sharded_step

LOG2E = 1.4426950408889634


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def slice_stats(z):
    """Base-2 softmax statistics of logits z[..., v] (one slice): max, sum 2^(x-m),
    sum 2^(x-m)(x-m), argmax (lowest index), x = z log2 e."""
    x = z * LOG2E
    m = x.max(-1)
    e = np.exp2(x - m[..., None])
    return m, e.sum(-1), (e * (x - m[..., None])).sum(-1), x.argmax(-1)


def merge(parts):
    """Merge slices' (m, s, t, a) in order, lowest index on ties of the max."""
    m, s, t, a = parts[0]
    for m2, s2, t2, a2 in parts[1:]:
        mm = np.maximum(m, m2)
        al, al2 = np.exp2(m - mm), np.exp2(m2 - mm)
        t = al * (t + (m - mm) * s) + al2 * (t2 + (m2 - mm) * s2)
        s = al * s + al2 * s2
        a = np.where(m > m2, a, np.where(m2 > m, a2, np.minimum(a, a2)))
        m = mm
    return m, s, t, a


class FakeShardContext:
    """Stands in for the library on a CPU rank: its "statistics" are those of its slice of a
    logit matrix shared by the test, with global argmax indices."""

    def __init__(self, K, z, v0, v1):
        self.K, self.z, self.v0, self.v1 = K, z, v0, v1
        self.gathered = None

    def step_shard_partials(self, hidden, mask, out):
        m, s, t, a = slice_stats(self.z[..., self.v0:self.v1])
        out.copy_(torch.from_numpy(np.stack([m, s, t, (a + self.v0).astype(np.float64)], -1)))

    def step_shard_finish(self, gathered, mask, tau, budget, out_commit, out_token, out_stats):
        self.gathered = gathered.clone()


def _worker(rank, world, port, V, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    K, N = 3, 5
    z = np.random.default_rng(7).normal(scale=4.0, size=(K, N, V))
    z[1, 2, 300] = z[1, 2, 700] = z[1, 2].max() + 1.0   # a tie across slices: lower index wins
    v0, v1 = shard_bounds(V, world, rank)
    ctx = FakeShardContext(K, z, v0, v1)
    mask = torch.ones(N, dtype=torch.uint8)
    # the exchange works on float32 tensors; here the statistics are carried in float64 views
    partials = torch.empty(K, N, 4, dtype=torch.float64)
    gathered = torch.empty(world, K, N, 4, dtype=torch.float64)
    sharded_step(ctx, None, mask, 0.9, 1.0, None, None, None, partials=partials, gathered=gathered)
    g = ctx.gathered.numpy()
    parts = [(g[r, ..., 0], g[r, ..., 1], g[r, ..., 2], g[r, ..., 3].astype(np.int64)) for r in range(world)]
    m, s, t, a = merge(parts)
    fm, fs, ft, fa = slice_stats(z)
    out[rank] = dict(bounds=(v0, v1), ok_m=np.allclose(m, fm), ok_s=np.allclose(s, fs),
                     ok_t=np.allclose(t, ft), ok_a=bool(np.array_equal(a, fa)),
                     tie=int(a[1, 2]), same=g.tobytes())
    dist.barrier()
    dist.destroy_process_group()


def test_shard_bounds_cover_the_vocabulary_in_aligned_slices():
    for V in (256, 257, 1000, 126464, 152064):
        for world in (1, 2, 3, 8):
            b = [shard_bounds(V, world, r) for r in range(world)]
            assert b[0][0] == 0 and b[-1][1] == V
            assert all(b[r][1] == b[r + 1][0] for r in range(world - 1))
            assert all(lo % 256 == 0 for lo, _ in b)


def test_two_rank_exchange_merges_to_the_whole_vocabulary():
    world, V = 2, 1000
    port = _free_port()
    out = mp.get_context("spawn").Manager().dict()
    mp.spawn(_worker, args=(world, port, V, out), nprocs=world, join=True)
    assert out[0]["bounds"] == (0, 512) and out[1]["bounds"] == (512, V)
    for r in range(world):
        assert out[r]["ok_m"] and out[r]["ok_s"] and out[r]["ok_t"] and out[r]["ok_a"], out[r]
        assert out[r]["tie"] == 300
    assert out[0]["same"] == out[1]["same"]      # every rank holds the same gathered statistics
