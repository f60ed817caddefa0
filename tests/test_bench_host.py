"""Host-side pieces of bench.py that need no GPU: the launch count it reports and the
traffic table keyed on the head kernels' sources."""
import argparse

import bench


def args(projection="all"):
    return argparse.Namespace(projection=projection)


def test_launches_per_step():
    one = {"K": 4, "N": 256, "B": 1}
    # compaction, gather, head, merge with the score/commit of the single canvas
    assert bench.launches_per_step(one, args("all")) == 4
    # lazy: band selection and a second gather/head/merge pass
    assert bench.launches_per_step(one, args("lazy")) == 8
    assert bench.launches_per_step(one, args("auto")) == 8
    batched = {"K": 6, "N": 1024, "B": 8}
    assert bench.launches_per_step(batched, args("all")) == 5      # separate score/commit
    long_canvas = {"K": 2, "N": 4096, "B": 1}
    assert bench.launches_per_step(long_canvas, args("all")) == 5
    tiny = {"K": 1, "N": 64, "B": 1}                                # auto never goes lazy at K = 1
    assert bench.launches_per_step(tiny, args("auto")) == 4


def test_traffic_table_is_from_one_capture_of_the_sources():
    hashes = {h for (_, h) in bench.HEAD_TRAFFIC}
    assert len(hashes) == 1
    assert all(v > 1e9 for v in bench.HEAD_TRAFFIC.values())
    assert len(bench.head_source_hash()) == 16
