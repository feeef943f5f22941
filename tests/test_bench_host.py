"""bench.py's host-side arithmetic (no GPU): the roofline numerators it reports.

The level-2 figure is the per-routed-scene unit of the hot-path scope (one scene's
P x d_k key block) times the routed scenes, plus the queries, the outputs and the
token ids; the step adds routing (queries, centroids, bias, scene/norm outputs) and
the injection (k value rows per kept token, one hidden read and write per layer,
the records), counting the queries once.
"""
from __future__ import annotations

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def test_single_image_numerators():
    import bench
    from paper_2607_16305_gb300 import workloads as W

    w = W.WORKLOADS["single_image"]
    ab = bench.algorithmic_bytes(w, n_routed=654, n_sel=256)
    keys = 654 * 256 * 256 * 2            # routed scenes x one scene's bf16 key block
    queries = 1024 * 256 * 2
    outputs = 1024 * 8 * (4 + 4)          # primitive index and weight per selected entry
    assert ab["score"] == keys + queries + outputs + 1024 * 4 == 86_315_008
    route = queries + 1024 * 256 * 2 + 1024 * 4 + 1024 * 8
    inject = 256 * 8 * 2048 * 2 + 2 * 1 * 256 * 2048 * 2 + 256 * 8 * 8
    assert ab["route"] == route and ab["inject"] == inject
    assert ab["step"] == ab["score"] + route + inject + 1024 * 4 * 3 - queries == 97_366_016
    # 14.4 us at the measured copy peak of 6,752.8 GB/s
    assert abs(ab["step"] / 6752.8e9 * 1e6 - 14.42) < 0.01


def test_value_width_changes_values_only():
    from paper_2607_16305_gb300 import workloads as W

    w = W.WORKLOADS["batched_zipf"]
    v = w.scaled(d_value=256)
    assert v.name == w.name and v.d_value == 256
    for f in ("n_tokens", "d_key", "n_scenes", "n_prims", "top_k", "keep_ratio", "zipf", "n_segments", "seed"):
        assert getattr(v, f) == getattr(w, f), f
    # the level-2 numerator does not depend on the value width
    import bench

    assert bench.algorithmic_bytes(v, 2930, 8192)["score"] == bench.algorithmic_bytes(w, 2930, 8192)["score"]
