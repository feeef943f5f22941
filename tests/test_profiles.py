"""The committed ncu summaries match the code they describe (no GPU needed).

bench.py reports the level-2 kernel's DRAM traffic from
profiles/ncu_score_single_image.md only while the hash recorded there matches
the kernel source; a kernel change without a new capture would silently turn
the figure into null.
"""
from __future__ import annotations

import os
import re
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def test_score_profile_matches_the_kernel_source():
    import bench

    txt = open(os.path.join(ROOT, "profiles", "ncu_score_single_image.md")).read()
    m = re.search(r"source_sha:\s*([0-9a-f]+)", txt)
    assert m, "the summary records no source hash"
    assert m.group(1) == bench.kernel_source_sha(), "k_score_tc.cu changed since the ncu capture: capture it again"
    assert bench.profiled_traffic("single_image") > 0


def test_profiles_are_short_text_with_their_command():
    for name in os.listdir(os.path.join(ROOT, "profiles")):
        path = os.path.join(ROOT, "profiles", name)
        assert name.endswith((".md", ".txt")), name
        assert os.path.getsize(path) < 16384, name
        assert "ncu " in open(path).read(), f"{name} does not give the command that made it"
