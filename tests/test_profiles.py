"""The committed ncu summaries match the code they describe (no GPU needed).

bench.py reports a kernel's DRAM traffic from its summary under profiles/
only while the hash recorded there matches the kernel's sources, so a stale
capture is never presented as the current kernel's traffic.
"""
from __future__ import annotations

import os
import re
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def test_profiled_traffic_only_from_a_current_capture():
    """bench.py takes a kernel's DRAM traffic from its ncu summary only while the
    source hash recorded there is the hash of the kernel's sources now."""
    import bench

    for name in os.listdir(os.path.join(ROOT, "profiles")):
        txt = open(os.path.join(ROOT, "profiles", name)).read()
        m = re.search(r"source_sha:\s*([0-9a-f]+)", txt)
        k = re.match(r"ncu_(\w+?)_(single_image|batched_zipf|large_table|multilayer_host)\.md$", name)
        if not m or not k or k.group(1) not in bench.KERNEL_SOURCES:
            continue
        traffic = bench.profiled_traffic(k.group(1), k.group(2))
        if m.group(1) == bench.kernel_source_sha(k.group(1)):
            assert traffic and traffic > 0, name
        else:
            assert traffic is None, name


def test_profiles_are_short_text_with_their_command():
    for name in os.listdir(os.path.join(ROOT, "profiles")):
        path = os.path.join(ROOT, "profiles", name)
        assert name.endswith((".md", ".txt")), name
        assert os.path.getsize(path) < 16384, name
        assert "ncu " in open(path).read(), f"{name} does not give the command that made it"
