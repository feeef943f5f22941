"""Grids sized for fewer SMs (lookme_set_grids; GPU required).

The settings change only how the steps are spread over CTAs, so every output
must be bit-identical to the default's, on every path they reach: the
tcgen05 and SIMT routing, the one-CTA bucketing with the gate beside it, the
three-launch bucketing of large calls, and the tcgen05 level 2 on fewer CTAs
(its work list then taken from the shared counter by fewer CTAs).  One case
per path is also checked against the oracle."""
from __future__ import annotations

import pytest
import torch

import gpu_harness as H
from paper_2607_16305_gb300 import workloads as W
from test_gpu_parity import run_case

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
# (routing and bucketing SMs, level-2 CTAs)
GRIDS = ((1, 0), (8, 0), (24, 0), (64, 0), (4096, 0), (0, 1), (0, 7), (16, 56), (24, 100), (0, 4096))


def _run_inject(t, w, q, hidden0, grids):
    t.set_grids(*grids)
    hs = [h.clone() for h in hidden0]
    out = t.lookup_inject(q, w.top_k, hs, w.keep_ratio, seg_offsets=w.segment_offsets if w.n_segments > 1 else None)
    torch.cuda.synchronize()
    assert t.device_status() == 0
    return [o.clone() for o in out] + hs


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_grids_lookup_inject_identical(lookme_lib, dtype):
    """Single-image shape (d_v cut to 512): the fused call at every grid size
    against the default grid, bit for bit (scene, primitives, weights, gate
    and every hidden row)."""
    from paper_2607_16305_gb300 import lookme

    w = W.small(f"grid_{dtype}", n_tokens=1024, n_scenes=1024, n_prims=256, d_key=256, d_value=512, top_k=8,
                keep_ratio=0.25, dtype=dtype)
    mu = W.means(w, DEV)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=dtype, device=0) as t:
        H.load_table(t, w, 0, DEV, mu)
        q = W.queries(w, DEV, mu)
        h0 = [W.hidden(w, l, DEV) for l in range(w.layers_per_table)]
        ref = _run_inject(t, w, q, h0, (0, 0))
        for grids in GRIDS:
            got = _run_inject(t, w, q, h0, grids)
            for i, (a, b) in enumerate(zip(ref, got)):
                assert torch.equal(a, b), f"grids {grids}: output {i} differs from the default grids'"


def test_grids_large_call_identical(lookme_lib):
    """A call above the one-CTA bucketing limit (three bucketing launches,
    no gate): lookme_lookup at every grid size against the default."""
    from paper_2607_16305_gb300 import lookme

    w = W.small("grid_large", n_tokens=20000, n_scenes=2048, n_prims=64, d_key=128, d_value=64, top_k=8)
    mu = W.means(w, DEV)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype="bf16", device=0) as t:
        H.load_table(t, w, 0, DEV, mu)
        q = W.queries(w, DEV, mu)
        ref = [o.clone() for o in t.lookup(q, w.top_k)]
        for grids in GRIDS:
            t.set_grids(*grids)
            got = t.lookup(q, w.top_k)
            torch.cuda.synchronize()
            assert t.device_status() == 0
            for i, (a, b) in enumerate(zip(ref, got)):
                assert torch.equal(a, b), f"grids {grids}: output {i} differs from the default grids'"


@pytest.mark.parametrize("dtype,grids", [("bf16", (24, 0)), ("bf16", (1, 3)), ("bf16", (16, 56)), ("fp32", (8, 0))])
def test_grids_against_oracle(oracle, lookme_lib, dtype, grids):
    """The fused call with small grids against the oracle (segments, gate, injection)."""
    w = W.small(f"grid_oracle_{dtype}_{grids[0]}_{grids[1]}", n_tokens=700, n_scenes=300, n_prims=96, d_key=128,
                d_value=128, top_k=8, keep_ratio=0.3, n_segments=3, dtype=dtype)
    run_case(oracle, lookme_lib, w, fused=True, grids=grids)


def test_grids_rejects_negative(lookme_lib):
    from paper_2607_16305_gb300 import lookme

    with lookme.Table(8, 16, 64, 64, device=0) as t:
        with pytest.raises(lookme.LookmeError):
            t.set_grids(-1, 0)
        with pytest.raises(lookme.LookmeError):
            t.set_grids(0, -1)
        t.set_grids(0, 0)
