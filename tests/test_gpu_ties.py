"""Exact ties on the GPU: the kernels' order against the order include/lookme.h
promises (lowest scene, then lower primitive, then lower token), on tables and
priorities built to tie exactly, for the separate kernels and the fused step
(GPU required).

The parity tests excuse decisions within 1e-3 of the oracle's boundary; these
cases make the tie exact, so the order is the only thing left to check.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from paper_2607_16305_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
PATHS = ["separate", "step"]


def _table(t, cent, keys, vals):
    t.load_scenes(0, keys, vals, centroids=cent)


@pytest.fixture(params=PATHS)
def path(request, monkeypatch):
    monkeypatch.setenv("LOOKME_STEP", "on" if request.param == "step" else "off")
    return request.param


def test_duplicated_centroids_route_to_the_lower_scene(oracle, lookme_lib, path):
    """Scenes 4 and 9 share one centroid (and so every score): every token
    that routes to either goes to scene 4, as the oracle's tie rule says."""
    from paper_2607_16305_gb300 import lookme

    w = W.small("tie_scene", n_tokens=600, n_scenes=16, n_prims=64, d_key=64, d_value=32, top_k=4, keep_ratio=0.25)
    cent, keys, vals = W.full_table(w, device=DEV)
    cent[9] = cent[4]
    q = W.queries(w, DEV)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, device=0) as t:
        _table(t, cent, keys, vals)
        h = W.hidden(w, 0, DEV)
        scene, prim, weight, mask = t.lookup_inject(q, w.top_k, [h], w.keep_ratio)
        s2, _, _ = t.lookup(q, w.top_k)
        torch.cuda.synchronize()
        assert t.device_status() == 0
    gs = scene.cpu().numpy()
    assert (gs == 4).sum() > 0, "no token routed to the tied pair"
    assert (gs != 9).all()
    assert torch.equal(scene, s2)
    r = oracle.route(q.float().cpu().numpy(), cent.float().cpu().numpy())
    tied = np.isin(r["scene"], [4, 9])
    assert (r["scene"][tied] == 4).all() and (gs[tied] == 4).all()


@pytest.mark.parametrize("n_prims", [64, 512])
def test_equal_keys_take_the_lower_primitives(lookme_lib, path, n_prims):
    """Scene 2: every key equal, so every logit ties and the top-k is
    primitives 0..k-1 in that order, each weighted exactly 1/k.  Scene 1: keys
    repeat with period 4, so the top-8 is the eight lowest members of the best
    of the four groups, in increasing order, each weighted 1/8.  With 512
    primitives the logits come from two N-tiles, and the equal keys of the
    second must not displace the lower ones of the first."""
    from paper_2607_16305_gb300 import lookme

    w = W.small(f"tie_prim_{n_prims}", n_tokens=800, n_scenes=4, n_prims=n_prims, d_key=64, d_value=32, top_k=8,
                keep_ratio=0.25)
    cent, keys, vals = W.full_table(w, device=DEV)
    keys[2] = keys[2, 0:1].expand(w.n_prims, -1)
    keys[1] = keys[1, 0:4].repeat(w.n_prims // 4, 1)
    q = W.queries(w, DEV)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, device=0) as t:
        _table(t, cent, keys, vals)
        h = W.hidden(w, 0, DEV)
        scene, prim, weight, _ = t.lookup_inject(q, w.top_k, [h], w.keep_ratio)
        torch.cuda.synchronize()
        assert t.device_status() == 0
    gs, gp, gw = scene.cpu().numpy(), prim.cpu().numpy(), weight.cpu().numpy()
    in2, in1 = gs == 2, gs == 1
    assert in2.sum() > 0 and in1.sum() > 0
    assert (gp[in2] == np.arange(8)).all()
    assert (gw[in2] == np.float32(0.125)).all()
    # scene 1: one residue class mod 4, its eight lowest members in order
    rows = gp[in1]
    j = rows[:, :1]
    assert (rows == j + 4 * np.arange(8)).all()
    assert (gw[in1] == np.float32(0.125)).all()
    # the chosen class is the one with the largest logit (ties: the lower class)
    z = (q[torch.from_numpy(in1).to(DEV)].float() @ keys[1, 0:4].float().T).cpu().numpy()
    best = np.argmax(z, axis=1)
    clear = np.sort(z, axis=1)[:, -1] - np.sort(z, axis=1)[:, -2] > 1e-3
    assert (j[clear, 0] == best[clear]).all()


@pytest.mark.parametrize("n_seg", [1, 3])
def test_equal_priorities_keep_the_lower_tokens(oracle, lookme_lib, path, n_seg):
    """Caller priorities with ten distinct values over 900 tokens (so exact
    ties straddle every segment's r-th place): the kept set is exactly the
    oracle's (larger priority first, then the lower token)."""
    from paper_2607_16305_gb300 import lookme

    w = W.small("tie_gate", n_tokens=900, n_scenes=64, n_prims=64, d_key=64, d_value=32, top_k=4, keep_ratio=0.25)
    cent, keys, vals = W.full_table(w, device=DEV)
    q = W.queries(w, DEV)
    pri = torch.tensor([float((t * 37) % 10) for t in range(w.n_tokens)], dtype=torch.float32, device=DEV)
    seg = [0, 250, 610, 900] if n_seg == 3 else None
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, device=0) as t:
        _table(t, cent, keys, vals)
        h1, h2 = W.hidden(w, 0, DEV), W.hidden(w, 0, DEV)
        _, _, _, m1 = t.lookup_inject(q, w.top_k, [h1], w.keep_ratio, priority=pri, seg_offsets=seg)
        s, p, wt = t.lookup(q, w.top_k)
        m2 = t.inject(s, p, wt, [h2], w.keep_ratio, priority=pri, seg_offsets=seg)
        torch.cuda.synchronize()
        assert t.device_status() == 0
    want = oracle.select(pri.cpu().numpy(), w.keep_ratio, seg)["mask"]
    assert (m1.cpu().numpy() == want).all()
    assert (m2.cpu().numpy() == want).all()
    assert torch.equal(h1, h2)
