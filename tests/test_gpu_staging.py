"""Pinned-host tables: the HBM slot cache kept across calls (GPU required).

Every call is checked against the oracle; the cache statistics are checked
against what the routed-scene lists imply (hits are the scenes a call shares
with what the cache held, copies are the rest)."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import gpu_harness as H
from paper_2607_16305_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None


def _check(o, w, t, q, cent, mu=None, table=0):
    scene, prim, weight = t.lookup(q, w.top_k)
    torch.cuda.synchronize()
    assert t.device_status() == 0, "device status set (timeout or staging overflow)"
    qs = H.f32(q)
    gscene = scene.cpu().numpy()
    r = o.route(qs, H.f32(cent))
    need = np.union1d(r["scene"], gscene)
    kb, kbos = H.scene_blocks(w, need, table, DEV, mu, cent, "keys")
    H.check_lookup(o, qs, H.f32(cent), None, gscene, prim.cpu().numpy(), weight.cpu().numpy(), kb, kbos,
                   w.top_k, w.n_scenes)
    return gscene, prim.clone(), weight.clone(), t.stats()


def _queries_on(w, scenes, n, seed, mu):
    """n queries drawn around the means of the given scenes."""
    g = torch.Generator(device=DEV)
    g.manual_seed(seed)
    pick = torch.tensor(scenes, device=DEV)[torch.randint(len(scenes), (n,), generator=g, device=DEV)]
    q = mu[pick] + w.sigma_q * torch.randn(n, w.d_key, generator=g, device=DEV)
    return q.to(w.torch_dtype).contiguous()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_slot_cache_hits_and_invalidate(oracle, lookme_lib, dtype):
    from paper_2607_16305_gb300 import lookme

    w = W.small(f"cache_{dtype}", n_tokens=300, n_scenes=40, n_prims=64, d_key=128, d_value=64, top_k=8,
                keep_ratio=0.25, residency="host", dtype=dtype)
    mu = W.means(w, DEV)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=dtype, residency="host", device=0) as t:
        cent = H.load_table(t, w, 0, DEV, mu)
        q = W.queries(w, DEV, mu)
        s1, p1, w1, st1 = _check(oracle, w, t, q, cent, mu)
        routed = len(np.unique(s1))
        assert st1["staged_hits"] == 0 and st1["staged_bytes"] > 0
        block = st1["staged_bytes"] // routed
        assert st1["staged_bytes"] == routed * block
        # The same queries again: every routed scene is a hit, nothing is copied.
        s2, p2, w2, st2 = _check(oracle, w, t, q, cent, mu)
        assert st2["staged_hits"] == routed and st2["staged_bytes"] == 0
        assert (s1 == s2).all() and torch.equal(p1, p2) and torch.equal(w1, w2)
        # Queries on a different scene subset: hits are the shared scenes.
        q3 = _queries_on(w, list(range(0, 40, 3)), 200, 5, mu)
        s3, _, _, st3 = _check(oracle, w, t, q3, cent, mu)
        shared = np.intersect1d(np.unique(s3), np.unique(s1)).size
        assert st3["staged_hits"] == shared
        assert st3["staged_bytes"] == (np.unique(s3).size - shared) * block
        # Emptied cache: everything is copied again.
        t.stage_invalidate()
        _, _, _, st4 = _check(oracle, w, t, q3, cent, mu)
        assert st4["staged_hits"] == 0 and st4["staged_bytes"] == np.unique(s3).size * block


class ClockCache:
    """The slot policy the library documents: routed scenes (in increasing
    scene order) that the cache holds are hits; each miss takes, in order, the
    next slot from the clock hand that no routed scene of the call uses."""

    def __init__(self, n_slots):
        self.scene = [-1] * n_slots
        self.stamp = [0] * n_slots
        self.hand = 0
        self.epoch = 0

    def call(self, routed):
        self.epoch += 1
        where = {s: j for j, s in enumerate(self.scene) if s >= 0}
        misses = []
        for s in sorted(routed):
            if s in where:
                self.stamp[where[s]] = self.epoch
            else:
                misses.append(s)
        n = len(self.scene)
        victims = [(self.hand + k) % n for k in range(n) if self.stamp[(self.hand + k) % n] != self.epoch]
        for s, j in zip(misses, victims):
            self.scene[j] = s
            self.stamp[j] = self.epoch
        if misses:
            self.hand = (victims[len(misses) - 1] + 1) % n
        return len(routed) - len(misses), len(misses)


def test_slot_cache_eviction(oracle, lookme_lib):
    """A cache of 24 slots for 96 scenes: calls of 24 tokens on moving scene
    windows evict earlier scenes.  Every call matches the oracle, and the hit
    and copy counts match the documented clock policy."""
    from paper_2607_16305_gb300 import lookme

    w = W.small("evict", n_tokens=24, n_scenes=96, n_prims=32, d_key=64, d_value=32, top_k=4, keep_ratio=0.25,
                residency="host")
    mu = W.means(w, DEV)
    model = ClockCache(24)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype="bf16", residency="host", device=0,
                      stage_slots=24) as t:
        cent = H.load_table(t, w, 0, DEV, mu)
        block = None
        for i, lo in enumerate([0, 8, 16, 40, 0, 70, 72, 74, 90, 0, 8]):
            scenes = [(lo + j) % 96 for j in range(16)]
            q = _queries_on(w, scenes, 24, 100 + i, mu)
            gs, _, _, st = _check(oracle, w, t, q, cent, mu)
            hits, copies = model.call(set(np.unique(gs).tolist()))
            assert st["staged_hits"] == hits, (i, st, hits)
            if copies:
                block = block or st["staged_bytes"] // copies
                assert st["staged_bytes"] == copies * block, (i, st, copies)
            else:
                assert st["staged_bytes"] == 0


def test_staged_call_under_graph_capture(oracle, lookme_lib):
    """The staging fork and join are captured with the call; replays give the same results."""
    from paper_2607_16305_gb300 import lookme

    w = W.small("cap_host", n_tokens=256, n_scenes=48, n_prims=64, d_key=128, d_value=64, top_k=8,
                keep_ratio=0.25, residency="host")
    mu = W.means(w, DEV)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype="bf16", residency="host", device=0,
                      max_tokens=w.n_tokens) as t:
        cent = H.load_table(t, w, 0, DEV, mu)
        q = W.queries(w, DEV, mu)
        scene = torch.empty(w.n_tokens, dtype=torch.int32, device=DEV)
        prim = torch.empty(w.n_tokens, w.top_k, dtype=torch.int32, device=DEV)
        weight = torch.empty(w.n_tokens, w.top_k, dtype=torch.float32, device=DEV)
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            t.lookup(q, w.top_k, scene_out=scene, prim_out=prim, weight_out=weight)
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        ref = (scene.clone(), prim.clone(), weight.clone())
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            t.lookup(q, w.top_k, scene_out=scene, prim_out=prim, weight_out=weight)
        for _ in range(3):
            t.stage_invalidate()
            scene.zero_()
            g.replay()
            torch.cuda.synchronize()
            assert torch.equal(scene, ref[0]) and torch.equal(prim, ref[1]) and torch.equal(weight, ref[2])
        assert t.device_status() == 0
