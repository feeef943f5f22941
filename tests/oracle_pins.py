"""Pins of the CPU oracle to facts outside itself.

Each check raises AssertionError on failure.  They are used twice: as tests of
the oracle (tests/test_oracle_pins.py) and, against deliberately mutated
builds of the oracle, to show that a plausible mistake in any of its steps is
caught by at least one of them.

What pins what
  two_scene_*       hand-worked closed forms (golden fixture) for routing,
                    logits, weights, selection and injection
  tie_*             the tie-break readings (lowest scene, lower primitive,
                    lower token)
  centroid_mean     Level-1 centroid against numpy's mean
  flat_bruteforce   on well-separated data the two-level lookup equals flat
                    top-k over the whole table (the paper's 1-L(sim) case),
                    checked by numpy argsort over every key
  invariants        one scene, k distinct primitives, weights sum to 1,
                    r tokens per segment, unselected rows untouched
  select_lexsort    top-r against numpy.lexsort per segment
  softmax_scipy     weights against scipy.special.softmax of the logits
  onehot_decode     with one-hot value rows the injected delta spells out the
                    scene, primitives and weights the lookup chose
  round_bf16        against torch's float32 -> bfloat16 conversion and
                    hand-picked ties
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "two_scene_example.json")


def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def _close(a, b, tol=1e-9, what=""):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    assert a.shape == b.shape, f"{what}: shape {a.shape} vs {b.shape}"
    err = np.max(np.abs(a - b)) if a.size else 0.0
    assert err <= tol, f"{what}: max abs error {err} > {tol}"


def check_two_scene_example(o):
    g = _golden()
    x, e = g["inputs"], g["expected"]
    q = np.array(x["queries"], np.float32)
    r = o.route(q, np.array(x["centroids"]))
    assert r["scene"].tolist() == e["scene"], r["scene"]
    _close(r["gap1"], e["gap1"], what="gap1")
    _close(r["qnorm"], e["qnorm"], what="qnorm")
    _close(o.query_norms(q), e["qnorm"], what="query_norms")
    p = o.primitives(q, r["scene"], np.array(x["keys"]), x["top_k"])
    assert p["prim"].tolist() == e["prim"], p["prim"]
    _close(p["logit"], e["logit"], what="logit")
    _close(p["weight"], e["weight"], what="weight")
    s = o.select(r["qnorm"], x["keep_ratio"])
    assert s["mask"].tolist() == e["mask"], s["mask"]
    h = o.inject(r["scene"], p["prim"], p["weight"], s["mask"], np.array(x["values"], np.float32),
                 np.array(x["hidden"], np.float32))
    _close(h[0], e["hidden_out"], what="hidden")


def check_two_scene_variants(o):
    g = _golden()
    x, v = g["inputs"], g["variants"]
    q = np.array(x["queries"], np.float32)
    rb = o.route(q, np.array(x["centroids"]), np.array(v["bias"]["bias"]))
    assert rb["scene"].tolist() == v["bias"]["scene"], rb["scene"]
    _close(rb["gap1"][0], v["bias"]["gap1_A"], what="gap1 with bias")
    r = o.route(q, np.array(x["centroids"]))
    p1 = o.primitives(q, r["scene"], np.array(x["keys"]), 1)
    assert p1["prim"].tolist() == v["top1"]["prim"]
    _close(p1["weight"], v["top1"]["weight"], what="top1 weight")
    ru = o.route(q, np.array(v["unnormalised_centroid"]["centroids"]))
    assert ru["scene"].tolist() == v["unnormalised_centroid"]["scene"], ru["scene"]


def check_ties(o):
    # Two identical centroids: the lower scene index wins and the gap is 0.
    q = np.array([[1.0, 2.0, 3.0]], np.float32)
    c = np.array([[1.0, 0.0, 0.0], [3.0, 2.0, 1.0], [3.0, 2.0, 1.0]], np.float32)
    r = o.route(q, c)
    assert r["scene"].tolist() == [1] and r["gap1"][0] == 0.0
    # Equal primitive logits: lower primitive index first.
    keys = np.array([[[1.0, 0.0, 0.0], [0.0, 1.0, 0.0], [0.0, 1.0, 0.0], [0.0, 0.0, 1.0]]], np.float32)
    qq = np.array([[0.0, 1.0, 0.0]], np.float32)
    p = o.primitives(qq, np.array([0]), keys, 3)
    assert p["prim"].tolist() == [[1, 2, 0]], p["prim"]
    assert p["gap_adj"][0] == 0.0
    # Equal priorities: lower token index is kept; r = floor(len * ratio).
    s = o.select(np.array([1.0, 2.0, 2.0, 2.0, 0.5]), 0.5)
    assert s["mask"].tolist() == [0, 1, 1, 0, 0], s["mask"]
    s = o.select(np.array([1.0, 2.0, 3.0]), 0.99)
    assert int(s["mask"].sum()) == 2


def check_centroid_mean(o):
    rng = np.random.default_rng(1)
    keys = rng.standard_normal((5, 7, 9)).astype(np.float32)
    _close(o.centroids(keys), keys.astype(np.float64).mean(axis=1), tol=1e-12, what="centroid")


def _flat_topk(q, keys, k):
    """1-L(sim): top-k over every key of the table by q.k / sqrt(d_k)."""
    S, P, dk = keys.shape
    flat = keys.reshape(S * P, dk).astype(np.float64)
    z = q.astype(np.float64) @ flat.T / math.sqrt(dk)
    rows = np.empty((q.shape[0], k), np.int64)
    for t in range(q.shape[0]):
        order = np.lexsort((np.arange(S * P), -z[t]))
        rows[t] = order[:k]
    return rows, np.take_along_axis(z, rows, axis=1)


def check_flat_bruteforce(o, workloads=None):
    from paper_2607_16305_gb300 import workloads as W

    cases = workloads or [W.WORKLOADS["tiny_fp32"],
                          W.small(n_tokens=200, d_key=16, n_scenes=8, n_prims=8, d_value=8, top_k=3,
                                  dtype="fp32", sigma_q=0.01)]
    for w in cases:
        cent, keys, _ = W.full_table(w)
        q = W.queries(w).numpy()
        keys = keys.numpy()
        r = o.route(q, cent.numpy())
        p = o.primitives(q, r["scene"], keys, w.top_k)
        rows, zf = _flat_topk(q, keys, w.top_k)
        same = (rows // w.n_prims == r["scene"][:, None]).all(axis=1) & (rows % w.n_prims == p["prim"]).all(axis=1)
        assert same.mean() >= 0.999, f"{w.name}: flat == two-level for only {same.mean():.4f} of tokens"
        wf = np.exp(zf - zf[:, :1])
        wf /= wf.sum(axis=1, keepdims=True)
        _close(p["weight"][same], wf[same], tol=1e-12, what=f"{w.name} flat weights")
        _close(p["logit"][same], zf[same], tol=1e-9, what=f"{w.name} flat logits")


def _random_case(seed, N, S, P, dk, dv, k, L=2):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((N, dk)).astype(np.float32)
    c = rng.standard_normal((S, dk)).astype(np.float32)
    keys = rng.standard_normal((S, P, dk)).astype(np.float32)
    vals = rng.standard_normal((S, P, dv)).astype(np.float32)
    hid = rng.standard_normal((L, N, dv)).astype(np.float32)
    bias = (0.1 * rng.standard_normal(S)).astype(np.float32)
    return q, c, keys, vals, hid, bias


def check_invariants(o):
    for seed, (N, S, P, dk, dv, k, ratio, nseg) in enumerate([
        (300, 7, 3, 16, 8, 2, 0.25, 3), (64, 1, 5, 8, 4, 5, 1.0, 1), (50, 3, 64, 32, 16, 1, 0.0, 2),
        (129, 2, 2, 4, 3, 1, 0.5, 4),
    ]):
        q, c, keys, vals, hid, bias = _random_case(seed, N, S, P, dk, dv, k)
        r = o.route(q, c, bias)
        assert ((r["scene"] >= 0) & (r["scene"] < S)).all()
        p = o.primitives(q, r["scene"], keys, k)
        assert ((p["prim"] >= 0) & (p["prim"] < P)).all()
        assert all(len(set(row)) == k for row in p["prim"].tolist())
        assert (p["weight"] > 0).all()
        _close(p["weight"].sum(axis=1), np.ones(N), tol=1e-12, what="sum of weights")
        assert (np.diff(p["logit"], axis=1) <= 0).all(), "logits not descending"
        seg = [i * N // nseg for i in range(nseg + 1)]
        s = o.select(r["qnorm"], ratio, seg)
        for i in range(nseg):
            assert int(s["mask"][seg[i]:seg[i + 1]].sum()) == math.floor((seg[i + 1] - seg[i]) * ratio)
        h = o.inject(r["scene"], p["prim"], p["weight"], s["mask"], vals, hid)
        un = s["mask"] == 0
        assert (h[:, un, :] == hid[:, un, :].astype(np.float64)).all(), "unselected rows changed"
        # The delta of a selected row is a convex combination of its k value rows.
        for t in np.nonzero(s["mask"])[0][:20]:
            rows = vals[r["scene"][t], p["prim"][t]].astype(np.float64)
            for l in range(hid.shape[0]):
                _close(h[l, t] - hid[l, t], p["weight"][t] @ rows, tol=1e-9, what="delta")
            lo, hi = rows.min(axis=0) - 1e-9, rows.max(axis=0) + 1e-9
            d = h[0, t] - hid[0, t]
            assert ((d >= lo) & (d <= hi)).all(), "delta outside the hull of its rows"


def check_select_lexsort(o):
    rng = np.random.default_rng(7)
    for N, nseg, ratio in [(1000, 1, 0.25), (1024, 32, 0.25), (97, 5, 0.3), (10, 2, 1.0), (10, 2, 0.0)]:
        pr = np.round(rng.standard_normal(N), 1)    # many exact ties
        seg = [i * N // nseg for i in range(nseg + 1)]
        s = o.select(pr, ratio, seg)
        want = np.zeros(N, np.uint8)
        for i in range(nseg):
            b, e = seg[i], seg[i + 1]
            r = math.floor((e - b) * ratio)
            order = np.lexsort((np.arange(b, e), -pr[b:e]))
            want[b + order[:r]] = 1
        assert (s["mask"] == want).all()


def check_softmax_scipy(o):
    from scipy.special import softmax

    q, c, keys, _, _, _ = _random_case(11, 80, 4, 40, 24, 4, 6)
    r = o.route(q, c)
    p = o.primitives(q, r["scene"], keys, 6)
    _close(p["weight"], softmax(p["logit"], axis=1), tol=1e-12, what="softmax")
    # The logits are those of the named primitives in the routed scene.
    z = np.einsum("td,tkd->tk", q.astype(np.float64),
                  keys[r["scene"][:, None], p["prim"]].astype(np.float64)) / math.sqrt(24)
    _close(p["logit"], z, tol=1e-9, what="logits of chosen primitives")
    _close(o.weights_for(q, r["scene"], p["prim"], keys), p["weight"], tol=1e-12, what="weights_for")


def check_onehot_decode(o):
    rng = np.random.default_rng(5)
    S, P, dk, k, N = 3, 5, 12, 3, 40
    q = rng.standard_normal((N, dk)).astype(np.float32)
    c = rng.standard_normal((S, dk)).astype(np.float32)
    keys = rng.standard_normal((S, P, dk)).astype(np.float32)
    vals = np.eye(S * P, dtype=np.float32).reshape(S, P, S * P)   # row (s,p) = e_{s*P+p}
    hid = np.zeros((1, N, S * P), np.float32)
    r = o.route(q, c)
    p = o.primitives(q, r["scene"], keys, k)
    mask = np.ones(N, np.uint8)
    h = o.inject(r["scene"], p["prim"], p["weight"], mask, vals, hid)[0]
    for t in range(N):
        nz = np.nonzero(h[t])[0]
        assert set((nz // P).tolist()) == {int(r["scene"][t])}
        assert set((nz % P).tolist()) == set(p["prim"][t].tolist())
        _close(h[t, r["scene"][t] * P + p["prim"][t]], p["weight"][t], tol=1e-15, what="decoded weights")


def check_round_bf16(o):
    import torch

    rng = np.random.default_rng(3)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-30, 30, 20000),
                        rng.standard_normal(2000)]).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = o.round_bf16(x.astype(np.float64))
    assert (got == want).all(), f"{int((got != want).sum())} bf16 roundings differ"
    ties = np.array([1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, -(1 + 2.0 ** -8), 0.0, 2.0 ** -140])
    got = o.round_bf16(ties)
    bits = np.array([0x3F80, 0x3F82, 0xBF80, 0x0000, 0x0000], np.uint16)
    assert (got == bits).all(), [hex(v) for v in got]


ALL_CHECKS = [
    check_two_scene_example, check_two_scene_variants, check_ties, check_centroid_mean,
    check_flat_bruteforce, check_invariants, check_select_lexsort, check_softmax_scipy,
    check_onehot_decode, check_round_bf16,
]


def failing_checks(o):
    """Names of the checks that fail (or crash) for oracle ``o``."""
    bad = []
    for chk in ALL_CHECKS:
        try:
            chk(o)
        except Exception:  # noqa: BLE001 - any failure counts
            bad.append(chk.__name__)
    return bad
