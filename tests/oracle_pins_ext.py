"""Pins of the oracle's second part (lookme_oracle_ext.c) to facts outside it.

What pins what
  golden_*          the hand-worked example (tests/golden/paper_level2_example.json):
                    MLP relevance with and without the bf16 hidden rounding,
                    top-T, cos + tanh softmax weights, the gate, the router,
                    SwiGLU, the propagation's orientation, the text lookup
  linear_numpy      x W^T + b against numpy's matmul
  ranker_*          invariants: a zero centroid half makes r independent of
                    the scene; relabelling scenes with their centroids leaves
                    r unchanged; the bf16 hidden rounding moves r by at most
                    |W2| times half an ulp of each hidden value
  level2_brute      top-T equals the T-subset of largest total relevance
                    (enumerated); weights equal scipy's softmax of
                    (1 - scipy cosine distance) + numpy tanh
  gate_expit        g = [scipy.special.expit(logit) > 0.5]
  text_onehot       with E = identity the injected delta spells out the id
  swiglu_special    W_a = W_b = W_o = I gives x^2 expit(x); swapped roles of
                    W_a and W_b give a different, predicted result; a
                    permutation W_o permutes the output
  propagate_special W_p = 0 is the identity (the hot path's reading), W_p = -I
                    gives 0, W_p = I doubles
  router_special    one scale returns it; equal scales return that value for
                    any H; weights sum to 1; a large score margin picks the
                    scale
  combine_onehot    one-hot value rows decode the chosen primitives and weights
"""
from __future__ import annotations

import itertools
import json
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "paper_level2_example.json")


def _g():
    with open(GOLDEN) as f:
        return json.load(f)


def _close(a, b, tol=1e-12, what=""):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    assert a.shape == b.shape, f"{what}: shape {a.shape} vs {b.shape}"
    err = float(np.max(np.abs(a - b))) if a.size else 0.0
    assert err <= tol, f"{what}: max abs error {err} > {tol}"


def check_golden_level2(o):
    g = _g()
    x = g["inputs"]
    scene = np.zeros(1, np.int32)
    for key, rh in (("expected_exact_hidden", False), ("expected_bf16_hidden", True)):
        e = g[key]
        r = o.ranker_relevance(x["v"], scene, x["centroid"], x["W1"], x["b1"], x["W2"], x["b2"], round_hidden=rh)
        _close(r[0], e["r"], 1e-14, f"{key} relevance")
        res = o.ranked_level2(x["v"], scene, np.asarray(x["keys"], np.float32), r, x["top_t"])
        assert res["prim"][0].tolist() == e["prim"], f"{key} primitives {res['prim'][0]}"
        _close(res["weight"][0], e["weight"], 1e-12, f"{key} weights")
        _close(o.ranked_weights_for(x["v"], scene, res["prim"], np.asarray(x["keys"], np.float32), r)[0],
               e["weight"], 1e-12, "weights_for")


def check_golden_gate_router_swiglu_propagate_text(o):
    g = _g()
    gate, logit = o.ska_gate(g["gate"]["delta"], g["gate"]["wg"])
    assert gate.tolist() == g["gate"]["gate"] and np.allclose(logit, g["gate"]["logit"])
    out, att = o.scale_router(g["router"]["H"], g["router"]["Whe"], g["router"]["Rs"])
    _close(att[0], g["router"]["att"], 1e-12, "router weights")
    _close(out[0], g["router"]["out"], 1e-12, "router output")
    I = np.eye(2)
    _close(o.swiglu(g["swiglu"]["x"], I, I, I, round_mid=False)[0], g["swiglu"]["y_exact"], 1e-12, "swiglu")
    _close(o.swiglu(g["swiglu"]["x"], I, I, I, round_mid=True)[0], g["swiglu"]["y_bf16_mid"], 0, "swiglu bf16")
    _close(o.propagate(g["propagate"]["R"], g["propagate"]["Wp"])[0], g["propagate"]["out"], 0, "propagate")
    t = g["text"]
    h = np.zeros((2, len(t["ids"]), 2), np.float32)
    out = o.text_inject(t["E"], t["ids"], np.asarray(t["gate"], np.uint8), h)
    for l in range(2):
        _close(out[l], t["delta"], 0, f"text layer {l}")


def check_linear_numpy(o):
    rng = np.random.default_rng(3)
    x, W, b = rng.normal(size=(5, 7)), rng.normal(size=(4, 7)), rng.normal(size=4)
    x, W, b = (a.astype(np.float32) for a in (x, W, b))
    _close(o.linear(x, W, b), x.astype(np.float64) @ W.astype(np.float64).T + b, 1e-12, "linear")


def _ranker_case(rng, S=5, de=6, dm=7, P=9, N=11):
    v = rng.normal(size=(N, de)).astype(np.float32)
    cent = rng.normal(size=(S, de)).astype(np.float32)
    W1 = rng.normal(size=(dm, 2 * de)).astype(np.float32) * 0.5
    b1 = rng.normal(size=dm).astype(np.float32) * 0.1
    W2 = rng.normal(size=(P, dm)).astype(np.float32) * 0.5
    b2 = rng.normal(size=P).astype(np.float32) * 0.1
    scene = rng.integers(0, S, N).astype(np.int32)
    return v, scene, cent, W1, b1, W2, b2


def check_ranker_invariants(o):
    rng = np.random.default_rng(4)
    v, scene, cent, W1, b1, W2, b2 = _ranker_case(rng)
    de = v.shape[1]
    W1z = W1.copy()
    W1z[:, de:] = 0
    r1 = o.ranker_relevance(v, scene, cent, W1z, b1, W2, b2, round_hidden=False)
    r2 = o.ranker_relevance(v, (scene + 1) % cent.shape[0], cent, W1z, b1, W2, b2, round_hidden=False)
    _close(r1, r2, 0, "zero centroid half")
    perm = rng.permutation(cent.shape[0])
    inv = np.argsort(perm)
    ra = o.ranker_relevance(v, scene, cent, W1, b1, W2, b2, round_hidden=False)
    rb = o.ranker_relevance(v, inv[scene].astype(np.int32), cent[perm], W1, b1, W2, b2, round_hidden=False)
    _close(ra, rb, 0, "relabelled scenes")
    # The scene's centroid matters when its half is not zero.
    rc = o.ranker_relevance(v, (scene + 1) % cent.shape[0], cent, W1, b1, W2, b2, round_hidden=False)
    assert np.abs(ra - rc).max() > 1e-3
    # bf16 hidden rounding: |r_rounded - r| <= sum_m |W2[p,m]| * 2^-9 |h_m| <= sum |W2| * 2^-9 * max|h|
    rr = o.ranker_relevance(v, scene, cent, W1, b1, W2, b2, round_hidden=True)
    pre = np.concatenate([v, cent[scene]], 1).astype(np.float64) @ W1.astype(np.float64).T + b1
    hmax = np.abs(pre).max() + 1.0
    bound = np.abs(W2).sum(1).max() * hmax * 2.0 ** -8
    assert 0 < np.abs(rr - ra).max() <= bound


def check_level2_bruteforce(o):
    from scipy.spatial.distance import cosine
    from scipy.special import softmax

    rng = np.random.default_rng(5)
    N, P, de, T = 40, 6, 5, 3
    v = rng.normal(size=(N, de)).astype(np.float32)
    keys = rng.normal(size=(2, P, de)).astype(np.float32)
    scene = rng.integers(0, 2, N).astype(np.int32)
    r = rng.normal(size=(N, P))
    res = o.ranked_level2(v, scene, keys, r, T)
    for t in range(N):
        best = max(itertools.combinations(range(P), T), key=lambda c: sum(r[t, list(c)]))
        assert sorted(res["prim"][t].tolist()) == sorted(best), f"token {t}"
        assert all(r[t, res["prim"][t][j]] >= r[t, res["prim"][t][j + 1]] for j in range(T - 1))
        s = [1 - cosine(v[t].astype(np.float64), keys[scene[t], p].astype(np.float64)) + np.tanh(r[t, p])
             for p in res["prim"][t]]
        _close(res["weight"][t], softmax(s), 1e-12, "weights vs scipy")
    # Ties: equal relevance keeps the lower primitive.
    rt = np.zeros((1, P))
    assert o.ranked_level2(v[:1], scene[:1], keys, rt, T)["prim"][0].tolist() == [0, 1, 2]


def check_gate_expit(o):
    from scipy.special import expit

    rng = np.random.default_rng(6)
    delta = rng.normal(size=(300, 16)).astype(np.float32)
    wg = rng.normal(size=16).astype(np.float32)
    gate, logit = o.ska_gate(delta, wg)
    _close(logit, delta.astype(np.float64) @ wg.astype(np.float64), 1e-12, "gate logit")
    assert (gate == (expit(logit) > 0.5)).all()
    assert 0 < gate.sum() < 300


def check_text_onehot(o):
    V, d, N = 6, 6, 9
    E = np.eye(V, d, dtype=np.float32)
    ids = np.array([0, 5, -3, 2, 6, 1, 1, 4, 3], np.int32)
    gate = np.array([1, 1, 1, 0, 1, 1, 1, 1, 0], np.uint8)
    h = np.zeros((1, N, d), np.float32)
    out = o.text_inject(E, ids, gate, h)[0]
    for t in range(N):
        want = np.zeros(d)
        if gate[t] and 0 <= ids[t] < V:
            want[ids[t]] = 1
        _close(out[t], want, 0, f"text token {t}")
    # No gate array: every text position.
    out = o.text_inject(E, ids, None, h)[0]
    assert out[3, 2] == 1 and out[8, 3] == 1 and out[2].sum() == 0 and out[4].sum() == 0


def check_swiglu_special(o):
    from scipy.special import expit

    x = np.array([[0.5, -1.5, 2.0]], np.float32)
    I = np.eye(3, dtype=np.float32)
    xd = x.astype(np.float64)
    _close(o.swiglu(x, I, I, I, False), xd ** 2 * expit(xd), 1e-12, "identity")
    _close(o.swiglu(x, I, 2 * I, I, False), 2 * xd ** 2 * expit(xd), 1e-12, "W_b = 2I")
    _close(o.swiglu(x, 2 * I, I, I, False), 2 * xd ** 2 * expit(2 * xd), 1e-12, "W_a = 2I")
    Pm = np.eye(3, dtype=np.float32)[[2, 0, 1]]
    _close(o.swiglu(x, I, I, Pm, False), (xd ** 2 * expit(xd))[:, [2, 0, 1]], 1e-12, "permuted W_o")
    W = np.random.default_rng(7).normal(size=(4, 3)).astype(np.float32)
    _close(o.swiglu(x, W, W, np.zeros((2, 4), np.float32), True), np.zeros((1, 2)), 0, "W_o = 0")


def check_propagate_special(o):
    R = np.random.default_rng(8).normal(size=(4, 5)).astype(np.float32)
    Z, I = np.zeros((5, 5), np.float32), np.eye(5, dtype=np.float32)
    _close(o.propagate(R, Z), R, 0, "W_p = 0")
    _close(o.propagate(R, -I), np.zeros_like(R), 0, "W_p = -I")
    _close(o.propagate(R, I), 2 * R.astype(np.float64), 0, "W_p = I")


def check_router_special(o):
    rng = np.random.default_rng(9)
    N, dh, de = 7, 6, 4
    H = rng.normal(size=(N, dh)).astype(np.float32)
    Whe = rng.normal(size=(dh, de)).astype(np.float32)
    R1 = rng.normal(size=(1, N, de)).astype(np.float32)
    out, att = o.scale_router(H, Whe, R1)
    _close(out, R1[0], 1e-12, "one scale")
    _close(att, np.ones((N, 1)), 1e-12, "one scale weight")
    Rs = np.repeat(R1, 3, axis=0)
    out, att = o.scale_router(H, Whe, Rs)
    _close(out, R1[0], 1e-12, "equal scales")
    _close(att, np.full((N, 3), 1 / 3), 1e-12, "equal scale weights")
    Rs = rng.normal(size=(3, N, de)).astype(np.float32)
    out, att = o.scale_router(H, Whe, Rs)
    _close(att.sum(1), np.ones(N), 1e-12, "weights sum to 1")
    # A scale aligned with q and scaled up wins outright.
    q = H.astype(np.float64) @ Whe.astype(np.float64)
    Rs[1] = (q * 50).astype(np.float32)
    out, att = o.scale_router(H, Whe, Rs)
    assert (att.argmax(1) == 1).all() and att[:, 1].min() > 0.999


def check_combine_onehot(o):
    S, P, T, N = 3, 4, 2, 6
    V = np.zeros((S, P, S * P), np.float32)
    for s in range(S):
        for p in range(P):
            V[s, p, s * P + p] = 1
    rng = np.random.default_rng(10)
    scene = rng.integers(0, S, N).astype(np.int32)
    prim = np.stack([rng.permutation(P)[:T] for _ in range(N)]).astype(np.int32)
    w = rng.dirichlet(np.ones(T), N)
    R = o.combine(scene, prim, w, V)
    for t in range(N):
        want = np.zeros(S * P)
        want[scene[t] * P + prim[t]] = w[t]
        _close(R[t], want, 1e-15, f"combine token {t}")


ALL_CHECKS = [check_golden_level2, check_golden_gate_router_swiglu_propagate_text, check_linear_numpy,
              check_ranker_invariants, check_level2_bruteforce, check_gate_expit, check_text_onehot,
              check_swiglu_special, check_propagate_special, check_router_special, check_combine_onehot]


def failing_checks(o):
    bad = []
    for c in ALL_CHECKS:
        try:
            c(o)
        except (AssertionError, ValueError, IndexError) as e:
            bad.append((c.__name__, str(e)[:200]))
    return bad
