"""CUDA path against the CPU oracle, through the C ABI (GPU required)."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import gpu_harness as H
from paper_2607_16305_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None


def _bias(w, scale, seed=11):
    if not scale:
        return None
    g = torch.Generator(device=DEV)
    g.manual_seed(seed)
    return (scale * torch.randn(w.n_scenes, generator=g, device=DEV)).float()


def run_case(o, lookme_lib, w, *, sample=None, give_centroids=True, bias_scale=0.0, n_layers=None,
             residency=None, table=0, mu=None, report=None, with_sel=False, fused=False, grids=(0, 0)):
    """with_sel requests the kept-id list, which routes the injection through
    the separate selection kernel; without it short segments take the fused
    select + inject kernel.  fused uses lookme_lookup_inject instead of the
    two calls.  grids = (routing and bucketing SMs, level-2 CTAs) for
    lookme_set_grids (0: the whole device)."""
    from paper_2607_16305_gb300 import lookme

    L = n_layers or w.layers_per_table
    N = w.n_tokens
    seg_off = w.segment_offsets
    bias = _bias(w, bias_scale)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype,
                      residency=residency or w.residency, device=0) as t:
        cent = H.load_table(t, w, table, DEV, mu, give_centroids, bias)
        t.set_grids(*grids)
        q = W.queries(w, DEV, mu)
        hs = [W.hidden(w, l, DEV) for l in range(L)]
        h0 = [h.clone() for h in hs]
        n_sel = sum(int(np.floor((seg_off[i + 1] - seg_off[i]) * w.keep_ratio)) for i in range(len(seg_off) - 1))
        if fused:
            qn = None
            with_sel = False
            scene, prim, weight, mask = t.lookup_inject(q, w.top_k, hs, w.keep_ratio,
                                                        seg_offsets=seg_off if w.n_segments > 1 else None)
        else:
            qn = torch.empty(N, dtype=torch.float32, device=DEV)
            scene, prim, weight = t.lookup(q, w.top_k, qnorm_out=qn)
            sel = torch.empty(max(n_sel, 1), dtype=torch.int32, device=DEV) if with_sel else None
            mask = t.inject(scene, prim, weight, hs, w.keep_ratio,
                            seg_offsets=seg_off if w.n_segments > 1 else None, sel_out=sel)
        torch.cuda.synchronize()
        assert t.device_status() == 0, "a device-side wait timed out"
        stats = t.stats()
    assert stats["n_tokens"] == N

    idx = np.arange(N) if sample is None else np.sort(np.asarray(sample))
    tidx = torch.from_numpy(idx).to(DEV)
    qs = H.f32(q.index_select(0, tidx))
    gscene = scene.index_select(0, tidx).cpu().numpy()
    gprim = prim.index_select(0, tidx).cpu().numpy()
    gw = weight.index_select(0, tidx).cpu().numpy()
    bias_np = None if bias is None else bias.cpu().numpy()
    if give_centroids:
        cent_np = H.f32(cent)
    else:
        _, keys_all, _ = W.full_table(w, table, DEV, mu)
        cent_np = o.centroids(H.f32(keys_all)).astype(np.float32)
        # The table stores the mean in its own dtype: the oracle routes with the exact mean.
        del keys_all

    # ---- lookup
    r = o.route(qs, cent_np, bias_np)
    need = np.union1d(r["scene"], gscene)
    kb, kbos = H.scene_blocks(w, need, table, DEV, mu, cent, "keys")
    res = H.check_lookup(o, qs, cent_np, bias_np, gscene, gprim, gw, kb, kbos, w.top_k, w.n_scenes)

    # ---- mask / selection over all N tokens (priorities are cheap)
    qn_all = o.query_norms(H.f32(q))
    if qn is not None:
        assert np.abs(qn.cpu().numpy() - qn_all).max() <= 1e-4 * max(1.0, qn_all.max())
    gmask = mask.cpu().numpy()
    mask_ties = H.check_mask(o, qn_all, gmask, w.keep_ratio, seg_off)
    if n_sel and with_sel:
        H.check_sel(sel[:n_sel].cpu().numpy(), gmask, w.keep_ratio, seg_off)

    # ---- hidden: untouched rows bit-identical, kept rows against the oracle
    keep_t = mask.bool()
    for l in range(L):
        assert torch.equal(hs[l][~keep_t], h0[l][~keep_t]), f"layer {l}: an unselected row changed"
    rows = np.nonzero(gmask[idx] == 1)[0]
    if rows.size:
        vb, vbos = H.scene_blocks(w, gscene[rows], table, DEV, mu, cent, "values")
        trow = torch.from_numpy(idx[rows]).to(DEV)
        hin = np.stack([H.f32(h.index_select(0, trow)) for h in h0])
        hout = np.stack([H.f32(h.index_select(0, trow)) for h in hs])
        ref = o.inject(gscene[rows], gprim[rows], res["wref"][rows], np.ones(rows.size, np.uint8), vb, hin,
                       vbos, w.n_scenes)
        err = np.abs(hout - ref).max()
        assert err <= H.hidden_tol(w.dtype), f"hidden max abs error {err}"
        res["hidden_err"] = float(err)
    res["mask_ties"] = mask_ties
    res.pop("wref")
    if report is not None:
        report.update(res, stats=stats, scene=gscene)
    print(f"{w.name}: {res} stats={stats}")
    return res


# ------------------------------------------------------------ the workloads
def test_tiny_fp32_full(oracle, lookme_lib):
    run_case(oracle, lookme_lib, W.WORKLOADS["tiny_fp32"])


@pytest.mark.parametrize("mode", ["fused_select", "select_list", "lookup_inject"])
def test_single_image_full(oracle, lookme_lib, mode):
    res = run_case(oracle, lookme_lib, W.WORKLOADS["single_image"], with_sel=mode == "select_list",
                   fused=mode == "lookup_inject")
    assert res["scene_ties"] == 0


@pytest.mark.slow
def test_batched_zipf_sampled(oracle, lookme_lib):
    w = W.WORKLOADS["batched_zipf"]
    rng = np.random.default_rng(0)
    run_case(oracle, lookme_lib, w, sample=rng.choice(w.n_tokens, 4096, replace=False))
    run_case(oracle, lookme_lib, w, sample=rng.choice(w.n_tokens, 1024, replace=False), with_sel=True)
    run_case(oracle, lookme_lib, w, sample=rng.choice(w.n_tokens, 4096, replace=False), fused=True)


@pytest.mark.slow
def test_large_table_sampled(oracle, lookme_lib):
    w = W.WORKLOADS["large_table"]
    rng = np.random.default_rng(1)
    # 4,096 sampled tokens in two calls (the oracle needs each routed scene's
    # 2 MiB key block on the host, so the sample is split to bound that).
    run_case(oracle, lookme_lib, w, sample=rng.choice(w.n_tokens, 2048, replace=False))
    run_case(oracle, lookme_lib, w, sample=rng.choice(w.n_tokens, 2048, replace=False), fused=True)


@pytest.mark.slow
def test_multilayer_host_staged_all_tables(oracle, lookme_lib):
    """Config with 7 tables x 4 layers in pinned host memory: every table, every token."""
    w = W.WORKLOADS["multilayer_host"]
    mu = W.means(w, DEV)
    for table in range(w.n_tables):
        run_case(oracle, lookme_lib, w, table=table, mu=mu, fused=table % 2 == 1)


# ---------------------------------------------------- shapes and edge cases
SMALL_CASES = [
    # name, overrides
    ("s1", dict(n_tokens=1, n_scenes=1, n_prims=1, top_k=1, keep_ratio=1.0)),
    ("s2", dict(n_tokens=300, n_scenes=7, n_prims=3, top_k=3, keep_ratio=0.25, d_key=16, d_value=8)),
    ("s3", dict(n_tokens=129, n_scenes=64, n_prims=64, top_k=64, keep_ratio=0.0, d_key=64, d_value=64)),
    ("s4", dict(n_tokens=257, n_scenes=2, n_prims=7, top_k=1, keep_ratio=1.0, d_key=40, d_value=24)),
    ("s5", dict(n_tokens=200, n_scenes=3, n_prims=64, top_k=4, keep_ratio=0.25, d_key=520, d_value=16)),
    ("s6", dict(n_tokens=1000, n_scenes=300, n_prims=33, top_k=5, keep_ratio=0.3, d_key=128, d_value=40,
                n_segments=7)),
    ("s7", dict(n_tokens=130, n_scenes=1, n_prims=2048, top_k=16, keep_ratio=0.5, d_key=64, d_value=8)),
    ("s8", dict(n_tokens=96, n_scenes=5, n_prims=100, top_k=64, keep_ratio=0.5, d_key=512, d_value=32)),
]


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
@pytest.mark.parametrize("name,kw", SMALL_CASES, ids=[c[0] for c in SMALL_CASES])
def test_small_shapes(oracle, lookme_lib, dtype, name, kw):
    w = W.small(f"{name}_{dtype}", dtype=dtype, **kw)
    run_case(oracle, lookme_lib, w, with_sel=(name in ("s2", "s6", "s8")))


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_routing_bias_and_mean_centroids(oracle, lookme_lib, dtype):
    w = W.small(f"bias_{dtype}", n_tokens=400, n_scenes=50, n_prims=32, d_key=64, d_value=64, top_k=8,
                keep_ratio=0.25, dtype=dtype)
    run_case(oracle, lookme_lib, w, bias_scale=0.05)
    run_case(oracle, lookme_lib, w, give_centroids=False)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_many_layers(oracle, lookme_lib, dtype):
    w = W.small(f"layers_{dtype}", n_tokens=256, n_scenes=16, n_prims=32, d_key=64, d_value=128, top_k=4,
                keep_ratio=0.5, dtype=dtype)
    run_case(oracle, lookme_lib, w, n_layers=5)


def test_host_staged_small(oracle, lookme_lib):
    w = W.small("staged", n_tokens=300, n_scenes=40, n_prims=64, d_key=128, d_value=64, top_k=8, keep_ratio=0.25,
                residency="host")
    run_case(oracle, lookme_lib, w)


def test_empty_and_errors(lookme_lib):
    from paper_2607_16305_gb300 import lookme

    w = W.small("err", n_tokens=16)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, device=0) as t:
        q = W.queries(w, DEV)
        with pytest.raises(lookme.LookmeError) as e:
            t.lookup(q, w.top_k)          # no scene loaded yet
        assert e.value.status == lookme.ERR_STATE
        H.load_table(t, w, 0, DEV)
        with pytest.raises(lookme.LookmeError) as e:
            t.lookup(q, w.n_prims + 1)    # top_k > P
        assert e.value.status == lookme.ERR_INVALID_ARG
        s, p, wt = t.lookup(q[:0], w.top_k)
        assert s.numel() == 0
        s, p, wt = t.lookup(q, w.top_k)
        h = W.hidden(w, 0, DEV)
        with pytest.raises(lookme.LookmeError):
            t.inject(s, p, wt, [h], 1.5)  # keep_ratio > 1
        with pytest.raises(lookme.LookmeError):
            t.inject(s, p, wt, [h], 0.5, seg_offsets=[0, 3, 2, 16])
        t.inject(s, p, wt, [h], 0.5)
        torch.cuda.synchronize()
        assert t.device_status() == 0


def test_graph_capture_replay(oracle, lookme_lib):
    """lookup + inject captured in a CUDA graph after reserve(); replays match an eager run."""
    from paper_2607_16305_gb300 import lookme

    w = W.WORKLOADS["single_image"].scaled(n_scenes=256, n_prims=64, d_value=256)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, device=0) as t:
        H.load_table(t, w, 0, DEV)
        t.reserve(w.n_tokens)
        q = W.queries(w, DEV)
        h = W.hidden(w, 0, DEV)
        h_ref = h.clone()
        s_ref, p_ref, w_ref = t.lookup(q, w.top_k)
        t.inject(s_ref, p_ref, w_ref, [h_ref], w.keep_ratio)
        scene = torch.empty_like(s_ref)
        prim = torch.empty_like(p_ref)
        weight = torch.empty_like(w_ref)
        hg = h.clone()
        stream = torch.cuda.Stream()
        stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(stream):
            t.lookup(q, w.top_k, scene, prim, weight)   # warm-up outside capture
        torch.cuda.current_stream().wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            t.lookup(q, w.top_k, scene, prim, weight)
            t.inject(scene, prim, weight, [hg], w.keep_ratio)
        hg.copy_(h)
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(scene, s_ref) and torch.equal(prim, p_ref) and torch.equal(weight, w_ref)
        assert torch.equal(hg, h_ref)


@pytest.mark.parametrize("case", ["single_image", "s6"])
def test_cuda_core_variants(oracle, lookme_lib, monkeypatch, case):
    """The CUDA-core level-1 and level-2 kernels (selected per table by the
    LOOKME_ROUTE / LOOKME_SCORE switches) against the oracle on bf16 tables."""
    monkeypatch.setenv("LOOKME_ROUTE", "simt")
    monkeypatch.setenv("LOOKME_SCORE", "simt")
    if case == "single_image":
        w = W.WORKLOADS["single_image"]
    else:
        w = W.small("s6_simt", **dict(SMALL_CASES)["s6"])
    run_case(oracle, lookme_lib, w)


@pytest.mark.parametrize("name", ["s1", "s2", "s4", "s5", "s6", "s7", "layers"])
def test_lookup_inject_small_against_oracle(oracle, lookme_lib, name):
    """lookme_lookup_inject on bf16 tables (gate decided beside the
    bucketing, level 2 on the tensor cores, injection of the kept tokens)
    against the oracle, over the small shapes and three layers."""
    kw = dict(SMALL_CASES).get(name) or dict(n_tokens=256, n_scenes=16, n_prims=32, d_key=64, d_value=128, top_k=4,
                                           keep_ratio=0.5)
    w = W.small(f"lif_{name}", dtype="bf16", **kw)
    run_case(oracle, lookme_lib, w, fused=True, n_layers=3 if name == "layers" else None)


@pytest.mark.parametrize("P,dk,top_k", [(512, 256, 8), (384, 256, 8), (600, 128, 4), (1024, 64, 1), (264, 256, 8),
                                          (1024, 512, 16)])
def test_lookup_inject_ntile_topk(oracle, lookme_lib, P, dk, top_k):
    """Several N-tiles of primitives (MMAs of 256 keys each, a partial last one
    included: 600 = 2 x 256 + 88, 264 = 256 + 8) with small top-k, against the
    oracle; 1,024 x 512 with top-16 is the large-table shape, whose level-2
    shared memory is the closest to the per-CTA limit."""
    n_scenes = 20 if dk >= 512 else 60
    w = W.small(f"ntile_{P}_{dk}_{top_k}", n_tokens=1500, n_scenes=n_scenes, n_prims=P, d_key=dk, d_value=128,
                top_k=top_k, keep_ratio=0.25, n_segments=2, dtype="bf16")
    run_case(oracle, lookme_lib, w, fused=True)


@pytest.mark.parametrize("extra", [0, 1])
def test_lookup_inject_many_items(oracle, lookme_lib, extra):
    """32 tokens per SM (and one more) spread over 32,768 scenes, so most
    tokens are alone in their scene and every level-2 CTA takes about 30 work
    items, with the work-list counters against the routed scenes."""
    n_sms = torch.cuda.get_device_properties(0).multi_processor_count
    n = n_sms * 32 + extra
    w = W.small(f"limit_{extra}", dtype="bf16", n_tokens=n, n_scenes=32768, n_prims=16, d_key=32, d_value=16,
                top_k=4, keep_ratio=0.25)
    rep = {}
    run_case(oracle, lookme_lib, w, fused=True, report=rep)
    st = rep["stats"]
    counts = np.bincount(rep["scene"], minlength=w.n_scenes)
    assert st["n_routed_scenes"] == int((counts > 0).sum())
    assert st["n_work_items"] == int(((counts + 7) // 8).sum())


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
@pytest.mark.parametrize("fused", [False, True])
def test_large_call_bucketing(oracle, lookme_lib, dtype, fused):
    """More than 8,192 tokens (the bucketing runs as three launches over all
    SMs) in 64 scenes of ~140 tokens each, so every scene splits into many
    work items, with three segments for the gate."""
    w = W.small(f"bigcall_{dtype}", dtype=dtype, n_tokens=9000, n_scenes=64, n_prims=32, d_key=64, d_value=64,
                top_k=4, keep_ratio=0.25, n_segments=3)
    rep = {}
    run_case(oracle, lookme_lib, w, fused=fused, report=rep)
    counts = np.bincount(rep["scene"], minlength=w.n_scenes)
    assert rep["stats"]["n_work_items"] == int(((counts + 7) // 8).sum())
    assert rep["stats"]["n_routed_scenes"] == int((counts > 0).sum())


def test_large_call_bucketing_host_staged(oracle, lookme_lib):
    """The three-launch bucketing feeding the staging of a pinned-host table
    (the routed-scene list and counts come from its scan)."""
    w = W.small("bigcall_host", n_tokens=9000, n_scenes=96, n_prims=32, d_key=64, d_value=64, top_k=4,
                keep_ratio=0.25, residency="host")
    rep = {}
    run_case(oracle, lookme_lib, w, report=rep)
    counts = np.bincount(rep["scene"], minlength=w.n_scenes)
    assert rep["stats"]["n_routed_scenes"] == int((counts > 0).sum())
    # A fresh table's slot cache is empty: every routed scene's key block is
    # copied (bf16 blocks are stored as 128-row tiles: 128 x 64 x 2 bytes here).
    assert rep["stats"]["staged_hits"] == 0
    assert rep["stats"]["staged_bytes"] == int((counts > 0).sum()) * 128 * 64 * 2


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
@pytest.mark.parametrize("name", ["s2", "s3", "s6", "s8", "layers"])
def test_lookup_inject_matches_separate_calls(lookme_lib, dtype, name):
    """lookme_lookup_inject gives bit-identical results to lookme_lookup +
    lookme_inject on the same inputs."""
    from paper_2607_16305_gb300 import lookme

    kw = dict(SMALL_CASES).get(name) or dict(n_tokens=256, n_scenes=16, n_prims=32, d_key=64, d_value=128, top_k=4,
                                           keep_ratio=0.5)
    w = W.small(f"li_{name}_{dtype}", dtype=dtype, **kw)
    L = 3 if name == "layers" else 1
    seg = w.segment_offsets if w.n_segments > 1 else None
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, device=0) as t:
        H.load_table(t, w, 0, DEV)
        q = W.queries(w, DEV)
        h_a = [W.hidden(w, l, DEV) for l in range(L)]
        h_b = [h.clone() for h in h_a]
        s1, p1, w1 = t.lookup(q, w.top_k)
        m1 = t.inject(s1, p1, w1, h_a, w.keep_ratio, seg_offsets=seg)
        s2, p2, w2, m2 = t.lookup_inject(q, w.top_k, h_b, w.keep_ratio, seg_offsets=seg)
        torch.cuda.synchronize()
        assert t.device_status() == 0
    assert torch.equal(s1, s2) and torch.equal(p1, p2) and torch.equal(w1, w2)
    assert torch.equal(m1, m2)
    for a, b in zip(h_a, h_b):
        assert torch.equal(a, b)

