"""The fused step kernel (LOOKME_STEP=on): a whole lookme_lookup_inject or
lookme_lookup call as one launch -- routing, bucketing, level 2, the gate and
the injection -- against the CPU oracle, and bit for bit against the separate
kernels on the same inputs (GPU required).

Each case first checks that the call really ran as one launch, so that a
shape the fused kernel declines (it falls back to the separate kernels) cannot
pass unnoticed.
"""
from __future__ import annotations

import pytest
import torch

import gpu_harness as H
from paper_2607_16305_gb300 import workloads as W
from test_gpu_parity import DEV, run_case

pytestmark = pytest.mark.gpu

STEP_CASES = {
    # name: (workload overrides, run_case options)
    "single_image": (None, {}),
    "segments": (dict(n_tokens=1000, n_scenes=300, n_prims=64, d_key=128, d_value=40, top_k=5, keep_ratio=0.3,
                      n_segments=7), {}),
    "layers": (dict(n_tokens=256, n_scenes=16, n_prims=32, d_key=64, d_value=128, top_k=4, keep_ratio=0.5),
               {"n_layers": 3}),
    "bias": (dict(n_tokens=400, n_scenes=50, n_prims=32, d_key=64, d_value=64, top_k=8, keep_ratio=0.25),
             {"bias_scale": 0.05}),
    "mean_centroids": (dict(n_tokens=400, n_scenes=50, n_prims=32, d_key=64, d_value=64, top_k=8, keep_ratio=0.25),
                       {"give_centroids": False}),
    "one_token": (dict(n_tokens=1, n_scenes=3, n_prims=16, d_key=32, d_value=16, top_k=4, keep_ratio=1.0), {}),
    # ~500 tokens per scene: one CTA owns ~63 items (past the on-chip item and
    # tile caches) and ~250 kept tokens (past the kept-token queue).
    "hot_scene": (dict(n_tokens=2000, n_scenes=4, n_prims=256, d_key=64, d_value=64, top_k=8, keep_ratio=0.5), {}),
}


def _workload(name):
    kw, _ = STEP_CASES[name]
    if kw is None:
        return W.WORKLOADS[name]
    return W.small(f"step_{name}", dtype="bf16", **kw)


def _one_launch(w):
    """lookup_inject on a fresh table counts as one library launch."""
    from paper_2607_16305_gb300 import lookme

    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, device=0) as t:
        H.load_table(t, w, 0, DEV)
        q = W.queries(w, DEV)
        h = W.hidden(w, 0, DEV)
        t.reserve(w.n_tokens)
        c0 = t.launch_count()
        t.lookup_inject(q, w.top_k, [h], w.keep_ratio, seg_offsets=w.segment_offsets if w.n_segments > 1 else None)
        torch.cuda.synchronize()
        return t.launch_count() - c0


@pytest.mark.parametrize("name", list(STEP_CASES))
def test_step_against_oracle(oracle, lookme_lib, monkeypatch, name):
    monkeypatch.setenv("LOOKME_STEP", "on")
    w = _workload(name)
    assert _one_launch(w) == 1, "the fused step did not take this call"
    run_case(oracle, lookme_lib, w, fused=True, **STEP_CASES[name][1])


def _run_path(w, step, layers=1):
    from paper_2607_16305_gb300 import lookme

    seg = w.segment_offsets if w.n_segments > 1 else None
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, device=0) as t:
        H.load_table(t, w, 0, DEV)
        q = W.queries(w, DEV)
        hs = [W.hidden(w, l, DEV) for l in range(layers)]
        s, p, wt, m = t.lookup_inject(q, w.top_k, hs, w.keep_ratio, seg_offsets=seg)
        # and the lookup alone, then the injection kernel on its results
        hs2 = [W.hidden(w, l, DEV) for l in range(layers)]
        s2, p2, wt2 = t.lookup(q, w.top_k)
        m2 = t.inject(s2, p2, wt2, hs2, w.keep_ratio, seg_offsets=seg)
        torch.cuda.synchronize()
        assert t.device_status() == 0
    return (s, p, wt, m, hs), (s2, p2, wt2, m2, hs2)


@pytest.mark.parametrize("name", ["single_image", "segments", "layers", "hot_scene"])
def test_step_bit_identical_to_separate_kernels(lookme_lib, monkeypatch, name):
    """The fused step and the separate kernels give the same bits: scenes,
    primitives (same order), weights, mask and hidden states; and the fused
    lookup followed by the injection kernel gives what the fused lookup_inject
    gives."""
    w = _workload(name)
    layers = STEP_CASES[name][1].get("n_layers", 1)
    monkeypatch.setenv("LOOKME_STEP", "off")
    ref, _ = _run_path(w, False, layers)
    monkeypatch.setenv("LOOKME_STEP", "on")
    fused, fused_then_inject = _run_path(w, True, layers)
    for a, b in zip(ref[:4], fused[:4]):
        assert torch.equal(a, b)
    for a, b in zip(ref[4], fused[4]):
        assert torch.equal(a, b)
    for a, b in zip(fused[:4], fused_then_inject[:4]):
        assert torch.equal(a, b)
    for a, b in zip(fused[4], fused_then_inject[4]):
        assert torch.equal(a, b)


def test_step_repeated_calls(lookme_lib, monkeypatch):
    """Calls alternate the fused kernel's argmax-key and barrier buffers by
    parity; ten calls in a row (different token counts) all match the
    separate kernels."""
    from paper_2607_16305_gb300 import lookme

    monkeypatch.setenv("LOOKME_STEP", "on")
    w = W.small("step_rep", dtype="bf16", n_tokens=700, n_scenes=120, n_prims=64, d_key=64, d_value=32, top_k=4,
                keep_ratio=0.25)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, device=0) as t:
        H.load_table(t, w, 0, DEV)
        q = W.queries(w, DEV)
        outs = []
        for i in range(10):
            n = [700, 333, 1, 700, 512][i % 5]
            outs.append([x.clone() for x in t.lookup(q[:n], w.top_k)])
        torch.cuda.synchronize()
        assert t.device_status() == 0
    monkeypatch.setenv("LOOKME_STEP", "off")
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=w.dtype, device=0) as t:
        H.load_table(t, w, 0, DEV)
        q = W.queries(w, DEV)
        for i in range(10):
            n = [700, 333, 1, 700, 512][i % 5]
            ref = t.lookup(q[:n], w.top_k)
            for a, b in zip(outs[i], ref):
                assert torch.equal(a, b), f"call {i}"
