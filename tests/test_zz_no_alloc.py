"""lookme_route_scenes_static: level-1 routing for callers that cannot allocate.

Some callers of this library cannot allocate device memory at the moment they
route tokens (their device memory belongs to another allocator, or they must
not risk the synchronisation an allocation can cause).  The allocation-free
entry point keeps its scratch in fixed arrays inside the library.  This test
calls it through the C ABI twice in a row, with different token counts, and
checks that it assigns exactly the scenes lookme_lookup assigns (scene ids are
integers: bit-exact), for a bf16 table (tensor-core routing) and an fp32 table
(CUDA-core routing); it also checks the size limit is enforced up front.

The file name sorts last so that a run stopping at its first failure has
already run every other test.
"""
import ctypes

import pytest
import torch

from paper_2607_16305_gb300 import lookme
from paper_2607_16305_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _route_static(lib, table, q, out):
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return lib.lookme_route_scenes_static(table.handle, ctypes.c_void_p(q.data_ptr()), q.shape[0],
                                          ctypes.c_void_p(out.data_ptr()), stream)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_route_static_matches_lookup(dtype):
    lib = lookme.load()
    dev = torch.device("cuda", 0)
    w = W.small(f"static_{dtype}", n_tokens=1500, n_scenes=300, n_prims=16, d_key=128, d_value=16, top_k=4,
                keep_ratio=0.25, dtype=dtype)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=dtype, device=0) as t:
        cent = W.centroids(w, 0, dev)
        for c in range(w.n_chunks):
            k, v = W.table_chunk(w, 0, c, dev, None, cent)
            s0 = c * w.scenes_per_chunk
            t.load_scenes(s0, k, v, centroids=cent[s0:s0 + k.shape[0]])
        q_all = W.queries(w, dev)
        # Two calls in a row: the second is smaller, so it runs on top of the
        # first call's leftovers in the shared scratch.
        batches = [q_all, q_all[200:900].contiguous()]
        refs = [t.lookup(q, w.top_k)[0].clone() for q in batches]
        outs = [torch.full((q.shape[0],), -1, dtype=torch.int32, device=dev) for q in batches]
        for q, out in zip(batches, outs):
            assert _route_static(lib, t, q, out) == lookme.OK, lib.lookme_last_error()
        torch.cuda.synchronize()
        for ref, out in zip(refs, outs):
            assert torch.equal(out, ref)
        assert t.device_status() == 0

        too_many = lookme.ROUTE_STATIC_MAX_TOKENS + 1
        assert _route_static_n(lib, t, q_all, outs[0], too_many) == lookme.ERR_INVALID_ARG
        assert b"fixed scratch" in lib.lookme_last_error()


def _route_static_n(lib, table, q, out, n):
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return lib.lookme_route_scenes_static(table.handle, ctypes.c_void_p(q.data_ptr()), n,
                                          ctypes.c_void_p(out.data_ptr()), stream)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_route_static_takes_no_device_memory(dtype):
    """On a table that has never looked anything up (no per-call scratch
    reserved), routing through the allocation-free entry point leaves the
    device's free memory unchanged: after one warm-up call (which may load the
    kernels' code), two more calls allocate nothing."""
    lib = lookme.load()
    dev = torch.device("cuda", 0)
    w = W.small(f"static_mem_{dtype}", n_tokens=4000, n_scenes=200, n_prims=16, d_key=64, d_value=16, top_k=4,
                keep_ratio=0.25, dtype=dtype)
    with lookme.Table(w.n_scenes, w.n_prims, w.d_key, w.d_value, dtype=dtype, device=0) as t:
        cent = W.centroids(w, 0, dev)
        for c in range(w.n_chunks):
            k, v = W.table_chunk(w, 0, c, dev, None, cent)
            s0 = c * w.scenes_per_chunk
            t.load_scenes(s0, k, v, centroids=cent[s0:s0 + k.shape[0]])
        q = W.queries(w, dev)
        out = torch.full((q.shape[0],), -1, dtype=torch.int32, device=dev)
        assert _route_static(lib, t, q, out) == lookme.OK, lib.lookme_last_error()
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info(dev)[0]
        for _ in range(2):
            assert _route_static(lib, t, q, out) == lookme.OK, lib.lookme_last_error()
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info(dev)[0] >= free0
        assert int(out.min()) >= 0 and int(out.max()) < w.n_scenes
        assert t.device_status() == 0
