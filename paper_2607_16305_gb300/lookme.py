"""Thin Python binding of liblookme.so (the C ABI in include/lookme.h).

Only argument marshalling happens here: torch tensors are checked for device,
dtype and contiguity and passed as raw pointers together with the current CUDA
stream.  Every step of the lookup and injection runs in the library's CUDA
kernels.  If the compiled library is missing, ``load()`` raises; there is no
fallback of any kind.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "liblookme.so")

OK, ERR_INVALID_ARG, ERR_CUDA, ERR_OOM, ERR_TIMEOUT, ERR_STATE, ERR_UNSUPPORTED = range(7)
BF16, FP32 = 0, 1
RES_DEVICE, RES_HOST_STAGED = 0, 1
MAX_TOP_K, MAX_LAYERS, MAX_SEGMENTS = 64, 64, 1024
ROUTE_STATIC_MAX_TOKENS = 65536

EXPORTS = [
    "lookme_table_create", "lookme_table_destroy", "lookme_load_scenes", "lookme_lookup", "lookme_inject",
    "lookme_reserve", "lookme_stage_invalidate", "lookme_set_grids", "lookme_last_lookup_stats", "lookme_device_status", "lookme_launch_count",
    "lookme_trace_enable", "lookme_trace_read", "lookme_kernel_name", "lookme_status_string",
    "lookme_last_error", "lookme_route_scenes_static", "lookme_lookup_inject",
    "lookme_set_ranker", "lookme_lookup_ranked", "lookme_ska_gate", "lookme_inject_gated", "lookme_combine",
    "lookme_text_inject", "lookme_project", "lookme_scale_router", "lookme_fusion_create", "lookme_fusion_load",
    "lookme_fusion_apply", "lookme_fusion_status", "lookme_fusion_destroy",
]


class LookmeError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"lookme status {status}: {message}")
        self.status = status


class TableDesc(ctypes.Structure):
    _fields_ = [
        ("n_scenes", ctypes.c_int64), ("n_prims", ctypes.c_int64), ("d_key", ctypes.c_int64),
        ("d_value", ctypes.c_int64), ("dtype", ctypes.c_int32), ("residency", ctypes.c_int32),
        ("device", ctypes.c_int32), ("reserved0", ctypes.c_int32), ("max_tokens", ctypes.c_int64),
        ("stage_slots", ctypes.c_int64),
    ]


class LookupStats(ctypes.Structure):
    _fields_ = [("n_tokens", ctypes.c_int64), ("n_routed_scenes", ctypes.c_int32),
                ("n_work_items", ctypes.c_int32), ("staged_bytes", ctypes.c_int64),
                ("staged_hits", ctypes.c_int32), ("reserved0", ctypes.c_int32)]


class TraceRecord(ctypes.Structure):
    _fields_ = [("kernel", ctypes.c_int32), ("ms", ctypes.c_float)]


_lib = None


def load(path: str = LIB_PATH):
    """Load liblookme.so (built by build.py); raises if it is not there."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise LookmeError(-1, f"{path} is missing: build it with paper_2607_16305_gb300/build.py")
    lib = ctypes.CDLL(path)
    P, I32, I64, D = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
    sig = {
        "lookme_table_create": ([ctypes.POINTER(TableDesc), ctypes.POINTER(P)], I32),
        "lookme_table_destroy": ([P], I32),
        "lookme_load_scenes": ([P, I64, I64, P, P, P, P, I32, P], I32),
        "lookme_lookup": ([P, P, I64, I32, P, P, P, P, P], I32),
        "lookme_inject": ([P, P, P, P, I64, I32, P, P, I32, D, P, I32, P, P, P], I32),
        "lookme_reserve": ([P, I64], I32),
        "lookme_stage_invalidate": ([P, P], I32),
        "lookme_set_grids": ([P, I32, I32], I32),
        "lookme_last_lookup_stats": ([P, ctypes.POINTER(LookupStats), P], I32),
        "lookme_device_status": ([P, ctypes.POINTER(ctypes.c_uint32), I32, P], I32),
        "lookme_launch_count": ([P], ctypes.c_uint64),
        "lookme_trace_enable": ([P, I32], I32),
        "lookme_trace_read": ([P, ctypes.POINTER(TraceRecord), I32, ctypes.POINTER(I32)], I32),
        "lookme_kernel_name": ([I32], ctypes.c_char_p),
        "lookme_status_string": ([I32], ctypes.c_char_p),
        "lookme_last_error": ([], ctypes.c_char_p),
        "lookme_route_scenes_static": ([P, P, I64, P, P], I32),
        "lookme_lookup_inject": ([P, P, I64, I32, P, P, I32, D, P, I32, P, P, P, P, P], I32),
        "lookme_set_ranker": ([P, I64, P, P, P, P, P], I32),
        "lookme_lookup_ranked": ([P, P, I64, I32, P, P, P, P], I32),
        "lookme_ska_gate": ([P, P, I64, I64, I32, P, P, P], I32),
        "lookme_inject_gated": ([P, P, P, P, I64, I32, P, P, I32, P], I32),
        "lookme_combine": ([P, P, P, P, I64, I32, P, I64, P, P], I32),
        "lookme_text_inject": ([P, I64, I64, I32, P, P, I64, P, I32, P], I32),
        "lookme_project": ([P, P, P, I64, I64, I64, P, P], I32),
        "lookme_scale_router": ([P, P, P, I32, I64, I64, I64, P, P, P, P], I32),
        "lookme_fusion_create": ([I32, I64, I64, I64, I32, I64, ctypes.POINTER(P)], I32),
        "lookme_fusion_load": ([P, I32, P, P, P, P, P], I32),
        "lookme_fusion_apply": ([P, P, P, I64, P, P], I32),
        "lookme_fusion_status": ([P, ctypes.POINTER(ctypes.c_uint32), P], I32),
        "lookme_fusion_destroy": ([P], I32),
    }
    for name, (argtypes, restype) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = argtypes
        fn.restype = restype
    _lib = lib
    return lib


def _check(status: int):
    if status != OK:
        msg = _lib.lookme_last_error().decode(errors="replace")
        raise LookmeError(status, msg)


def _stream(stream, device):
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


_DT = {"bf16": (BF16, torch.bfloat16), "fp32": (FP32, torch.float32)}


class Table:
    """A LookME two-level table (keys [S, P, d_key], values [S, P, d_value]) on one GPU."""

    def __init__(self, n_scenes, n_prims, d_key, d_value, dtype="bf16", residency="device", device=0,
                 max_tokens=0, stage_slots=0):
        self.lib = load()
        self.dtype_code, self.torch_dtype = _DT[dtype]
        self.dtype = dtype
        self.device = torch.device("cuda", device) if isinstance(device, int) else torch.device(device)
        self.shape = (n_scenes, n_prims, d_key, d_value)
        desc = TableDesc(n_scenes, n_prims, d_key, d_value, self.dtype_code,
                         RES_HOST_STAGED if residency == "host" else RES_DEVICE,
                         self.device.index or 0, 0, max_tokens, stage_slots)
        h = ctypes.c_void_p()
        _check(self.lib.lookme_table_create(ctypes.byref(desc), ctypes.byref(h)))
        self.handle = h

    # ------------------------------------------------------------------ life
    def close(self):
        if getattr(self, "handle", None):
            self.lib.lookme_table_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:  # noqa: BLE001 - interpreter shutdown
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # ----------------------------------------------------------------- calls
    def _tensor(self, t, name, dtype=None, device=True):
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
        if dtype is not None and t.dtype != dtype:
            raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
        if device and t.device != self.device:
            raise ValueError(f"{name} must be on {self.device}")
        return t

    def load_scenes(self, scene_begin, keys, values, centroids=None, bias=None, stream=None):
        """Copy scenes [scene_begin, scene_begin + keys.shape[0]) from device or host tensors."""
        n = keys.shape[0]
        on_dev = keys.is_cuda
        for name, t in (("keys", keys), ("values", values), ("centroids", centroids)):
            if t is not None:
                self._tensor(t, name, self.torch_dtype, device=False)
        if bias is not None:
            self._tensor(bias, "bias", torch.float32, device=False)
        S, P, dk, dv = self.shape
        if tuple(keys.shape) != (n, P, dk) or tuple(values.shape) != (n, P, dv):
            raise ValueError("keys/values shape mismatch")
        if centroids is not None and tuple(centroids.shape) != (n, dk):
            raise ValueError("centroids shape mismatch")
        _check(self.lib.lookme_load_scenes(self.handle, scene_begin, n, _ptr(centroids), _ptr(keys), _ptr(values),
                                           _ptr(bias), int(on_dev), _stream(stream, self.device)))

    def lookup(self, queries, top_k, scene_out=None, prim_out=None, weight_out=None, qnorm_out=None, stream=None):
        """Two-level lookup of every query; returns (scene [N], prim [N, k], weight [N, k])."""
        self._tensor(queries, "queries", self.torch_dtype)
        N = queries.shape[0]
        dev = self.device
        scene_out = torch.empty(N, dtype=torch.int32, device=dev) if scene_out is None else scene_out
        prim_out = torch.empty(N, top_k, dtype=torch.int32, device=dev) if prim_out is None else prim_out
        weight_out = torch.empty(N, top_k, dtype=torch.float32, device=dev) if weight_out is None else weight_out
        _check(self.lib.lookme_lookup(self.handle, _ptr(queries), N, top_k, _ptr(scene_out), _ptr(prim_out),
                                      _ptr(weight_out), _ptr(qnorm_out), _stream(stream, dev)))
        return scene_out, prim_out, weight_out

    def inject(self, scene, prim, weight, hidden, keep_ratio, priority=None, seg_offsets=None, mask_out=None,
               sel_out=None, stream=None):
        """Add the looked-up rows into the kept rows of every hidden tensor (in place); returns the mask."""
        hidden = list(hidden) if isinstance(hidden, (list, tuple)) else [hidden]
        N, top_k = prim.shape
        for i, h in enumerate(hidden):
            self._tensor(h, f"hidden[{i}]", self.torch_dtype)
        if mask_out is None:
            mask_out = torch.empty(N, dtype=torch.uint8, device=self.device)
        arr = (ctypes.c_void_p * len(hidden))(*[h.data_ptr() for h in hidden])
        if seg_offsets is not None:
            seg = (ctypes.c_int64 * len(seg_offsets))(*[int(x) for x in seg_offsets])
            n_seg = len(seg_offsets) - 1
        else:
            seg, n_seg = None, 0
        _check(self.lib.lookme_inject(self.handle, _ptr(scene), _ptr(prim), _ptr(weight), N, top_k,
                                      _ptr(priority), seg, n_seg, float(keep_ratio), arr, len(hidden),
                                      _ptr(mask_out), _ptr(sel_out), _stream(stream, self.device)))
        return mask_out

    def lookup_inject(self, queries, top_k, hidden, keep_ratio, priority=None, seg_offsets=None, scene_out=None,
                      prim_out=None, weight_out=None, mask_out=None, stream=None):
        """Lookup and injection in one call; returns (scene, prim, weight, mask)."""
        self._tensor(queries, "queries", self.torch_dtype)
        hidden = list(hidden) if isinstance(hidden, (list, tuple)) else [hidden]
        for i, h in enumerate(hidden):
            self._tensor(h, f"hidden[{i}]", self.torch_dtype)
        N = queries.shape[0]
        dev = self.device
        scene_out = torch.empty(N, dtype=torch.int32, device=dev) if scene_out is None else scene_out
        prim_out = torch.empty(N, top_k, dtype=torch.int32, device=dev) if prim_out is None else prim_out
        weight_out = torch.empty(N, top_k, dtype=torch.float32, device=dev) if weight_out is None else weight_out
        mask_out = torch.empty(N, dtype=torch.uint8, device=dev) if mask_out is None else mask_out
        arr = (ctypes.c_void_p * len(hidden))(*[h.data_ptr() for h in hidden])
        if seg_offsets is not None:
            seg = (ctypes.c_int64 * len(seg_offsets))(*[int(x) for x in seg_offsets])
            n_seg = len(seg_offsets) - 1
        else:
            seg, n_seg = None, 0
        _check(self.lib.lookme_lookup_inject(self.handle, _ptr(queries), N, top_k, _ptr(priority), seg, n_seg,
                                             float(keep_ratio), arr, len(hidden), _ptr(scene_out), _ptr(prim_out),
                                             _ptr(weight_out), _ptr(mask_out), _stream(stream, dev)))
        return scene_out, prim_out, weight_out, mask_out

    def reserve(self, max_tokens):
        _check(self.lib.lookme_reserve(self.handle, max_tokens))

    def stats(self, stream=None):
        s = LookupStats()
        _check(self.lib.lookme_last_lookup_stats(self.handle, ctypes.byref(s), _stream(stream, self.device)))
        return dict(n_tokens=s.n_tokens, n_routed_scenes=s.n_routed_scenes, n_work_items=s.n_work_items,
                    staged_bytes=s.staged_bytes, staged_hits=s.staged_hits)

    def stage_invalidate(self, stream=None):
        """Empty the HBM slot cache of a pinned-host table (the next lookup copies every routed scene)."""
        _check(self.lib.lookme_stage_invalidate(self.handle, _stream(stream, self.device)))

    def set_grids(self, route_sms=0, level2_ctas=0):
        """Grid sizes of later calls: routing and bucketing for `route_sms` SMs, level 2 on
        `level2_ctas` CTAs (0: the whole device)."""
        _check(self.lib.lookme_set_grids(self.handle, int(route_sms), int(level2_ctas)))

    def device_status(self, reset=False, stream=None):
        v = ctypes.c_uint32()
        _check(self.lib.lookme_device_status(self.handle, ctypes.byref(v), int(reset), _stream(stream, self.device)))
        return v.value

    def launch_count(self):
        return int(self.lib.lookme_launch_count(self.handle))

    def trace_enable(self, on=True):
        _check(self.lib.lookme_trace_enable(self.handle, int(on)))

    def trace_read(self, max_records=1 << 16):
        buf = (TraceRecord * max_records)()
        n = ctypes.c_int32()
        _check(self.lib.lookme_trace_read(self.handle, buf, max_records, ctypes.byref(n)))
        return [(self.lib.lookme_kernel_name(buf[i].kernel).decode(), buf[i].ms) for i in range(n.value)]


# ------------------------------------------------------------------------------
# The pieces around the two-level lookup (Sec. "Level-2", "Text", "Sparse
# Injection", "Multi-scale image retrieval"): thin marshalling, as above.
def _ptrs(ts):
    return (ctypes.c_void_p * len(ts))(*[t.data_ptr() for t in ts])


def _set_ranker(self, W1, b1, W2, b2, stream=None):
    """Install the ranker MLP: W1 [d_m, 2 d_key] bf16, b1 [d_m] fp32, W2 [n_prims, d_m] bf16, b2 [n_prims] fp32."""
    for name, t, dt in (("W1", W1, torch.bfloat16), ("b1", b1, torch.float32), ("W2", W2, torch.bfloat16),
                        ("b2", b2, torch.float32)):
        self._tensor(t, name, dt, device=False)
    _check(self.lib.lookme_set_ranker(self.handle, W1.shape[0], _ptr(W1), _ptr(b1), _ptr(W2), _ptr(b2),
                                      _stream(stream, self.device)))


def _lookup_ranked(self, queries, top_t, scene_out=None, prim_out=None, weight_out=None, stream=None):
    """Level 1, then the paper's level 2 (MLP relevance, top-T, cos + tanh softmax)."""
    self._tensor(queries, "queries", self.torch_dtype)
    N, dev = queries.shape[0], self.device
    scene_out = torch.empty(N, dtype=torch.int32, device=dev) if scene_out is None else scene_out
    prim_out = torch.empty(N, top_t, dtype=torch.int32, device=dev) if prim_out is None else prim_out
    weight_out = torch.empty(N, top_t, dtype=torch.float32, device=dev) if weight_out is None else weight_out
    _check(self.lib.lookme_lookup_ranked(self.handle, _ptr(queries), N, top_t, _ptr(scene_out), _ptr(prim_out),
                                         _ptr(weight_out), _stream(stream, dev)))
    return scene_out, prim_out, weight_out


def _inject_gated(self, scene, prim, weight, gate, hidden, stream=None):
    """h_l[t] += sum_j w V rows for every gated t (in place)."""
    hidden = list(hidden) if isinstance(hidden, (list, tuple)) else [hidden]
    for i, h in enumerate(hidden):
        self._tensor(h, f"hidden[{i}]", self.torch_dtype)
    N, k = prim.shape
    _check(self.lib.lookme_inject_gated(self.handle, _ptr(scene), _ptr(prim), _ptr(weight), N, k, _ptr(gate),
                                        _ptrs(hidden), len(hidden), _stream(stream, self.device)))


def _combine(self, scene, prim, weight, rows, out=None, stream=None):
    """Retrieved embeddings of the listed tokens, bf16 [len(rows), d_value]."""
    n, k = rows.shape[0], prim.shape[1]
    out = torch.empty(n, self.shape[3], dtype=torch.bfloat16, device=self.device) if out is None else out
    _check(self.lib.lookme_combine(self.handle, _ptr(scene), _ptr(prim), _ptr(weight), scene.shape[0], k, _ptr(rows),
                                   n, _ptr(out), _stream(stream, self.device)))
    return out


Table.set_ranker = _set_ranker
Table.lookup_ranked = _lookup_ranked
Table.inject_gated = _inject_gated
Table.combine = _combine


def _code(dtype):
    return BF16 if dtype == torch.bfloat16 else FP32


def ska_gate(delta, w_g, gate_out=None, logit_out=None, stream=None):
    """Hard SKA gate g = [delta . w_g > 0]; returns (gate u8, logit fp32 or None)."""
    lib = load()
    N, dh = delta.shape
    gate_out = torch.empty(N, dtype=torch.uint8, device=delta.device) if gate_out is None else gate_out
    _check(lib.lookme_ska_gate(_ptr(delta), _ptr(w_g), N, dh, _code(delta.dtype), _ptr(gate_out), _ptr(logit_out),
                               _stream(stream, delta.device)))
    return gate_out, logit_out


def text_inject(E, ids, hidden, gate=None, stream=None):
    """h_l[t] += E[ids[t]] on gated text positions (ids outside [0, V) are skipped); in place."""
    lib = load()
    hidden = list(hidden) if isinstance(hidden, (list, tuple)) else [hidden]
    V, d = E.shape
    _check(lib.lookme_text_inject(_ptr(E), V, d, _code(E.dtype), _ptr(ids), _ptr(gate), ids.shape[0], _ptrs(hidden),
                                  len(hidden), _stream(stream, E.device)))


def project(x, W, bias=None, out=None, stream=None):
    """x W^T + bias in bf16 on the tensor cores (W [d_out, d_in])."""
    lib = load()
    N, d_in = x.shape
    d_out = W.shape[0]
    out = torch.empty(N, d_out, dtype=torch.bfloat16, device=x.device) if out is None else out
    _check(lib.lookme_project(_ptr(x), _ptr(W), _ptr(bias), N, d_in, d_out, _ptr(out), _stream(stream, x.device)))
    return out


def scale_router(H, W_he, scales, out=None, att_out=None, workspace=None, stream=None):
    """Softmax router over the scales' results (W_he [d_e, d_h]); returns (out bf16 [N, d_e], att or None)."""
    lib = load()
    N, dh = H.shape
    de = W_he.shape[0]
    workspace = torch.empty(N, de, dtype=torch.float32, device=H.device) if workspace is None else workspace
    out = torch.empty(N, de, dtype=torch.bfloat16, device=H.device) if out is None else out
    _check(lib.lookme_scale_router(_ptr(H), _ptr(W_he), _ptrs(scales), len(scales), N, dh, de, _ptr(workspace),
                                   _ptr(out), _ptr(att_out), _stream(stream, H.device)))
    return out, att_out


class Fusion:
    """SwiGLU fusion f and the R W_p + R propagation over n_stages layers (bf16)."""

    def __init__(self, n_stages, d_embed, d_ff, d_hidden, device=0, max_rows=4096):
        self.lib = load()
        self.device = torch.device("cuda", device) if isinstance(device, int) else torch.device(device)
        h = ctypes.c_void_p()
        _check(self.lib.lookme_fusion_create(n_stages, d_embed, d_ff, d_hidden, self.device.index or 0, max_rows,
                                             ctypes.byref(h)))
        self.handle = h
        self.n_stages = n_stages

    def load_stage(self, stage, W_a, W_b, W_o, W_p=None, stream=None):
        """W_a, W_b [d_ff, d_e]; W_o [d_h, d_ff]; W_p [d_e, d_e] as a linear weight (paper's W_p transposed)."""
        _check(self.lib.lookme_fusion_load(self.handle, stage, _ptr(W_a), _ptr(W_b), _ptr(W_o), _ptr(W_p),
                                           _stream(stream, self.device)))

    def apply(self, R, rows, hidden, stream=None):
        """h_k[rows] += f^k(R^(k)) for every stage k (in place)."""
        _check(self.lib.lookme_fusion_apply(self.handle, _ptr(R), _ptr(rows), rows.shape[0], _ptrs(hidden),
                                            _stream(stream, self.device)))

    def status(self, stream=None):
        v = ctypes.c_uint32()
        _check(self.lib.lookme_fusion_status(self.handle, ctypes.byref(v), _stream(stream, self.device)))
        return v.value

    def close(self):
        if getattr(self, "handle", None):
            self.lib.lookme_fusion_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:  # noqa: BLE001 - interpreter shutdown
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
