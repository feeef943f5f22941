"""LookME CPU oracle: TEST INFRASTRUCTURE ONLY.

A plain, slow, double-precision restatement of the hierarchical two-level
lookup and sparse injection of arXiv 2607.16305 (Sec. "Image Embedding
Hierarchical Two-Level Lookup", Sec. "Sparse Injection").  The arithmetic is
in ``lookme_oracle.c``; this module compiles it with gcc, loads it with
ctypes and marshals numpy arrays.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The CUDA library never does, and the two
share no code.

Every function takes float32 arrays that hold the exact input values (bf16
inputs widened to float32 are exact) and computes in float64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "lookme_oracle.c")
_LIB = os.path.join(_HERE, "liblookme_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB) -> str:
    """Compile the C oracle into a shared library (gcc -O2 -fopenmp)."""
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


_I64 = ctypes.c_int64
_I32 = ctypes.c_int32
_P = ctypes.c_void_p
_D = ctypes.c_double

_SIGS = {
    "lkm_centroids": [_I64, _I64, _I64, _P, _P],
    "lkm_query_norms": [_I64, _I64, _P, _P],
    "lkm_route": [_I64, _I64, _I64, _P, _P, _P, _P, _P, _P, _P],
    "lkm_primitives": [_I64, _I64, _I64, _I32, _P, _P, _P, _P, _P, _P, _P, _P, _P],
    "lkm_weights_for": [_I64, _I64, _I64, _I32, _P, _P, _P, _P, _P, _P],
    "lkm_select": [_I64, _P, _I32, _P, _D, _P, _P, _P],
    "lkm_inject": [_I64, _I64, _I64, _I32, _P, _P, _P, _P, _P, _P, _I32, _P, _P],
    "lkm_round_bf16": [_I64, _P, _P],
}


def load(path: str | None = None):
    """Build (if needed) and load the oracle library.  A path loads that file instead."""
    global _lib
    if path is not None:
        lib = ctypes.CDLL(path)
        for name, argtypes in _SIGS.items():
            fn = getattr(lib, name)
            fn.argtypes = argtypes
            fn.restype = None
        return lib
    with _lock:
        if _lib is None:
            _lib = load(build())
    return _lib


def _f32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def _ptr(a):
    return None if a is None else a.ctypes.data


def _blocks(blocks, block_of_scene, n_scene):
    """Scene blocks [n_blocks, P, d] plus the scene -> block map (identity if None)."""
    blocks = _f32(blocks)
    if block_of_scene is None:
        block_of_scene = np.arange(n_scene, dtype=np.int64)
    return blocks, np.ascontiguousarray(block_of_scene, dtype=np.int64)


class Oracle:
    """numpy front end to the C oracle.  ``lib`` may be a mutated build (tests)."""

    def __init__(self, lib=None):
        self.lib = lib if lib is not None else load()

    def centroids(self, keys):
        """e_img[s] = mean over primitives of K[s] (Level-1, first equation)."""
        keys = _f32(keys)
        S, P, dk = keys.shape
        out = np.empty((S, dk), np.float64)
        self.lib.lkm_centroids(S, P, dk, _ptr(keys), _ptr(out))
        return out

    def query_norms(self, q):
        """||q_t||_2 in float64 (the default token-selection priority)."""
        q = _f32(q)
        out = np.empty(q.shape[0], np.float64)
        self.lib.lkm_query_norms(q.shape[0], q.shape[1], _ptr(q), _ptr(out))
        return out

    def route(self, q, cent, bias=None):
        """Level-1 routing.  Returns dict(scene, score, gap1, qnorm)."""
        q, cent = _f32(q), _f32(cent)
        N, dk = q.shape
        S = cent.shape[0]
        bias = None if bias is None else _f32(bias)
        scene = np.empty(N, np.int32)
        score, gap1, qnorm = (np.empty(N, np.float64) for _ in range(3))
        self.lib.lkm_route(N, S, dk, _ptr(q), _ptr(cent), _ptr(bias),
                           _ptr(scene), _ptr(score), _ptr(gap1), _ptr(qnorm))
        return dict(scene=scene, score=score, gap1=gap1, qnorm=qnorm)

    def primitives(self, q, scene, key_blocks, top_k, block_of_scene=None, n_scene=None):
        """Level-2 scoring, top-k and softmax.  Returns dict(prim, weight, logit, gap_k, gap_adj)."""
        q = _f32(q)
        N, dk = q.shape
        kb = np.asarray(key_blocks)
        P = kb.shape[1]
        kb, bos = _blocks(kb, block_of_scene, n_scene if n_scene is not None else kb.shape[0])
        scene = np.ascontiguousarray(scene, dtype=np.int32)
        if N and (scene.min() < 0 or scene.max() >= bos.shape[0] or (bos[scene] < 0).any()):
            raise ValueError("a token's scene block is missing")
        if not 1 <= top_k <= min(P, 64):
            raise ValueError("top_k out of range")
        prim = np.empty((N, top_k), np.int32)
        weight, logit = np.empty((N, top_k), np.float64), np.empty((N, top_k), np.float64)
        gap_k, gap_adj = np.empty(N, np.float64), np.empty(N, np.float64)
        self.lib.lkm_primitives(N, P, dk, top_k, _ptr(q), _ptr(scene), _ptr(kb), _ptr(bos),
                                _ptr(prim), _ptr(weight), _ptr(logit), _ptr(gap_k), _ptr(gap_adj))
        return dict(prim=prim, weight=weight, logit=logit, gap_k=gap_k, gap_adj=gap_adj)

    def weights_for(self, q, scene, prim, key_blocks, block_of_scene=None, n_scene=None):
        """Softmax weights of a given primitive set (conditional oracle)."""
        q = _f32(q)
        N, dk = q.shape
        kb = np.asarray(key_blocks)
        P = kb.shape[1]
        kb, bos = _blocks(kb, block_of_scene, n_scene if n_scene is not None else kb.shape[0])
        prim = np.ascontiguousarray(prim, dtype=np.int32)
        top_k = prim.shape[1]
        if top_k > 64:
            raise ValueError("top_k out of range")
        scene = np.ascontiguousarray(scene, dtype=np.int32)
        weight = np.empty((N, top_k), np.float64)
        self.lib.lkm_weights_for(N, P, dk, top_k, _ptr(q), _ptr(scene), _ptr(prim),
                                 _ptr(kb), _ptr(bos), _ptr(weight))
        return weight

    def select(self, priority, keep_ratio, seg_off=None):
        """Top-r token selection per segment.  Returns dict(mask, pi_r, pi_r1, seg_off)."""
        pr = np.ascontiguousarray(priority, dtype=np.float64)
        N = pr.shape[0]
        if seg_off is None:
            seg_off = [0, N]
        seg_off = np.ascontiguousarray(seg_off, dtype=np.int64)
        n_seg = seg_off.shape[0] - 1
        mask = np.empty(N, np.uint8)
        pi_r, pi_r1 = np.empty(n_seg, np.float64), np.empty(n_seg, np.float64)
        self.lib.lkm_select(N, _ptr(pr), n_seg, _ptr(seg_off), float(keep_ratio),
                            _ptr(mask), _ptr(pi_r), _ptr(pi_r1))
        return dict(mask=mask, pi_r=pi_r, pi_r1=pi_r1, seg_off=seg_off)

    def inject(self, scene, prim, weight, mask, value_blocks, hidden, block_of_scene=None, n_scene=None):
        """h' = h + sum_j w_j V[scene, prim_j] on masked rows of every layer.  Returns float64 [L,N,dv]."""
        hidden = _f32(hidden)
        if hidden.ndim == 2:
            hidden = hidden[None]
        L, N, dv = hidden.shape
        vb = np.asarray(value_blocks)
        P = vb.shape[1]
        vb, bos = _blocks(vb, block_of_scene, n_scene if n_scene is not None else vb.shape[0])
        prim = np.ascontiguousarray(prim, dtype=np.int32)
        top_k = prim.shape[1]
        weight = np.ascontiguousarray(weight, dtype=np.float64)
        mask = np.ascontiguousarray(mask, dtype=np.uint8)
        scene = np.ascontiguousarray(scene, dtype=np.int32)
        sel_scenes = scene[mask.astype(bool)]
        if sel_scenes.size and (bos[sel_scenes] < 0).any():
            raise ValueError("a selected token's value block is missing")
        out = np.empty((L, N, dv), np.float64)
        self.lib.lkm_inject(N, P, dv, top_k, _ptr(scene), _ptr(prim), _ptr(weight), _ptr(mask),
                            _ptr(vb), _ptr(bos), L, _ptr(hidden), _ptr(out))
        return out

    def round_bf16(self, x):
        """Round-to-nearest-even to bf16; returns the uint16 bit patterns."""
        x = np.ascontiguousarray(x, dtype=np.float64)
        out = np.empty(x.shape, np.uint16)
        self.lib.lkm_round_bf16(x.size, _ptr(x), _ptr(out))
        return out


def bf16_bits_to_f32(bits):
    """Widen bf16 bit patterns (uint16) to float32 values (exact)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32)


# ---------------------------------------------------------------------------
# Second part (lookme_oracle_ext.c): the paper-exact level 2 with the MLP
# ranker, the SKA gate, the text pathway, the dense ends and the multi-scale
# router.  Same rules: test infrastructure only.
_SRC_EXT = os.path.join(_HERE, "lookme_oracle_ext.c")
_LIB_EXT = os.path.join(_HERE, "liblookme_oracle_ext.so")
_lib_ext = None

_SIGS_EXT = {
    "lkx_linear": [_I64, _I64, _I64, _P, _P, _P, _P],
    "lkx_ranker_relevance": [_I64, _I64, _I64, _I64, _I64, _P, _P, _P, _P, _P, _P, _P, _I32, _P],
    "lkx_ranked_level2": [_I64, _I64, _I64, _I32, _P, _P, _P, _P, _P, _P, _P, _P, _P],
    "lkx_ranked_weights_for": [_I64, _I64, _I64, _I32, _P, _P, _P, _P, _P, _P, _P],
    "lkx_ska_gate": [_I64, _I64, _P, _P, _P, _P],
    "lkx_combine": [_I64, _I64, _I64, _I32, _P, _P, _P, _P, _P, _P],
    "lkx_text_inject": [_I64, _I64, _I64, _P, _P, _P, _I32, _P, _P],
    "lkx_swiglu": [_I64, _I64, _I64, _I64, _P, _P, _P, _P, _I32, _P],
    "lkx_propagate": [_I64, _I64, _P, _P, _P],
    "lkx_scale_router": [_I64, _I64, _I64, _I32, _P, _P, _P, _P, _P],
}


def build_ext(force: bool = False, src: str = _SRC_EXT, out: str = _LIB_EXT) -> str:
    """Compile the second part of the C oracle (gcc -O2 -fopenmp)."""
    return build(force, src, out)


def load_ext(path: str | None = None):
    """Build (if needed) and load the second part; a path loads that file instead."""
    global _lib_ext
    if path is not None:
        lib = ctypes.CDLL(path)
        for name, argtypes in _SIGS_EXT.items():
            fn = getattr(lib, name)
            fn.argtypes = argtypes
            fn.restype = None
        return lib
    with _lock:
        if _lib_ext is None:
            _lib_ext = load_ext(build_ext())
    return _lib_ext


def _i32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


class PaperOracle:
    """numpy front end to lookme_oracle_ext.c.  ``lib`` may be a mutated build (tests)."""

    def __init__(self, lib=None):
        self.lib = lib if lib is not None else load_ext()

    def linear(self, x, W, b=None):
        """x W^T + b with W [dout][din] (float64 result)."""
        x, W = _f32(x), _f32(W)
        n, din = x.shape
        dout = W.shape[0]
        assert W.shape[1] == din
        y = np.empty((n, dout), np.float64)
        self.lib.lkx_linear(n, din, dout, _ptr(x), _ptr(W), _ptr(None if b is None else _f32(b)), _ptr(y))
        return y

    def ranker_relevance(self, v, scene, cent, W1, b1, W2, b2, round_hidden=True):
        """r = W2 silu(W1 [v ; e_img[scene]] + b1) + b2 (Level-2, first equation) [N][P]."""
        v, cent, W1, b1, W2, b2 = (_f32(a) for a in (v, cent, W1, b1, W2, b2))
        N, de = v.shape
        S = cent.shape[0]
        dm, P = W1.shape[0], W2.shape[0]
        assert W1.shape[1] == 2 * de and W2.shape[1] == dm
        r = np.empty((N, P), np.float64)
        self.lib.lkx_ranker_relevance(N, S, de, dm, P, _ptr(v), _ptr(_i32(scene)), _ptr(cent), _ptr(W1), _ptr(b1),
                                      _ptr(W2), _ptr(b2), 1 if round_hidden else 0, _ptr(r))
        return r

    def ranked_level2(self, v, scene, key_blocks, r, top_t, block_of_scene=None, n_scene=None):
        """Top-T by r, weights softmax(cos + tanh r).  Returns dict(prim, weight, gap_T, gap_adj)."""
        v = _f32(v)
        N, de = v.shape
        kb = np.asarray(key_blocks)
        P = kb.shape[1]
        kb, bos = _blocks(kb, block_of_scene, n_scene if n_scene is not None else kb.shape[0])
        r = np.ascontiguousarray(r, dtype=np.float64)
        if not 1 <= top_t <= min(P, 64):
            raise ValueError("top_t out of range")
        prim = np.empty((N, top_t), np.int32)
        weight = np.empty((N, top_t), np.float64)
        gap_T, gap_adj = np.empty(N, np.float64), np.empty(N, np.float64)
        self.lib.lkx_ranked_level2(N, P, de, top_t, _ptr(v), _ptr(_i32(scene)), _ptr(kb), _ptr(bos), _ptr(r),
                                   _ptr(prim), _ptr(weight), _ptr(gap_T), _ptr(gap_adj))
        return dict(prim=prim, weight=weight, gap_T=gap_T, gap_adj=gap_adj)

    def ranked_weights_for(self, v, scene, prim, key_blocks, r, block_of_scene=None, n_scene=None):
        """The cos + tanh softmax of a given primitive set (conditional oracle)."""
        v = _f32(v)
        N, de = v.shape
        kb = np.asarray(key_blocks)
        P = kb.shape[1]
        kb, bos = _blocks(kb, block_of_scene, n_scene if n_scene is not None else kb.shape[0])
        prim = _i32(prim)
        r = np.ascontiguousarray(r, dtype=np.float64)
        w = np.empty(prim.shape, np.float64)
        self.lib.lkx_ranked_weights_for(N, P, de, prim.shape[1], _ptr(v), _ptr(_i32(scene)), _ptr(prim), _ptr(kb),
                                        _ptr(bos), _ptr(r), _ptr(w))
        return w

    def ska_gate(self, delta, wg):
        """Hard SKA gate: returns (gate u8 [N], logit float64 [N])."""
        delta, wg = _f32(delta), _f32(wg)
        N, dh = delta.shape
        gate, logit = np.empty(N, np.uint8), np.empty(N, np.float64)
        self.lib.lkx_ska_gate(N, dh, _ptr(delta), _ptr(wg), _ptr(gate), _ptr(logit))
        return gate, logit

    def combine(self, scene, prim, weight, value_blocks, block_of_scene=None, n_scene=None):
        """R_t = sum_j w_tj V[scene_t, prim_tj] (float64 [N][dv])."""
        vb = np.asarray(value_blocks)
        P, dv = vb.shape[1], vb.shape[2]
        vb, bos = _blocks(vb, block_of_scene, n_scene if n_scene is not None else vb.shape[0])
        prim = _i32(prim)
        N, T = prim.shape
        R = np.empty((N, dv), np.float64)
        self.lib.lkx_combine(N, P, dv, T, _ptr(_i32(scene)), _ptr(prim),
                             _ptr(np.ascontiguousarray(weight, dtype=np.float64)), _ptr(vb), _ptr(bos), _ptr(R))
        return R

    def text_inject(self, E, ids, gate, hidden):
        """h + E[ids] on gated text positions of every layer (float64 [L][N][d])."""
        E, hidden = _f32(E), _f32(hidden)
        if hidden.ndim == 2:
            hidden = hidden[None]
        L, N, d = hidden.shape
        out = np.empty((L, N, d), np.float64)
        g = None if gate is None else np.ascontiguousarray(gate, dtype=np.uint8)
        self.lib.lkx_text_inject(N, E.shape[0], d, _ptr(E), _ptr(_i32(ids)), _ptr(g), L, _ptr(hidden), _ptr(out))
        return out

    def swiglu(self, x, Wa, Wb, Wo, round_mid=True):
        """(silu(x Wa^T) * (x Wb^T)) Wo^T (float64)."""
        x, Wa, Wb, Wo = (_f32(a) for a in (x, Wa, Wb, Wo))
        n, de = x.shape
        dff, dh = Wa.shape[0], Wo.shape[0]
        y = np.empty((n, dh), np.float64)
        self.lib.lkx_swiglu(n, de, dff, dh, _ptr(x), _ptr(Wa), _ptr(Wb), _ptr(Wo), 1 if round_mid else 0, _ptr(y))
        return y

    def propagate(self, R, Wp):
        """R W_p + R (W_p [de][de], paper orientation)."""
        R, Wp = _f32(R), _f32(Wp)
        n, de = R.shape
        out = np.empty((n, de), np.float64)
        self.lib.lkx_propagate(n, de, _ptr(R), _ptr(Wp), _ptr(out))
        return out

    def scale_router(self, H, Whe, Rs):
        """Token-wise softmax router over M scales.  Returns (out [N][de], att [N][M])."""
        H, Whe, Rs = _f32(H), _f32(Whe), _f32(Rs)
        N, dh = H.shape
        de = Whe.shape[1]
        M = Rs.shape[0]
        if not 1 <= M <= 64:
            raise ValueError("1 <= M <= 64")
        out, att = np.empty((N, de), np.float64), np.empty((N, M), np.float64)
        self.lib.lkx_scale_router(N, dh, de, M, _ptr(H), _ptr(Whe), _ptr(Rs), _ptr(out), _ptr(att))
        return out, att
