"""Seeded synthetic LookME workloads.

The paper evaluates on Qwen2.5-VL image tokens drawn from public benchmarks
(Sec. "Experimental Setup").  Neither those tokens nor the trained tables are
available, so these generators stand in for them: a Gaussian mixture of scene
means, queries drawn around the means, primitive keys scattered around their
scene centroid, small random values and unit-normal hidden states.

This module holds no part of the method's arithmetic: it only draws random
numbers (torch generators, seeded per workload, per table and per chunk of
scenes) and casts them to the workload's dtype.  Both the CUDA path and the
CPU oracle consume what it returns.

Recipe (every workload):
  mu[c]   ~ N(0, 1)^{d_k}                       c < n_components (= n_scenes)
  comp[t] ~ Uniform(n_components), or Zipf(a) over ranks mapped through a
            seeded permutation of the components
  q[t]    = mu[comp[t]] + sigma_q * N(0, 1)
  C_i[s]  = mu[perm_i[s]]  (perm_i = identity for a single table)
  K_i[s,p]= C_i[s] + sigma_key * N(0, 1)
  V_i[s,p]~ sigma_value * N(0, 1)
  h_l[t]  ~ N(0, 1)
then a cast to bf16 for the bf16 workloads.
"""
from __future__ import annotations

import dataclasses
import math

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n_tokens: int
    d_key: int
    n_scenes: int
    n_prims: int
    d_value: int
    top_k: int
    keep_ratio: float
    dtype: str = "bf16"            # "fp32" or "bf16"
    n_segments: int = 1            # equal-length token-selection segments
    n_tables: int = 1
    layers_per_table: int = 1
    residency: str = "device"      # "device" or "host" (pinned host, staged to HBM)
    zipf: float | None = None      # scene popularity exponent; None = uniform
    scale_lengths: tuple = ()      # multi-scale query groups (concatenated)
    sigma_q: float = 0.1
    sigma_key: float = 0.3
    sigma_value: float = 0.02
    seed: int = 0
    scenes_per_chunk: int = 256    # table generation granularity

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "fp32" else torch.bfloat16

    @property
    def elem_bytes(self):
        return 4 if self.dtype == "fp32" else 2

    @property
    def n_chunks(self):
        return (self.n_scenes + self.scenes_per_chunk - 1) // self.scenes_per_chunk

    @property
    def segment_offsets(self):
        n, k = self.n_tokens, self.n_segments
        return [i * n // k for i in range(k + 1)]

    def scaled(self, **kw):
        return dataclasses.replace(self, **kw)


WORKLOADS = {
    # Tiny, fp32: 256 tokens, 64 scenes x 64 primitives, d_k 128, d_v 256, top-4, keep 25%.
    "tiny_fp32": Workload("tiny_fp32", 256, 128, 64, 64, 256, 4, 0.25, dtype="fp32"),
    # One image: 1,024 tokens, 1,024 x 256 table (1 GiB of bf16 values), top-8, keep 25%.
    "single_image": Workload("single_image", 1024, 256, 1024, 256, 2048, 8, 0.25),
    # Batched serving: 32 images x 1,024 tokens, 4,096 x 512 table (8 GiB), Zipf(1.1) scenes.
    "batched_zipf": Workload("batched_zipf", 32768, 256, 4096, 512, 2048, 8, 0.25,
                             n_segments=32, zipf=1.1, scenes_per_chunk=128),
    # Multi-layer, multi-scale: 4,096 tokens (1,024 + 2,048 + 1,024), 7 tables x 4 layers,
    # each table 2,048 x 256 with d_v 1,536 in pinned host memory, keep 12.5%.
    "multilayer_host": Workload("multilayer_host", 4096, 256, 2048, 256, 1536, 8, 0.125,
                                n_tables=7, layers_per_table=4, residency="host",
                                scale_lengths=(1024, 2048, 1024)),
    # Large table: 65,536 tokens, 16,384 x 1,024 table (64 GiB of values), d_k 512, top-16.
    "large_table": Workload("large_table", 65536, 512, 16384, 1024, 2048, 16, 0.25,
                            scenes_per_chunk=64),
}


def _gen(device, *key):
    """A torch generator seeded from a tuple of small integers."""
    s = 0
    for k in key:
        s = (s * 1000003 + int(k)) % (2**62)
    g = torch.Generator(device=device)
    g.manual_seed(s)
    return g


def _randn(shape, g, device):
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32)


def means(w: Workload, device="cpu"):
    """Mixture component means mu [n_scenes, d_key], float32."""
    return _randn((w.n_scenes, w.d_key), _gen(device, w.seed, 1), device)


def scene_permutation(w: Workload, table: int, device="cpu"):
    """Table i's centroid s is mu[perm_i[s]]; identity when there is one table."""
    if w.n_tables == 1:
        return torch.arange(w.n_scenes, device=device)
    return torch.randperm(w.n_scenes, generator=_gen(device, w.seed, 2, table), device=device)


def centroids(w: Workload, table: int = 0, device="cpu", mu=None):
    """Scene centroids [n_scenes, d_key] in the workload dtype."""
    mu = means(w, device) if mu is None else mu
    return mu[scene_permutation(w, table, device)].to(w.torch_dtype)


def token_components(w: Workload, device="cpu"):
    """Mixture component of every token (int64 [n_tokens])."""
    g = _gen(device, w.seed, 3)
    C = w.n_scenes
    if w.zipf is None:
        return torch.randint(0, C, (w.n_tokens,), generator=g, device=device)
    ranks = torch.arange(1, C + 1, device=device, dtype=torch.float64)
    p = ranks.pow(-w.zipf)
    p = p / p.sum()
    rank_of_token = torch.multinomial(p.float(), w.n_tokens, replacement=True, generator=g)
    rank_to_comp = torch.randperm(C, generator=_gen(device, w.seed, 4), device=device)
    return rank_to_comp[rank_of_token]


def queries(w: Workload, device="cpu", mu=None):
    """Queries [n_tokens, d_key] in the workload dtype."""
    mu = means(w, device) if mu is None else mu
    comp = token_components(w, device)
    noise = _randn((w.n_tokens, w.d_key), _gen(device, w.seed, 5), device)
    return (mu[comp] + w.sigma_q * noise).to(w.torch_dtype)


def table_chunk(w: Workload, table: int, chunk: int, device="cpu", mu=None, cent=None):
    """Keys [n, P, d_key] and values [n, P, d_value] of scenes
    [chunk * scenes_per_chunk, ...), in the workload dtype."""
    s0 = chunk * w.scenes_per_chunk
    s1 = min(w.n_scenes, s0 + w.scenes_per_chunk)
    if cent is None:
        cent = centroids(w, table, device, mu)
    c = cent[s0:s1].float()
    gk = _gen(device, w.seed, 6, table, chunk)
    keys = (c[:, None, :] + w.sigma_key * _randn((s1 - s0, w.n_prims, w.d_key), gk, device))
    gv = _gen(device, w.seed, 7, table, chunk)
    values = w.sigma_value * _randn((s1 - s0, w.n_prims, w.d_value), gv, device)
    return keys.to(w.torch_dtype), values.to(w.torch_dtype)


def scene_block(w: Workload, table: int, scene: int, device="cpu", mu=None, cent=None):
    """Keys and values of one scene (regenerates its chunk)."""
    chunk = scene // w.scenes_per_chunk
    k, v = table_chunk(w, table, chunk, device, mu, cent)
    i = scene - chunk * w.scenes_per_chunk
    return k[i], v[i]


def full_table(w: Workload, table: int = 0, device="cpu", mu=None):
    """Centroids, keys and values of a whole table (small workloads only)."""
    cent = centroids(w, table, device, mu)
    ks, vs = zip(*(table_chunk(w, table, c, device, mu, cent) for c in range(w.n_chunks)))
    return cent, torch.cat(ks), torch.cat(vs)


def hidden(w: Workload, layer: int, device="cpu"):
    """Hidden states of one layer [n_tokens, d_value] in the workload dtype."""
    g = _gen(device, w.seed, 8, layer)
    return _randn((w.n_tokens, w.d_value), g, device).to(w.torch_dtype)


def small(name: str = "mini", **kw) -> Workload:
    """A small ad-hoc workload for property tests."""
    base = dict(n_tokens=64, d_key=64, n_scenes=8, n_prims=16, d_value=64, top_k=4, keep_ratio=0.25)
    base.update(kw)
    return Workload(name, **base)


def expected_distinct(n_tokens: int, n_scenes: int) -> float:
    """Expected number of distinct scenes hit by uniform routing."""
    return n_scenes * (1.0 - math.pow(1.0 - 1.0 / n_scenes, n_tokens))
