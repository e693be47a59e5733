"""Seeded synthetic inputs for the RippleKV serving path.

This module draws random tensors and nothing else: it holds no step of the
method (no scoring, selection, allocation or attention arithmetic). The same
generators feed the CPU oracle tests, the CUDA parity tests and the benchmark,
so both sides of every comparison read identical bytes.

Recipe (the stand-in for the prefill KV caches of the paper's Llama / Mistral
backbones on LongBench, none of which exist here):

* every tensor comes from its own torch generator, seeded by a splitmix64 hash
  of (workload seed, tensor tag, layer, decode step);
* "plain" workloads: Q, K, V ~ N(0, 1);
* "scaled_sinks" workloads: K = N(0, 1) * c[h, ch] with a per-(layer, kv head,
  channel) scale c ~ lognormal(0, 0.5), and the first four tokens shifted by
  +3 c (attention-sink keys); V, window queries and decode queries ~ N(0, 1);
  decode keys N(0, 1) * c (same channel scales, no sink shift);
* values are drawn in fp32 and rounded to nearest-even into the workload dtype;
* profiling inputs (the stand-in for one calibration example's outputs):
  perturbation draws eps ~ N(0, 1) in fp32; reference logits over a
  vocabulary = 2.5 N(0, 1) with +12 added to four random tokens per position
  (a peaked next-token distribution), and the logits of perturbed run s =
  reference + sigma_s N(0, 1), sigma_s from 0.02 to 0.3 across the sets;
* layer sensitivity profiles follow the shape the paper reports for
  Llama-3.1-8B (Sec. 3.1: maximum at an intermediate layer, ~18x spread):
  "bump" = a mid-depth Gaussian bump times lognormal(0, 0.3) noise,
  "two_peaks" = two interior bumps, "fixed" = a literal vector.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

_MASK64 = (1 << 64) - 1


def _splitmix64(x: int) -> int:
    x = (x + 0x9E3779B97F4A7C15) & _MASK64
    x = ((x ^ (x >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
    x = ((x ^ (x >> 27)) * 0x94D049BB133111EB) & _MASK64
    return x ^ (x >> 31)


_TAGS = {"k": 1, "v": 2, "q_win": 3, "scale": 4, "dq": 5, "dk": 6, "dv": 7, "sens": 8,
         "votes": 9, "ck": 10, "cv": 11, "eps": 12, "lp": 13, "lq": 14}


def stream_seed(seed: int, tag: str, layer: int = 0, step: int = 0) -> int:
    """63-bit seed of one tensor's generator."""
    h = _splitmix64(seed)
    for part in (_TAGS[tag], layer, step):
        h = _splitmix64(h ^ (part & _MASK64))
    return h & ((1 << 63) - 1)


def _generator(device, seed: int, tag: str, layer: int = 0, step: int = 0) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(stream_seed(seed, tag, layer, step))
    return g


_TORCH_DTYPES = {"f32": torch.float32, "bf16": torch.bfloat16}


@dataclass(frozen=True)
class Workload:
    """Shape, dtype, seed and hyper-parameters of one synthetic serving workload."""

    name: str
    n_layers: int
    batch: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    seq_len: int
    dtype: str
    window: int
    pool_kernel: int
    ratio: float
    avg_budget: int
    decode_steps: int
    seed: int
    profile: str
    kv_dist: str
    fixed_profile: tuple = field(default=())
    gamma: float = math.inf

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def global_budget(self) -> int:
        return self.avg_budget * self.n_layers

    @property
    def torch_dtype(self) -> torch.dtype:
        return _TORCH_DTYPES[self.dtype]

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def replace(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


WORKLOADS = {
    "tiny": Workload(
        name="tiny-4L-4q2kv-d64-B1-T512-f32", n_layers=4, batch=1, n_q_heads=4,
        n_kv_heads=2, head_dim=64, seq_len=512, dtype="f32", window=32, pool_kernel=7,
        ratio=4.0, avg_budget=128, decode_steps=1, seed=0, profile="fixed",
        kv_dist="plain", fixed_profile=(0.2, 1.0, 0.6, 0.1)),
    "llama8b-8k": Workload(
        name="llama3-8b-32L-32q8kv-d128-B1-T8192-bf16", n_layers=32, batch=1,
        n_q_heads=32, n_kv_heads=8, head_dim=128, seq_len=8192, dtype="bf16", window=32,
        pool_kernel=7, ratio=4.0, avg_budget=512, decode_steps=64, seed=1,
        profile="bump", kv_dist="scaled_sinks"),
    "llama8b-32k": Workload(
        name="llama3-8b-32L-32q8kv-d128-B4-T32768-bf16", n_layers=32, batch=4,
        n_q_heads=32, n_kv_heads=8, head_dim=128, seq_len=32768, dtype="bf16", window=32,
        pool_kernel=7, ratio=8.0, avg_budget=1024, decode_steps=128, seed=2,
        profile="bump", kv_dist="scaled_sinks"),
    "mistral7b-16k": Workload(
        name="mistral-7b-32L-32q8kv-d128-B8-T16384-bf16", n_layers=32, batch=8,
        n_q_heads=32, n_kv_heads=8, head_dim=128, seq_len=16384, dtype="bf16", window=32,
        pool_kernel=7, ratio=4.0, avg_budget=128, decode_steps=256, seed=3,
        profile="bump", kv_dist="scaled_sinks"),
    "llama70b-128k": Workload(
        name="llama-70b-80L-64q8kv-d128-B1-T131072-bf16", n_layers=80, batch=1,
        n_q_heads=64, n_kv_heads=8, head_dim=128, seq_len=131072, dtype="bf16", window=32,
        pool_kernel=7, ratio=8.0, avg_budget=2048, decode_steps=64, seed=4,
        profile="two_peaks", kv_dist="scaled_sinks"),
}


def sensitivity_profile(wl: Workload) -> list:
    """Per-layer sensitivity vector s (float64), the input of budget allocation."""
    L = wl.n_layers
    if wl.profile == "fixed":
        return [float(x) for x in wl.fixed_profile]
    rng = np.random.Generator(np.random.Philox(key=stream_seed(wl.seed, "sens")))
    z = rng.standard_normal(L)
    ell = np.arange(L, dtype=np.float64)
    if wl.profile == "bump":
        base = 0.003 + 0.05 * np.exp(-((ell - 0.45 * (L - 1)) ** 2) / (2.0 * (0.15 * L) ** 2))
    elif wl.profile == "two_peaks":
        w = 0.08 * L
        base = (0.003 + 0.05 * np.exp(-((ell - 0.3 * (L - 1)) ** 2) / (2.0 * w * w))
                + 0.04 * np.exp(-((ell - 0.7 * (L - 1)) ** 2) / (2.0 * w * w)))
    else:
        raise ValueError(f"unknown profile {wl.profile}")
    return [float(x) for x in base * np.exp(0.3 * z)]


def _normal(shape, gen, device) -> torch.Tensor:
    return torch.randn(shape, generator=gen, device=device, dtype=torch.float32)


def channel_scales(wl: Workload, layer: int, device="cpu") -> torch.Tensor:
    """fp32 [Hkv][d] key channel scales (all ones for "plain" workloads)."""
    if wl.kv_dist == "plain":
        return torch.ones(wl.n_kv_heads, wl.head_dim, device=device)
    z = _normal((wl.n_kv_heads, wl.head_dim), _generator(device, wl.seed, "scale", layer), device)
    return torch.exp(0.5 * z)


def layer_keys(wl: Workload, layer: int, device="cpu") -> torch.Tensor:
    """K of one layer, [B][Hkv][T][d] in the workload dtype."""
    shape = (wl.batch, wl.n_kv_heads, wl.seq_len, wl.head_dim)
    k = _normal(shape, _generator(device, wl.seed, "k", layer), device)
    if wl.kv_dist == "scaled_sinks":
        c = channel_scales(wl, layer, device)[None, :, None, :]
        k.mul_(c)
        n_sink = min(4, wl.seq_len)
        k[:, :, :n_sink, :].add_(3.0 * c)
    return k.to(wl.torch_dtype)


def layer_values(wl: Workload, layer: int, device="cpu") -> torch.Tensor:
    """V of one layer, [B][Hkv][T][d] in the workload dtype."""
    shape = (wl.batch, wl.n_kv_heads, wl.seq_len, wl.head_dim)
    return _normal(shape, _generator(device, wl.seed, "v", layer), device).to(wl.torch_dtype)


def layer_window_queries(wl: Workload, layer: int, device="cpu") -> torch.Tensor:
    """The last `window` prompt queries of one layer, [B][Hq][w][d]."""
    shape = (wl.batch, wl.n_q_heads, wl.window, wl.head_dim)
    return _normal(shape, _generator(device, wl.seed, "q_win", layer), device).to(wl.torch_dtype)


def decode_inputs(wl: Workload, step: int, device="cpu", layers=None):
    """(q [L][B][Hq][d], k_new [L][B][Hkv][d], v_new [L][B][Hkv][d]) of one decode step."""
    layers = range(wl.n_layers) if layers is None else layers
    qs, ks, vs = [], [], []
    for layer in layers:
        q = _normal((wl.batch, wl.n_q_heads, wl.head_dim),
                    _generator(device, wl.seed, "dq", layer, step), device)
        k = _normal((wl.batch, wl.n_kv_heads, wl.head_dim),
                    _generator(device, wl.seed, "dk", layer, step), device)
        if wl.kv_dist == "scaled_sinks":
            k.mul_(channel_scales(wl, layer, device)[None])
        v = _normal((wl.batch, wl.n_kv_heads, wl.head_dim),
                    _generator(device, wl.seed, "dv", layer, step), device)
        qs.append(q)
        ks.append(k)
        vs.append(v)
    dt = wl.torch_dtype
    return (torch.stack(qs).to(dt), torch.stack(ks).to(dt), torch.stack(vs).to(dt))


def to_f64(t: torch.Tensor) -> np.ndarray:
    """Exact float64 copy of a tensor's values (bf16 and fp32 embed exactly)."""
    return t.detach().to("cpu", torch.float64).numpy()


def synthetic_votes(seed: int, units: int, prefix: int, levels: int = 0, device="cpu") -> torch.Tensor:
    """fp32 [units][prefix] non-negative vote arrays for selection checks.

    levels > 0 quantises the values to that many levels, which makes many exact
    ties; levels == 0 keeps continuous values.
    """
    g = _generator(device, seed, "votes")
    x = torch.rand((units, prefix), generator=g, device=device, dtype=torch.float32)
    if levels > 0:
        x = torch.floor(x * levels) / levels
    return x * 0.01


def decode_caches(wl: Workload, layer: int, cap: int, device="cpu"):
    """Seeded K/V caches [B][Hkv][cap][d] of one layer for decode checks
    (keys with the layer's channel scales, values N(0, 1))."""
    shape = (wl.batch, wl.n_kv_heads, cap, wl.head_dim)
    k = _normal(shape, _generator(device, wl.seed, "ck", layer), device)
    if wl.kv_dist == "scaled_sinks":
        k.mul_(channel_scales(wl, layer, device)[None, :, None, :])
    v = _normal(shape, _generator(device, wl.seed, "cv", layer), device)
    return k.to(wl.torch_dtype), v.to(wl.torch_dtype)


def perturb_draws(wl: Workload, layer: int, n_rows: int, device="cpu") -> torch.Tensor:
    """fp32 [B][Hkv][n_rows][d] standard normal draws for one layer's Value
    perturbation (one d-vector per eligible position)."""
    shape = (wl.batch, wl.n_kv_heads, n_rows, wl.head_dim)
    return _normal(shape, _generator(device, wl.seed, "eps", layer), device)


def window_logits(seed: int, n_sets: int, n_pos: int, vocab: int, dtype=torch.float32,
                  device="cpu", sigmas=None):
    """(p [n_pos][vocab], q [n_sets][n_pos][vocab]) synthetic output logits of a
    reference run and of n_sets perturbed runs over an evaluation window.

    p = 2.5 N(0, 1) with +12 on four random tokens per position; q[s] = p +
    sigma_s N(0, 1), sigma_s spaced from 0.02 to 0.3 unless given.
    """
    g = _generator(device, seed, "lp")
    p = 2.5 * _normal((n_pos, vocab), g, device)
    top = torch.randint(0, vocab, (n_pos, 4), generator=g, device=device)
    p.scatter_add_(1, top, torch.full((n_pos, 4), 12.0, device=device))
    if sigmas is None:
        sigmas = [0.02 + 0.28 * s / max(1, n_sets - 1) for s in range(n_sets)]
    gq = _generator(device, seed, "lq")
    q = torch.empty((n_sets, n_pos, vocab), device=device, dtype=torch.float32)
    for s in range(n_sets):
        q[s] = p + float(sigmas[s]) * _normal((n_pos, vocab), gq, device)
    return p.to(dtype), q.to(dtype)
