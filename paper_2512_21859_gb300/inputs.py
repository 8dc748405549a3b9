"""Seeded synthetic workloads for the eviction + decode-attention path.

This module only draws inputs. It holds none of the scoring, pooling,
selection or attention arithmetic: both the CUDA path and the CPU oracle
receive the arrays it returns, so they see identical bytes.

The paper's experiments run Qwen2.5-7B-Instruct on LongBench (Section
"Experimental Setup"); neither the weights nor the dataset are used here.
Random tensors with the same attention shapes stand in for them:

* queries ~ N(0, 1);
* keys and values ~ N(0, 1)/sqrt(d) for the bf16 model shapes (unit-norm
  rows on average), N(0, 1) for the small fp32 case;
* "heavy hitter" prefix positions whose keys are pushed towards the mean
  window query of their KV-head group, so that a correct scorer must keep
  them (and, through the max-pool, their neighbours);
* for the 128K shape, a milder push on the last 2048 prefix positions
  (a recency band).

bf16 tensors are returned as uint16 bit patterns (round-to-nearest-even
from float32); ``bf16_to_f32`` turns them back into exact float32 values.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional

import numpy as np

__all__ = [
    "Workload",
    "WORKLOADS",
    "f32_to_bf16",
    "bf16_to_f32",
    "as_f32",
    "request_shapes",
    "make_layer",
    "make_decode_step",
]


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and value recipe of one synthetic workload."""

    name: str
    layers: int
    hq: int
    hkv: int
    head_dim: int
    dtype: str  # "f32" or "bf16"
    batch: int
    window: int
    pool_k: int
    decode_steps: int
    seed: int
    # prompt lengths: fixed, or drawn uniformly from [n_lo, n_hi] per request
    n_fixed: Optional[int] = None
    n_lo: int = 0
    n_hi: int = 0
    # eviction ratio: fixed, or drawn per request from alpha_choices
    alpha: Optional[float] = None
    alpha_choices: tuple = ()
    # heavy hitters: an absolute count, or a fraction of the prefix
    heavy_count: Optional[int] = None
    heavy_frac: float = 0.0
    heavy_scale: float = 3.0
    # True: keys/values scaled by 1/sqrt(d) and the push is heavy_scale * unit
    # direction of the mean window query; False: push is heavy_scale * mean query
    unit_keys: bool = True
    recency_band: int = 0
    recency_scale: float = 1.0
    # alphas the workload is swept over (informational; the bench picks one)
    alpha_sweep: tuple = ()

    @property
    def group(self) -> int:
        return self.hq // self.hkv


WORKLOADS: Dict[str, Workload] = {
    # 1 layer, 4q/2kv, d 64, fp32, N 512, W 16, pool 7, alpha 0.5, 16 decode steps
    "tiny": Workload(
        name="tiny", layers=1, hq=4, hkv=2, head_dim=64, dtype="f32", batch=1,
        window=16, pool_k=7, decode_steps=16, seed=0, n_fixed=512, alpha=0.5,
        heavy_count=5, unit_keys=False),
    # 28 layers, 28q/4kv, d 128, bf16, N 4096, W 32, alpha in {0,.25,.5,.75}
    "7b": Workload(
        name="7b", layers=28, hq=28, hkv=4, head_dim=128, dtype="bf16", batch=1,
        window=32, pool_k=7, decode_steps=256, seed=1, n_fixed=4096, alpha=0.5,
        heavy_frac=0.01, alpha_sweep=(0.0, 0.25, 0.5, 0.75)),
    # same shape, N 32768, alpha swept 0.00..0.95 in steps of 0.05
    "32k": Workload(
        name="32k", layers=28, hq=28, hkv=4, head_dim=128, dtype="bf16", batch=1,
        window=32, pool_k=7, decode_steps=512, seed=2, n_fixed=32768, alpha=0.5,
        heavy_frac=0.01,
        alpha_sweep=tuple(round(0.05 * i, 2) for i in range(20))),
    # 16 requests, N_b ~ U{1024..16384}, alpha_b from {.1,.3,.5,.7,.9}
    "ragged": Workload(
        name="ragged", layers=28, hq=28, hkv=4, head_dim=128, dtype="bf16",
        batch=16, window=32, pool_k=7, decode_steps=256, seed=3, n_lo=1024,
        n_hi=16384, alpha_choices=(0.1, 0.3, 0.5, 0.7, 0.9), heavy_frac=0.01),
    # 32 layers, 32q/8kv, d 128, bf16, N 131072, W 64, alpha 0.9
    "128k": Workload(
        name="128k", layers=32, hq=32, hkv=8, head_dim=128, dtype="bf16",
        batch=1, window=64, pool_k=7, decode_steps=1024, seed=4,
        n_fixed=131072, alpha=0.9, heavy_frac=0.005, recency_band=2048),
}


# ----------------------------------------------------------------------------
# bf16 storage (bit patterns in uint16)
# ----------------------------------------------------------------------------

def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); returns uint16 bits."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    out = np.empty(b.shape, dtype=np.uint16)
    flat_b, flat_o = b.reshape(-1), out.reshape(-1)
    step = 1 << 22
    for s in range(0, flat_b.size, step):
        chunk = flat_b[s:s + step]
        r = chunk >> np.uint32(16)
        r &= np.uint32(1)
        r += np.uint32(0x7FFF)
        r += chunk
        r >>= np.uint32(16)
        flat_o[s:s + step] = r
    return out


def bf16_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact float32 values of bf16 bit patterns."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32)
            << np.uint32(16)).view(np.float32)


def as_f32(x: np.ndarray, dtype: str) -> np.ndarray:
    """Storage array (float32, or uint16 bf16 bits) -> float32 values."""
    return bf16_to_f32(x) if dtype == "bf16" else np.asarray(x, dtype=np.float32)


def _store(x: np.ndarray, dtype: str) -> np.ndarray:
    return f32_to_bf16(x) if dtype == "bf16" else np.ascontiguousarray(x, np.float32)


# ----------------------------------------------------------------------------
# shapes
# ----------------------------------------------------------------------------

def request_shapes(wl: Workload, alpha: Optional[float] = None):
    """Per-request prompt lengths (int64) and eviction ratios (float64).

    ``alpha`` overrides the workload's own ratio for every request.
    """
    if wl.n_fixed is not None:
        n = np.full(wl.batch, wl.n_fixed, dtype=np.int64)
    else:
        rng = np.random.Generator(np.random.PCG64(wl.seed * 1000 + 999))
        n = rng.integers(wl.n_lo, wl.n_hi + 1, size=wl.batch).astype(np.int64)
    if alpha is not None:
        a = np.full(wl.batch, float(alpha), dtype=np.float64)
    elif wl.alpha is not None:
        a = np.full(wl.batch, float(wl.alpha), dtype=np.float64)
    else:
        rng = np.random.Generator(np.random.PCG64(wl.seed * 1000 + 998))
        a = rng.choice(np.asarray(wl.alpha_choices, np.float64), size=wl.batch)
    return n, a


def _normal(rng, shape, scale=1.0):
    x = rng.standard_normal(size=shape, dtype=np.float32)
    if scale != 1.0:
        x *= np.float32(scale)
    return x


def make_layer(wl: Workload, layer: int = 0, alpha: Optional[float] = None,
               n_override: Optional[List[int]] = None) -> dict:
    """One layer's eviction inputs.

    Returns a dict with
      q_win  [B][Hq][W][d]        storage dtype
      K, V   [Hkv][sum N][d]      storage dtype (requests packed along rows)
      n      [B] int64, alpha [B] float64, kv_offset [B] int64
      heavy  list of per-request int64 arrays of planted prefix positions
    ``n_override`` replaces the prompt lengths (used for small parity cases).
    """
    n, a = request_shapes(wl, alpha)
    if n_override is not None:
        n = np.asarray(n_override, dtype=np.int64)
        a = np.resize(a, n.shape[0]).astype(np.float64)
    B = n.shape[0]
    d, W, G = wl.head_dim, wl.window, wl.group
    rng = np.random.Generator(np.random.PCG64(wl.seed * 1000 + layer))
    kv_offset = np.zeros(B, dtype=np.int64)
    kv_offset[1:] = np.cumsum(n)[:-1]
    rows = int(n.sum())
    kscale = 1.0 / np.sqrt(d) if wl.unit_keys else 1.0

    q_win = _normal(rng, (B, wl.hq, W, d))
    K = _normal(rng, (wl.hkv, rows, d), kscale)
    V = _normal(rng, (wl.hkv, rows, d), kscale)

    heavy = []
    for b in range(B):
        P = int(n[b]) - W
        cnt = wl.heavy_count if wl.heavy_count is not None else int(round(wl.heavy_frac * P))
        cnt = max(0, min(cnt, P))
        pos = np.sort(rng.choice(P, size=cnt, replace=False)).astype(np.int64) if cnt else \
            np.zeros(0, np.int64)
        heavy.append(pos)
        off = int(kv_offset[b])
        for g in range(wl.hkv):
            qbar = q_win[b, g * G:(g + 1) * G].reshape(-1, d).mean(axis=0)
            if wl.unit_keys:
                push = qbar / np.float32(np.linalg.norm(qbar) + 1e-30)
            else:
                push = qbar
            K[g, off + pos] += np.float32(wl.heavy_scale) * push
            if wl.recency_band:
                lo = max(0, P - wl.recency_band)
                K[g, off + lo:off + P] += np.float32(wl.recency_scale) * push

    return {
        "q_win": _store(q_win, wl.dtype),
        "K": _store(K, wl.dtype),
        "V": _store(V, wl.dtype),
        "n": n,
        "alpha": a,
        "kv_offset": kv_offset,
        "heavy": heavy,
    }


def make_decode_step(wl: Workload, layer: int, step: int, batch: int) -> dict:
    """Decode step ``step`` (1-based): the new query and the new token's K/V row.

    Returns q [B][Hq][d], k_new / v_new [Hkv][B][d] in storage dtype.
    """
    d = wl.head_dim
    rng = np.random.Generator(np.random.PCG64((wl.seed * 1000 + layer) * 1000003 + step))
    kscale = 1.0 / np.sqrt(d) if wl.unit_keys else 1.0
    q = _normal(rng, (batch, wl.hq, d))
    k_new = _normal(rng, (wl.hkv, batch, d), kscale)
    v_new = _normal(rng, (wl.hkv, batch, d), kscale)
    return {"q": _store(q, wl.dtype), "k_new": _store(k_new, wl.dtype),
            "v_new": _store(v_new, wl.dtype)}
