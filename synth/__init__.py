"""Seeded synthetic inputs for SelKV: GQA-shaped KV caches, observation-window queries and
decode-step tokens.

This module serves both the fp64 oracle and the CUDA library's tests and benchmark. It holds
no arithmetic of the method itself: it only draws random numbers, lays them out and rounds
them to the storage dtype.

Recipe (one unit = one (layer, sequence, KV head)):

* The sequence is cut into segments.  Either fixed-length segments, or lengths drawn
  uniformly from an integer range with the last segment truncated at n.
* Each segment draws independent N(0, I_d) centroids for K and for V, and a noise scale
  sigma (fixed, or uniform in a range per segment).  Token t of the segment is
  centroid + sigma * N(0, I_d), for K and V separately (same segmentation, same sigma).
* Heavy hitters: a set of positions, drawn uniformly without replacement per (layer,
  sequence) and shared by every KV head, has its key rows multiplied by 4.
* Observation-window queries Q_obs[h] (the last W query rows of each query head) are drawn
  with the same segmented distribution, independently per query head.
* Decode steps draw fresh i.i.d. N(0, 1) queries q[b][h] and fresh N(0, 1) key/value rows
  appended to the cache.
* Values are drawn in fp32 and rounded (round-to-nearest-even) to bf16 where the workload
  stores bf16; both sides of every comparison consume the same rounded values.

Every stream is a numpy PCG64 generator seeded by SeedSequence([seed, layer, seq, unit,
purpose]), so any unit can be regenerated alone and threads may generate units in any order.
"""
from __future__ import annotations

import dataclasses
import math
from concurrent.futures import ThreadPoolExecutor
from typing import Optional, Sequence

import numpy as np

# purpose codes for SeedSequence streams
_KV, _Q, _HEAVY, _DECODE, _LENGTHS = 0, 1, 2, 3, 4


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic workload: attention shape, cache length, budget and generator recipe."""
    name: str
    dtype: str                    # "bf16" or "fp32": storage dtype of K, V, Q_obs, q
    batch: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    obs_window: int
    n: int                        # prefill length (the capacity n_cap when ragged)
    layers: int
    rho: float                    # KV retention ratio
    decode_steps: int
    seg_len: tuple                # ("fixed", L) or ("uniform", lo, hi)
    sigma: tuple                  # (lo, hi); lo == hi means a fixed sigma
    heavy: tuple                  # ("count", k) or ("frac", f)
    ragged: Optional[tuple] = None  # (lo_frac, hi_frac): n_b ~ U[lo*n, hi*n]
    seed: int = 0

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


_LLAMA = dict(dtype="bf16", num_q_heads=32, num_kv_heads=8, head_dim=128, obs_window=64,
              seg_len=("uniform", 4, 64), sigma=(0.1, 0.8), heavy=("frac", 0.01))

#: The five workloads.  tiny: single layer, fp32, GQA group 2.  llama_layer: one
#: Llama-3-8B-shaped layer at 16k.  llama_32l_b4: 32 layers, batch 4, 32k.  long_100k: 32
#: layers at 100k context.  sweep(): the batched serving grid with ragged lengths.
#: longchat_mha_31k: the MHA shape of the per-head selection mode.
WORKLOADS = {
    "tiny": Workload(name="tiny", dtype="fp32", batch=1, num_q_heads=4, num_kv_heads=2,
                     head_dim=64, obs_window=32, n=1024, layers=1, rho=0.25, decode_steps=16,
                     seg_len=("fixed", 16), sigma=(0.3, 0.3), heavy=("count", 8)),
    "llama_layer": Workload(name="llama_layer", batch=1, n=16384, layers=1, rho=0.25,
                            decode_steps=128, **_LLAMA),
    "llama_32l_b4": Workload(name="llama_32l_b4", batch=4, n=32768, layers=32, rho=0.25,
                             decode_steps=256, **_LLAMA),
    "long_100k": Workload(name="long_100k", batch=1, n=100000, layers=32, rho=0.25,
                          decode_steps=256, **_LLAMA),
    # a wider GQA group (Llama-3-70B attention shape: 64 query heads over 8 KV heads, G = 8),
    # one layer at 16k: G W = 512 window rows per KV head
    "llama70b_layer": Workload(name="llama70b_layer", batch=1, n=16384, layers=1, rho=0.25,
                               decode_steps=128, **dict(_LLAMA, num_q_heads=64)),
    # the same G = 8 shape over 32 layers at 100k context (the long-context setting of the paper
    # with the wider group)
    "llama70b_100k": Workload(name="llama70b_100k", batch=1, n=100000, layers=32, rho=0.25,
                              decode_steps=256, **dict(_LLAMA, num_q_heads=64)),
    # the paper's MHA setting (LongChat-7B-shaped: 32 query heads = 32 KV heads, 31,500-token
    # inputs, W = 32), for the per-head selection mode
    "longchat_mha_31k": Workload(name="longchat_mha_31k", batch=1, n=31500, layers=32, rho=0.25,
                                 decode_steps=256, **dict(_LLAMA, num_kv_heads=32, obs_window=32)),
}


def sweep(batch: int, n: int, rho: float) -> Workload:
    """One point of the batched serving sweep (ragged n_b ~ U[0.5 n, n], one layer)."""
    return Workload(name=f"sweep_b{batch}_n{n}_r{int(round(rho * 100))}", batch=batch, n=n,
                    layers=1, rho=rho, decode_steps=16, ragged=(0.5, 1.0), **_LLAMA)


SWEEP_POINTS = [(b, n, r) for b in (1, 8, 32, 64) for n in (8192, 32768, 131072)
                for r in (0.10, 0.25, 0.50)]


def _rng(*key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(list(key))))


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even); returned as fp32 values."""
    return bf16_bits_to_f32(f32_to_bf16_bits(x))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns (uint16), round to nearest even.  Inputs are finite."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def seq_lengths(wl: Workload) -> np.ndarray:
    """Prefill length n_b of every sequence (all equal to n unless the workload is ragged)."""
    if wl.ragged is None:
        return np.full(wl.batch, wl.n, dtype=np.int32)
    lo = int(math.ceil(wl.ragged[0] * wl.n))
    hi = int(math.floor(wl.ragged[1] * wl.n))
    out = np.empty(wl.batch, dtype=np.int32)
    for b in range(wl.batch):
        out[b] = _rng(wl.seed, 0, b, 0, _LENGTHS).integers(lo, hi + 1)
    return out


def _segmented(rng: np.random.Generator, n: int, d: int, wl: Workload, pair: bool):
    """Segmented-centroid rows: one (or, with pair=True, two sharing the segmentation) [n, d]."""
    kind = wl.seg_len[0]
    if kind == "fixed":
        L = wl.seg_len[1]
        lens = np.full((n + L - 1) // L, L, dtype=np.int64)
    else:
        lo, hi = wl.seg_len[1], wl.seg_len[2]
        lens = rng.integers(lo, hi + 1, size=n // lo + 1)
    ends = np.cumsum(lens)
    nseg = int(np.searchsorted(ends, n, side="left")) + 1
    lens = lens[:nseg].copy()
    lens[-1] -= int(ends[nseg - 1] - n)
    seg = np.repeat(np.arange(nseg), lens)
    lo_s, hi_s = wl.sigma
    sig = (np.full(nseg, lo_s, dtype=np.float32) if lo_s == hi_s
           else rng.uniform(lo_s, hi_s, size=nseg).astype(np.float32))
    outs = []
    for _ in range(2 if pair else 1):
        cent = rng.standard_normal((nseg, d), dtype=np.float32)
        noise = rng.standard_normal((n, d), dtype=np.float32)
        noise *= sig[seg][:, None]
        noise += cent[seg]
        outs.append(noise)
    return outs


def heavy_positions(wl: Workload, layer: int, b: int, n_b: int) -> np.ndarray:
    kind, v = wl.heavy
    k = int(v) if kind == "count" else int(math.floor(v * n_b))
    k = min(k, n_b)
    return np.sort(_rng(wl.seed, layer, b, 0, _HEAVY).choice(n_b, size=k, replace=False))


def _store(x: np.ndarray, dtype: str) -> np.ndarray:
    return round_bf16(x) if dtype == "bf16" else x


def gen_sequence(wl: Workload, layer: int, b: int, threads: int = 1) -> dict:
    """Sequence b of gen_layer(wl, layer) alone (the same values): K, V [Hkv][n_b][d] and
    Q_obs [Hq][W][d] (fp32 arrays holding storage-dtype values) and its length n_b."""
    Hq, Hkv, d, W = wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.obs_window
    n_b = int(seq_lengths(wl)[b])
    K = np.empty((Hkv, n_b, d), dtype=np.float32)
    V = np.empty((Hkv, n_b, d), dtype=np.float32)
    Q = np.empty((Hq, W, d), dtype=np.float32)
    heavy = heavy_positions(wl, layer, b, n_b)

    def kv_unit(kv):
        k, v = _segmented(_rng(wl.seed, layer, b, kv, _KV), n_b, d, wl, pair=True)
        k[heavy] *= 4.0
        K[kv] = _store(k, wl.dtype)
        V[kv] = _store(v, wl.dtype)

    def q_unit(h):
        (q,) = _segmented(_rng(wl.seed, layer, b, h, _Q), W, d, wl, pair=False)
        Q[h] = _store(q, wl.dtype)

    if threads > 1:
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(kv_unit, range(Hkv)))
            list(ex.map(q_unit, range(Hq)))
    else:
        for kv in range(Hkv):
            kv_unit(kv)
        for h in range(Hq):
            q_unit(h)
    return dict(K=K, V=V, Q_obs=Q, n=n_b)


def gen_layer(wl: Workload, layer: int, threads: int = 1) -> dict:
    """K, V [B][Hkv][n_cap][d], Q_obs [B][Hq][W][d] (fp32 arrays holding storage-dtype
    values; rows at or beyond n_b are zero) and n_len [B]."""
    B, Hq, Hkv, d, W = wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.obs_window
    n_len = seq_lengths(wl)
    n_cap = wl.n
    K = np.zeros((B, Hkv, n_cap, d), dtype=np.float32)
    V = np.zeros((B, Hkv, n_cap, d), dtype=np.float32)
    Q = np.zeros((B, Hq, W, d), dtype=np.float32)

    def kv_unit(args):
        b, kv = args
        n_b = int(n_len[b])
        k, v = _segmented(_rng(wl.seed, layer, b, kv, _KV), n_b, d, wl, pair=True)
        k[heavy_positions(wl, layer, b, n_b)] *= 4.0
        K[b, kv, :n_b] = _store(k, wl.dtype)
        V[b, kv, :n_b] = _store(v, wl.dtype)

    def q_unit(args):
        b, h = args
        (q,) = _segmented(_rng(wl.seed, layer, b, h, _Q), W, d, wl, pair=False)
        Q[b, h] = _store(q, wl.dtype)

    units_kv = [(b, kv) for b in range(B) for kv in range(Hkv)]
    units_q = [(b, h) for b in range(B) for h in range(Hq)]
    if threads > 1:
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(kv_unit, units_kv))
            list(ex.map(q_unit, units_q))
    else:
        for u in units_kv:
            kv_unit(u)
        for u in units_q:
            q_unit(u)
    return dict(K=K, V=V, Q_obs=Q, n_len=n_len)


def gen_decode(wl: Workload, layer: int, steps: int, start: int = 0) -> dict:
    """Decode-step inputs for `steps` consecutive steps: q [T][B][Hq][d], k_new and v_new
    [T][B][Hkv][d], all i.i.d. N(0, 1) in the storage dtype."""
    B, Hq, Hkv, d = wl.batch, wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    q = np.empty((steps, B, Hq, d), dtype=np.float32)
    k = np.empty((steps, B, Hkv, d), dtype=np.float32)
    v = np.empty((steps, B, Hkv, d), dtype=np.float32)
    for t in range(steps):
        rng = _rng(wl.seed, layer, start + t, 0, _DECODE)
        q[t] = rng.standard_normal((B, Hq, d), dtype=np.float32)
        k[t] = rng.standard_normal((B, Hkv, d), dtype=np.float32)
        v[t] = rng.standard_normal((B, Hkv, d), dtype=np.float32)
    return dict(q=_store(q, wl.dtype), k_new=_store(k, wl.dtype), v_new=_store(v, wl.dtype))


def workload_names() -> Sequence[str]:
    return list(WORKLOADS)
