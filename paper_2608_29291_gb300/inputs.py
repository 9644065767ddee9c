"""Seeded synthetic inputs for the token-routed compacted block.

This module is the one piece shared by the CUDA path (tests, bench, smoke) and the
CPU oracle's tests.  It holds none of the method's arithmetic: only

* a counter-based generator, SplitMix64 (Steele, Lea and Flood, "Fast splittable
  pseudorandom number generators", OOPSLA 2014), evaluated at counter i as
  ``mix64(seed + (i + 1) * 0x9E3779B97F4A7C15)``;
* uniforms and Box-Muller normals drawn from it, in fp64;
* conversion of the drawn fp32 values to bf16 bit patterns (round to nearest even);
* a Fisher-Yates draw of the static FFN channel keep set (Sec. 3.4, FFN pruning:
  the static mask P_l is an input of the method, not something it computes);
* the workload descriptions (shapes, routable ranges, keep counts, seeds).

Everything is numpy on the host, so both sides read the very same bit patterns.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 22


def _mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function on a uint64 array (wrapping arithmetic), in place."""
    t = np.empty_like(z)
    np.right_shift(z, np.uint64(30), out=t)
    z ^= t
    z *= _M1
    np.right_shift(z, np.uint64(27), out=t)
    z ^= t
    z *= _M2
    np.right_shift(z, np.uint64(31), out=t)
    z ^= t
    return z


def _fnv1a64(name: str) -> int:
    h = 0xCBF29CE484222325
    for b in name.encode():
        h ^= b
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def substream_seed(seed: int, name: str) -> int:
    """Seed of the named tensor's stream: mix64(seed XOR fnv1a64(name))."""
    z = np.array([(seed ^ _fnv1a64(name)) & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64)
    with np.errstate(over="ignore"):
        return int(_mix64(z)[0])


def raw_u64(seed: int, start: int, count: int) -> np.ndarray:
    """Counter-based SplitMix64 words for counters start .. start+count-1."""
    with np.errstate(over="ignore"):
        z = np.arange(start + 1, start + count + 1, dtype=np.uint64)
        z *= _GAMMA
        z += np.uint64(seed)
        return _mix64(z)


def uniform01(seed: int, count: int, start: int = 0) -> np.ndarray:
    """fp64 uniforms in the open interval (0, 1): ((w >> 11) + 0.5) * 2^-53."""
    w = raw_u64(seed, start, count)
    return ((w >> np.uint64(11)).astype(np.float64) + 0.5) * (2.0 ** -53)


def normal(seed: int, count: int) -> np.ndarray:
    """fp64 standard normals by Box-Muller; element i uses counters 2i and 2i+1."""
    out = np.empty(count, dtype=np.float64)
    for s in range(0, count, _CHUNK):
        n = min(_CHUNK, count - s)
        u = uniform01(seed, 2 * n, start=2 * s)
        u1, u2 = u[0::2], u[1::2]
        out[s:s + n] = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * math.pi * u2)
    return out


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (nearest, ties to even); returns uint16 bit patterns.

    Inputs here are finite draws, so no NaN handling is needed.
    """
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))
    return (b >> np.uint64(16)).astype(np.uint16)


def bf16_normal(seed: int, name: str, shape, std: float) -> np.ndarray:
    """bf16 bit patterns of N(0, std^2) draws, uint16 array of the given shape.

    One SplitMix64 word per element: its top 24 bits and its low 24 bits give
    the two Box-Muller uniforms ((k + 0.5) * 2^-24), enough for a bf16 result.
    """
    count = int(np.prod(shape))
    out = np.empty(count, dtype=np.uint16)
    ss = substream_seed(seed, name)
    for s in range(0, count, _CHUNK):
        n = min(_CHUNK, count - s)
        w = raw_u64(ss, s, n)
        u1 = ((w >> np.uint64(40)).astype(np.float64) + 0.5) * (2.0 ** -24)
        u2 = ((w & np.uint64(0xFFFFFF)).astype(np.float64) + 0.5) * (2.0 ** -24)
        z = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * math.pi * u2)
        out[s:s + n] = f32_to_bf16_bits((z * std).astype(np.float32))
    return out.reshape(shape)


def f32_normal(seed: int, name: str, shape, std: float) -> np.ndarray:
    count = int(np.prod(shape))
    return (normal(substream_seed(seed, name), count) * std).astype(np.float32).reshape(shape)


def f32_uniform(seed: int, name: str, count: int) -> np.ndarray:
    """fp32 uniforms in [0, 1) with 24 random bits each (exact in fp32)."""
    w = raw_u64(substream_seed(seed, name), 0, count)
    return ((w >> np.uint64(40)).astype(np.float64) * (2.0 ** -24)).astype(np.float32)


def channel_keep_set(seed: int, name: str, n_channels: int, n_keep: int) -> np.ndarray:
    """Static FFN channel keep set: the first n_keep entries of a Fisher-Yates
    permutation of [0, n_channels), sorted ascending (int32)."""
    perm = np.arange(n_channels, dtype=np.int64)
    w = raw_u64(substream_seed(seed, name), 0, max(n_channels - 1, 0))
    for k, i in enumerate(range(n_channels - 1, 0, -1)):
        j = int(w[k] % np.uint64(i + 1))
        perm[i], perm[j] = perm[j], perm[i]
    return np.sort(perm[:n_keep]).astype(np.int32)


def keep_count(ratio: float, n_routable: int) -> int:
    """Routable tokens kept per sequence: K = floor(ratio * N_r + 0.5) in fp64,
    clamped to [0, N_r] (the keep ratio is r = K/N, App. A.2 training table)."""
    k = int(math.floor(ratio * n_routable + 0.5))
    return max(0, min(n_routable, k))


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and synthesis recipe of one routed-block workload."""
    name: str
    B: int
    N: int
    d: int
    I: int            # full SwiGLU intermediate width
    C: int            # kept intermediate channels
    r0: int           # routable token range [r0, r1); the rest is always kept
    r1: int
    K: int            # routable tokens kept per sequence
    Hc: int           # core scorer hidden width
    He: int           # expansion scorer hidden width (0: understanding only)
    E: int            # sinusoidal embedding width of the expansion
    task: int         # 0 = understanding, 1 = generation
    n_segments: int = 1
    t_fixed: Optional[float] = None   # None: t_b ~ U[0,1) per sequence
    visual_lognormal: bool = False    # scale routable rows by lognormal(0, 0.5)
    core_bias: bool = False
    seed: int = 0

    @property
    def k_tot(self) -> int:
        return self.K + (self.N - (self.r1 - self.r0))

    @property
    def M(self) -> int:
        return self.B * self.k_tot

    def ffn_flops(self) -> int:
        return 6 * self.M * self.d * self.C

    def score_flops(self) -> int:
        h = self.Hc + (self.He if self.task == 1 else 0)
        return 2 * self.B * self.N * self.d * h

    def attn_heads(self):
        """(query heads, key/value heads) of the Qwen2.5 backbone with this
        width (head size 128): 12/2 for the 1.5B model, 28/4 for the 7B."""
        known = {1536: (12, 2), 3584: (28, 4)}
        return known.get(self.d, (max(1, self.d // 128), 1))

    def attn_flops(self, causal: bool) -> int:
        """Q K^T and P V over the packed sequences (only the admissible pairs
        when causal)."""
        Hq, _ = self.attn_heads()
        L = self.k_tot
        pairs = L * (L + 1) // 2 if causal else L * L
        return 4 * self.B * Hq * 128 * pairs


def tiny() -> Workload:
    return Workload("tiny_b1_n256_d256", B=1, N=256, d=256, I=1024, C=512, r0=0, r1=256,
                    K=128, Hc=64, He=64, E=64, task=1, t_fixed=0.5)


def und_1p5b() -> Workload:
    return Workload("und_1p5b_b4_n1024_d1536", B=4, N=1024, d=1536, I=8960,
                    C=keep_count(0.75, 8960), r0=0, r1=729, K=keep_count(0.4, 729),
                    Hc=256, He=0, E=0, task=0, visual_lognormal=True)


def gen_1p5b() -> Workload:
    return Workload("gen_1p5b_b8_n1088_d1536", B=8, N=1088, d=1536, I=8960,
                    C=keep_count(0.5, 8960), r0=64, r1=1088, K=keep_count(0.5, 1024),
                    Hc=256, He=256, E=256, task=1)


def long_7b() -> Workload:
    return Workload("long_7b_b2_n4096_d3584", B=2, N=4096, d=3584, I=18944,
                    C=keep_count(0.5, 18944), r0=0, r1=3840, K=keep_count(0.3, 3840),
                    Hc=512, He=512, E=256, task=1, t_fixed=0.25)


def sweep(n: int, token_ratio: float, ffn_ratio: float) -> Workload:
    return Workload(f"sweep_7b_n{n}_r{token_ratio}_f{ffn_ratio}", B=1, N=n, d=3584, I=18944,
                    C=keep_count(ffn_ratio, 18944), r0=0, r1=n, K=keep_count(token_ratio, n),
                    Hc=512, He=512, E=256, task=1)


WORKLOADS = {"tiny": tiny, "und_1p5b": und_1p5b, "gen_1p5b": gen_1p5b, "long_7b": long_7b}


def make_inputs(w: Workload, ffn_weights: Optional[tuple] = None) -> dict:
    """All tensors of one workload as host numpy arrays (bf16 as uint16 bits).

    Recipe: h ~ N(0,1) (routable rows times lognormal(0, 0.5) per row when
    ``visual_lognormal``); every weight ~ N(0, 1/fan_in); scorer output vectors
    w2 fp32; t_b fixed or ~ U[0,1); channel keep set by Fisher-Yates.
    ``ffn_weights`` may pass (Wg, Wu, WdT) drawn earlier for the same (seed, I, d).
    """
    s = w.seed
    h_shape = (w.B, w.N, w.d)
    if w.visual_lognormal:
        z = normal(substream_seed(s, "h"), w.B * w.N * w.d).reshape(h_shape)
        scale = np.exp(0.5 * normal(substream_seed(s, "h_rowscale"), w.B * w.N)).reshape(w.B, w.N)
        scale[:, :w.r0] = 1.0
        scale[:, w.r1:] = 1.0
        h = f32_to_bf16_bits((z * scale[:, :, None]).astype(np.float32)).reshape(h_shape)
    else:
        h = bf16_normal(s, "h", h_shape, 1.0)
    inp = {
        "h": h,
        "W1": bf16_normal(s, "W1", (w.Hc, w.d), 1.0 / math.sqrt(w.d)),
        "w2": f32_normal(s, "w2", (w.Hc,), 1.0 / math.sqrt(w.Hc)),
        "b1": f32_normal(s, "b1", (w.Hc,), 0.1) if w.core_bias else None,
        "Wg": ffn_weights[0] if ffn_weights else bf16_normal(s, "Wg", (w.I, w.d), 1.0 / math.sqrt(w.d)),
        "Wu": ffn_weights[1] if ffn_weights else bf16_normal(s, "Wu", (w.I, w.d), 1.0 / math.sqrt(w.d)),
        "WdT": ffn_weights[2] if ffn_weights else bf16_normal(s, "WdT", (w.I, w.d), 1.0 / math.sqrt(w.I)),
        "chan": channel_keep_set(s, "chan", w.I, w.C),
    }
    if w.t_fixed is not None:
        inp["t"] = np.full(w.B, w.t_fixed, dtype=np.float32)
    else:
        inp["t"] = f32_uniform(s, "t", w.B)
    if w.He > 0:
        S = w.n_segments
        inp["W1e"] = bf16_normal(s, "W1e", (S, w.He, w.d), 1.0 / math.sqrt(w.d))
        inp["w2e"] = f32_normal(s, "w2e", (S, w.He), 1.0 / math.sqrt(w.He))
        inp["Ue"] = bf16_normal(s, "Ue", (S, w.He, w.E), 1.0 / math.sqrt(w.E)) if w.E > 0 else None
        inp["b1e"] = None
    return inp
