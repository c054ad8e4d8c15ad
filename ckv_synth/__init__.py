"""Seeded synthetic inputs for the CompressKV prefill-time KV-compression step.

This module draws the inputs that both the CUDA path and the fp64 oracle consume: window
queries, keys, values, per-layer head-selection masks, per-layer budgets, sequence lengths and
planted structure.  It holds none of the method's arithmetic (no attention, pooling, selection
or budget allocation); it only decides *what data* the method is run on.

Random numbers come from a counter-based generator: output ``i`` of stream ``key`` is the
SplitMix64 finaliser (Steele, Lea & Flood, "Fast splittable pseudorandom number generators",
OOPSLA 2014) applied to ``key + (i + 1) * 0x9E3779B97F4A7C15`` (mod 2**64).  Normals use the
Box-Muller transform on the two 32-bit halves of each 64-bit draw, in double precision, rounded
to float32.  Every tensor of every layer has its own stream, so any layer (or any subset of
layers) is generated on its own, in any order, with the same bits.  The bulk draws run in a
small C library (``synth.c``, built with gcc on first use, OpenMP over the draws); the stream
itself is also written out in numpy (``uniform_u64``), and the two agree bit for bit.

Recipe per tensor (generate fp32 -> outlier channels -> planted keys -> round to bf16 once):
  * Q window rows, K, V ~ N(0, 1).
  * K: per (layer, KV head) ``outlier_channels`` seeded channels scaled by ``outlier_scale``
    (the per-channel key outliers of Llama-family models).
  * Planted keys: ``k = beta * u_g (+ N(0,1) noise)`` with ``u_g`` the unit mean of KV group
    g's selected window query rows (after their bf16 rounding), ``beta = c * sqrt(d)``.  Either
    a few isolated tokens (``plant="tokens"``) or one contiguous span at a seeded depth
    (``plant="span"``, the needle-in-a-haystack analogue).
  * Head mask: ``heads_per_group`` distinct heads per (layer, KV group), drawn without
    replacement.
  * Budgets: start every layer at ``budget_mean`` and apply seeded pairwise transfers that keep
    each layer within [budget_min, 3 * budget_mean]; the total stays ``num_layers *
    budget_mean``.  This is only a way to obtain non-uniform layer budgets with a fixed sum;
    it is not the paper's allocation rule.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
import ctypes
import math
import os
import subprocess

import numpy as np

__all__ = [
    "Workload", "LayerInputs", "WORKLOADS", "WORKLOAD_ORDER", "workload",
    "bf16_bits", "bf16_to_f32", "normals", "normals_bf16", "uniform_u64", "build",
]

_GOLDEN = 0x9E3779B97F4A7C15
_M64 = (1 << 64) - 1

# stream kinds (high bits of the stream id)
_K_Q, _K_K, _K_V, _K_OUTLIER, _K_MASK, _K_BUDGET, _K_PLANT_POS, _K_PLANT_NOISE, _K_SEQLEN = range(1, 10)


def _mix64_int(z: int) -> int:
    z &= _M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def _stream_key(seed: int, kind: int, a: int = 0, b: int = 0) -> int:
    sid = (kind << 56) | ((a & 0xFFFFFF) << 32) | (b & 0xFFFFFFFF)
    return _mix64_int(_mix64_int(seed * _GOLDEN + 0x5851F42D4C957F2D) ^ sid)


def uniform_u64(key: int, start: int, count: int) -> np.ndarray:
    """Draws ``start .. start+count-1`` of the counter-based stream ``key`` as uint64."""
    i = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    z = i * np.uint64(_GOLDEN) + np.uint64(key & _M64)
    z ^= z >> np.uint64(30)
    z *= np.uint64(0xBF58476D1CE4E5B9)
    z ^= z >> np.uint64(27)
    z *= np.uint64(0x94D049BB133111EB)
    z ^= z >> np.uint64(31)
    return z


_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB_PATH = os.path.join(_HERE, "libckv_synth.so")
_lib = None


def build(force: bool = False) -> str:
    """Compiles the bulk-draw library (gcc, C11, OpenMP, no FMA contraction) next to this file."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                               "-ffp-contract=off", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        P, I64, U64 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64
        lib.synth_u64.argtypes = [U64, I64, I64, P]
        lib.synth_normals_f32.argtypes = [U64, I64, P]
        lib.synth_normals_bf16.argtypes = [U64, I64, P, I64, P]
        _lib = lib
    return _lib


def uniform_u64_fast(key: int, start: int, count: int) -> np.ndarray:
    """The same draws as ``uniform_u64``, from the C library."""
    out = np.empty(count, dtype=np.uint64)
    _load().synth_u64(key & _M64, start, count, out.ctypes.data_as(ctypes.c_void_p))
    return out


def normals(key: int, count: int) -> np.ndarray:
    """``count`` standard normals (float32) from stream ``key`` (Box-Muller, 2 per draw)."""
    out = np.empty(count, dtype=np.float32)
    _load().synth_normals_f32(key & _M64, count, out.ctypes.data_as(ctypes.c_void_p))
    return out


def normals_bf16(key: int, count: int, scale: np.ndarray | None = None) -> np.ndarray:
    """The first ``count`` normals of stream ``key``, element i multiplied in float32 by
    ``scale.flat[i % scale.size]`` (when given), rounded to bfloat16; returns the uint16 bits."""
    out = np.empty(count, dtype=np.uint16)
    sc = None if scale is None else np.ascontiguousarray(scale, dtype=np.float32).ravel()
    _load().synth_normals_bf16(key & _M64, count, None if sc is None else sc.ctypes.data_as(ctypes.c_void_p),
                               0 if sc is None else sc.size, out.ctypes.data_as(ctypes.c_void_p))
    return out


def _randint(key: int, start: int, count: int, lo: int, hi: int) -> np.ndarray:
    """Integers in [lo, hi] (inclusive), by 64-bit multiply-shift (Lemire) of the stream."""
    z = uniform_u64(key, start, count)
    span = hi - lo + 1
    # (z * span) >> 64 without 128-bit ints: split z into 32-bit halves.
    hi32 = (z >> np.uint64(32)).astype(np.float64)
    lo32 = (z & np.uint64(0xFFFFFFFF)).astype(np.float64)
    frac = (hi32 + lo32 / 4294967296.0) / 4294967296.0
    return lo + np.minimum(np.floor(frac * span).astype(np.int64), span - 1)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (round to nearest, ties to even); returns the uint16 bits."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = ((b >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((b + r) >> np.uint32(16)).astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bfloat16 bits (uint16) to float32."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclass
class LayerInputs:
    """One layer's inputs as bf16 bit patterns (uint16), packed row-major.

    q_win: [S, w, H_q, d] the last ``w`` query rows of every sequence (rows with a negative
           query position, when L_s < w, are present and hold ordinary random values).
    k, v:  [T, H_kv, d] varlen-packed keys / values (T = sum of L_s).
    planted: sequence-local positions of planted keys, [S, n_planted] (empty if none).
    """
    q_win: np.ndarray
    k: np.ndarray
    v: np.ndarray
    planted: np.ndarray


@dataclass(frozen=True)
class Workload:
    name: str
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    seqlens: tuple
    window: int
    heads_per_group: int
    budget_mean: int
    pool_kernel: int = 7
    pool_type: str = "max"           # "max" | "avg"
    head_order: str = "pool_then_sum"  # "pool_then_sum" | "sum_then_pool"
    head_dim: int = 128
    budget_min: int = 32
    budget_uniform: bool = False
    outlier_channels: int = 0
    outlier_scale: float = 10.0
    plant: str = "none"              # "none" | "tokens" | "span"
    plant_count: int = 0
    plant_beta: float = 0.0          # beta / sqrt(d)
    plant_noise: bool = False
    seed: int = 20250802
    description: str = ""
    heads_per_layer: int = 0         # > 0: that many selected heads per layer, from any group
    scope: str = "kv_head"           # "kv_head" | "layer": one selection per KV head / per layer

    # ---- shapes -------------------------------------------------------------------------
    @property
    def num_seqs(self) -> int:
        return len(self.seqlens)

    @property
    def group_size(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def total_tokens(self) -> int:
        return int(sum(self.seqlens))

    def cu_seqlens(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.seqlens)]).astype(np.int32)

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)

    # ---- per-layer head mask and budgets -------------------------------------------------
    def head_mask(self) -> np.ndarray:
        """uint8 [num_layers, H_q]: 1 marks a selected (semantic retrieval) head."""
        m = np.zeros((self.num_layers, self.num_q_heads), dtype=np.uint8)
        if self.heads_per_layer > 0:  # heads_per_layer of the layer's heads, any groups
            n = self.heads_per_layer
            if n > self.num_q_heads:
                raise ValueError("heads_per_layer must be at most num_q_heads")
            for l in range(self.num_layers):
                key = _stream_key(self.seed, _K_MASK, l, 1 << 16)
                order = np.argsort(uniform_u64(key, 0, self.num_q_heads), kind="stable")
                m[l, order[:n]] = 1
            return m
        G, n = self.group_size, self.heads_per_group
        if not 1 <= n <= G:
            raise ValueError("heads_per_group must be in [1, group size]")
        for l in range(self.num_layers):
            for g in range(self.num_kv_heads):
                key = _stream_key(self.seed, _K_MASK, l, g)
                order = np.argsort(uniform_u64(key, 0, G), kind="stable")
                m[l, g * G + order[:n]] = 1
        return m

    def budgets(self) -> np.ndarray:
        """int32 [num_layers]: tokens kept per KV head in each layer, window included."""
        L, mean = self.num_layers, self.budget_mean
        b = np.full(L, mean, dtype=np.int64)
        if self.budget_uniform or L == 1:
            return b.astype(np.int32)
        lo, hi = self.budget_min, 3 * mean
        key = _stream_key(self.seed, _K_BUDGET)
        steps = 8 * L
        pa = _randint(key, 0, steps, 0, L - 1)
        pb = _randint(key, steps, steps, 0, L - 1)
        amt = _randint(key, 2 * steps, steps, 0, mean)
        for a, c, d in zip(pa, pb, amt):
            if a == c:
                continue
            d = int(min(d, b[a] - lo, hi - b[c]))
            if d > 0:
                b[a] -= d
                b[c] += d
        assert b.sum() == L * mean and b.min() >= lo and b.max() <= hi
        return b.astype(np.int32)

    # ---- tensors -------------------------------------------------------------------------
    def layer(self, l: int) -> LayerInputs:
        S, w, Hq, Hkv, d = self.num_seqs, self.window, self.num_q_heads, self.num_kv_heads, self.head_dim
        T, G = self.total_tokens, self.group_size
        cu = self.cu_seqlens()
        q_bits = normals_bf16(_stream_key(self.seed, _K_Q, l), S * w * Hq * d).reshape(S, w, Hq, d)
        scale = None
        if self.outlier_channels:
            scale = np.ones((Hkv, d), dtype=np.float32)
            for g in range(Hkv):
                key = _stream_key(self.seed, _K_OUTLIER, l, g)
                ch = np.argsort(uniform_u64(key, 0, d), kind="stable")[: self.outlier_channels]
                scale[g, ch] = np.float32(self.outlier_scale)
        k_bits = normals_bf16(_stream_key(self.seed, _K_K, l), T * Hkv * d, scale).reshape(T, Hkv, d)
        planted = self._plant(l, q_bits, k_bits, cu)
        v_bits = normals_bf16(_stream_key(self.seed, _K_V, l), T * Hkv * d).reshape(T, Hkv, d)
        return LayerInputs(q_win=q_bits, k=k_bits, v=v_bits, planted=planted)

    def _plant(self, l, q_bits, k_bits, cu) -> np.ndarray:
        """Overwrites the planted keys' rows of ``k_bits`` (bf16 bits) in place."""
        S, w, d, G = self.num_seqs, self.window, self.head_dim, self.group_size
        if self.plant == "none" or self.plant_count == 0:
            return np.zeros((S, 0), dtype=np.int64)
        mask = self.head_mask()[l]
        beta = self.plant_beta * math.sqrt(d)
        qf = bf16_to_f32(q_bits).astype(np.float64)
        out = np.zeros((S, self.plant_count), dtype=np.int64)
        for s in range(S):
            Ls = int(cu[s + 1] - cu[s])
            P = Ls - w
            n = self.plant_count
            if P < n:
                out[s] = -1
                continue
            key = _stream_key(self.seed, _K_PLANT_POS, l, s)
            if self.plant == "tokens":
                pos = np.sort(np.argsort(uniform_u64(key, 0, P), kind="stable")[:n]) if P <= 1 << 20 \
                    else np.sort(_randint(key, 0, n, 0, P - 1))
            elif self.plant == "span":
                depth = int(_randint(key, 0, 1, 0, P - n)[0])
                pos = np.arange(depth, depth + n)
            else:
                raise ValueError(self.plant)
            out[s] = pos
            for g in range(self.num_kv_heads):
                heads = np.nonzero(mask[g * G:(g + 1) * G])[0] + g * G
                if heads.size == 0:  # a group without a selected head: the layer's heads
                    heads = np.nonzero(mask)[0]
                u = qf[s][:, heads, :].reshape(-1, d).mean(axis=0)
                u /= np.linalg.norm(u)
                rows = np.broadcast_to(beta * u, (n, d)).copy()
                if self.plant_noise:
                    rows += normals(_stream_key(self.seed, _K_PLANT_NOISE, l, s * 4096 + g),
                                    n * d).reshape(n, d)
                k_bits[cu[s] + pos, g, :] = bf16_bits(rows.astype(np.float32))
        return out


def _ragged_lengths(seed: int, n: int, lo: int, hi: int) -> tuple:
    key = _stream_key(seed, _K_SEQLEN)
    return tuple(int(x) for x in _randint(key, 0, n, lo, hi))


# The five workloads.  Shapes follow the backbone models (Llama-3.1-8B: 32 layers, 32 query /
# 8 KV heads; Qwen2.5-7B: 28 layers, 28 / 4 heads; head_dim 128).  Where a workload leaves the
# pool or head count open, max pooling with kernel 7 and 2 selected heads per group are used.
_W = [
    Workload(name="single_layer_l2048", num_layers=1, num_q_heads=32, num_kv_heads=8,
             seqlens=(2048,), window=32, heads_per_group=1, budget_mean=128, budget_uniform=True,
             plant="tokens", plant_count=4, plant_beta=6.0, seed=20250802 + 0,
             description="1 layer, 1 seq, L=2048, 32/8 heads, 4 planted keys, w=32, 1 head per "
                         "group, maxpool 7, budget 128"),
    Workload(name="llama8b_l8192", num_layers=32, num_q_heads=32, num_kv_heads=8,
             seqlens=(8192,), window=32, heads_per_group=2, budget_mean=256,
             outlier_channels=8, seed=20250802 + 1,
             description="Llama-3.1-8B-shaped 32 layers, L=8192, key outliers, w=32, 2 heads per "
                         "group, layer budgets summing to 32x256"),
    Workload(name="llama8b_l32768", num_layers=32, num_q_heads=32, num_kv_heads=8,
             seqlens=(32768,), window=32, heads_per_group=2, budget_mean=1024,
             outlier_channels=8, seed=20250802 + 2,
             description="Llama-3.1-8B-shaped 32 layers, L=32768, w=32, maxpool 7, mean budget 1024"),
    Workload(name="needle_l131072", num_layers=32, num_q_heads=32, num_kv_heads=8,
             seqlens=(131072,), window=32, heads_per_group=2, budget_mean=128, budget_uniform=True,
             outlier_channels=8, plant="span", plant_count=64, plant_beta=6.0, plant_noise=True,
             seed=20250802 + 3,
             description="needle-style L=131072, planted 64-token span, budget 128"),
    Workload(name="ragged_qwen7b", num_layers=28, num_q_heads=28, num_kv_heads=4,
             seqlens=_ragged_lengths(20250802 + 4, 8, 4096, 32768), window=32, heads_per_group=2,
             budget_mean=512, outlier_channels=8, seed=20250802 + 4,
             description="8 ragged sequences in [4096, 32768], Qwen2.5-7B-shaped 28 layers, 28/4 "
                         "heads, mean budget 512, varlen packed"),
    Workload(name="paper_llama8b_l8192", num_layers=32, num_q_heads=32, num_kv_heads=8,
             seqlens=(8192,), window=8, heads_per_group=1, heads_per_layer=4, scope="layer",
             pool_kernel=5, pool_type="avg", budget_mean=256, outlier_channels=8,
             plant="tokens", plant_count=4, plant_beta=6.0, seed=20250802 + 5,
             description="the paper's own hyper-parameters (App. A, Sec. 4.1): one index set per "
                         "layer from the top-4 heads of the layer, w=8, avg pool 5; "
                         "Llama-3.1-8B-shaped 32 layers, L=8192, 4 planted keys"),
]
WORKLOAD_ORDER = [w.name for w in _W]
WORKLOADS = {w.name: w for w in _W}


def workload(name: str) -> Workload:
    return WORKLOADS[name]
