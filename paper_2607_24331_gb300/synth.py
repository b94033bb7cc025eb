"""Seeded synthetic inputs for DynaCalKV latent-cache decode attention.

This module is shared by the oracle, the tests and the benchmark.  It holds
no arithmetic of the method itself (no reconstruction, RoPE, softmax or
projection): it only draws numbers and builds the shapes, group tables and
sequence lengths of the workloads.

Generator.  Every tensor is drawn from a counter-based stream so that any
element can be produced independently (the CUDA fill kernel in the library
implements the same definition and is checked bit-exact against this one):

* SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014; constants of Vigna's public-domain version):
  ``draw(key, i) = mix(key + (i + 1) * GAMMA)`` modulo 2**64, where ``mix`` is
  the SplitMix64 output finaliser.
* Stream key of (seed, layer, tensor id):
  ``mix(mix(mix(seed + GAMMA) + layer + GAMMA) + tid + GAMMA)``.
* Gaussian element i: the eight 16-bit fields of draws 2i and 2i+1 are summed
  as integers (Irwin-Hall with n = 8, an exact integer), centred as
  ``s2 = 2*s - 8*65535`` and scaled by one IEEE fp32 multiplication with
  ``c = float32(std / (65536*sqrt(8/3)))``.  The result is an fp32 value; for
  bf16 tensors it is rounded once more to bf16, round-to-nearest-even.
  All steps are exact integer work or single IEEE roundings, so numpy and
  CUDA give identical bits.
* Integers in [lo, hi]: ``lo + ((draw >> 32) * (hi - lo + 1) >> 32)``.

Workloads (shapes and value distributions of the paper's 7-8B MHA and GQA
models, stood in for by Gaussian data because no weights are used):
x, q ~ N(0, 1); the latent caches c = x A_g and v = x A_v with A ~ N(0, 1/D)
have unit variance, so they are drawn directly as N(0, 1); B_g ~ N(0, 1/r_g)
and B_v ~ N(0, 1/r_v), so reconstructed keys and values also have unit
variance.
"""

from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import numpy as np

MASK64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15
MIX_C1 = 0xBF58476D1CE4E5B9
MIX_C2 = 0x94D049BB133111EB

# Tensor ids of the stream keys.  The CUDA fill kernel only receives the
# 64-bit key, so these ids live here alone.
TID = {
    "q": 1, "kcache": 2, "vcache": 3, "B_k": 4, "B_v": 5, "x": 6,
    "A_k": 7, "A_v": 8, "perm": 9, "lens": 10, "x_step": 11, "q_prefill": 12,
}


# ---------------------------------------------------------------------------
# SplitMix64
# ---------------------------------------------------------------------------

def mix64_int(z: int) -> int:
    """SplitMix64 output finaliser on a Python int (mod 2**64)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * MIX_C1) & MASK64
    z = ((z ^ (z >> 27)) * MIX_C2) & MASK64
    return z ^ (z >> 31)


def stream_key(seed: int, layer: int, tid: int) -> int:
    """64-bit key of the stream for (seed, layer, tensor id)."""
    k = mix64_int(seed + GAMMA)
    k = mix64_int(k + layer + GAMMA)
    return mix64_int(k + tid + GAMMA)


def _mix64_np(z: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * np.uint64(MIX_C1)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(MIX_C2)
        return z ^ (z >> np.uint64(31))


def draws(key: int, start: int, count: int) -> np.ndarray:
    """SplitMix64 outputs number start .. start+count-1 of stream ``key``."""
    idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(key) + idx * np.uint64(GAMMA)
    return _mix64_np(z)


def gauss_scale(std: float) -> np.float32:
    """fp32 multiplier mapping the centred Irwin-Hall sum to N(0, std^2)."""
    return np.float32(std / (65536.0 * math.sqrt(8.0 / 3.0)))


_CHUNK = 1 << 20
_POOL = None


def _pool():
    global _POOL
    if _POOL is None:
        import concurrent.futures
        import os
        n = max(1, min(32, len(os.sched_getaffinity(0))))
        _POOL = concurrent.futures.ThreadPoolExecutor(max_workers=n)
    return _POOL


_M2 = np.uint64(0x0000FFFF0000FFFF)
_M32 = np.uint64(0xFFFFFFFF)


def _gauss_chunk(out: np.ndarray, key: int, first_draw: int, c: np.float32) -> None:
    n = out.shape[0]
    with np.errstate(over="ignore"):
        z = np.arange(first_draw + 1, first_draw + 2 * n + 1, dtype=np.uint64)
        z *= np.uint64(GAMMA)
        z += np.uint64(key)
        z ^= z >> np.uint64(30)
        z *= np.uint64(MIX_C1)
        z ^= z >> np.uint64(27)
        z *= np.uint64(MIX_C2)
        z ^= z >> np.uint64(31)
        # sum of the four 16-bit fields of each draw, two lanes at a time
        t = (z & _M2) + ((z >> np.uint64(16)) & _M2)
        t = (t & _M32) + (t >> np.uint64(32))
        s = t.view(np.int64)
        s2 = 2 * (s[0::2] + s[1::2]) - 8 * 65535
        np.multiply(s2.astype(np.float32), c, out=out)


def gaussian_f32(key: int, start: int, count: int, std: float) -> np.ndarray:
    """Gaussian elements start .. start+count-1 of stream ``key`` as fp32."""
    out = np.empty(count, dtype=np.float32)
    c = gauss_scale(std)
    offs = list(range(0, count, _CHUNK))
    if len(offs) <= 1:
        if count:
            _gauss_chunk(out, key, 2 * start, c)
        return out
    futs = [_pool().submit(_gauss_chunk, out[o:o + _CHUNK], key, 2 * (start + o), c) for o in offs]
    for f in futs:
        f.result()
    return out


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_to(a: np.ndarray, dtype: str) -> np.ndarray:
    """Values of ``a`` after storage in ``dtype`` ('bf16' or 'f32'), as fp32."""
    if dtype == "bf16":
        return bf16_bits_to_f32(f32_to_bf16_bits(a))
    return np.asarray(a, dtype=np.float32)


def gaussian(key: int, shape: Sequence[int], std: float, dtype: str,
             start: int = 0) -> np.ndarray:
    """Seeded Gaussian tensor, already rounded to its storage dtype (fp32 array)."""
    n = int(np.prod(shape)) if len(shape) else 1
    return round_to(gaussian_f32(key, start, n, std), dtype).reshape(shape)


def uniform_ints(key: int, count: int, lo: int, hi: int) -> np.ndarray:
    """Integers in [lo, hi] from stream ``key`` (multiply-shift mapping)."""
    d = draws(key, 0, count) >> np.uint64(32)
    span = np.uint64(hi - lo + 1)
    with np.errstate(over="ignore"):
        v = (d * span) >> np.uint64(32)
    return (v.astype(np.int64) + lo).astype(np.int64)


def permutation(key: int, n: int) -> List[int]:
    """Fisher-Yates shuffle of range(n) driven by the stream (draw i picks slot i)."""
    p = list(range(n))
    d = draws(key, 0, n)
    for i in range(n - 1, 0, -1):
        j = int(d[i]) % (i + 1)
        p[i], p[j] = p[j], p[i]
    return p


# ---------------------------------------------------------------------------
# Layer and workload descriptions
# ---------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class LayerSpec:
    """One attention layer with a DynaCalKV-compressed KV cache.

    groups[g] lists the KV heads of key group g in the column-block order of
    B_g; ranks[g] = r_g; rank_v = r_v (one whole-matrix value latent).
    """
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    groups: Tuple[Tuple[int, ...], ...]
    ranks: Tuple[int, ...]
    rank_v: int
    dtype: str = "bf16"
    rope_theta: float = 1e4

    @property
    def n_groups(self) -> int:
        return len(self.groups)

    @property
    def rank_k(self) -> int:
        return int(sum(self.ranks))

    def group_offsets(self) -> List[int]:
        off = [0]
        for g in self.groups:
            off.append(off[-1] + len(g))
        return off

    def group_heads(self) -> List[int]:
        return [h for g in self.groups for h in g]

    def rank_offsets(self) -> List[int]:
        off = [0]
        for r in self.ranks:
            off.append(off[-1] + r)
        return off

    def bk_offsets(self) -> List[int]:
        """Element offset of each group's block [r_g, n_g*d] in the packed B_k."""
        off = [0]
        for g, r in zip(self.groups, self.ranks):
            off.append(off[-1] + r * len(g) * self.head_dim)
        return off

    def validate(self) -> None:
        hs = sorted(self.group_heads())
        assert hs == list(range(self.n_kv_heads)), "groups must partition the KV heads"
        assert self.n_q_heads % self.n_kv_heads == 0
        assert len(self.ranks) == len(self.groups)


@dataclasses.dataclass(frozen=True)
class Workload:
    """A decode batch: one query per sequence at position len_b - 1."""
    name: str
    layer: LayerSpec
    seq_lens: Tuple[int, ...]
    seed: int = 0
    n_layers: int = 1
    append_tokens: int = 0  # tokens per sequence of a latent-append prefill

    @property
    def batch(self) -> int:
        return len(self.seq_lens)


def groups_from_sizes(sizes: Sequence[int], order: Sequence[int]) -> Tuple[Tuple[int, ...], ...]:
    out, i = [], 0
    for s in sizes:
        out.append(tuple(order[i:i + s]))
        i += s
    return tuple(out)


def tiny_mha_layer() -> LayerSpec:
    """fp32 MHA layer: D 512, 8 heads of 64, groups {0-2},{3-7}, ranks {48,96}, r_v 160."""
    return LayerSpec(512, 8, 8, 64, ((0, 1, 2), (3, 4, 5, 6, 7)), (48, 96), 160, "f32", 1e4)


def llama2_mha_layer(seed: int = 0, layer: int = 0) -> LayerSpec:
    """Llama-2-7B-like MHA layer: 32 heads of 128, uneven groups over a seeded head permutation."""
    perm = permutation(stream_key(seed, layer, TID["perm"]), 32)
    sizes = (2, 3, 3, 4, 4, 5, 5, 6)
    return LayerSpec(4096, 32, 32, 128, groups_from_sizes(sizes, perm),
                     (64, 96, 96, 128, 128, 160, 160, 192), 1024, "bf16", 1e4)


def mistral_gqa_layer() -> LayerSpec:
    """Mistral-7B-like GQA layer: 32 q-heads, 8 KV heads of 128, groups {1,1,2,2,2}."""
    return LayerSpec(4096, 32, 8, 128, groups_from_sizes((1, 1, 2, 2, 2), range(8)),
                     (96, 96, 160, 192, 224), 512, "bf16", 1e6)


def llama3_gqa_layer() -> LayerSpec:
    """Llama-3-8B-like long-context GQA layer: 8 KV heads, groups {2,3,3}."""
    return LayerSpec(4096, 32, 8, 128, groups_from_sizes((2, 3, 3), range(8)),
                     (192, 256, 256), 384, "bf16", 5e5)


def recalkv_mha_layer() -> LayerSpec:
    """The Llama-2-7B-like MHA layer with ReCalKV's fixed grouping (Sec. III-C): groups of
    four consecutive heads and one uniform rank r/K per group, at the same total rank
    (sum r_g = 1024) and value rank as the DynaCalKV layer."""
    return LayerSpec(4096, 32, 32, 128, groups_from_sizes((4,) * 8, range(32)), (128,) * 8, 1024, "bf16", 1e4)


def ragged_lens(seed: int, batch: int, lo: int = 1024, hi: int = 16384) -> Tuple[int, ...]:
    key = stream_key(seed, 1000 + batch, TID["lens"])
    return tuple(int(v) for v in uniform_ints(key, batch, lo, hi))


def workload(cfg: int, batch: Optional[int] = None) -> Workload:
    """The five benchmark workloads (0: tiny fp32 MHA ... 4: 32-layer ragged MHA step), and
    5: the MHA layer of workload 1 with ReCalKV's fixed groups of four at equal total rank."""
    if cfg == 0:
        return Workload("tiny-fp32-mha D512 H8 d64 B1 T512", tiny_mha_layer(), (512,))
    if cfg == 1:
        return Workload("llama2-7b-mha D4096 H32 d128 B16 T4096", llama2_mha_layer(), (4096,) * 16)
    if cfg == 2:
        return Workload("mistral-7b-gqa Hq32 Hkv8 d128 B8 T32768", mistral_gqa_layer(), (32768,) * 8)
    if cfg == 3:
        return Workload("llama3-8b-gqa Hq32 Hkv8 d128 B2 T131072", llama3_gqa_layer(), (131072,) * 2,
                        append_tokens=8192)
    if cfg == 4:
        b = 8 if batch is None else batch
        return Workload(f"llama2-7b-mha 32 layers B{b} ragged T~U[1024,16384]",
                        llama2_mha_layer(), ragged_lens(0, b), n_layers=32)
    if cfg == 5:
        return Workload("llama2-7b-mha recalkv-groups D4096 H32 d128 B16 T4096", recalkv_mha_layer(), (4096,) * 16)
    raise ValueError(cfg)


def layer_for(w: Workload, layer: int) -> LayerSpec:
    """Layer spec of layer ``layer``: every layer keeps the workload's grouping and ranks;
    only the data streams are re-seeded per layer (stream key uses the layer index)."""
    del layer
    return w.layer


# ---------------------------------------------------------------------------
# Tensors of one layer
# ---------------------------------------------------------------------------

@dataclasses.dataclass
class DecodeInputs:
    """Host copies of one layer's decode inputs, already rounded to storage dtype.

    kcache [n_rows, R_k] and vcache [n_rows, r_v] hold the sequences back to
    back: sequence b owns rows seq_start[b] .. seq_start[b] + seq_lens[b] - 1.
    B_k packs group g's [r_g, n_g*d] block at bk_offsets()[g]; B_v is
    [r_v, Hkv*d]; q is [B, Hq, d] before RoPE.
    """
    spec: LayerSpec
    q: np.ndarray
    kcache: np.ndarray
    vcache: np.ndarray
    B_k: np.ndarray
    B_v: np.ndarray
    seq_start: np.ndarray
    seq_lens: np.ndarray


def seq_starts(seq_lens: Sequence[int]) -> np.ndarray:
    return np.concatenate([[0], np.cumsum(seq_lens)[:-1]]).astype(np.int64)


def factor_keys(seed: int, layer: int) -> dict:
    return {n: stream_key(seed, layer, TID[n]) for n in ("B_k", "B_v")}


def make_bk(spec: LayerSpec, seed: int, layer: int) -> np.ndarray:
    """Packed B_k: group g's block ~ N(0, 1/r_g), drawn from one stream at its packed offset."""
    key = stream_key(seed, layer, TID["B_k"])
    off = spec.bk_offsets()
    out = np.empty(off[-1], dtype=np.float32)
    for g, r in enumerate(spec.ranks):
        n = off[g + 1] - off[g]
        out[off[g]:off[g + 1]] = round_to(gaussian_f32(key, off[g], n, 1.0 / math.sqrt(r)), spec.dtype)
    return out


def make_bv(spec: LayerSpec, seed: int, layer: int) -> np.ndarray:
    key = stream_key(seed, layer, TID["B_v"])
    return gaussian(key, (spec.rank_v, spec.n_kv_heads * spec.head_dim),
                    1.0 / math.sqrt(spec.rank_v), spec.dtype)


def make_decode_inputs(spec: LayerSpec, seq_lens: Sequence[int], seed: int = 0, layer: int = 0,
                       q_std: float = 1.0) -> DecodeInputs:
    """All decode inputs of one layer (host, fp32 arrays holding storage-dtype values)."""
    spec.validate()
    lens = np.asarray(seq_lens, dtype=np.int64)
    n_rows = int(lens.sum())
    B = len(lens)
    q = gaussian(stream_key(seed, layer, TID["q"]), (B, spec.n_q_heads, spec.head_dim), q_std, spec.dtype)
    kc = gaussian(stream_key(seed, layer, TID["kcache"]), (n_rows, spec.rank_k), 1.0, spec.dtype)
    vc = gaussian(stream_key(seed, layer, TID["vcache"]), (n_rows, spec.rank_v), 1.0, spec.dtype)
    return DecodeInputs(spec, q, kc, vc, make_bk(spec, seed, layer), make_bv(spec, seed, layer),
                        seq_starts(lens), lens)


def make_prefill_q(spec: LayerSpec, batch: int, q_max: int, seed: int = 0, layer: int = 0,
                   q_std: float = 1.0) -> np.ndarray:
    """Prefill queries [B, q_max, Hq, d] before RoPE, ~ N(0, q_std^2), storage dtype."""
    return gaussian(stream_key(seed, layer, TID["q_prefill"]), (batch, q_max, spec.n_q_heads, spec.head_dim),
                    q_std, spec.dtype)


def cache_rows(spec: LayerSpec, seed: int, layer: int, which: str, row0: int, n: int) -> np.ndarray:
    """Rows row0 .. row0+n-1 of one layer's key or value latent cache (random access)."""
    width = spec.rank_k if which == "kcache" else spec.rank_v
    key = stream_key(seed, layer, TID[which])
    return round_to(gaussian_f32(key, row0 * width, n * width, 1.0), spec.dtype).reshape(n, width)


def make_append_inputs(spec: LayerSpec, n_tok: int, seed: int = 0, layer: int = 0):
    """x [n_tok, D] ~ N(0,1); A_k [D, R_k], A_v [D, r_v] ~ N(0, 1/D)."""
    D = spec.hidden
    x = gaussian(stream_key(seed, layer, TID["x"]), (n_tok, D), 1.0, spec.dtype)
    A_k = gaussian(stream_key(seed, layer, TID["A_k"]), (D, spec.rank_k), 1.0 / math.sqrt(D), spec.dtype)
    A_v = gaussian(stream_key(seed, layer, TID["A_v"]), (D, spec.rank_v), 1.0 / math.sqrt(D), spec.dtype)
    return x, A_k, A_v
