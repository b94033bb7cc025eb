"""Decode attention over a DynaCalKV compressed KV cache, fp64, plain definition.

TEST INFRASTRUCTURE ONLY (see the package docstring): never imported by the
library.

What is computed (one decode query per sequence):

Sec. III-A: a rank-r factorisation W ~ L R lets the cache keep z = x L and
rebuild x W ~ z R.  Sec. III-C splits the key projection column-wise into
head groups, W_i ~ L_i R_i, so group g caches c_t^g = x_t L_g (r_g values per
token) and rebuilds the keys of all its heads as c_t^g R_g.  Sec. III-D keeps
one whole-matrix value factorisation W^(v) ~ L_v R_v, so the cache keeps
v_t = x_t L_v (r_v values) and rebuilds every head's value as v_t R_v.
In the library's names A_g = L_g, B_g = R_g, A_v = L_v, B_v = R_v.

For sequence b of length L, query head j, KV head h = kv(j), group g that
holds h at column-block slot s:

1. k_t = c_t^g . B_g[:, s*d:(s+1)*d]            for t in [0, L)
   v'_t = v_t . B_v[:, h*d:(h+1)*d]
2. RoPE, rotate-half pairing (i, i + d/2), omega_i = theta^(-2i/d):
   keys at position t, the query at position L - 1 (the decode step's own
   token is the cache's last row), both shifted by ``pos_offset``.
3. sigma_t = <RoPE(q_j), RoPE(k_t)> / sqrt(d);  p = softmax(sigma) over t.
4. o_j = sum_t p_t v'_t.

The paper does not describe decode, RoPE, the query position or the GQA head
mapping; the readings used here (RoPE after reconstruction on keys and query,
rotate-half pairing, q at L-1, kv(j) = floor(j*Hkv/Hq)) are the ones stated in
the design notes.  Everything is fp64; the inputs are the stored (already
rounded) values.
"""

from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np


def rope_freqs(d: int, theta: float) -> np.ndarray:
    """omega_i = theta^(-2i/d) for i in [0, d/2), fp64."""
    i = np.arange(d // 2, dtype=np.float64)
    return np.power(float(theta), -2.0 * i / d)


def rope(x: np.ndarray, pos, theta: float) -> np.ndarray:
    """Rotate-half RoPE of x[..., d] at integer positions ``pos`` (broadcast over x[..., 0]).

    Pair (i, i + d/2) is rotated by the angle pos * omega_i:
      y[i]       = x[i] cos - x[i + d/2] sin
      y[i + d/2] = x[i] sin + x[i + d/2] cos
    """
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    ang = np.asarray(pos, dtype=np.float64)[..., None] * rope_freqs(d, theta)
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def kv_head_of(j: int, n_q_heads: int, n_kv_heads: int) -> int:
    """KV head of query head j: consecutive query heads share one KV head."""
    return (j * n_kv_heads) // n_q_heads


def _group_slot(groups: Sequence[Sequence[int]], h: int):
    for g, heads in enumerate(groups):
        for s, hh in enumerate(heads):
            if hh == h:
                return g, s
    raise ValueError(f"KV head {h} is in no group")


def decode_attention(spec, q, kcache, vcache, B_k, B_v, seq_start, seq_lens,
                     pos_offset: int = 0, return_probs: bool = False,
                     heads: Optional[Sequence[int]] = None, batch_ids: Optional[Sequence[int]] = None):
    """Decode attention output o [B, Hq, d] in fp64.

    spec      : LayerSpec-like (hidden, n_q_heads, n_kv_heads, head_dim, groups,
                ranks, rank_v, rope_theta)
    q         : [B, Hq, d] query before RoPE
    kcache    : [n_rows, R_k]; group g's latent in columns [sum_{g'<g} r_g', +r_g)
    vcache    : [n_rows, r_v]
    B_k       : packed 1-D; group g's block [r_g, n_g*d] row-major at sum_{g'<g} r_g' n_g' d
    B_v       : [r_v, Hkv*d]
    seq_start : first cache row of each sequence; seq_lens: its length L_b >= 1
    heads, batch_ids : optional subsets to evaluate (others are left as NaN)
    return_probs : also return {(b, j): p} with the softmax rows
    """
    Hq, Hkv, d = spec.n_q_heads, spec.n_kv_heads, spec.head_dim
    groups, ranks = spec.groups, spec.ranks
    q = np.asarray(q, dtype=np.float64)
    kcache = np.asarray(kcache, dtype=np.float64)
    vcache = np.asarray(vcache, dtype=np.float64)
    B_k = np.asarray(B_k, dtype=np.float64).reshape(-1)
    B_v = np.asarray(B_v, dtype=np.float64)
    B = q.shape[0]

    rank_off = np.concatenate([[0], np.cumsum(ranks)]).astype(int)
    blk_off = [0]
    for heads_g, r in zip(groups, ranks):
        blk_off.append(blk_off[-1] + r * len(heads_g) * d)

    out = np.full((B, Hq, d), np.nan, dtype=np.float64)
    probs = {}
    bs = range(B) if batch_ids is None else batch_ids
    js = range(Hq) if heads is None else heads
    for b in bs:
        L = int(seq_lens[b])
        r0 = int(seq_start[b])
        t_pos = np.arange(L) + pos_offset
        q_pos = L - 1 + pos_offset
        kv_cache = {}  # KV head -> (rotated keys, values): shared by its query heads
        for j in js:
            h = kv_head_of(j, Hq, Hkv)
            if h not in kv_cache:
                g, s = _group_slot(groups, h)
                r_g, n_g = ranks[g], len(groups[g])
                Bg = B_k[blk_off[g]:blk_off[g + 1]].reshape(r_g, n_g * d)
                C_g = kcache[r0:r0 + L, rank_off[g]:rank_off[g] + r_g]
                k = C_g @ Bg[:, s * d:(s + 1) * d]                     # step 1, keys
                v = vcache[r0:r0 + L] @ B_v[:, h * d:(h + 1) * d]      # step 1, values
                kv_cache[h] = (rope(k, t_pos, spec.rope_theta), v)      # step 2, keys
            k_rot, v = kv_cache[h]
            q_rot = rope(q[b, j], q_pos, spec.rope_theta)               # step 2, query
            sigma = (k_rot @ q_rot) / math.sqrt(d)                  # step 3
            e = np.exp(sigma - sigma.max())
            p = e / e.sum()
            out[b, j] = p @ v                                       # step 4
            if return_probs:
                probs[(b, j)] = p
    if return_probs:
        return out, probs
    return out


def max_rel_err(got: np.ndarray, ref: np.ndarray) -> float:
    """max |got - ref| / ||ref||_inf, the parity measure of the decode output.

    Only the entries the reference evaluated (finite in ``ref``; a subset of
    heads or sequences leaves the rest NaN) are compared, and the scale is the
    reference's largest magnitude over those entries.  A non-finite ``got`` at
    any compared entry gives +inf, so it fails every tolerance; so does a
    reference with nothing evaluated or all zeros (nothing to normalise by).
    """
    ref = np.asarray(ref, dtype=np.float64)
    got = np.asarray(got, dtype=np.float64)
    if got.shape != ref.shape:
        raise ValueError(f"shape mismatch: got {got.shape}, reference {ref.shape}")
    m = np.isfinite(ref)
    if not m.any():
        return math.inf
    g, r = got[m], ref[m]
    if not np.isfinite(g).all():
        return math.inf
    scale = np.abs(r).max()
    if scale == 0.0:
        return 0.0 if (g == 0.0).all() else math.inf
    return float(np.abs(g - r).max() / scale)
