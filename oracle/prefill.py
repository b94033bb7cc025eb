"""Prefill attention over a DynaCalKV compressed KV cache, fp64, plain definition.

TEST INFRASTRUCTURE ONLY (see the package docstring): never imported by the
library.

Prefill is decode with many queries per sequence: the Q_b new tokens of
sequence b are the last Q_b rows of its cache (appended before attention, as
in decode), the i-th of them sits at position p_i = L_b - Q_b + i and attends,
causally, to the keys at positions 0 .. p_i.  Keys and values are rebuilt from
the latents exactly as in decode (Sec. III-A z = x L, x W ~ z R; Sec. III-C one
factorisation per head group; Sec. III-D one value factorisation for all
heads), so for each sequence the reconstruction K_h = C_g B_g[:, slot] and
V_h = C_v B_v[:, h] is computed once and serves all of its queries.

For sequence b, query i at position p, query head j, KV head h = kv(j):

1. k_t, v'_t rebuilt from the latents, t in [0, L)        (Sec. III-A, III-C, III-D)
2. RoPE of the keys at position t, of the query at position p
3. sigma_t = <RoPE(q_ij), RoPE(k_t)> / sqrt(d) for t <= p; p = softmax over t <= p
4. o_ij = sum_{t <= p} p_t v'_t

The causal mask and the query positions are this library's readings (the paper
describes neither); Q_b = 1 is the decode call.
"""

from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np

from .decode import _group_slot, kv_head_of, rope


def prefill_attention(spec, q, q_lens, kcache, vcache, B_k, B_v, seq_start, seq_lens,
                      return_probs: bool = False, heads: Optional[Sequence[int]] = None):
    """Causal prefill attention output o [B, Qmax, Hq, d] in fp64.

    spec      : LayerSpec-like (n_q_heads, n_kv_heads, head_dim, groups, ranks, rope_theta)
    q         : [B, Qmax, Hq, d] queries before RoPE; sequence b uses rows [0, q_lens[b])
    q_lens    : Q_b, new tokens of each sequence (1 <= Q_b <= L_b)
    kcache, vcache, B_k, B_v, seq_start, seq_lens : as for the decode oracle
    heads     : optional subset of query heads (others are left as NaN)
    return_probs : also return {(b, i, j): p} with each query's softmax row (length p + 1)
    """
    Hq, Hkv, d = spec.n_q_heads, spec.n_kv_heads, spec.head_dim
    groups, ranks = spec.groups, spec.ranks
    q = np.asarray(q, dtype=np.float64)
    kcache = np.asarray(kcache, dtype=np.float64)
    vcache = np.asarray(vcache, dtype=np.float64)
    B_k = np.asarray(B_k, dtype=np.float64).reshape(-1)
    B_v = np.asarray(B_v, dtype=np.float64)
    B, Qmax = q.shape[0], q.shape[1]

    rank_off = np.concatenate([[0], np.cumsum(ranks)]).astype(int)
    blk_off = [0]
    for heads_g, r in zip(groups, ranks):
        blk_off.append(blk_off[-1] + r * len(heads_g) * d)

    out = np.full((B, Qmax, Hq, d), np.nan, dtype=np.float64)
    probs = {}
    js = range(Hq) if heads is None else heads
    for b in range(B):
        L, Q, r0 = int(seq_lens[b]), int(q_lens[b]), int(seq_start[b])
        if not 1 <= Q <= L:
            raise ValueError("each sequence needs 1 <= q_len <= seq_len")
        for j in js:
            h = kv_head_of(j, Hq, Hkv)
            g, s = _group_slot(groups, h)
            r_g, n_g = ranks[g], len(groups[g])
            Bg = B_k[blk_off[g]:blk_off[g + 1]].reshape(r_g, n_g * d)
            k = kcache[r0:r0 + L, rank_off[g]:rank_off[g] + r_g] @ Bg[:, s * d:(s + 1) * d]  # step 1
            v = vcache[r0:r0 + L] @ B_v[:, h * d:(h + 1) * d]
            k_rot = rope(k, np.arange(L), spec.rope_theta)                                  # step 2
            for i in range(Q):
                p_pos = L - Q + i
                q_rot = rope(q[b, i, j], p_pos, spec.rope_theta)
                sigma = (k_rot[:p_pos + 1] @ q_rot) / math.sqrt(d)                           # step 3
                e = np.exp(sigma - sigma.max())
                p = e / e.sum()
                out[b, i, j] = p @ v[:p_pos + 1]                                             # step 4
                if return_probs:
                    probs[(b, i, j)] = p
    if return_probs:
        return out, probs
    return out
