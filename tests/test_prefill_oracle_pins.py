"""Pins of the prefill oracle (oracle/prefill.py), each independent of its code:

* full rank with A.B = I: torch's scaled_dot_product_attention with an explicit
  causal mask (bottom-right aligned: the new tokens are the cache's last rows)
  on RoPE written in complex form, MHA and GQA;
* one new token is the decode call (the decode oracle is pinned on its own);
* causality: latents after a query's position do not change its output;
* softmax rows over the visible keys sum to one, and a query sees exactly its
  position + 1 keys."""

import math

import numpy as np
import pytest
import torch

from oracle.decode import decode_attention
from oracle.prefill import prefill_attention
from paper_2607_24331_gb300 import synth as S
from test_oracle_pins import random_inputs, rope_complex, small_spec


def _queries(spec, q_lens, seed, std=1.0):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((len(q_lens), max(q_lens), spec.n_q_heads, spec.head_dim)) * std


@pytest.mark.parametrize("Hq,Hkv,groups", [(4, 4, ((2, 0), (1,), (3,))), (8, 2, ((1, 0),))])
def test_full_rank_identity_factors_equal_masked_textbook_attention(Hq, Hkv, groups):
    d = 8
    ranks = tuple(len(g) * d for g in groups)
    spec = small_spec(Hq, Hkv, d, groups, ranks, Hkv * d, 1e4)
    lens, q_lens = [6, 3, 9], [6, 1, 4]
    n = sum(lens)
    starts = S.seq_starts(lens)
    rng = np.random.default_rng(13)
    K = [rng.standard_normal((n, d)) for _ in range(Hkv)]
    V = [rng.standard_normal((n, d)) for _ in range(Hkv)]
    q = _queries(spec, q_lens, 14, 2.0)
    kc_cols, Bk = [], []
    for g in groups:
        Kg = np.concatenate([K[h] for h in g], axis=1)
        M = rng.standard_normal((Kg.shape[1], Kg.shape[1])) + 3 * np.eye(Kg.shape[1])
        kc_cols.append(Kg @ np.linalg.inv(M))
        Bk.append(M.ravel())
    kc = np.concatenate(kc_cols, axis=1)
    Mv = rng.standard_normal((Hkv * d, Hkv * d)) + 3 * np.eye(Hkv * d)
    vc = np.concatenate(V, axis=1) @ np.linalg.inv(Mv)
    got = prefill_attention(spec, q, q_lens, kc, vc, np.concatenate(Bk), Mv, starts, lens)
    rep = Hq // Hkv
    for b, (L, Q) in enumerate(zip(lens, q_lens)):
        r0 = int(starts[b])
        k = np.stack([rope_complex(K[h][r0:r0 + L], np.arange(L), 1e4) for h in range(Hkv)])
        v = np.stack([V[h][r0:r0 + L] for h in range(Hkv)])
        pos = np.arange(L - Q, L)
        qq = np.stack([rope_complex(q[b, :Q, j], pos, 1e4) for j in range(Hq)])     # [Hq, Q, d]
        mask = torch.from_numpy(np.arange(L)[None, :] <= pos[:, None])              # [Q, L]
        o = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(qq)[None], torch.from_numpy(k).repeat_interleave(rep, 0)[None],
            torch.from_numpy(v).repeat_interleave(rep, 0)[None], attn_mask=mask, scale=1.0 / math.sqrt(d))
        np.testing.assert_allclose(got[b, :Q], o[0].permute(1, 0, 2).numpy(), atol=1e-10, rtol=1e-10)
        assert np.isnan(got[b, Q:]).all()


def test_one_new_token_is_the_decode_call():
    spec = small_spec()
    lens = [7, 1, 12]
    q, kc, vc, Bk, Bv, starts, lens_a = random_inputs(spec, lens, seed=21, q_std=3.0)
    got = prefill_attention(spec, q[:, None], [1, 1, 1], kc, vc, Bk, Bv, starts, lens_a)
    ref = decode_attention(spec, q, kc, vc, Bk, Bv, starts, lens_a)
    np.testing.assert_allclose(got[:, 0], ref, atol=1e-13, rtol=1e-12)


def test_later_latents_do_not_change_earlier_queries():
    spec = small_spec()
    lens, q_lens = [10], [6]
    _, kc, vc, Bk, Bv, starts, lens_a = random_inputs(spec, lens, seed=5)
    q = _queries(spec, q_lens, 6)
    base = prefill_attention(spec, q, q_lens, kc, vc, Bk, Bv, starts, lens_a)
    kc2, vc2 = kc.copy(), vc.copy()
    kc2[8:] += 50.0   # tokens at positions 8, 9
    vc2[8:] -= 30.0
    moved = prefill_attention(spec, q, q_lens, kc2, vc2, Bk, Bv, starts, lens_a)
    # queries at positions 4..7 (rows 0..3) see only tokens 0..7; positions 8, 9 see the change
    np.testing.assert_array_equal(moved[0, :4], base[0, :4])
    assert np.abs(moved[0, 4:] - base[0, 4:]).max() > 1e-3


def test_each_query_sees_its_prefix_and_rows_sum_to_one():
    spec = small_spec(Hq=8, Hkv=2, groups=((1, 0),), ranks=(24,))
    lens, q_lens = [9, 4], [5, 4]
    _, kc, vc, Bk, Bv, starts, lens_a = random_inputs(spec, lens, seed=8)
    q = _queries(spec, q_lens, 9, 6.0)
    _, probs = prefill_attention(spec, q, q_lens, kc, vc, Bk, Bv, starts, lens_a, return_probs=True)
    for (b, i, j), p in probs.items():
        assert len(p) == lens[b] - q_lens[b] + i + 1
        assert abs(p.sum() - 1.0) <= 1e-12
