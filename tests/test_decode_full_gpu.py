"""Full-size and planted-needle parity of decode attention through the C ABI.

* Every query head of two whole sequences of each full-size workload against
  the fp64 oracle, one of them (where the workload has any) in the leftover
  tiles that the tensor-core path splits below tile granularity.
* A planted needle (one token whose key, for one query head, scores far above
  every other: the softmax must select it) at a 128-token tile boundary,
  inside a leftover tile, and at a position near 1.3e5.
* Peaked scores (q x 8) on the long-context GQA layer.

The needle helper is checked on the CPU (the oracle must give the needle
almost all the probability) before any GPU use.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2607_24331_gb300 import synth as S
from gpu_util import assert_parity, gpu_decode, leftover_sequences, oracle_decode, plant_needle, sm_count


def test_planted_needle_takes_the_softmax_on_the_oracle():
    """CPU check of plant_needle: the oracle gives the needle p > 0.999 and the
    output is the needle's value row projected by its head's B_v block."""
    spec = S.workload(3).layer
    lens = (300, 200)
    di = S.make_decode_inputs(spec, lens, seed=4)
    plant_needle(di, 0, 128, 5)
    plant_needle(di, 1, 77, 30)
    out, probs = oracle.decode_attention(spec, di.q, di.kcache, di.vcache, di.B_k, di.B_v, di.seq_start,
                                         di.seq_lens, return_probs=True, heads=[5, 30])
    assert probs[(0, 5)][128] > 0.999 and probs[(1, 30)][77] > 0.999
    d = spec.head_dim
    for b, t, j in ((0, 128, 5), (1, 77, 30)):
        h = oracle.kv_head_of(j, spec.n_q_heads, spec.n_kv_heads)
        v = di.vcache[int(di.seq_start[b]) + t].astype(np.float64) @ di.B_v[:, h * d:(h + 1) * d]
        assert np.abs(out[b, j] - v).max() < 1e-2 * np.abs(v).max()


@pytest.mark.gpu
@pytest.mark.parametrize("cfg", [1, 2, 3, 5])
def test_full_size_every_head_of_two_sequences(cfg):
    w = S.workload(cfg)
    spec = w.layer
    di = S.make_decode_inputs(spec, w.seq_lens, seed=w.seed)
    got, _ = gpu_decode(spec, w.seq_lens, di=di)
    assert np.isfinite(got).all()
    left = leftover_sequences(w.seq_lens, sm_count())
    bs = sorted({0, left[-1] if left else w.batch - 1})
    for b in bs:
        ref = oracle_decode(di, batch_ids=[b])
        tag = "leftover tiles" if b in left else "whole tiles"
        assert_parity(got[b:b + 1], ref[b:b + 1], "bf16", f"cfg{cfg} b{b} every head ({tag})")


@pytest.mark.gpu
@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_needles_at_a_tile_boundary_and_in_a_leftover_tile(cfg):
    sms = sm_count()
    nt = sms + 5
    lens = (64 * 128, (nt - 64 - 1) * 128 + 77)
    spec = S.workload(cfg).layer
    di = S.make_decode_inputs(spec, lens, seed=31 + cfg)
    left = leftover_sequences(lens, sms)
    assert 1 in left
    k_left = nt - 64 - 2                          # second-last tile of sequence 1: a leftover tile
    # a pair-tile boundary (2560: the first token of pair tile 10, 2559: the last of
    # pair tile 9), the boundary between the two halves of pair tile 10 (2688),
    # and a token inside a leftover tile
    needles = [(0, 20 * 128, 3), (0, 20 * 128 - 1, spec.n_q_heads - 1), (0, 21 * 128, 17),
               (1, k_left * 128 + 61, 9)]
    for b, t, j in needles:
        plant_needle(di, b, t, j)
    got, _ = gpu_decode(spec, lens, di=di)
    ref, probs = oracle.decode_attention(spec, di.q, di.kcache, di.vcache, di.B_k, di.B_v, di.seq_start,
                                         di.seq_lens, return_probs=True)
    for b, t, j in needles:
        assert probs[(b, j)][t] > 0.999, (b, t, j)
    assert_parity(got, ref, "bf16", f"cfg{cfg} needles")
    d = spec.head_dim
    for b, t, j in needles:   # the selected value row, directly
        h = oracle.kv_head_of(j, spec.n_q_heads, spec.n_kv_heads)
        v = di.vcache[int(di.seq_start[b]) + t].astype(np.float64) @ di.B_v[:, h * d:(h + 1) * d]
        assert np.abs(got[b, j] - v).max() <= 2e-2 * np.abs(v).max(), (b, t, j)


@pytest.mark.gpu
def test_needle_near_position_130000():
    spec = S.workload(3).layer
    lens = (131071, 3)
    di = S.make_decode_inputs(spec, lens, seed=7)
    t, j = 130_003, 13
    plant_needle(di, 0, t, j)
    got, _ = gpu_decode(spec, lens, di=di)
    ref, probs = oracle.decode_attention(spec, di.q, di.kcache, di.vcache, di.B_k, di.B_v, di.seq_start,
                                         di.seq_lens, return_probs=True, batch_ids=[0])
    assert probs[(0, j)][t] > 0.999
    assert_parity(got[:1], ref[:1], "bf16", "cfg3 needle at 130003")


@pytest.mark.gpu
def test_peaked_scores_long_context_gqa():
    """q scaled x8 on the long-context GQA layer (scores ~ N(0, 64))."""
    spec = S.workload(3).layer
    lens = (700, 45, 1031, 5000)
    got, di = gpu_decode(spec, lens, seed=5, q_std=8.0)
    assert_parity(got, oracle_decode(di), "bf16", "cfg3 peaked")
