"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

Each test is chosen so that a plausible slip in the oracle (a dropped term, a
transposed factor, a wrong head or group index, a wrong RoPE pairing or sign,
a wrong query position or scale) fails at least one of them:

* full rank with A.B = I (non-symmetric B) reduces to textbook MHA / GQA,
  computed by torch's scaled_dot_product_attention with RoPE written in the
  complex form of RoFormer;
* softmax rows sum to one;
* agreement with a pure-Python brute force that materialises K and V element
  by element in a different loop order, on ragged tiny inputs;
* T = 1 closed form, needle case, position-shift invariance of RoPE,
  GQA-as-replicated-MHA, group-order invariance;
* the parameter counts of Sec. III-C against Table I.
"""

import cmath
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle.decode import decode_attention, max_rel_err, rope
from paper_2607_24331_gb300 import synth as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def small_spec(Hq=4, Hkv=4, d=16, groups=((2, 0), (1,), (3,)), ranks=(8, 16, 4), rank_v=12, theta=1e4):
    return S.LayerSpec(64, Hq, Hkv, d, tuple(tuple(g) for g in groups), tuple(ranks), rank_v, "f32", theta)


def random_inputs(spec, lens, seed=1, q_std=1.0):
    rng = np.random.default_rng(seed)
    n = int(sum(lens))
    B = len(lens)
    q = rng.standard_normal((B, spec.n_q_heads, spec.head_dim)) * q_std
    kc = rng.standard_normal((n, spec.rank_k))
    vc = rng.standard_normal((n, spec.rank_v))
    Bk = np.concatenate([rng.standard_normal((r, len(g) * spec.head_dim)).ravel() / math.sqrt(r)
                         for g, r in zip(spec.groups, spec.ranks)])
    Bv = rng.standard_normal((spec.rank_v, spec.n_kv_heads * spec.head_dim)) / math.sqrt(spec.rank_v)
    starts = S.seq_starts(lens)
    return q, kc, vc, Bk, Bv, starts, np.asarray(lens)


# ---------------------------------------------------------------------------
# RoPE in complex form (RoFormer): pair (i, i + d/2) is the complex number
# x[i] + 1j x[i+d/2], multiplied by exp(1j * pos * theta^(-2i/d)).
# ---------------------------------------------------------------------------

def rope_complex(x, pos, theta):
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    h = d // 2
    z = x[..., :h] + 1j * x[..., h:]
    w = np.array([theta ** (-2.0 * i / d) for i in range(h)])
    z = z * np.exp(1j * np.asarray(pos, dtype=np.float64)[..., None] * w)
    return np.concatenate([z.real, z.imag], axis=-1)


def test_rope_matches_complex_form_and_basic_identities():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((7, 32))
    pos = np.array([0, 1, 5, 127, 4095, 131071, 77])
    for theta in (1e4, 5e5, 1e6):
        y = rope(x, pos, theta)
        np.testing.assert_allclose(y, rope_complex(x, pos, theta), atol=1e-12)
        np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    np.testing.assert_allclose(rope(x, np.zeros(7), 1e4), x, atol=0)
    # composition: R_a R_b = R_{a+b}
    np.testing.assert_allclose(rope(rope(x, pos, 1e4), pos + 3, 1e4), rope(x, 2 * pos + 3, 1e4), atol=1e-9)


# ---------------------------------------------------------------------------
# (i) full rank, A.B = I: reduces to textbook attention
# ---------------------------------------------------------------------------

def _textbook(q, K, V, lens, starts, theta, Hq, Hkv):
    """torch SDPA (fp64) over explicit per-KV-head keys/values, RoPE in complex form."""
    B, _, d = q.shape
    out = np.zeros((B, Hq, d))
    rep = Hq // Hkv
    for b in range(B):
        L, r0 = int(lens[b]), int(starts[b])
        k = np.stack([rope_complex(K[h][r0:r0 + L], np.arange(L), theta) for h in range(Hkv)])
        v = np.stack([V[h][r0:r0 + L] for h in range(Hkv)])
        qq = rope_complex(q[b], np.full(Hq, L - 1), theta)
        kt = torch.from_numpy(k).repeat_interleave(rep, dim=0)[None]
        vt = torch.from_numpy(v).repeat_interleave(rep, dim=0)[None]
        qt = torch.from_numpy(qq)[None, :, None, :]
        o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, scale=1.0 / math.sqrt(d))
        out[b] = o[0, :, 0, :].numpy()
    return out


@pytest.mark.parametrize("Hq,Hkv,groups", [(4, 4, ((2, 0), (1,), (3,))), (8, 2, ((1, 0),)), (6, 3, ((2,), (0, 1)))])
def test_full_rank_identity_factors_equal_textbook_attention(Hq, Hkv, groups):
    d = 8
    ranks = tuple(len(g) * d for g in groups)
    spec = small_spec(Hq, Hkv, d, groups, ranks, Hkv * d, 1e4)
    lens = [5, 1, 9]
    n = sum(lens)
    starts = S.seq_starts(lens)
    rng = np.random.default_rng(3)
    K = [rng.standard_normal((n, d)) for _ in range(Hkv)]
    V = [rng.standard_normal((n, d)) for _ in range(Hkv)]
    q = rng.standard_normal((len(lens), Hq, d)) * 2.0
    # B_g = M_g (random, non-symmetric), cache = K_g M_g^{-1}, so cache . B_g = K_g
    kc_cols, Bk = [], []
    for g in groups:
        Kg = np.concatenate([K[h] for h in g], axis=1)
        M = rng.standard_normal((Kg.shape[1], Kg.shape[1])) + 3 * np.eye(Kg.shape[1])
        kc_cols.append(Kg @ np.linalg.inv(M))
        Bk.append(M.ravel())
    kc = np.concatenate(kc_cols, axis=1)
    Vall = np.concatenate(V, axis=1)
    Mv = rng.standard_normal((Hkv * d, Hkv * d)) + 3 * np.eye(Hkv * d)
    vc = Vall @ np.linalg.inv(Mv)
    got = decode_attention(spec, q, kc, vc, np.concatenate(Bk), Mv, starts, lens)
    ref = _textbook(q, K, V, lens, starts, spec.rope_theta, Hq, Hkv)
    np.testing.assert_allclose(got, ref, atol=1e-10, rtol=1e-10)


# ---------------------------------------------------------------------------
# (ii) softmax rows sum to one
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("q_std", [1.0, 8.0, 40.0])
def test_softmax_rows_sum_to_one(q_std):
    spec = small_spec()
    lens = [1, 17, 64]
    args = random_inputs(spec, lens, seed=5, q_std=q_std)
    _, probs = decode_attention(spec, *args, return_probs=True)
    assert len(probs) == len(lens) * spec.n_q_heads
    for (b, j), p in probs.items():
        assert p.shape == (lens[b],)
        assert abs(p.sum() - 1.0) <= 1e-12
        assert (p >= 0).all()


# ---------------------------------------------------------------------------
# (iii) brute force, element by element, different loop order
# ---------------------------------------------------------------------------

def brute_force(spec, q, kc, vc, Bk, Bv, starts, lens):
    Hq, Hkv, d = spec.n_q_heads, spec.n_kv_heads, spec.head_dim
    rep = Hq // Hkv
    half = d // 2
    # locate every KV head: (group, slot, rank column offset, packed B_k offset)
    where = {}
    roff, boff = 0, 0
    for g, heads in enumerate(spec.groups):
        r = spec.ranks[g]
        for s, h in enumerate(heads):
            where[h] = (s, r, roff, boff, len(heads))
        roff += r
        boff += r * len(heads) * d
    out = np.zeros((len(lens), Hq, d))
    for b in range(len(lens)):
        L, r0 = int(lens[b]), int(starts[b])
        P = L - 1
        for j in range(Hq):
            h = j // rep
            s, r, ro, bo, ng = where[h]
            zq = [complex(q[b][j][i], q[b][j][i + half]) for i in range(half)]
            scores = []
            vals = []
            for t in range(L):
                key = [0.0] * d
                for e in range(d):
                    acc = 0.0
                    for i in range(r):
                        acc += kc[r0 + t][ro + i] * Bk[bo + i * ng * d + s * d + e]
                    key[e] = acc
                sc = 0.0
                for i in range(half):
                    w = spec.rope_theta ** (-2.0 * i / d)
                    zk = complex(key[i], key[i + half]) * cmath.exp(1j * t * w)
                    zqr = zq[i] * cmath.exp(1j * P * w)
                    sc += (zqr.conjugate() * zk).real
                scores.append(sc / math.sqrt(d))
                vals.append([sum(vc[r0 + t][i] * Bv[i][h * d + e] for i in range(spec.rank_v)) for e in range(d)])
            m = max(scores)
            w_ = [math.exp(x - m) for x in scores]
            z = sum(w_)
            for e in range(d):
                out[b][j][e] = sum(w_[t] * vals[t][e] for t in range(L)) / z
    return out


@pytest.mark.parametrize("Hq,Hkv,groups,ranks", [
    (4, 4, ((2, 0), (1,), (3,)), (5, 3, 4)),
    (6, 2, ((1, 0),), (7,)),
    (4, 2, ((1,), (0,)), (3, 6)),
])
def test_oracle_matches_brute_force(Hq, Hkv, groups, ranks):
    spec = small_spec(Hq, Hkv, 8, groups, ranks, 6, 1e4)
    lens = [1, 5, 3]
    args = random_inputs(spec, lens, seed=11, q_std=3.0)
    got = decode_attention(spec, *args)
    ref = brute_force(spec, *args)
    np.testing.assert_allclose(got, ref, atol=1e-12, rtol=1e-11)


# ---------------------------------------------------------------------------
# closed forms and invariants
# ---------------------------------------------------------------------------

def test_single_token_returns_its_value_projection():
    spec = small_spec()
    q, kc, vc, Bk, Bv, starts, lens = random_inputs(spec, [1, 1], seed=2, q_std=5.0)
    got = decode_attention(spec, q, kc, vc, Bk, Bv, starts, lens)
    for b in range(2):
        for j in range(spec.n_q_heads):
            h = oracle.kv_head_of(j, spec.n_q_heads, spec.n_kv_heads)
            np.testing.assert_allclose(got[b, j], vc[b] @ Bv[:, h * 16:(h + 1) * 16], atol=1e-13)


def test_needle_token_dominates():
    spec = small_spec(4, 4, 16, ((0, 1, 2, 3),), (64,), 12)
    lens = [40]
    q, kc, vc, Bk, Bv, starts, _ = random_inputs(spec, lens, seed=4)
    # the group factor is square and invertible: choose token 17's latent so that
    # its RoPE'd key for head 2 is 60 * RoPE'd query direction
    Bg = Bk.reshape(64, 64)
    d = 16
    qrot = rope(q[0, 2], 39, spec.rope_theta)
    k_rot = 60.0 * qrot / np.linalg.norm(qrot)
    k = rope(k_rot, -17, spec.rope_theta)      # undo the key's own rotation at t = 17
    full = np.linalg.solve(Bg.T, np.concatenate([np.zeros(2 * d), k, np.zeros(d)]))
    kc[17] = full
    got = decode_attention(spec, q, kc, vc, Bk, Bv, starts, np.asarray(lens))
    np.testing.assert_allclose(got[0, 2], vc[17] @ Bv[:, 2 * d:3 * d], atol=1e-6)


def test_position_shift_invariance():
    spec = small_spec(theta=1e4)
    lens = [9, 33]
    args = random_inputs(spec, lens, seed=8, q_std=4.0)
    a = decode_attention(spec, *args)
    for shift in (1, 1000, 125000):
        b = decode_attention(spec, *args, pos_offset=shift)
        assert max_rel_err(b, a) < 1e-9


def test_gqa_equals_mha_with_replicated_kv_heads():
    Hq, Hkv, d = 8, 2, 8
    spec = small_spec(Hq, Hkv, d, ((1, 0),), (6,), 5)
    lens = [7, 2]
    q, kc, vc, Bk, Bv, starts, lens_a = random_inputs(spec, lens, seed=21, q_std=2.0)
    rep = Hq // Hkv
    Bg = Bk.reshape(6, 2 * d)              # column blocks: slot 0 = head 1, slot 1 = head 0
    slot = {1: 0, 0: 1}
    cols = [Bg[:, slot[j // rep] * d:(slot[j // rep] + 1) * d] for j in range(Hq)]
    Bk_mha = np.concatenate(cols, axis=1).ravel()
    Bv_mha = np.concatenate([Bv[:, (j // rep) * d:(j // rep + 1) * d] for j in range(Hq)], axis=1)
    mha = small_spec(Hq, Hq, d, (tuple(range(Hq)),), (6,), 5)
    a = decode_attention(spec, q, kc, vc, Bk, Bv, starts, lens_a)
    b = decode_attention(mha, q, kc, vc, Bk_mha, Bv_mha, starts, lens_a)
    np.testing.assert_allclose(a, b, atol=1e-13)


def test_group_order_and_slot_order_invariance():
    spec = small_spec(4, 4, 8, ((2, 0), (1, 3)), (5, 7), 6)
    lens = [6, 11]
    q, kc, vc, Bk, Bv, starts, la = random_inputs(spec, lens, seed=31, q_std=2.0)
    d = 8
    # reorder: groups swapped, and heads inside the first group swapped
    B0 = Bk[:5 * 16].reshape(5, 16)
    B1 = Bk[5 * 16:].reshape(7, 16)
    B0s = np.concatenate([B0[:, d:], B0[:, :d]], axis=1)         # heads (0, 2)
    spec2 = small_spec(4, 4, 8, ((1, 3), (0, 2)), (7, 5), 6)
    kc2 = np.concatenate([kc[:, 5:12], kc[:, 0:5]], axis=1)
    Bk2 = np.concatenate([B1.ravel(), B0s.ravel()])
    a = decode_attention(spec, q, kc, vc, Bk, Bv, starts, la)
    b = decode_attention(spec2, q, kc2, vc, Bk2, Bv, starts, la)
    np.testing.assert_allclose(a, b, atol=1e-13)


def test_subset_evaluation_matches_full():
    spec = small_spec()
    args = random_inputs(spec, [4, 9], seed=9)
    full = decode_attention(spec, *args)
    part = decode_attention(spec, *args, heads=[1, 3], batch_ids=[1])
    np.testing.assert_array_equal(part[1, [1, 3]], full[1, [1, 3]])
    assert np.isnan(part[0]).all()


# ---------------------------------------------------------------------------
# latent append
# ---------------------------------------------------------------------------

def test_latent_append_identity_and_brute_force():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((5, 12))
    A_k = np.eye(12)[:, [3, 0, 7]]
    A_v = np.eye(12)[:, [11, 2]]
    c, v = oracle.latent_append(x, A_k, A_v)
    np.testing.assert_array_equal(c, x[:, [3, 0, 7]])
    np.testing.assert_array_equal(v, x[:, [11, 2]])
    A_k = rng.standard_normal((12, 4))
    A_v = rng.standard_normal((12, 3))
    c, v = oracle.latent_append(x, A_k, A_v)
    for t in range(5):
        for j in range(4):
            assert abs(c[t, j] - sum(x[t, i] * A_k[i, j] for i in range(12))) < 1e-12
        for j in range(3):
            assert abs(v[t, j] - sum(x[t, i] * A_v[i, j] for i in range(12))) < 1e-12


# ---------------------------------------------------------------------------
# Sec. III-C parameter counts and Table I
# ---------------------------------------------------------------------------

def test_grouped_params_identities():
    rng = np.random.default_rng(0)
    for _ in range(20):
        h = int(rng.choice([8, 16, 32]))
        d_h = int(rng.choice([64, 128]))
        m = 2048
        n = h * d_h
        sizes = []
        left = h
        while left:
            s = int(rng.integers(1, left + 1))
            sizes.append(s)
            left -= s
        ranks = [int(rng.integers(1, 200)) for _ in sizes]
        # sum_i (m r_i + r_i h_i d_h) = m sum r_i + n sum r_i alpha_i, alpha_i = h_i / h
        lhs = oracle.grouped_key_params(m, d_h, sizes, ranks)
        rhs = m * sum(ranks) + n * sum(r * s / h for r, s in zip(ranks, sizes))
        assert abs(lhs - rhs) < 1e-6
    # ReCalKV: four heads per group, r_i = r / K, K = h / 4  ->  m r + r n 4 / h
    for h, d_h, r in [(8, 64, 64), (16, 128, 256), (32, 64, 512)]:
        K = h // 4
        assert oracle.grouped_key_params(2048, d_h, [4] * K, [r // K] * K) == \
            oracle.recalkv_key_params(2048, h * d_h, h, r)


def test_table1_key_param_counts():
    with open(os.path.join(GOLDEN, "table1_key_params.json")) as f:
        tab = json.load(f)["models"]
    for name, row in tab.items():
        assert row["recalkv"] + row["difference"] == row["dynacalkv"], name
        assert round(-100.0 * row["difference"] / row["recalkv"], 2) == row["percent"], name
        # ReCalKV entries are sum over layers of (m r + r n 4/h): linear in r, so the
        # summed rank must be a whole number under the stated shapes
        per_rank = oracle.recalkv_key_params(row["m"], row["n"], row["h"], 1)
        assert row["recalkv"] % per_rank == 0, name
        r_sum = row["recalkv"] // per_rank
        assert oracle.recalkv_key_params(row["m"], row["n"], row["h"], r_sum) == row["recalkv"]


# ---------------------------------------------------------------------------
# the parity measure itself: max |got - ref| / ||ref||_inf over the entries the
# reference evaluated (hand-computed cases)
# ---------------------------------------------------------------------------

def test_max_rel_err_hand_computed():
    ref = np.array([[1.0, 2.5], [3.0, -5.0]])
    got = np.array([[1.0, 2.0], [3.0, -4.0]])
    # |d| = 0, 0.5, 0, 1.0 -> 1.0; ||ref||_inf = 5
    assert max_rel_err(got, ref) == pytest.approx(0.2, abs=1e-15)
    assert max_rel_err(ref, ref) == 0.0


def test_max_rel_err_normalises_by_the_reference():
    ref = np.array([2.0, -4.0])
    got = np.array([2.0, -3.0])
    assert max_rel_err(got, ref) == pytest.approx(0.25, abs=1e-15)   # 1 / 4, not 1 / 3
    # scaling `got` alone moves the numerator only
    assert max_rel_err(10 * got, ref) == pytest.approx(26.0 / 4.0, abs=1e-12)   # |20-2|, |-30+4|


def test_max_rel_err_non_finite_got_fails_every_tolerance():
    ref = np.array([1.0, 2.0, 3.0])
    for bad in (np.nan, np.inf, -np.inf):
        got = np.array([1.0, bad, 3.0])
        e = max_rel_err(got, ref)
        assert e == math.inf and not e <= 1e30


def test_max_rel_err_ignores_entries_the_reference_did_not_evaluate():
    ref = np.array([[1.0, np.nan], [np.nan, -2.0]])
    got = np.array([[1.1, 123.0], [np.nan, -2.0]])
    assert max_rel_err(got, ref) == pytest.approx(0.05, abs=1e-15)   # 0.1 / 2
    with pytest.raises(ValueError):
        max_rel_err(got[:1], ref)
    assert max_rel_err(got, np.full_like(ref, np.nan)) == math.inf


def test_oracle_kv_reuse_equals_one_head_at_a_time():
    """Evaluating all heads at once (keys and values of a KV head reused by its
    query heads) equals evaluating each head alone."""
    spec = small_spec(8, 4, 16, ((2, 0), (1,), (3,)), (8, 16, 4), 12)
    lens = [7, 30]
    args = random_inputs(spec, lens, seed=13, q_std=2.0)
    full = decode_attention(spec, *args)
    for j in range(8):
        one = decode_attention(spec, *args, heads=[j])
        np.testing.assert_array_equal(one[:, j], full[:, j])
