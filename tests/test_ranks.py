"""Rank allocation of the grouped key factorization (Sec. III-C, Algorithm 1's
InitRanksByEnergy and GreedyAdjust), checked against facts outside its own
arithmetic: the Frobenius norm and explicit truncated SVDs (numpy), ReCalKV's
layout as the boundary of the parameter constraint, and greedy steps worked
out by hand."""

import numpy as np
import pytest

from paper_2607_24331_gb300 import dck
from paper_2607_24331_gb300 import ranks as R
from paper_2607_24331_gb300 import synth as S


def _rand(m, n, seed):
    return np.random.default_rng(seed).standard_normal((m, n))


def test_energy_is_the_squared_frobenius_norm():
    for seed, (m, n) in enumerate([(40, 12), (9, 30), (16, 16)]):
        W = _rand(m, n, seed)
        sigma = np.linalg.svd(W, compute_uv=False)
        assert R.group_energy(sigma) == pytest.approx(np.linalg.norm(W, "fro") ** 2, rel=1e-12)


def test_whole_matrix_energy_is_the_sum_over_column_groups():
    # the denominator of the energy ratio: groups partition W^(k) column-wise
    W = _rand(64, 8 * 16, 3)
    cols = [(0, 32), (32, 48), (48, 128)]
    parts = [R.group_energy(np.linalg.svd(W[:, a:b], compute_uv=False)) for a, b in cols]
    whole = R.group_energy(np.linalg.svd(W, compute_uv=False))
    assert sum(parts) == pytest.approx(whole, rel=1e-12)


def test_truncation_error_matches_an_explicit_truncated_svd():
    W = _rand(30, 20, 7)
    U, s, Vt = np.linalg.svd(W, full_matrices=False)
    for k in (0, 1, 5, 19, 20):
        Wk = (U[:, :k] * s[:k]) @ Vt[:k]
        assert R.truncation_error(s, k) == pytest.approx(np.linalg.norm(W - Wk, "fro") ** 2, rel=1e-10, abs=1e-10)


def test_init_ranks_are_proportional_to_energy():
    assert R.init_ranks_by_energy([1.0, 1.0, 1.0, 1.0], 256) == [64, 64, 64, 64]
    assert R.init_ranks_by_energy([1.0, 3.0], 64) == [16, 48]
    assert R.init_ranks_by_energy([2.0, 1.0, 1.0], 100) == [50, 25, 25]
    with pytest.raises(ValueError):
        R.init_ranks_by_energy([0.0, 0.0], 10)


def test_recalkv_layout_sits_on_the_constraint_and_is_left_unchanged():
    # K = h/4 groups of four heads at rank r/K each: sum r_i alpha_i = r/K = 4r/h
    h, r = 32, 1024
    heads = [4] * 8
    ranks = [r // 8] * 8
    spectra = [np.linspace(5.0, 0.1, 512) for _ in heads]
    load = sum(ri * hi / h for ri, hi in zip(ranks, heads))
    assert load == pytest.approx(R.budget_bound(r, h))
    assert R.greedy_adjust(ranks, heads, spectra, r, h) == ranks


def test_greedy_steps_worked_by_hand():
    # h = 8, alpha = (0.25, 0.75), r = 8: bound 4r/h = 4; start (2, 6): load 0.5 + 4.5 = 5.
    h, r, heads = 8, 8, [2, 6]
    sig1 = [5.0, 4.0, 3.0, 2.0, 1.5, 1.0]
    # group 0 spectrum (10, 1): dropping its 2nd value costs 1 / 0.25 = 4; group 1 dropping
    # 1.0 costs 1 / 0.75 = 1.33 -> group 1 (5); then 1.5^2 / 0.75 = 3 < 4 -> group 1 (4);
    # load 0.5 + 3.0 = 3.5 <= 4
    assert R.greedy_adjust([2, 6], heads, [[10.0, 1.0], sig1], r, h) == [2, 4]
    # group 0 spectrum (10, 0.5): 0.25 / 0.25 = 1 < 1.33 -> group 0 (1); load 4.75; then
    # 100 / 0.25 = 400 against 1.33 -> group 1 (5); load 0.25 + 3.75 = 4.0 <= 4
    assert R.greedy_adjust([2, 6], heads, [[10.0, 0.5], sig1], r, h) == [1, 5]


def test_greedy_result_meets_the_budget_and_only_lowers_ranks():
    rng = np.random.default_rng(11)
    for trial in range(20):
        h = 32
        sizes = rng.multinomial(h - 8, np.ones(8) / 8) + 1
        r = int(rng.integers(256, 2048))
        spectra = [np.sort(rng.gamma(2.0, 1.0, size=min(4096, s * 128)))[::-1] * rng.uniform(0.5, 3.0)
                   for s in sizes]
        r0 = R.init_ranks_by_energy([R.group_energy(sp) for sp in spectra], r)
        out = R.greedy_adjust(r0, list(sizes), spectra, r, h)
        assert sum(ri * s / h for ri, s in zip(out, sizes)) <= R.budget_bound(r, h) + 1e-9
        assert all(0 <= a <= b for a, b in zip(out, r0))


def test_parameter_count_closed_form():
    # sum_i (m r_i + r_i h_i d_h) = m sum r_i + n sum r_i alpha_i, n = h d_h; ReCalKV: m r + r n 4/h
    m, d, h = 2048, 64, 32
    rng = np.random.default_rng(5)
    sizes = [2, 3, 3, 4, 4, 5, 5, 6]
    ranks = [int(x) for x in rng.integers(16, 200, size=len(sizes))]
    n = h * d
    closed = m * sum(ranks) + n * sum(ri * s / h for ri, s in zip(ranks, sizes))
    assert R.key_param_count(m, d, sizes, ranks) == pytest.approx(closed, rel=1e-12)
    r = 1024
    assert R.key_param_count(m, d, [4] * 8, [r // 8] * 8) == m * r + r * n * 4 // h


def test_cluster_objective_with_explicit_factorizations():
    rng = np.random.default_rng(2)
    Ws = [rng.standard_normal((48, 32)), rng.standard_normal((48, 64))]
    ranks, r = [10, 30], 48
    err = 0.0
    for W, k in zip(Ws, ranks):
        U, s, Vt = np.linalg.svd(W, full_matrices=False)
        L, Rm = U[:, :k] * np.sqrt(s[:k]), np.sqrt(s[:k])[:, None] * Vt[:k]  # L = U S^1/2, R = S^1/2 V^T
        err += np.linalg.norm(W - L @ Rm, "fro") ** 2
    spectra = [np.linalg.svd(W, compute_uv=False) for W in Ws]
    assert R.cluster_objective(spectra, ranks, r) == pytest.approx(err + (r - 40), rel=1e-10)
    assert R.cluster_objective(spectra, ranks, r, lam=0.0) == pytest.approx(err, rel=1e-10)


def test_kernel_sized_allocation_gives_a_layer_the_library_accepts():
    # DynaCalKV grouping of the benchmark MHA layer, synthetic group spectra, rank step 16
    base = S.workload(1).layer
    groups = base.groups
    h, r = base.n_kv_heads, 1024
    rng = np.random.default_rng(0)
    spectra = [np.sort(rng.gamma(1.5, 1.0, size=len(g) * 128))[::-1] * (1.0 + 0.3 * i)
               for i, g in enumerate(groups)]
    r0 = R.kernel_ranks(R.init_ranks_by_energy([R.group_energy(s) for s in spectra], r))
    out = R.greedy_adjust(r0, [len(g) for g in groups], spectra, r, h, step=16)
    assert all(x % 16 == 0 and x > 0 for x in out)
    assert sum(x * len(g) / h for x, g in zip(out, groups)) <= R.budget_bound(r, h) + 1e-9
    spec = S.LayerSpec(base.hidden, base.n_q_heads, base.n_kv_heads, base.head_dim, groups, tuple(out),
                       base.rank_v, base.dtype, base.rope_theta)
    assert dck.dck_validate_desc(dck.Layer.from_spec(spec)) == dck.DCK_OK
