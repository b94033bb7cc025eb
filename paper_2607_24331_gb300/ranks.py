"""Rank allocation of DynaCalKV's grouped key factorization (host tooling).

Given the key projection W^(k) [m x n] of one layer, split column-wise into K
head groups W_i [m x h_i d_h] (Sec. III-C), and the layer's rank budget r, this
module allocates the group ranks r_i the way Sec. III-C and Algorithm 1 describe:

* ``init_ranks_by_energy``: r_i = round(r * energy(W_i) / energy(W^(k))), the
  energy of a matrix being the sum of its squared singular values;
* ``greedy_adjust``: while sum_i r_i alpha_i > 4 r / h (alpha_i = h_i / h, the
  bound being ReCalKV's parameter count), lower by one the rank of the group
  whose reduction loses the least energy per unit of alpha, Delta E_i / alpha_i;
* ``key_param_count``: sum_i (m r_i + r_i h_i d_h) = m sum_i r_i + n sum_i r_i alpha_i;
* ``cluster_objective``: sum_i ||W_i - L_i R_i||_F^2 + lambda (r - sum_i r_i),
  the criterion that picks the number of groups (lambda = 1 in the paper), with
  the truncated-SVD error of each group taken from its singular values.

The head clustering itself (CKA similarity, agglomerative clustering) and the
SVD of real weights run offline on calibration data and are not part of this
library; the functions here take the groups' singular values as input.  The
decode kernels need every rank to be a multiple of 16, which the paper does not;
``kernel_ranks`` rounds an allocation down to that grid and ``greedy_adjust``
accepts the rank step it lowers by.
"""

from __future__ import annotations

from typing import List, Sequence

import numpy as np


def group_energy(sigma: Sequence[float]) -> float:
    """Energy of a matrix from its singular values: sum of their squares (Sec. III-C)."""
    s = np.asarray(sigma, dtype=np.float64)
    return float(np.dot(s, s))


def init_ranks_by_energy(energies: Sequence[float], r: int) -> List[int]:
    """Initial group ranks proportional to the groups' energies (Sec. III-C):
    r_i = round(r * E_i / E) with E the energy of the whole key matrix, which is the
    sum of the groups' energies because the groups partition its columns."""
    e = np.asarray(energies, dtype=np.float64)
    if e.ndim != 1 or len(e) == 0 or (e < 0).any() or e.sum() <= 0:
        raise ValueError("energies must be a non-empty list of non-negative numbers with a positive sum")
    if r < 0:
        raise ValueError("rank budget must be non-negative")
    # numpy's round is round-half-to-even; the paper says only "rounded to the nearest integer"
    return [int(np.round(r * ei / e.sum())) for ei in e]


def budget_bound(r: int, h: int) -> float:
    """Right-hand side of the parameter constraint sum_i r_i alpha_i <= 4 r / h (Sec. III-C):
    ReCalKV's count with groups of four heads at rank r / K each."""
    return 4.0 * r / h


def _energy_loss(sigma: np.ndarray, rank: int, step: int) -> float:
    """Energy lost when a group truncated at ``rank`` drops to ``rank - step``: the squares of
    the singular values sigma[rank - step : rank] (singular values in descending order)."""
    lo = max(rank - step, 0)
    part = sigma[lo:rank]
    return float(np.dot(part, part))


def greedy_adjust(ranks: Sequence[int], group_heads: Sequence[int], spectra: Sequence[Sequence[float]], r: int,
                  h: int, step: int = 1) -> List[int]:
    """Greedy rank adjustment of Sec. III-C.

    ranks        initial r_i (e.g. from ``init_ranks_by_energy``)
    group_heads  h_i, heads of each group (alpha_i = h_i / h)
    spectra      singular values of each W_i, in descending order
    r, h         the layer's rank budget and head count
    step         rank decrement per iteration (1 in the paper; 16 keeps kernel-sized ranks)

    While sum_i r_i alpha_i exceeds 4 r / h, the group with the smallest normalized
    energy loss Delta E_i / alpha_i (Delta E_i: the energy of the singular values the
    decrement drops) loses ``step`` ranks; ties go to the lower group index.  A rank
    above the group's number of singular values first drops to that number (those
    ranks carry no energy).  Returns the adjusted ranks.
    """
    k = len(ranks)
    if len(group_heads) != k or len(spectra) != k:
        raise ValueError("ranks, group_heads and spectra must have one entry per group")
    if step < 1:
        raise ValueError("step must be positive")
    if sum(group_heads) != h:
        raise ValueError("group head counts must add up to h")
    sig = [np.sort(np.asarray(s, dtype=np.float64))[::-1] for s in spectra]
    alpha = [hi / h for hi in group_heads]
    cur = [min(int(ri), len(si)) for ri, si in zip(ranks, sig)]
    bound = budget_bound(r, h)

    def load(rs):
        return sum(ri * ai for ri, ai in zip(rs, alpha))

    # tolerance for the float comparison of equal sums (e.g. the ReCalKV layout itself)
    eps = 1e-9 * max(1.0, bound)
    while load(cur) > bound + eps:
        best, best_cost = -1, np.inf
        for i in range(k):
            if cur[i] <= 0:
                continue
            cost = _energy_loss(sig[i], cur[i], step) / alpha[i]
            if cost < best_cost:
                best, best_cost = i, cost
        if best < 0:
            break  # every rank is zero: nothing left to lower
        cur[best] = max(cur[best] - step, 0)
    return cur


def kernel_ranks(ranks: Sequence[int], multiple: int = 16) -> List[int]:
    """Ranks rounded down to the decode kernels' grid (multiples of ``multiple``), at least one
    step each.  Rounding down keeps the parameter constraint satisfied unless a rank below one
    step is raised to it."""
    return [max(multiple, (int(ri) // multiple) * multiple) for ri in ranks]


def key_param_count(m: int, d_h: int, group_heads: Sequence[int], ranks: Sequence[int]) -> int:
    """Parameters of the factorized key projection, sum_i (m r_i + r_i h_i d_h) (Sec. III-C)."""
    return int(sum(m * ri + ri * hi * d_h for ri, hi in zip(ranks, group_heads)))


def truncation_error(sigma: Sequence[float], rank: int) -> float:
    """||W_i - L_i R_i||_F^2 of the rank-``rank`` truncated SVD: the energy of the dropped
    singular values (Eckart-Young)."""
    s = np.sort(np.asarray(sigma, dtype=np.float64))[::-1]
    tail = s[rank:]
    return float(np.dot(tail, tail))


def cluster_objective(spectra: Sequence[Sequence[float]], ranks: Sequence[int], r: int, lam: float = 1.0) -> float:
    """Selection criterion for the number of groups (Sec. III-C):
    sum_i ||W_i - L_i R_i||_F^2 + lambda (r - sum_i r_i)."""
    err = sum(truncation_error(s, ri) for s, ri in zip(spectra, ranks))
    return float(err + lam * (r - sum(int(ri) for ri in ranks)))


def allocate(group_heads: Sequence[int], spectra: Sequence[Sequence[float]], r: int, step: int = 1) -> List[int]:
    """InitRanksByEnergy followed by GreedyAdjust (Algorithm 1) for one clustering."""
    h = int(sum(group_heads))
    r0 = init_ranks_by_energy([group_energy(s) for s in spectra], r)
    return greedy_adjust(r0, group_heads, spectra, r, h, step=step)
