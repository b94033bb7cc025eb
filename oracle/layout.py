"""Parameter counts of the key factors (Sec. III-C, Table I).

TEST INFRASTRUCTURE ONLY (see the package docstring).

A key projection W^(k) in R^{m x n}, n = h d_h, is split into K head groups
W_i (h_i heads each) with W_i ~ L_i R_i, L_i in R^{m x r_i},
R_i in R^{r_i x h_i d_h}.  The factors hold sum_i (m r_i + r_i h_i d_h)
numbers.  ReCalKV's fixed grouping (four heads per group, r_i = r/K,
K = h/4) gives m r + r n 4/h.
"""

from __future__ import annotations

from typing import Sequence


def grouped_key_params(m: int, d_h: int, group_sizes: Sequence[int], ranks: Sequence[int]) -> int:
    """sum_i (m r_i + r_i h_i d_h): entries of all L_i and R_i of one key projection."""
    return int(sum(m * r + r * h * d_h for h, r in zip(group_sizes, ranks)))


def recalkv_key_params(m: int, n: int, h: int, r: int) -> int:
    """m r + r n 4/h: the fixed four-head grouping with a uniform rank split."""
    return int(m * r + (r * n * 4) // h)
