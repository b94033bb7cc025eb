"""Latent append, fp64: the cached representation of new tokens.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Sec. III-A caches z = x L instead of x W.  Sec. III-C gives every key group
its own L_g (columns of A_k, concatenated in group order), Sec. III-D one
L_v for the values (A_v).  For tokens x [n, D]:
    key latents   = x . A_k   [n, R_k]
    value latents = x . A_v   [n, r_v]
"""

from __future__ import annotations

import numpy as np


def latent_append(x, A_k, A_v):
    """(x A_k, x A_v) in fp64 from the stored (rounded) inputs."""
    x = np.asarray(x, dtype=np.float64)
    return x @ np.asarray(A_k, dtype=np.float64), x @ np.asarray(A_v, dtype=np.float64)
