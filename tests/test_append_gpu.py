"""Latent append through the C ABI vs the fp64 oracle.

Bound per element (derived from the arithmetic): the kernel accumulates
fp32 products of stored values and rounds once to the storage dtype, so
|c_gpu - c| <= u_store |c| + K * 2^-23 * sum_k |x_k a_k|, with u_store = 2^-8
for bf16 (one rounding, half an ulp, plus slack of a second half-ulp) and
2^-23 for fp32.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2607_24331_gb300 import dck, device
from paper_2607_24331_gb300 import synth as S

pytestmark = pytest.mark.gpu


def _check(spec, n_tok, rows, n_rows, seed=0):
    x, A_k, A_v = S.make_append_inputs(spec, n_tok, seed=seed)
    buf = device.AppendBuffers(spec, n_tok, n_rows).load_host(x, A_k, A_v, rows)
    dck.check(buf.run(), "dck_latent_append")
    torch.cuda.synchronize()
    assert dck.dck_last_device_error() == dck.DCK_OK
    c, v = oracle.latent_append(x, A_k, A_v)
    u = 2.0 ** -8 if spec.dtype == "bf16" else 2.0 ** -23
    ck = buf.kcache.float().cpu().numpy().astype(np.float64)
    cv = buf.vcache.float().cpu().numpy().astype(np.float64)
    for got, ref, A in ((ck, c, A_k), (cv, v, A_v)):
        absdot = np.abs(x.astype(np.float64)) @ np.abs(A.astype(np.float64))
        bound = u * np.abs(ref) + spec.hidden * 2.0 ** -23 * absdot
        diff = np.abs(got[rows] - ref)
        assert (diff <= bound).all(), float((diff / np.maximum(bound, 1e-30)).max())
        untouched = np.setdiff1d(np.arange(n_rows), rows)
        assert (got[untouched] == 0).all()


@pytest.mark.parametrize("cfg", [0, 1, 2, 3])
@pytest.mark.parametrize("n_tok", [1, 16, 200])
def test_append_small(cfg, n_tok):
    spec = S.workload(cfg).layer
    rng = np.random.default_rng(n_tok)
    n_rows = 3 * n_tok + 5
    rows = rng.choice(n_rows, size=n_tok, replace=False)
    _check(spec, n_tok, rows, n_rows, seed=cfg)


@pytest.mark.parametrize("cfg,n_tok", [(1, 300), (3, 1000), (2, 257)])
def test_append_long_ragged(cfg, n_tok):
    """Appends above the split-K size run as persistent CTA pairs over 256-token x 256-column tiles:
    token counts that leave a ragged last block, scattered destination rows, a key width (704) whose
    last tile reaches past R_k."""
    spec = S.workload(cfg).layer
    rng = np.random.default_rng(n_tok + cfg)
    n_rows = 2 * n_tok + 3
    rows = rng.choice(n_rows, size=n_tok, replace=False)
    _check(spec, n_tok, rows, n_rows, seed=10 + cfg)


def test_append_prefill_8192_tokens_per_sequence():
    """Latent-append prefill of 2 x 8192 tokens of the long-context GQA layer."""
    spec = S.workload(3).layer
    n_tok = 2 * 8192
    rows = np.arange(n_tok, dtype=np.int64)
    _check(spec, n_tok, rows, n_tok, seed=3)


def test_append_bad_row_is_reported():
    spec = S.workload(1).layer
    x, A_k, A_v = S.make_append_inputs(spec, 4)
    buf = device.AppendBuffers(spec, 4, 8).load_host(x, A_k, A_v, [0, 1, 99, 3])
    dck.check(buf.run(), "append")
    assert dck.dck_last_device_error() == dck.DCK_ERR_INVALID
