"""Prefill attention through the C ABI (dck_prefill_attention) against the
fp64 oracle's prefill_attention: causal attention of each sequence's last Q_b
cache rows over its prefix, keys and values rebuilt from the latents
(Sec. III-A, III-C, III-D).

Cases (the value reconstruction by the pair GEMM in all but the max_len case,
where the reconstruction kernel rebuilds values too): Q = 1 (the decode call), Q = L (a whole prompt), ragged Q across the
batch, query and key tiles cut at and around the 128-row boundaries, MHA and
both GQA layers, Q = 0 (nothing written), invalid sequences (recorded and
zeroed), and a full 4096-token prompt sampled on two heads.  The tolerance is
the decode one: max|o - o_ref| / ||o_ref||_inf <= 2e-2 for bf16 latents with
fp32 accumulation (probabilities rounded to bf16 before the value product).
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2607_24331_gb300 import dck, device
from paper_2607_24331_gb300 import synth as S
from gpu_util import assert_parity

pytestmark = pytest.mark.gpu

SENTINEL = 7.0


def _run(spec, lens, q_lens, seed, q_max=None, q_std=1.0, max_len=None):
    di = S.make_decode_inputs(spec, lens, seed=seed)
    B = len(lens)
    q_max = max(max(q_lens), 1) if q_max is None else q_max
    q = S.make_prefill_q(spec, B, q_max, seed=seed, q_std=q_std)
    buf = device.DecodeBuffers(spec, lens).load_host(di)
    dt = device.TORCH_DTYPE[spec.dtype]
    qd = torch.from_numpy(q).to("cuda", dt)
    ql = torch.tensor(q_lens, dtype=torch.int32, device="cuda")
    out = torch.full((B, q_max, spec.n_q_heads, spec.head_dim), SENTINEL, dtype=dt, device="cuda")
    ws_bytes = dck.dck_prefill_workspace_size(buf.layer, buf.n_rows)
    assert ws_bytes > 0
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    max_len = max(lens) if max_len is None else max_len
    dck.check(dck.dck_prefill_attention(buf.layer, qd, ql, q_max, buf.kcache, buf.vcache, buf.n_rows, buf.B_k,
                                        buf.B_v, buf.seq_start, buf.seq_len, B, max_len, spec.rope_theta, out, ws,
                                        ws_bytes), "dck_prefill_attention")
    torch.cuda.synchronize()
    # values rebuilt by the pair GEMM over all cache rows when the rows in use can be most of the
    # cache (then three launches), else by the reconstruction kernel with the keys (two)
    assert dck.dck_last_launch_count() == (3 if buf.n_rows <= 2 * B * max_len else 2)
    return out.float().cpu().numpy().astype(np.float64), q, di


def _oracle(spec, q, q_lens, di, heads=None):
    return oracle.prefill_attention(spec, q, q_lens, di.kcache, di.vcache, di.B_k, di.B_v, di.seq_start,
                                    di.seq_lens, heads=heads)


def _check(got, ref, q_lens, what):
    for b, Q in enumerate(q_lens):
        assert np.isfinite(got[b, :Q]).all(), (what, b)
        assert (got[b, Q:] == SENTINEL).all(), (what, b, "rows past Q_b must stay untouched")
    mask = np.isfinite(ref)
    return assert_parity(np.where(mask, got, np.nan), ref, "bf16", what)


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_prefill_q1_qL_and_ragged(cfg):
    spec = S.workload(cfg).layer
    lens = (300, 129, 1000, 128)
    q_lens = (300, 1, 37, 128)          # Q = L, Q = 1, ragged, Q = L at one whole tile
    assert dck.dck_last_device_error() == dck.DCK_OK
    got, q, di = _run(spec, lens, q_lens, seed=70 + cfg)
    assert dck.dck_last_device_error() == dck.DCK_OK
    _check(got, _oracle(spec, q, q_lens, di), q_lens, f"prefill cfg{cfg}")


@pytest.mark.parametrize("cfg", [1, 3])
def test_prefill_tile_edges(cfg):
    """Sequence lengths and query counts at and around the 128-row tiles of keys
    and of queries (a query tile holds 128 / (Hq / Hkv) query positions)."""
    spec = S.workload(cfg).layer
    lens = (127, 256, 257, 385, 16, 640)
    q_lens = (127, 255, 129, 17, 16, 640)
    got, q, di = _run(spec, lens, q_lens, seed=80 + cfg)
    assert dck.dck_last_device_error() == dck.DCK_OK
    _check(got, _oracle(spec, q, q_lens, di), q_lens, f"prefill edges cfg{cfg}")


def test_prefill_q1_equals_decode():
    """Q_b = 1 is the decode call: the prefill kernels against the decode kernels
    (both within tolerance of the oracle, and of each other)."""
    spec = S.workload(2).layer
    lens = (2000, 77, 4096)
    got, q, di = _run(spec, lens, (1, 1, 1), seed=90)
    di_dec = S.DecodeInputs(spec, q[:, 0].copy(), di.kcache, di.vcache, di.B_k, di.B_v, di.seq_start, di.seq_lens)
    buf = device.DecodeBuffers(spec, lens).load_host(di_dec)
    dck.check(buf.run(), "dck_decode_attention")
    dec = buf.out.float().cpu().numpy().astype(np.float64)
    ref = oracle.decode_attention(spec, di_dec.q, di.kcache, di.vcache, di.B_k, di.B_v, di.seq_start, di.seq_lens)
    assert_parity(got[:, 0], ref, "bf16", "prefill Q=1 vs decode oracle")
    assert_parity(got[:, 0], dec, "bf16", "prefill Q=1 vs decode kernels")


def test_prefill_zero_queries_and_invalid_sequences():
    spec = S.workload(1).layer
    lens = (200, 50, 300, 40)
    q_lens = (20, 0, 301, 40)            # sequence 2 asks for more queries than it has rows
    got, q, di = _run(spec, lens, q_lens, seed=95, q_max=301)
    assert dck.dck_last_device_error() == dck.DCK_ERR_INVALID
    assert (got[1] == SENTINEL).all(), "Q_b = 0 writes nothing"
    assert (got[2] == 0).all(), "an invalid sequence's output is zero"
    ok = [0, 3]
    ref = oracle.prefill_attention(spec, q[ok], [q_lens[b] for b in ok], di.kcache, di.vcache, di.B_k, di.B_v,
                                   di.seq_start[ok], di.seq_lens[ok])
    for i, b in enumerate(ok):
        Q = q_lens[b]
        assert_parity(got[b, :Q], ref[i, :Q], "bf16", f"valid sequence {b} beside invalid ones")


def test_prefill_longer_than_max_seq_len_is_reported():
    spec = S.workload(2).layer
    lens = (300, 200)
    got, q, di = _run(spec, lens, (5, 5), seed=96, max_len=256)
    assert dck.dck_last_device_error() != dck.DCK_OK
    assert (got[0] == 0).all()
    ref = oracle.prefill_attention(spec, q[1:], [5], di.kcache, di.vcache, di.B_k, di.B_v, di.seq_start[1:],
                                   di.seq_lens[1:])
    assert_parity(got[1, :5], ref[0, :5], "bf16", "the valid sequence")


def test_prefill_peaked_scores():
    spec = S.workload(3).layer
    lens = (700, 333)
    q_lens = (700, 100)
    got, q, di = _run(spec, lens, q_lens, seed=97, q_std=8.0)
    assert dck.dck_last_device_error() == dck.DCK_OK
    _check(got, _oracle(spec, q, q_lens, di), q_lens, "prefill peaked")


def test_prefill_full_prompt_4096_sampled_heads():
    """Two 4096-token prompts of the 7B MHA layer (Q = L), every query of two heads."""
    spec = S.workload(1).layer
    lens = (4096, 4096)
    got, q, di = _run(spec, lens, lens, seed=98)
    assert dck.dck_last_device_error() == dck.DCK_OK
    heads = [0, 31]
    ref = _oracle(spec, q, lens, di, heads=heads)
    for j in heads:
        assert_parity(got[:, :, j], ref[:, :, j], "bf16", f"4096-token prompt head {j}")
