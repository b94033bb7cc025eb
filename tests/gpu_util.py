"""Helpers of the GPU parity tests: run the library, compare with the oracle."""

import numpy as np
import torch

import oracle
from oracle.decode import max_rel_err
from paper_2607_24331_gb300 import dck, device
from paper_2607_24331_gb300 import synth as S

# Tolerances of the decode output, max|o_gpu - o_oracle| / ||o_oracle||_inf:
# bf16 latents with fp32 accumulation, and the fp32 layer.
TOL = {"bf16": 2e-2, "f32": 1e-5}


def gpu_decode(spec, lens, di=None, seed=0, q_std=1.0, kernel=0):
    if di is None:
        di = S.make_decode_inputs(spec, lens, seed=seed, q_std=q_std)
    buf = device.DecodeBuffers(spec, lens).load_host(di)
    prev = dck.dck_set_decode_kernel(kernel)
    try:
        dck.check(buf.run(), "dck_decode_attention")
        torch.cuda.synchronize()
    finally:
        dck.dck_set_decode_kernel(prev)
    assert dck.dck_last_device_error() == dck.DCK_OK
    return buf.out.float().cpu().numpy().astype(np.float64), di


def oracle_decode(di, heads=None, batch_ids=None):
    return oracle.decode_attention(di.spec, di.q, di.kcache, di.vcache, di.B_k, di.B_v, di.seq_start,
                                   di.seq_lens, heads=heads, batch_ids=batch_ids)


def assert_parity(got, ref, dtype, what=""):
    err = max_rel_err(got, ref)
    print(f"{what} max|d|/||o||inf = {err:.3e}")
    assert err <= TOL[dtype], (what, err)
    return err


def sm_count():
    return torch.cuda.get_device_properties(0).multi_processor_count


def leftover_sequences(lens, sms):
    """Sequences with tiles in the finely split leftover range of the tensor-core
    path: sequences are cut into 256-token pair tiles, split over the CTA pairs
    (sms // 2 of them on a GPU whose TPCs all hold two SMs); with fewer than 8
    pair tiles per pair, those from floor(NP / P) * P on are shared out by
    groups of heads."""
    nts = [(int(L) + 255) // 256 for L in lens]
    NP, P = sum(nts), sms // 2
    NPm = NP // P * P if NP // P < 8 else NP
    out, pre = [], 0
    for b, n in enumerate(nts):
        if n and pre + n > NPm:
            out.append(b)
        pre += n
    return out


def plant_needle(di, b, t, j, score=30.0):
    """Rewrites token t of sequence b so that its key, for query head j, scores
    `score` (natural-log units, after the 1/sqrt(d) scale) against that head's
    query: the group latent is the direction that maximises the score,
    c = alpha w / |w| with w = B_slot RoPE(RoPE(q_j, L - 1), -t), rounded to the
    storage dtype.  Returns the row written."""
    spec = di.spec
    d = spec.head_dim
    h = oracle.kv_head_of(j, spec.n_q_heads, spec.n_kv_heads)
    g = next(i for i, hs in enumerate(spec.groups) if h in hs)
    s = spec.groups[g].index(h)
    r_g, n_g = spec.ranks[g], len(spec.groups[g])
    off = spec.bk_offsets()
    Bg = np.asarray(di.B_k[off[g]:off[g + 1]], dtype=np.float64).reshape(r_g, n_g * d)
    B_slot = Bg[:, s * d:(s + 1) * d]
    L = int(di.seq_lens[b])
    qr = oracle.rope(np.asarray(di.q[b, j], dtype=np.float64), L - 1, spec.rope_theta)
    w = B_slot @ oracle.rope(qr, -t, spec.rope_theta)
    c = w * (score * np.sqrt(d) / (w @ w))
    row = int(di.seq_start[b]) + t
    r0 = spec.rank_offsets()[g]
    di.kcache[row, r0:r0 + r_g] = S.round_to(c.astype(np.float32), spec.dtype)
    return row
