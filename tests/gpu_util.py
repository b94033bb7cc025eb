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
