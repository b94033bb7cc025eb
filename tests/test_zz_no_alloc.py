"""dck_decode_attention_noalloc: decode attention for callers that cannot
allocate device memory (a runtime whose memory is all reserved by its own
pool, a plug-in given only its tensors, a loop that must not allocate after
start-up).  It must give the regular entry point's results, call after call,
from its fixed library-owned scratch, and refuse requests larger than that
scratch.  This file is collected last so that a failure here comes after
every other test has run."""

import numpy as np
import pytest
import torch

from paper_2607_24331_gb300 import dck, device
from paper_2607_24331_gb300 import synth as S
from gpu_util import TOL

pytestmark = pytest.mark.gpu


def _regular_and_noalloc(spec, lens, seed):
    buf = device.DecodeBuffers(spec, lens).load_host(S.make_decode_inputs(spec, lens, seed=seed, q_std=3.0))
    dck.check(buf.run(), "dck_decode_attention")
    ref = buf.out.clone()
    out = torch.full_like(buf.out, float("nan"))
    r = dck.dck_decode_attention_noalloc(buf.layer, buf.q, buf.kcache, buf.vcache, buf.n_rows, buf.B_k, buf.B_v,
                                         buf.seq_start, buf.seq_len, buf.B, spec.rope_theta, out)
    dck.check(r, "dck_decode_attention_noalloc")
    torch.cuda.synchronize()
    assert dck.dck_last_device_error() == dck.DCK_OK
    return ref.float().cpu().numpy(), out.float().cpu().numpy()


def test_noalloc_matches_regular_entry_point_on_two_calls_in_a_row():
    cases = [(S.workload(1).layer, (300, 1, 129), 11),   # MHA, tensor-core kernel
             (S.workload(2).layer, (517, 64), 12)]       # GQA, different partial layout
    for spec, lens, seed in cases:
        ref, got = _regular_and_noalloc(spec, lens, seed)
        assert np.isfinite(got).all()
        err = np.abs(got - ref).max() / np.abs(ref).max()
        assert err <= TOL[spec.dtype], err


def test_noalloc_rejects_requests_beyond_its_scratch():
    # 4096 one-token sequences with r_v = 2048 need about 150 MB of partials
    spec = S.LayerSpec(4096, 32, 32, 128, (tuple(range(32)),), (256,), 2048, "bf16", 1e4)
    lens = (1,) * 4096
    buf = device.DecodeBuffers(spec, lens).synth(seed=1)   # valid buffers of the full request
    assert dck.dck_decode_workspace_size(buf.layer, buf.B, buf.n_rows) > (32 << 20)
    r = dck.dck_decode_attention_noalloc(buf.layer, buf.q, buf.kcache, buf.vcache, buf.n_rows, buf.B_k, buf.B_v,
                                         buf.seq_start, buf.seq_len, buf.B, spec.rope_theta, buf.out)
    assert r == dck.DCK_ERR_WORKSPACE
