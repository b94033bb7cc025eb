"""dck_decode_attention_noalloc: decode attention for callers that cannot
allocate device memory (a runtime whose memory is all reserved by its own
pool, a plug-in given only its tensors, a loop that must not allocate after
start-up).  It runs the regular entry point's kernels on the same inputs, so
its output must equal the regular entry point's bit for bit, call after call,
from its fixed library-owned scratch, without changing the device's free
memory; it must refuse requests larger than that scratch.  This file is
collected last so that a failure here comes after every other test has run."""

import numpy as np
import pytest
import torch

from paper_2607_24331_gb300 import dck, device
from paper_2607_24331_gb300 import synth as S
from gpu_util import TOL, assert_parity, oracle_decode

pytestmark = pytest.mark.gpu


def _noalloc(buf, spec, out):
    return dck.dck_decode_attention_noalloc(buf.layer, buf.q, buf.kcache, buf.vcache, buf.n_rows, buf.B_k, buf.B_v,
                                            buf.seq_start, buf.seq_len, buf.B, spec.rope_theta, out)


def test_noalloc_matches_regular_entry_point_on_two_calls_in_a_row():
    cases = [(S.workload(1).layer, (300, 1, 129), 11),   # MHA, query-folded tensor-core kernels
             (S.workload(2).layer, (517, 64), 12)]       # GQA, key-mode kernels, other partial layout
    for spec, lens, seed in cases:
        di = S.make_decode_inputs(spec, lens, seed=seed, q_std=3.0)
        buf = device.DecodeBuffers(spec, lens).load_host(di)
        dck.check(buf.run(), "dck_decode_attention")
        torch.cuda.synchronize()
        ref = buf.out.clone()
        outs = [torch.full_like(buf.out, float("nan")) for _ in range(3)]
        dck.check(_noalloc(buf, spec, outs[0]), "dck_decode_attention_noalloc (first call on the device)")
        torch.cuda.synchronize()
        free0, _ = torch.cuda.mem_get_info()
        for o in outs[1:]:   # two calls in a row on the same scratch
            dck.check(_noalloc(buf, spec, o), "dck_decode_attention_noalloc")
        torch.cuda.synchronize()
        free1, _ = torch.cuda.mem_get_info()
        assert free1 == free0, f"free device memory changed across the calls: {free0} -> {free1}"
        assert dck.dck_last_device_error() == dck.DCK_OK
        for o in outs:
            assert torch.equal(o.view(torch.int16), ref.view(torch.int16)), "not bit-identical to the regular call"
        got = outs[-1].float().cpu().numpy().astype(np.float64)
        assert_parity(got, oracle_decode(di), spec.dtype, f"noalloc Hkv={spec.n_kv_heads} vs oracle")
        assert TOL[spec.dtype] > 0


def test_noalloc_rejects_requests_beyond_its_scratch():
    # 4096 one-token sequences with r_v = 2048 need about 150 MB of partials
    spec = S.LayerSpec(4096, 32, 32, 128, (tuple(range(32)),), (256,), 2048, "bf16", 1e4)
    lens = (1,) * 4096
    buf = device.DecodeBuffers(spec, lens).synth(seed=1)   # valid buffers of the full request
    assert dck.dck_decode_workspace_size(buf.layer, buf.B, buf.n_rows) > (32 << 20)
    assert _noalloc(buf, spec, buf.out) == dck.DCK_ERR_WORKSPACE
