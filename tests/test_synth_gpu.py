"""The device-side generator gives the host generator's bits."""

import numpy as np
import pytest
import torch

from paper_2607_24331_gb300 import device
from paper_2607_24331_gb300 import synth as S

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_device_generator_bit_exact(dtype):
    key = S.stream_key(3, 7, S.TID["kcache"])
    n, start = 1_000_003, 12345
    t = torch.empty(n, dtype=device.TORCH_DTYPE[dtype], device="cuda")
    device.synth_fill(t, key, 0.37, start=start)
    host = S.round_to(S.gaussian_f32(key, start, n, 0.37), dtype)
    np.testing.assert_array_equal(t.float().cpu().numpy(), host)


def test_decode_buffers_synth_matches_host_inputs():
    spec = S.workload(1).layer
    lens = (300, 77)
    buf = device.DecodeBuffers(spec, lens).synth(seed=4, layer=2)
    di = S.make_decode_inputs(spec, lens, seed=4, layer=2)
    for name in ("q", "kcache", "vcache", "B_k", "B_v"):
        np.testing.assert_array_equal(getattr(buf, name).float().cpu().numpy(), getattr(di, name), err_msg=name)
