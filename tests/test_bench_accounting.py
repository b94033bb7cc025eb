"""The roofline numerators bench.py reports, pinned on CPU against sums
written out by hand for the 7B MHA workload (32 heads of 128, groups of
{2,3,3,4,4,5,5,6} KV heads at ranks {64,96,96,128,128,160,160,192}, r_v =
1024, B16 x T4096, bf16), so that a slip in the byte or flop accounting (a
factor counted per sequence, a missing query, fp32 element size) fails here,
not silently in the reported fraction."""

import types

import pytest

import bench
from paper_2607_24331_gb300 import device
from paper_2607_24331_gb300 import synth as S

ROWS = 16 * 4096          # cache rows read by one call
EL = 2                    # bf16
SUM_RN = 2 * 64 + 3 * 96 + 3 * 96 + 4 * 128 + 4 * 128 + 5 * 160 + 5 * 160 + 6 * 192   # sum_g r_g n_g = 4480
B_K = SUM_RN * 128 * EL   # every B_g once: 1,146,880 bytes
B_V = 1024 * 32 * 128 * EL  # B_v once: 8,388,608 bytes
QO = 16 * 32 * 128 * EL   # q in, out out: 131,072 bytes each


def _buf():
    w = S.workload(1)
    assert w.batch == 16 and set(w.seq_lens) == {4096}
    return types.SimpleNamespace(spec=w.layer, n_rows=sum(w.seq_lens), B=w.batch)


def test_hand_sums():
    assert SUM_RN == 4480 and B_K == 1_146_880 and B_V == 8_388_608 and QO == 131_072


def test_call_bytes_and_flops():
    buf = _buf()
    assert device.DecodeBuffers.algorithmic_bytes(buf) == ROWS * (1024 + 1024) * EL + B_K + B_V + 2 * QO == 278_233_088
    # key reconstruction 2 r_g d per head and token, value absorption 2 r_v per query head and token
    assert device.DecodeBuffers.tensor_flops(buf) == ROWS * (2 * SUM_RN * 128 + 2 * 32 * 1024) == 79_456_894_976


@pytest.mark.parametrize("name,bytes_,flops", [
    ("scores", ROWS * 1024 * EL + B_K + QO, ROWS * 2 * SUM_RN * 128),
    ("absorb", ROWS * 1024 * EL, ROWS * 2 * 32 * 1024),
    ("combine", B_V + QO, 0),
    # the step's append: [A_k | A_v] once and the 16 tokens' x and latents; B_g and q for the factor images
    ("factor_prep+append", B_K + QO + 4096 * 2048 * EL + 16 * (4096 + 2048) * EL, 2 * 16 * 4096 * 2048),
])
def test_per_kernel_work(name, bytes_, flops):
    assert bench.kernel_work(_buf(), name) == (bytes_, flops)


def test_step_bytes_are_the_call_plus_the_append():
    """The bench line's numerator: 295,206,912 bytes per decode-step call of this workload."""
    buf = _buf()
    app = 4096 * 2048 * EL + 16 * (4096 + 2048) * EL
    assert device.DecodeBuffers.algorithmic_bytes(buf) + app == 295_206_912
