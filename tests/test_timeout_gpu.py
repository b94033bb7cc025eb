"""Failure detection on the GPU without a fault: a bounded wait on a barrier
that nothing arrives at gives up by its own limit, the kernel reports the
timeout through the device error word, and the context keeps working."""

import time

import pytest

from gpu_util import assert_parity, gpu_decode, oracle_decode
from paper_2607_24331_gb300 import dck
from paper_2607_24331_gb300 import synth as S

pytestmark = pytest.mark.gpu


def test_bounded_wait_gives_up_and_the_context_stays_usable():
    assert dck.dck_last_device_error() == dck.DCK_OK  # start from a clear error word
    t0 = time.perf_counter()
    dck.check(dck.dck_selftest_bounded_wait(2_000_000), "dck_selftest_bounded_wait")  # about 1 ms of SM clock
    assert dck.dck_last_device_error() == dck.DCK_ERR_TIMEOUT
    assert time.perf_counter() - t0 < 10.0
    assert dck.dck_last_device_error() == dck.DCK_OK  # reading the word cleared it
    # a regular call on the same context afterwards
    spec = S.workload(1).layer
    got, di = gpu_decode(spec, (129, 7), seed=4)
    assert_parity(got, oracle_decode(di), "bf16", "after the timeout")
