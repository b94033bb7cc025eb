"""dck_decode_step through the C ABI: the latent append of the batch's new
tokens (Sec. III-A z = x L) and decode attention over the caches that hold
them, in one call, against the fp64 oracle's latent_append followed by its
decode_attention on the appended caches.

The appended rows are checked element by element with the append bound of
test_append_gpu (fp32 accumulation of stored values, one rounding to the
cache dtype); the decode output with the decode tolerance.  The oracle
rounds its fp64 append to the cache dtype itself, so no expected value comes
from the GPU.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2607_24331_gb300 import dck, device
from paper_2607_24331_gb300 import synth as S
from gpu_util import TOL, assert_parity, oracle_decode

pytestmark = pytest.mark.gpu


def _step(spec, lens, seed, sample_heads=None):
    di = S.make_decode_inputs(spec, lens, seed=seed)
    B = len(lens)
    x, A_k, A_v = S.make_append_inputs(spec, B, seed=seed + 100)
    rows = (di.seq_start + np.asarray(lens) - 1).astype(np.int64)
    # the oracle: append in fp64, rounded to the cache dtype, written into the last rows
    c, v = oracle.latent_append(x, A_k, A_v)
    ref_k, ref_v = di.kcache.copy(), di.vcache.copy()
    ref_k[rows] = S.round_to(c.astype(np.float32), spec.dtype)
    ref_v[rows] = S.round_to(v.astype(np.float32), spec.dtype)
    di_ref = S.DecodeInputs(spec, di.q, ref_k, ref_v, di.B_k, di.B_v, di.seq_start, di.seq_lens)
    # the library: the caches as they were before the step
    buf = device.DecodeBuffers(spec, lens).load_host(di)
    dt = device.TORCH_DTYPE[spec.dtype]
    xd, Akd, Avd = (torch.from_numpy(np.ascontiguousarray(t, dtype=np.float32)).to("cuda", dt) for t in (x, A_k, A_v))
    rd = torch.from_numpy(rows).cuda()
    ws_bytes = dck.dck_decode_step_workspace_size(buf.layer, B, buf.n_rows)
    ws = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    dck.check(dck.dck_decode_step(buf.layer, xd, Akd, Avd, rd, buf.q, buf.kcache, buf.vcache, buf.n_rows, buf.B_k,
                                  buf.B_v, buf.seq_start, buf.seq_len, B, spec.rope_theta, buf.out, ws, ws_bytes),
              "dck_decode_step")
    torch.cuda.synchronize()
    assert dck.dck_last_device_error() == dck.DCK_OK
    launches = dck.dck_last_launch_count()
    # appended rows, per element
    u = 2.0 ** -8 if spec.dtype == "bf16" else 2.0 ** -23
    gk = buf.kcache.float().cpu().numpy().astype(np.float64)
    gv = buf.vcache.float().cpu().numpy().astype(np.float64)
    for got, ref, A in ((gk, c, A_k), (gv, v, A_v)):
        absdot = np.abs(x.astype(np.float64)) @ np.abs(A.astype(np.float64))
        bound = u * np.abs(ref) + spec.hidden * 2.0 ** -23 * absdot
        assert (np.abs(got[rows] - ref) <= bound).all()
    others = np.setdiff1d(np.arange(buf.n_rows), rows)
    assert (gk[others] == di.kcache[others]).all() and (gv[others] == di.vcache[others]).all()
    # decode output against the oracle on the appended caches
    got = buf.out.float().cpu().numpy().astype(np.float64)
    assert np.isfinite(got).all()
    if sample_heads is None:
        assert_parity(got, oracle_decode(di_ref), spec.dtype, f"step {spec.dtype} Hkv={spec.n_kv_heads} {lens}")
    else:
        for b, j in sample_heads:
            ref = oracle_decode(di_ref, heads=[j], batch_ids=[b])
            assert_parity(got[b:b + 1, j:j + 1], ref[b:b + 1, j:j + 1], spec.dtype, f"step b{b} j{j}")
    return launches


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_step_fused_append_then_decode(cfg):
    """Fused path (bf16 tensor-core kernels): the append runs in the call's first launch."""
    n = _step(S.workload(cfg).layer, (300, 1, 129, 1000), seed=40 + cfg)
    assert n == 4, f"expected the four decode kernels with the append fused, got {n} launches"


def test_step_fused_64_sequences():
    spec = S.workload(1).layer
    lens = tuple(int(x) for x in np.random.default_rng(3).integers(1, 400, size=64))
    _step(spec, lens, seed=51)


def test_step_unfused_paths():
    """fp32 layer (CUDA-core kernels) and a batch above the fused limit: append, then decode."""
    assert _step(S.workload(0).layer, (512, 33), seed=60) >= 3
    spec = S.workload(2).layer
    _step(spec, tuple([17] * 65), seed=61)


def test_step_full_size_mha():
    """The 7B MHA workload, B16 x T4096, sampled heads of the first and last sequence."""
    w = S.workload(1)
    _step(w.layer, w.seq_lens, seed=w.seed, sample_heads=[(0, 0), (0, 17), (15, 5), (15, 31)])


def test_timing_hook_brackets():
    """dck_set_timing_events: with kernels + 1 events every kernel is bracketed, in launch order; with
    two, the call is bracketed.  The events are recorded once beforehand (so that they exist), then a
    mark; every event the hooked call records again must come after the mark, in order."""
    w = S.workload(1)
    buf = device.DecodeBuffers(w.layer, (700, 300)).synth(seed=7)
    dck.check(buf.run(), "dck_decode_attention")
    torch.cuda.synchronize()
    kernels = dck.dck_last_launch_count()
    assert kernels == 4
    for n in (kernels + 1, 2):
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
        for e_ in evs:
            e_.record()
        mark, after = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        mark.record()
        dck.check(dck.dck_set_timing_events(evs), "timing events")
        try:
            dck.check(buf.run(), "dck_decode_attention")
        finally:
            dck.check(dck.dck_set_timing_events(None), "timing events")
        after.record()
        torch.cuda.synchronize()
        chain = [mark] + evs + [after]
        gaps = [chain[i].elapsed_time(chain[i + 1]) for i in range(len(chain) - 1)]
        assert all(g >= 0 for g in gaps), (n, gaps)
        assert evs[0].elapsed_time(evs[-1]) > 0
