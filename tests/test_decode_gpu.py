"""Decode attention through the C ABI vs the fp64 oracle, element by element.

Small cases span several 128-token tiles and ragged tails; the benchmark
workloads run at full size with the oracle evaluated on sampled (sequence,
head) pairs.  Tolerance: max|d| / ||o||_inf <= 2e-2 for bf16 latents with fp32
accumulation, <= 1e-5 for the fp32 layer.
"""

import numpy as np
import pytest
import torch

from paper_2607_24331_gb300 import dck, device
from paper_2607_24331_gb300 import synth as S
from gpu_util import TOL, assert_parity, gpu_decode, oracle_decode

pytestmark = pytest.mark.gpu

KERNELS = [0, 1]  # automatic (tensor-core where supported), CUDA-core


@pytest.mark.parametrize("kernel", KERNELS)
def test_tiny_fp32_config_full(kernel):
    w = S.workload(0)
    got, di = gpu_decode(w.layer, w.seq_lens, kernel=kernel)
    assert_parity(got, oracle_decode(di), "f32", "cfg0")


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("cfg", [1, 2, 3])
@pytest.mark.parametrize("lens", [(1, 127, 128, 129, 300, 517), (255, 2, 384)])
def test_ragged_small_bf16(cfg, lens, kernel):
    spec = S.workload(cfg).layer
    got, di = gpu_decode(spec, lens, seed=3, kernel=kernel)
    assert_parity(got, oracle_decode(di), "bf16", f"cfg{cfg} {lens}")


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("cfg", [1, 2])
def test_peaked_scores_bf16(cfg, kernel):
    """q scaled x8: scores ~ N(0, 64), the softmax is dominated by few tokens."""
    spec = S.workload(cfg).layer
    got, di = gpu_decode(spec, (700, 45, 1031), seed=5, q_std=8.0, kernel=kernel)
    assert_parity(got, oracle_decode(di), "bf16", f"cfg{cfg} peaked")


@pytest.mark.parametrize("kernel", KERNELS)
def test_fp32_ragged(kernel):
    spec = S.workload(0).layer
    got, di = gpu_decode(spec, (1, 129, 64, 1000), seed=9, q_std=3.0, kernel=kernel)
    assert_parity(got, oracle_decode(di), "f32", "cfg0 ragged")


@pytest.mark.parametrize("kernel", KERNELS)
def test_long_positions_bf16(kernel):
    """One sequence near 131k tokens: RoPE angles up to 1.3e5 rad."""
    spec = S.workload(3).layer
    got, di = gpu_decode(spec, (131071, 3), seed=2, q_std=4.0, kernel=kernel)
    assert_parity(got, oracle_decode(di), "bf16", "cfg3 long positions")


def test_zero_length_and_invalid_sequences():
    spec = S.workload(2).layer
    lens = (40, 0, 70)
    di = S.make_decode_inputs(spec, (40, 0, 70), seed=1)
    buf = device.DecodeBuffers(spec, lens).load_host(di)
    dck.check(buf.run(), "decode")
    assert dck.dck_last_device_error() == dck.DCK_OK
    out = buf.out.float().cpu().numpy()
    assert (out[1] == 0).all()
    ref = oracle_decode(di, batch_ids=[0, 2])
    assert_parity(out[[0, 2]], ref[[0, 2]], "bf16", "zero-length neighbours")
    # a sequence whose rows run past the cache: reported, treated as empty
    buf.seq_len[2] = 10_000
    dck.check(buf.run(), "decode")
    assert dck.dck_last_device_error() == dck.DCK_ERR_INVALID
    out = buf.out.float().cpu().numpy()
    assert (out[2] == 0).all()
    assert_parity(out[[0]], ref[[0]], "bf16", "valid neighbour")


def test_workspace_and_argument_errors():
    spec = S.workload(1).layer
    buf = device.DecodeBuffers(spec, (16, 16)).synth()
    L = buf.layer
    r = dck.dck_decode_attention(L, buf.q, buf.kcache, buf.vcache, buf.n_rows, buf.B_k, buf.B_v, buf.seq_start,
                                 buf.seq_len, buf.B, 1e4, buf.out, buf.workspace, buf.ws_bytes - 256)
    assert r == dck.DCK_ERR_WORKSPACE
    r = dck.dck_decode_attention(L, buf.q, buf.kcache, buf.vcache, buf.n_rows, buf.B_k, buf.B_v, buf.seq_start,
                                 buf.seq_len, buf.B, -1.0, buf.out, buf.workspace, buf.ws_bytes)
    assert r == dck.DCK_ERR_INVALID
    r = dck.dck_decode_attention(L, None, buf.kcache, buf.vcache, buf.n_rows, buf.B_k, buf.B_v, buf.seq_start,
                                 buf.seq_len, buf.B, 1e4, buf.out, buf.workspace, buf.ws_bytes)
    assert r == dck.DCK_ERR_INVALID
    assert dck.dck_decode_attention(L, buf.q, buf.kcache, buf.vcache, buf.n_rows, buf.B_k, buf.B_v, buf.seq_start,
                                    buf.seq_len, 0, 1e4, buf.out, buf.workspace, buf.ws_bytes) == dck.DCK_OK


def _sample_pairs(B, Hq, n, seed):
    rng = np.random.default_rng(seed)
    pairs = {(0, 0), (B - 1, Hq - 1)}
    while len(pairs) < n:
        pairs.add((int(rng.integers(B)), int(rng.integers(Hq))))
    return sorted(pairs)


@pytest.mark.parametrize("cfg", [1, 2, 3, 5])
def test_full_size_configs_sampled(cfg):
    """Full benchmark workload, inputs from the host generator, sampled oracle outputs."""
    w = S.workload(cfg)
    spec = w.layer
    di = S.make_decode_inputs(spec, w.seq_lens, seed=w.seed)
    got, _ = gpu_decode(spec, w.seq_lens, di=di)
    pairs = _sample_pairs(w.batch, spec.n_q_heads, 12, cfg)
    errs = []
    for b, j in pairs:
        ref = oracle_decode(di, heads=[j], batch_ids=[b])
        errs.append(assert_parity(got[b:b + 1, j:j + 1], ref[b:b + 1, j:j + 1], "bf16", f"cfg{cfg} b{b} j{j}"))
    assert np.isfinite(got).all()


# Layers beyond the benchmark configs that the tensor-core path takes: a head
# count that pads to the MMA width (24 -> 32), two and eight query heads per KV
# head, and ranks whose latent pieces include 32- and 16-column widths.
TC_SHAPES = {
    "mha24_pad": S.LayerSpec(1024, 24, 24, 128, ((0, 1, 2, 3, 4, 5), (6, 7, 8, 9, 10, 11, 12, 13),
                                                  tuple(range(14, 24))), (64, 128, 80), 256, "bf16", 1e4),
    "gqa_qpg2": S.LayerSpec(2048, 16, 8, 128, ((0, 1), (2, 3, 4), (5, 6, 7)), (96, 160, 48), 384, "bf16", 5e5),
    "gqa_qpg8": S.LayerSpec(2048, 32, 4, 128, ((0, 1), (2, 3)), (112, 64), 128, "bf16", 1e6),
}


@pytest.mark.parametrize("name", sorted(TC_SHAPES))
def test_tensor_core_layer_shapes(name):
    spec = TC_SHAPES[name]
    lens = (1, 200, 700, 129)
    got, di = gpu_decode(spec, lens, seed=17, q_std=3.0)
    n = dck.dck_last_launch_count()
    assert n == 4, f"the tensor-core path (factor preparation, scores, absorption, combine) did not run: {n} launches"
    assert_parity(got, oracle_decode(di), "bf16", name)


@pytest.mark.parametrize("cfg", [1, 2])
@pytest.mark.parametrize("extra", [5, -1, 1])
def test_leftover_tiles_split_finely(cfg, extra):
    """More 256-token pair tiles than CTA pairs: whole pair tiles per pair, then the
    leftover pair tiles shared out by groups of heads (scores) and their 128-token
    halves by r_v chunks (absorption), each half with its own partial slot.
    extra = -1: one pair tile short of two per pair; extra = 1 with an odd last
    128-token tile: the leftover pair tile's second half is empty."""
    P = torch.cuda.get_device_properties(0).multi_processor_count // 2
    npt = P + (extra if extra > 0 else P - 1)
    tail = 77 if extra != 1 else 256 + 100
    lens = (32 * 256, (npt - 32 - 2) * 256 + tail)
    spec = S.workload(cfg).layer
    di = S.make_decode_inputs(spec, lens, seed=21 + cfg)
    got, _ = gpu_decode(spec, lens, di=di)
    for b, j in _sample_pairs(2, spec.n_q_heads, 8, cfg + 40):
        ref = oracle_decode(di, heads=[j], batch_ids=[b])
        assert_parity(got[b:b + 1, j:j + 1], ref[b:b + 1, j:j + 1], "bf16", f"cfg{cfg} npt{npt} b{b} j{j}")
    assert np.isfinite(got).all()


@pytest.mark.parametrize("batch", [1, 8, 32, 64])
def test_32_layer_ragged_sampled(batch):
    """32-layer ragged workload: device-generated inputs (checked bit-exact against the host
    generator elsewhere); sampled layers and sequences against the oracle."""
    w = S.workload(4, batch)
    spec = w.layer
    rng = np.random.default_rng(batch)
    for layer in (0, 31, int(rng.integers(1, 31))):
        buf = device.DecodeBuffers(spec, w.seq_lens).synth(seed=w.seed, layer=layer)
        dck.check(buf.run(), "decode")
        torch.cuda.synchronize()
        assert dck.dck_last_device_error() == dck.DCK_OK
        got = buf.out.float().cpu().numpy().astype(np.float64)
        assert np.isfinite(got).all()
        for b in sorted({0, batch - 1, int(rng.integers(batch))}):
            L = w.seq_lens[b]
            row0 = int(S.seq_starts(w.seq_lens)[b])
            di = S.DecodeInputs(
                spec,
                S.gaussian(S.stream_key(w.seed, layer, S.TID["q"]), (batch, spec.n_q_heads, spec.head_dim), 1.0,
                           "bf16")[b:b + 1],
                S.cache_rows(spec, w.seed, layer, "kcache", row0, L),
                S.cache_rows(spec, w.seed, layer, "vcache", row0, L),
                S.make_bk(spec, w.seed, layer), S.make_bv(spec, w.seed, layer),
                np.array([0]), np.array([L]))
            j = int(rng.integers(spec.n_q_heads))
            ref = oracle_decode(di, heads=[j])
            assert_parity(got[b:b + 1, j:j + 1], ref[:, j:j + 1], "bf16", f"L{layer} b{b} j{j}")
