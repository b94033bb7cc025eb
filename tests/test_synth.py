"""The seeded input generator: determinism, random access, rounding, shapes."""

import math

import numpy as np

from paper_2607_24331_gb300 import synth as S


def _draw_py(key, i):
    return S.mix64_int(key + (i + 1) * S.GAMMA)


def test_splitmix64_reference_values():
    # SplitMix64 with state 0: the first outputs of Vigna's reference generator
    assert _draw_py(0, 0) == 0xE220A8397B1DCDAF
    assert _draw_py(0, 1) == 0x6E789E6AA1B965F4
    assert _draw_py(0, 2) == 0x06C45D188009454F
    d = S.draws(0, 0, 3)
    assert [int(v) for v in d] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_gaussian_definition_and_random_access():
    key = S.stream_key(7, 3, S.TID["kcache"])
    g = S.gaussian_f32(key, 0, 4096 + 17, 1.0)
    for i in (0, 1, 99, 4096 + 16):
        a, b = _draw_py(key, 2 * i), _draw_py(key, 2 * i + 1)
        s = sum((a >> sh) & 0xFFFF for sh in (0, 16, 32, 48)) + sum((b >> sh) & 0xFFFF for sh in (0, 16, 32, 48))
        assert np.float32(2 * s - 8 * 65535) * S.gauss_scale(1.0) == g[i]
    np.testing.assert_array_equal(S.gaussian_f32(key, 1000, 3000, 1.0), g[1000:4000])
    big = S.gaussian_f32(key, 0, 1 << 21, 2.0)
    assert abs(big.mean()) < 0.01 and abs(big.std() - 2.0) < 0.01


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -8 + 2 ** -20, -2.5, 0.0, 3e38],
                 dtype=np.float32)
    r = S.round_to(x, "bf16")
    assert r[0] == 1.0
    assert r[1] == 1.0                     # tie -> even
    assert r[2] == 1.0 + 4 * 2 ** -8       # tie -> even (up)
    assert r[3] == 1.0 + 2 * 2 ** -8       # above the tie -> up
    assert r[4] == -2.5 and r[5] == 0.0
    assert np.isfinite(r[6]) or r[6] == np.inf
    # round trip of representable values
    b = S.f32_to_bf16_bits(r[:6])
    np.testing.assert_array_equal(S.bf16_bits_to_f32(b), r[:6])


def test_workload_shapes():
    for cfg in range(5):
        w = S.workload(cfg)
        w.layer.validate()
    w1 = S.workload(1)
    assert sorted(len(g) for g in w1.layer.groups) == [2, 3, 3, 4, 4, 5, 5, 6]
    assert w1.layer.rank_k == 1024 and w1.layer.rank_v == 1024
    assert S.workload(2).layer.rank_k == 768
    assert S.workload(3).layer.rank_k == 704
    lens = S.ragged_lens(0, 64)
    assert len(lens) == 64 and min(lens) >= 1024 and max(lens) <= 16384
    assert S.ragged_lens(0, 64) == lens


def test_decode_inputs_layout():
    spec = S.tiny_mha_layer()
    di = S.make_decode_inputs(spec, [5, 3], seed=0)
    assert di.kcache.shape == (8, 144) and di.vcache.shape == (8, 160)
    assert di.B_k.shape == (48 * 3 * 64 + 96 * 5 * 64,)
    assert list(di.seq_start) == [0, 5]
    rows = S.cache_rows(spec, 0, 0, "kcache", 5, 3)
    np.testing.assert_array_equal(rows, di.kcache[5:8])
    # factor scale: B_g ~ N(0, 1/r_g)
    assert abs(di.B_k[:48 * 192].std() - 1 / math.sqrt(48)) < 0.02
