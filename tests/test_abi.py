"""The C ABI library loads, exports every declared entry point, and rejects
malformed descriptors on the host (no GPU needed: nothing is launched)."""

import ctypes
import os
import re

import pytest

from paper_2607_24331_gb300 import dck
from paper_2607_24331_gb300 import synth as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", fn)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names += re.findall(r"\b(dck_[a-z0-9_]+)\s*\(", txt)
    return sorted(set(names))


def test_library_exports_every_declared_symbol():
    L = dck.lib()
    names = declared_functions()
    assert "dck_decode_attention" in names and "dck_latent_append" in names
    for n in names:
        assert hasattr(L, n), n
    assert set(names) <= set(dck.EXPORTED)


def test_status_strings():
    for s in (0, -1, -2, -3, -4, -5):
        assert dck.status_string(s)
    assert dck.status_string(-99) == "unknown status"


def _layer(**kw):
    spec = dict(hidden=4096, n_q_heads=32, n_kv_heads=8, head_dim=128, groups=[[0, 1], [2, 3, 4], [5, 6, 7]],
                ranks=[192, 256, 256], rank_v=384, dtype="bf16")
    spec.update(kw)
    return dck.Layer(**spec)


def test_valid_descriptors():
    for cfg in range(5):
        assert dck.dck_validate_desc(dck.Layer.from_spec(S.workload(cfg).layer)) == dck.DCK_OK


@pytest.mark.parametrize("kw,expect", [
    (dict(n_q_heads=30), dck.DCK_ERR_INVALID),                         # Hq not a multiple of Hkv
    (dict(groups=[[0, 1], [2, 3, 4], [5, 6, 6]]), dck.DCK_ERR_INVALID),  # not a permutation
    (dict(groups=[[0, 1], [2, 3, 4], [5, 6]], ranks=[192, 256, 256]), dck.DCK_ERR_INVALID),
    (dict(ranks=[192, 250, 256]), dck.DCK_ERR_UNSUPPORTED),           # rank not a multiple of 16
    (dict(ranks=[192, 0, 256]), dck.DCK_ERR_INVALID),
    (dict(rank_v=100), dck.DCK_ERR_UNSUPPORTED),
    (dict(head_dim=96), dck.DCK_ERR_UNSUPPORTED),
    (dict(head_dim=0), dck.DCK_ERR_INVALID),
    (dict(hidden=0), dck.DCK_ERR_INVALID),
    (dict(n_q_heads=128), dck.DCK_ERR_UNSUPPORTED),                    # 16 query heads per KV head
])
def test_malformed_descriptors(kw, expect):
    assert dck.dck_validate_desc(_layer(**kw)) == expect


def test_null_descriptor():
    assert dck.lib().dck_validate_desc(None) == dck.DCK_ERR_INVALID


def test_selftest_rejects_limits_out_of_range_without_launching():
    # checked on the host before any CUDA call (stream handle 0 is never used)
    assert dck.dck_selftest_bounded_wait(10, 0) == dck.DCK_ERR_INVALID
    assert dck.dck_selftest_bounded_wait(5_000_000_000, 0) == dck.DCK_ERR_INVALID


def test_decode_entry_points_check_arguments_before_any_cuda_call():
    """Both decode entry points run the same host-side checks, in the same
    order, before touching the device: nothing here needs a GPU (stream 0 and
    fake aligned addresses are never used)."""
    L = dck.Layer.from_spec(S.workload(1).layer)
    p = 1 << 20   # aligned, never dereferenced
    lib = dck.lib()
    args = dict(q=p, kc=p, vc=p, n_rows=100, bk=p, bv=p, st=p, ln=p, batch=2, theta=1e4, out=p)

    def both(**kw):
        a = dict(args, **kw)
        r1 = lib.dck_decode_attention(L.ref, a["q"], a["kc"], a["vc"], a["n_rows"], a["bk"], a["bv"], a["st"],
                                      a["ln"], a["batch"], a["theta"], a["out"], p, 1 << 30, 0)
        r2 = lib.dck_decode_attention_noalloc(L.ref, a["q"], a["kc"], a["vc"], a["n_rows"], a["bk"], a["bv"],
                                              a["st"], a["ln"], a["batch"], a["theta"], a["out"], 0)
        return r1, r2

    assert both(n_rows=-1) == (dck.DCK_ERR_INVALID,) * 2
    assert both(q=None) == (dck.DCK_ERR_INVALID,) * 2
    assert both(theta=-1.0) == (dck.DCK_ERR_INVALID,) * 2
    assert both(batch=-3) == (dck.DCK_ERR_INVALID,) * 2
    assert both(batch=5000) == (dck.DCK_ERR_INVALID,) * 2       # beyond the batch limit
    assert both(q=p + 1) == (dck.DCK_ERR_INVALID,) * 2          # misaligned bf16 pointer
    assert both(batch=0) == (dck.DCK_OK,) * 2                   # nothing to do, nothing launched


def test_timing_hook_arguments():
    lib = dck.lib()
    assert lib.dck_set_timing_events(None, 0) == dck.DCK_OK
    assert lib.dck_set_timing_events(None, 2) == dck.DCK_ERR_INVALID
    import ctypes
    one = (ctypes.c_void_p * 1)(1)
    assert lib.dck_set_timing_events(one, 1) == dck.DCK_ERR_INVALID
    nulls = (ctypes.c_void_p * 2)(None, None)
    assert lib.dck_set_timing_events(nulls, 2) == dck.DCK_ERR_INVALID
