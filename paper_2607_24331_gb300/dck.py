"""Python binding of libdck (ctypes): argument marshalling only.

Every function here has the name of the C entry point it calls and passes
raw device pointers (taken from torch tensors) and the current CUDA stream.
No step of the computation runs in Python: if ``libdck.so`` is missing the
import of this module's entry points raises.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libdck.so")

DCK_OK = 0
DCK_ERR_INVALID = -1
DCK_ERR_UNSUPPORTED = -2
DCK_ERR_WORKSPACE = -3
DCK_ERR_CUDA = -4
DCK_ERR_TIMEOUT = -5
DCK_BF16 = 0
DCK_F32 = 1

EXPORTED = (
    "dck_status_string", "dck_validate_desc", "dck_latent_append_workspace_size", "dck_latent_append",
    "dck_decode_workspace_size", "dck_decode_attention", "dck_last_device_error", "dck_set_decode_kernel",
    "dck_last_launch_count", "dck_synth_gaussian", "dck_set_timing_events", "dck_decode_attention_noalloc",
    "dck_selftest_bounded_wait", "dck_decode_step", "dck_decode_step_workspace_size",
    "dck_prefill_workspace_size", "dck_prefill_attention",
)


class DckError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} ({status})")


class LayerDesc(ctypes.Structure):
    _fields_ = [
        ("hidden", ctypes.c_int32),
        ("n_q_heads", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("n_groups", ctypes.c_int32),
        ("group_offsets", ctypes.POINTER(ctypes.c_int32)),
        ("group_heads", ctypes.POINTER(ctypes.c_int32)),
        ("ranks", ctypes.POINTER(ctypes.c_int32)),
        ("rank_v", ctypes.c_int32),
        ("dtype", ctypes.c_int32),
    ]


_lib: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    """The loaded libdck.so; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"libdck.so is not built ({LIB_PATH}); run __graft_entry__.build()")
    L = ctypes.CDLL(LIB_PATH)
    P, I32, I64, U64, F32, SZ = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64,
                                 ctypes.c_float, ctypes.c_size_t)
    D = ctypes.POINTER(LayerDesc)
    L.dck_status_string.restype = ctypes.c_char_p
    L.dck_status_string.argtypes = [I32]
    L.dck_validate_desc.restype = I32
    L.dck_validate_desc.argtypes = [D]
    L.dck_latent_append_workspace_size.restype = SZ
    L.dck_latent_append_workspace_size.argtypes = [D, I32]
    L.dck_latent_append.restype = I32
    L.dck_latent_append.argtypes = [D, P, I32, P, P, P, P, P, I64, P, SZ, P]
    L.dck_decode_workspace_size.restype = SZ
    L.dck_decode_workspace_size.argtypes = [D, I32, I64]
    L.dck_decode_attention.restype = I32
    L.dck_decode_attention.argtypes = [D, P, P, P, I64, P, P, P, P, I32, F32, P, P, SZ, P]
    L.dck_prefill_workspace_size.restype = SZ
    L.dck_prefill_workspace_size.argtypes = [D, I64]
    L.dck_prefill_attention.restype = I32
    L.dck_prefill_attention.argtypes = [D, P, P, I32, P, P, I64, P, P, P, P, I32, I32, F32, P, P, SZ, P]
    L.dck_decode_step_workspace_size.restype = SZ
    L.dck_decode_step_workspace_size.argtypes = [D, I32, I64]
    L.dck_decode_step.restype = I32
    L.dck_decode_step.argtypes = [D, P, P, P, P, P, P, P, I64, P, P, P, P, I32, F32, P, P, SZ, P]
    L.dck_decode_attention_noalloc.restype = I32
    L.dck_decode_attention_noalloc.argtypes = [D, P, P, P, I64, P, P, P, P, I32, F32, P, P]
    L.dck_last_device_error.restype = I32
    L.dck_last_device_error.argtypes = [P]
    L.dck_set_decode_kernel.restype = I32
    L.dck_set_decode_kernel.argtypes = [I32]
    L.dck_last_launch_count.restype = I32
    L.dck_last_launch_count.argtypes = []
    L.dck_set_timing_events.restype = I32
    L.dck_set_timing_events.argtypes = [P, I32]
    L.dck_selftest_bounded_wait.restype = I32
    L.dck_selftest_bounded_wait.argtypes = [I64, P]
    L.dck_synth_gaussian.restype = I32
    L.dck_synth_gaussian.argtypes = [P, I64, U64, I64, F32, I32, P]
    _lib = L
    return L


def status_string(status: int) -> str:
    return lib().dck_status_string(int(status)).decode()


class Layer:
    """A dck_layer_desc and the host arrays it points to (kept alive here)."""

    def __init__(self, hidden: int, n_q_heads: int, n_kv_heads: int, head_dim: int,
                 groups: Sequence[Sequence[int]], ranks: Sequence[int], rank_v: int, dtype: str):
        self.groups = [list(g) for g in groups]
        offs = [0]
        for g in self.groups:
            offs.append(offs[-1] + len(g))
        heads = [h for g in self.groups for h in g]
        self._offs = (ctypes.c_int32 * len(offs))(*offs)
        self._heads = (ctypes.c_int32 * max(1, len(heads)))(*heads)
        self._ranks = (ctypes.c_int32 * max(1, len(ranks)))(*ranks)
        self.dtype = dtype
        self.desc = LayerDesc(hidden, n_q_heads, n_kv_heads, head_dim, len(self.groups),
                              ctypes.cast(self._offs, ctypes.POINTER(ctypes.c_int32)),
                              ctypes.cast(self._heads, ctypes.POINTER(ctypes.c_int32)),
                              ctypes.cast(self._ranks, ctypes.POINTER(ctypes.c_int32)),
                              rank_v, DCK_F32 if dtype == "f32" else DCK_BF16)

    @classmethod
    def from_spec(cls, spec) -> "Layer":
        return cls(spec.hidden, spec.n_q_heads, spec.n_kv_heads, spec.head_dim, spec.groups,
                   spec.ranks, spec.rank_v, spec.dtype)

    @property
    def ref(self):
        return ctypes.byref(self.desc)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def dck_validate_desc(layer: Layer) -> int:
    return lib().dck_validate_desc(layer.ref)


def dck_decode_workspace_size(layer: Layer, batch: int, n_rows: int) -> int:
    return lib().dck_decode_workspace_size(layer.ref, batch, n_rows)


def dck_latent_append_workspace_size(layer: Layer, n_tok: int) -> int:
    return lib().dck_latent_append_workspace_size(layer.ref, n_tok)


def dck_decode_attention(layer: Layer, q, kcache, vcache, n_rows: int, B_k, B_v, seq_start, seq_len,
                         batch: int, rope_theta: float, out, workspace, ws_bytes: int, stream=None) -> int:
    return lib().dck_decode_attention(layer.ref, _ptr(q), _ptr(kcache), _ptr(vcache), int(n_rows), _ptr(B_k),
                                      _ptr(B_v), _ptr(seq_start), _ptr(seq_len), int(batch), float(rope_theta),
                                      _ptr(out), _ptr(workspace), int(ws_bytes), _stream(stream))


def dck_decode_step_workspace_size(layer: Layer, batch: int, n_rows: int) -> int:
    return lib().dck_decode_step_workspace_size(layer.ref, batch, n_rows)


def dck_decode_step(layer: Layer, x, A_k, A_v, rows, q, kcache, vcache, n_rows: int, B_k, B_v, seq_start, seq_len,
                    batch: int, rope_theta: float, out, workspace, ws_bytes: int, stream=None) -> int:
    """Latent append of the batch's new tokens, then decode attention (one call)."""
    return lib().dck_decode_step(layer.ref, _ptr(x), _ptr(A_k), _ptr(A_v), _ptr(rows), _ptr(q), _ptr(kcache),
                                 _ptr(vcache), int(n_rows), _ptr(B_k), _ptr(B_v), _ptr(seq_start), _ptr(seq_len),
                                 int(batch), float(rope_theta), _ptr(out), _ptr(workspace), int(ws_bytes),
                                 _stream(stream))


def dck_prefill_workspace_size(layer: Layer, n_rows: int) -> int:
    return lib().dck_prefill_workspace_size(layer.ref, int(n_rows))


def dck_prefill_attention(layer: Layer, q, q_len, q_max: int, kcache, vcache, n_rows: int, B_k, B_v, seq_start,
                          seq_len, batch: int, max_seq_len: int, rope_theta: float, out, workspace, ws_bytes: int,
                          stream=None) -> int:
    return lib().dck_prefill_attention(layer.ref, _ptr(q), _ptr(q_len), int(q_max), _ptr(kcache), _ptr(vcache),
                                       int(n_rows), _ptr(B_k), _ptr(B_v), _ptr(seq_start), _ptr(seq_len), int(batch),
                                       int(max_seq_len), float(rope_theta), _ptr(out), _ptr(workspace),
                                       int(ws_bytes), _stream(stream))


def dck_decode_attention_noalloc(layer: Layer, q, kcache, vcache, n_rows: int, B_k, B_v, seq_start, seq_len,
                                 batch: int, rope_theta: float, out, stream=None) -> int:
    """dck_decode_attention without a workspace argument (library-owned fixed scratch)."""
    return lib().dck_decode_attention_noalloc(layer.ref, _ptr(q), _ptr(kcache), _ptr(vcache), int(n_rows),
                                              _ptr(B_k), _ptr(B_v), _ptr(seq_start), _ptr(seq_len), int(batch),
                                              float(rope_theta), _ptr(out), _stream(stream))


def dck_latent_append(layer: Layer, x, n_tok: int, A_k, A_v, rows, kcache, vcache, n_rows: int,
                      workspace, ws_bytes: int, stream=None) -> int:
    return lib().dck_latent_append(layer.ref, _ptr(x), int(n_tok), _ptr(A_k), _ptr(A_v), _ptr(rows), _ptr(kcache),
                                   _ptr(vcache), int(n_rows), _ptr(workspace), int(ws_bytes), _stream(stream))


def dck_last_device_error(stream=None) -> int:
    return lib().dck_last_device_error(_stream(stream))


def dck_set_decode_kernel(which: int) -> int:
    return lib().dck_set_decode_kernel(int(which))


def dck_last_launch_count() -> int:
    return lib().dck_last_launch_count()


def dck_synth_gaussian(dst, n: int, key: int, start: int, scale: float, dtype: int, stream=None) -> int:
    return lib().dck_synth_gaussian(_ptr(dst), int(n), int(key) & ((1 << 64) - 1), int(start), float(scale),
                                    int(dtype), _stream(stream))


def dck_set_timing_events(events) -> int:
    """``events``: torch.cuda.Event objects (already recorded once, so that the CUDA
    events exist), or None / [] to switch this thread's hook off."""
    if not events:
        return lib().dck_set_timing_events(None, 0)
    arr = (ctypes.c_void_p * len(events))(*[e.cuda_event for e in events])
    return lib().dck_set_timing_events(arr, len(events))


def dck_selftest_bounded_wait(limit_cycles: int, stream=None) -> int:
    """One kernel whose bounded wait on a barrier nothing arrives at gives up after
    ``limit_cycles`` SM cycles; the timeout shows in the next dck_last_device_error."""
    return lib().dck_selftest_bounded_wait(int(limit_cycles), _stream(stream))


def check(status: int, what: str) -> None:
    if status != DCK_OK:
        raise DckError(status, what)
