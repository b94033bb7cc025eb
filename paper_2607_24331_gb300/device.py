"""Device buffers for the C ABI (PyTorch used for memory and streams only).

``DecodeBuffers`` holds one layer's decode inputs, output and workspace in
HBM and calls ``dck_decode_attention`` through the binding; ``AppendBuffers``
does the same for ``dck_latent_append``.  Inputs come either from host arrays
(the seeded generator's values) or from the library's device-side generator
(``dck_synth_gaussian``), which produces the same bits.
"""

from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np
import torch

from . import dck
from . import synth as S

TORCH_DTYPE = {"bf16": torch.bfloat16, "f32": torch.float32}
DCK_DTYPE = {"bf16": dck.DCK_BF16, "f32": dck.DCK_F32}


def upload(a: np.ndarray, dtype: str, device="cuda") -> torch.Tensor:
    """Host fp32 array holding storage-dtype values -> device tensor (exact)."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(device=device, dtype=TORCH_DTYPE[dtype])


def synth_fill(t: torch.Tensor, key: int, std: float, start: int = 0, stream=None) -> None:
    """Fill a device tensor with stream ``key`` of the seeded Gaussian generator."""
    dtype = dck.DCK_F32 if t.dtype == torch.float32 else dck.DCK_BF16
    scale = float(S.gauss_scale(std))
    dck.check(dck.dck_synth_gaussian(t, t.numel(), key, start, scale, dtype, stream), "dck_synth_gaussian")


class DecodeBuffers:
    """One layer's decode call: inputs resident in HBM, output and workspace."""

    def __init__(self, spec: S.LayerSpec, seq_lens: Sequence[int], device="cuda"):
        self.spec = spec
        self.layer = dck.Layer.from_spec(spec)
        self.lens_host = np.asarray(seq_lens, dtype=np.int64)
        self.B = len(self.lens_host)
        self.n_rows = int(self.lens_host.sum())
        self.device = device
        dt = TORCH_DTYPE[spec.dtype]
        self.seq_start = torch.from_numpy(S.seq_starts(self.lens_host)).to(device)
        self.seq_len = torch.from_numpy(self.lens_host.astype(np.int32)).to(device)
        self.out = torch.empty((self.B, spec.n_q_heads, spec.head_dim), dtype=dt, device=device)
        self.ws_bytes = dck.dck_decode_workspace_size(self.layer, self.B, self.n_rows)
        self.workspace = torch.empty(max(self.ws_bytes, 256), dtype=torch.uint8, device=device)
        self.q = self.kcache = self.vcache = self.B_k = self.B_v = None

    def load_host(self, di: S.DecodeInputs) -> "DecodeBuffers":
        d = self.spec.dtype
        self.q = upload(di.q, d, self.device)
        self.kcache = upload(di.kcache, d, self.device)
        self.vcache = upload(di.vcache, d, self.device)
        self.B_k = upload(di.B_k, d, self.device)
        self.B_v = upload(di.B_v, d, self.device)
        return self

    def synth(self, seed: int = 0, layer: int = 0, q_std: float = 1.0) -> "DecodeBuffers":
        """Device-side generation of the same tensors as synth.make_decode_inputs."""
        spec, dt, dev = self.spec, TORCH_DTYPE[self.spec.dtype], self.device
        self.q = torch.empty((self.B, spec.n_q_heads, spec.head_dim), dtype=dt, device=dev)
        self.kcache = torch.empty((self.n_rows, spec.rank_k), dtype=dt, device=dev)
        self.vcache = torch.empty((self.n_rows, spec.rank_v), dtype=dt, device=dev)
        off = spec.bk_offsets()
        self.B_k = torch.empty((off[-1],), dtype=dt, device=dev)
        self.B_v = torch.empty((spec.rank_v, spec.n_kv_heads * spec.head_dim), dtype=dt, device=dev)
        synth_fill(self.q, S.stream_key(seed, layer, S.TID["q"]), q_std)
        synth_fill(self.kcache, S.stream_key(seed, layer, S.TID["kcache"]), 1.0)
        synth_fill(self.vcache, S.stream_key(seed, layer, S.TID["vcache"]), 1.0)
        kb = S.stream_key(seed, layer, S.TID["B_k"])
        for g, r in enumerate(spec.ranks):
            synth_fill(self.B_k[off[g]:off[g + 1]], kb, 1.0 / math.sqrt(r), start=off[g])
        synth_fill(self.B_v, S.stream_key(seed, layer, S.TID["B_v"]), 1.0 / math.sqrt(spec.rank_v))
        return self

    def run(self, stream=None, out: Optional[torch.Tensor] = None) -> int:
        return dck.dck_decode_attention(self.layer, self.q, self.kcache, self.vcache, self.n_rows, self.B_k,
                                        self.B_v, self.seq_start, self.seq_len, self.B, self.spec.rope_theta,
                                        self.out if out is None else out, self.workspace, self.ws_bytes, stream)

    def algorithmic_bytes(self) -> int:
        """Latent rows read once, both factors once, q and out once."""
        s = self.spec
        el = 2 if s.dtype == "bf16" else 4
        fac = s.bk_offsets()[-1] + s.rank_v * s.n_kv_heads * s.head_dim
        return el * (self.n_rows * (s.rank_k + s.rank_v) + fac + 2 * self.B * s.n_q_heads * s.head_dim)

    def tensor_flops(self) -> int:
        """Key reconstruction plus value absorption on the tensor pipe."""
        s = self.spec
        per_tok = 2 * sum(r * len(g) for g, r in zip(s.groups, s.ranks)) * s.head_dim + 2 * s.n_q_heads * s.rank_v
        return self.n_rows * per_tok


class AppendBuffers:
    """Latent append of n_tok tokens into caches of n_rows rows."""

    def __init__(self, spec: S.LayerSpec, n_tok: int, n_rows: int, device="cuda"):
        self.spec = spec
        self.layer = dck.Layer.from_spec(spec)
        self.n_tok = n_tok
        self.n_rows = n_rows
        dt = TORCH_DTYPE[spec.dtype]
        self.kcache = torch.zeros((n_rows, spec.rank_k), dtype=dt, device=device)
        self.vcache = torch.zeros((n_rows, spec.rank_v), dtype=dt, device=device)
        self.ws_bytes = dck.dck_latent_append_workspace_size(self.layer, n_tok)
        self.workspace = torch.empty(max(self.ws_bytes, 256), dtype=torch.uint8, device=device)
        self.x = self.A_k = self.A_v = self.rows = None
        self.device = device

    def load_host(self, x, A_k, A_v, rows) -> "AppendBuffers":
        d = self.spec.dtype
        self.x = upload(x, d, self.device)
        self.A_k = upload(A_k, d, self.device)
        self.A_v = upload(A_v, d, self.device)
        self.rows = torch.as_tensor(np.asarray(rows, dtype=np.int64)).to(self.device)
        return self

    def run(self, stream=None) -> int:
        return dck.dck_latent_append(self.layer, self.x, self.n_tok, self.A_k, self.A_v, self.rows, self.kcache,
                                     self.vcache, self.n_rows, self.workspace, self.ws_bytes, stream)

    def flops(self) -> int:
        return 2 * self.n_tok * self.spec.hidden * (self.spec.rank_k + self.spec.rank_v)
