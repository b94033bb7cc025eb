"""fp64 CPU oracle for DynaCalKV latent-cache decode attention.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package.  The library
(the CUDA kernels behind the C ABI and their Python binding) never imports,
links or calls it, and it shares no code with them: the two meet only in the
seeded input generator ``paper_2607_24331_gb300.synth``, which holds none of
the method's arithmetic.

Contents
* ``decode.py``  - decode attention over grouped low-rank key latents and a
  whole-matrix value latent (Sec. III-A, III-C, III-D), with RoPE applied to
  the reconstructed keys and to the query; plain definition, fp64.
* ``prefill.py`` - causal prefill attention over the same caches: many new
  tokens per sequence, each attending to its prefix (the decode call is one
  new token); plain definition, fp64.
* ``append.py``  - the latent projection z = x L of new tokens (Sec. III-A).
* ``layout.py``  - parameter counts of grouped key factors (Sec. III-C,
  Table I).

Parity status: every function is pinned by ``tests/test_oracle_pins.py`` and
``tests/test_prefill_oracle_pins.py`` (closed forms, library routines,
invariants and brute force); none is "parity unpinned".
"""

from .decode import decode_attention, rope, rope_freqs, kv_head_of  # noqa: F401
from .prefill import prefill_attention  # noqa: F401
from .append import latent_append  # noqa: F401
from .layout import grouped_key_params, recalkv_key_params  # noqa: F401
