"""fp64 CPU oracle for fork-decode attention over a shared reasoning prefix.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import, call or
link anything under ``oracle/``; only the test suite, the package smoke check
and the benchmark's CPU-baseline leg use it.  It shares no code with the CUDA
path: it computes the plain definition of softmax attention in float64 from
the bf16 bit patterns the GPU path also reads, and the plain row copies of a
decode step's append into paged suffixes (``paging.py``).

Every function here is pinned by ``tests/test_oracle_pins.py`` (closed forms,
brute force, library cross-checks and invariants); no function carries the
"parity unpinned" mark.
"""

from .attention import (  # noqa: F401
    NEG_INF,
    bf16_bits_to_f64,
    gather_logical,
    attention_rows,
    lse_merge,
    fork_attn_decode,
    fork_attn_decode_rows,
    fork_attn_split_merge,
    fork_prefill,
    fork_cascade_decode,
)
from .paging import append_kv, pack_pages, unpack_pages  # noqa: F401
