"""fp64 CPU oracle for prefix-cached paged attention.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``, never by the library.  It shares no
code with the CUDA path (see ``pkv_oracle.c`` for the definitions it follows).
"""

from .oracle import (  # noqa: F401
    attention,
    bf16_to_f64,
    build,
    cache_write,
    gather,
    paged_request_attention,
    request_attention,
    slot_mapping,
)
