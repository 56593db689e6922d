"""fp64 CPU oracle (test infrastructure only; never used by the product path).

Only the test suite, the smoke check and the benchmark's CPU-baseline and
reference arms may import this package.
"""

from .crc_oracle import (  # noqa: F401
    attention,
    bias_matrix,
    chunk_pose,
    correspond,
    current_key_frames,
    fill_slots,
    gather,
    key_table,
    reproject,
    rope_frequencies,
    rope_reposition,
    retrieval_terms,
    retrieve,
)
