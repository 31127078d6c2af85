"""CPU oracle of the FOVEA retrieve+fuse path (test infrastructure only).

Only tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package; the product path never does.
"""

from .fovea_oracle import (  # noqa: F401
    Memory, Selection, build_memory, fold_keys, fuse, layer_norm, query, query_input, readout,
    lm_head_topk, retrieve_fuse, rms_norm, round_bf16, scores, select, sigmoid, silu,
)
