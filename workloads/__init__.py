"""Seeded synthetic workloads: checkpoint manifests shaped like real models, and blob bytes.

Input infrastructure only.  Both the oracle side and the GPU side consume what this package
produces; it contains none of the loader's arithmetic (no address computation, no cast, no
checksum), only the description of a checkpoint and the bytes it would hold.
"""
from .gen import fill, fill_ptr, splitmix64_word  # noqa: F401
from .manifests import (  # noqa: F401
    DTYPE_SIZE,
    Manifest,
    tiny_config,
    dense_config,
    fp8_block_config,
    moe_config,
    named_config,
    NAMED_CONFIGS,
)
