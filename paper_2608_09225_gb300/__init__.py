"""KVGov salted block-hash chain and block prefix-cache probe on GB300 (sm_103a).

The compute path is the CUDA library libkvgov.so (C ABI in include/kvgov.h);
``paper_2608_09225_gb300.kvgov`` is its ctypes binding.  ``workloads`` holds the
seeded synthetic input generators.  Importing the package loads nothing; the
first binding call loads the library and raises if it or a GPU is missing.
"""
from .kvgov import (BLOCK, BOUNDARY, DIGEST_BYTES, ROOT, UNSALTED, KVGovError, block_offsets,  # noqa: F401
                    chain_hash, chain_hash_arrival, chain_hash_probe, derive_salts, divergence_boundary, insert, insert_arrival, insert_uncached, new_owner,
                    new_table, origami, owner_init, probe, probe_arrival, response_key, set_spin_limit, status_string, table_init)
