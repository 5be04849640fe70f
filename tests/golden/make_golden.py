"""Write tests/golden/oracle_small.json from the CPU oracle alone.

Run from the repository root:  python tests/golden/make_golden.py

The file stores, for a small fixed input, the oracle's salts, its chain
digests in all three salt placements and its prefix lengths against a table
holding the first requests' ROOT chains.  The CPU suite checks that the
oracle still reproduces it; the GPU suite checks the CUDA path against it.
"""
import json
import os
import sys

import numpy as np

ROOT_DIR = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT_DIR)

import oracle  # noqa: E402
from paper_2608_09225_gb300 import workloads as W  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_small.json")

# Ragged request lengths (tokens) covering empty, sub-block, exact, tail, and
# a boundary offset cycle of 0, 15, 16, 17, 31, 32, 64 and "past the end".
LENGTHS = [0, 15, 16, 17, 31, 32, 33, 64, 100, 129, 256, 7]
SEED = 20260
SECRET = bytes(range(100, 132))
N_PRINCIPALS = 8
N_FILL = 6


def compute():
    b = W.ragged(SEED, LENGTHS)
    ids, id_off = W.principal_ids(N_PRINCIPALS)
    salts = oracle.derive_salts(SECRET, ids, id_off)
    blk = oracle.block_offsets(b.tok_off)
    out = {"seed": SEED, "lengths": LENGTHS, "secret_hex": SECRET.hex(), "n_principals": N_PRINCIPALS,
           "n_fill": N_FILL, "salts": [s.tobytes().hex() for s in salts], "blk_off": blk.tolist()}
    for name, mode in (("unsalted", oracle.UNSALTED), ("root", oracle.ROOT), ("boundary", oracle.BOUNDARY)):
        d = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
        out["digests_" + name] = [row.tobytes().hex() for row in d]
    root = oracle.chain_hash(oracle.ROOT, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    ks = oracle.KeySet(1)
    ks.insert(root[: blk[N_FILL]])
    # probe a second copy of the batch with principal 0 everywhere: only the
    # filled requests whose principal is 0 hit
    b0 = np.zeros_like(b.principal)
    q = oracle.chain_hash(oracle.ROOT, b.tokens, b.tok_off, b0, salts, b.boundary_tok)
    out["prefix_root_self"] = ks.prefix_blocks(root, blk).tolist()
    out["prefix_root_principal0"] = ks.prefix_blocks(q, blk).tolist()
    return out


if __name__ == "__main__":
    with open(OUT, "w") as f:
        json.dump(compute(), f, indent=1)
    print("wrote", OUT)
