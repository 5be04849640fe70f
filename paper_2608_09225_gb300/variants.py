"""Build-time variants of libkvgov's chain kernel, timed side by side.

    python -m paper_2608_09225_gb300.variants [name:flags ...]

Each variant is the library compiled with extra nvcc -D flags (for example
KVGOV_COMPACT_ROUNDS=0|1, KVGOV_CHAIN_R=64|128|256, KVGOV_FMA_ADDS=0|1) into
_build/variants/<name>/libkvgov.so.  kvgov_chain_hash is timed on three
workload shapes (15 launches each, CUDA events, median) and every variant's
digests must equal the first variant's, byte for byte.  Prints one JSON line
per variant.  Needs a GPU.
"""
from __future__ import annotations

import ctypes
import json
import os
import subprocess
import sys

import numpy as np

from . import build as kbuild
from . import workloads as W

DEFAULT = ["compact128:-DKVGOV_COMPACT_ROUNDS=1 -DKVGOV_CHAIN_R=128",
           "unroll128:-DKVGOV_COMPACT_ROUNDS=0 -DKVGOV_CHAIN_R=128",
           "compact256:-DKVGOV_COMPACT_ROUNDS=1 -DKVGOV_CHAIN_R=256",
           "unroll256:-DKVGOV_COMPACT_ROUNDS=0 -DKVGOV_CHAIN_R=256",
           "unroll128_imad:-DKVGOV_COMPACT_ROUNDS=0 -DKVGOV_FMA_ADDS=1"]
SOURCES = ["kvgov_chain.cu", "kvgov_salts.cu", "kvgov_table.cu"]


def build_variant(name: str, flags: list[str]) -> str:
    out = os.path.join(kbuild.BUILD_DIR, "variants", name)
    os.makedirs(out, exist_ok=True)
    cc = kbuild.nvcc()
    procs, objs = [], []
    for src in SOURCES:
        obj = os.path.join(out, src.replace(".cu", ".o"))
        objs.append(obj)
        procs.append(subprocess.Popen([cc, *kbuild.ARCH, *kbuild.FLAGS, *flags, "-c", os.path.join(kbuild.CSRC, src),
                                       "-o", obj]))
    if any(p.wait() != 0 for p in procs):
        raise RuntimeError(f"variant {name}: nvcc failed")
    lib = os.path.join(out, "libkvgov.so")
    subprocess.run([cc, *kbuild.ARCH, "-shared", "-o", lib, *objs], check=True)
    return lib


def main(argv):
    import torch
    specs = argv or DEFAULT
    p = ctypes.c_void_p
    cases = []
    for name, mode, w in (("wide_boundary", 2, W.make("wide", seed=5)),
                          ("probe_root", 1, W.probe(seed=6, n_req=65536, n_prior=64, capacity=1 << 12, n_random=10)),
                          ("template_unsalted", 0, W.make("template"))):
        b = w.batch

        def dev(a):
            return torch.from_numpy(np.ascontiguousarray(a)).cuda()

        cases.append(dict(name=name, mode=mode, w=w, toks=dev(b.tokens), tok_off=dev(b.tok_off), pr=dev(b.principal),
                          bt=dev(b.boundary_tok), ids=dev(w.ids), id_off=dev(w.id_off), n=b.n,
                          nblk=int((np.diff(b.tok_off) // 16).sum())))
    stream = torch.cuda.current_stream().cuda_stream
    ref = {}
    for spec in specs:
        name, _, flags = spec.partition(":")
        L = ctypes.CDLL(build_variant(name, flags.split()))
        L.kvgov_block_offsets.argtypes = [p, ctypes.c_int32, p, p, p]
        L.kvgov_derive_salts.argtypes = [p, ctypes.c_size_t, p, p, ctypes.c_int32, p, p, p]
        L.kvgov_chain_hash.argtypes = [ctypes.c_int, p, p, ctypes.c_int32, p, p, ctypes.c_int32, p, p, p, p, p]
        res = {}
        for c in cases:
            n_p = len(c["id_off"]) - 1
            salts = torch.empty((n_p, 32), dtype=torch.uint8, device="cuda")
            sec = ctypes.create_string_buffer(c["w"].secret, len(c["w"].secret))
            assert L.kvgov_derive_salts(ctypes.cast(sec, p), len(c["w"].secret), c["ids"].data_ptr(),
                                        c["id_off"].data_ptr(), n_p, salts.data_ptr(), None, stream) == 0
            blk = torch.empty(c["n"] + 1, dtype=torch.int64, device="cuda")
            assert L.kvgov_block_offsets(c["tok_off"].data_ptr(), c["n"], blk.data_ptr(), None, stream) == 0
            dig = torch.empty((c["nblk"], 32), dtype=torch.uint8, device="cuda")
            st = torch.zeros(1, dtype=torch.int32, device="cuda")

            def run():
                assert L.kvgov_chain_hash(c["mode"], c["toks"].data_ptr(), c["tok_off"].data_ptr(), c["n"],
                                          c["pr"].data_ptr(), salts.data_ptr(), n_p, c["bt"].data_ptr(),
                                          blk.data_ptr(), dig.data_ptr(), st.data_ptr(), stream) == 0

            for _ in range(3):
                run()
            ts = []
            for _ in range(15):
                a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                run()
                e.record()
                torch.cuda.synchronize()
                ts.append(a.elapsed_time(e))
            d = dig.cpu().numpy()
            ref.setdefault(c["name"], d)
            res[c["name"]] = {"ms_median": float(np.median(ts)), "blocks_per_s": c["nblk"] / (np.median(ts) / 1e3),
                              "same_digests_as_first": bool((d == ref[c["name"]]).all()) and int(st.item()) == 0}
        print(json.dumps({"variant": name, "flags": flags, **res}), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main(sys.argv[1:]))
