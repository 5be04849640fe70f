"""Build-time variants of libkvgov, timed side by side.

    python -m paper_2608_09225_gb300.variants [name:flags ...]
    python -m paper_2608_09225_gb300.variants --insert [name:flags ...]
    python -m paper_2608_09225_gb300.variants --probe [name:flags ...]

Each variant is the library compiled with extra nvcc -D flags into
_build/variants/<name>/libkvgov.so.

Chain mode (default; flags such as KVGOV_COMPACT_ROUNDS=0|1,
KVGOV_CHAIN_R=64|128|256, KVGOV_FMA_ADDS=0|1): kvgov_chain_hash is timed on
three workload shapes (15 launches each, CUDA events, median) and every
variant's digests must equal the first variant's, byte for byte.

Insert mode (flags KVGOV_INSERT_LOOK, _DEDUP, _PACK, _ST16 = 0|1): 80 serving
steps of the wide batch (131,072 x 128 tokens, BOUNDARY at token 64) against
a 2^25-slot table under a new secret epoch per step, flushed before a step
would take it past load factor 0.5; CUDA events around every kernel.  Reports
the median steady-state insert, the insert of the first step after a flush
(where every request's shared-prefix blocks are new, a hot key), probe and
step times; the number of keys inserted must equal the closed form.

Probe mode (flags KVGOV_PROBE_{MANY,MID,FEW}_{G,PER,PAIR,FIRST},
_MANY_MIN, _MID_MIN): kvgov_probe on every workload's probed requests against its table
as bench.py --configs fills it, plus two mid-size batches (all 8192 template
requests, the first 16,384 probe-heavy requests); mean of 20 back-to-back
launches queued behind a GPU spin.  Every variant's prefix lengths must
equal the first variant's.

Split mode (flag KVGOV_SPLIT_CTAS_PER_SM = 0..3: the largest batch the
small-batch chain kernel takes, in CTAs of 64 chains per SM; 0 never uses it):
kvgov_chain_hash in ROOT mode on batches of 512-token requests from a quarter
to four times the SM count x 64 requests (mean of 10 back-to-back launches
queued behind a GPU spin); every variant's digests must equal the first
variant's.

Prints one JSON line per variant.  Needs a GPU.
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
SOURCES = kbuild.LIBS[kbuild.LIB]


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


INSERT_DEFAULT = ["st16_pack1:-DKVGOV_INSERT_ST16=1 -DKVGOV_INSERT_PACK=1",
                  "st8_pack1:-DKVGOV_INSERT_ST16=0 -DKVGOV_INSERT_PACK=1",
                  "st16_pack0:-DKVGOV_INSERT_ST16=1 -DKVGOV_INSERT_PACK=0",
                  "st8_pack0:-DKVGOV_INSERT_ST16=0 -DKVGOV_INSERT_PACK=0",
                  "st16_pack1_dedup1:-DKVGOV_INSERT_ST16=1 -DKVGOV_INSERT_PACK=1 -DKVGOV_INSERT_DEDUP=1",
                  "st16_pack1_look0:-DKVGOV_INSERT_ST16=1 -DKVGOV_INSERT_PACK=1 -DKVGOV_INSERT_LOOK=0"]


def _bind(L):
    p = ctypes.c_void_p
    L.kvgov_block_offsets.argtypes = [p, ctypes.c_int32, p, p, p]
    L.kvgov_derive_salts.argtypes = [p, ctypes.c_size_t, p, p, ctypes.c_int32, p, p, p]
    L.kvgov_chain_hash.argtypes = [ctypes.c_int, p, p, ctypes.c_int32, p, p, ctypes.c_int32, p, p, p, p, p]
    L.kvgov_table_init.argtypes = [p, ctypes.c_uint64, p]
    L.kvgov_probe.argtypes = [p, ctypes.c_uint64, p, p, ctypes.c_int32, p, p, p]
    L.kvgov_insert_uncached.argtypes = [p, ctypes.c_uint64, p, p, ctypes.c_int32, p, p, p, p]
    return L


def insert_mode(specs):
    import torch
    n_pool, steps, cap = 4, 80, 1 << 25
    pool = [W.make("wide", seed=300 + i) for i in range(n_pool)]
    p0 = pool[0].batch.tokens.reshape(-1, 128)[0, :64].copy()
    for w in pool:                               # one service-wide 64-token prefix
        w.batch.tokens.reshape(-1, 128)[:, :64] = p0
    w0 = pool[0]
    n = w0.batch.n
    nblk = n * 8

    def dev(a):
        return torch.from_numpy(np.ascontiguousarray(a)).cuda()

    dp = [(dev(w.batch.tokens), dev(w.batch.tok_off), dev(w.batch.principal), dev(w.batch.boundary_tok))
          for w in pool]
    ids, id_off = dev(w0.ids), dev(w0.id_off)
    stream = torch.cuda.current_stream().cuda_stream
    for spec in specs:
        name, _, flags = spec.partition(":")
        L = _bind(ctypes.CDLL(build_variant(name, flags.split())))
        slots = torch.empty((cap, 32), dtype=torch.uint8, device="cuda")
        salts = torch.empty((4096, 32), dtype=torch.uint8, device="cuda")
        blk = torch.empty(n + 1, dtype=torch.int64, device="cuda")
        dig = torch.empty((nblk, 32), dtype=torch.uint8, device="cuda")
        pre = torch.empty(n, dtype=torch.int32, device="cuda")
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        n_new = torch.zeros(1, dtype=torch.int64, device="cuda")
        in_table, expect, fresh = 0, 0, True
        t = {"insert_steady": [], "insert_after_flush": [], "probe": [], "step": []}
        assert L.kvgov_table_init(slots.data_ptr(), cap, stream) == 0
        for s_i in range(steps):
            if not fresh and in_table + 4 * n > cap // 2:
                assert L.kvgov_table_init(slots.data_ptr(), cap, stream) == 0
                in_table, fresh = 0, True
            add = 4 * n + (4 if fresh else 0)
            first = fresh
            in_table, expect, fresh = in_table + add, expect + add, False
            toks, toff, prin, bt = dp[s_i % n_pool]
            sec = w0.secret[:24] + s_i.to_bytes(8, "little")
            buf = ctypes.create_string_buffer(sec, len(sec))
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
            ev[0].record()
            assert L.kvgov_derive_salts(ctypes.cast(buf, ctypes.c_void_p), len(sec), ids.data_ptr(),
                                        id_off.data_ptr(), 4096, salts.data_ptr(), st.data_ptr(), stream) == 0
            assert L.kvgov_block_offsets(toff.data_ptr(), n, blk.data_ptr(), st.data_ptr(), stream) == 0
            assert L.kvgov_chain_hash(2, toks.data_ptr(), toff.data_ptr(), n, prin.data_ptr(), salts.data_ptr(),
                                      4096, bt.data_ptr(), blk.data_ptr(), dig.data_ptr(), st.data_ptr(),
                                      stream) == 0
            ev[1].record()
            assert L.kvgov_probe(slots.data_ptr(), cap, dig.data_ptr(), blk.data_ptr(), n, pre.data_ptr(),
                                 st.data_ptr(), stream) == 0
            ev[2].record()
            assert L.kvgov_insert_uncached(slots.data_ptr(), cap, dig.data_ptr(), blk.data_ptr(), n, pre.data_ptr(),
                                           n_new.data_ptr(), st.data_ptr(), stream) == 0
            ev[3].record()
            torch.cuda.synchronize()
            if s_i >= 2:
                t["insert_after_flush" if first else "insert_steady"].append(ev[2].elapsed_time(ev[3]))
                t["probe"].append(ev[1].elapsed_time(ev[2]))
                t["step"].append(ev[0].elapsed_time(ev[3]))
        ok = int(st.item()) == 0 and int(n_new.item()) == expect
        res = {k: round(float(np.median(v)) * 1e3, 1) for k, v in t.items() if v}
        print(json.dumps({"variant": name, "flags": flags, "us_median": res, "keys_inserted": int(n_new.item()),
                          "keys_expected": expect, "ok": ok}), flush=True)
        del slots
    return 0


PROBE_DEFAULT = [
    "default:",
    "all_single:-DKVGOV_PROBE_MID_PAIR=0 -DKVGOV_PROBE_FEW_PAIR=0",
    "all_pair:-DKVGOV_PROBE_MANY_PAIR=1",
    "mid_single:-DKVGOV_PROBE_MID_PAIR=0",
    "mid_8x1_first8:-DKVGOV_PROBE_MID_G=8 -DKVGOV_PROBE_MID_PER=1 -DKVGOV_PROBE_MID_FIRST=8",
    "many_8x1_first8:-DKVGOV_PROBE_MANY_G=8 -DKVGOV_PROBE_MANY_FIRST=8",
]


def probe_cases(torch, seed=2030):
    """Each workload's digests, table and probed range, made with the default
    library (the fill of bench.py --configs)."""
    from . import kvgov as K
    from .pipeline import DeviceBatch, PrefixCache, next_pow2
    tmpl = W.make("template")
    cases = []
    for name, mode, w in (("tiny", W.ROOT, W.make("tiny")), ("sysprompt", W.ROOT, W.make("sysprompt")),
                          ("template_unsalted", W.UNSALTED, tmpl), ("template_root", W.ROOT, tmpl),
                          ("probe", W.ROOT, W.make("probe")), ("long", W.BOUNDARY, W.make("long", seed=seed)),
                          ("wide", W.BOUNDARY, W.make("wide", seed=seed + 1))):
        b = w.batch
        cap = w.capacity or next_pow2(4 * int((b.lengths() // 16).sum()))
        cache = PrefixCache(cap, w.secret, w.ids, w.id_off)
        db = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
        blk, dig = cache.hash(mode, db)
        blk_np = blk.cpu().numpy()
        keys = []
        if w.fill_from == "prior":
            pdb = DeviceBatch.from_host(w.prior.tokens, w.prior.tok_off, w.prior.principal, w.prior.boundary_tok)
            keys.append(cache.hash(mode, pdb)[1])
        elif w.fill[1] > w.fill[0]:
            keys.append(dig[blk_np[w.fill[0]]:blk_np[w.fill[1]]])
        else:
            keys.append(dig[: blk_np[b.n // 2]])
        if w.random_keys is not None:
            keys.append(torch.from_numpy(w.random_keys).cuda())
        K.insert(cache.slots, torch.cat(keys), cache.status)
        torch.cuda.synchronize()
        cache.check_status()
        p0, p1 = w.probe if w.probe[1] > w.probe[0] else (0, b.n)
        cases.append(dict(name=name, slots=cache.slots, cap=cap, dig=dig, blk=blk[p0:p1 + 1], n=p1 - p0))
        if name in ("template_root", "probe"):      # mid-size batches: every template request, 16,384 probes
            q1 = b.n if name == "template_root" else 16384
            cases.append(dict(name=name + f"_{q1}", slots=cache.slots, cap=cap, dig=dig, blk=blk[:q1 + 1], n=q1))
    return cases


def probe_mode(specs):
    import torch
    cases = probe_cases(torch)
    stream = torch.cuda.current_stream().cuda_stream
    ref = {}
    for spec in specs:
        name, _, flags = spec.partition(":")
        L = _bind(ctypes.CDLL(build_variant(name, flags.split())))
        res, same = {}, True
        for c in cases:
            pre = torch.full((c["n"],), -1, dtype=torch.int32, device="cuda")
            st = torch.zeros(1, dtype=torch.int32, device="cuda")

            def run():
                assert L.kvgov_probe(c["slots"].data_ptr(), c["cap"], c["dig"].data_ptr(), c["blk"].data_ptr(),
                                     c["n"], pre.data_ptr(), st.data_ptr(), stream) == 0

            for _ in range(3):
                run()
            torch.cuda.synchronize()
            a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda._sleep(4_000_000)
            a.record()
            for _ in range(20):
                run()
            e.record()
            torch.cuda.synchronize()
            res[c["name"]] = round(a.elapsed_time(e) / 20 * 1e3, 2)
            got = pre.cpu().numpy()
            same = same and int(st.item()) == 0 and (c["name"] not in ref or (got == ref[c["name"]]).all())
            ref.setdefault(c["name"], got)
        print(json.dumps({"variant": name, "flags": flags, "probe_us": res, "same_prefix_as_first": bool(same)}),
              flush=True)
    return 0


SPLIT_DEFAULT = ["split0:-DKVGOV_SPLIT_CTAS_PER_SM=0", "split1:-DKVGOV_SPLIT_CTAS_PER_SM=1",
                 "split2:-DKVGOV_SPLIT_CTAS_PER_SM=2", "split3:-DKVGOV_SPLIT_CTAS_PER_SM=3"]


def split_mode(specs):
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    sizes = [sms * 64 * f // 4 for f in (1, 2, 4, 6, 8, 12, 16)]
    b = W.ragged(11, [512] * sizes[-1])
    salts = torch.from_numpy(np.random.default_rng(3).integers(0, 256, (8, 32), dtype=np.uint8)).cuda()
    toks = torch.from_numpy(b.tokens).cuda()
    tok_off = torch.from_numpy(b.tok_off).cuda()
    pr = torch.from_numpy(b.principal).cuda()
    stream = torch.cuda.current_stream().cuda_stream
    ref = {}
    for spec in specs:
        name, _, flags = spec.partition(":")
        L = _bind(ctypes.CDLL(build_variant(name, flags.split())))
        res, same = {}, True
        for n in sizes:
            blk = torch.empty(n + 1, dtype=torch.int64, device="cuda")
            assert L.kvgov_block_offsets(tok_off.data_ptr(), n, blk.data_ptr(), None, stream) == 0
            dig = torch.empty((n * 32, 32), dtype=torch.uint8, device="cuda")
            st = torch.zeros(1, dtype=torch.int32, device="cuda")

            def run():
                assert L.kvgov_chain_hash(1, toks.data_ptr(), tok_off.data_ptr(), n, pr.data_ptr(), salts.data_ptr(),
                                          8, None, blk.data_ptr(), dig.data_ptr(), st.data_ptr(), stream) == 0

            for _ in range(3):
                run()
            torch.cuda.synchronize()
            a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda._sleep(4_000_000)
            a.record()
            for _ in range(10):
                run()
            e.record()
            torch.cuda.synchronize()
            res[str(n)] = round(a.elapsed_time(e) / 10 * 1e3, 1)
            got = dig.cpu().numpy()
            same = same and int(st.item()) == 0 and (n not in ref or (got == ref[n]).all())
            ref.setdefault(n, got)
        print(json.dumps({"variant": name, "flags": flags, "chain_us_by_requests": res,
                          "same_digests_as_first": bool(same)}), flush=True)
    return 0


def main(argv):
    import torch
    if argv and argv[0] == "--split":
        return split_mode(argv[1:] or SPLIT_DEFAULT)
    if argv and argv[0] == "--insert":
        return insert_mode(argv[1:] or INSERT_DEFAULT)
    if argv and argv[0] == "--probe":
        return probe_mode(argv[1:] or PROBE_DEFAULT)
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
