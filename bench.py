#!/usr/bin/env python3
"""Benchmark: KVGov salted block-hash chain + prefix-cache probe on GB300.

One step = one serving batch through the whole hot path, every step a
libkvgov kernel: per-principal salts (HMAC-SHA-256, 4096 principals) ->
blocking (block offsets) -> BOUNDARY-salted chain hash (salt at token 64,
block 4) -> probe of the resident prefix-cache table -> insert of each
request's uncached blocks.  DevicePipeline runs each batch's insert inside
the next batch's chain-hash launch (the last one after the timed loop,
still inside the timed region).  Workload: 131,072 requests x 128 tokens (8 blocks
each; the largest batch), a 64-token prefix shared by all requests, 4096
principals.

Serving regime: a pool of distinct batches (inputs resident in HBM) is
cycled, and every step runs under a new secret epoch, so each step is new
traffic: the 4 unsalted shared-prefix blocks of every request hit the cache,
the 4 salted blocks miss and are inserted (524,288 new keys per step).  The
table is sized so that its load factor stays at or below 0.5 at the end.

Timed region: `--steps` steps after `--warmup` untimed ones, bracketed by a
barrier and cuda synchronize, CUDA events on the launching stream, max over
ranks.  Prints ONE JSON line (rank 0).  `--impl reference` times the CPU
oracle (plain C) on a bounded sample of the same step as the reference arm.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, HERE)

METRIC = "salted block digests/s and tokens hashed/s on 1 GB300; % of INT32 issue peak"
UNIT = "block digests/s"
WORKLOAD = {"workload": "wide: 131072 requests x 128 tokens, BOUNDARY salt at token 64, 4096 principals",
            "requests": 131072, "tokens_per_request": 128, "block": 16, "blocks_per_step": 131072 * 8,
            "principals": 4096, "mode": "BOUNDARY (k=4)"}
SM_MAX_MHZ = 2070.0            # maximum SM clock of a GB300 (profiling recipe)
DRIFT_LIMIT = 0.05             # the two halves of the timed steps must agree to within 5 % ...
DRIFT_LIMIT_SHORT = 0.10       # ... (10 % when each half has fewer than DRIFT_FULL_HALF steps) ...
DRIFT_FULL_HALF = 50
DRIFT_MIN_HALF = 10            # ... when each half has at least 10 steps
INT32_LANES_PER_SM = 64        # 4 SMSPs x 16 lanes of the integer ALU pipe (LOP3 and SHF microbench: 64/clk/SM)
CHAIN_SOURCES = ["paper_2608_09225_gb300/csrc/kvgov_chain.cu", "paper_2608_09225_gb300/csrc/sha256_dev.cuh",
                 "paper_2608_09225_gb300/csrc/kvgov_internal.cuh", "paper_2608_09225_gb300/csrc/kvgov_lookup.cuh",
                 "paper_2608_09225_gb300/csrc/kvgov_insert.cuh", "paper_2608_09225_gb300/csrc/kvgov_stash.cuh"]
CHAIN_HEADER = "include/kvgov.h"      # only its #define lines reach the chain kernel's code
# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) per launch of the
# step's chain kernel from one ncu capture, and the SHA-256 (chain_source_hash)
# of the sources it was captured from: reported as roofline.traffic only while
# the kernel's sources still hash to that value.
CHAIN_TRAFFIC = {"chain_prev_kernel": {"bytes_per_launch": 200526208,
                 "source_sha256": "85d072705de98f8ea01e70bcc93f66213122131b53e0fc6a62e5e966b7fa9585"},
                 "chain_serve_kernel": {"bytes_per_launch": 200615680,
                                        "source_sha256": "0619a12914dd648e870c7a6cacd06f92e38e46c2757b83ac2424d8d226fd7827"}}


# DRAM bytes per launch of the probe on the probe-heavy workload from one ncu
# capture, with the SHA-256 of the table kernels' sources it was taken from.
TABLE_SOURCES = ["paper_2608_09225_gb300/csrc/kvgov_table.cu", "paper_2608_09225_gb300/csrc/kvgov_lookup.cuh",
                 "paper_2608_09225_gb300/csrc/kvgov_stash.cuh", "paper_2608_09225_gb300/csrc/kvgov_internal.cuh",
                 "paper_2608_09225_gb300/csrc/kvgov_insert.cuh"]
TABLE_TRAFFIC = {"probe_share_kernel<16, true>": {
    "bytes_per_launch": 74561792, "source_sha256": "c4f89d4058529d0c53f612bec5fb827b26dad802c885253c7535f69eebcba2aa"}}


def load_peaks() -> dict:
    """Measured copy bandwidth of this GPU pool (written beside the repository
    by the pool's driver); the profiling fallback of 6.8 TB/s without it."""
    try:
        with open(os.path.join(HERE, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except (OSError, ValueError):
        return {"hbm_gbs": 6800.0, "fallback": True}


PEAKS = load_peaks()


def sources_hash(sources) -> str:
    """SHA-256 over a kernel's translation-unit sources and the constants
    (#define lines) of the public header they include."""
    import hashlib
    h = hashlib.sha256()
    for rel in sources:
        with open(os.path.join(HERE, rel), "rb") as f:
            h.update(f.read())
    with open(os.path.join(HERE, CHAIN_HEADER), "rb") as f:
        h.update(b"".join(line for line in f.read().splitlines(keepends=True) if line.lstrip().startswith(b"#define")))
    return h.hexdigest()


def table_traffic(kernel: str):
    """DRAM bytes per launch of a table kernel from its last ncu capture, if
    that capture was taken of the current sources; else None."""
    rec = TABLE_TRAFFIC.get(kernel, {})
    if rec.get("bytes_per_launch") is None:
        return None, "no capture recorded"
    if rec.get("source_sha256") != sources_hash(TABLE_SOURCES):
        return None, "the last capture was of other sources"
    return rec["bytes_per_launch"], "ncu capture of the current sources"


def chain_source_hash() -> str:
    """sources_hash of the chain kernel's translation unit."""
    return sources_hash(CHAIN_SOURCES)


def profiled_traffic(kernel: str):
    """DRAM bytes per launch of the step's chain kernel from its last ncu
    capture, if that capture was taken of the chain kernel's current sources;
    else None."""
    rec = CHAIN_TRAFFIC.get(kernel, {})
    if rec.get("bytes_per_launch") is None:
        return None, "no capture recorded"
    if rec.get("source_sha256") != chain_source_hash():
        return None, "the last capture was of other sources"
    return rec["bytes_per_launch"], "ncu capture of the current sources"


# --------------------------------------------------------------------------- helpers
def rank_seed(seed: int, rank: int, i: int) -> int:
    """Seed of batch i on rank `rank`: ranks draw disjoint streams of batches
    (weak scaling: requests are sharded, nothing is exchanged)."""
    return seed + 1000003 * rank + i


def max_over_ranks(ms: float, world: int, dist, device) -> float:
    """Slowest rank's time (the whole job finishes when it does)."""
    if world <= 1:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def nominal_chain_ops(nb: np.ndarray, mode: int, k: np.ndarray | None) -> int:
    """Nominal integer ops of the chain kernel: 1384 per scheduled compression,
    904 per compression whose schedule is a compile-time constant (padding
    block).  Per block: 64-byte message 1384 + 904; 96-byte 2 x 1384;
    128-byte (boundary block, k >= 1) 2 x 1384 + 904."""
    nb = np.asarray(nb, dtype=np.int64)
    m64, m96, m128 = 1384 + 904, 2 * 1384, 2 * 1384 + 904
    if mode == 0:
        return int(np.where(nb > 0, m64 + (nb - 1) * m96, 0).sum())
    if mode == 1:
        return int((nb * m96).sum())
    k = np.asarray(k, dtype=np.int64)
    salted = k < nb
    tot = np.zeros_like(nb)
    # k = 0: ROOT chain; k >= 1 inside: 64 + (nb-2) x 96 + one 128; k >= nb: UNSALTED
    tot = np.where(salted & (k == 0), nb * m96, tot)
    tot = np.where(salted & (k > 0), m64 + (nb - 2) * m96 + m128, tot)
    tot = np.where(~salted & (nb > 0), m64 + (nb - 1) * m96, tot)
    return int(tot.sum())


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.t.join(timeout=2)

    def summary(self):
        sm, mx, pw, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
                pw.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:8]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "power_w_max": max(pw),
                "reasons": sorted(reasons), "samples": len(sm)}


def measure_int_peak(torch, peak_lib_path):
    """Thread-ops per SM clock of LOP3, SHF, IADD3, IMAD and SHA-256 (adds on
    the ALU / as IMAD), from libkvgov_peak."""
    import ctypes
    L = ctypes.CDLL(peak_lib_path)
    L.kvgov_peak_int.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                 ctypes.c_void_p, ctypes.c_void_p]
    L.kvgov_peak_ops_per_iter.argtypes = [ctypes.c_int]
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    out = {}
    for kind, name, threads, blocks_per_sm, iters in ((0, "lop3", 256, 8, 4000), (1, "shf", 256, 8, 4000),
                                                      (2, "iadd3", 256, 8, 4000), (3, "sha_alu", 256, 4, 200),
                                                      (4, "sha_fma", 256, 4, 200), (5, "imad", 256, 8, 4000),
                                                      (8, "lop3+iadd3", 256, 8, 4000), (9, "lop3+imad", 256, 8, 4000),
                                                      (10, "shf+iadd3", 256, 8, 4000),
                                                      (11, "sha_msg96", 256, 4, 100), (12, "sha_msg96_split", 256, 4, 100),
                                                      (11, "sha_msg96_8w", 256, 8, 100),
                                                      (12, "sha_msg96_split_8w", 256, 8, 100)):
        blocks = n_sm * blocks_per_sm
        sink = torch.zeros(1, dtype=torch.int32, device="cuda")
        clocks = torch.zeros(blocks * 3, dtype=torch.int64, device="cuda")
        for _ in range(2):
            rc = L.kvgov_peak_int(kind, iters, blocks, threads, sink.data_ptr(), clocks.data_ptr(),
                                  torch.cuda.current_stream().cuda_stream)
            assert rc == 0, rc
        torch.cuda.synchronize()
        c = clocks.view(blocks, 3).cpu().numpy()
        per_sm = {}
        for sm, t0, t1 in c:
            lo, hi, cnt = per_sm.get(int(sm), (t0, t1, 0))
            per_sm[int(sm)] = (min(lo, t0), max(hi, t1), cnt + 1)
        ops_iter = L.kvgov_peak_ops_per_iter(kind)
        rates = [cnt * threads * iters * ops_iter / max(hi - lo, 1) for lo, hi, cnt in per_sm.values()]
        out[name] = float(np.median(rates))
    out["n_sm"] = n_sm
    return out


def measure_lone_warp_round(torch, peak_lib_path) -> float:
    """SM clock cycles of one SHA-256 round for a warp alone on its SM
    sub-partition (libkvgov_peak kind 6: rounds only, K_t + W_t in
    registers, one CTA of four warps per SM): the latency floor of the
    small-batch chain kernel, whose round warp runs alone."""
    import ctypes
    L = ctypes.CDLL(peak_lib_path)
    L.kvgov_peak_int.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                 ctypes.c_void_p, ctypes.c_void_p]
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    iters = 400
    sink = torch.zeros(1, dtype=torch.int32, device="cuda")
    clocks = torch.zeros(n_sm * 3, dtype=torch.int64, device="cuda")
    for _ in range(2):
        assert L.kvgov_peak_int(6, iters, n_sm, 128, sink.data_ptr(), clocks.data_ptr(),
                                torch.cuda.current_stream().cuda_stream) == 0
    torch.cuda.synchronize()
    c = clocks.view(n_sm, 3).cpu().numpy()
    return float(np.median(c[:, 2] - c[:, 1])) / (iters * 64)


def main_slots(table) -> int:
    """The main slots of a table tensor (a power of two; the side store's
    slots follow them)."""
    return 1 << (table.shape[0].bit_length() - 1)


def measure_gather(torch, peak_lib_path, table: "torch.Tensor", n_reads: int = 1 << 25) -> dict:
    """Random-slot read rate (GB/s of bytes read, best of 5) over `table`,
    reading whole 32-byte slots and first halves, from libkvgov_peak."""
    import ctypes
    L = ctypes.CDLL(peak_lib_path)
    L.kvgov_peak_gather.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int, ctypes.c_int64,
                                    ctypes.c_uint64, ctypes.c_void_p, ctypes.c_void_p]
    sink = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = {"table_bytes": table.numel() * table.element_size(), "reads": n_reads}
    for slot_bytes in (32, 16):
        best = float("inf")
        for rep in range(6):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            rc = L.kvgov_peak_gather(table.data_ptr(), main_slots(table), slot_bytes, n_reads, 12345 + rep,
                                     sink.data_ptr(), torch.cuda.current_stream().cuda_stream)
            b.record()
            assert rc == 0, rc
            b.synchronize()
            if rep:
                best = min(best, a.elapsed_time(b))
        out[f"gbs_{slot_bytes}B"] = n_reads * slot_bytes / (best / 1e3) / 1e9
        out[f"reads_per_s_{slot_bytes}B"] = n_reads / (best / 1e3)
    return out


def measure_slot_ops(torch, peak_lib_path, table: "torch.Tensor", n_ops: int) -> dict:
    """Random-slot claims per second (best of 5) on `table`, zeroed before
    each run: 128-bit CAS; CAS + 16-byte store; 16-byte read + CAS + store."""
    import ctypes
    L = ctypes.CDLL(peak_lib_path)
    L.kvgov_peak_slot_ops.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int, ctypes.c_int64,
                                      ctypes.c_uint64, ctypes.c_void_p, ctypes.c_void_p]
    sink = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = {"table_bytes": table.numel() * table.element_size(), "ops": n_ops}
    for kind, name in ((0, "cas"), (1, "cas_store"), (2, "read_cas_store")):
        best = float("inf")
        for rep in range(6):
            table.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            rc = L.kvgov_peak_slot_ops(table.data_ptr(), main_slots(table), kind, n_ops, 777 + rep, sink.data_ptr(),
                                       torch.cuda.current_stream().cuda_stream)
            b.record()
            assert rc == 0, rc
            b.synchronize()
            if rep:
                best = min(best, a.elapsed_time(b))
        out[f"{name}_per_s"] = n_ops / (best / 1e3)
    return out


# --------------------------------------------------------------------------- reference arm
def epoch_secret(base: bytes, step: int) -> bytes:
    """The server secret of step `step` (an input of the step, not a hash)."""
    return base[:24] + int(step).to_bytes(8, "little")


def share_prefix(pool_host):
    """Give every pool batch the first batch's 64-token prefix (the prefix
    every request of the service starts with)."""
    p0 = pool_host[0].batch.tokens.reshape(-1, 128)[0, :64].copy()
    for w in pool_host:
        w.batch.tokens.reshape(-1, 128)[:, :64] = p0


class FlushPolicy:
    """Host bookkeeping of the cache's flush policy and the closed-form key
    counts: after a flush the next batch misses everywhere (it inserts the 4
    shared-prefix blocks once plus 4 salted blocks per request); later batches
    hit the shared prefix and insert their 4 salted blocks."""

    def __init__(self, capacity: int, new_per_step: int):
        self.capacity, self.new_per_step = capacity, new_per_step
        self.in_table, self.expected_new, self.flushes, self.last_prefix = 0, 0, 0, 0
        self.fresh = True
        self.seen = []

    def mean_load_factor(self) -> float:
        """Mean load factor the steps so far probed against (the table before
        each step's insert)."""
        return float(np.mean(self.seen)) / self.capacity if self.seen else 0.0

    def before_step(self) -> bool:
        flushed = False
        if not self.fresh and self.in_table + self.new_per_step > self.capacity // 2:
            self.in_table, self.fresh, flushed = 0, True, True
            self.flushes += 1
        add = self.new_per_step + (4 if self.fresh else 0)
        self.seen.append(self.in_table)
        self.last_prefix = 0 if self.fresh else 4
        self.in_table += add
        self.expected_new += add
        self.fresh = False
        return flushed


def cpu_oracle_step(w, sample_req, n_threads, secret):
    """The oracle on the first `sample_req` requests of one step: salts under
    `secret`, the chain (threaded over request chunks), the probe against a
    set holding the shared prefix's 4 blocks, and the insert of the uncached
    blocks.  Returns (blocks hashed, digests)."""
    import concurrent.futures as cf

    import oracle
    b = w.batch
    salts = oracle.derive_salts(secret, w.ids, w.id_off)
    n = sample_req
    chunks = np.array_split(np.arange(n), n_threads)

    def run(ix):
        if len(ix) == 0:
            return np.zeros((0, 32), np.uint8)
        lo, hi = int(ix[0]), int(ix[-1]) + 1
        off = b.tok_off[lo:hi + 1] - b.tok_off[lo]
        toks = b.tokens[b.tok_off[lo]:b.tok_off[hi]]
        return oracle.chain_hash(oracle.BOUNDARY, toks, off, b.principal[lo:hi], salts, b.boundary_tok[lo:hi])

    with cf.ThreadPoolExecutor(n_threads) as ex:
        d = np.concatenate(list(ex.map(run, chunks)))
    blk = oracle.block_offsets(b.tok_off[:n + 1])
    ks = oracle.KeySet(1)
    ks.insert(d[:4])                     # the shared prefix's blocks are cached
    pre = ks.prefix_blocks(d, blk)
    suffix = np.concatenate([d[blk[r] + pre[r]:blk[r + 1]] for r in range(n)])
    ks.insert(suffix)
    return int(blk[-1]), d


def reference_arm(args):
    import oracle
    from paper_2608_09225_gb300 import workloads as W
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    oracle.build()
    cores = len(os.sched_getaffinity(0))
    w = W.make("wide", seed=args.seed)
    sample = args.cpu_sample
    for i in range(args.warmup):
        cpu_oracle_step(w, sample, cores, epoch_secret(w.secret, i))
    t0 = time.perf_counter()
    blocks = 0
    for i in range(args.steps):
        blocks += cpu_oracle_step(w, sample, cores, epoch_secret(w.secret, args.warmup + i))[0]
    dt = time.perf_counter() - t0
    value = blocks / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32", "data": "synthetic",
            "config": dict(WORKLOAD, sample_requests=sample),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"first {sample} requests of the batch per step (salts for all 4096 "
                                       f"principals, chain on {cores} threads, probe, insert of the uncached blocks)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "tokens_per_s": 16 * value}
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------------- GPU arm
def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="kvgov", choices=["kvgov", "reference"])
    ap.add_argument("--pool", type=int, default=16, help="distinct resident batches cycled by the steps")
    ap.add_argument("--e2e-steps", type=int, default=100)
    ap.add_argument("--arrival-steps", type=int, default=50)
    ap.add_argument("--table-slots", type=int, default=1 << 25, help="cache capacity (power of two)")
    ap.add_argument("--seed", type=int, default=None, help="base seed (default: fresh per run)")
    ap.add_argument("--cpu-sample", type=int, default=16384, help="requests per oracle step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--schedule", default="one_launch", choices=["insert_in_chain", "inline", "one_launch"],
                    help="insert_in_chain: each batch's insert runs inside the next batch's chain-hash launch, and "
                         "each batch is probed after its chain hash; inline: chain hash with the fused probe, then "
                         "the insert; one_launch: each batch's lookups and insert in its own chain-hash launch "
                         "(kvgov_chain_hash_serve, the table's generations telling the batch's keys from older ones)")
    ap.add_argument("--configs", action="store_true",
                    help="instead of the timed serving step: per-kernel rates on every workload, one JSON line each")
    ap.add_argument("--only", default=None,
                    help="with --configs: comma-separated workloads to run (tiny, sysprompt, template, probe, long, "
                         "wide, audit)")
    ap.add_argument("--microbench", action="store_true",
                    help="instead of the timed serving step: the integer issue-rate microbenchmark alone, one JSON line")
    ap.add_argument("--probe-heavy", action="store_true",
                    help="instead of the timed serving step: the probe-heavy table leg alone, one JSON line")
    args = ap.parse_args()
    if args.seed is None:
        args.seed = int.from_bytes(os.urandom(4), "little")
    args.warmup = max(args.warmup, 3)
    if args.impl == "reference":
        return reference_arm(args)
    if args.configs:
        return run_configs(args)
    if args.microbench or args.probe_heavy:
        return run_single_leg(args)

    import torch
    import torch.distributed as dist

    from paper_2608_09225_gb300 import build as kbuild
    from paper_2608_09225_gb300 import kvgov as K
    from paper_2608_09225_gb300 import workloads as W
    from paper_2608_09225_gb300.pipeline import DeviceBatch, DevicePipeline, PrefixCache

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    kbuild.build()
    K.lib()

    # ---- inputs: a pool of distinct batches, resident in HBM (weak scaling: per-rank seeds)
    pool_host = [W.make("wide", seed=rank_seed(args.seed, rank, i)) for i in range(args.pool)]
    share_prefix(pool_host)
    w0 = pool_host[0]
    n_req = w0.batch.n
    n_blocks, w0_blk = K.count_blocks(w0.batch.tok_off)
    new_per_step = 4 * n_req                       # the salted blocks 4..7 of every request
    pool = [DeviceBatch.from_host(w.batch.tokens, w.batch.tok_off, w.batch.principal, w.batch.boundary_tok)
            for w in pool_host]
    cache = PrefixCache(args.table_slots, w0.secret, w0.ids, w0.id_off)
    flush = FlushPolicy(args.table_slots, new_per_step)
    bufs = {"blk_off": torch.empty(n_req + 1, dtype=torch.int64, device="cuda"),
            "digests": torch.empty((n_blocks, 32), dtype=torch.uint8, device="cuda"),
            "prefix": torch.empty(n_req, dtype=torch.int32, device="cuda")}

    # ---- gate before timing: the first serve into the empty table (closed forms)
    cache.set_secret(epoch_secret(w0.secret, 0))
    flush.before_step()
    prefix, digests, _ = cache.serve(W.BOUNDARY, pool[0], bufs)
    torch.cuda.synchronize()
    cache.check_status()
    gate_digests = digests.view(n_req, -1, 32)[: args.cpu_sample].cpu().numpy().reshape(-1, 32)
    gate = {"prefix_all_zero_on_empty_table": bool((prefix == 0).all().item()),
            "n_new": int(cache.n_new.item()), "n_new_expected": flush.expected_new}
    if not gate["prefix_all_zero_on_empty_table"] or gate["n_new"] != gate["n_new_expected"]:
        raise SystemExit(f"gate failed: {gate}")

    # ---- the timed steps: DevicePipeline computes each batch's salts and block
    # offsets on a prep stream beside the previous batch's chain hash
    in_chain = args.schedule == "insert_in_chain"
    one = args.schedule == "one_launch"
    pipe = DevicePipeline(cache, W.BOUNDARY, n_req, n_blocks, insert_in_chain=in_chain, one_launch=one)
    epoch = [1]
    launches = [0]
    table_timed = []

    def step(db, ev=None, tab_ev=None):
        cache.set_secret(epoch_secret(w0.secret, epoch[0]))
        epoch[0] += 1
        flushed = flush.before_step()              # load factor would pass 0.5: flush the cache
        pending = pipe.pending
        if one or (in_chain and (flushed or not pending)):
            tab_ev = None                          # this step runs no probe of its own (its chain launch looks up)
        if tab_ev is not None:
            table_timed.append(tab_ev)
        prefix, _ = pipe.submit(db, flushed, ev, tab_ev)
        if one:
            # salts, block offsets (2), the chain hash with the batch's lookups and insert (+ table init)
            launches[0] += 4 + int(flushed)
        elif in_chain:
            # salts, block offsets (2), then the chain hash with the previous batch's insert and the probe or,
            # after a flush (which runs the pending insert and the table init first), the chain hash with
            # the probe fused in
            launches[0] += 3 + (2 + int(pending) if flushed else (2 if pending else 1))
        else:
            # salts, block offsets (2), chain hash with the fused probe, insert (+ table init)
            launches[0] += 5 + int(flushed)
        return prefix

    for i in range(args.warmup):
        step(pool[(1 + i) % args.pool])
    torch.cuda.synchronize()
    table_timed.clear()
    n_new_before = int(cache.n_new.item())

    # time the chain launch and the table kernel of every 4th step (steps 0, 4, 8, ...): the other steps
    # carry no timing event between their launches
    timing_every = 4
    chain_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                if i % timing_every == 0 else None for i in range(args.steps)]
    table_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                if i % timing_every == 0 else None for i in range(args.steps)]
    t_start, t_stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_mid = torch.cuda.Event(enable_timing=True)   # between the two halves of the timed steps (drift gate)
    t_last = torch.cuda.Event(enable_timing=True)  # after the last step, before the pending insert runs
    # create every timing event now (a CUDA event is created on its first record, which costs the host far
    # more than a step's launches): inside the timed loop they are only recorded
    for pair in [e for e in chain_ev + table_ev if e is not None] + [(t_start, t_stop), (t_mid, t_last)]:
        for e in pair:
            e.record(pipe.compute_stream)
    torch.cuda.synchronize()
    launches[0] = 0
    flushes_before = flush.flushes
    with ClockSampler(local) as clk:
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        # a 1 ms spin ahead of the start event, so that the GPU reaches the timed steps with the first ones
        # already queued (otherwise it waits at the start for the host to enqueue step 0: about 0.2 ms)
        with torch.cuda.stream(pipe.compute_stream):
            torch.cuda._sleep(2_000_000)
        t_start.record(pipe.compute_stream)
        pipe.prep_stream.wait_event(t_start)
        h0 = time.perf_counter()
        half = args.steps // 2
        for i in range(args.steps):
            if i == half:
                t_mid.record(pipe.compute_stream)
            last_prefix = step(pool[(1 + args.warmup + i) % args.pool], chain_ev[i], table_ev[i])
        t_last.record(pipe.compute_stream)
        if in_chain:
            pipe.drain()                           # the last batch's insert
            launches[0] += 1
        host_ms = (time.perf_counter() - h0) * 1e3
        t_stop.record(pipe.compute_stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
    cache.check_status()
    gate["n_new_total"] = int(cache.n_new.item())
    gate["n_new_total_expected"] = flush.expected_new
    gate["flushes_in_timed_steps"] = flush.flushes - flushes_before
    gate["last_step_prefix_expected"] = flush.last_prefix
    gate["last_step_prefix_ok"] = bool((last_prefix == flush.last_prefix).all().item())
    if gate["n_new_total"] != gate["n_new_total_expected"] or not gate["last_step_prefix_ok"]:
        raise SystemExit(f"gate failed: {gate}")
    kernel_launches = launches[0]
    ms = t_start.elapsed_time(t_stop)
    # gate: two independent halves of the timed steps must agree (the paper's section 5.7 gates ask two
    # independent blocks of a measurement to agree)
    if half > 0:
        ms_a, ms_b = t_start.elapsed_time(t_mid) / half, t_mid.elapsed_time(t_last) / (args.steps - half)
        drift = abs(ms_a - ms_b) / ((ms_a + ms_b) / 2)
        gated = half >= DRIFT_MIN_HALF
        limit = DRIFT_LIMIT if half >= DRIFT_FULL_HALF else DRIFT_LIMIT_SHORT
        def mean_ms(pairs):
            t = [p[0].elapsed_time(p[1]) for p in pairs if p is not None]
            return float(np.mean(t)) if t else None
        chain_a, chain_b = mean_ms(chain_ev[:half]), mean_ms(chain_ev[half:])
        gate["drift"] = {"ms_per_step_first_half": ms_a, "ms_per_step_second_half": ms_b, "drift": drift,
                         "limit": limit, "gated": gated, "chain_ms_first_half": chain_a,
                         "chain_ms_second_half": chain_b,
                         "first_chain_start_ms": t_start.elapsed_time(chain_ev[0][0])}
        if gated and drift > limit:
            raise SystemExit(f"gate failed: the two halves of the timed steps differ by {100 * drift:.2f} % "
                             f"(limit {100 * limit:.0f} %): {gate['drift']}")
    chain_ms = float(np.mean([p[0].elapsed_time(p[1]) for p in chain_ev if p is not None]))
    table_ms = float(np.mean([a.elapsed_time(b) for a, b in table_timed]))
    inserted_per_step = (gate["n_new_total"] - n_new_before) / args.steps
    ms = max_over_ranks(ms, world, dist, "cuda")
    value = world * args.steps * n_blocks / (ms / 1e3)

    # ---- arrival-order serving of the same batches (kvgov_chain_hash_arrival), each into an empty cache
    arrival = arrival_leg(torch, K, W, pool, n_req, n_blocks, cache, args.arrival_steps, chain_ms)

    # ---- end to end through the public API with host buffers
    e2e = e2e_leg(torch, K, W, w0, pool_host[: min(4, args.pool)], args.e2e_steps, world, dist, args.table_slots,
                  in_chain, one)

    # ---- roofline of the chain kernel (integer-pipe bound)
    micro = measure_int_peak(torch, kbuild.PEAK_LIB)
    ops = nominal_chain_ops(np.diff(w0_blk), 2, w0.batch.boundary_tok // K.BLOCK)
    achieved = ops / (chain_ms / 1e3) / 1e12
    clock = clk.summary()
    n_sm = micro["n_sm"]
    # the SHA-256 ceiling: the chain kernel's own steady-block code (a 96-byte message, two compact
    # compressions) register-resident with no memory traffic, the better of two occupancies
    sha_rate = max(micro["sha_msg96"], micro["sha_msg96_8w"])
    peak_tops = n_sm * sha_rate * SM_MAX_MHZ * 1e6 / 1e12
    traffic, traffic_src = profiled_traffic("chain_serve_kernel" if one else "chain_prev_kernel")
    roofline = {"bound": "alu", "achieved": achieved, "peak": peak_tops, "unit": "Tops/s (int32)",
                "frac": achieved / peak_tops, "traffic": traffic,
                "kernel": ("chain_serve_kernel<BOUNDARY> (kvgov_chain_hash_serve: the chain hash with the batch's "
                           "own lookups and insert)" if one else
                           "chain_prev_kernel<BOUNDARY, insert + lookups> (kvgov_chain_hash_insert_prev: the chain "
                           "hash with the previous batch's insert and this batch's lookups)" if in_chain else
                           "chain_kernel<BOUNDARY, probe> (kvgov_chain_hash_probe)"), "ops_per_launch": ops,
                "kernel_ms": chain_ms, "timed_launches": f"every {timing_every}th step of the timed region",
                "ops_counted": "SHA-256 ops of the chain only; the fused " +
                               ("lookups and insert of the batch" if one else
                                "inserts of the previous batch and lookups of this one" if in_chain else "lookups") +
                               " are extra",
                "algorithmic_bytes_per_launch": 96 * n_blocks,
                "peak_basis": f"{n_sm} SMs x {sha_rate:.2f} nominal SHA-256 ops per SM per clock x {SM_MAX_MHZ:.0f} MHz:"
                              " the rate of the chain kernel's own steady-block code (a 96-byte message: two "
                              "compressions of 1384 nominal ops) with its data in registers, measured in this run "
                              "(libkvgov_peak kind 11). SHF and LOP3 (10 of a round's 14 ops) issue only to the "
                              "integer ALU pipe, 16 lanes per SM sub-partition (64 per SM per clock); IMAD issues to "
                              "the FMA-heavy pipe (64), alongside (a LOP3 + IMAD mix: 95.7); the compiler sends a "
                              "share of the adds there (ncu: 45 % of a pure IADD3 chain, 74.7 per clock; 8 % of "
                              "SHA-256's), which is how SHA-256 exceeds 64; issuing its off-chain adds as IMAD "
                              "explicitly measured slower (kind 12)",
                "int_ops_per_clk_per_sm_measured": {k: round(v, 2) for k, v in micro.items() if k != "n_sm"},
                "frac_of_alu_pipe_64": achieved / (n_sm * INT32_LANES_PER_SM * SM_MAX_MHZ * 1e6 / 1e12),
                "frac_of_issue_peak_128": achieved / (n_sm * 128 * SM_MAX_MHZ * 1e6 / 1e12),
                "traffic_source": traffic_src}
    # the table kernel of the step (insert of the uncached blocks) against HBM and a random-read ceiling
    gather = measure_gather(torch, kbuild.PEAK_LIB, cache.slots)
    claims = measure_slot_ops(torch, kbuild.PEAK_LIB, cache.slots, int(inserted_per_step))
    if one:
        table_roofline = {
            "kernel": None, "frac": None,
            "note": "no table kernel of its own: each batch's lookups (blocks 0-4 of every request: 4 hits and a "
                    "miss) and its insert (blocks 4-7) run inside its chain launch, told apart by the table's "
                    "generations; the DRAM-bound table case is table_roofline_cfg4",
            "lookups_in_chain_launch_per_step": 5 * n_req,
            "keys_inserted_per_step": inserted_per_step,
            "random_read_microbench": gather,
            "claim_ceiling_per_s": claims["read_cas_store_per_s"], "slot_op_microbench": claims}
    elif in_chain:
        # the probe resumes each request's walk where the chain launch's own lookups stopped: they found the 4
        # shared-prefix blocks (L2 hits, as they were hashed), so the probe looks up block 4, a miss walking
        # (1 + 1/(1-a)^2)/2 slots at the table's mean load factor a
        lf = flush.mean_load_factor()
        miss_walk = (1 + 1 / (1 - lf) ** 2) / 2
        lookups = n_req
        tab_bytes = n_req * (32 + miss_walk * 32) + 24 * n_req
        tab_gbs = tab_bytes / (table_ms / 1e3) / 1e9
        slot_bytes = n_req * 32 * miss_walk
        table_roofline = {
            "kernel": "probe_share_kernel<16, true> (kvgov_probe_resume: the step's probe, each walk resumed where "
                      "the chain launch's lookups stopped)", "bound": "hbm", "achieved": tab_gbs,
            "peak": PEAKS.get("hbm_gbs"), "unit": "GB/s",
            "frac": tab_gbs / PEAKS["hbm_gbs"] if PEAKS.get("hbm_gbs") else None,
            "peak_source": "of fallback (6.8 TB/s)" if PEAKS.get("fallback") else
                           "of measured (MEASURED_PEAKS.json hbm_gbs, a copy)",
            "note": "one dependent lookup per request after reading its offsets and lower bound: latency, not "
                    "bandwidth; the DRAM-bound table case is table_roofline_cfg4",
            "slot_bytes_per_launch": slot_bytes,
            "random_read_ceiling_gbs": gather["gbs_32B"],
            "frac_of_random_read_ceiling_slots": slot_bytes / (table_ms / 1e3) / 1e9 / gather["gbs_32B"],
            "kernel_ms": table_ms, "timed_launches": f"every {timing_every}th step of the timed region",
            "lookups_per_launch": lookups, "lookups_per_s": lookups / (table_ms / 1e3),
            "lookups_in_chain_launch_per_step": 5 * n_req,
            "mean_load_factor": lf, "algorithmic_bytes_per_launch": tab_bytes,
            "bytes_basis": "per request its block-4 digest (32 B), 32 B per slot its miss walks at the mean load "
                           "factor, 16 B offsets, 4 B lower bound in and 4 B prefix out (counted as if the chain "
                           "launch's lookups missed nothing: a lookup racing the insert of its own key adds work)",
            "random_read_microbench": gather,
            "insert": {"where": "inside the next batch's chain launch (kvgov_chain_hash_insert_prev)",
                       "keys_inserted_per_step": inserted_per_step,
                       "claim_ceiling_per_s": claims["read_cas_store_per_s"], "slot_op_microbench": claims}}
    else:
        ins_bytes = 96 * inserted_per_step + 20 * n_req
        ins_gbs = ins_bytes / (table_ms / 1e3) / 1e9
        table_roofline = {
            "kernel": "insert_uncached_packed_kernel (kvgov_insert_uncached)", "bound": "hbm", "achieved": ins_gbs,
            "peak": PEAKS.get("hbm_gbs"), "unit": "GB/s",
            "frac": ins_gbs / PEAKS["hbm_gbs"] if PEAKS.get("hbm_gbs") else None,
            "peak_source": "of fallback (6.8 TB/s)" if PEAKS.get("fallback") else
                           "of measured (MEASURED_PEAKS.json hbm_gbs, a copy)",
            "random_read_ceiling_gbs": gather["gbs_32B"], "frac_of_random_read_ceiling": ins_gbs / gather["gbs_32B"],
            "kernel_ms": table_ms, "timed_launches": f"every {timing_every}th step of the timed region",
            "keys_inserted_per_launch": inserted_per_step,
            "inserts_per_s": inserted_per_step / (table_ms / 1e3),
            "algorithmic_bytes_per_launch": ins_bytes,
            "bytes_basis": "per new key 32 B read + one 32 B slot read + 32 B written; per request 4 B prefix + "
                           "16 B offsets",
            "random_read_microbench": gather,
            "claim_ceiling_per_s": claims["read_cas_store_per_s"],
            "frac_of_claim_ceiling": (inserted_per_step / (table_ms / 1e3)) / claims["read_cas_store_per_s"],
            "slot_op_microbench": claims}
    if clock.get("sm_mhz"):
        roofline["frac_at_run_clock"] = achieved / (n_sm * sha_rate * clock["sm_mhz"] * 1e6 / 1e12)

    # ---- the probe-heavy workload: the table kernels on a 512 MiB table (larger than L2)
    table_cfg4 = probe_heavy_leg(torch, K, W, kbuild)

    # gate: no kernel may run above its own ceiling (the paper's section 5.7 gate rejects a result that
    # implies more than 100 % of the GPU's peak)
    fracs = {"roofline.frac": roofline["frac"], "table_roofline.frac": table_roofline["frac"] or 0.0,
             "table_roofline_cfg4.probe.frac": table_cfg4["probe"]["frac"],
             "table_roofline_cfg4.insert.frac": table_cfg4["insert"]["frac"]}
    gate["frac_ok"] = all(f is not None and f <= 1.0 for f in fracs.values())
    gate["fracs"] = fracs
    if not gate["frac_ok"]:
        raise SystemExit(f"gate failed: a kernel measured above its ceiling: {fracs}")

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "u32", "data": "synthetic",
            "config": dict(WORKLOAD, pool_batches=args.pool, seed=args.seed,
                           l2=f"{args.pool} distinct resident batches cycled (each re-read after "
                              f"{args.pool - 1} others); table {cache.capacity * 32 >> 20} MiB",
                           table_slots=cache.capacity,
                           regime="new secret epoch per step: the 4 shared-prefix blocks hit, the 4 salted blocks "
                                  "miss and are inserted; the cache is flushed (table re-initialised, inside the "
                                  "timed steps) whenever the next step would take it past load factor 0.5"),
            "tokens_per_s": 16 * value, "chain_digests_per_s": world * n_blocks / (chain_ms / 1e3),
            "host_enqueue_ms_per_step": host_ms / args.steps,
            "schedule": ("DevicePipeline over the library's serving engine (kvgov_pipeline_submit, one call per "
                         "step), one launch: salts (new epoch) and block offsets of batch i+1 on a prep stream "
                         "beside the chain launch of batch i, which on a higher-priority compute stream hashes "
                         "the batch, looks its blocks up and inserts its uncached ones" if one else
                         "DevicePipeline over the library's serving engine (kvgov_pipeline_submit, one call per "
                         "step), insert in chain: salts (new epoch) and block offsets of batch i+1 on a "
                         "prep stream beside the chain hash of batch i; on a higher-priority compute stream the "
                         "chain hash of batch i with batch i-1's insert in the same launch, then the probe of batch "
                         "i" if in_chain else
                         "DevicePipeline (inline): salts (new epoch) and block offsets of batch i+1 on a prep stream "
                         "beside the chain hash of batch i; chain hash with the fused probe, then the insert, on a "
                         "higher-priority compute stream"),
            "e2e": e2e, "gpu_launches": kernel_launches, "clocks": clock, "roofline": roofline,
            "table_roofline": table_roofline, "table_roofline_cfg4": table_cfg4,
            "arrival": arrival, "gate": gate}
    if rank == 0 and not args.no_cpu_baseline and world == 1:
        line["cpu_baseline"] = cpu_baseline(pool_host[0], args.cpu_sample, gate_digests)
        if not line["cpu_baseline"]["gate_sample_digests_equal_gpu"]:
            raise SystemExit("parity: GPU digests of the gate step differ from the oracle's")
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def probe_heavy_leg(torch, K, W, kbuild, reps: int = 10) -> dict:
    """The table kernels where the table is larger than L2: the probe-heavy
    workload (65,536 requests x 512 tokens, ROOT, 1024 principals; 30 % reuse
    the first 0-31 blocks of one of 8192 prior requests) probed against a
    2^24-slot (512 MiB) table at load factor 0.5 (the prior requests' chains
    and 8,126,464 random keys), and that table's fill from empty.  Each probe
    is timed alone with CUDA events after a 256 MiB write that flushes L2;
    each fill is a table initialisation then the insert, timed around the
    insert.  Both against the random-read ceiling measured on the same table."""
    from paper_2608_09225_gb300.pipeline import DeviceBatch, PrefixCache
    w = W.make("probe")
    b, p = w.batch, w.prior
    cache = PrefixCache(w.capacity, w.secret, w.ids, w.id_off)
    db = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
    dp = DeviceBatch.from_host(p.tokens, p.tok_off, p.principal, p.boundary_tok)
    blk, pblk = K.block_offsets(db.tok_off), K.block_offsets(dp.tok_off)
    dig = K.chain_hash(W.ROOT, db.tokens, db.tok_off, blk, db.principal, cache.salts, n_blocks=db.n_blocks)
    pdig = K.chain_hash(W.ROOT, dp.tokens, dp.tok_off, pblk, dp.principal, cache.salts, n_blocks=dp.n_blocks)
    keys = torch.cat([pdig, torch.from_numpy(w.random_keys).cuda()])
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    pre = torch.empty(b.n, dtype=torch.int32, device="cuda")
    n_new = torch.zeros(1, dtype=torch.int64, device="cuda")
    ins_ms, probe_ms = [], []
    for i in range(3 + reps):
        K.table_init(cache.slots)
        n_new.zero_()
        a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        K.insert(cache.slots, keys, cache.status, n_new)
        e.record()
        for _ in range(2):                         # two probes per fill, each after an L2 flush
            flush.zero_()
            pa, pe = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            pa.record()
            K.probe(cache.slots, dig, blk, pre, cache.status)
            pe.record()
            torch.cuda.synchronize()
            if i >= 3:
                probe_ms.append(pa.elapsed_time(pe))
        if i >= 3:
            ins_ms.append(a.elapsed_time(e))
    cache.check_status()
    n_keys, stored = keys.shape[0], int(n_new.item())
    L = pre.cpu().numpy().astype(np.int64)
    nb = np.diff(K.count_blocks(b.tok_off)[1])
    if stored != n_keys:
        raise SystemExit(f"probe-heavy leg: {stored} of {n_keys} keys stored")
    reuse, cut = w.info["reuse"], w.info["cut"]
    if not (L == np.where(reuse, cut, 0)).all():          # closed form: a reused request hits its cut, else 0
        raise SystemExit("probe-heavy leg: prefix lengths differ from the closed form")
    gather = measure_gather(torch, kbuild.PEAK_LIB, cache.slots)
    ceiling = gather["gbs_32B"]
    cap = K.capacity_of(cache.slots)
    alpha = n_keys / cap
    hit_walk, miss_walk = (1 + 1 / (1 - alpha)) / 2, (1 + 1 / (1 - alpha) ** 2) / 2
    hits = int(np.minimum(L, nb).sum())
    misses = int((L < nb).sum())
    hbm = PEAKS["hbm_gbs"]
    # the time a kernel needs at best: its random 32-byte slot accesses at the random-read ceiling plus its
    # streamed bytes (a request's consecutive digest rows, offsets, results, keys) at the copy bandwidth
    probe_random = (hits * hit_walk + misses * miss_walk) * 32
    probe_stream = (hits + misses) * 32 + 20 * b.n
    probe_bytes = probe_random + probe_stream
    t_probe = float(np.mean(probe_ms))
    probe_gbs = probe_bytes / (t_probe / 1e3) / 1e9
    probe_floor_ms = 1e3 * (probe_random / (ceiling * 1e9) + probe_stream / (hbm * 1e9))
    fill_walk = np.mean([(1 + 1 / (1 - a) ** 2) / 2 for a in np.linspace(0, alpha, 64, endpoint=False)])
    ins_random = n_keys * 32 * (fill_walk + 1)            # the slots walked, and the claimed slot written back
    ins_stream = n_keys * 32                               # the keys
    ins_bytes = ins_random + ins_stream
    t_ins = float(np.mean(ins_ms))
    ins_gbs = ins_bytes / (t_ins / 1e3) / 1e9
    ins_floor_ms = 1e3 * (ins_random / (ceiling * 1e9) + ins_stream / (hbm * 1e9))
    traffic, traffic_src = table_traffic("probe_share_kernel<16, true>")
    return {"workload": "probe-heavy: 65536 requests x 512 tokens, ROOT, 1024 principals, table 2^24 slots "
                        "(512 MiB) at load factor 0.5", "table_bytes": cap * 32, "load_factor": alpha,
            "random_read_ceiling_gbs": ceiling, "random_read_microbench": gather,
            "probe": {"kernel": "probe_share_kernel<16, true> (kvgov_probe)", "bound": "hbm (random 32-byte reads)",
                      "kernel_ms": t_probe, "timed_launches": len(probe_ms), "l2": "flushed before each launch",
                      "algorithmic_probes": hits + misses, "probes_per_s": (hits + misses) / (t_probe / 1e3),
                      "algorithmic_bytes_per_launch": probe_bytes, "random_bytes_per_launch": probe_random,
                      "streamed_bytes_per_launch": probe_stream, "achieved": probe_gbs, "unit": "GB/s",
                      "floor_ms": probe_floor_ms, "frac": probe_floor_ms / t_probe,
                      "frac_basis": "floor / measured time; floor = random slot bytes at the random-read ceiling "
                                    "(measured on this table) + streamed bytes at the copy bandwidth (of measured)",
                      "random_read_ceiling_gbs": ceiling, "frac_of_hbm_copy_peak": probe_gbs / hbm,
                      "traffic": traffic, "traffic_source": traffic_src,
                      "bytes_basis": "per lookup up to the first miss: its 32 B digest and 32 B per slot walked "
                                     "(linear probing at the load factor: (1 + 1/(1-a))/2 for a hit, "
                                     "(1 + 1/(1-a)^2)/2 for a miss); per request 16 B offsets + 4 B prefix"},
            "insert": {"kernel": "insert_kernel (kvgov_insert)", "bound": "hbm (random 32-byte slots)",
                       "kernel_ms": t_ins, "timed_launches": len(ins_ms), "keys": n_keys,
                       "inserts_per_s": n_keys / (t_ins / 1e3), "algorithmic_bytes_per_launch": ins_bytes,
                       "random_bytes_per_launch": ins_random, "streamed_bytes_per_launch": ins_stream,
                       "achieved": ins_gbs, "unit": "GB/s", "floor_ms": ins_floor_ms, "frac": ins_floor_ms / t_ins,
                       "frac_basis": "floor / measured time, as for the probe",
                       "bytes_basis": "per key its 32 B (streamed), 32 B per slot walked while the table fills "
                                      "from empty to the load factor and the 32 B slot written back (random)"}}


def arrival_leg(torch, K, W, pool, n_req, n_blocks, cache, steps, chain_ms):
    """kvgov_chain_hash_arrival on the pool's batches: each batch is served in
    arrival order into an empty 2^22-slot cache (re-initialised before the
    timed call), CUDA events around the call on its stream."""
    cap = 1 << 22
    slots, owner = K.new_table(cap), K.new_owner(cap)
    blk = torch.empty(n_req + 1, dtype=torch.int64, device="cuda")
    dig = torch.empty((n_blocks, 32), dtype=torch.uint8, device="cuda")
    slot_of = torch.empty(n_blocks, dtype=torch.int32, device="cuda")
    pre = torch.empty(n_req, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    n_new = torch.zeros(1, dtype=torch.int64, device="cuda")
    seq, times, means = 1, [], []
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps + 3)]
    for pair in evs:                               # created here, only recorded in the loop
        for e in pair:
            e.record()
    torch.cuda.synchronize()
    for i in range(steps + 3):
        db = pool[i % len(pool)]
        K.table_init(slots)
        K.block_offsets(db.tok_off, blk, status)
        a, b = evs[i]
        a.record()
        K.chain_hash_arrival(W.BOUNDARY, db.tokens, db.tok_off, blk, slots, owner, seq, status, db.principal,
                             cache.salts, db.boundary_tok, dig, slot_of, pre, n_new=n_new)
        b.record()
        seq += n_blocks
        if i >= 3:
            times.append((a, b))
            if i == 3:
                means.append(float(pre.float().mean().item()))
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise SystemExit(f"arrival leg: device status {int(status.item())}")
    ms = float(np.mean([x.elapsed_time(y) for x, y in times]))
    return {"api": "kvgov_chain_hash_arrival (chain hash, arrival-order insert fused into it, owner min, probe)",
            "ms_per_batch": ms, "blocks_per_s": n_blocks / (ms / 1e3), "steps": steps,
            "chain_hash_probe_ms": chain_ms, "extra_over_chain_hash_probe_ms": ms - chain_ms,
            "mean_prefix_blocks": means[0] if means else None,
            "cache": f"empty {cap}-slot table per batch (re-initialised outside the timed call)"}


def e2e_leg(torch, K, W, w0, hosts, steps, world, dist, table_slots, in_chain=True, one_launch=False):
    """Same step with host buffers, through the public HostPipeline: each
    step's inputs are copied from pinned host memory (a copy stream, which
    overlaps the previous step's serving) and its prefix lengths are copied
    back to pinned host memory, all inside the timed region."""
    from paper_2608_09225_gb300.pipeline import HostPipeline, PrefixCache
    pinned = []
    for w in hosts:
        b = w.batch
        pinned.append(tuple(torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
                            for a in (b.tokens, b.tok_off, b.principal, b.boundary_tok)))
    n_req = hosts[0].batch.n
    n_tok = int(hosts[0].batch.tok_off[-1])
    n_blocks, _ = K.count_blocks(hosts[0].batch.tok_off)
    cache = PrefixCache(table_slots, w0.secret, w0.ids, w0.id_off)
    pipe = HostPipeline(cache, W.BOUNDARY, n_req, n_tok, insert_in_chain=in_chain, one_launch=one_launch)
    flush = FlushPolicy(table_slots, 4 * n_req)
    h2d = sum(t.numel() * t.element_size() for t in pinned[0])
    d2h = n_req * 4

    def one(i):
        cache.set_secret(epoch_secret(w0.secret, i))
        return pipe.submit(*pinned[i % len(pinned)], n_blocks, flush.before_step())

    warm = len(pinned) + 1                         # every pinned input set is copied once before timing
    for i in range(warm):
        one(i)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    a.record(pipe.copy_stream)
    h0 = time.perf_counter()
    for i in range(steps):
        out, ev = one(warm + i)
    pipe.drain()                                   # the last batch's insert
    host_ms = (time.perf_counter() - h0) * 1e3
    b.record(pipe.compute_stream)
    torch.cuda.synchronize()
    cache.check_status()
    last_ok = bool((out == 4).all()) if flush.last_prefix == 4 else bool((out == 0).all())
    ms = max_over_ranks(a.elapsed_time(b), world, dist, "cuda")
    # the host link alone: one plain pinned -> device copy of a step's tokens
    link = []
    dst = torch.empty_like(pinned[0][0], device="cuda")
    for _ in range(5):
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        c0.record()
        dst.copy_(pinned[0][0], non_blocking=True)
        c1.record()
        c1.synchronize()
        link.append(c0.elapsed_time(c1))
    link_gbs = pinned[0][0].numel() * 4 / (min(link) / 1e3) / 1e9
    value = world * steps * n_blocks / (ms / 1e3)
    copy_bound = world * n_blocks / (h2d / (link_gbs * 1e9))
    return {"value": value, "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps, "last_step_prefix_ok": last_ok,
            "host_enqueue_ms_per_step": host_ms / steps, "ms_per_step": ms / steps,
            "h2d_link_gbs": link_gbs, "copy_bound_value": copy_bound, "frac_of_copy_bound": value / copy_bound,
            "api": "paper_2608_09225_gb300.pipeline.HostPipeline (copy of step i+1 overlaps serving of step i; "
                   "each step's insert inside the next step's chain launch)"}


def cpu_baseline(w, sample, gpu_digests):
    """The oracle, as it stands, on the machine's host cores: a bounded sample of
    the step.  Its digests of the gate step are compared with the GPU's."""
    import oracle
    oracle.build()
    cores = len(os.sched_getaffinity(0))
    _, d0 = cpu_oracle_step(w, sample, cores, epoch_secret(w.secret, 0))
    same = bool(d0.shape == gpu_digests.shape and (d0 == gpu_digests).all())
    reps, blocks, t0 = 0, 0, time.perf_counter()
    while reps < 2 or time.perf_counter() - t0 < 5.0:
        blocks += cpu_oracle_step(w, sample, cores, epoch_secret(w.secret, 1 + reps))[0]
        reps += 1
    dt = time.perf_counter() - t0
    one_reps, one_blocks, t1 = 0, 0, time.perf_counter()   # the same step on one thread
    one_sample = max(1, sample // 8)
    while one_reps < 1 or time.perf_counter() - t1 < 4.0:
        one_blocks += cpu_oracle_step(w, one_sample, 1, epoch_secret(w.secret, 100 + one_reps))[0]
        one_reps += 1
    dt1 = time.perf_counter() - t1
    return {"value": blocks / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{reps} steps over the first {sample} requests of one batch (salts for 4096 principals, "
                      f"chain on {cores} threads, probe, insert of the uncached blocks); {dt:.1f} s",
            "value_1_thread": one_blocks / dt1,
            "sample_1_thread": f"{one_reps} steps over the first {one_sample} requests, one thread; {dt1:.1f} s",
            "gate_sample_digests_equal_gpu": same}


def run_single_leg(args):
    """One measurement leg of the default run on its own (for a short run or
    an ncu capture of that leg's kernels)."""
    import torch

    from paper_2608_09225_gb300 import build as kbuild
    from paper_2608_09225_gb300 import kvgov as K
    from paper_2608_09225_gb300 import workloads as W
    kbuild.build()
    K.lib()
    if args.microbench:
        out = {"int_ops_per_clk_per_sm_measured": measure_int_peak(torch, kbuild.PEAK_LIB),
               "lone_warp_cycles_per_round": measure_lone_warp_round(torch, kbuild.PEAK_LIB)}
    else:
        out = {"table_roofline_cfg4": probe_heavy_leg(torch, K, W, kbuild)}
    print(json.dumps(out), flush=True)
    return 0


# --------------------------------------------------------------------------- per-workload rates
def _time(torch, fn, reps=10, warm=3):
    """Mean CUDA-event time of fn() in ms over `reps` back-to-back calls (fn
    enqueues on the current stream).  A GPU spin of about 2 ms is queued first,
    so that every call is already queued when the first one starts: the time
    is the GPU's, not the host's launch latency."""
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(4_000_000)
    a.record()
    for _ in range(reps):
        fn()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def _oracle_rate(w, mode, cores, budget_s=3.0):
    """Oracle digests/s on 1 thread and on `cores` threads over request chunks."""
    import concurrent.futures as cf

    import oracle
    b = w.batch
    salts = oracle.derive_salts(w.secret, w.ids, w.id_off)

    def run(lo, hi):
        off = b.tok_off[lo:hi + 1] - b.tok_off[lo]
        return len(oracle.chain_hash(mode, b.tokens[b.tok_off[lo]:b.tok_off[hi]], off, b.principal[lo:hi], salts,
                                     b.boundary_tok[lo:hi]))

    out = {}
    for threads in (1, cores):
        n = 1
        while True:                                 # grow the sample until it takes ~budget/4
            t0 = time.perf_counter()
            step = max(1, n // threads)
            with cf.ThreadPoolExecutor(threads) as ex:
                blocks = sum(ex.map(lambda i: run(i, min(i + step, n)), range(0, n, step)))
            dt = time.perf_counter() - t0
            if dt > budget_s / 4 or n >= b.n:
                break
            n = min(b.n, n * 4)
        out[f"oracle_digests_per_s_{threads}_threads"] = blocks / dt
    return out


def run_configs(args):
    """Per-kernel GPU rates (and the oracle's) on every workload at full size."""
    import torch

    import oracle
    from paper_2608_09225_gb300 import build as kbuild
    from paper_2608_09225_gb300 import kvgov as K
    from paper_2608_09225_gb300 import workloads as W
    from paper_2608_09225_gb300.pipeline import DeviceBatch, PrefixCache, next_pow2
    kbuild.build()
    oracle.build()
    K.lib()
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    micro = measure_int_peak(torch, kbuild.PEAK_LIB)
    peak = n_sm * max(micro["sha_msg96"], micro["sha_msg96_8w"]) * SM_MAX_MHZ * 1e6   # the SHA-256 ceiling
    cores = len(os.sched_getaffinity(0))
    l2 = torch.cuda.get_device_properties(0).L2_cache_size
    seed = args.seed
    scratch_table = K.new_table(1 << 25)
    gather = measure_gather(torch, kbuild.PEAK_LIB, scratch_table)
    del scratch_table
    round_cycles = measure_lone_warp_round(torch, kbuild.PEAK_LIB)
    print(json.dumps({"random_read_microbench": gather, "hbm_gbs": PEAKS.get("hbm_gbs"),
                      "lone_warp_cycles_per_round": round_cycles}), flush=True)
    only = set(args.only.split(",")) if args.only else None
    want = (lambda n: only is None or n in only)
    plan = []
    if want("tiny"):
        plan.append(("tiny", W.make("tiny"), W.ROOT))
    if want("sysprompt"):
        plan.append(("sysprompt", W.make("sysprompt"), W.ROOT))
    if want("template"):
        tmpl = W.make("template")
        plan += [("template", tmpl, m) for m in (W.UNSALTED, W.ROOT, W.BOUNDARY)]
    if want("probe"):
        plan.append(("probe", W.make("probe"), W.ROOT))
    if want("long"):
        plan.append(("long", W.make("long", seed=seed), W.BOUNDARY))
    if want("wide"):
        plan.append(("wide", W.make("wide", seed=seed + 1), W.BOUNDARY))
    names = {W.UNSALTED: "UNSALTED", W.ROOT: "ROOT", W.BOUNDARY: "BOUNDARY"}
    for name, w, mode in plan:
        b = w.batch
        nb_all = np.diff(K.count_blocks(b.tok_off)[1])     # blocks per request
        cap = w.capacity or next_pow2(4 * int(nb_all.sum()))
        cache = PrefixCache(cap, w.secret, w.ids, w.id_off)
        db = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
        n_blocks = db.n_blocks
        blk = torch.empty(b.n + 1, dtype=torch.int64, device="cuda")
        dig = torch.empty((n_blocks, 32), dtype=torch.uint8, device="cuda")
        pre = torch.empty(b.n, dtype=torch.int32, device="cuda")
        salted = mode != W.UNSALTED
        pr, sl, bt = (db.principal if salted else None), (cache.salts if salted else None), \
            (db.boundary_tok if mode == W.BOUNDARY else None)
        K.block_offsets(db.tok_off, blk)
        t_salts = _time(torch, lambda: K.derive_salts(w.secret, cache.ids, cache.id_off, cache.salts))
        t_blk = _time(torch, lambda: K.block_offsets(db.tok_off, blk))
        t_chain = _time(torch, lambda: K.chain_hash(mode, db.tokens, db.tok_off, blk, pr, sl, bt, dig))
        # the workload's table content
        blk_np = blk.cpu().numpy()
        fill_keys = []
        if w.fill_from == "prior":
            p = w.prior
            dp = DeviceBatch.from_host(p.tokens, p.tok_off, p.principal, p.boundary_tok)
            pblk = torch.empty(p.n + 1, dtype=torch.int64, device="cuda")
            K.block_offsets(dp.tok_off, pblk)
            pd = K.chain_hash(mode, dp.tokens, dp.tok_off, pblk, dp.principal if salted else None, sl,
                              dp.boundary_tok if mode == W.BOUNDARY else None, n_blocks=dp.n_blocks)
            fill_keys.append(pd)
        elif w.fill[1] > w.fill[0]:
            fill_keys.append(dig[blk_np[w.fill[0]]:blk_np[w.fill[1]]])
        else:                                    # long / wide: the first half of the batch
            fill_keys.append(dig[: blk_np[b.n // 2]])
        if w.random_keys is not None:
            fill_keys.append(torch.from_numpy(w.random_keys).cuda())
        keys = torch.cat(fill_keys)
        t_insert = _time(torch, lambda: (K.table_init(cache.slots), K.insert(cache.slots, keys, cache.status)),
                         reps=3, warm=1)
        t_init = _time(torch, lambda: K.table_init(cache.slots), reps=3, warm=1)
        K.insert(cache.slots, keys, cache.status)
        p0, p1 = w.probe if w.probe[1] > w.probe[0] else (0, b.n)
        pblk_view = blk[p0:p1 + 1]
        t_probe = _time(torch, lambda: K.probe(cache.slots, dig, pblk_view, pre[: p1 - p0]))
        t_fused = _time(torch, lambda: K.chain_hash_probe(mode, db.tokens, db.tok_off, blk, cache.slots, pr, sl, bt,
                                                          dig, pre))
        # divergence boundaries against the workload's registered shared preamble
        n_pre = {"tiny": 128, "sysprompt": 1024, "template": 96, "long": 64, "wide": 64}.get(name, 0)
        t0 = int(b.tok_off[0])
        pre_tok = db.tokens[t0:t0 + n_pre].contiguous() if n_pre else db.tokens[:4].contiguous()
        pre_off = torch.tensor([0, n_pre], dtype=torch.int64, device="cuda")
        tid = torch.full((b.n,), 0 if n_pre else K.TEMPLATE_NONE, dtype=torch.int32, device="cuda")
        bnd = torch.empty(b.n, dtype=torch.int32, device="cuda")
        t_bnd = _time(torch, lambda: K.divergence_boundary(db.tokens, db.tok_off, tid, pre_tok, pre_off, bnd,
                                                           cache.status))
        bnd_np = bnd.cpu().numpy()
        bnd_bytes = 4 * int(np.minimum(bnd_np + 1, b.lengths()).sum()) if n_pre else 0

        # exact-response keys of the whole prompts (salted when the workload is)
        rmode = W.UNSALTED if mode == W.UNSALTED else W.ROOT
        rkeys = torch.empty((b.n, 32), dtype=torch.uint8, device="cuda")
        t_resp = _time(torch, lambda: K.response_key(rmode, db.tokens, db.tok_off, db.principal, cache.salts, rkeys,
                                                     cache.status))
        resp_comp = int((((8 if rmode == W.ROOT else 0) + b.lengths() + 3 + 15) // 16).sum())

        # arrival order: the whole batch served request by request into an empty cache
        acap = next_pow2(4 * n_blocks)
        aslots, owner = K.new_table(acap), K.new_owner(acap)
        slot_of = torch.empty(n_blocks, dtype=torch.int32, device="cuda")
        pre_a = torch.empty(b.n, dtype=torch.int32, device="cuda")
        seq = [1]

        def arrival(probe=True):
            K.table_init(aslots)
            K.insert_arrival(aslots, owner, dig, blk, seq[0], cache.status, slot_of)
            if probe:
                K.probe_arrival(owner, slot_of, blk, seq[0], pre_a, cache.status)
            seq[0] += n_blocks

        def arrival_fused():
            K.table_init(aslots)
            K.chain_hash_arrival(mode, db.tokens, db.tok_off, blk, aslots, owner, seq[0], cache.status, pr, sl, bt,
                                 dig, slot_of, pre_a)
            seq[0] += n_blocks

        t_arr_fused = _time(torch, arrival_fused, reps=5, warm=1)
        t_arr = _time(torch, arrival, reps=5, warm=1)
        t_arr_ins = _time(torch, lambda: arrival(False), reps=5, warm=1)
        t_ainit = _time(torch, lambda: K.table_init(aslots), reps=5, warm=1)
        arrival()
        La = pre_a.cpu().numpy()
        del aslots, owner, slot_of
        torch.cuda.synchronize()
        cache.check_status()
        L = K.probe(cache.slots, dig, pblk_view).cpu().numpy()
        nb = np.diff(blk_np[p0:p1 + 1])
        algo_probes = int(np.minimum(L + 1, nb).sum())
        ops = nominal_chain_ops(nb_all, mode, b.boundary_tok // K.BLOCK)
        # algorithmic table bytes, linear probing at load factor a: a hit walks 1/2 (1 + 1/(1-a)) slots,
        # a miss 1/2 (1 + 1/(1-a)^2); a fill from empty to a averages 1/2 (1 + 1/(1-a)) per insert
        a = keys.shape[0] / cap
        hits = int(np.minimum(L, nb).sum())
        misses = int((L < nb).sum())
        probe_bytes = hits * (32 + 16 * (1 + 1 / (1 - a))) + misses * (32 + 16 * (1 + 1 / (1 - a) ** 2)) + 4 * (p1 - p0)
        insert_bytes = keys.shape[0] * (32 + 16 * (1 + 1 / (1 - a)) + 32)
        # floors: random slot bytes at the random-read ceiling, streamed bytes (digests, keys, results) at
        # the copy bandwidth
        probe_random = hits * 16 * (1 + 1 / (1 - a)) + misses * 16 * (1 + 1 / (1 - a) ** 2)
        probe_floor = 1e3 * (probe_random / (gather["gbs_32B"] * 1e9) +
                             (probe_bytes - probe_random) / (PEAKS["hbm_gbs"] * 1e9))
        insert_random = keys.shape[0] * (16 * (1 + 1 / (1 - a)) + 32)
        insert_floor = 1e3 * (insert_random / (gather["gbs_32B"] * 1e9) +
                              (insert_bytes - insert_random) / (PEAKS["hbm_gbs"] * 1e9))
        # a batch that leaves every round warp alone on its sub-partition (at most 64 chains
        # per SM) is bound by the latency of its longest chain: 2 compressions per block,
        # one more for a boundary block, 64 rounds each at the lone-warp round time
        k_all = b.boundary_tok // K.BLOCK
        comp = 2 * nb_all + ((k_all >= 1) & (k_all < nb_all) if mode == W.BOUNDARY else 0)
        lat_ms = (float(comp.max()) * 64 * round_cycles / (SM_MAX_MHZ * 1e3)
                  if 0 < b.n <= 64 * n_sm else None)
        line = {"workload": name, "mode": names[mode], "requests": b.n, "blocks": n_blocks,
                "table_slots": cap, "table_fits_l2": cap * 32 <= l2,
                "chain_ms": t_chain, "chain_digests_per_s": n_blocks / (t_chain / 1e3),
                "chain_tokens_per_s": 16 * n_blocks / (t_chain / 1e3),
                "chain_frac_sha256_ceiling": ops / (t_chain / 1e3) / peak,
                "chain_us_per_block_per_chain": 1e3 * t_chain / max(1, int(nb_all.max())),
                "chain_latency_bound_ms": lat_ms,
                "chain_frac_latency_bound": (lat_ms / t_chain) if lat_ms else None,
                "fused_chain_probe_ms": t_fused, "salts_ms": t_salts, "block_offsets_ms": t_blk,
                "probe_ms": t_probe, "probed_requests": p1 - p0, "algorithmic_probes": algo_probes,
                "probes_per_s": algo_probes / (t_probe / 1e3), "mean_prefix_blocks": float(L.mean()),
                "insert_keys": int(keys.shape[0]), "insert_ms": t_insert - t_init,
                "inserts_per_s": keys.shape[0] / ((t_insert - t_init) / 1e3), "load_factor": a,
                "probe_gbs": probe_bytes / (t_probe / 1e3) / 1e9,
                "probe_frac_hbm": probe_bytes / (t_probe / 1e3) / 1e9 / PEAKS["hbm_gbs"],
                "probe_floor_ms": probe_floor, "probe_frac_floor": probe_floor / t_probe,
                "response_key_ms": t_resp, "response_keys_per_s": b.n / (t_resp / 1e3),
                "response_tokens_per_s": float(b.lengths().sum()) / (t_resp / 1e3),
                "response_compressions": resp_comp,
                "response_frac_sha256_ceiling": resp_comp * 1384 / (t_resp / 1e3) / peak,
                "boundary_preamble_tokens": n_pre, "boundary_ms": t_bnd,
                "boundary_mean_tokens": float(bnd_np.mean()) if b.n else 0.0,
                "boundary_gbs": bnd_bytes / (t_bnd / 1e3) / 1e9,
                "arrival_insert_ms": t_arr_ins - t_ainit, "arrival_probe_ms": t_arr - t_arr_ins,
                "chain_arrival_ms": t_arr_fused - t_ainit,
                "chain_arrival_blocks_per_s": n_blocks / ((t_arr_fused - t_ainit) / 1e3),
                "arrival_blocks_per_s": n_blocks / ((t_arr - t_ainit) / 1e3),
                "arrival_mean_prefix_blocks": float(La.mean()),
                "arrival_hit_fraction": float(La.sum()) / max(1, n_blocks),
                "insert_gbs": insert_bytes / ((t_insert - t_init) / 1e3) / 1e9,
                "insert_floor_ms": insert_floor, "insert_frac_floor": insert_floor / (t_insert - t_init)}
        if not args.no_cpu_baseline:
            line.update(_oracle_rate(w, mode, cores))
            line["oracle_cores"] = cores
        print(json.dumps(line), flush=True)
        del cache, keys, dig
        torch.cuda.empty_cache()
    if want("audit"):
        print(json.dumps(audit_rates(torch, K, W, seed, cores, args.no_cpu_baseline)), flush=True)
    return 0


def audit_rates(torch, K, W, seed, cores, no_cpu):
    """ORIGAMI allocation (kvgov_origami) on 2^20 problems of the section 5.5
    setting: 50 tenants with Pareto(1.29) values, K = 10."""
    import oracle
    b = W.audit(seed=seed, n_prob=1 << 20)
    v = torch.from_numpy(b.values).cuda()
    off = torch.from_numpy(b.off).cuda()
    bud = torch.from_numpy(b.budget).cuda()
    p = torch.empty_like(v)
    lam = torch.empty(b.n, dtype=torch.float32, device="cuda")
    util = torch.empty(b.n, dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    t = _time(torch, lambda: K.origami(v, off, bud, p, lam, util, st))
    n_val = int(b.off[-1])
    bytes_ = 8 * n_val + 8 * (b.n + 1) + 12 * b.n         # values in, p out; offsets, budget, lambda, utility
    line = {"workload": "audit", "problems": b.n, "tenants_per_problem": 50, "budget": 10.0,
            "values": "Pareto(1.29), x_m = 1", "origami_ms": t, "problems_per_s": b.n / (t / 1e3),
            "gbs": bytes_ / (t / 1e3) / 1e9, "frac_hbm": bytes_ / (t / 1e3) / 1e9 / PEAKS["hbm_gbs"],
            "mean_lambda": float(lam.mean().item()), "status": int(st.item())}
    if not no_cpu:
        sample = W.audit(seed=seed, n_prob=1 << 16)
        t0 = time.perf_counter()
        oracle.origami(sample.values, sample.off, sample.budget)
        dt = time.perf_counter() - t0
        line["oracle_problems_per_s_1_thread"] = sample.n / dt
    return line


if __name__ == "__main__":
    sys.exit(main())
