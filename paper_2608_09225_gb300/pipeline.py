"""The hot path as one call sequence: salts -> blocking -> chain -> probe -> insert.

``PrefixCache`` owns the device-resident state of one KVGov prefix-cache
index (the slot table and the per-principal salts) and runs a batch of
requests through the library's kernels on one CUDA stream.
``DevicePipeline`` and ``HostPipeline`` serve a stream of batches (resident
on the device, or in pinned host memory) through the library's serving
engine (include/kvgov_pipeline.h), with each batch's salts, block offsets and
host-to-device copy overlapping the previous batch's kernels.  Nothing here
computes; every step is a libkvgov entry point (include/kvgov.h).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

from . import kvgov as K


def next_pow2(n: int) -> int:
    return 1 << max(int(n) - 1, 0).bit_length()


@dataclass
class DeviceBatch:
    """Device copies of one batch of requests (CSR tokens)."""
    tokens: torch.Tensor        # int32 [T]
    tok_off: torch.Tensor       # int64 [n + 1]
    principal: torch.Tensor     # int32 [n]
    boundary_tok: torch.Tensor  # int32 [n]
    n_blocks: int               # sum of floor(len / 16), known on the host

    @property
    def n(self) -> int:
        return self.tok_off.numel() - 1

    @staticmethod
    def from_host(tokens, tok_off, principal, boundary_tok, device="cuda", non_blocking=False) -> "DeviceBatch":
        tok_off_np = np.asarray(tok_off, dtype=np.int64)
        n_blocks, _ = K.count_blocks(tok_off_np)

        def put(a, dt):
            t = a if isinstance(a, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(a, dtype=dt))
            return t.to(device, non_blocking=non_blocking)

        return DeviceBatch(put(tokens, np.int32), put(tok_off_np, np.int64), put(principal, np.int32),
                           put(boundary_tok, np.int32), n_blocks)


class PrefixCache:
    """A GPU-resident block prefix-cache index with per-principal salts.

    capacity   main table slots (power of two, >= 32), 32 bytes each; the
               table also holds the side store's K.STASH_SLOTS slots.
    secret     the server secret K (HMAC key of section 4.1).
    ids/id_off principal-id bytes in CSR form (host numpy or device tensors).
    """

    def __init__(self, capacity: int, secret: bytes, ids, id_off, device="cuda", stream=None):
        self.device = torch.device(device)
        self.stream = stream
        self.capacity = int(capacity)
        self.secret = bytes(secret)
        self.ids = torch.as_tensor(np.asarray(ids, dtype=np.uint8)).to(self.device)
        self.id_off = torch.as_tensor(np.asarray(id_off, dtype=np.int64)).to(self.device)
        self.n_principals = self.id_off.numel() - 1
        self.salts = torch.empty((self.n_principals, 32), dtype=torch.uint8, device=self.device)
        self.slots = torch.empty((self.capacity + K.STASH_SLOTS, 32), dtype=torch.uint8, device=self.device)
        self.status = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.n_new = torch.zeros(1, dtype=torch.int64, device=self.device)
        self.gen = None        # the table's generations, made by the first one-launch engine on it
        K.table_init(self.slots, self.stream)
        self.derive_salts()

    def set_secret(self, secret: bytes):
        """Change the server secret; salts are derived again on the next serve."""
        self.secret = bytes(secret)

    # -- individual steps ------------------------------------------------
    def derive_salts(self):
        K.derive_salts(self.secret, self.ids, self.id_off, self.salts, self.status, self.stream)
        return self.salts

    def hash(self, mode: int, b: DeviceBatch, blk_off=None, digests=None):
        if blk_off is None:
            blk_off = torch.empty(b.n + 1, dtype=torch.int64, device=self.device)
        K.block_offsets(b.tok_off, blk_off, self.status, self.stream)
        if digests is None:
            digests = torch.empty((b.n_blocks, 32), dtype=torch.uint8, device=self.device)
        salted = mode != K.UNSALTED
        K.chain_hash(mode, b.tokens, b.tok_off, blk_off, b.principal if salted else None,
                     self.salts if salted else None, b.boundary_tok if mode == K.BOUNDARY else None,
                     digests, status=self.status, stream=self.stream)
        return blk_off, digests

    def insert(self, keys: torch.Tensor):
        K.insert(self.slots, keys, self.status, self.n_new, self.stream)

    def probe(self, digests, blk_off, prefix_blocks=None):
        return K.probe(self.slots, digests, blk_off, prefix_blocks, self.status, self.stream)

    def insert_uncached(self, digests, blk_off, prefix_blocks):
        K.insert_uncached(self.slots, digests, blk_off, prefix_blocks, self.status, self.n_new, self.stream)

    # -- one serving step -------------------------------------------------
    def serve(self, mode: int, b: DeviceBatch, bufs: dict | None = None, derive_salts: bool = True):
        """Salts, blocking, chain hash with the probe fused in, and insert of
        the uncached blocks for one batch.  Returns (prefix_blocks, digests,
        blk_off), on the device."""
        bufs = bufs if bufs is not None else {}
        if derive_salts:
            self.derive_salts()
        blk_off = bufs.get("blk_off")
        if blk_off is None:
            blk_off = torch.empty(b.n + 1, dtype=torch.int64, device=self.device)
        K.block_offsets(b.tok_off, blk_off, self.status, self.stream)
        salted = mode != K.UNSALTED
        digests, prefix = K.chain_hash_probe(mode, b.tokens, b.tok_off, blk_off, self.slots,
                                             b.principal if salted else None, self.salts if salted else None,
                                             b.boundary_tok if mode == K.BOUNDARY else None, bufs.get("digests"),
                                             bufs.get("prefix"), n_blocks=b.n_blocks, status=self.status,
                                             stream=self.stream)
        self.insert_uncached(digests, blk_off, prefix)
        return prefix, digests, blk_off

    def check_status(self):
        s = int(self.status.item()) & 0xFFFFFFFF
        if s:
            raise K.KVGovError(s, "device status")
        return s


class _Pipelined:
    """Buffers, events and streams of one serving engine (kvgov_pipeline.h),
    shared by DevicePipeline and HostPipeline.  The stream schedule itself
    -- batch i's salts and block offsets on a prep stream beside batch i-1's
    chain launch; on the compute stream (higher priority) the chain hash,
    the probe and the insert; slots reused only once free -- is the
    library's: one foreign call per batch (kvgov_pipeline_submit).

    insert_in_chain=True (default): batch i's chain hash runs in one launch
    with the insert of batch i-1's uncached blocks
    (kvgov_chain_hash_insert_prev), then batch i is probed against the table
    as batch i-1 left it; batch i's own insert waits for the next batch's
    chain launch (or drain()), and three slots rotate.
    insert_in_chain=False: the chain hash with the probe fused in, then the
    insert; two slots.
    one_launch=True (overrides insert_in_chain): batch i's lookups and its
    own insert in its chain launch (kvgov_chain_hash_serve), told apart by
    the table's generations (cache.gen); two slots, nothing left pending.
    The keys already in the cache count as cached from the first submit on;
    after that the cache must change only through this pipeline.

    Either way every probe sees the table exactly as the previous batch's
    insert left it.  A flush (submit(..., flush=True)) first runs a pending
    insert, then empties the table.  Nothing here computes.
    """

    def __init__(self, cache: PrefixCache, mode: int, max_req: int, max_blocks: int, device="cuda",
                 insert_in_chain: bool = True, one_launch: bool = False):
        self.cache, self.mode = cache, mode
        self.device = torch.device(device)
        self.one_launch = one_launch
        self.insert_in_chain = insert_in_chain and not one_launch
        schedule = K.SCHEDULE_ONE_LAUNCH if one_launch else int(bool(insert_in_chain))
        if one_launch and getattr(cache, "gen", None) is None:
            cache.gen = K.new_gen(cache.slots)       # the table's generations, zeroed with it
        self.prep_stream = torch.cuda.Stream(self.device)
        self.compute_stream = torch.cuda.Stream(self.device, priority=-1)
        cache.stream = self.compute_stream
        n_slots = 3 if schedule == 1 else 2
        self.slots = []
        for _ in range(n_slots):
            self.slots.append({
                "salts": torch.empty((max(cache.n_principals, 1), 32), dtype=torch.uint8, device=self.device),
                "blk_off": torch.empty(max_req + 1, dtype=torch.int64, device=self.device),
                "digests": torch.empty((max(max_blocks, 1), 32), dtype=torch.uint8, device=self.device),
                "prefix": torch.empty(max(max_req, 1), dtype=torch.int32, device=self.device),
                "prepared": torch.cuda.Event(), "chain_start": torch.cuda.Event(), "probed": torch.cuda.Event(),
                "free": torch.cuda.Event(),
            })
        d = K.PipelineDesc()
        d.mode, d.insert_in_chain, d.n_slots = int(mode), schedule, n_slots
        d.max_req, d.max_blocks = int(max_req), int(max_blocks)
        d.d_slots, d.capacity = cache.slots.data_ptr(), cache.capacity
        d.d_status, d.d_n_new = cache.status.data_ptr(), cache.n_new.data_ptr()
        d.d_ids, d.d_id_off, d.n_principals = cache.ids.data_ptr(), cache.id_off.data_ptr(), cache.n_principals
        cs = self.compute_stream
        for i, sl in enumerate(self.slots):
            d.d_salts[i], d.d_blk_off[i] = sl["salts"].data_ptr(), sl["blk_off"].data_ptr()
            d.d_digests[i], d.d_prefix[i] = sl["digests"].data_ptr(), sl["prefix"].data_ptr()
            d.prepared[i] = K.event_handle(sl["prepared"], cs)
            d.chain_start[i] = K.event_handle(sl["chain_start"], cs)
            d.probed[i] = K.event_handle(sl["probed"], cs)
            d.free_ev[i] = K.event_handle(sl["free"], cs)
        d.prep_stream, d.compute_stream = self.prep_stream.cuda_stream, cs.cuda_stream
        d.d_gen = cache.gen.data_ptr() if one_launch else None
        self.engine = K.Engine(d)
        self._after = [torch.cuda.Event() for _ in self.slots]
        self._i = 0

    @property
    def pending(self) -> bool:
        return self.engine.pending()

    def drain(self):
        """Run the pending insert, if any; returns an event recorded after it
        on the compute stream."""
        self.engine.drain()
        ev = torch.cuda.Event()
        ev.record(self.compute_stream)
        return ev

    def _submit(self, db: DeviceBatch, after: torch.cuda.Event, flush: bool, chain_events, table_events) -> int:
        cs = self.compute_stream
        ce = tuple(K.event_handle(e, cs) for e in chain_events) if chain_events is not None else (None, None)
        te = tuple(K.event_handle(e, cs) for e in table_events) if table_events is not None else (None, None)
        salted = self.mode != K.UNSALTED
        return self.engine.submit(self.cache.secret, db.tokens.data_ptr(), db.tok_off.data_ptr(), db.n,
                                  db.principal.data_ptr() if salted else None,
                                  db.boundary_tok.data_ptr() if self.mode == K.BOUNDARY else None,
                                  db.n_blocks, K.event_handle(after, cs), flush, ce, te)


class DevicePipeline(_Pipelined):
    """Serve device-resident batches back to back through the library's
    serving engine (see _Pipelined).

    submit() returns (prefix_blocks, event) on the device: prefix_blocks is
    valid once event has completed and is overwritten by a later submit (the
    second or third after it).  The batch's uncached blocks are in the table
    once the next submit's chain launch or drain() has run (with one_launch,
    once its own chain launch has: when the event has completed).  The batch's
    tensors are used on the pipeline's streams after the work queued so far
    on the caller's current stream.
    """

    def submit(self, db: DeviceBatch, flush: bool = False, chain_events=None, table_events=None):
        """Queue one device-resident batch.  flush empties the cache before
        it (after any pending insert).  chain_events and table_events, pairs
        of CUDA events, are recorded around the chain-hash launch and the
        table kernel after it (the probe, or the insert)."""
        after = self._after[self._i % len(self._after)]
        self._i += 1
        after.record(torch.cuda.current_stream(self.device))
        for t in (db.tokens, db.tok_off, db.principal, db.boundary_tok):
            t.record_stream(self.prep_stream)
            t.record_stream(self.compute_stream)
        slot = self._submit(db, after, flush, chain_events, table_events)
        sl = self.slots[slot]
        return sl["prefix"][:db.n], sl["probed"]


class HostPipeline(_Pipelined):
    """Serve batches that live in pinned host memory: each batch's
    host-to-device copy runs on a copy stream while the previous batch is
    served, then the library's serving engine serves it (see _Pipelined) and
    an output stream copies its prefix lengths back into a pinned host buffer
    once its probe is done.  A slot's buffers are reused only after its
    batch has been inserted and its output copied.

    submit() returns (prefix_host, event): prefix_host is valid once event has
    completed (event.synchronize()) and is overwritten by a later submit (the
    second or third after it).
    """

    def __init__(self, cache: PrefixCache, mode: int, max_req: int, max_tokens: int, device="cuda",
                 insert_in_chain: bool = True, one_launch: bool = False):
        max_blocks, _ = K.count_blocks([0, max_tokens])        # no batch of max_tokens tokens has more
        super().__init__(cache, mode, max_req, max_blocks, device, insert_in_chain, one_launch)
        self.copy_stream = torch.cuda.Stream(self.device)
        self.out_stream = torch.cuda.Stream(self.device)
        for s in self.slots:
            s.update({
                "tokens": torch.empty(max(max_tokens, 4), dtype=torch.int32, device=self.device),
                "tok_off": torch.empty(max_req + 1, dtype=torch.int64, device=self.device),
                "principal": torch.empty(max(max_req, 1), dtype=torch.int32, device=self.device),
                "boundary_tok": torch.empty(max(max_req, 1), dtype=torch.int32, device=self.device),
                "out": torch.empty(max(max_req, 1), dtype=torch.int32).pin_memory(),
                "copied": torch.cuda.Event(), "out_done": torch.cuda.Event(), "used": False,
            })

    def submit(self, tokens, tok_off, principal, boundary_tok, n_blocks: int, flush: bool = False,
               chain_events=None):
        """Queue one batch given as pinned host tensors (int32 tokens, int64
        offsets, int32 principal rows and boundary offsets).  flush empties
        the cache before it (after any pending insert); chain_events as in
        DevicePipeline.submit."""
        s = self.slots[self._i % len(self.slots)]   # the slot the engine gives this batch
        n, t = tok_off.numel() - 1, tokens.numel()
        with torch.cuda.stream(self.copy_stream):
            if s["used"]:
                self.copy_stream.wait_event(s["free"])
                self.copy_stream.wait_event(s["out_done"])
            s["tokens"][:t].copy_(tokens, non_blocking=True)
            s["tok_off"][:n + 1].copy_(tok_off, non_blocking=True)
            s["principal"][:n].copy_(principal, non_blocking=True)
            s["boundary_tok"][:n].copy_(boundary_tok, non_blocking=True)
            s["copied"].record(self.copy_stream)
        db = DeviceBatch(s["tokens"][:max(t, 4)], s["tok_off"][:n + 1], s["principal"][:n],
                         s["boundary_tok"][:n], n_blocks)
        self._i += 1
        slot = self._submit(db, s["copied"], flush, chain_events, None)
        assert self.slots[slot] is s
        with torch.cuda.stream(self.out_stream):
            self.out_stream.wait_event(s["probed"])
            s["out"][:n].copy_(s["prefix"][:n], non_blocking=True)
            s["out_done"].record(self.out_stream)
        s["used"] = True
        return s["out"][:n], s["out_done"]
