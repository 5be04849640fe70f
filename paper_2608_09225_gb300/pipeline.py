"""The hot path as one call sequence: salts -> blocking -> chain -> probe -> insert.

``PrefixCache`` owns the device-resident state of one KVGov prefix-cache
index (the slot table and the per-principal salts) and runs a batch of
requests through the library's kernels on one CUDA stream.
``DevicePipeline`` and ``HostPipeline`` serve a stream of batches (resident
on the device, or in pinned host memory) with each batch's salts, block
offsets and host-to-device copy overlapping the previous batch's kernels.
Nothing here computes; every step is a libkvgov entry point (include/kvgov.h).
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
        n_blocks = int((np.diff(tok_off_np) // K.BLOCK).sum())

        def put(a, dt):
            t = a if isinstance(a, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(a, dtype=dt))
            return t.to(device, non_blocking=non_blocking)

        return DeviceBatch(put(tokens, np.int32), put(tok_off_np, np.int64), put(principal, np.int32),
                           put(boundary_tok, np.int32), n_blocks)


class PrefixCache:
    """A GPU-resident block prefix-cache index with per-principal salts.

    capacity   table slots (power of two, >= 32), 32 bytes each.
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
        self.slots = torch.empty((self.capacity, 32), dtype=torch.uint8, device=self.device)
        self.status = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.n_new = torch.zeros(1, dtype=torch.int64, device=self.device)
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
    """Per-batch device buffers in rotating slots and the stream schedule
    shared by DevicePipeline and HostPipeline.

    Batch i's salts (under the secret current when it is submitted) and block
    offsets are computed on a prep stream once batch i-1's chain hash has
    started, so their small CTAs run in the room the chain kernel leaves on
    the SMs instead of in front of batch i's chain hash.  The compute stream
    (higher priority, so its CTAs are placed first) then serves the batch:

    insert_in_chain=True (default): batch i's chain hash runs in one launch
    with the insert of batch i-1's uncached blocks
    (kvgov_chain_hash_insert_prev), then batch i is probed against the table
    as batch i-1 left it.  Batch i's own insert is left pending for the next
    batch's chain launch (or drain()); three slots rotate, since batch i's
    buffers are read by batch i+1's chain launch while batch i+2 is prepared.

    insert_in_chain=False: the chain hash with the probe fused in, then the
    insert of the uncached blocks; two slots.

    Either way every probe sees the table exactly as the previous batch's
    insert left it, and every step runs on the GPU; nothing here computes.
    A cache flush (before_serve) first runs a pending insert, so that the
    flush follows it.
    """

    def __init__(self, cache: PrefixCache, mode: int, max_req: int, max_blocks: int, device="cuda",
                 insert_in_chain: bool = True):
        self.cache, self.mode = cache, mode
        self.device = torch.device(device)
        self.insert_in_chain = insert_in_chain
        self.prep_stream = torch.cuda.Stream(self.device)
        self.compute_stream = torch.cuda.Stream(self.device, priority=-1)
        cache.stream = self.compute_stream
        self.slots = []
        for _ in range(3 if insert_in_chain else 2):
            self.slots.append({
                "salts": torch.empty((max(cache.n_principals, 1), 32), dtype=torch.uint8, device=self.device),
                "blk_off": torch.empty(max_req + 1, dtype=torch.int64, device=self.device),
                "digests": torch.empty((max(max_blocks, 1), 32), dtype=torch.uint8, device=self.device),
                "prefix": torch.empty(max(max_req, 1), dtype=torch.int32, device=self.device),
                "prepared": torch.cuda.Event(), "chain_start": torch.cuda.Event(), "probed": torch.cuda.Event(),
                "free": torch.cuda.Event(), "used": False, "n": 0, "n_blocks": 0,
            })
        self.i = 0
        self.last_chain_start = None
        self.pending = None          # the slot whose batch's insert has not run yet

    def _next_slot(self):
        s = self.slots[self.i % len(self.slots)]
        self.i += 1
        return s

    def _prepare(self, s, db: DeviceBatch, after=None):
        """Salts and block offsets of one batch on the prep stream."""
        c = self.cache
        ps = self.prep_stream
        if after is not None:
            ps.wait_event(after)
        if self.last_chain_start is not None:
            ps.wait_event(self.last_chain_start)    # start beside the previous batch's chain hash
        if s["used"]:
            ps.wait_event(s["free"])                # the slot's previous batch has been inserted
        if self.mode != K.UNSALTED:
            K.derive_salts(c.secret, c.ids, c.id_off, s["salts"], c.status, ps)
        K.block_offsets(db.tok_off, s["blk_off"][:db.n + 1], c.status, ps)
        s["prepared"].record(ps)

    def _views(self, s):
        return s["blk_off"][:s["n"] + 1], s["digests"][:s["n_blocks"]], s["prefix"][:s["n"]]

    def _insert_pending(self):
        """The pending batch's insert as its own launch (compute stream)."""
        q = self.pending
        if q is None:
            return
        c = self.cache
        blk, dig, pre = self._views(q)
        K.insert_uncached(c.slots, dig, blk, pre, c.status, c.n_new, self.compute_stream)
        q["free"].record(self.compute_stream)
        self.pending = None

    def drain(self):
        """Run the pending insert, if any; returns an event recorded after it
        on the compute stream."""
        with torch.cuda.stream(self.compute_stream):
            self._insert_pending()
        ev = torch.cuda.Event()
        ev.record(self.compute_stream)
        return ev

    def _serve(self, s, db: DeviceBatch, before_serve=None, chain_events=None, table_events=None):
        """Serve one batch on the compute stream (see the class docstring).
        chain_events are recorded around the chain-hash launch, table_events
        around the batch's table kernel after it: the probe (when the chain
        launch carried the previous batch's insert) or the insert
        (insert_in_chain=False)."""
        c = self.cache
        cs = self.compute_stream
        n = db.n
        s["n"], s["n_blocks"] = n, db.n_blocks
        blk_off, digests, prefix = self._views(s)
        salted = self.mode != K.UNSALTED
        kw = dict(principal=db.principal if salted else None, salts=s["salts"] if salted else None,
                  boundary_tok=db.boundary_tok if self.mode == K.BOUNDARY else None, digests=digests,
                  stream=cs)
        with torch.cuda.stream(cs):
            cs.wait_event(s["prepared"])
            if before_serve is not None:
                self._insert_pending()
                before_serve()
            if chain_events is not None:
                chain_events[0].record(cs)
            # the last command before the chain launch: the prep of the next
            # batch starts only once the chain kernel is being placed
            s["chain_start"].record(cs)
            self.last_chain_start = s["chain_start"]
            q = self.pending if self.insert_in_chain else None
            if q is not None:
                qb, qd, qp = self._views(q)
                K.chain_hash_insert_prev(self.mode, db.tokens, db.tok_off, blk_off, c.slots, qd, qb, qp, c.status,
                                         n_new=c.n_new, **kw)
            else:
                K.chain_hash_probe(self.mode, db.tokens, db.tok_off, blk_off, c.slots, prefix_blocks=prefix,
                                   n_blocks=db.n_blocks, status=c.status, **kw)
            if chain_events is not None:
                chain_events[1].record(cs)
            if q is not None:
                if table_events is not None:
                    table_events[0].record(cs)
                K.probe(c.slots, digests, blk_off, prefix, c.status, cs)
                if table_events is not None:
                    table_events[1].record(cs)
            if q is not None:
                q["free"].record(cs)
                self.pending = None
            if not self.insert_in_chain:
                if table_events is not None:
                    table_events[0].record(cs)
                K.insert_uncached(c.slots, digests, blk_off, prefix, c.status, c.n_new, cs)
                if table_events is not None:
                    table_events[1].record(cs)
            s["probed"].record(cs)
            if self.insert_in_chain:
                self.pending = s
            else:
                s["free"].record(cs)
        s["used"] = True
        return prefix, digests, blk_off


class DevicePipeline(_Pipelined):
    """Serve device-resident batches back to back, each batch's salts and
    block offsets computed beside the previous batch's chain hash and (by
    default) its insert run inside the next batch's chain launch.

    submit() returns (prefix_blocks, event) on the device: prefix_blocks is
    valid once event has completed and is overwritten by a later submit (the
    second or third after it).  The batch's uncached blocks are in the table
    once the next submit's chain launch or drain() has run.  The batch's
    tensors are used on the pipeline's streams after the work queued so far
    on the caller's current stream.
    """

    def __init__(self, cache: PrefixCache, mode: int, max_req: int, max_blocks: int, device="cuda",
                 insert_in_chain: bool = True):
        super().__init__(cache, mode, max_req, max_blocks, device, insert_in_chain)
        self._ready = [torch.cuda.Event() for _ in self.slots]

    def submit(self, db: DeviceBatch, before_serve=None, chain_events=None, table_events=None):
        """Queue one device-resident batch.  before_serve, if given, is called
        with the compute stream current just before the chain hash, after any
        pending insert (for instance to flush the cache); chain_events and
        table_events, pairs of CUDA events, are recorded around the
        chain-hash launch and the table kernel after it (the probe, or the
        insert)."""
        ready = self._ready[self.i % len(self.slots)]
        ready.record(torch.cuda.current_stream(self.device))
        for t in (db.tokens, db.tok_off, db.principal, db.boundary_tok):
            t.record_stream(self.prep_stream)
            t.record_stream(self.compute_stream)
        self.compute_stream.wait_event(ready)
        s = self._next_slot()
        self._prepare(s, db, after=ready)
        prefix, _, _ = self._serve(s, db, before_serve, chain_events, table_events)
        return prefix, s["probed"]


class HostPipeline(_Pipelined):
    """Serve batches that live in pinned host memory: each batch's
    host-to-device copy runs on a copy stream while the previous batch is
    served, its salts and block offsets follow on the prep stream, the
    compute stream serves it as in DevicePipeline and copies its prefix
    lengths back into a pinned host buffer.  A slot's buffers are reused
    only after its batch has been inserted.

    submit() returns (prefix_host, event): prefix_host is valid once event has
    completed (event.synchronize()) and is overwritten by a later submit (the
    second or third after it).
    """

    def __init__(self, cache: PrefixCache, mode: int, max_req: int, max_tokens: int, device="cuda",
                 insert_in_chain: bool = True):
        super().__init__(cache, mode, max_req, max_tokens // K.BLOCK, device, insert_in_chain)
        self.copy_stream = torch.cuda.Stream(self.device)
        for s in self.slots:
            s.update({
                "tokens": torch.empty(max(max_tokens, 4), dtype=torch.int32, device=self.device),
                "tok_off": torch.empty(max_req + 1, dtype=torch.int64, device=self.device),
                "principal": torch.empty(max(max_req, 1), dtype=torch.int32, device=self.device),
                "boundary_tok": torch.empty(max(max_req, 1), dtype=torch.int32, device=self.device),
                "out": torch.empty(max(max_req, 1), dtype=torch.int32).pin_memory(),
                "copied": torch.cuda.Event(), "out_done": torch.cuda.Event(),
            })

    def submit(self, tokens, tok_off, principal, boundary_tok, n_blocks: int, before_serve=None,
               chain_events=None):
        """Queue one batch given as pinned host tensors (int32 tokens, int64
        offsets, int32 principal rows and boundary offsets).  before_serve, if
        given, is called with the compute stream current just before the
        chain hash, after any pending insert (for instance to flush the
        cache); chain_events as in DevicePipeline.submit."""
        s = self._next_slot()
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
        self._prepare(s, db, after=s["copied"])
        prefix, _, _ = self._serve(s, db, before_serve, chain_events)
        with torch.cuda.stream(self.compute_stream):
            s["out"][:n].copy_(prefix, non_blocking=True)
            s["out_done"].record(self.compute_stream)
        return s["out"][:n], s["out_done"]
