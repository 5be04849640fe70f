"""The hot path as one call sequence: salts -> blocking -> chain -> probe -> insert.

``PrefixCache`` owns the device-resident state of one KVGov prefix-cache
index (the slot table and the per-principal salts) and runs a batch of
requests through the library's kernels on one CUDA stream.  Nothing here
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


class HostPipeline:
    """Serve batches that live in pinned host memory, overlapping each batch's
    host-to-device copy with the serving of the previous one.

    Two device input slots alternate: ``submit`` copies the batch into the next
    slot on a copy stream, and the compute stream serves it (salts, blocking,
    chain hash with the fused probe, insert) once that copy has landed, then
    copies the prefix lengths back into a pinned host buffer.  A slot is reused
    only after the compute stream has finished with it.

    submit() returns (prefix_host, event): prefix_host is valid once event has
    completed (event.synchronize()) and is overwritten two submits later.
    Every step runs on the GPU; nothing here computes.
    """

    def __init__(self, cache: PrefixCache, mode: int, max_req: int, max_tokens: int, device="cuda"):
        self.cache, self.mode = cache, mode
        dev = torch.device(device)
        self.copy_stream = torch.cuda.Stream(dev)
        self.compute_stream = torch.cuda.Stream(dev)
        cache.stream = self.compute_stream
        max_blocks = max_tokens // K.BLOCK
        self.slots = []
        for _ in range(2):
            self.slots.append({
                "tokens": torch.empty(max(max_tokens, 4), dtype=torch.int32, device=dev),
                "tok_off": torch.empty(max_req + 1, dtype=torch.int64, device=dev),
                "principal": torch.empty(max(max_req, 1), dtype=torch.int32, device=dev),
                "boundary_tok": torch.empty(max(max_req, 1), dtype=torch.int32, device=dev),
                "blk_off": torch.empty(max_req + 1, dtype=torch.int64, device=dev),
                "digests": torch.empty((max(max_blocks, 1), 32), dtype=torch.uint8, device=dev),
                "prefix": torch.empty(max(max_req, 1), dtype=torch.int32, device=dev),
                "out": torch.empty(max(max_req, 1), dtype=torch.int32).pin_memory(),
                "copied": torch.cuda.Event(), "free": torch.cuda.Event(), "used": False,
            })
        self.i = 0

    def submit(self, tokens, tok_off, principal, boundary_tok, n_blocks: int, before_serve=None):
        """Queue one batch given as pinned host tensors (int32 tokens, int64
        offsets, int32 principal rows and boundary offsets).  before_serve, if
        given, is called with the compute stream current just before serving
        (for instance to flush the cache)."""
        s = self.slots[self.i % 2]
        self.i += 1
        n, t = tok_off.numel() - 1, tokens.numel()
        with torch.cuda.stream(self.copy_stream):
            if s["used"]:
                self.copy_stream.wait_event(s["free"])
            s["tokens"][:t].copy_(tokens, non_blocking=True)
            s["tok_off"][:n + 1].copy_(tok_off, non_blocking=True)
            s["principal"][:n].copy_(principal, non_blocking=True)
            s["boundary_tok"][:n].copy_(boundary_tok, non_blocking=True)
            s["copied"].record(self.copy_stream)
        s["used"] = True
        with torch.cuda.stream(self.compute_stream):
            self.compute_stream.wait_event(s["copied"])
            if before_serve is not None:
                before_serve()
            db = DeviceBatch(s["tokens"][:max(t, 4)], s["tok_off"][:n + 1], s["principal"][:n],
                             s["boundary_tok"][:n], n_blocks)
            bufs = {"blk_off": s["blk_off"][:n + 1], "digests": s["digests"][:n_blocks], "prefix": s["prefix"][:n]}
            prefix, _, _ = self.cache.serve(self.mode, db, bufs)
            s["out"][:n].copy_(prefix, non_blocking=True)
            s["free"].record(self.compute_stream)
        return s["out"][:n], s["free"]
