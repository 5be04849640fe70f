"""ctypes binding of libkvgov (include/kvgov.h).

Argument marshalling only: every function checks tensor devices, dtypes and
contiguity, passes raw device pointers and the current torch CUDA stream to the
C entry point of the same name, and raises KVGovError on a non-zero return.
All work runs in the library's CUDA kernels; there is no CPU path.  If the
library is missing or CUDA is unavailable the first call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

UNSALTED, ROOT, BOUNDARY = 0, 1, 2
BLOCK = 16
DIGEST_BYTES = 32
MAX_SECRET = 1024
MIN_CAPACITY = 32
STASH_SLOTS = 64          # slots after the capacity main ones: the table's side store
STASH_KEYS = 56

OK, EINVAL, ECUDA = 0, 1, 2
F_BADINDEX, F_SENTINEL, F_TABLE_FULL, F_TIMEOUT = 0x10, 0x20, 0x40, 0x80
TEMPLATE_NONE, TEMPLATE_ANY = -1, -2

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libkvgov.so")
_lock = threading.Lock()
_lib = None

_p = ctypes.c_void_p


MAX_SLOTS = 3
SCHEDULE_ONE_LAUNCH = 2   # kvgov_pipeline_desc.insert_in_chain: KVGOV_SCHEDULE_ONE_LAUNCH
_S3 = _p * MAX_SLOTS


class PipelineDesc(ctypes.Structure):
    """kvgov_pipeline_desc (include/kvgov_pipeline.h)."""
    _fields_ = [("mode", ctypes.c_int), ("insert_in_chain", ctypes.c_int), ("n_slots", ctypes.c_int),
                ("max_req", ctypes.c_int32), ("max_blocks", ctypes.c_int64),
                ("d_slots", _p), ("capacity", ctypes.c_uint64), ("d_status", _p), ("d_n_new", _p),
                ("d_ids", _p), ("d_id_off", _p), ("n_principals", ctypes.c_int32),
                ("d_salts", _S3), ("d_blk_off", _S3), ("d_digests", _S3), ("d_prefix", _S3),
                ("prepared", _S3), ("chain_start", _S3), ("probed", _S3), ("free_ev", _S3),
                ("prep_stream", _p), ("compute_stream", _p), ("d_gen", _p)]


class KVGovError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status) if _lib is not None else status}")


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not torch.cuda.is_available():
            raise RuntimeError("libkvgov needs a CUDA device; none is available (no CPU fallback)")
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libkvgov.so is not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        L.kvgov_status_string.argtypes = [ctypes.c_int]
        L.kvgov_status_string.restype = ctypes.c_char_p
        L.kvgov_block_offsets.argtypes = [_p, ctypes.c_int32, _p, _p, _p]
        L.kvgov_count_blocks.argtypes = [_p, ctypes.c_int32, _p, _p]
        L.kvgov_derive_salts.argtypes = [_p, ctypes.c_size_t, _p, _p, ctypes.c_int32, _p, _p, _p]
        L.kvgov_chain_hash.argtypes = [ctypes.c_int, _p, _p, ctypes.c_int32, _p, _p, ctypes.c_int32, _p, _p, _p,
                                       _p, _p]
        L.kvgov_chain_hash_probe.argtypes = [ctypes.c_int, _p, _p, ctypes.c_int32, _p, _p, ctypes.c_int32, _p, _p,
                                             _p, _p, ctypes.c_uint64, _p, _p, _p]
        L.kvgov_chain_hash_insert_prev.argtypes = [ctypes.c_int, _p, _p, ctypes.c_int32, _p, _p, ctypes.c_int32,
                                                   _p, _p, _p, _p, ctypes.c_uint64, _p, _p, ctypes.c_int32, _p, _p,
                                                   _p, _p, _p]
        L.kvgov_table_init.argtypes = [_p, ctypes.c_uint64, _p]
        L.kvgov_table_gen_stamp.argtypes = [_p, ctypes.c_uint64, _p, ctypes.c_uint32, _p]
        L.kvgov_chain_hash_serve.argtypes = [ctypes.c_int, _p, _p, ctypes.c_int32, _p, _p, ctypes.c_int32, _p, _p, _p,
                                             _p, ctypes.c_uint64, _p, ctypes.c_uint32, ctypes.c_uint32, _p, _p, _p,
                                             _p]
        L.kvgov_insert.argtypes = [_p, ctypes.c_uint64, _p, ctypes.c_int64, _p, _p, _p]
        L.kvgov_probe.argtypes = [_p, ctypes.c_uint64, _p, _p, ctypes.c_int32, _p, _p, _p]
        L.kvgov_probe_resume.argtypes = [_p, ctypes.c_uint64, _p, _p, ctypes.c_int32, _p, _p, _p]
        L.kvgov_insert_uncached.argtypes = [_p, ctypes.c_uint64, _p, _p, ctypes.c_int32, _p, _p, _p, _p]
        L.kvgov_owner_init.argtypes = [_p, ctypes.c_uint64, _p]
        L.kvgov_insert_arrival.argtypes = [_p, _p, ctypes.c_uint64, _p, _p, ctypes.c_int32, ctypes.c_uint64, _p, _p,
                                           _p, _p]
        L.kvgov_probe_arrival.argtypes = [_p, ctypes.c_uint64, _p, _p, ctypes.c_int32, ctypes.c_uint64, _p, _p, _p]
        L.kvgov_chain_hash_arrival.argtypes = [ctypes.c_int, _p, _p, ctypes.c_int32, _p, _p, ctypes.c_int32, _p, _p,
                                               _p, _p, _p, ctypes.c_uint64, ctypes.c_uint64, _p, _p, _p, _p, _p]
        L.kvgov_divergence_boundary.argtypes = [_p, _p, ctypes.c_int32, _p, _p, _p, ctypes.c_int32, _p, _p, _p]
        L.kvgov_response_key.argtypes = [ctypes.c_int, _p, _p, ctypes.c_int32, _p, _p, ctypes.c_int32, _p, _p, _p]
        L.kvgov_origami.argtypes = [_p, _p, ctypes.c_int32, _p, _p, _p, _p, _p, _p]
        L.kvgov_serve_arrival_static.argtypes = [_p, _p, ctypes.c_uint64, _p, _p, ctypes.c_int32, ctypes.c_int64,
                                                 ctypes.c_uint64, _p, _p, _p, _p]
        L.kvgov_set_spin_limit.argtypes = [ctypes.c_uint32]
        L.kvgov_set_spin_limit.restype = ctypes.c_uint32
        L.kvgov_pipeline_create.argtypes = [ctypes.POINTER(PipelineDesc), ctypes.POINTER(_p)]
        L.kvgov_pipeline_submit.argtypes = [_p, ctypes.c_char_p, ctypes.c_size_t, _p, _p, ctypes.c_int32, _p, _p,
                                            ctypes.c_int64, _p, ctypes.c_int, _p, _p, _p, _p,
                                            ctypes.POINTER(ctypes.c_int32)]
        L.kvgov_pipeline_drain.argtypes = [_p]
        L.kvgov_pipeline_pending.argtypes = [_p]
        L.kvgov_pipeline_destroy.argtypes = [_p]
        L.kvgov_pipeline_destroy.restype = None
        for fn in ("kvgov_block_offsets", "kvgov_count_blocks", "kvgov_derive_salts", "kvgov_chain_hash", "kvgov_table_init",
                   "kvgov_insert", "kvgov_probe", "kvgov_probe_resume", "kvgov_insert_uncached",
                   "kvgov_table_gen_stamp", "kvgov_chain_hash_serve",
                   "kvgov_chain_hash_probe",
                   "kvgov_owner_init", "kvgov_insert_arrival", "kvgov_probe_arrival", "kvgov_chain_hash_arrival",
                   "kvgov_divergence_boundary", "kvgov_response_key", "kvgov_origami",
                   "kvgov_serve_arrival_static", "kvgov_pipeline_create", "kvgov_pipeline_submit",
                   "kvgov_pipeline_drain", "kvgov_pipeline_pending"):
            getattr(L, fn).restype = ctypes.c_int
        _lib = L
        return L


def lib():
    return _lib if _lib is not None else _load()


def status_string(status: int) -> str:
    return lib().kvgov_status_string(int(status)).decode()


def _check(rc: int, where: str):
    if rc != OK:
        raise KVGovError(rc, where)


def _dev(t: torch.Tensor | None, dtype, name: str, allow_none: bool = False):
    if t is None:
        if allow_none:
            return None
        raise ValueError(f"{name} is required")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr() if t.numel() else None


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def capacity_of(slots: torch.Tensor) -> int:
    """The capacity of a table tensor: its rows minus the side store's."""
    return slots.shape[0] - STASH_SLOTS


def _owner_capacity(owner: torch.Tensor) -> int:
    return owner.numel() - STASH_SLOTS


def block_offsets(tok_off: torch.Tensor, blk_off: torch.Tensor | None = None,
                  status: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """blk_off[r+1] - blk_off[r] = floor(len_r / 16) (paper section 2.1)."""
    L = lib()
    n = tok_off.numel() - 1
    if blk_off is None:
        blk_off = torch.empty(n + 1, dtype=torch.int64, device=tok_off.device)
    _check(L.kvgov_block_offsets(_dev(tok_off, torch.int64, "tok_off"), n,
                                 _dev(blk_off, torch.int64, "blk_off"),
                                 _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_block_offsets")
    return blk_off


def count_blocks(tok_off) -> tuple[int, "np.ndarray"]:
    """kvgov_count_blocks on host offsets (numpy or a CPU tensor): the batch's
    block count and its block offsets, as kvgov_block_offsets computes them."""
    import numpy as np
    off = np.ascontiguousarray(tok_off.cpu().numpy() if isinstance(tok_off, torch.Tensor) else tok_off,
                               dtype=np.int64)
    n = off.size - 1
    blk = np.empty(max(n, 0) + 1, dtype=np.int64)
    total = ctypes.c_int64(0)
    if n < 0:
        raise ValueError("tok_off needs at least one entry")
    _check(lib().kvgov_count_blocks(off.ctypes.data, n, blk.ctypes.data, ctypes.byref(total)), "kvgov_count_blocks")
    return int(total.value), blk


def derive_salts(secret: bytes, ids: torch.Tensor, id_off: torch.Tensor, salts: torch.Tensor | None = None,
                 status: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """sigma_p = HMAC-SHA-256(secret, id_p) for every principal (paper section 4.1)."""
    L = lib()
    n = id_off.numel() - 1
    if salts is None:
        salts = torch.empty((n, 32), dtype=torch.uint8, device=id_off.device)
    if ids.numel() == 0:   # every id is empty: hand the kernel a valid (unread) buffer
        ids = torch.zeros(1, dtype=torch.uint8, device=id_off.device)
    sec = bytes(secret)
    buf = ctypes.create_string_buffer(sec, len(sec)) if sec else None
    _check(L.kvgov_derive_salts(ctypes.cast(buf, _p) if buf is not None else None, len(sec),
                                _dev(ids, torch.uint8, "ids"), _dev(id_off, torch.int64, "id_off"), n,
                                _dev(salts, torch.uint8, "salts"),
                                _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_derive_salts")
    return salts


def chain_hash(mode: int, tokens: torch.Tensor, tok_off: torch.Tensor, blk_off: torch.Tensor,
               principal: torch.Tensor | None = None, salts: torch.Tensor | None = None,
               boundary_tok: torch.Tensor | None = None, digests: torch.Tensor | None = None,
               n_blocks: int | None = None, status: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Chained block digests, request-major [sum n_b, 32] (paper sections 2.1, 4.1, 4.2).

    digests (or n_blocks = blk_off[-1]) sizes the output; with neither, the
    total is read back from the device, which synchronises.
    """
    L = lib()
    n = tok_off.numel() - 1
    if digests is None:
        if n_blocks is None:
            n_blocks = int(blk_off[-1].item())
        digests = torch.empty((n_blocks, 32), dtype=torch.uint8, device=tokens.device)
    if tokens.numel() == 0:
        tokens = torch.zeros(4, dtype=torch.int32, device=tok_off.device)
    n_p = 0 if salts is None else salts.shape[0]
    _check(L.kvgov_chain_hash(int(mode), _dev(tokens, torch.int32, "tokens"), _dev(tok_off, torch.int64, "tok_off"),
                              n, _dev(principal, torch.int32, "principal", True),
                              _dev(salts, torch.uint8, "salts", True), n_p,
                              _dev(boundary_tok, torch.int32, "boundary_tok", True),
                              _dev(blk_off, torch.int64, "blk_off"),
                              _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(tokens),
                              _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_chain_hash")
    return digests


def chain_hash_probe(mode: int, tokens: torch.Tensor, tok_off: torch.Tensor, blk_off: torch.Tensor,
                     slots: torch.Tensor, principal: torch.Tensor | None = None, salts: torch.Tensor | None = None,
                     boundary_tok: torch.Tensor | None = None, digests: torch.Tensor | None = None,
                     prefix_blocks: torch.Tensor | None = None, n_blocks: int | None = None,
                     status: torch.Tensor | None = None, stream=None):
    """chain_hash and probe in one launch; returns (digests, prefix_blocks)."""
    L = lib()
    n = tok_off.numel() - 1
    if digests is None:
        if n_blocks is None:
            n_blocks = int(blk_off[-1].item())
        digests = torch.empty((n_blocks, 32), dtype=torch.uint8, device=tokens.device)
    if prefix_blocks is None:
        prefix_blocks = torch.empty(n, dtype=torch.int32, device=tok_off.device)
    if tokens.numel() == 0:
        tokens = torch.zeros(4, dtype=torch.int32, device=tok_off.device)
    n_p = 0 if salts is None else salts.shape[0]
    _check(L.kvgov_chain_hash_probe(int(mode), _dev(tokens, torch.int32, "tokens"),
                                    _dev(tok_off, torch.int64, "tok_off"), n,
                                    _dev(principal, torch.int32, "principal", True),
                                    _dev(salts, torch.uint8, "salts", True), n_p,
                                    _dev(boundary_tok, torch.int32, "boundary_tok", True),
                                    _dev(blk_off, torch.int64, "blk_off"),
                                    _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(tokens),
                                    _dev(slots, torch.uint8, "slots"), capacity_of(slots),
                                    _dev(prefix_blocks, torch.int32, "prefix_blocks") if n else _dummy(tokens),
                                    _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_chain_hash_probe")
    return digests, prefix_blocks


def new_gen(slots: torch.Tensor) -> torch.Tensor:
    """A zeroed generation array for a table (kvgov_chain_hash_serve)."""
    return torch.zeros(slots.shape[0], dtype=torch.int32, device=slots.device)


def table_gen_stamp(slots: torch.Tensor, gen: torch.Tensor, value: int, stream=None):
    """gen[h] = value for every handle holding a key, 0 for the others."""
    _check(lib().kvgov_table_gen_stamp(_dev(slots, torch.uint8, "slots"), capacity_of(slots),
                                       _dev(gen, torch.int32, "gen"), int(value), _stream(stream)),
           "kvgov_table_gen_stamp")


def chain_hash_serve(mode: int, tokens: torch.Tensor, tok_off: torch.Tensor, blk_off: torch.Tensor,
                     slots: torch.Tensor, gen: torch.Tensor, g: int, gen_floor: int, status: torch.Tensor,
                     principal: torch.Tensor | None = None, salts: torch.Tensor | None = None,
                     boundary_tok: torch.Tensor | None = None, digests: torch.Tensor | None = None,
                     n_blocks: int | None = None, n_new: torch.Tensor | None = None,
                     prefix_blocks: torch.Tensor | None = None, stream=None):
    """The serving step of one batch in one launch: its digests, its prefix
    lengths against the keys of generation [gen_floor, g), and its uncached
    blocks inserted with generation g.  Returns (digests, prefix_blocks)."""
    L = lib()
    n = tok_off.numel() - 1
    if digests is None:
        if n_blocks is None:
            n_blocks = int(blk_off[-1].item())
        digests = torch.empty((n_blocks, 32), dtype=torch.uint8, device=tokens.device)
    if prefix_blocks is None:
        prefix_blocks = torch.empty(max(n, 0), dtype=torch.int32, device=tokens.device)
    if tokens.numel() == 0:
        tokens = torch.zeros(4, dtype=torch.int32, device=tok_off.device)
    n_p = 0 if salts is None else salts.shape[0]
    _check(L.kvgov_chain_hash_serve(
        int(mode), _dev(tokens, torch.int32, "tokens"), _dev(tok_off, torch.int64, "tok_off"), n,
        _dev(principal, torch.int32, "principal", True), _dev(salts, torch.uint8, "salts", True), n_p,
        _dev(boundary_tok, torch.int32, "boundary_tok", True), _dev(blk_off, torch.int64, "blk_off"),
        _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(tokens),
        _dev(slots, torch.uint8, "slots"), capacity_of(slots), _dev(gen, torch.int32, "gen"), int(g), int(gen_floor),
        _dev(prefix_blocks, torch.int32, "prefix_blocks") if n else _dummy(tokens),
        _dev(n_new, torch.int64, "n_new", True), _dev(status, torch.int32, "status"), _stream(stream)),
        "kvgov_chain_hash_serve")
    return digests, prefix_blocks


def chain_hash_insert_prev(mode: int, tokens: torch.Tensor, tok_off: torch.Tensor, blk_off: torch.Tensor,
                           slots: torch.Tensor, prev_digests: torch.Tensor, prev_blk_off: torch.Tensor,
                           prev_prefix_blocks: torch.Tensor, status: torch.Tensor,
                           principal: torch.Tensor | None = None, salts: torch.Tensor | None = None,
                           boundary_tok: torch.Tensor | None = None, digests: torch.Tensor | None = None,
                           n_blocks: int | None = None, n_new: torch.Tensor | None = None,
                           prefix_blocks: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """chain_hash of this batch with insert_uncached of the previous batch
    (prev_digests, prev_blk_off, prev_prefix_blocks) and, if prefix_blocks
    is given, the probe of this batch after that insert; returns this
    batch's digests."""
    L = lib()
    n = tok_off.numel() - 1
    pn = prev_blk_off.numel() - 1
    if digests is None:
        if n_blocks is None:
            n_blocks = int(blk_off[-1].item())
        digests = torch.empty((n_blocks, 32), dtype=torch.uint8, device=tokens.device)
    if tokens.numel() == 0:
        tokens = torch.zeros(4, dtype=torch.int32, device=tok_off.device)
    n_p = 0 if salts is None else salts.shape[0]
    _check(L.kvgov_chain_hash_insert_prev(
        int(mode), _dev(tokens, torch.int32, "tokens"), _dev(tok_off, torch.int64, "tok_off"), n,
        _dev(principal, torch.int32, "principal", True), _dev(salts, torch.uint8, "salts", True), n_p,
        _dev(boundary_tok, torch.int32, "boundary_tok", True), _dev(blk_off, torch.int64, "blk_off"),
        _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(tokens),
        _dev(slots, torch.uint8, "slots"), capacity_of(slots),
        _dev(prev_digests, torch.uint8, "prev_digests") if prev_digests.numel() else _dummy(tokens),
        _dev(prev_blk_off, torch.int64, "prev_blk_off"), pn,
        _dev(prev_prefix_blocks, torch.int32, "prev_prefix_blocks") if pn else _dummy(tokens),
        (_dev(prefix_blocks, torch.int32, "prefix_blocks") if n else _dummy(tokens))
        if prefix_blocks is not None else None,
        _dev(n_new, torch.int64, "n_new", True), _dev(status, torch.int32, "status"), _stream(stream)),
        "kvgov_chain_hash_insert_prev")
    return digests


def _dummy(like: torch.Tensor):
    global _dummy_buf
    if _dummy_buf is None or _dummy_buf.device != like.device:
        _dummy_buf = torch.zeros(64, dtype=torch.uint8, device=like.device)
    return _dummy_buf.data_ptr()


_dummy_buf = None


def table_init(slots: torch.Tensor, stream=None) -> torch.Tensor:
    """Mark every slot of a [capacity + STASH_SLOTS, 32] u8 table empty."""
    _check(lib().kvgov_table_init(_dev(slots, torch.uint8, "slots"), capacity_of(slots), _stream(stream)),
           "kvgov_table_init")
    return slots


def new_table(capacity: int, device="cuda", stream=None) -> torch.Tensor:
    """An empty table of `capacity` main slots and the side store."""
    slots = torch.empty((capacity + STASH_SLOTS, 32), dtype=torch.uint8, device=device)
    return table_init(slots, stream)


def insert(slots: torch.Tensor, keys: torch.Tensor, status: torch.Tensor, n_new: torch.Tensor | None = None,
           stream=None):
    """Set-insert [n, 32] u8 keys; adds the number stored to n_new (int64[1])."""
    _check(lib().kvgov_insert(_dev(slots, torch.uint8, "slots"), capacity_of(slots),
                              _dev(keys, torch.uint8, "keys"), keys.shape[0] if keys.dim() == 2 else 0,
                              _dev(n_new, torch.int64, "n_new", True), _dev(status, torch.int32, "status"),
                              _stream(stream)),
           "kvgov_insert")


def probe(slots: torch.Tensor, digests: torch.Tensor, blk_off: torch.Tensor,
          prefix_blocks: torch.Tensor | None = None, status: torch.Tensor | None = None,
          stream=None) -> torch.Tensor:
    """prefix_blocks[r] = first j with h_j(r) not cached, or n_b(r) (paper section 2.1, Table 1)."""
    n = blk_off.numel() - 1
    if prefix_blocks is None:
        prefix_blocks = torch.empty(n, dtype=torch.int32, device=blk_off.device)
    _check(lib().kvgov_probe(_dev(slots, torch.uint8, "slots"), capacity_of(slots),
                             _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(blk_off),
                             _dev(blk_off, torch.int64, "blk_off"), n,
                             _dev(prefix_blocks, torch.int32, "prefix_blocks"),
                             _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_probe")
    return prefix_blocks


def probe_resume(slots: torch.Tensor, digests: torch.Tensor, blk_off: torch.Tensor, prefix_blocks: torch.Tensor,
                 status: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """probe, each request's walk starting at prefix_blocks[r] (a lower bound of
    its prefix on the table as it is now); prefix_blocks is overwritten with
    the prefix lengths and returned."""
    n = blk_off.numel() - 1
    _check(lib().kvgov_probe_resume(_dev(slots, torch.uint8, "slots"), capacity_of(slots),
                                    _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(blk_off),
                                    _dev(blk_off, torch.int64, "blk_off"), n,
                                    _dev(prefix_blocks, torch.int32, "prefix_blocks"),
                                    _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_probe_resume")
    return prefix_blocks


def insert_uncached(slots: torch.Tensor, digests: torch.Tensor, blk_off: torch.Tensor, prefix_blocks: torch.Tensor,
                    status: torch.Tensor, n_new: torch.Tensor | None = None, stream=None):
    """Insert each request's blocks from prefix_blocks[r] on (after probe)."""
    n = blk_off.numel() - 1
    _check(lib().kvgov_insert_uncached(_dev(slots, torch.uint8, "slots"), capacity_of(slots),
                                       _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(blk_off),
                                       _dev(blk_off, torch.int64, "blk_off"), n,
                                       _dev(prefix_blocks, torch.int32, "prefix_blocks"),
                                       _dev(n_new, torch.int64, "n_new", True), _dev(status, torch.int32, "status"),
                                       _stream(stream)),
           "kvgov_insert_uncached")


# ---- arrival-order serving (paper sections 2.1 and 4.2, request by request)
def owner_init(owner: torch.Tensor, stream=None) -> torch.Tensor:
    """Zero a table's owner array ([capacity + STASH_SLOTS] int64 holding u64
    arrival positions)."""
    _check(lib().kvgov_owner_init(_dev(owner, torch.int64, "owner"), _owner_capacity(owner), _stream(stream)),
           "kvgov_owner_init")
    return owner


def new_owner(capacity: int, device="cuda", stream=None) -> torch.Tensor:
    return owner_init(torch.empty(capacity + STASH_SLOTS, dtype=torch.int64, device=device), stream)


def insert_arrival(slots: torch.Tensor, owner: torch.Tensor, digests: torch.Tensor, blk_off: torch.Tensor,
                   seq_base: int, status: torch.Tensor, slot_of: torch.Tensor | None = None,
                   n_new: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Insert every block of the batch, block j of request r arriving at
    position seq_base + blk_off[r] + j; returns slot_of ([n_blocks] int32:
    the slot of each block, -1 if not stored)."""
    n = blk_off.numel() - 1
    n_blocks = digests.shape[0] if digests.dim() == 2 else 0
    if slot_of is None:
        slot_of = torch.empty(n_blocks, dtype=torch.int32, device=blk_off.device)
    _check(lib().kvgov_insert_arrival(_dev(slots, torch.uint8, "slots"), _dev(owner, torch.int64, "owner"),
                                      capacity_of(slots),
                                      _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(blk_off),
                                      _dev(blk_off, torch.int64, "blk_off"), n, int(seq_base),
                                      _dev(slot_of, torch.int32, "slot_of") if slot_of.numel() else _dummy(blk_off),
                                      _dev(n_new, torch.int64, "n_new", True), _dev(status, torch.int32, "status"),
                                      _stream(stream)),
           "kvgov_insert_arrival")
    return slot_of


def probe_arrival(owner: torch.Tensor, slot_of: torch.Tensor, blk_off: torch.Tensor, seq_base: int,
                  prefix_blocks: torch.Tensor | None = None, status: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    """prefix_blocks[r] = blocks of request r cached when it arrived (after insert_arrival)."""
    n = blk_off.numel() - 1
    if prefix_blocks is None:
        prefix_blocks = torch.empty(n, dtype=torch.int32, device=blk_off.device)
    _check(lib().kvgov_probe_arrival(_dev(owner, torch.int64, "owner"), _owner_capacity(owner),
                                     _dev(slot_of, torch.int32, "slot_of") if slot_of.numel() else _dummy(blk_off),
                                     _dev(blk_off, torch.int64, "blk_off"), n, int(seq_base),
                                     _dev(prefix_blocks, torch.int32, "prefix_blocks"),
                                     _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_probe_arrival")
    return prefix_blocks


def chain_hash_arrival(mode: int, tokens: torch.Tensor, tok_off: torch.Tensor, blk_off: torch.Tensor,
                       slots: torch.Tensor, owner: torch.Tensor, seq_base: int, status: torch.Tensor,
                       principal: torch.Tensor | None = None, salts: torch.Tensor | None = None,
                       boundary_tok: torch.Tensor | None = None, digests: torch.Tensor | None = None,
                       slot_of: torch.Tensor | None = None, prefix_blocks: torch.Tensor | None = None,
                       n_blocks: int | None = None, n_new: torch.Tensor | None = None, stream=None):
    """chain_hash, insert_arrival and probe_arrival in one call (the insert
    fused into the chain kernel for large batches); returns (digests,
    slot_of, prefix_blocks)."""
    L = lib()
    n = tok_off.numel() - 1
    if digests is None:
        if n_blocks is None:
            n_blocks = int(blk_off[-1].item())
        digests = torch.empty((n_blocks, 32), dtype=torch.uint8, device=tokens.device)
    if slot_of is None:
        slot_of = torch.empty(digests.shape[0], dtype=torch.int32, device=tokens.device)
    if prefix_blocks is None:
        prefix_blocks = torch.empty(n, dtype=torch.int32, device=tok_off.device)
    if tokens.numel() == 0:
        tokens = torch.zeros(4, dtype=torch.int32, device=tok_off.device)
    n_p = 0 if salts is None else salts.shape[0]
    _check(L.kvgov_chain_hash_arrival(int(mode), _dev(tokens, torch.int32, "tokens"),
                                      _dev(tok_off, torch.int64, "tok_off"), n,
                                      _dev(principal, torch.int32, "principal", True),
                                      _dev(salts, torch.uint8, "salts", True), n_p,
                                      _dev(boundary_tok, torch.int32, "boundary_tok", True),
                                      _dev(blk_off, torch.int64, "blk_off"),
                                      _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(tokens),
                                      _dev(slots, torch.uint8, "slots"), _dev(owner, torch.int64, "owner"),
                                      capacity_of(slots), int(seq_base),
                                      _dev(slot_of, torch.int32, "slot_of") if slot_of.numel() else _dummy(tokens),
                                      _dev(prefix_blocks, torch.int32, "prefix_blocks") if n else _dummy(tokens),
                                      _dev(n_new, torch.int64, "n_new", True), _dev(status, torch.int32, "status"),
                                      _stream(stream)),
           "kvgov_chain_hash_arrival")
    return digests, slot_of, prefix_blocks


def divergence_boundary(tokens: torch.Tensor, tok_off: torch.Tensor, template_id: torch.Tensor,
                        tpl_tokens: torch.Tensor | None = None, tpl_off: torch.Tensor | None = None,
                        boundary_tok: torch.Tensor | None = None, status: torch.Tensor | None = None,
                        stream=None) -> torch.Tensor:
    """Boundary token offset of each request: its longest common prefix with
    its registered preamble (paper sections 4.2 and 5.7); template_id[r] is a
    preamble index, TEMPLATE_NONE or TEMPLATE_ANY."""
    n = tok_off.numel() - 1
    n_tpl = 0 if tpl_off is None else tpl_off.numel() - 1
    if boundary_tok is None:
        boundary_tok = torch.empty(max(n, 0), dtype=torch.int32, device=tok_off.device)
    if tokens.numel() == 0:
        tokens = torch.zeros(4, dtype=torch.int32, device=tok_off.device)
    if tpl_tokens is not None and tpl_tokens.numel() == 0:
        tpl_tokens = torch.zeros(4, dtype=torch.int32, device=tok_off.device)
    _check(lib().kvgov_divergence_boundary(_dev(tokens, torch.int32, "tokens"), _dev(tok_off, torch.int64, "tok_off"), n,
                                           _dev(template_id, torch.int32, "template_id") if n else _dummy(tokens),
                                           _dev(tpl_tokens, torch.int32, "tpl_tokens", True),
                                           _dev(tpl_off, torch.int64, "tpl_off", True), n_tpl,
                                           _dev(boundary_tok, torch.int32, "boundary_tok") if n else _dummy(tokens),
                                           _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_divergence_boundary")
    return boundary_tok


def response_key(mode: int, tokens: torch.Tensor, tok_off: torch.Tensor, principal: torch.Tensor | None = None,
                 salts: torch.Tensor | None = None, keys: torch.Tensor | None = None,
                 status: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Exact-response cache key per request: SHA-256(sigma_p || prompt bytes)
    (ROOT) or SHA-256(prompt bytes) (UNSALTED); returns [n, 32] u8."""
    n = tok_off.numel() - 1
    if keys is None:
        keys = torch.empty((max(n, 0), 32), dtype=torch.uint8, device=tok_off.device)
    if tokens.numel() == 0:
        tokens = torch.zeros(4, dtype=torch.int32, device=tok_off.device)
    n_p = 0 if salts is None else salts.shape[0]
    _check(lib().kvgov_response_key(int(mode), _dev(tokens, torch.int32, "tokens"), _dev(tok_off, torch.int64, "tok_off"),
                                    n, _dev(principal, torch.int32, "principal", True),
                                    _dev(salts, torch.uint8, "salts", True), n_p,
                                    _dev(keys, torch.uint8, "keys") if n else _dummy(tokens),
                                    _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_response_key")
    return keys


def origami(values: torch.Tensor, off: torch.Tensor, budget: torch.Tensor, p: torch.Tensor | None = None,
            lam: torch.Tensor | None = None, utility: torch.Tensor | None = None, status: torch.Tensor | None = None,
            stream=None):
    """ORIGAMI audit probabilities per problem (paper section 4.3): float32
    values in CSR by off, float32 budgets; returns (p, lambda, utility)."""
    n = off.numel() - 1
    if p is None:
        p = torch.empty_like(values)
    if lam is None:
        lam = torch.empty(max(n, 0), dtype=torch.float32, device=off.device)
    if utility is None:
        utility = torch.empty(max(n, 0), dtype=torch.float32, device=off.device)
    if values.numel() == 0:
        values = torch.zeros(1, dtype=torch.float32, device=off.device)
        p_arg = _dummy(off)
    else:
        p_arg = _dev(p, torch.float32, "p")
    _check(lib().kvgov_origami(_dev(values, torch.float32, "values"), _dev(off, torch.int64, "off"), n,
                               _dev(budget, torch.float32, "budget") if n else _dummy(off), p_arg,
                               _dev(lam, torch.float32, "lambda") if n else None,
                               _dev(utility, torch.float32, "utility") if n else None,
                               _dev(status, torch.int32, "status", True), _stream(stream)),
           "kvgov_origami")
    return p, lam, utility


def serve_arrival_static(slots: torch.Tensor, owner: torch.Tensor, digests: torch.Tensor, blk_off: torch.Tensor,
                         seq_base: int, status: torch.Tensor, prefix_blocks: torch.Tensor | None = None,
                         n_new: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """insert_arrival + probe_arrival with the slot handles kept in the
    library's own device array (at most 2^21 blocks; calls must not overlap)."""
    n = blk_off.numel() - 1
    n_blocks = digests.shape[0] if digests.dim() == 2 else 0
    if prefix_blocks is None:
        prefix_blocks = torch.empty(max(n, 0), dtype=torch.int32, device=blk_off.device)
    _check(lib().kvgov_serve_arrival_static(_dev(slots, torch.uint8, "slots"), _dev(owner, torch.int64, "owner"),
                                            capacity_of(slots),
                                            _dev(digests, torch.uint8, "digests") if digests.numel() else _dummy(blk_off),
                                            _dev(blk_off, torch.int64, "blk_off"), n, n_blocks, int(seq_base),
                                            _dev(prefix_blocks, torch.int32, "prefix_blocks") if n else _dummy(blk_off),
                                            _dev(n_new, torch.int64, "n_new", True),
                                            _dev(status, torch.int32, "status"), _stream(stream)),
           "kvgov_serve_arrival_static")
    return prefix_blocks


def set_spin_limit(limit: int) -> int:
    return int(lib().kvgov_set_spin_limit(int(limit)))


# ---- the serving engine (include/kvgov_pipeline.h)
def event_handle(ev: torch.cuda.Event, stream) -> int:
    """The cudaEvent_t of a torch event, created (by one record on stream) if it has none yet."""
    if ev.cuda_event == 0:
        ev.record(stream)
    return ev.cuda_event


class Engine:
    """A kvgov_pipeline engine over caller-owned buffers, events and streams
    (kept alive by the caller).  submit() is one foreign call per batch."""

    def __init__(self, desc: PipelineDesc):
        self._desc = desc
        self._h = _p()
        _check(lib().kvgov_pipeline_create(ctypes.byref(desc), ctypes.byref(self._h)), "kvgov_pipeline_create")
        self._slot = ctypes.c_int32(0)

    def submit(self, secret: bytes, tokens: int, tok_off: int, n_req: int, principal: int | None,
               boundary_tok: int | None, n_blocks: int, after: int | None, flush: bool,
               chain_ev=(None, None), table_ev=(None, None)) -> int:
        _check(lib().kvgov_pipeline_submit(self._h, secret, len(secret), tokens, tok_off, n_req, principal,
                                           boundary_tok, n_blocks, after, int(bool(flush)), chain_ev[0],
                                           chain_ev[1], table_ev[0], table_ev[1], ctypes.byref(self._slot)),
               "kvgov_pipeline_submit")
        return self._slot.value

    def drain(self):
        _check(lib().kvgov_pipeline_drain(self._h), "kvgov_pipeline_drain")

    def pending(self) -> bool:
        return bool(lib().kvgov_pipeline_pending(self._h))

    def __del__(self):
        if getattr(self, "_h", None) and _lib is not None:
            _lib.kvgov_pipeline_destroy(self._h)
            self._h = None
