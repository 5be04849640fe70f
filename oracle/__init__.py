"""CPU oracle for KVGov's salted block-hash chain and prefix lookup.

TEST INFRASTRUCTURE: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The CUDA library
and its Python binding never import it.

This module only marshals numpy arrays into the plain C implementation in
``oracle.c`` (FIPS 180-4 SHA-256, RFC 2104 HMAC, the paper's chain equations
of sections 2.1, 4.1 and 4.2, and the block prefix lookup of section 2.1 /
Table 1).  The shared library is compiled with gcc on first use.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

UNSALTED, ROOT, BOUNDARY = 0, 1, 2
FLAG_ZERO_KEY = 1

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

_p = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_sz = ctypes.c_size_t


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so (plain gcc, no vector extensions)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-std=c11", "-Wall", "-Wextra", "-shared", "-fPIC",
                        "-o", tmp, _SRC], check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _configure(L):
    L.oracle_sha256.argtypes = [_p, _sz, _p]
    L.oracle_sha256.restype = None
    L.oracle_hmac_sha256.argtypes = [_p, _sz, _p, _sz, _p]
    L.oracle_hmac_sha256.restype = None
    L.oracle_sha256_constants.argtypes = [_p, _p]
    L.oracle_sha256_constants.restype = None
    L.oracle_derive_salts.argtypes = [_p, _sz, _p, _p, _i32, _p]
    L.oracle_derive_salts.restype = ctypes.c_int
    L.oracle_block_offsets.argtypes = [_p, _i32, _p]
    L.oracle_block_offsets.restype = ctypes.c_int
    L.oracle_chain_hash.argtypes = [ctypes.c_int, _p, _p, _i32, _p, _p, _i32, _p, _p]
    L.oracle_chain_hash.restype = ctypes.c_int
    L.oracle_key_is_zero.argtypes = [_p]
    L.oracle_key_is_zero.restype = ctypes.c_int
    L.oracle_set_insert.argtypes = [_p, _p, _i64, _p, _i64, _p]
    L.oracle_set_insert.restype = _i64
    L.oracle_prefix_blocks.argtypes = [_p, _i64, _p, _p, _i32, _p]
    L.oracle_prefix_blocks.restype = ctypes.c_int
    L.oracle_arrival_prefix.argtypes = [_p, _i64, _p, _p, _i32, _p, _p]
    L.oracle_arrival_prefix.restype = ctypes.c_int
    L.oracle_divergence_boundary.argtypes = [_p, _p, _i32, _p, _p, _p, _i32, _p]
    L.oracle_divergence_boundary.restype = ctypes.c_int
    L.oracle_response_key.argtypes = [ctypes.c_int, _p, _p, _i32, _p, _p, _i32, _p]
    L.oracle_response_key.restype = ctypes.c_int
    L.oracle_origami.argtypes = [_p, _p, _i32, _p, _p, _p, _p]
    L.oracle_origami.restype = ctypes.c_int
    return L


_override = None


def load_library(path: str):
    """A separately built copy of the oracle (the tests build copies with a
    planted mistake to show that the pins catch it)."""
    return _configure(ctypes.CDLL(path))


class using_library:
    """Context manager: route this module's functions through library L."""

    def __init__(self, L):
        self.L = L

    def __enter__(self):
        global _override
        self.prev, _override = _override, self.L
        return self.L

    def __exit__(self, *exc):
        global _override
        _override = self.prev


def lib():
    global _lib
    if _override is not None:
        return _override
    with _lock:
        if _lib is None:
            build()
            _lib = _configure(ctypes.CDLL(_LIB))
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p) if a is not None and a.size else None


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def sha256(msg: bytes) -> bytes:
    m = np.frombuffer(bytes(msg), dtype=np.uint8)
    out = np.zeros(32, np.uint8)
    lib().oracle_sha256(_ptr(m), len(m), _ptr(out))
    return out.tobytes()


def hmac_sha256(key: bytes, msg: bytes) -> bytes:
    k = np.frombuffer(bytes(key), dtype=np.uint8)
    m = np.frombuffer(bytes(msg), dtype=np.uint8)
    out = np.zeros(32, np.uint8)
    lib().oracle_hmac_sha256(_ptr(k), len(k), _ptr(m), len(m), _ptr(out))
    return out.tobytes()


def sha256_constants():
    k = np.zeros(64, np.uint32)
    iv = np.zeros(8, np.uint32)
    lib().oracle_sha256_constants(_ptr(k), _ptr(iv))
    return k, iv


def derive_salts(secret: bytes, ids: np.ndarray, id_off: np.ndarray) -> np.ndarray:
    """sigma_p = HMAC-SHA-256(secret, id bytes of p) for every principal p."""
    ids = _c(ids, np.uint8)
    id_off = _c(id_off, np.int64)
    n = len(id_off) - 1
    s = np.frombuffer(bytes(secret), dtype=np.uint8)
    salts = np.zeros((n, 32), np.uint8)
    rc = lib().oracle_derive_salts(_ptr(s), len(s), _ptr(ids), _ptr(id_off), n, _ptr(salts))
    if rc != 0:
        raise ValueError("oracle_derive_salts: malformed id offsets")
    return salts


def block_offsets(tok_off: np.ndarray) -> np.ndarray:
    tok_off = _c(tok_off, np.int64)
    n = len(tok_off) - 1
    blk = np.zeros(n + 1, np.int64)
    if lib().oracle_block_offsets(_ptr(tok_off), n, _ptr(blk)) != 0:
        raise ValueError("oracle_block_offsets: negative request length")
    return blk


def chain_hash(mode: int, tokens: np.ndarray, tok_off: np.ndarray,
               principal: np.ndarray | None = None, salts: np.ndarray | None = None,
               boundary_tok: np.ndarray | None = None) -> np.ndarray:
    """Digests [sum n_b, 32] u8 of every request's block chain, request-major."""
    tokens = _c(tokens, np.int32)
    tok_off = _c(tok_off, np.int64)
    n = len(tok_off) - 1
    blk = block_offsets(tok_off)
    out = np.zeros((int(blk[-1]), 32), np.uint8)
    principal = None if principal is None else _c(principal, np.int32)
    salts = None if salts is None else _c(salts, np.uint8)
    boundary_tok = None if boundary_tok is None else _c(boundary_tok, np.int32)
    n_p = 0 if salts is None else salts.shape[0]
    if mode != UNSALTED and (principal is None or salts is None):
        raise ValueError("salted modes need principal and salts")
    if mode == BOUNDARY and boundary_tok is None:
        raise ValueError("BOUNDARY needs boundary_tok")
    rc = lib().oracle_chain_hash(mode, _ptr(tokens), _ptr(tok_off), n, _ptr(principal),
                                 _ptr(salts), n_p, _ptr(boundary_tok), _ptr(out))
    if rc != 0:
        raise ValueError("oracle_chain_hash: invalid argument")
    return out


def divergence_boundary(tokens: np.ndarray, tok_off: np.ndarray, template_id: np.ndarray,
                        tpl_tokens: np.ndarray, tpl_off: np.ndarray):
    """Boundary token offset per request: the longest common prefix with its
    registered preamble (ids: index, -1 none, -2 best of all).  Returns
    (boundary_tok int32 [n], flag) -- flag set if an id was out of range."""
    tokens = _c(tokens, np.int32)
    if tokens.size == 0:
        tokens = np.zeros(1, np.int32)
    tok_off = _c(tok_off, np.int64)
    template_id = _c(template_id, np.int32)
    tpl_tokens = _c(tpl_tokens, np.int32)
    if tpl_tokens.size == 0:
        tpl_tokens = np.zeros(1, np.int32)
    tpl_off = _c(tpl_off, np.int64)
    n = len(tok_off) - 1
    out = np.zeros(max(n, 1), np.int32)
    flag = lib().oracle_divergence_boundary(_ptr(tokens), _ptr(tok_off), n, _ptr(template_id), _ptr(tpl_tokens),
                                            _ptr(tpl_off), len(tpl_off) - 1, _ptr(out))
    return out[:n], bool(flag)


def response_key(mode: int, tokens: np.ndarray, tok_off: np.ndarray, principal: np.ndarray,
                 salts: np.ndarray) -> np.ndarray:
    """Exact-response cache keys [n, 32]: SHA-256(sigma_p || prompt bytes) for
    ROOT, SHA-256(prompt bytes) for UNSALTED (paper Table 1, section 4.1)."""
    tokens = _c(tokens, np.int32)
    if tokens.size == 0:
        tokens = np.zeros(1, np.int32)
    tok_off = _c(tok_off, np.int64)
    principal = _c(principal, np.int32)
    salts = _c(salts, np.uint8).reshape(-1, 32)
    n = len(tok_off) - 1
    out = np.zeros((max(n, 1), 32), np.uint8)
    rc = lib().oracle_response_key(int(mode), _ptr(tokens), _ptr(tok_off), n, _ptr(principal), _ptr(salts),
                                   salts.shape[0], _ptr(out))
    if rc != 0:
        raise ValueError("oracle_response_key: bad mode, range or principal")
    return out[:n]


def origami(values: np.ndarray, off: np.ndarray, budget: np.ndarray):
    """ORIGAMI audit probabilities (paper section 4.3): float32 values in CSR
    by off, float32 budgets.  Returns (p fp64, lambda fp64, utility fp64, flag)."""
    values = _c(values, np.float32)
    if values.size == 0:
        values = np.zeros(1, np.float32)
    off = _c(off, np.int64)
    budget = _c(budget, np.float32)
    n = len(off) - 1
    p = np.zeros(max(values.size, 1), np.float64)
    lam = np.zeros(max(n, 1), np.float64)
    u = np.zeros(max(n, 1), np.float64)
    rc = lib().oracle_origami(_ptr(values), _ptr(off), n, _ptr(budget), _ptr(p), _ptr(lam), _ptr(u))
    if rc < 0:
        raise MemoryError("oracle_origami")
    return p[: int(off[-1])], lam[:n], u[:n], bool(rc)


def key_is_zero(key: bytes) -> bool:
    """The one key the set refuses: all 32 bytes zero."""
    k = np.frombuffer(bytes(key), dtype=np.uint8)
    return bool(lib().oracle_key_is_zero(_ptr(k)))


class KeySet:
    """The cache index as a mathematical set of 32-byte keys (sorted array)."""

    def __init__(self, capacity: int):
        self.keys = np.zeros((max(int(capacity), 1), 32), np.uint8)
        self.n = 0

    def insert(self, keys: np.ndarray):
        """Returns (n_new, zero_key_flag): the keys the set gained, and whether
        an all-zero key was given (and skipped)."""
        keys = _c(keys, np.uint8).reshape(-1, 32)
        if self.n + keys.shape[0] > self.keys.shape[0]:
            grown = np.zeros((self.n + keys.shape[0], 32), np.uint8)
            grown[: self.n] = self.keys[: self.n]
            self.keys = grown
        n_set = ctypes.c_int64(self.n)
        n_new = ctypes.c_int64(0)
        rc = lib().oracle_set_insert(_ptr(self.keys), ctypes.byref(n_set), self.keys.shape[0],
                                     _ptr(keys), keys.shape[0], ctypes.byref(n_new))
        if rc < 0:
            raise ValueError("KeySet capacity exceeded")
        self.n = n_set.value
        return n_new.value, bool(rc & FLAG_ZERO_KEY)

    def contents(self) -> np.ndarray:
        return self.keys[: self.n]

    def prefix_blocks(self, digests: np.ndarray, blk_off: np.ndarray) -> np.ndarray:
        digests = _c(digests, np.uint8).reshape(-1, 32)
        blk_off = _c(blk_off, np.int64)
        n = len(blk_off) - 1
        out = np.zeros(n, np.int32)
        rc = lib().oracle_prefix_blocks(_ptr(self.keys), self.n, _ptr(digests), _ptr(blk_off),
                                        n, _ptr(out))
        if rc != 0:
            raise ValueError("oracle_prefix_blocks: malformed block offsets")
        return out

    def arrival_prefix(self, digests: np.ndarray, blk_off: np.ndarray):
        """Arrival-order serving of a batch against this set (left unchanged):
        request r's prefix counts the set's keys and every block of requests
        before r; returns (prefix_blocks, n_new), n_new = keys the batch adds."""
        digests = _c(digests, np.uint8).reshape(-1, 32)
        blk_off = _c(blk_off, np.int64)
        n = len(blk_off) - 1
        out = np.zeros(n, np.int32)
        n_new = ctypes.c_int64(0)
        rc = lib().oracle_arrival_prefix(_ptr(self.keys), self.n, _ptr(digests), _ptr(blk_off), n, _ptr(out),
                                         ctypes.byref(n_new))
        if rc != 0:
            raise ValueError("oracle_arrival_prefix: malformed block offsets or out of memory")
        return out, n_new.value
