"""CPU-only checks: the C-ABI library builds, loads and exports every symbol
the header declares; host-side argument validation; the golden file is still
what the oracle computes; the seeded workloads have the structure they claim.
No GPU and no kernel launch is involved."""
import ctypes
import json
import os
import re

import numpy as np
import pytest

import oracle
from paper_2608_09225_gb300 import build as kbuild
from paper_2608_09225_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "kvgov.h")


@pytest.fixture(scope="module")
def libkv():
    path = kbuild.build()
    return ctypes.CDLL(path)


def declared_functions(header=HEADER):
    text = open(header).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kvgov_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ("kvgov_derive_salts", "kvgov_block_offsets", "kvgov_chain_hash", "kvgov_table_init",
                 "kvgov_insert", "kvgov_probe", "kvgov_insert_uncached", "kvgov_chain_hash_probe",
                 "kvgov_owner_init", "kvgov_insert_arrival", "kvgov_probe_arrival", "kvgov_chain_hash_arrival",
                 "kvgov_divergence_boundary", "kvgov_response_key", "kvgov_origami", "kvgov_status_string",
                 "kvgov_set_spin_limit"):
        assert want in names


def test_library_exports_every_declared_symbol(libkv):
    for name in declared_functions():
        assert hasattr(libkv, name), name


def test_peak_library_exports_every_declared_symbol():
    kbuild.build()
    lib = ctypes.CDLL(kbuild.PEAK_LIB)
    names = declared_functions(os.path.join(ROOT, "include", "kvgov_peak.h"))
    assert {"kvgov_peak_int", "kvgov_peak_gather", "kvgov_peak_ops_per_iter"} <= set(names)
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(os.listdir(os.path.join(ROOT, "include"))) == ["kvgov.h", "kvgov_peak.h", "kvgov_pipeline.h"]


def test_library_exports_the_serving_engine(libkv):
    names = declared_functions(os.path.join(ROOT, "include", "kvgov_pipeline.h"))
    assert {"kvgov_pipeline_create", "kvgov_pipeline_submit", "kvgov_pipeline_drain", "kvgov_pipeline_pending",
            "kvgov_pipeline_destroy"} <= set(names)
    for name in names:
        assert hasattr(libkv, name), name


def _engine_desc(insert_in_chain=1):
    """A description whose pointers are never dereferenced on the host (the
    checks below run before any CUDA call)."""
    from paper_2608_09225_gb300.kvgov import PipelineDesc
    d = PipelineDesc()
    d.mode, d.insert_in_chain, d.n_slots = 2, insert_in_chain, 3 if insert_in_chain == 1 else 2
    d.d_gen = 0x60000 if insert_in_chain == 2 else None
    d.max_req, d.max_blocks = 100, 800
    d.d_slots, d.capacity, d.d_status, d.d_n_new = 0x10000, 1 << 10, 0x20000, 0x30000
    d.d_ids, d.d_id_off, d.n_principals = 0x40000, 0x50000, 4
    for i in range(d.n_slots):
        d.d_salts[i], d.d_blk_off[i], d.d_digests[i], d.d_prefix[i] = (0x100000 * (i + 1) + 0x1000 * k
                                                                       for k in range(4))
        d.prepared[i], d.chain_start[i], d.probed[i], d.free_ev[i] = (0x9000000 + 0x100 * i + k for k in range(4))
    d.prep_stream, d.compute_stream = 0x7000, 0x7100
    return d


def test_serving_engine_checks_its_arguments(libkv):
    """kvgov_pipeline_create refuses bad descriptions and kvgov_pipeline_submit
    bad batches with KVGOV_EINVAL, on the host, before anything is queued."""
    from paper_2608_09225_gb300.kvgov import PipelineDesc
    P = ctypes.c_void_p
    libkv.kvgov_pipeline_create.argtypes = [ctypes.POINTER(PipelineDesc), ctypes.POINTER(P)]
    libkv.kvgov_pipeline_submit.argtypes = [P, ctypes.c_char_p, ctypes.c_size_t, P, P, ctypes.c_int32, P, P,
                                            ctypes.c_int64, P, ctypes.c_int, P, P, P, P,
                                            ctypes.POINTER(ctypes.c_int32)]
    libkv.kvgov_pipeline_destroy.argtypes = [P]
    libkv.kvgov_pipeline_destroy.restype = None
    libkv.kvgov_pipeline_drain.argtypes = [P]
    libkv.kvgov_pipeline_pending.argtypes = [P]
    h = P()
    bad = []
    d = _engine_desc(); d.n_slots = 2; bad.append(d)                 # insert in chain needs 3 slots
    d = _engine_desc(0); d.n_slots = 3; bad.append(d)                # inline takes 2
    d = _engine_desc(); d.mode = 7; bad.append(d)
    d = _engine_desc(); d.capacity = 1000; bad.append(d)             # not a power of two
    d = _engine_desc(); d.d_digests[2] = 0x100008; bad.append(d)     # misaligned
    d = _engine_desc(); d.probed[1] = 0; bad.append(d)               # missing event
    d = _engine_desc(); d.d_ids = 0; bad.append(d)                   # salted mode without ids
    d = _engine_desc(); d.max_req = -1; bad.append(d)
    d = _engine_desc(3); d.n_slots = 2; bad.append(d)                # no such schedule
    d = _engine_desc(2); d.d_gen = None; bad.append(d)              # one launch needs the generations
    d = _engine_desc(2); d.n_slots = 3; bad.append(d)                # ... and takes 2 slots
    for d in bad:
        assert libkv.kvgov_pipeline_create(ctypes.byref(d), ctypes.byref(h)) == 1
    d = _engine_desc()
    assert libkv.kvgov_pipeline_create(ctypes.byref(d), ctypes.byref(h)) == 0 and h.value
    slot = ctypes.c_int32(-1)
    sec = b"s" * 32
    args = dict(tokens=0x800000, tok_off=0x810000, n_req=10, principal=0x820000, boundary=0x830000, n_blocks=80)

    def submit(**kw):
        a = dict(args, **kw)
        return libkv.kvgov_pipeline_submit(h, kw.get("secret", sec), kw.get("secret_len", len(sec)), a["tokens"],
                                           a["tok_off"], a["n_req"], a["principal"], a["boundary"], a["n_blocks"],
                                           None, 0, kw.get("ev0"), None, None, None, ctypes.byref(slot))
    assert submit(n_req=101) == 1                                     # above max_req
    assert submit(n_blocks=801) == 1                                  # above max_blocks
    assert submit(principal=None) == 1                                # salted mode
    assert submit(boundary=None) == 1                                 # BOUNDARY mode
    assert submit(tok_off=None) == 1
    assert submit(secret_len=2000) == 1                               # longer than KVGOV_MAX_SECRET
    assert submit(ev0=0x1234) == 1                                    # an unpaired timing event
    assert slot.value == -1 and libkv.kvgov_pipeline_pending(h) == 0
    assert libkv.kvgov_pipeline_drain(h) == 0                         # nothing pending: nothing queued
    libkv.kvgov_pipeline_destroy(h)
    libkv.kvgov_pipeline_destroy(None)
    d = _engine_desc(2)                                               # one launch: generations, 2 slots
    assert libkv.kvgov_pipeline_create(ctypes.byref(d), ctypes.byref(h)) == 0 and h.value
    assert submit(n_req=101) == 1 and libkv.kvgov_pipeline_pending(h) == 0
    libkv.kvgov_pipeline_destroy(h)


def test_peak_gather_rejects_bad_arguments():
    """Argument checks run on the host and launch nothing."""
    kbuild.build()
    f = ctypes.CDLL(kbuild.PEAK_LIB).kvgov_peak_gather
    f.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int, ctypes.c_int64, ctypes.c_uint64, ctypes.c_void_p,
                  ctypes.c_void_p]
    fake, sink = 1 << 20, 1 << 21          # never dereferenced: every call below fails its checks first
    assert f(None, 1024, 32, 10, 0, sink, None) == 1
    assert f(fake, 1000, 32, 10, 0, sink, None) == 1          # not a power of two
    assert f(fake, 1024, 24, 10, 0, sink, None) == 1          # 16 or 32 bytes per read
    assert f(fake, 1024, 32, -1, 0, sink, None) == 1
    assert f(fake + 8, 1024, 32, 10, 0, sink, None) == 1      # not 16-byte aligned
    assert f(fake, 1024, 32, 10, 0, None, None) == 1
    assert f(fake, 1024, 32, 0, 0, sink, None) == 0           # nothing to read: nothing launched


def test_status_strings(libkv):
    f = libkv.kvgov_status_string
    f.restype = ctypes.c_char_p
    f.argtypes = [ctypes.c_int]
    assert f(0) == b"KVGOV_OK"
    assert b"EINVAL" in f(1)
    for flag, word in ((0x10, b"BADINDEX"), (0x20, b"SENTINEL"), (0x40, b"FULL"), (0x80, b"TIMEOUT")):
        assert word in f(flag)
    assert f(12345)


def test_spin_limit_roundtrip(libkv):
    f = libkv.kvgov_set_spin_limit
    f.restype = ctypes.c_uint32
    f.argtypes = [ctypes.c_uint32]
    prev = f(77)
    assert f(0) == 77
    assert f(prev) == 1 << 23


def test_host_validation_rejects_bad_arguments(libkv):
    """Arguments the host can check are refused with KVGOV_EINVAL before any
    CUDA call (these calls never reach the GPU)."""
    p = ctypes.c_void_p
    fake = p(1 << 20)          # never dereferenced: every call below fails validation first
    odd = p((1 << 20) + 4)     # not 16-byte aligned
    ch = libkv.kvgov_chain_hash
    ch.argtypes = [ctypes.c_int, p, p, ctypes.c_int32, p, p, ctypes.c_int32, p, p, p, p, p]
    assert ch(7, fake, fake, 4, fake, fake, 1, fake, fake, fake, None, None) == 1          # bad mode
    assert ch(0, odd, fake, 4, None, None, 0, None, fake, fake, None, None) == 1            # misaligned tokens
    assert ch(0, fake, fake, 4, None, None, 0, None, fake, odd, None, None) == 1            # misaligned digests
    assert ch(1, fake, fake, 4, None, fake, 1, None, fake, fake, None, None) == 1           # ROOT without principal
    assert ch(2, fake, fake, 4, fake, fake, 1, None, fake, fake, None, None) == 1           # BOUNDARY without offsets
    assert ch(0, fake, fake, -1, None, None, 0, None, fake, fake, None, None) == 1          # negative n_req
    assert ch(0, fake, fake, 0, None, None, 0, None, fake, fake, None, None) == 0           # empty batch: no-op
    cp = libkv.kvgov_chain_hash_probe
    cp.argtypes = [ctypes.c_int, p, p, ctypes.c_int32, p, p, ctypes.c_int32, p, p, p, p, ctypes.c_uint64, p, p, p]
    assert cp(0, fake, fake, 4, None, None, 0, None, fake, fake, fake, 64, None, None, None) == 1   # no output
    assert cp(0, fake, fake, 4, None, None, 0, None, fake, fake, fake, 100, fake, None, None) == 1  # capacity
    assert cp(0, fake, fake, 4, None, None, 0, None, fake, fake, odd, 64, fake, None, None) == 1    # misaligned
    assert cp(0, fake, fake, 0, None, None, 0, None, fake, fake, fake, 64, fake, None, None) == 0   # empty batch
    ti = libkv.kvgov_table_init
    ti.argtypes = [p, ctypes.c_uint64, p]
    for cap in (0, 16, 48, 1000):
        assert ti(fake, cap, None) == 1
    ins = libkv.kvgov_insert
    ins.argtypes = [p, ctypes.c_uint64, p, ctypes.c_int64, p, p, p]
    assert ins(fake, 64, fake, 5, None, None, None) == 1      # status is required
    assert ins(fake, 64, fake, -1, None, fake, None) == 1
    assert ins(fake, 64, None, 0, None, fake, None) == 0      # nothing to insert
    pr = libkv.kvgov_probe
    pr.argtypes = [p, ctypes.c_uint64, p, p, ctypes.c_int32, p, p, p]
    assert pr(fake, 100, fake, fake, 3, fake, None, None) == 1
    assert pr(fake, 64, odd, fake, 3, fake, None, None) == 1
    iu = libkv.kvgov_insert_uncached
    iu.argtypes = [p, ctypes.c_uint64, p, p, ctypes.c_int32, p, p, p, p]
    assert iu(fake, 64, fake, fake, 3, fake, None, None, None) == 1     # status is required
    assert iu(fake, 64, odd, fake, 3, fake, None, fake, None) == 1      # misaligned digests
    assert iu(fake, 64, fake, fake, 0, None, None, fake, None) == 0     # empty batch
    sa = libkv.kvgov_derive_salts
    sa.argtypes = [p, ctypes.c_size_t, p, p, ctypes.c_int32, p, p, p]
    assert sa(None, 1025, fake, fake, 3, fake, None, None) == 1
    assert sa(None, 5, fake, fake, 3, fake, None, None) == 1
    assert sa(None, 0, fake, fake, 0, fake, None, None) == 0
    bo = libkv.kvgov_block_offsets
    bo.argtypes = [p, ctypes.c_int32, p, p, p]
    assert bo(fake, -2, fake, None, None) == 1
    oi = libkv.kvgov_owner_init
    oi.argtypes = [p, ctypes.c_uint64, p]
    assert oi(None, 64, None) == 1
    assert oi(odd, 64, None) == 1
    assert oi(fake, 100, None) == 1
    assert oi(fake, 1 << 32, None) == 1                                   # slot index must fit in u32
    ia = libkv.kvgov_insert_arrival
    ia.argtypes = [p, p, ctypes.c_uint64, p, p, ctypes.c_int32, ctypes.c_uint64, p, p, p, p]
    assert ia(fake, fake, 64, fake, fake, 3, 0, fake, None, fake, None) == 1            # position 0 is reserved
    assert ia(fake, fake, 64, fake, fake, 3, (1 << 62) + 1, fake, None, fake, None) == 1   # past 2^62
    assert ia(fake, fake, 64, fake, fake, 3, 1, fake, None, None, None) == 1            # status is required
    assert ia(fake, fake, 64, fake, fake, 3, 1, None, None, fake, None) == 1            # no slot_of
    assert ia(fake, fake, 64, odd, fake, 3, 1, fake, None, fake, None) == 1             # misaligned digests
    assert ia(fake, fake, 64, None, None, 0, 1, None, None, fake, None) == 0            # empty batch
    ca = libkv.kvgov_chain_hash_arrival
    ca.argtypes = [ctypes.c_int, p, p, ctypes.c_int32, p, p, ctypes.c_int32, p, p, p, p, p, ctypes.c_uint64,
                   ctypes.c_uint64, p, p, p, p, p]
    assert ca(0, fake, fake, 4, None, None, 0, None, fake, fake, fake, fake, 64, 1, fake, fake, None, None,
              None) == 1                                                                 # status is required
    assert ca(0, fake, fake, 4, None, None, 0, None, fake, fake, fake, None, 64, 1, fake, fake, None, fake,
              None) == 1                                                                 # no owner array
    assert ca(0, fake, fake, 4, None, None, 0, None, fake, fake, fake, fake, 64, 0, fake, fake, None, fake,
              None) == 1                                                                 # position 0
    assert ca(0, fake, fake, 0, None, None, 0, None, fake, fake, fake, fake, 64, 1, fake, fake, None, fake,
              None) == 0                                                                 # empty batch
    db = libkv.kvgov_divergence_boundary
    db.argtypes = [p, p, ctypes.c_int32, p, p, p, ctypes.c_int32, p, p, p]
    assert db(fake, fake, -1, fake, None, None, 0, fake, None, None) == 1                # negative n_req
    assert db(fake, fake, 3, None, None, None, 0, fake, None, None) == 1                 # no template ids
    assert db(fake, fake, 3, fake, None, None, 2, fake, None, None) == 1                 # preambles missing
    assert db(None, fake, 0, None, None, None, 0, None, None, None) == 0                 # empty batch
    rk = libkv.kvgov_response_key
    rk.argtypes = [ctypes.c_int, p, p, ctypes.c_int32, p, p, ctypes.c_int32, p, p, p]
    assert rk(2, fake, fake, 3, fake, fake, 1, fake, None, None) == 1                    # BOUNDARY has no meaning
    assert rk(1, fake, fake, 3, None, fake, 1, fake, None, None) == 1                    # ROOT without principals
    assert rk(0, odd, fake, 3, None, None, 0, fake, None, None) == 1                     # misaligned tokens
    assert rk(0, fake, fake, 0, None, None, 0, None, None, None) == 0                    # empty batch
    og = libkv.kvgov_origami
    og.argtypes = [p, p, ctypes.c_int32, p, p, p, p, p, p]
    assert og(fake, fake, -1, fake, fake, None, None, None, None) == 1                   # negative count
    assert og(fake, fake, 3, None, fake, None, None, None, None) == 1                    # no budgets
    assert og(None, fake, 0, None, None, None, None, None, None) == 0                    # no problems
    pa = libkv.kvgov_probe_arrival
    pa.argtypes = [p, ctypes.c_uint64, p, p, ctypes.c_int32, ctypes.c_uint64, p, p, p]
    assert pa(fake, 64, fake, fake, 3, 0, fake, None, None) == 1
    assert pa(fake, 64, fake, fake, 3, 1, None, None, None) == 1
    assert pa(fake, 64, None, None, 0, 1, None, None, None) == 0


def test_golden_file_is_what_the_oracle_computes():
    import importlib.util
    spec = importlib.util.spec_from_file_location("make_golden", os.path.join(ROOT, "tests", "golden",
                                                                              "make_golden.py"))
    mg = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mg)
    with open(mg.OUT) as f:
        stored = json.load(f)
    assert mg.compute() == stored


# ----------------------------------------------------------------- workloads
def test_workloads_are_deterministic():
    a, b = W.make("template", n_req=64), W.make("template", n_req=64)
    assert a.secret == b.secret and (a.batch.tokens == b.batch.tokens).all()
    c = W.make("wide", seed=5, n_req=32)
    d = W.make("wide", seed=6, n_req=32)
    assert not (c.batch.tokens == d.batch.tokens).all()


def test_workload_structure():
    w = W.make("tiny")
    t = w.batch.tokens.reshape(64, 256)
    assert (t[:32, :128] == t[0, :128]).all() and not (t[32:, :128] == t[0, :128]).all(axis=1).any()
    assert t.min() >= 0 and t.max() < W.VOCAB
    s = W.sysprompt(n_req=64)
    ts = s.batch.tokens.reshape(64, 2119)
    assert (ts[:, :1024] == ts[0, :1024]).all()
    assert 0.4 < s.info["gini"] < 0.9
    tp = W.template(n_req=128)
    tt = tp.batch.tokens.reshape(128, 512)
    mask = np.ones(512, bool)
    for off in W.FIELD_OFFSETS:
        mask[off:off + 8] = False
    assert (tt[:, mask] == tt[0, mask]).all()
    assert (tp.batch.boundary_tok == 96).all()
    pw = W.probe(n_req=256, n_prior=32, capacity=1 << 12, n_random=100)
    reuse, src, cut = pw.info["reuse"], pw.info["src"], pw.info["cut"]
    pt, prt = pw.batch.tokens.reshape(256, 512), pw.prior.tokens.reshape(32, 512)
    for r in np.nonzero(reuse)[0]:
        c = 16 * int(cut[r])
        assert (pt[r, :c] == prt[src[r], :c]).all()
        assert pw.batch.principal[r] == pw.prior.principal[src[r]]
    keys = pw.random_keys
    assert not any(oracle.key_is_zero(k.tobytes()) for k in keys)
    lw = W.make("long", n_req=4)
    assert lw.batch.tokens.shape[0] == 4 * 32768 and (lw.batch.boundary_tok == 64).all()


def test_full_size_shapes():
    """The full-size definitions (sizes only; generation is cheap except probe)."""
    assert W.make("wide").batch.n == 131072
    assert W.make("sysprompt").batch.lengths()[0] == 2119


def test_oracle_zero_key_rule():
    """Only the all-zero key is refused by the oracle's set."""
    one = b"\x01" * 8
    assert oracle.key_is_zero(bytes(32))
    for k in (bytes(16) + one + one, one + one + bytes(8) + one, one + one + one + bytes(8), bytes(31) + b"\x01",
              b"\x01" + bytes(31), bytes(8) + one + one + one):
        assert not oracle.key_is_zero(k)


def test_count_blocks_on_the_host(libkv):
    """kvgov_count_blocks (host code, no device) against the oracle's
    blocking: the same block offsets on ragged lengths (tails of 0..15 tokens,
    empty requests, the workloads' shapes), a negative length counting 0 as
    on the device, and its argument checks."""
    p = ctypes.c_void_p
    cb = libkv.kvgov_count_blocks
    cb.argtypes = [p, ctypes.c_int32, p, p]
    rng = np.random.default_rng(41)
    for lens in (np.array([0, 1, 15, 16, 17, 31, 32, 2119, 128, 0], np.int64), rng.integers(0, 5000, 777),
                 np.full(64, 256), np.zeros(0, np.int64)):
        tok_off = np.zeros(len(lens) + 1, np.int64)
        tok_off[1:] = np.cumsum(lens)
        blk = np.empty(len(lens) + 1, np.int64)
        total = ctypes.c_int64(-1)
        assert cb(tok_off.ctypes.data, len(lens), blk.ctypes.data, ctypes.byref(total)) == 0
        want = oracle.block_offsets(tok_off)
        assert (blk == want).all() and total.value == int(want[-1])
        assert cb(tok_off.ctypes.data, len(lens), None, ctypes.byref(total)) == 0 and total.value == int(want[-1])
    bad = np.array([0, 40, 20, 60], np.int64)                 # request 1 has length -20
    blk = np.empty(4, np.int64)
    total = ctypes.c_int64(-1)
    assert cb(bad.ctypes.data, 3, blk.ctypes.data, ctypes.byref(total)) == 0
    assert list(blk) == [0, 2, 2, 4] and total.value == 4
    assert cb(None, 3, None, ctypes.byref(total)) == 1
    assert cb(bad.ctypes.data, -1, None, ctypes.byref(total)) == 1
    assert cb(bad.ctypes.data, 3, None, None) == 1
