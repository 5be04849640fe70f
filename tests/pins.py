"""Pins for the CPU oracle: checks against things other than the oracle itself.

Every check here compares the oracle with an independent implementation of a
special case (Python's hashlib / hmac, i.e. OpenSSL), with an invariant the
paper states, with a number the paper prints for a worked example
(tests/golden/paper_examples.json), with a closed form of a synthetic
workload, or with brute force on tiny inputs.  They are plain functions so
that tests/test_oracle_pins.py can also run them against copies of the oracle
with a planted mistake and show that some pin fails.
"""
from __future__ import annotations

import hashlib
import hmac
import json
import os
import struct

import numpy as np

import oracle
from paper_2608_09225_gb300 import workloads as W

UNSALTED, ROOT, BOUNDARY = oracle.UNSALTED, oracle.ROOT, oracle.BOUNDARY
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def H(b: bytes) -> bytes:
    return hashlib.sha256(b).digest()


def block_le(tokens) -> bytes:
    """Little-endian int32 serialisation, written with struct (not numpy)."""
    return struct.pack("<%di" % len(tokens), *[int(t) for t in tokens])


def _batch(lengths, seed=3):
    return W.ragged(seed, lengths)


def _rows(blk_off, r):
    return range(int(blk_off[r]), int(blk_off[r + 1]))


# --------------------------------------------------------------- SHA-256 / HMAC
def pin_sha256_every_length():
    """FIPS 180-4 SHA-256 == hashlib on every length 0..300 (all padding edges)."""
    rng = np.random.default_rng(11)
    for n in range(301):
        m = rng.integers(0, 256, n, dtype=np.uint8).tobytes()
        assert oracle.sha256(m) == H(m), f"length {n}"


def pin_sha256_long_and_classic():
    """Multi-block messages: short ASCII, a two-block 56-byte message, 1 MB."""
    for m in (b"abc", b"abcdbcdecdefdefgefghfghighijhijkijkljklmklmnlmnomnopnopq",
              b"a" * 1_000_000, bytes(range(256)) * 17):
        assert oracle.sha256(m) == H(m)


def pin_hmac():
    """RFC 2104 HMAC-SHA-256 == Python hmac for keys shorter than, equal to and
    longer than the 64-byte block, and messages across the padding edges."""
    rng = np.random.default_rng(12)
    for kl in (0, 1, 20, 32, 63, 64, 65, 131, 1024):
        key = rng.integers(0, 256, kl, dtype=np.uint8).tobytes()
        for ml in (0, 4, 50, 55, 56, 64, 119, 152, 1000):
            msg = rng.integers(0, 256, ml, dtype=np.uint8).tobytes()
            assert oracle.hmac_sha256(key, msg) == hmac.new(key, msg, "sha256").digest(), (kl, ml)


def pin_salts():
    """sigma_p = HMAC_K(secret, principal_id) (section 4.1) == Python hmac,
    for 4-byte ids and for variable-length ids including the empty one."""
    secret = bytes(range(32))
    ids, id_off = W.principal_ids(64)
    s = oracle.derive_salts(secret, ids, id_off)
    for p in range(64):
        assert s[p].tobytes() == hmac.new(secret, struct.pack("<I", p), "sha256").digest()
    rng = np.random.default_rng(13)
    lens = [0, 1, 55, 56, 64, 100, 200]
    raw = [rng.integers(0, 256, L, dtype=np.uint8).tobytes() for L in lens]
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    buf = np.frombuffer(b"".join(raw), np.uint8)
    long_key = bytes(rng.integers(0, 256, 100, dtype=np.uint8))
    s = oracle.derive_salts(long_key, buf, off)
    for i, m in enumerate(raw):
        assert s[i].tobytes() == hmac.new(long_key, m, "sha256").digest()


# ----------------------------------------------------------------- the chain
def pin_token_serialisation():
    """A token's hashed bytes are its int32 little-endian bytes; a block of
    16 tokens hashes as H(T_0) (section 2.1, j = 0)."""
    toks = np.array([0x04030201, -1, -(2 ** 31), 2 ** 31 - 1, 0, 1, 256, 65536,
                     152063, 7, 0x7F00FF00, -2, 3, 4, 5, 6], dtype=np.int32)
    d = oracle.chain_hash(UNSALTED, toks, np.array([0, 16]))
    assert d[0].tobytes() == H(block_le(toks))
    assert block_le(toks[:1]) == b"\x01\x02\x03\x04"


def pin_chain_unsalted():
    """Section 2.1: h_0 = H(T_0), h_j = H(h_{j-1} || T_j); partial tails unhashed."""
    b = _batch([16, 33, 48, 0, 15, 16 * 9 + 5])
    d = oracle.chain_hash(UNSALTED, b.tokens, b.tok_off)
    blk = oracle.block_offsets(b.tok_off)
    assert list(np.diff(blk)) == [1, 2, 3, 0, 0, 9]
    for r in range(b.n):
        t = b.tokens[b.tok_off[r]:b.tok_off[r + 1]]
        prev = None
        for j, row in enumerate(_rows(blk, r)):
            T = block_le(t[16 * j:16 * j + 16])
            want = H(T) if j == 0 else H(prev + T)
            assert d[row].tobytes() == want, (r, j)
            prev = want


def pin_chain_root():
    """Section 4.1: h_0 = H(sigma_p || T_0); later blocks chained as before."""
    b = _batch([16, 40, 64, 16 * 7])
    salts = np.random.default_rng(5).integers(0, 256, (8, 32), dtype=np.uint8)
    d = oracle.chain_hash(ROOT, b.tokens, b.tok_off, b.principal, salts)
    blk = oracle.block_offsets(b.tok_off)
    for r in range(b.n):
        t = b.tokens[b.tok_off[r]:b.tok_off[r + 1]]
        sig = salts[b.principal[r]].tobytes()
        prev = None
        for j, row in enumerate(_rows(blk, r)):
            T = block_le(t[16 * j:16 * j + 16])
            want = H(sig + T) if j == 0 else H(prev + T)
            assert d[row].tobytes() == want, (r, j)
            prev = want


def pin_chain_boundary():
    """Section 4.2: blocks j < k unsalted; h_k = H(sigma_p || h_{k-1} || T_k)
    (H(sigma_p || T_0) at k = 0); j > k chained; k = floor(b / 16)."""
    bounds = [0, 1, 15, 16, 17, 31, 32, 47, 48, 63, 64, 100, 10 ** 6]
    n = len(bounds)
    rng = np.random.default_rng(6)
    toks = rng.integers(0, W.VOCAB, (n, 16 * 6), dtype=np.int32)
    tok_off = np.arange(n + 1, dtype=np.int64) * 96
    principal = np.arange(n, dtype=np.int32) % 4
    salts = rng.integers(0, 256, (4, 32), dtype=np.uint8)
    bt = np.array(bounds, dtype=np.int32)
    d = oracle.chain_hash(BOUNDARY, toks.reshape(-1), tok_off, principal, salts, bt)
    for r in range(n):
        k = bounds[r] // 16
        sig = salts[principal[r]].tobytes()
        prev = None
        for j in range(6):
            T = block_le(toks[r, 16 * j:16 * j + 16])
            if j == k:
                want = H(sig + T) if j == 0 else H(sig + prev + T)
            else:
                want = H(T) if j == 0 else H(prev + T)
            assert d[6 * r + j].tobytes() == want, (r, j)
            prev = want


def pin_boundary_invariants():
    """Section 4.2: for j < k the digests are principal-independent and equal
    to the unsalted chain (shared, routable); for j >= k they differ across
    principals and from the unsalted chain; BOUNDARY with b < 16 is ROOT."""
    rng = np.random.default_rng(8)
    toks = rng.integers(0, W.VOCAB, 16 * 8, dtype=np.int32)
    n_p = 6
    tokens = np.tile(toks, n_p)
    tok_off = np.arange(n_p + 1, dtype=np.int64) * 128
    principal = np.arange(n_p, dtype=np.int32)
    salts = oracle.derive_salts(b"k" * 32, *W.principal_ids(n_p))
    un = oracle.chain_hash(UNSALTED, toks, np.array([0, 128]))
    for b in (16 * 3, 16 * 3 + 9):
        d = oracle.chain_hash(BOUNDARY, tokens, tok_off, principal, salts, np.full(n_p, b, np.int32))
        d = d.reshape(n_p, 8, 32)
        for j in range(3):
            for p in range(n_p):
                assert (d[p, j] == un[j]).all()
        for j in range(3, 8):
            rows = {d[p, j].tobytes() for p in range(n_p)}
            assert len(rows) == n_p and un[j].tobytes() not in rows
    root = oracle.chain_hash(ROOT, tokens, tok_off, principal, salts)
    for b in (0, 7, 15):
        d = oracle.chain_hash(BOUNDARY, tokens, tok_off, principal, salts, np.full(n_p, b, np.int32))
        assert (d == root).all()


def pin_disjoint_and_deterministic():
    """Section 4.1: over identical tokens, ROOT chains of different principals
    share no digest at any position; the same (principal, tokens) gives the
    same chain at any batch position."""
    rng = np.random.default_rng(9)
    n_p, per = 8, 8
    base = rng.integers(0, W.VOCAB, (per, 64), dtype=np.int32)
    tokens = np.tile(base.reshape(-1), n_p)
    tok_off = np.arange(n_p * per + 1, dtype=np.int64) * 64
    principal = np.repeat(np.arange(n_p, dtype=np.int32), per)
    salts = oracle.derive_salts(b"s" * 32, *W.principal_ids(n_p))
    d = oracle.chain_hash(ROOT, tokens, tok_off, principal, salts).reshape(n_p, per, 4, 32)
    seen = {}
    for p in range(n_p):
        for q in range(per):
            for j in range(4):
                key = d[p, q, j].tobytes()
                assert seen.setdefault(key, (p, q, j)) == (p, q, j)
    # same chain at another batch position (request reordered)
    perm = np.random.default_rng(10).permutation(n_p * per)
    t2 = tokens.reshape(-1, 64)[perm].reshape(-1)
    d2 = oracle.chain_hash(ROOT, t2, tok_off, principal[perm], salts).reshape(-1, 4, 32)
    assert (d2 == d.reshape(-1, 4, 32)[perm]).all()


# ------------------------------------------------------------------- lookup
def _prefix(mode, fill_tokens, fill_principal, probe_tokens, probe_principal, salts=None, b=0, L=None):
    """Fill a set with one request's chain, probe another; returns hit blocks."""
    L = L or len(fill_tokens)
    ks = oracle.KeySet(1)
    d = oracle.chain_hash(mode, fill_tokens, np.array([0, L]), np.array([fill_principal]), salts,
                          np.array([b], np.int32))
    ks.insert(d)
    q = oracle.chain_hash(mode, probe_tokens, np.array([0, L]), np.array([probe_principal]), salts,
                          np.array([b], np.int32))
    return int(ks.prefix_blocks(q, oracle.block_offsets(np.array([0, L])))[0])


def _paper():
    with open(os.path.join(GOLDEN, "paper_examples.json")) as f:
        return json.load(f)


def pin_paper_divergence_layout():
    """Section 5.7: a 2119-token shared preamble diverging at token 1990 keeps
    124 block hits; diverging at token 5 keeps none."""
    ex = _paper()["divergence_layout"]
    n = ex["prompt_tokens"]
    rng = np.random.default_rng(14)
    a = rng.integers(0, W.VOCAB, n, dtype=np.int32)
    for i, want in zip(ex["diverge_at_token"], ex["hit_blocks"]):
        bq = a.copy()
        bq[i] = (bq[i] + 1) % W.VOCAB
        assert _prefix(UNSALTED, a, 0, bq, 0) == want


def pin_paper_boundary_efficiency():
    """Section 4.2: with the salt at the end of a 2000-token shared preamble of
    a 2119-token prompt, another principal reuses the preamble's full blocks
    and prefills 8 blocks (7 full + the partial tail) instead of 133."""
    ex = _paper()["boundary_salting_efficiency"]
    n, pre = ex["prompt_tokens"], ex["shared_preamble_tokens"]
    total_blocks = -(-n // 16)
    rng = np.random.default_rng(15)
    a = rng.integers(0, W.VOCAB, n, dtype=np.int32)
    salts = oracle.derive_salts(b"x" * 32, *W.principal_ids(2))
    hits_b = _prefix(BOUNDARY, a, 0, a, 1, salts, b=pre)
    hits_r = _prefix(ROOT, a, 0, a, 1, salts)
    assert total_blocks - hits_b == ex["blocks_to_prefill_boundary"]
    assert total_blocks - hits_r == ex["blocks_to_prefill_root"]
    assert _prefix(BOUNDARY, a, 1, a, 1, salts, b=pre) == n // 16   # same principal: all full blocks


def pin_cross_principal_all_miss():
    """Section 4.1: a prober on another principal sees all-MISS on the victim's
    cached prompt; the same principal hits every full block."""
    rng = np.random.default_rng(16)
    salts = oracle.derive_salts(b"y" * 32, *W.principal_ids(4))
    for L in (16, 100, 512):
        a = rng.integers(0, W.VOCAB, L, dtype=np.int32)
        assert _prefix(ROOT, a, 2, a, 3, salts) == 0
        assert _prefix(ROOT, a, 2, a, 2, salts) == L // 16
        assert _prefix(UNSALTED, a, 2, a, 3) == L // 16


def pin_prefix_brute_force():
    """Lookup == a Python-set brute force: first missing block, later hits
    ignored (section 2.1 longest common prefix from position 0)."""
    rng = np.random.default_rng(17)
    for trial in range(20):
        nb = rng.integers(0, 12, 30)
        off = np.concatenate([[0], np.cumsum(nb)]).astype(np.int64)
        pool = rng.integers(0, 256, (8, 32), dtype=np.uint8)
        pool[:, 31] |= 1                                  # no all-zero key
        pool[0, :16] = 0                                  # zero first half: an ordinary key
        pool[1, 16:24] = 0                                # a zero 8-byte word: an ordinary key
        digests = pool[rng.integers(0, 8, int(off[-1]))]
        member = rng.random(8) < 0.6
        ks = oracle.KeySet(1)
        ks.insert(pool[member])
        S = {pool[i].tobytes() for i in range(8) if member[i]}
        got = ks.prefix_blocks(digests, off)
        for r in range(30):
            L = 0
            while L < nb[r] and digests[off[r] + L].tobytes() in S:
                L += 1
            assert got[r] == L


def pin_set_semantics():
    """Set insert (section 2.1: the cache index holds the keys of cached
    blocks): duplicates are no-ops in any order; every key but the all-zero
    one becomes a member -- keys with a zero half or zero 8-byte words
    included -- and the all-zero key is refused and flagged.  Contents and
    lookups are checked against a Python set."""
    rng = np.random.default_rng(18)
    keys = rng.integers(0, 256, (50, 32), dtype=np.uint8)
    keys[:, 0] |= 1
    batch = np.concatenate([keys, keys[::-1], keys[:10]])
    ks = oracle.KeySet(1)
    n_new, flag = ks.insert(batch)
    assert n_new == 50 and not flag
    n_new, flag = ks.insert(keys[:20])
    assert n_new == 0 and not flag
    odd = np.full((8, 32), 7, np.uint8)
    odd[0, :16] = 0             # first half zero
    odd[1, 16:24] = 0           # third word zero
    odd[2, 24:] = 0             # fourth word zero
    odd[3, 16:] = 0             # second half zero
    odd[4, :8] = 0              # first word zero
    odd[5, :24] = 0             # only the last word non-zero
    odd[6, 1:] = 0              # one non-zero byte, first
    odd[7, :31] = 0             # one non-zero byte, last
    n_new, flag = ks.insert(np.concatenate([odd, odd[::-1]]))
    assert n_new == 8 and not flag and ks.n == 58
    n_new, flag = ks.insert(np.zeros((2, 32), np.uint8))
    assert n_new == 0 and flag and ks.n == 58
    S = {k.tobytes() for k in np.concatenate([keys, odd])}
    assert {k.tobytes() for k in ks.contents()} == S
    probe = np.concatenate([odd, np.zeros((1, 32), np.uint8), keys[:3]])
    assert list(ks.prefix_blocks(probe, np.array([0, 8, 12, 12], np.int64))) == [8, 0, 0]
    assert list(ks.prefix_blocks(probe[9:], np.array([0, 3], np.int64))) == [3]
    ks2 = oracle.KeySet(1)
    ks2.insert(np.concatenate([odd, batch])[rng.permutation(len(batch) + 8)])
    assert (ks2.contents() == ks.contents()).all()


# ------------------------------------------------------ workload closed forms
def run_workload_oracle(w, mode):
    """Salts, chains, table fill and probe of a workload, all with the oracle."""
    salts = oracle.derive_salts(w.secret, w.ids, w.id_off)
    b = w.batch
    d = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    blk = oracle.block_offsets(b.tok_off)
    ks = oracle.KeySet(1)
    if w.fill_from == "prior":
        p = w.prior
        dp = oracle.chain_hash(mode, p.tokens, p.tok_off, p.principal, salts, p.boundary_tok)
        ks.insert(dp)
    else:
        f0, f1 = w.fill
        ks.insert(d[blk[f0]:blk[f1]])
    if w.random_keys is not None:
        ks.insert(w.random_keys)
    p0, p1 = w.probe
    L = ks.prefix_blocks(d, blk[p0:p1 + 1])
    return salts, d, blk, ks, L


def pin_tiny_closed_form():
    """Tiny workload: the table holds requests 0-15; requests 16-31 share the
    128-token template (8 blocks) with request r-16 of the same principal;
    requests 32-63 share nothing."""
    w = W.make("tiny")
    _, _, _, _, L = run_workload_oracle(w, ROOT)
    assert list(L) == [16] * 16 + [8] * 16 + [0] * 32


def pin_sysprompt_closed_form():
    """Shared system prompt (reduced): filled requests hit all 132 blocks;
    others hit the 64 system-prefix blocks iff their principal filled."""
    w = W.sysprompt(n_req=96, fill_n=24)
    _, _, _, _, L = run_workload_oracle(w, ROOT)
    filled = set(w.batch.principal[:24].tolist())
    want = [132] * 24 + [64 if int(p) in filled else 0 for p in w.batch.principal[24:]]
    assert list(L) == want


def pin_probe_closed_form():
    """Probe-heavy (reduced): a request reusing c blocks of a prior request
    (with that request's principal) hits exactly c; a fresh one hits 0."""
    w = W.probe(n_req=512, n_prior=64, capacity=1 << 12, n_random=1000)
    _, _, _, _, L = run_workload_oracle(w, ROOT)
    assert (L == w.info["cut"]).all()


def pin_template_ordering():
    """Template workload (reduced): per request, hits under UNSALTED >=
    BOUNDARY >= ROOT; BOUNDARY (k = 6) keeps the 6 template blocks before the
    first field for every request."""
    w = W.template(n_req=1024)
    Ls = {m: run_workload_oracle(w, m)[4] for m in (UNSALTED, ROOT, BOUNDARY)}
    assert (Ls[UNSALTED] >= Ls[BOUNDARY]).all() and (Ls[BOUNDARY] >= Ls[ROOT]).all()
    assert (Ls[BOUNDARY] >= 6).all() and (Ls[UNSALTED] >= 6).all()
    assert Ls[UNSALTED].mean() > Ls[BOUNDARY].mean()


# ------------------------------------------------------ arrival-order serving
def _zero_py(k: bytes) -> bool:
    return not any(k)


def _replay_python(S0, digests, off):
    """Serve the requests one at a time with a Python set: count the leading
    cached blocks, then cache the request's blocks."""
    S = {bytes(k) for k in S0}
    before, out = len(S), []
    for r in range(len(off) - 1):
        rows = [digests[i].tobytes() for i in range(int(off[r]), int(off[r + 1]))]
        L = 0
        while L < len(rows) and rows[L] in S:
            L += 1
        out.append(L)
        S.update(k for k in rows if not _zero_py(k))
    return out, len(S) - before


def pin_arrival_brute_force():
    """Arrival-order serving == a Python-set replay, request by request, on
    batches whose requests copy leading keys of earlier ones, with keys cached
    before the batch, keys with a zero half or word (ordinary members) and
    the odd all-zero key (never cached)."""
    rng = np.random.default_rng(19)
    for trial in range(40):
        n_req = int(rng.integers(1, 40))
        pool = rng.integers(0, 256, (16, 32), dtype=np.uint8)
        pool[:, 0] |= 1
        pool[13, :16] = 0                                  # zero first half: an ordinary key
        pool[14, 24:] = 0                                  # zero last word: an ordinary key
        pool[15] = 0                                       # the all-zero key: never cached
        reqs = []
        for r in range(n_req):
            nb = int(rng.integers(0, 10))
            keys = list(rng.integers(0, 16, nb))
            if reqs and rng.random() < 0.6:               # start with a copy of an earlier request's prefix
                src = reqs[int(rng.integers(0, len(reqs)))]
                c = int(rng.integers(0, len(src) + 1))
                keys = list(src[:c]) + keys
            reqs.append(keys)
        off = np.concatenate([[0], np.cumsum([len(k) for k in reqs])]).astype(np.int64)
        digests = pool[np.array([i for k in reqs for i in k], dtype=np.int64)].reshape(-1, 32)
        s0 = pool[:15][rng.random(15) < 0.3]
        ks = oracle.KeySet(1)
        ks.insert(s0)
        got, n_new = ks.arrival_prefix(digests, off)
        want, want_new = _replay_python(s0, digests, off)
        assert list(got) == want and n_new == want_new, trial


def pin_arrival_repeats_and_turns():
    """Closed forms: a request repeated by its principal hits every block the
    second time; the turns of one conversation, each an exact prefix extension
    of the one before (section 6: multi-turn reuse), hit all blocks of the
    previous turn."""
    salts = oracle.derive_salts(b"q" * 32, *W.principal_ids(4))
    rng = np.random.default_rng(20)
    t = rng.integers(0, W.VOCAB, 100, dtype=np.int32)
    toks = np.tile(t, 5)
    off = np.arange(0, 501, 100, dtype=np.int64)
    d = oracle.chain_hash(ROOT, toks, off, np.full(5, 2, np.int32), salts, np.zeros(5, np.int32))
    L, n_new = oracle.KeySet(1).arrival_prefix(d, oracle.block_offsets(off))
    assert list(L) == [0, 6, 6, 6, 6] and n_new == 6
    conv = rng.integers(0, W.VOCAB, 200, dtype=np.int32)
    turns = [conv[: 16 * (r + 1) + 5] for r in range(10)]
    toks = np.concatenate(turns)
    off = np.concatenate([[0], np.cumsum([len(x) for x in turns])]).astype(np.int64)
    d = oracle.chain_hash(ROOT, toks, off, np.ones(10, np.int32), salts, np.zeros(10, np.int32))
    L, n_new = oracle.KeySet(1).arrival_prefix(d, oracle.block_offsets(off))
    assert list(L) == list(range(10)) and n_new == 10


def pin_arrival_per_principal():
    """Sixteen requests with one prompt, principal r mod 4: salted at the
    root, a principal's first request misses and its later ones hit every
    block (section 4.1); unsalted, only request 0 misses; salted at block 2
    (section 4.2), the first request of principals 1-3 still hits the 2 shared
    blocks."""
    salts = oracle.derive_salts(b"r" * 32, *W.principal_ids(4))
    t = np.random.default_rng(21).integers(0, W.VOCAB, 130, dtype=np.int32)
    toks = np.tile(t, 16)
    off = np.arange(0, 16 * 130 + 1, 130, dtype=np.int64)
    pr = (np.arange(16) % 4).astype(np.int32)
    b = np.full(16, 32, np.int32)
    blk = oracle.block_offsets(off)
    want = {ROOT: [0] * 4 + [8] * 12, UNSALTED: [0] + [8] * 15, BOUNDARY: [0] + [2] * 3 + [8] * 12}
    for mode, w in want.items():
        d = oracle.chain_hash(mode, toks, off, pr, salts, b)
        L, _ = oracle.KeySet(1).arrival_prefix(d, blk)
        assert list(L) == w, mode


def pin_arrival_tiny_closed_form():
    """Tiny workload served in arrival order into an empty cache: request r of
    the 32 template requests hits the 8 template blocks once request r-8 (same
    principal) has been served; the 32 others share nothing."""
    w = W.make("tiny")
    salts = oracle.derive_salts(w.secret, w.ids, w.id_off)
    b = w.batch
    d = oracle.chain_hash(ROOT, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    L, n_new = oracle.KeySet(1).arrival_prefix(d, oracle.block_offsets(b.tok_off))
    assert list(L) == [0] * 8 + [8] * 24 + [0] * 32
    assert n_new == 64 * 16 - 24 * 8


# ------------------------------------------------------ divergence boundary
def _lcp_python(a, b):
    n = 0
    for x, y in zip(a, b):
        if int(x) != int(y):
            break
        n += 1
    return n


def pin_boundary_brute_force():
    """Boundary detection == a Python zip comparison: the longest common
    prefix with the named preamble, the longest over all preambles for id -2,
    0 for id -1 and for ids out of range (flagged)."""
    rng = np.random.default_rng(22)
    for trial in range(30):
        tpls = [rng.integers(0, 5, int(rng.integers(0, 40)), dtype=np.int32) for _ in range(int(rng.integers(0, 4)))]
        reqs, ids = [], []
        for r in range(int(rng.integers(1, 30))):
            base = tpls[int(rng.integers(0, len(tpls)))] if tpls and rng.random() < 0.8 else np.zeros(0, np.int32)
            cut = int(rng.integers(0, len(base) + 1))
            tail = rng.integers(0, 5, int(rng.integers(0, 10)), dtype=np.int32)
            reqs.append(np.concatenate([base[:cut], tail]).astype(np.int32))
            ids.append(int(rng.integers(-3, len(tpls) + 1)))
        tok_off = np.concatenate([[0], np.cumsum([len(x) for x in reqs])]).astype(np.int64)
        tpl_off = np.concatenate([[0], np.cumsum([len(x) for x in tpls])]).astype(np.int64)
        toks = np.concatenate(reqs + [np.zeros(0, np.int32)]).astype(np.int32)
        tt = np.concatenate(tpls + [np.zeros(0, np.int32)]).astype(np.int32)
        got, flag = oracle.divergence_boundary(toks, tok_off, np.array(ids, np.int32), tt, tpl_off)
        want, bad = [], False
        for req, i in zip(reqs, ids):
            if i < -2 or i >= len(tpls):
                want.append(0)
                bad = True
            elif i == -1:
                want.append(0)
            elif i == -2:
                want.append(max([_lcp_python(req, t) for t in tpls], default=0))
            else:
                want.append(_lcp_python(req, tpls[i]))
        assert list(got) == want and flag == bad, trial


def pin_boundary_paper_layout():
    """Section 5.7 again, through boundary detection: a 2119-token request
    whose preamble is registered and which diverges at token 1990 gets its
    boundary at block 124; diverging at token 5, at block 0.  Salting there
    (section 4.2) leaves another principal exactly those leading blocks."""
    ex = _paper()["divergence_layout"]
    n = ex["prompt_tokens"]
    rng = np.random.default_rng(23)
    pre = rng.integers(0, W.VOCAB, n, dtype=np.int32)
    salts = oracle.derive_salts(b"z" * 32, *W.principal_ids(2))
    for i, want in zip(ex["diverge_at_token"], ex["hit_blocks"]):
        req = pre.copy()
        req[i] = (req[i] + 1) % W.VOCAB
        b, _ = oracle.divergence_boundary(req, np.array([0, n], np.int64), np.array([0], np.int32), pre,
                                          np.array([0, n], np.int64))
        assert int(b[0]) == i and int(b[0]) // 16 == want
        assert _prefix(BOUNDARY, req, 0, req, 1, salts, b=int(b[0])) == want


def pin_boundary_workload_preambles():
    """Registering the template's first 96 tokens (up to its first field) gives
    every template request boundary 96, and the wide batch's shared 64-token
    prefix gives 64: the boundaries those workloads are built with."""
    w = W.template(n_req=512)
    b = w.batch
    first = b.tokens[int(b.tok_off[0]):int(b.tok_off[0]) + 96]
    got, flag = oracle.divergence_boundary(b.tokens, b.tok_off, np.zeros(b.n, np.int32), first,
                                           np.array([0, 96], np.int64))
    assert not flag and (got == 96).all() and (got == b.boundary_tok).all()
    w = W.wide(seed=5, n_req=300)
    b = w.batch
    got, _ = oracle.divergence_boundary(b.tokens, b.tok_off, np.full(b.n, -2, np.int32), b.tokens[:64],
                                        np.array([0, 64], np.int64))
    assert (got == 64).all() and (got == b.boundary_tok).all()


# ------------------------------------------------------ exact-response key
def pin_response_key_hashlib():
    """Exact-response keys == hashlib over sigma_p || struct-packed tokens
    (and over the tokens alone unsalted), for prompts of every length 0..70
    tokens (all padding edges of a 32-byte salt plus 4-byte tokens) and a
    2119-token prompt."""
    salts = oracle.derive_salts(b"resp", *W.principal_ids(3))
    rng = np.random.default_rng(24)
    lens = list(range(71)) + [2119]
    reqs = [rng.integers(0, W.VOCAB, n, dtype=np.int32) for n in lens]
    tok_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    toks = np.concatenate(reqs).astype(np.int32)
    pr = (np.arange(len(lens)) % 3).astype(np.int32)
    root = oracle.response_key(ROOT, toks, tok_off, pr, salts)
    plain = oracle.response_key(UNSALTED, toks, tok_off, pr, salts)
    for r, t in enumerate(reqs):
        assert root[r].tobytes() == H(salts[pr[r]].tobytes() + block_le(t)), r
        assert plain[r].tobytes() == H(block_le(t)), r


def pin_response_key_whole_prompt():
    """The exact-response key covers every token (a change in a 7-token tail
    changes it, while the block chain ignores the tail), and it separates
    principals on identical prompts (section 4.1)."""
    salts = oracle.derive_salts(b"resp2", *W.principal_ids(2))
    rng = np.random.default_rng(25)
    a = rng.integers(0, W.VOCAB, 2119, dtype=np.int32)
    b = a.copy()
    b[-1] = (b[-1] + 1) % W.VOCAB
    toks = np.concatenate([a, b, a]).astype(np.int32)
    off = np.array([0, 2119, 4238, 6357], np.int64)
    pr = np.array([0, 0, 1], np.int32)
    k = oracle.response_key(ROOT, toks, off, pr, salts)
    assert k[0].tobytes() != k[1].tobytes() and k[0].tobytes() != k[2].tobytes()
    d = oracle.chain_hash(UNSALTED, toks[:4238], off[:3], pr[:2], salts, np.zeros(2, np.int32))
    assert (d[:132] == d[132:]).all()                  # the blocks never see the tail


# ------------------------------------------------------ ORIGAMI (section 4.3)
def pin_origami_linear_program():
    """The allocation == scipy's LP solution of the epigraph form the paper's
    proof uses: minimise t subject to v_i (1 - p_i) <= t, sum p = K,
    0 <= p <= 1.  t* is the water level and p* the probabilities."""
    from scipy.optimize import linprog
    rng = np.random.default_rng(26)
    for trial in range(25):
        n = int(rng.integers(2, 12))
        v = (1.0 + rng.pareto(1.29, n)).astype(np.float32)
        K = float(np.float32(rng.uniform(0.2, n - 0.2)))
        c = np.zeros(n + 1)
        c[-1] = 1.0
        A = np.zeros((n, n + 1))
        A[np.arange(n), np.arange(n)] = -v.astype(np.float64)
        A[:, -1] = -1.0
        res = linprog(c, A_ub=A, b_ub=-v.astype(np.float64), A_eq=np.concatenate([np.ones(n), [0.0]])[None],
                      b_eq=[K], bounds=[(0, 1)] * n + [(None, None)], method="highs")
        assert res.status == 0
        p, lam, u, flag = oracle.origami(v, np.array([0, n], np.int64), np.array([K], np.float32))
        assert not flag
        assert abs(lam[0] - res.x[-1]) <= 1e-7 * max(1.0, res.x[-1]), trial
        assert np.abs(p - res.x[:n]).max() <= 1e-6, trial
        assert abs(u[0] - res.fun) <= 1e-7 * max(1.0, res.fun)


def pin_origami_bisection():
    """The paper finds lambda by bisection on sum_i max(0, 1 - lambda/v_i) = K;
    a plain Python bisection (fp64, 200 halvings) lands on the oracle's level."""
    rng = np.random.default_rng(27)
    b = W.audit(seed=27, n_prob=40, n_tenants=50)
    p, lam, _, _ = oracle.origami(b.values, b.off, b.budget)
    for q in range(b.n):
        v = [float(x) for x in b.values[b.off[q]:b.off[q + 1]]]
        K = float(b.budget[q])
        lo, hi = 0.0, max(v)
        for _ in range(200):
            mid = (lo + hi) / 2
            if sum(max(0.0, 1.0 - mid / x) for x in v) > K:
                lo = mid
            else:
                hi = mid
        assert abs((lo + hi) / 2 - lam[q]) <= 1e-12 * lam[q], q
    del rng


def pin_origami_closed_forms():
    """Equal values: p = K/n, the same as uniform random audit (section 5.4);
    K >= n: every tenant audited, lambda = 0; K = 0: none, lambda = max v;
    tenants of value <= 0 get nothing; and on Pareto batches the water-filling
    properties: sum p = K, 0 <= p <= 1, v (1 - p) = lambda where p > 0,
    v <= lambda where p = 0, utility = lambda."""
    v = np.array([3.0] * 10 + [2, 4, 8] + [5, 1] + [-1.0, 0.0, 7.0], np.float32)
    off = np.array([0, 10, 13, 15, 18], np.int64)
    K = np.array([5, 3.5, 0, 1], np.float32)
    p, lam, u, flag = oracle.origami(v, off, K)
    assert not flag
    assert np.allclose(p[:10], 0.5) and abs(lam[0] - 1.5) < 1e-12 and abs(u[0] - 1.5) < 1e-12
    assert np.allclose(p[10:13], 1.0) and lam[1] == 0.0           # K capped at n
    assert np.allclose(p[13:15], 0.0) and lam[2] == 5.0 and u[2] == 5.0
    assert list(p[15:18]) == [0.0, 0.0, 1.0] and lam[3] == 0.0     # one usable tenant, K = 1
    b = W.audit(seed=28, n_prob=200, n_tenants=50)
    p, lam, u, _ = oracle.origami(b.values, b.off, b.budget)
    for q in range(b.n):
        s, e = int(b.off[q]), int(b.off[q + 1])
        pq, vq = p[s:e], b.values[s:e].astype(np.float64)
        assert abs(pq.sum() - b.budget[q]) < 1e-9 and (pq >= 0).all() and (pq <= 1).all()
        act = pq > 0
        assert np.allclose(vq[act] * (1 - pq[act]), lam[q], rtol=1e-12)
        assert (vq[~act] <= lam[q] * (1 + 1e-12)).all() and abs(u[q] - lam[q]) <= 1e-12 * lam[q]


PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_") and callable(v)]
