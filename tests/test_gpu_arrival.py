"""Arrival-order serving on the GPU (kvgov_insert_arrival + kvgov_probe_arrival)
against the oracle's request-by-request replay: bit-exact prefix lengths,
insert counts, table contents and slot handles, on synthetic key sequences
and on the workloads.  Marked gpu."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_09225_gb300 import workloads as W
from paper_2608_09225_gb300.pipeline import DeviceBatch, PrefixCache, next_pow2
from tests.table_layout import table_keys

pytestmark = pytest.mark.gpu
DEV = "cuda"
NO_SLOT = -1          # 0xFFFFFFFF read as int32


def dev(a, dtype=None):
    return torch.from_numpy(np.ascontiguousarray(a if dtype is None else np.asarray(a, dtype=dtype))).to(DEV)


def status_tensor():
    return torch.zeros(1, dtype=torch.int32, device=DEV)




class Arrival:
    """A table with its owner array, served batch after batch."""

    def __init__(self, kv, capacity):
        self.kv = kv
        self.slots = kv.new_table(capacity)
        self.owner = kv.new_owner(capacity)
        self.status = status_tensor()
        self.n_new = torch.zeros(1, dtype=torch.int64, device=DEV)
        self.seq = 1

    def serve(self, digests, blk_off):
        d, b = dev(digests, np.uint8).reshape(-1, 32), dev(blk_off, np.int64)
        slot_of = self.kv.insert_arrival(self.slots, self.owner, d, b, self.seq, self.status, n_new=self.n_new)
        pre = self.kv.probe_arrival(self.owner, slot_of, b, self.seq, status=self.status)
        self.seq += int(blk_off[-1])
        torch.cuda.synchronize()
        return pre.cpu().numpy(), slot_of.cpu().numpy()


def sequences(seed, n_req, pool_n=64, max_blocks=12, side=0, zero=False):
    """Requests as key sequences that often start with a copy of an earlier
    request's leading keys (the structure of shared prefixes).  `side` pool
    keys take the patterns a main slot cannot hold (zero first half, zero
    third or fourth 8-byte word); `zero` makes the last pool key all-zero."""
    rng = np.random.default_rng(seed)
    pool = rng.integers(0, 256, (pool_n, 32), dtype=np.uint8)
    pool[:, 0] |= 1
    for i in range(side):
        pool[i, (slice(0, 16), slice(16, 24), slice(24, 32))[i % 3]] = 0
    if zero:
        pool[-1] = 0
    reqs = []
    for _ in range(n_req):
        keys = list(rng.integers(0, pool_n, int(rng.integers(0, max_blocks))))
        if reqs and rng.random() < 0.7:
            src = reqs[int(rng.integers(0, len(reqs)))]
            keys = list(src[: int(rng.integers(0, len(src) + 1))]) + keys
        reqs.append(keys)
    off = np.concatenate([[0], np.cumsum([len(k) for k in reqs])]).astype(np.int64)
    idx = np.array([i for k in reqs for i in k], dtype=np.int64)
    return pool, pool[idx].reshape(-1, 32), off


@pytest.mark.parametrize("n_req,cap_log2", [(1, 6), (37, 10), (600, 12), (5000, 16)])
def test_arrival_matches_replay(kv, n_req, cap_log2):
    pool, d, off = sequences(100 + n_req, n_req)
    a = Arrival(kv, 1 << cap_log2)
    pre, slot_of = a.serve(d, off)
    want, n_new = oracle.KeySet(1).arrival_prefix(d, off)
    assert int(a.status.item()) == 0
    assert (pre == want).all()
    assert int(a.n_new.item()) == n_new
    s = a.slots.cpu().numpy()
    assert (s[slot_of] == d).all()                     # each block's handle holds its key
    assert table_keys(a.slots) == {r.tobytes() for r in d}


def test_arrival_batches_in_sequence_and_plain_inserts(kv):
    """Keys cached before a batch -- by kvgov_insert (owner 0) or by an earlier
    arrival batch -- count as cached for every request of the batch."""
    pool, d1, off1 = sequences(7, 300)
    _, d2, off2 = sequences(8, 400)
    plain = np.random.default_rng(9).integers(1, 256, (41, 32), dtype=np.uint8)
    # batch 2: request 0 = three plainly inserted keys and a new one; then the
    # random requests; then one request made of batch 1's first 50 keys
    d2 = np.concatenate([plain[:3], plain[40:41], d2, d1[:50]])
    off2 = np.concatenate([[0], 4 + off2, [4 + off2[-1] + 50]]).astype(np.int64)
    plain = plain[:40]
    a = Arrival(kv, 1 << 14)
    kv.insert(a.slots, dev(plain), a.status, a.n_new)
    pre1, _ = a.serve(d1, off1)
    pre2, _ = a.serve(d2, off2)
    ks = oracle.KeySet(1)
    ks.insert(plain)
    w1, n1 = ks.arrival_prefix(d1, off1)
    ks.insert(d1)
    w2, n2 = ks.arrival_prefix(d2, off2)
    assert int(a.status.item()) == 0
    assert (pre1 == w1).all() and (pre2 == w2).all()
    assert int(a.n_new.item()) == 40 + n1 + n2
    assert pre2[-1] == 50 and pre2[0] == 3


def test_arrival_side_store_keys_and_the_zero_key(kv):
    """Keys a main slot cannot hold (zero first half or a zero 8-byte word in
    the second half), shared by many requests' prefixes, are served like any
    other key: their handles point into the side store and hold them, and
    prefix lengths and key counts match the oracle's replay.  The all-zero
    key is flagged, gets no handle and ends its request's prefix."""
    for seed, n_req in ((11, 50), (12, 3000)):
        pool, d, off = sequences(seed, n_req, pool_n=20, side=6, zero=True)
        a = Arrival(kv, 1 << 12)
        pre, slot_of = a.serve(d, off)
        want, n_new = oracle.KeySet(1).arrival_prefix(d, off)
        zero_rows = ~d.any(axis=1)
        assert zero_rows.any() and int(a.status.item()) == kv.F_SENTINEL
        assert (slot_of[zero_rows] == NO_SLOT).all()
        assert (pre == want).all() and int(a.n_new.item()) == n_new
        s = a.slots.cpu().numpy()
        ok = ~zero_rows
        assert (s[slot_of[ok]] == d[ok]).all()                   # each handle holds its block's key
        side_rows = ok & (~d[:, :16].any(axis=1) | ~d[:, 16:24].any(axis=1) | ~d[:, 24:].any(axis=1))
        assert side_rows.any() and (slot_of[side_rows] >= (1 << 12)).all()
        assert table_keys(a.slots) == {r.tobytes() for r in d[ok]}


def test_arrival_full_and_empty(kv):
    """A full table flags and ends the prefix at the block it could not
    store; empty batches and empty requests are no-ops."""
    # a 32-slot table and 64 distinct keys
    k = np.random.default_rng(12).integers(1, 256, (64, 32), dtype=np.uint8)
    b = Arrival(kv, 32)
    off = np.arange(0, 65, 8, dtype=np.int64)
    pre, slot_of = b.serve(np.concatenate([k]), off)
    assert int(b.status.item()) & kv.F_TABLE_FULL
    assert int(b.n_new.item()) == 32 and (slot_of == NO_SLOT).sum() == 32
    # empty batch, empty requests
    c = Arrival(kv, 64)
    pre, _ = c.serve(np.zeros((0, 32), np.uint8), np.zeros(1, np.int64))
    assert pre.shape == (0,)
    pre, _ = c.serve(np.zeros((0, 32), np.uint8), np.zeros(4, np.int64))
    assert list(pre) == [0, 0, 0] and int(c.status.item()) == 0


def test_arrival_rejects_bad_sequence_numbers(kv):
    a = Arrival(kv, 64)
    d, b = dev(np.ones((2, 32), np.uint8)), dev(np.array([0, 1, 2], np.int64))
    for seq in (0, (1 << 62) + 1):
        with pytest.raises(kv.KVGovError):
            kv.insert_arrival(a.slots, a.owner, d, b, seq, a.status)
    with pytest.raises(kv.KVGovError):
        kv.probe_arrival(a.owner, torch.zeros(2, dtype=torch.int32, device=DEV), b, 0)


# ------------------------------------------------------------ the workloads
def serve_workload(kv, w, mode, fill=False):
    """Chains on the GPU, then one arrival-order batch into an empty cache
    (or, with fill, a cache holding the workload's table content)."""
    b = w.batch
    cap = w.capacity if fill else next_pow2(4 * int((b.lengths() // 16).sum()))
    cache = PrefixCache(cap, w.secret, w.ids, w.id_off)
    db = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
    blk, d = cache.hash(mode, db)
    owner = kv.new_owner(cache.capacity)
    if fill and w.random_keys is not None:
        cache.insert(torch.from_numpy(w.random_keys).cuda())
    slot_of = kv.insert_arrival(cache.slots, owner, d, blk, 1, cache.status, n_new=cache.n_new)
    pre = kv.probe_arrival(owner, slot_of, blk, 1, status=cache.status)
    torch.cuda.synchronize()
    cache.check_status()
    return cache, d.cpu().numpy(), blk.cpu().numpy(), pre.cpu().numpy()


def oracle_arrival(w, mode, fill=False):
    salts = oracle.derive_salts(w.secret, w.ids, w.id_off)
    b = w.batch
    d = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    blk = oracle.block_offsets(b.tok_off)
    ks = oracle.KeySet(1)
    if fill and w.random_keys is not None:
        ks.insert(w.random_keys)
    L, n_new = ks.arrival_prefix(d, blk)
    return d, L, n_new + ks.n


def test_arrival_tiny_closed_form(kv):
    _, _, _, pre = serve_workload(kv, W.make("tiny"), W.ROOT)
    assert list(pre) == [0] * 8 + [8] * 24 + [0] * 32


@pytest.mark.parametrize("mode", [W.UNSALTED, W.ROOT, W.BOUNDARY])
def test_arrival_template_full(kv, mode):
    """The 8192-request template workload served in arrival order: the hit
    blocks a serving cache sees, per salt placement, equal the replay's."""
    w = W.make("template")
    cache, d, _, pre = serve_workload(kv, w, mode)
    dref, L, n_keys = oracle_arrival(w, mode)
    assert (d == dref).all()
    assert (pre == L).all()
    assert int(cache.n_new.item()) == n_keys


def test_arrival_sysprompt_full(kv):
    w = W.make("sysprompt")
    cache, _, _, pre = serve_workload(kv, w, W.ROOT)
    _, L, n_keys = oracle_arrival(w, W.ROOT)
    assert (pre == L).all() and int(cache.n_new.item()) == n_keys


def test_arrival_probe_heavy_full(kv):
    """65,536 requests into the 2^24-slot table holding 8.1 M random keys."""
    w = W.make("probe")
    cache, _, _, pre = serve_workload(kv, w, W.ROOT, fill=True)
    _, L, n_keys = oracle_arrival(w, W.ROOT, fill=True)
    assert (pre == L).all() and int(cache.n_new.item()) == n_keys


def test_arrival_wide_full(kv):
    w = W.make("wide", seed=41)
    cache, _, _, pre = serve_workload(kv, w, W.BOUNDARY)
    _, L, n_keys = oracle_arrival(w, W.BOUNDARY)
    assert (pre == L).all() and int(cache.n_new.item()) == n_keys
    assert pre[0] == 0 and (pre[1:] >= 4).all()         # the shared 64-token prefix is unsalted


# ------------------------------------------------- chain hash + arrival in one call
def shared_prefix_batch(seed, n_req):
    """Requests that start with one of four 200-token prompts (cut at a
    random length, then their own tokens), a tenth of them an exact repeat
    of an earlier request by the same principal; principals 0..7; boundary
    offsets cycling as in workloads.ragged."""
    rng = np.random.default_rng(seed)
    prompts = rng.integers(0, W.VOCAB, (4, 200), dtype=np.int32)
    reqs, principal = [], []
    for r in range(n_req):
        if reqs and rng.random() < 0.1:
            src = int(rng.integers(0, len(reqs)))
            reqs.append(reqs[src].copy())
            principal.append(principal[src])
            continue
        cut = int(rng.integers(0, 200))
        own = rng.integers(0, W.VOCAB, int(rng.integers(0, 120)), dtype=np.int32)
        reqs.append(np.concatenate([prompts[int(rng.integers(0, 4))][:cut], own]).astype(np.int32))
        principal.append(int(rng.integers(0, 8)))
    tok_off = np.concatenate([[0], np.cumsum([len(t) for t in reqs])]).astype(np.int64)
    cyc = np.array([0, 15, 16, 17, 31, 32, 64, 10 ** 6], dtype=np.int32)
    return W.Batch(tokens=np.concatenate(reqs).astype(np.int32), tok_off=tok_off,
                   principal=np.array(principal, np.int32), boundary_tok=cyc[np.arange(n_req) % len(cyc)])


@pytest.mark.parametrize("mode", [W.UNSALTED, W.ROOT, W.BOUNDARY])
@pytest.mark.parametrize("n_req", [180, 40960], ids=["separate_launches", "fused"])
def test_chain_hash_arrival_matches_oracle_and_separate_calls(kv, mode, n_req):
    """kvgov_chain_hash_arrival gives the oracle's digests and arrival-order
    prefix lengths, and the table, key count and prefix lengths of the
    separate calls, for a batch small enough for separate launches and one
    that takes the fused kernel; keys cached before the batch count."""
    b = shared_prefix_batch(500 + n_req + mode, n_req)
    salts = oracle.derive_salts(b"arrival", *W.principal_ids(8))
    ref = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    blk_ref = oracle.block_offsets(b.tok_off)
    early = ref[np.random.default_rng(mode).random(len(ref)) < 0.05]     # cached before the batch
    ks = oracle.KeySet(1)
    ks.insert(early)
    want, n_batch = ks.arrival_prefix(ref, blk_ref)
    cap = next_pow2(4 * len(ref))
    toks, tok_off = dev(b.tokens, np.int32), dev(b.tok_off, np.int64)
    pr, sl, bt = dev(b.principal, np.int32), dev(salts), dev(b.boundary_tok, np.int32)
    outs = []
    for fused_call in (True, False):
        a = Arrival(kv, cap)
        kv.insert(a.slots, dev(early), a.status, a.n_new)
        blk = kv.block_offsets(tok_off, status=a.status)
        if fused_call:
            d, slot_of, pre = kv.chain_hash_arrival(mode, toks, tok_off, blk, a.slots, a.owner, 7, a.status, pr, sl, bt,
                                                    n_blocks=len(ref), n_new=a.n_new)
        else:
            d = kv.chain_hash(mode, toks, tok_off, blk, pr, sl, bt, n_blocks=len(ref), status=a.status)
            slot_of = kv.insert_arrival(a.slots, a.owner, d, blk, 7, a.status, n_new=a.n_new)
            pre = kv.probe_arrival(a.owner, slot_of, blk, 7, status=a.status)
        torch.cuda.synchronize()
        assert int(a.status.item()) == 0
        assert (d.cpu().numpy() == ref).all()
        so = slot_of.cpu().numpy()
        assert (a.slots.cpu().numpy()[so] == ref).all()
        assert (pre.cpu().numpy() == want).all()
        assert int(a.n_new.item()) == ks.n + n_batch
        outs.append(table_keys(a.slots))
    assert outs[0] == outs[1]
    assert want.max() > 0 and (want == 0).any()


@pytest.mark.parametrize("name", ["wide", "probe", "template"])
def test_chain_hash_arrival_full_workloads(kv, name):
    """The one-call path at full size: the wide batch (131,072 requests, the
    fused kernel, 4 shared-prefix keys inserted by every request), the
    probe-heavy batch into its table of 8.1 M keys (fused), and the 8192
    template requests (separate launches)."""
    w = W.make(name, seed=43) if name == "wide" else W.make(name)
    mode = W.BOUNDARY if name != "probe" else W.ROOT
    fill = name == "probe"
    b = w.batch
    n_blocks = int((b.lengths() // 16).sum())
    cap = w.capacity if fill else next_pow2(4 * n_blocks)
    cache = PrefixCache(cap, w.secret, w.ids, w.id_off)
    db = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
    owner = kv.new_owner(cap)
    if fill:
        cache.insert(torch.from_numpy(w.random_keys).cuda())
    blk = kv.block_offsets(db.tok_off, status=cache.status)
    d, slot_of, pre = kv.chain_hash_arrival(mode, db.tokens, db.tok_off, blk, cache.slots, owner, 1 << 40,
                                            cache.status, db.principal, cache.salts, db.boundary_tok,
                                            n_blocks=n_blocks, n_new=cache.n_new)
    torch.cuda.synchronize()
    cache.check_status()
    dref, L, n_keys = oracle_arrival(w, mode, fill)
    assert (d.cpu().numpy() == dref).all()
    assert (pre.cpu().numpy() == L).all()
    assert int(cache.n_new.item()) == n_keys
    so = slot_of.cpu().numpy()
    assert (so >= 0).all() and (cache.slots.cpu().numpy()[so] == dref).all()
