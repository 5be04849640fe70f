"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle,
bit-exact on every salt, block offset, digest, prefix length and insert
count; plus the device-detected error flags.  Marked gpu."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2608_09225_gb300 import workloads as W
from tests.table_layout import table_keys

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
DEV = "cuda"


def dev(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a if dtype is None else np.asarray(a, dtype=dtype)))
    return t.to(DEV)


def status_tensor():
    return torch.zeros(1, dtype=torch.int32, device=DEV)


def gpu_chain(kv, mode, b: W.Batch, salts_np, status=None):
    toks = dev(b.tokens, np.int32)
    tok_off = dev(b.tok_off, np.int64)
    blk = kv.block_offsets(tok_off, status=status)
    n_blocks = int((np.diff(b.tok_off) // 16).sum())
    d = kv.chain_hash(mode, toks, tok_off, blk, dev(b.principal, np.int32), dev(salts_np, np.uint8),
                      dev(b.boundary_tok, np.int32), n_blocks=n_blocks, status=status)
    torch.cuda.synchronize()
    return blk.cpu().numpy(), d.cpu().numpy()


# ----------------------------------------------------------------- salts
@pytest.mark.parametrize("secret_len", [0, 1, 32, 63, 64, 65, 200, 1024])
def test_salts_match_oracle(kv, secret_len):
    rng = np.random.default_rng(secret_len)
    secret = rng.integers(0, 256, secret_len, dtype=np.uint8).tobytes()
    ids, id_off = W.principal_ids(4096)
    s = kv.derive_salts(secret, dev(ids), dev(id_off))
    torch.cuda.synchronize()
    assert (s.cpu().numpy() == oracle.derive_salts(secret, ids, id_off)).all()


def test_salts_variable_length_ids(kv):
    rng = np.random.default_rng(21)
    lens = rng.integers(0, 300, 777)
    lens[:10] = [0, 1, 55, 56, 63, 64, 119, 120, 0, 200]
    off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    ids = rng.integers(0, 256, int(off[-1]), dtype=np.uint8)
    secret = b"server secret"
    s = kv.derive_salts(secret, dev(ids), dev(off))
    torch.cuda.synchronize()
    assert (s.cpu().numpy() == oracle.derive_salts(secret, ids, off)).all()


def test_salts_bad_offsets_flagged(kv):
    ids, off = W.principal_ids(4)
    off = off.copy()
    off[2] = 1          # principal 1 has a decreasing range
    st = status_tensor()
    salts = torch.zeros((4, 32), dtype=torch.uint8, device=DEV)
    kv.derive_salts(b"k", dev(ids), dev(off), salts, st)
    torch.cuda.synchronize()
    assert int(st.item()) & kv.F_BADINDEX
    ref = oracle.derive_salts(b"k", ids, W.principal_ids(4)[1])
    assert (salts.cpu().numpy()[[0, 3]] == ref[[0, 3]]).all()


# --------------------------------------------------------- block offsets
@pytest.mark.parametrize("n", [0, 1, 5, 127, 1024, 1025, 4097, 10000, 131073, 1000003, 1 << 20, (1 << 20) + 1,
                               3000001])
def test_block_offsets(kv, n):
    rng = np.random.default_rng(n)
    lens = rng.integers(0, 200, n)
    tok_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    st = status_tensor()
    blk = kv.block_offsets(dev(tok_off), status=st)
    torch.cuda.synchronize()
    assert (blk.cpu().numpy() == oracle.block_offsets(tok_off)).all()
    assert int(st.item()) == 0


def test_block_offsets_reused_output_and_side_stream(kv):
    """The output array doubles as the scan's mailboxes: values left in it by
    an earlier call must not leak into the next one, and the scan must give
    the same result on a second stream while a chain-hash launch runs."""
    rng = np.random.default_rng(5)
    offs = [np.concatenate([[0], np.cumsum(rng.integers(0, 300, 200000))]).astype(np.int64) for _ in range(3)]
    out = torch.full((200001,), -7, dtype=torch.int64, device="cuda")
    b = W.make("wide", seed=3, n_req=16384)
    db_tok, db_off = dev(b.batch.tokens), dev(b.batch.tok_off)
    blk_b = kv.block_offsets(db_off)
    side = torch.cuda.Stream()
    for t in offs:
        st = status_tensor()
        kv.chain_hash(0, db_tok, db_off, blk_b, n_blocks=16384 * 8)
        ev = torch.cuda.Event()
        ev.record()
        side.wait_event(ev)
        kv.block_offsets(dev(t), out, st, side)
        torch.cuda.synchronize()
        assert (out.cpu().numpy() == oracle.block_offsets(t)).all()
        assert int(st.item()) == 0


def test_block_offsets_negative_length_flagged(kv):
    tok_off = np.array([0, 16, 8, 40], dtype=np.int64)
    st = status_tensor()
    kv.block_offsets(dev(tok_off), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & kv.F_BADINDEX


# ------------------------------------------------------------------ chain
RAGGED = [0, 15, 16, 17, 31, 32, 33, 2119, 64, 100, 7, 48, 3, 19, 257, 1, 128, 129, 130, 131]


def split_limit():
    """Largest batch the chain hash runs on its small-batch kernel (one
    round warp and one schedule warp per 32 chains, 64 chains per SM)."""
    return 64 * torch.cuda.get_device_properties(0).multi_processor_count


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("lengths", [RAGGED, RAGGED * 17, [3, 16], [1, 16 * 9 + 2], [5] * 300, RAGGED * 600],
                         ids=["ragged", "ragged_many_ctas", "tail_at_array_end", "tail2", "all_short",
                              "ragged_above_split_limit"])
def test_chain_matches_oracle(kv, mode, lengths):
    b = W.ragged(31 + len(lengths), lengths)
    salts = oracle.derive_salts(b"salt key", *W.principal_ids(8))
    st = status_tensor()
    blk, d = gpu_chain(kv, mode, b, salts, st)
    assert int(st.item()) == 0
    ref = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    assert (blk == oracle.block_offsets(b.tok_off)).all()
    assert d.shape == ref.shape
    bad = np.nonzero((d != ref).any(axis=1))[0]
    assert len(bad) == 0, f"{len(bad)} digests differ, first rows {bad[:5]}"


@pytest.mark.parametrize("boundary", [0, 15, 16, 17, 100, 16 * 20, 16 * 39, 16 * 40, 16 * 41, 10 ** 9])
@pytest.mark.parametrize("n_req", [150, 12000], ids=["split_kernel", "chain_kernel"])
def test_chain_boundary_positions(kv, boundary, n_req):
    """k = 0, interior, last block (k = n_b - 1), past the end."""
    b = W.ragged(5, [16 * 40] * n_req)
    b.boundary_tok[:] = boundary
    salts = oracle.derive_salts(b"B", *W.principal_ids(8))
    _, d = gpu_chain(kv, 2, b, salts)
    ref = oracle.chain_hash(2, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    assert (d == ref).all()


@pytest.mark.parametrize("delta", [-1, 0, 1])
def test_chain_at_the_split_limit(kv, delta):
    """Batches at the small-batch kernel's limit and one past it, every mode,
    ragged lengths (empty, sub-block, unaligned starts, a long chain) and a
    boundary per request anywhere from block 0 to past the end."""
    n = split_limit() + delta
    lengths = (RAGGED * (n // len(RAGGED) + 1))[:n]
    b = W.ragged(77 + delta, lengths)
    rng = np.random.default_rng(5 + delta)
    b.boundary_tok[:] = rng.integers(0, 2200, n)
    salts = oracle.derive_salts(b"limit", *W.principal_ids(8))
    for mode in (0, 1, 2):
        st = status_tensor()
        _, d = gpu_chain(kv, mode, b, salts, st)
        assert int(st.item()) == 0
        ref = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
        bad = np.nonzero((d != ref).any(axis=1))[0]
        assert len(bad) == 0, f"mode {mode}: {len(bad)} digests differ, first rows {bad[:5]}"


def test_chain_against_golden_file(kv):
    with open(os.path.join(GOLDEN, "oracle_small.json")) as f:
        g = json.load(f)
    b = W.ragged(g["seed"], g["lengths"])
    ids, id_off = W.principal_ids(g["n_principals"])
    s = kv.derive_salts(bytes.fromhex(g["secret_hex"]), dev(ids), dev(id_off))
    torch.cuda.synchronize()
    salts = s.cpu().numpy()
    assert [x.tobytes().hex() for x in salts] == g["salts"]
    for name, mode in (("unsalted", 0), ("root", 1), ("boundary", 2)):
        blk, d = gpu_chain(kv, mode, b, salts)
        assert blk.tolist() == g["blk_off"]
        assert [x.tobytes().hex() for x in d] == g["digests_" + name]


def test_chain_bad_principal_flagged(kv):
    b = W.ragged(9, [64, 64, 64])
    b.principal[:] = [0, 99, 1]
    salts = oracle.derive_salts(b"k", *W.principal_ids(8))
    st = status_tensor()
    _, d = gpu_chain(kv, 1, b, salts, st)
    assert int(st.item()) & kv.F_BADINDEX
    good = b.principal.copy()
    good[1] = 0
    ref = oracle.chain_hash(1, b.tokens, b.tok_off, good, salts)
    assert (d[:4] == ref[:4]).all() and (d[8:] == ref[8:]).all()


def test_chain_negative_boundary_flagged(kv):
    b = W.ragged(9, [64, 64])
    b.boundary_tok[:] = [-5, 16]
    st = status_tensor()
    gpu_chain(kv, 2, b, oracle.derive_salts(b"k", *W.principal_ids(8)), st)
    assert int(st.item()) & kv.F_BADINDEX


# ------------------------------------------------------------------ table
def keys_np(n, seed):
    k = np.random.default_rng(seed).integers(0, 256, (n, 32), dtype=np.uint8)
    k[:, 0] |= 1
    return k




def test_insert_set_semantics(kv):
    k = keys_np(5000, 1)
    batch = np.concatenate([k, k[::-1], k[:100], k[:100]])
    slots = kv.new_table(1 << 14)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    kv.insert(slots, dev(batch), st, n_new)
    kv.insert(slots, dev(k[:777]), st, n_new)
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(n_new.item()) == 5000
    assert table_keys(slots) == {r.tobytes() for r in k}


def test_insert_heavy_in_batch_duplicates(kv):
    """One key repeated 100,000 times plus 64 keys each 512 times: every
    concurrent claim of the same key stores it once."""
    k = keys_np(65, 2)
    batch = np.concatenate([np.repeat(k[:1], 100000, axis=0), np.tile(k[1:], (512, 1))])
    batch = batch[np.random.default_rng(3).permutation(len(batch))]
    slots = kv.new_table(1 << 10)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    kv.insert(slots, dev(batch), st, n_new)
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(n_new.item()) == 65
    assert table_keys(slots) == {r.tobytes() for r in k}


def side_store_keys(n, seed):
    """n distinct keys that a main slot cannot hold, cycling through the
    patterns: first half zero, third or fourth 8-byte word zero, second half
    zero, all but the last two bytes zero."""
    k = keys_np(n, seed)
    for i in range(n):
        kind = i % 5
        if kind == 0:
            k[i, :16] = 0
        elif kind == 1:
            k[i, 16:24] = 0
        elif kind == 2:
            k[i, 24:] = 0
        elif kind == 3:
            k[i, 16:] = 0
        else:
            k[i, :30] = 0
            k[i, 30] = seed & 0xff
            k[i, 31] = 1 + i // 5
    return k


def test_insert_side_store_keys(kv):
    """Keys with a zero first half or a zero 8-byte word in the second half
    -- which a main slot cannot hold -- are stored (in the side store) and
    found, like any other key; only the all-zero key is refused.  Checked
    against the oracle's set: contents, key count, each key's lookup, and a
    request of them all hitting to its end."""
    k = np.concatenate([keys_np(12, 4), side_store_keys(10, 40)])
    k[3, :] = 0                 # all zero: refused
    k[10, :8] = 0               # first word zero alone: a main slot holds it
    k[11, :8] = 255
    slots = kv.new_table(64)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    kv.insert(slots, dev(k), st, n_new)
    kv.insert(slots, dev(k[::-1].copy()), st, n_new)          # every key again: duplicates
    torch.cuda.synchronize()
    assert int(st.item()) == kv.F_SENTINEL
    ks = oracle.KeySet(1)
    n_ref, flagged = ks.insert(k)
    assert flagged and int(n_new.item()) == n_ref == 21
    assert table_keys(slots) == {r.tobytes() for r in ks.contents()}
    pre = kv.probe(slots, dev(k), dev(np.arange(23, dtype=np.int64)))
    whole = kv.probe(slots, dev(np.delete(k, 3, axis=0)), dev(np.array([0, 21], np.int64)))
    absent = kv.probe(slots, dev(side_store_keys(10, 41)), dev(np.arange(11, dtype=np.int64)))
    torch.cuda.synchronize()
    member = {r.tobytes() for r in ks.contents()}
    assert list(pre.cpu().numpy()) == [int(r.tobytes() in member) for r in k]
    assert int(whole.item()) == 21
    assert (absent.cpu().numpy() == 0).all()


def test_side_store_concurrent_duplicates(kv):
    """Ten side-store keys, each inserted 4000 times from every part of one
    shuffled batch (with 3000 ordinary keys around them) and then once more:
    each is stored once, the count matches the oracle, every key is found."""
    side = side_store_keys(10, 42)
    plain = keys_np(3000, 43)
    batch = np.concatenate([np.repeat(side, 4000, axis=0), plain])
    batch = batch[np.random.default_rng(44).permutation(len(batch))]
    slots = kv.new_table(1 << 14)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    kv.insert(slots, dev(batch), st, n_new)
    kv.insert(slots, dev(side), st, n_new)
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(n_new.item()) == 3010
    assert table_keys(slots) == {r.tobytes() for r in np.concatenate([side, plain])}
    pre = kv.probe(slots, dev(np.concatenate([side, plain[:6]])), dev(np.array([0, 16], np.int64)))
    torch.cuda.synchronize()
    assert int(pre.item()) == 16


def test_side_store_full(kv):
    """More distinct side-store keys than it holds: KVGOV_STASH_KEYS are
    stored, the rest flagged KVGOV_F_TABLE_FULL; every stored key is found
    and a key inserted again is a duplicate, not a new entry."""
    k = side_store_keys(70, 45)
    slots = kv.new_table(32)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    kv.insert(slots, dev(k), st, n_new)
    torch.cuda.synchronize()
    assert int(st.item()) == kv.F_TABLE_FULL
    stored = table_keys(slots)
    assert int(n_new.item()) == len(stored) == kv.STASH_KEYS and stored <= {r.tobytes() for r in k}
    st2 = status_tensor()
    kept = np.array([np.frombuffer(x, np.uint8) for x in sorted(stored)])
    kv.insert(slots, dev(kept), st2, n_new)
    pre = kv.probe(slots, dev(k), dev(np.arange(71, dtype=np.int64)))
    torch.cuda.synchronize()
    assert int(st2.item()) == 0 and int(n_new.item()) == kv.STASH_KEYS
    assert list(pre.cpu().numpy()) == [int(r.tobytes() in stored) for r in k]
    kv.table_init(slots)
    torch.cuda.synchronize()
    assert table_keys(slots) == set()


def test_table_full(kv):
    k = keys_np(40, 5)
    slots = kv.new_table(32)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    kv.insert(slots, dev(k), st, n_new)
    torch.cuda.synchronize()
    assert int(st.item()) & kv.F_TABLE_FULL
    assert int(n_new.item()) == 32 and len(table_keys(slots)) == 32


def test_full_table_inserts_and_lookups_stay_bounded(kv):
    """A table filled to the end: further inserts report TABLE_FULL after at
    most one probe window of slots, and lookups of absent keys end."""
    cap = 4096
    k = keys_np(cap + 500, 8)
    slots = kv.new_table(cap)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    kv.insert(slots, dev(k), st, n_new)
    torch.cuda.synchronize()
    assert int(st.item()) & kv.F_TABLE_FULL
    stored = table_keys(slots)
    # with the probe window a nearly full table may refuse a key before the
    # last slot is taken; every refusal is flagged and every store counted
    assert int(n_new.item()) == len(stored) and len(stored) > 0.9 * cap
    assert stored <= {r.tobytes() for r in k}
    absent = keys_np(300, 9)
    pre = kv.probe(slots, dev(absent), dev(np.arange(301, dtype=np.int64)))
    pre_k = kv.probe(slots, dev(k), dev(np.arange(cap + 501, dtype=np.int64)))
    torch.cuda.synchronize()
    assert (pre.cpu().numpy() == 0).all()
    assert list(pre_k.cpu().numpy()) == [int(r.tobytes() in stored) for r in k]


def test_insert_wait_times_out_on_a_slot_nobody_finishes(kv):
    """A slot holding a key's first 16 bytes whose second half is never
    written (as if its writer stopped): an insert of that key waits a bounded
    number of times, reports KVGOV_F_TIMEOUT and returns; a probe of the key
    does not match the half-written slot."""
    cap = 64
    k = keys_np(1, 6)
    home = int(k[0, :8].view(np.uint64)[0]) & (cap - 1)
    slots = kv.new_table(cap)
    slots[home, :16] = torch.from_numpy(k[0, :16].copy()).to(DEV)
    st = status_tensor()
    prev = kv.set_spin_limit(1000)
    try:
        kv.insert(slots, dev(k), st)
        torch.cuda.synchronize()
    finally:
        kv.set_spin_limit(prev)
    assert int(st.item()) == kv.F_TIMEOUT
    blk = dev(np.array([0, 1], np.int64))
    pre = kv.probe(slots, dev(k), blk)
    torch.cuda.synchronize()
    assert int(pre.item()) == 0


@pytest.mark.parametrize("cap_log2", [5, 10, 16])
def test_probe_matches_oracle(kv, cap_log2):
    """Random chains of known digests against a table holding a random subset:
    prefix length = first missing block (later hits ignored)."""
    rng = np.random.default_rng(cap_log2)
    pool = keys_np(min(1 << (cap_log2 - 1), 4000), cap_log2 + 100)
    nb = rng.integers(0, 70, 3000)
    nb[:5] = [0, 1, 33, 64, 69]
    off = np.concatenate([[0], np.cumsum(nb)]).astype(np.int64)
    digests = pool[rng.integers(0, len(pool), int(off[-1]))]
    member = rng.random(len(pool)) < 0.85
    slots = kv.new_table(1 << cap_log2)
    st = status_tensor()
    kv.insert(slots, dev(pool[member]), st)
    pre = kv.probe(slots, dev(digests), dev(off), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ks = oracle.KeySet(1)
    ks.insert(pool[member])
    assert (pre.cpu().numpy() == ks.prefix_blocks(digests, off)).all()


@pytest.mark.parametrize("n_req,max_nb,p_member", [(700, 400, 0.995), (3000, 70, 0.6), (20000, 150, 0.99),
                                                    (40000, 40, 0.9), (40000, 3, 0.5), (70000, 300, 0.999)],
                         ids=["few_long", "mid_short", "mid_long", "many", "many_tiny_requests", "many_long"])
def test_probe_layouts_match_oracle(kv, n_req, max_nb, p_member):
    """Every probe layout (a warp per request below 2048 requests, 16 lanes
    per request up to 32,768, above that 16 requests per warp sharing its
    lanes), with requests of 0, 1 and 2 blocks, prefixes that span several
    rounds (up to 400 blocks), and prefixes that end exactly at a window's
    edge."""
    rng = np.random.default_rng(n_req + max_nb)
    pool = keys_np(6000, n_req % 997 + 3)
    nb = rng.integers(0, max_nb + 1, n_req)
    nb[:8] = [0, 1, 2, 1, 0, max_nb, 33, 129][:8] if max_nb >= 129 else [0, 1, 2, 1, 0, max_nb, 0, 1]
    off = np.concatenate([[0], np.cumsum(nb)]).astype(np.int64)
    digests = pool[rng.integers(0, len(pool), int(off[-1]))]
    member = rng.random(len(pool)) < p_member
    # request 6 misses exactly at block 32 (the end of a warp's first window),
    # request 7 at block 128, when they are that long
    for r, j in ((6, 32), (7, 128)):
        if nb[r] > j:
            digests[off[r]:off[r] + j] = pool[np.nonzero(member)[0][:j]]
            digests[off[r] + j] = pool[np.nonzero(~member)[0][0]]
    slots = kv.new_table(1 << 14)
    st = status_tensor()
    kv.insert(slots, dev(pool[member]), st)
    pre = kv.probe(slots, dev(digests), dev(off), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ks = oracle.KeySet(1)
    ks.insert(pool[member])
    want = ks.prefix_blocks(digests, off)
    got = pre.cpu().numpy()
    assert (got == want).all(), f"{int((got != want).sum())} of {n_req} prefix lengths differ"
    if max_nb >= 129:
        assert want[6] == 32 and want[7] == 128
    assert want.max() > (100 if max_nb >= 300 else 0)


@pytest.mark.parametrize("n_req,max_nb", [(700, 400), (3000, 70), (40000, 40), (70000, 300)],
                         ids=["few", "mid", "many", "many_long"])
def test_probe_resume_from_lower_bounds(kv, n_req, max_nb):
    """kvgov_probe_resume, every layout: starting each request's walk at any
    lower bound of its prefix (0, the prefix itself, a random value between,
    a negative entry, a bound inside a window or at its edge) gives the
    prefix lengths of the oracle's set (paper section 2.1), as kvgov_probe
    does from block 0."""
    rng = np.random.default_rng(3 * n_req + max_nb)
    pool = keys_np(6000, n_req % 991 + 11)
    nb = rng.integers(0, max_nb + 1, n_req)
    nb[:6] = [0, 1, 2, max_nb, max_nb, max_nb]
    off = np.concatenate([[0], np.cumsum(nb)]).astype(np.int64)
    digests = pool[rng.integers(0, len(pool), int(off[-1]))]
    member = rng.random(len(pool)) < 0.97
    digests[off[3]:off[4]] = pool[np.nonzero(member)[0][:max_nb]]      # request 3: every block cached
    slots = kv.new_table(1 << 14)
    st = status_tensor()
    kv.insert(slots, dev(pool[member]), st)
    ks = oracle.KeySet(1)
    ks.insert(pool[member])
    want = ks.prefix_blocks(digests, off)
    assert want[3] == max_nb and want.max() > 3
    d_dig, d_off = dev(digests), dev(off)
    bounds = {
        "zero": np.zeros(n_req, np.int32),
        "exact": want.astype(np.int32),
        "between": (rng.random(n_req) * (want + 1)).astype(np.int32),
        "negative": np.where(rng.random(n_req) < 0.5, -rng.integers(1, 5, n_req), want).astype(np.int32),
        "window_edge": np.minimum(want, 32 * (want // 32)).astype(np.int32),
    }
    for name, lower in bounds.items():
        assert (lower <= want).all()
        pre = dev(lower)
        kv.probe_resume(slots, d_dig, d_off, pre, status=st)
        torch.cuda.synchronize()
        assert int(st.item()) == 0
        got = pre.cpu().numpy()
        assert (got == want).all(), f"{name}: {int((got != want).sum())} of {n_req} prefix lengths differ"


@pytest.mark.parametrize("n_req", [500, 5000, 40000], ids=["few", "mid", "many"])
@pytest.mark.parametrize("cap_log2,n_keys,clustered", [(12, 3686, 0), (12, 2400, 400), (5, 28, 0), (16, 49152, 0)],
                         ids=["load_0.9", "clustered_run", "window_is_table", "load_0.75"])
def test_probe_long_walks_match_oracle(kv, cap_log2, n_keys, clustered, n_req):
    """Every probe layout, where a warp's walks that go past their first two
    slots are finished together, on tables with long walks: load factor 0.9; `clustered` keys (and 32 absent ones) homed within
    16 slots, so that walks run for hundreds of slots (the longest run of
    filled slots is 809, under the 1024-slot window, so every insert fits);
    a 32-slot table whose window is the whole table.  Requests of 1-3 blocks
    drawn 80 % from the stored keys and 20 % from absent ones."""
    cap = 1 << cap_log2
    pool = keys_np(n_keys + n_keys // 2 + 64, 500 + cap_log2 + clustered)
    if clustered:
        idx = np.r_[0:clustered, n_keys:n_keys + 32]
        h = pool[idx, :8].copy().view(np.uint64)[:, 0]
        h = (h & ~np.uint64(cap - 1)) | (np.uint64(cap // 4) + (h & np.uint64(15)))
        pool[idx, :8] = h.reshape(-1, 1).view(np.uint8)
    present, absent = pool[:n_keys], pool[n_keys:]
    rng = np.random.default_rng(cap_log2 + clustered + n_req)
    nb = rng.integers(1, 4, n_req)
    off = np.concatenate([[0], np.cumsum(nb)]).astype(np.int64)
    n = int(off[-1])
    digests = np.where((rng.random(n) < 0.8)[:, None], present[rng.integers(0, n_keys, n)],
                       absent[rng.integers(0, len(absent), n)])
    if clustered:                                        # some requests walk the long run
        digests[off[1:100]] = absent[rng.integers(0, 32, 99)]
    slots = kv.new_table(cap)
    st = status_tensor()
    kv.insert(slots, dev(present), st)
    pre = kv.probe(slots, dev(digests), dev(off), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ks = oracle.KeySet(1)
    ks.insert(present)
    want = ks.prefix_blocks(digests, off)
    got = pre.cpu().numpy()
    assert (got == want).all(), f"{int((got != want).sum())} of {n_req} prefix lengths differ"
    assert 0 < (want == 0).sum() < n_req and (want == 3).any()


@pytest.mark.parametrize("n_req", [500, 5000, 40000], ids=["few", "mid", "many"])
def test_probe_bad_range_in_a_batch(kv, n_req):
    """A malformed range (its end before its start) in the middle of a batch
    is flagged and gets prefix 0; every other request, including the next one
    whose range now starts earlier, gets the oracle's prefix for its range."""
    rng = np.random.default_rng(n_req)
    pool = keys_np(2000, 41)
    nb = rng.integers(1, 12, n_req)
    off = np.concatenate([[0], np.cumsum(nb)]).astype(np.int64)
    digests = pool[rng.integers(0, len(pool), int(off[-1]))]
    member = rng.random(len(pool)) < 0.8
    k = n_req // 2
    off_bad = off.copy()
    off_bad[k + 1] = off[k] - 1                 # request k: -1 blocks; request k+1 starts one block early
    slots = kv.new_table(1 << 13)
    st = status_tensor()
    kv.insert(slots, dev(pool[member]), st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    pre = kv.probe(slots, dev(digests), dev(off_bad), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & kv.F_BADINDEX
    # the same requests laid out back to back for the oracle, the bad one empty
    ranges = [(int(off_bad[r]), max(0, int(off_bad[r + 1] - off_bad[r]))) for r in range(n_req)]
    ranges[k] = (0, 0)
    flat = np.concatenate([digests[b:b + n] for b, n in ranges])
    off2 = np.concatenate([[0], np.cumsum([n for _, n in ranges])]).astype(np.int64)
    ks = oracle.KeySet(1)
    ks.insert(pool[member])
    want = ks.prefix_blocks(flat, off2)
    assert (pre.cpu().numpy() == want).all()


@pytest.mark.parametrize("cap_log2", [6, 12, 16])
def test_insert_uncached_after_probe_matches_insert_all(kv, cap_log2):
    """Probe, then insert each request's suffix from its prefix length: the
    set and the count of new keys equal those of inserting every digest."""
    rng = np.random.default_rng(100 + cap_log2)
    pool = keys_np(min(1 << (cap_log2 - 1), 3000), cap_log2 + 200)
    nb = rng.integers(0, 40, 2000)
    nb[:4] = [0, 1, 39, 16]
    off = np.concatenate([[0], np.cumsum(nb)]).astype(np.int64)
    digests = pool[rng.integers(0, len(pool), int(off[-1]))]
    member = rng.random(len(pool)) < 0.5
    slots = kv.new_table(1 << cap_log2)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    kv.insert(slots, dev(pool[member]), st)
    d_dig, d_off = dev(digests), dev(off)
    pre = kv.probe(slots, d_dig, d_off, status=st)
    kv.insert_uncached(slots, d_dig, d_off, pre, st, n_new)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ks = oracle.KeySet(1)
    ks.insert(pool[member])
    assert (pre.cpu().numpy() == ks.prefix_blocks(digests, off)).all()
    n_ref, _ = ks.insert(digests)
    assert int(n_new.item()) == n_ref
    assert table_keys(slots) == {r.tobytes() for r in ks.contents()}


def test_insert_uncached_bad_offsets_flagged(kv):
    slots = kv.new_table(64)
    st = status_tensor()
    kv.insert_uncached(slots, dev(keys_np(4, 7)), dev(np.array([0, 4, 2], np.int64)),
                       dev(np.zeros(2, np.int32)), st)
    torch.cuda.synchronize()
    assert int(st.item()) & kv.F_BADINDEX


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("fill", [0.0, 0.5, 1.0])
@pytest.mark.parametrize("n_req", [180, 20000, 34000, 40960],
                         ids=["split_then_probe", "split_3_ctas_per_sm_then_probe", "chain_then_probe", "fused"])
def test_chain_hash_probe_matches_separate_calls(kv, mode, fill, n_req):
    """kvgov_chain_hash_probe writes the digests of kvgov_chain_hash and the
    prefix lengths of kvgov_probe, both equal to the oracle's, on each of its
    routes: the small-batch chain kernel then the probe kernel (up to 192
    requests per SM), the chain kernel then the probe kernel (up to two warps
    per SM sub-partition), and the chain kernel probing each digest as it
    computes it."""
    lengths = (RAGGED * 9 if n_req == 180 else
               list(np.random.default_rng(n_req + mode).integers(0, 260, n_req)))
    b = W.ragged(77, lengths)
    salts = oracle.derive_salts(b"fused", *W.principal_ids(8))
    ref = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    blk_ref = oracle.block_offsets(b.tok_off)
    rng = np.random.default_rng(int(fill * 10) + mode)
    member = rng.random(len(ref)) < fill
    member[blk_ref[5]:blk_ref[9]] = True          # some requests fully cached
    slots = kv.new_table(max(1 << 14, 1 << int(4 * member.sum()).bit_length()))
    st = status_tensor()
    if member.any():
        kv.insert(slots, dev(ref[member]), st)
    toks, tok_off = dev(b.tokens, np.int32), dev(b.tok_off, np.int64)
    blk = kv.block_offsets(tok_off, status=st)
    d, pre = kv.chain_hash_probe(mode, toks, tok_off, blk, slots, dev(b.principal, np.int32), dev(salts),
                                 dev(b.boundary_tok, np.int32), n_blocks=len(ref), status=st)
    pre_sep = kv.probe(slots, d, blk, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert (d.cpu().numpy() == ref).all()
    ks = oracle.KeySet(1)
    ks.insert(ref[member])
    pref = ks.prefix_blocks(ref, blk_ref)
    assert (pre.cpu().numpy() == pref).all() and (pre_sep.cpu().numpy() == pref).all()


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("n_req,prev_n", [(180, 150), (40960, 40960), (40960, 90000), (40960, 0), (0, 300)],
                         ids=["two_launches", "fused", "fused_more_prev", "no_prev", "empty_batch"])
def test_chain_hash_insert_prev_matches_separate_calls(kv, mode, n_req, prev_n):
    """kvgov_chain_hash_insert_prev writes kvgov_chain_hash's digests and
    leaves the table, key count and flags of kvgov_insert_uncached on the
    previous batch: on a batch small enough to take two launches, on fused
    batches (the previous one with more requests than the grid has threads,
    or none), and with an empty batch.  The previous batch holds the all-zero
    key, keys that live in the side store, a request whose prefix covers it
    whole, and out-of-range prefixes."""
    rng = np.random.default_rng(n_req + prev_n + mode)
    lengths = list(rng.integers(0, 200, n_req)) if n_req else []
    b = W.ragged(19 + mode, lengths) if n_req else None
    salts = oracle.derive_salts(b"prev", *W.principal_ids(8))
    # the previous batch: random keys, a third of them present already
    pnb = rng.integers(0, 12, prev_n)
    if prev_n:
        pnb[0] = max(int(pnb[0]), 1)
    poff = np.concatenate([[0], np.cumsum(pnb)]).astype(np.int64)
    pdig = keys_np(int(poff[-1]), 5 + mode) if prev_n else np.zeros((0, 32), np.uint8)
    ppre = rng.integers(-2, 14, prev_n).astype(np.int32)      # < 0 reads as 0, > n_b as n_b
    if prev_n:
        pdig[0] = 0                                           # the all-zero key, uncached
        ppre[0] = 0
        for i in range(1, min(len(pdig), 13), 4):             # keys that live in the side store
            pdig[i, (slice(0, 16), slice(16, 24), slice(24, 32))[(i // 4) % 3]] = 0
    present = pdig[rng.random(len(pdig)) < 0.3] if prev_n else pdig
    cap = 1 << 20
    def fresh_table():
        slots = kv.new_table(cap)
        st = status_tensor()
        if len(present):
            kv.insert(slots, dev(present[present.any(axis=1)]), st)
        return slots
    slots_a, slots_b = fresh_table(), fresh_table()
    st_a, st_b = status_tensor(), status_tensor()
    n_a = torch.zeros(1, dtype=torch.int64, device=DEV)
    n_b = torch.zeros(1, dtype=torch.int64, device=DEV)
    d_pdig, d_poff, d_ppre = dev(pdig), dev(poff), dev(ppre)
    if n_req:
        toks, tok_off = dev(b.tokens, np.int32), dev(b.tok_off, np.int64)
        pr, bt = dev(b.principal, np.int32), dev(b.boundary_tok, np.int32)
    else:
        toks, tok_off = torch.zeros(4, dtype=torch.int32, device=DEV), torch.zeros(1, dtype=torch.int64, device=DEV)
        # no requests; the salted modes still take non-NULL principal and boundary arrays
        pr, bt = torch.zeros(1, dtype=torch.int32, device=DEV), torch.zeros(1, dtype=torch.int32, device=DEV)
    blk = kv.block_offsets(tok_off, status=st_a)
    nbk = int(blk[-1].item())
    d_salts = dev(salts) if mode else None
    pr_, bt_ = (pr if mode else None), (bt if mode == 2 else None)
    d_a = kv.chain_hash_insert_prev(mode, toks, tok_off, blk, slots_a, d_pdig, d_poff, d_ppre, st_a,
                                    principal=pr_, salts=d_salts, boundary_tok=bt_, n_blocks=nbk, n_new=n_a)
    d_b = kv.chain_hash(mode, toks, tok_off, blk, pr_, d_salts, bt_, n_blocks=nbk, status=st_b)
    kv.insert_uncached(slots_b, d_pdig, d_poff, d_ppre, st_b, n_b)
    torch.cuda.synchronize()
    assert int(st_a.item()) == int(st_b.item())
    if prev_n:
        assert int(st_a.item()) & kv.F_SENTINEL
    assert (d_a.cpu().numpy() == d_b.cpu().numpy()).all()
    assert int(n_a.item()) == int(n_b.item())
    assert table_keys(slots_a) == table_keys(slots_b)
    if n_req:
        ref = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
        assert (d_a.cpu().numpy() == ref).all()
    # the oracle's set: the keys present before plus every uncached key of the previous batch
    ks = oracle.KeySet(1)
    ks.insert(present[present.any(axis=1)])
    before = ks.n
    rows = [np.arange(poff[r] + min(max(int(ppre[r]), 0), pnb[r]), poff[r + 1]) for r in range(prev_n)]
    rows = np.concatenate(rows + [np.zeros(0, np.int64)]).astype(np.int64)
    new_keys = pdig[rows]
    ks.insert(new_keys[new_keys.any(axis=1)])
    assert int(n_a.item()) == ks.n - before
    assert table_keys(slots_a) == {r.tobytes() for r in ks.contents()}


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("n_req,stride", [(180, 3), (40960, 3), (40960, 1)],
                         ids=["separate_launches", "fused", "fused_same_batch"])
def test_chain_hash_insert_prev_with_probe(kv, mode, n_req, stride):
    """With a prefix output, kvgov_chain_hash_insert_prev gives this batch's
    digests, the previous batch's insert, and this batch's prefix lengths
    against the table after that insert -- the results of kvgov_chain_hash,
    kvgov_insert_uncached and kvgov_probe in sequence.  The previous batch
    shares keys with this one (every third request's blocks, or every
    request's), so the probe must see the insert: in the fused launch the
    lookups of a block run while its own key is being inserted, and the
    resumed probe must make up what they missed."""
    rng = np.random.default_rng(7 * n_req + mode + stride)
    lengths = list(rng.integers(0, 300, n_req))
    b = W.ragged(23 + mode, lengths)
    salts = oracle.derive_salts(b"probe-after-insert", *W.principal_ids(8))
    ref = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
    blk_ref = oracle.block_offsets(b.tok_off)
    # the previous batch: this batch's digests of every stride-th request (so its insert makes them hit), plus
    # random keys; its prefix lengths cut some requests short
    prev_req = np.arange(0, n_req, stride)
    prev_rows = [ref[blk_ref[r]:blk_ref[r + 1]] for r in prev_req]
    pnb = np.array([len(x) for x in prev_rows], np.int64)
    poff = np.concatenate([[0], np.cumsum(pnb)]).astype(np.int64)
    pdig = np.concatenate(prev_rows + [np.zeros((0, 32), np.uint8)])
    ppre = np.where(rng.random(len(prev_req)) < 0.2, rng.integers(0, 5, len(prev_req)), 0).astype(np.int32)
    present = ref[rng.random(len(ref)) < 0.05]                 # a few keys cached before
    cap = 1 << 21
    slots_a, slots_b = kv.new_table(cap), kv.new_table(cap)
    st_a, st_b = status_tensor(), status_tensor()
    for sl in (slots_a, slots_b):
        kv.insert(sl, dev(present), st_b)
    n_a = torch.zeros(1, dtype=torch.int64, device=DEV)
    n_b = torch.zeros(1, dtype=torch.int64, device=DEV)
    toks, tok_off = dev(b.tokens, np.int32), dev(b.tok_off, np.int64)
    pr, bt = dev(b.principal, np.int32), dev(b.boundary_tok, np.int32)
    d_salts = dev(salts) if mode else None
    pr_, bt_ = (pr if mode else None), (bt if mode == 2 else None)
    blk = kv.block_offsets(tok_off, status=st_a)
    d_pdig, d_poff, d_ppre = dev(pdig), dev(poff), dev(ppre)
    pre_a = torch.full((n_req,), -5, dtype=torch.int32, device=DEV)
    d_a = kv.chain_hash_insert_prev(mode, toks, tok_off, blk, slots_a, d_pdig, d_poff, d_ppre, st_a,
                                    principal=pr_, salts=d_salts, boundary_tok=bt_, n_blocks=len(ref), n_new=n_a,
                                    prefix_blocks=pre_a)
    d_b = kv.chain_hash(mode, toks, tok_off, blk, pr_, d_salts, bt_, n_blocks=len(ref), status=st_b)
    kv.insert_uncached(slots_b, d_pdig, d_poff, d_ppre, st_b, n_b)
    pre_b = kv.probe(slots_b, d_b, blk, status=st_b)
    torch.cuda.synchronize()
    assert int(st_a.item()) == 0 and int(st_b.item()) == 0
    assert (d_a.cpu().numpy() == ref).all() and (d_b.cpu().numpy() == ref).all()
    assert int(n_a.item()) == int(n_b.item())
    assert table_keys(slots_a) == table_keys(slots_b)
    ks = oracle.KeySet(1)
    ks.insert(present)
    rows = np.concatenate([np.arange(poff[i] + ppre[i], poff[i + 1]) for i in range(len(prev_req))] +
                          [np.zeros(0, np.int64)]).astype(np.int64)
    ks.insert(pdig[rows])
    want = ks.prefix_blocks(ref, blk_ref)
    assert (pre_a.cpu().numpy() == want).all() and (pre_b.cpu().numpy() == want).all()
    assert (want[prev_req][ppre == 0] == (np.diff(blk_ref)[prev_req][ppre == 0])).all()   # inserted: all hit


def _repeat_requests(b: W.Batch, idx) -> W.Batch:
    """The batch of b's requests idx (repeats allowed), in that order."""
    parts = [b.tokens[b.tok_off[r]:b.tok_off[r + 1]] for r in idx]
    tok_off = np.concatenate([[0], np.cumsum([len(x) for x in parts])]).astype(np.int64)
    tokens = np.concatenate(parts + [np.zeros(4, np.int32)]).astype(np.int32)
    return W.Batch(tokens, tok_off, b.principal[idx].copy(), b.boundary_tok[idx].copy())


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("n_req", [180, 40960], ids=["separate_launches", "fused"])
def test_chain_hash_serve_matches_probe_then_insert(kv, mode, n_req):
    """kvgov_chain_hash_serve over a sequence of batches -- a fresh one, the
    same one again (every block now cached), a new batch whose requests come
    in pairs (a key the batch itself adds never counts as cached for it,
    whichever copy gets there first), then a flush with the floor raised and
    the first batch twice more -- gives, batch by batch, the digests of
    kvgov_chain_hash, the prefix lengths of the oracle's set before the
    batch's insert, and after it the set and key count of inserting every
    block past the prefix (paper section 2.1).  Keys in the table before the
    first batch are stamped with generation 1."""
    rng = np.random.default_rng(11 * n_req + mode)
    b0 = W.ragged(41 + mode, list(rng.integers(0, 300, n_req)))
    fresh = W.ragged(43 + mode, list(rng.integers(0, 300, n_req)))
    pairs = _repeat_requests(fresh, np.repeat(np.arange(n_req // 2), 2))
    salts = oracle.derive_salts(b"serve", *W.principal_ids(8))
    d_salts = dev(salts) if mode else None
    cap = 1 << 22
    slots = kv.new_table(cap)
    gen = kv.new_gen(slots)
    st, n_new = status_tensor(), torch.zeros(1, dtype=torch.int64, device=DEV)
    ref0 = oracle.chain_hash(mode, b0.tokens, b0.tok_off, b0.principal, salts, b0.boundary_tok)
    present = ref0[rng.random(len(ref0)) < 0.05]               # a few of the first batch's blocks, cached before
    kv.insert(slots, dev(present), st)
    kv.table_gen_stamp(slots, gen, 1)
    ks = oracle.KeySet(1)
    ks.insert(present)
    start_n = ks.n
    g, floor = 1, 1
    for step, (b, flush) in enumerate([(b0, False), (b0, False), (pairs, False), (b0, True), (b0, False)]):
        if flush:                                               # the table emptied; every generation so far below
            kv.table_init(slots)
            floor = g + 1
            ks, start_n = oracle.KeySet(1), 0
            n_new.zero_()
        g += 1
        toks, tok_off = dev(b.tokens, np.int32), dev(b.tok_off, np.int64)
        blk = kv.block_offsets(tok_off, status=st)
        pr = dev(b.principal, np.int32) if mode else None
        bt = dev(b.boundary_tok, np.int32) if mode == 2 else None
        blk_ref = oracle.block_offsets(b.tok_off)
        dig, pre = kv.chain_hash_serve(mode, toks, tok_off, blk, slots, gen, g, floor, st, principal=pr,
                                       salts=d_salts, boundary_tok=bt, n_blocks=int(blk_ref[-1]), n_new=n_new)
        torch.cuda.synchronize()
        assert int(st.item()) == 0
        ref = oracle.chain_hash(mode, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
        assert (dig.cpu().numpy() == ref).all(), f"step {step}: digests differ"
        want = ks.prefix_blocks(ref, blk_ref)
        got = pre.cpu().numpy()
        assert (got == want).all(), f"step {step}: {int((got != want).sum())} of {b.n} prefix lengths differ"
        rows = np.concatenate([np.arange(blk_ref[r] + want[r], blk_ref[r + 1]) for r in range(b.n)] +
                              [np.zeros(0, np.int64)]).astype(np.int64)
        ks.insert(ref[rows])
        assert int(n_new.item()) == ks.n - start_n, f"step {step}: key count"
        if step == 1 or step == 4:                              # the same batch again: every block cached
            assert (want == np.diff(blk_ref)).all()
        if step == 2:                                           # a new batch in pairs: nothing cached for it
            assert (want == 0).all() and len(rows) > 0
    assert table_keys(slots) == {r.tobytes() for r in ks.contents()}


def test_probe_empty_and_bad_offsets(kv):
    slots = kv.new_table(64)
    st = status_tensor()
    pre = kv.probe(slots, dev(keys_np(4, 7)), dev(np.array([0, 4, 2], np.int64)), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & kv.F_BADINDEX
    empty = kv.probe(slots, dev(keys_np(1, 7)), dev(np.array([0], np.int64)))
    assert empty.numel() == 0


def test_probe_resume_empty_and_bad_offsets(kv):
    """kvgov_probe_resume, as include/kvgov.h states it: a request whose
    block range is malformed is flagged and gets 0 whatever its entry; a
    negative entry reads as the lower bound 0; an entry past the request's
    blocks is clamped to them (and, being the caller's claim, not checked);
    an empty batch is a no-op."""
    keys = keys_np(6, 9)
    slots = kv.new_table(64)
    st = status_tensor()
    kv.insert(slots, dev(keys[:4]), st)
    off = np.array([0, 4, 2, 6], np.int64)                 # request 1 runs backwards; request 2: rows 2-5
    pre = dev(np.array([-5, 1, 8], np.int32))
    kv.probe_resume(slots, dev(keys), dev(off), pre, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & kv.F_BADINDEX
    assert pre.cpu().numpy().tolist() == [4, 0, 4]
    empty = torch.zeros(0, dtype=torch.int32, device=DEV)
    kv.probe_resume(slots, dev(keys[:1]), dev(np.array([0], np.int64)), empty)
    torch.cuda.synchronize()
