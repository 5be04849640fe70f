"""kvgov_serve_arrival_static (slot handles in the library's static device
array) against kvgov_insert_arrival + kvgov_probe_arrival (caller scratch):
the same prefix lengths, key counts and table contents on two consecutive
calls on one table; oversized batches are refused, and a batch whose offsets
run past the block count it is given is flagged without a read past that
count.  Marked gpu."""
import numpy as np
import pytest
import torch

from paper_2608_09225_gb300 import workloads as W
from paper_2608_09225_gb300.pipeline import DeviceBatch, PrefixCache, next_pow2
from tests.table_layout import table_keys

pytestmark = pytest.mark.gpu




def test_static_scratch_matches_caller_scratch(kv):
    ws = [W.make("wide", seed=90 + i, n_req=20000) for i in range(2)]
    ws[1].batch.tokens.reshape(-1, 128)[:, :64] = ws[0].batch.tokens[:64]
    w0 = ws[0]
    dbs = [DeviceBatch.from_host(w.batch.tokens, w.batch.tok_off, w.batch.principal, w.batch.boundary_tok)
           for w in ws]
    hasher = PrefixCache(1 << 10, w0.secret, w0.ids, w0.id_off)
    batches = [hasher.hash(W.BOUNDARY, db) for db in dbs]            # (blk_off, digests)
    cap = next_pow2(8 * dbs[0].n_blocks)
    ref_slots, ref_owner = kv.new_table(cap), kv.new_owner(cap)
    st_slots, st_owner = kv.new_table(cap), kv.new_owner(cap)
    ref_st, st_st = (torch.zeros(1, dtype=torch.int32, device="cuda") for _ in range(2))
    ref_new, st_new = (torch.zeros(1, dtype=torch.int64, device="cuda") for _ in range(2))
    seq = 1
    for blk, d in batches:                                           # two consecutive calls
        slot_of = kv.insert_arrival(ref_slots, ref_owner, d, blk, seq, ref_st, n_new=ref_new)
        want = kv.probe_arrival(ref_owner, slot_of, blk, seq, status=ref_st)
        got = kv.serve_arrival_static(st_slots, st_owner, d, blk, seq, st_st, n_new=st_new)
        torch.cuda.synchronize()
        assert int(ref_st.item()) == 0 and int(st_st.item()) == 0
        assert (got.cpu().numpy() == want.cpu().numpy()).all()
        assert int(st_new.item()) == int(ref_new.item())
        seq += d.shape[0]
    assert table_keys(st_slots) == table_keys(ref_slots)
    assert (st_owner.cpu().numpy()[st_slots.cpu().numpy()[:, :16].any(axis=1)] > 0).all()
    last = got.cpu().numpy()
    assert last[0] >= 4 and (last >= 4).all()                        # batch 2 reuses batch 1's shared prefix


def test_static_scratch_refuses_oversized_batches(kv):
    slots, owner = kv.new_table(64), kv.new_owner(64)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = torch.zeros(((1 << 21) + 1, 32), dtype=torch.uint8, device="cuda")
    blk = torch.tensor([0, (1 << 21) + 1], dtype=torch.int64, device="cuda")
    with pytest.raises(kv.KVGovError):
        kv.serve_arrival_static(slots, owner, d, blk, 1, st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0


@pytest.mark.parametrize("total", [96, (1 << 21) + 1])
def test_static_scratch_bounds_rows_by_n_blocks(kv, total):
    """d_blk_off[n_req] above the n_blocks argument (the digest buffer still
    holds d_blk_off[n_req] rows, so every read stays inside it either way):
    nothing is inserted, every request is flagged KVGOV_F_BADINDEX with
    prefix 0, and the table and owners are unchanged."""
    digests = torch.full((total, 32), 7, dtype=torch.uint8, device="cuda")
    digests[:, 0] = torch.arange(total, device="cuda").to(torch.uint8) | 1
    blk = torch.tensor([0, 40, total], dtype=torch.int64, device="cuda")
    slots, owner = kv.new_table(256), kv.new_owner(256)
    slots_before, owner_before = slots.clone(), owner.clone()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    n_new = torch.zeros(1, dtype=torch.int64, device="cuda")
    pre = kv.serve_arrival_static(slots, owner, digests[:64], blk, 1, st, n_new=n_new)
    torch.cuda.synchronize()
    assert int(st.item()) == kv.F_BADINDEX
    assert (pre.cpu().numpy() == 0).all()
    assert int(n_new.item()) == 0
    assert torch.equal(slots, slots_before) and torch.equal(owner, owner_before)


def test_static_scratch_with_side_store_keys(kv):
    """Keys that live in the table's side store (zero first half, zero third
    or fourth 8-byte word), shared across requests, and one all-zero key:
    the same prefix lengths, key count, flags and table as the caller-scratch
    calls, on two consecutive calls."""
    rng = np.random.default_rng(77)
    pool = rng.integers(1, 256, (24, 32), dtype=np.uint8)
    for i in range(6):
        pool[i, (slice(0, 16), slice(16, 24), slice(24, 32))[i % 3]] = 0
    pool[23] = 0
    cap = 1 << 10
    ref_slots, ref_owner = kv.new_table(cap), kv.new_owner(cap)
    st_slots, st_owner = kv.new_table(cap), kv.new_owner(cap)
    ref_st, st_st = (torch.zeros(1, dtype=torch.int32, device="cuda") for _ in range(2))
    ref_new, st_new = (torch.zeros(1, dtype=torch.int64, device="cuda") for _ in range(2))
    seq = 1
    for call in range(2):
        lens = rng.integers(0, 9, 400)
        off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
        d = torch.from_numpy(pool[rng.integers(0, 24, int(off[-1]))]).cuda()
        blk = torch.from_numpy(off).cuda()
        slot_of = kv.insert_arrival(ref_slots, ref_owner, d, blk, seq, ref_st, n_new=ref_new)
        want = kv.probe_arrival(ref_owner, slot_of, blk, seq, status=ref_st)
        got = kv.serve_arrival_static(st_slots, st_owner, d, blk, seq, st_st, n_new=st_new)
        torch.cuda.synchronize()
        assert int(ref_st.item()) == int(st_st.item()) == kv.F_SENTINEL
        assert (got.cpu().numpy() == want.cpu().numpy()).all()
        assert int(st_new.item()) == int(ref_new.item()) == 23
        seq += int(off[-1])
    assert table_keys(st_slots) == table_keys(ref_slots) == {r.tobytes() for r in pool[:23]}
