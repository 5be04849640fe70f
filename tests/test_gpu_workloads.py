"""The five workloads through the CUDA path, bit-exact against the oracle:
reduced sizes, then the full sizes in the launch configuration bench.py
times (PrefixCache.serve: salts, blocking, chain, probe, insert).  Marked gpu."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_09225_gb300 import workloads as W
from paper_2608_09225_gb300 import kvgov as K
from paper_2608_09225_gb300.pipeline import (DeviceBatch, DevicePipeline, HostPipeline, PrefixCache,
                                              next_pow2)
from tests.pins import run_workload_oracle

pytestmark = pytest.mark.gpu

# the serving engine's schedules: the insert in the next batch's chain launch, the insert after the
# chain hash and the probe, and the lookups and insert in the batch's own chain launch
SCHEDULES = ["insert_in_chain", "inline", "one_launch"]


def sched(schedule):
    return {"insert_in_chain": schedule == "insert_in_chain", "one_launch": schedule == "one_launch"}


def run_gpu(kv, w: W.Workload, mode: int):
    """Salts, chains, table fill (same content as the oracle's) and probe."""
    cap = w.capacity or 1024
    cache = PrefixCache(cap, w.secret, w.ids, w.id_off)
    b = w.batch
    db = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
    blk, d = cache.hash(mode, db)
    blk_np = blk.cpu().numpy()
    if w.fill_from == "prior":
        p = w.prior
        dp = DeviceBatch.from_host(p.tokens, p.tok_off, p.principal, p.boundary_tok)
        _, dpd = cache.hash(mode, dp)
        cache.insert(dpd)
    else:
        f0, f1 = w.fill
        if f1 > f0:
            cache.insert(d[blk_np[f0]:blk_np[f1]])
    if w.random_keys is not None:
        cache.insert(torch.from_numpy(w.random_keys).cuda())
    p0, p1 = w.probe
    pre = cache.probe(d, blk[p0:p1 + 1])
    torch.cuda.synchronize()
    cache.check_status()
    return cache, blk_np, d.cpu().numpy(), pre.cpu().numpy()


def check(kv, w, mode):
    cache, blk, d, pre = run_gpu(kv, w, mode)
    salts, dref, bref, ks, pref = run_workload_oracle(w, mode)
    assert (cache.salts.cpu().numpy() == salts).all()
    assert (blk == bref).all()
    bad = np.nonzero((d != dref).any(axis=1))[0]
    assert len(bad) == 0, f"{len(bad)} of {len(d)} digests differ"
    assert (pre == pref).all(), f"{int((pre != pref).sum())} prefix lengths differ"
    assert int(cache.n_new.item()) == ks.n
    return pre


def test_tiny_full(kv):
    pre = check(kv, W.make("tiny"), W.ROOT)
    assert list(pre) == [16] * 16 + [8] * 16 + [0] * 32


def test_sysprompt_reduced(kv):
    check(kv, W.sysprompt(n_req=128, fill_n=32), W.ROOT)


@pytest.mark.parametrize("mode", [W.UNSALTED, W.ROOT, W.BOUNDARY])
def test_template_reduced(kv, mode):
    check(kv, W.template(n_req=1024), mode)


def test_probe_reduced(kv):
    w = W.probe(n_req=2048, n_prior=256, capacity=1 << 16)
    pre = check(kv, w, W.ROOT)
    assert (pre == w.info["cut"]).all()


def test_long_reduced(kv):
    w = W.long(seed=11, n_req=8)
    w.capacity, w.fill, w.probe = 1 << 16, (0, 4), (0, 8)
    check(kv, w, W.BOUNDARY)


def test_wide_reduced(kv):
    w = W.wide(seed=12, n_req=4096)
    w.capacity, w.fill, w.probe = 1 << 16, (0, 2048), (0, 4096)
    pre = check(kv, w, W.BOUNDARY)
    assert (pre[:2048] == 8).all() and (pre[2048:] == 4).all()


# ------------------------------------------------------------- full sizes
def test_full_sysprompt(kv):
    w = W.make("sysprompt")
    pre = check(kv, w, W.ROOT)
    filled = set(w.batch.principal[:256].tolist())
    assert list(pre) == [132] * 256 + [64 if int(p) in filled else 0 for p in w.batch.principal[256:]]


@pytest.mark.parametrize("mode", [W.UNSALTED, W.ROOT, W.BOUNDARY])
def test_full_template(kv, mode):
    check(kv, W.make("template"), mode)


def test_full_probe(kv):
    w = W.make("probe")
    pre = check(kv, w, W.ROOT)
    assert (pre == w.info["cut"]).all()


def test_full_long(kv):
    w = W.make("long", seed=77)
    w.capacity, w.fill, w.probe = 1 << 20, (0, 128), (0, 256)
    pre = check(kv, w, W.BOUNDARY)
    assert (pre[:128] == 2048).all() and (pre[128:] == 4).all()


def test_full_wide_serving_steps(kv):
    """The bench's step (PrefixCache.serve) on the full 131,072 x 128 batch,
    three times: batch A into an empty cache, a fresh batch B with the same
    shared prefix (its 4 unsalted blocks hit), then A again (all 8 hit).
    Every salt, digest and prefix length is compared with the oracle."""
    wa, wb = W.make("wide", seed=101), W.make("wide", seed=102)
    wb.secret, wb.ids, wb.id_off = wa.secret, wa.ids, wa.id_off
    # B shares A's 64-token prefix (the prefix every request of the service starts with)
    wb.batch.tokens.reshape(-1, 128)[:, :64] = wa.batch.tokens[:64]
    n_blocks = wa.batch.n * 8
    cache = PrefixCache(next_pow2(4 * 3 * n_blocks), wa.secret, wa.ids, wa.id_off)
    salts = oracle.derive_salts(wa.secret, wa.ids, wa.id_off)
    ks = oracle.KeySet(1)
    seen = []
    for w in (wa, wb, wa):
        b = w.batch
        db = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
        pre, d, blk = cache.serve(W.BOUNDARY, db)
        torch.cuda.synchronize()
        cache.check_status()
        dref = oracle.chain_hash(W.BOUNDARY, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
        bref = oracle.block_offsets(b.tok_off)
        assert (cache.salts.cpu().numpy() == salts).all()
        assert (blk.cpu().numpy() == bref).all()
        assert (d.cpu().numpy() == dref).all()
        pref = ks.prefix_blocks(dref, bref)
        assert (pre.cpu().numpy() == pref).all()
        ks.insert(dref)
        assert int(cache.n_new.item()) == ks.n
        seen.append(int(pref.min()))
    assert seen == [0, 4, 8]


def test_full_wide_device_pipeline_matches_oracle(kv):
    """The bench's timed path at full size: DevicePipeline in its default
    schedule (each batch's insert inside the next batch's chain launch,
    chain_prev_kernel at 131,072 requests) over batches A, B, A, B under one
    secret, then A under a new secret epoch.  Every batch's prefix lengths,
    copied on the compute stream right after its submit, and the final key
    count equal the oracle's replay."""
    wa, wb = W.make("wide", seed=111), W.make("wide", seed=112)
    wb.secret, wb.ids, wb.id_off = wa.secret, wa.ids, wa.id_off
    wb.batch.tokens.reshape(-1, 128)[:, :64] = wa.batch.tokens[:64]
    n_blocks = wa.batch.n * 8
    cache = PrefixCache(next_pow2(4 * 5 * n_blocks), wa.secret, wa.ids, wa.id_off)
    pipe = DevicePipeline(cache, W.BOUNDARY, wa.batch.n, n_blocks)
    dbs = [DeviceBatch.from_host(w.batch.tokens, w.batch.tok_off, w.batch.principal, w.batch.boundary_tok)
           for w in (wa, wb)]
    plan = [(0, 0), (1, 0), (0, 0), (1, 0), (0, 1)]            # (batch, secret epoch)
    copies = []
    for k, e in plan:
        cache.set_secret(wa.secret[:24] + e.to_bytes(8, "little"))
        pre, _ = pipe.submit(dbs[k])
        with torch.cuda.stream(pipe.compute_stream):
            copies.append(pre.clone())
    pipe.drain()
    torch.cuda.synchronize()
    cache.check_status()
    ks = oracle.KeySet(1)
    mins = []
    for i, (k, e) in enumerate(plan):
        b = (wa, wb)[k].batch
        salts = oracle.derive_salts(wa.secret[:24] + e.to_bytes(8, "little"), wa.ids, wa.id_off)
        dref = oracle.chain_hash(W.BOUNDARY, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
        bref = oracle.block_offsets(b.tok_off)
        pref = ks.prefix_blocks(dref, bref)
        assert (copies[i].cpu().numpy() == pref).all(), f"batch {i}"
        ks.insert(dref)
        mins.append(int(pref.min()))
    assert int(cache.n_new.item()) == ks.n
    assert mins == [0, 4, 8, 8, 4]


@pytest.mark.parametrize("schedule", SCHEDULES)
def test_device_pipeline_empty_and_tiny_batches(kv, schedule):
    """Batches of no requests, of one request shorter than a block, and
    ordinary batches, mixed in one stream through the serving engine: the
    empty ones give empty results and leave the cache alone, the others match
    the oracle's replay."""
    w = W.make("tiny")
    b = w.batch
    full = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
    empty = DeviceBatch.from_host(np.zeros(4, np.int32), np.zeros(1, np.int64), np.zeros(0, np.int32),
                                  np.zeros(0, np.int32))
    short_toks = b.tokens[:7].copy()
    short = DeviceBatch.from_host(short_toks, np.array([0, 7], np.int64), b.principal[:1], b.boundary_tok[:1])
    cache = PrefixCache(1 << 12, w.secret, w.ids, w.id_off)
    pipe = DevicePipeline(cache, W.ROOT, b.n, full.n_blocks, **sched(schedule))
    order = [empty, full, empty, short, full, empty]
    copies = []
    for db in order:
        pre, _ = pipe.submit(db)
        with torch.cuda.stream(pipe.compute_stream):
            copies.append(pre.clone())
    pipe.drain()
    torch.cuda.synchronize()
    cache.check_status()
    salts = oracle.derive_salts(w.secret, w.ids, w.id_off)
    ks = oracle.KeySet(1)
    for db, got in zip(order, copies):
        got = got.cpu().numpy()
        if db is empty:
            assert got.shape == (0,)
            continue
        if db is short:
            assert list(got) == [0]
            continue
        d = oracle.chain_hash(W.ROOT, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
        blk = oracle.block_offsets(b.tok_off)
        assert (got == ks.prefix_blocks(d, blk)).all()
        ks.insert(d)
    assert int(cache.n_new.item()) == ks.n


@pytest.mark.parametrize("schedule", SCHEDULES)
def test_host_pipeline_matches_device_serving(kv, schedule):
    """Batches served from pinned host memory through HostPipeline (copies
    overlapping the previous batch's serving; each batch's result read only
    after the next batch is queued) give the prefix lengths of the same
    batches served from device memory, and the same cache contents."""
    ws = [W.make("wide", seed=200 + i, n_req=8192) for i in range(4)]
    for w in ws[1:]:
        w.batch.tokens.reshape(-1, 128)[:, :64] = ws[0].batch.tokens[:64]
    w0 = ws[0]
    dev_cache = PrefixCache(1 << 18, w0.secret, w0.ids, w0.id_off)
    host_cache = PrefixCache(1 << 18, w0.secret, w0.ids, w0.id_off)
    n_tok = int(w0.batch.tok_off[-1])
    pipe = HostPipeline(host_cache, W.BOUNDARY, w0.batch.n, n_tok, **sched(schedule))
    order = [0, 1, 2, 0, 3, 1]
    got, want, pending = [], [], None
    for i, k in enumerate(order):
        b = ws[k].batch
        secret = w0.secret[:24] + (0 if i < 4 else 1).to_bytes(8, "little")   # a new epoch from batch 4 on
        dev_cache.set_secret(secret)
        host_cache.set_secret(secret)
        pre, _, _ = dev_cache.serve(W.BOUNDARY, DeviceBatch.from_host(b.tokens, b.tok_off, b.principal,
                                                                       b.boundary_tok))
        want.append(pre.cpu().numpy())
        host = [torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
                for a in (b.tokens, b.tok_off, b.principal, b.boundary_tok)]
        out, ev = pipe.submit(*host, b.n * 8)
        if pending is not None:                  # the previous batch's result, read while this one runs
            pending[1].synchronize()
            got.append(pending[0].numpy().copy())
        pending = (out, ev)
    pending[1].synchronize()
    got.append(pending[0].numpy().copy())
    pipe.drain()
    torch.cuda.synchronize()
    dev_cache.check_status()
    host_cache.check_status()
    for g, w in zip(got, want):
        assert (g == w).all()
    assert int(dev_cache.n_new.item()) == int(host_cache.n_new.item())
    assert [int(x.min()) for x in want] == [0, 4, 4, 8, 4, 4]


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("mode", [W.UNSALTED, W.ROOT, W.BOUNDARY])
def test_device_pipeline_matches_sequential_serving(kv, mode, schedule):
    """DevicePipeline (salts and block offsets of batch i+1 on a prep stream
    beside batch i's chain hash; batch i's insert inside batch i+1's chain
    launch, or inline) gives the prefix lengths and the key count of serving
    the same batches one by one, across secret changes and a flush of the
    cache between batches."""
    ws = [W.make("wide", seed=300 + i, n_req=40960) for i in range(3)]   # the fused launches
    for w in ws[1:]:
        w.batch.tokens.reshape(-1, 128)[:, :64] = ws[0].batch.tokens[:64]
    w0 = ws[0]
    dbs = [DeviceBatch.from_host(w.batch.tokens, w.batch.tok_off, w.batch.principal, w.batch.boundary_tok)
           for w in ws]
    seq = PrefixCache(1 << 21, w0.secret, w0.ids, w0.id_off)
    pip = PrefixCache(1 << 21, w0.secret, w0.ids, w0.id_off)
    pipe = DevicePipeline(pip, mode, w0.batch.n, dbs[0].n_blocks, **sched(schedule))
    order = [0, 1, 2, 0, 1, 2, 0]
    got, want = [], []
    for i, k in enumerate(order):
        secret = w0.secret[:24] + (i // 3).to_bytes(8, "little")     # a new epoch every third batch
        flush = i == 5
        seq.set_secret(secret)
        if flush:
            K.table_init(seq.slots)
        pre, _, _ = seq.serve(mode, dbs[k])
        want.append(pre.cpu().numpy())
        pip.set_secret(secret)
        out, ev = pipe.submit(dbs[k], flush)
        ev.synchronize()
        got.append(out.cpu().numpy())
    pipe.drain()
    torch.cuda.synchronize()
    seq.check_status()
    pip.check_status()
    for g, w in zip(got, want):
        assert (g == w).all()
    assert int(seq.n_new.item()) == int(pip.n_new.item())
    assert int(want[0].min()) == 0
    if mode != W.ROOT:                 # the shared 64-token prefix is unsalted
        assert int(want[1].min()) == 4


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("flush_at", [None, 5])
def test_device_pipeline_back_to_back_matches_oracle(kv, flush_at, schedule):
    """Many batches queued without waiting in between (and a cache flush
    queued in the middle): every batch's prefix lengths, copied out on the
    compute stream right after its submit, match the oracle's replay of the
    same batches in order."""
    ws = [W.make("wide", seed=400 + i, n_req=4096) for i in range(4)]
    for w in ws[1:]:
        w.batch.tokens.reshape(-1, 128)[:, :64] = ws[0].batch.tokens[:64]
    w0 = ws[0]
    dbs = [DeviceBatch.from_host(w.batch.tokens, w.batch.tok_off, w.batch.principal, w.batch.boundary_tok)
           for w in ws]
    cache = PrefixCache(1 << 17, w0.secret, w0.ids, w0.id_off)
    pipe = DevicePipeline(cache, W.BOUNDARY, w0.batch.n, dbs[0].n_blocks, **sched(schedule))
    order = [0, 1, 2, 3, 2, 0, 1, 3]
    copies = []
    for i, k in enumerate(order):
        cache.set_secret(w0.secret[:24] + (i % 2).to_bytes(8, "little"))
        pre, _ = pipe.submit(dbs[k], i == flush_at)
        with torch.cuda.stream(pipe.compute_stream):
            copies.append(pre.clone())
    pipe.drain()
    torch.cuda.synchronize()
    cache.check_status()
    ks, before_flush = oracle.KeySet(1), 0
    for i, k in enumerate(order):
        if i == flush_at:
            ks, before_flush = oracle.KeySet(1), ks.n
        b = ws[k].batch
        salts = oracle.derive_salts(w0.secret[:24] + (i % 2).to_bytes(8, "little"), w0.ids, w0.id_off)
        d = oracle.chain_hash(W.BOUNDARY, b.tokens, b.tok_off, b.principal, salts, b.boundary_tok)
        blk = oracle.block_offsets(b.tok_off)
        assert (copies[i].cpu().numpy() == ks.prefix_blocks(d, blk)).all(), f"batch {i}"
        ks.insert(d)
    assert int(cache.n_new.item()) == before_flush + ks.n
