"""Divergence-boundary detection on the GPU (kvgov_divergence_boundary)
against the oracle, bit-exact, and fed into BOUNDARY salting.  Marked gpu."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_09225_gb300 import workloads as W
from paper_2608_09225_gb300.pipeline import DeviceBatch, PrefixCache, next_pow2

pytestmark = pytest.mark.gpu
DEV = "cuda"


def dev(a, dtype=None):
    return torch.from_numpy(np.ascontiguousarray(a if dtype is None else np.asarray(a, dtype=dtype))).to(DEV)


def gpu_boundary(kv, tokens, tok_off, ids, tpl_tokens, tpl_off):
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    tt = dev(tpl_tokens, np.int32) if tpl_off is not None and len(tpl_off) > 1 else None
    to = dev(tpl_off, np.int64) if tt is not None else None
    b = kv.divergence_boundary(dev(tokens, np.int32), dev(tok_off, np.int64), dev(ids, np.int32), tt, to, status=st)
    torch.cuda.synchronize()
    return b.cpu().numpy(), int(st.item())


def random_case(seed, n_req, n_tpl, max_tpl=3000, max_tail=2000):
    rng = np.random.default_rng(seed)
    tpls = [rng.integers(0, W.VOCAB, int(rng.integers(0, max_tpl)), dtype=np.int32) for _ in range(n_tpl)]
    reqs, ids = [], []
    for _ in range(n_req):
        base = tpls[int(rng.integers(0, n_tpl))] if n_tpl and rng.random() < 0.9 else np.zeros(0, np.int32)
        cut = int(rng.integers(0, len(base) + 1))
        if rng.random() < 0.3:
            cut = len(base)                       # the whole preamble, then private tokens
        tail = rng.integers(0, W.VOCAB, int(rng.integers(0, max_tail)), dtype=np.int32)
        reqs.append(np.concatenate([base[:cut], tail]).astype(np.int32))
        ids.append(int(rng.integers(-2, n_tpl)) if n_tpl else int(rng.integers(-2, 0)))
    tok_off = np.concatenate([[0], np.cumsum([len(x) for x in reqs])]).astype(np.int64)
    tpl_off = np.concatenate([[0], np.cumsum([len(x) for x in tpls])]).astype(np.int64)
    toks = np.concatenate(reqs + [np.zeros(0, np.int32)]).astype(np.int32)
    tt = np.concatenate(tpls + [np.zeros(0, np.int32)]).astype(np.int32)
    return toks, tok_off, np.array(ids, np.int32), tt, tpl_off


@pytest.mark.parametrize("n_req,n_tpl", [(1, 1), (50, 0), (700, 3), (5000, 8), (40000, 4)])
def test_boundary_matches_oracle(kv, n_req, n_tpl):
    """Random batches with every id kind; 40,000 requests take the
    four-requests-per-warp layout."""
    big = n_req >= 32 * 1024
    toks, tok_off, ids, tt, tpl_off = random_case(n_req * 7 + n_tpl, n_req, n_tpl, max_tpl=300 if big else 3000,
                                                  max_tail=100 if big else 2000)
    got, st = gpu_boundary(kv, toks, tok_off, ids, tt, tpl_off)
    want, flag = oracle.divergence_boundary(toks, tok_off, ids, tt, tpl_off)
    assert st == 0 and not flag
    assert (got == want).all()


def test_boundary_bad_ids_flagged(kv):
    toks, tok_off, ids, tt, tpl_off = random_case(9, 64, 2)
    ids[[3, 10]] = [2, -3]                     # one past the last preamble, below TEMPLATE_ANY
    got, st = gpu_boundary(kv, toks, tok_off, ids, tt, tpl_off)
    want, flag = oracle.divergence_boundary(toks, tok_off, ids, tt, tpl_off)
    assert flag and st == kv.F_BADINDEX
    assert (got == want).all() and got[3] == 0 and got[10] == 0


def test_boundary_edge_cases(kv):
    """Empty requests, a preamble longer than its request (the whole request
    matches), a mismatch at token 0, and a batch of no requests."""
    tpl = np.arange(1, 301, dtype=np.int32)
    reqs = [np.zeros(0, np.int32), tpl[:17], tpl[:300], np.concatenate([tpl, [5, 6]]), np.array([9], np.int32),
            np.concatenate([tpl[:127], [0], tpl[128:]])]
    tok_off = np.concatenate([[0], np.cumsum([len(x) for x in reqs])]).astype(np.int64)
    toks = np.concatenate(reqs).astype(np.int32)
    ids = np.zeros(len(reqs), np.int32)
    got, st = gpu_boundary(kv, toks, tok_off, ids, tpl, np.array([0, 300], np.int64))
    assert st == 0 and list(got) == [0, 17, 300, 300, 0, 127]
    got, st = gpu_boundary(kv, np.zeros(0, np.int32), np.zeros(1, np.int64), np.zeros(0, np.int32), tpl,
                           np.array([0, 300], np.int64))
    assert got.shape == (0,) and st == 0


@pytest.mark.parametrize("name", ["sysprompt", "template", "wide", "long"])
def test_boundary_workloads(kv, name):
    """The workloads' shared preambles registered: the system prompt's 1024
    tokens, the template up to its first field (96), the 64-token prefix of
    the sweep batches."""
    w = W.make(name, seed=61) if name in ("wide", "long") else W.make(name)
    b = w.batch
    n_pre = {"sysprompt": 1024, "template": 96, "wide": 64, "long": 64}[name]
    pre = b.tokens[int(b.tok_off[0]):int(b.tok_off[0]) + n_pre]
    tpl_off = np.array([0, n_pre], np.int64)
    ids = np.zeros(b.n, np.int32)
    got, st = gpu_boundary(kv, b.tokens, b.tok_off, ids, pre, tpl_off)
    want, _ = oracle.divergence_boundary(b.tokens, b.tok_off, ids, pre, tpl_off)
    assert st == 0 and (got == want).all() and (got == n_pre).all()


def test_detected_boundaries_share_the_preamble_across_principals(kv):
    """System-prompt batch: boundaries detected against the registered system
    prompt, then BOUNDARY salting and arrival-order serving.  Every request
    after the first hits the 64 system-prompt blocks whatever its principal,
    and no block past them is shared across principals; the oracle agrees on
    every digest and prefix length."""
    w = W.make("sysprompt")
    b = w.batch
    pre = b.tokens[:1024]
    tpl_off = np.array([0, 1024], np.int64)
    db = DeviceBatch.from_host(b.tokens, b.tok_off, b.principal, b.boundary_tok)
    cache = PrefixCache(next_pow2(4 * db.n_blocks), w.secret, w.ids, w.id_off)
    kv.divergence_boundary(db.tokens, db.tok_off, dev(np.zeros(b.n, np.int32)), dev(pre), dev(tpl_off),
                           boundary_tok=db.boundary_tok, status=cache.status)
    blk = kv.block_offsets(db.tok_off, status=cache.status)
    owner = kv.new_owner(cache.capacity)
    d, _, pre_len = kv.chain_hash_arrival(W.BOUNDARY, db.tokens, db.tok_off, blk, cache.slots, owner, 1, cache.status,
                                          db.principal, cache.salts, db.boundary_tok, n_blocks=db.n_blocks,
                                          n_new=cache.n_new)
    torch.cuda.synchronize()
    cache.check_status()
    bt, _ = oracle.divergence_boundary(b.tokens, b.tok_off, np.zeros(b.n, np.int32), pre, tpl_off)
    assert (db.boundary_tok.cpu().numpy() == bt).all() and (bt == 1024).all()
    salts = oracle.derive_salts(w.secret, w.ids, w.id_off)
    dref = oracle.chain_hash(W.BOUNDARY, b.tokens, b.tok_off, b.principal, salts, bt)
    L, _ = oracle.KeySet(1).arrival_prefix(dref, oracle.block_offsets(b.tok_off))
    got = pre_len.cpu().numpy()
    assert (d.cpu().numpy() == dref).all() and (got == L).all()
    assert got[0] == 0 and (got[1:] >= 64).all()
    first_of_principal = {}
    for r, p in enumerate(b.principal.tolist()):
        first_of_principal.setdefault(p, r)
    for p, r in first_of_principal.items():
        if r > 0:
            assert got[r] == 64          # a principal's first request: only the shared preamble
