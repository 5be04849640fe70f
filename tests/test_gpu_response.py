"""Exact-response cache keys on the GPU (kvgov_response_key) against the
oracle, bit-exact, and their use as table keys.  Marked gpu."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_09225_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


def dev(a, dtype=None):
    return torch.from_numpy(np.ascontiguousarray(a if dtype is None else np.asarray(a, dtype=dtype))).to(DEV)


def gpu_keys(kv, mode, toks, tok_off, pr, salts):
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    k = kv.response_key(mode, dev(toks, np.int32), dev(tok_off, np.int64), dev(pr, np.int32), dev(salts, np.uint8),
                        status=st)
    torch.cuda.synchronize()
    return k.cpu().numpy(), int(st.item())


@pytest.mark.parametrize("mode", [W.UNSALTED, W.ROOT])
def test_response_key_every_length(kv, mode):
    """Lengths 0..300 tokens (every padding edge, both with and without the
    32-byte salt), one request per length, packed back to back so that
    request starts fall on every 4-byte offset."""
    rng = np.random.default_rng(30 + mode)
    lens = np.arange(301)
    rng.shuffle(lens)
    tok_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    toks = rng.integers(0, W.VOCAB, int(tok_off[-1]), dtype=np.int32)
    salts = oracle.derive_salts(b"rk", *W.principal_ids(5))
    pr = rng.integers(0, 5, len(lens)).astype(np.int32)
    got, st = gpu_keys(kv, mode, toks, tok_off, pr, salts)
    assert st == 0
    assert (got == oracle.response_key(mode, toks, tok_off, pr, salts)).all()


@pytest.mark.parametrize("mode", [W.UNSALTED, W.ROOT])
@pytest.mark.parametrize("delta", [0, 1])
def test_response_key_at_the_split_limit(kv, mode, delta):
    """Batches at the small-batch kernel's limit (192 requests per SM, two
    warps per 32 requests) and one past it (one thread per request): lengths
    0..600 tokens, every start offset, empty prompts included."""
    n = 192 * torch.cuda.get_device_properties(0).multi_processor_count + delta
    rng = np.random.default_rng(40 + delta + 2 * mode)
    lens = rng.integers(0, 601, n)
    lens[:50] = 0
    tok_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    toks = rng.integers(0, W.VOCAB, int(tok_off[-1]), dtype=np.int32)
    salts = oracle.derive_salts(b"limit", *W.principal_ids(16))
    pr = rng.integers(0, 16, n).astype(np.int32)
    got, st = gpu_keys(kv, mode, toks, tok_off, pr, salts)
    assert st == 0
    assert (got == oracle.response_key(mode, toks, tok_off, pr, salts)).all()


@pytest.mark.parametrize("name", ["sysprompt", "wide", "long"])
def test_response_key_workloads(kv, name):
    w = W.make(name, seed=71) if name in ("wide", "long") else W.make(name)
    b = w.batch
    salts = oracle.derive_salts(w.secret, w.ids, w.id_off)
    got, st = gpu_keys(kv, W.ROOT, b.tokens, b.tok_off, b.principal, salts)
    assert st == 0
    assert (got == oracle.response_key(W.ROOT, b.tokens, b.tok_off, b.principal, salts)).all()


def test_response_key_cache_round_trip(kv):
    """Responses cached for some (principal, prompt) pairs: a repeat of the
    same prompt by the same principal hits, by another principal misses, and
    a prompt differing only in its last token misses."""
    rng = np.random.default_rng(33)
    prompts = [rng.integers(0, W.VOCAB, int(n), dtype=np.int32) for n in rng.integers(1, 500, 64)]
    salts = oracle.derive_salts(b"cache", *W.principal_ids(4))
    pr = (np.arange(64) % 4).astype(np.int32)
    off = np.concatenate([[0], np.cumsum([len(x) for x in prompts])]).astype(np.int64)
    keys, _ = gpu_keys(kv, W.ROOT, np.concatenate(prompts), off, pr, salts)
    slots = kv.new_table(1 << 10)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    kv.insert(slots, dev(keys[:32]), st)
    probe = [prompts[5], prompts[40], prompts[6], np.concatenate([prompts[7][:-1], [(prompts[7][-1] + 1) % W.VOCAB]])]
    ppr = np.array([pr[5], pr[40], (pr[6] + 1) % 4, pr[7]], np.int32)
    poff = np.concatenate([[0], np.cumsum([len(x) for x in probe])]).astype(np.int64)
    pk, _ = gpu_keys(kv, W.ROOT, np.concatenate(probe).astype(np.int32), poff, ppr, salts)
    hit = kv.probe(slots, dev(pk), dev(np.arange(5, dtype=np.int64)), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and list(hit.cpu().numpy()) == [1, 0, 0, 0]


def test_response_key_bad_principal_flagged(kv):
    toks = np.arange(40, dtype=np.int32)
    off = np.array([0, 10, 40], np.int64)
    salts = oracle.derive_salts(b"x", *W.principal_ids(2))
    got, st = gpu_keys(kv, W.ROOT, toks, off, np.array([0, 7], np.int32), salts)
    assert st == kv.F_BADINDEX
    assert (got[0] == oracle.response_key(W.ROOT, toks[:10], off[:2], np.zeros(1, np.int32), salts)[0]).all()
