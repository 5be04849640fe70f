"""Seeded synthetic workloads shaped like the paper's prompts.

Inputs only: this module draws tokens, principals, secrets and random table
keys with numpy's PCG64 (``np.random.default_rng(seed)``) in a fixed,
documented order.  It contains none of the hashing or lookup arithmetic, and it
is the only code that both the CUDA path's tests and the CPU oracle consume.

Token ids are uniform in [0, 152064), the size of the Qwen2.5 vocabulary the
paper's TTFT experiments use (section 3.4, section 5.7).  Principal p's id is
the 4-byte little-endian encoding of p.  The HMAC secret is 32 bytes drawn
first from each workload's generator.

Workloads (sizes at full scale; ``n_req`` shrinks a workload for tests):

  tiny       64 x 256 tokens, seed 1; requests 0-31 share one 128-token
             template prefix; principal = r mod 8; ROOT; a 1024-slot table
             holds the chains of requests 0-15; all 64 are probed.
  sysprompt  1024 x 2119 tokens (132 full blocks + a 7-token tail); one
             shared 1024-token system prefix, then uniform tokens; 64
             principals drawn Zipf(s = 1.1) over ranks 1..64; ROOT; a
             65,536-slot table holds the chains of requests 0-255; all probed.
             Stands in for the paper's 2119-token shared system prompt
             (section 5.7, Table 8).
  template   8192 x 512 tokens from one 512-token template with 4 fields of
             8 tokens at offsets 96/200/304/408, each field value drawn
             uniformly from its own seeded 1000-entry dictionary of 8-token
             strings; 256 principals uniform; UNSALTED, ROOT and BOUNDARY
             (b = 96, block 6) each with its own 262,144-slot table holding
             requests 0-4095; requests 4096-8191 are probed.  Stands in for
             the structured, form-filled prompts of section 3.4.
  probe      a 2^24-slot table at load factor 0.5: the ROOT chains of 8192
             prior 512-token requests (262,144 keys) plus 8,126,464 random
             32-byte keys; 65,536 x 512-token requests of which 30 % reuse a
             prior request's first c ~ U{0..31} blocks (and its principal),
             the rest are fresh; 1024 principals uniform; ROOT; all probed.
  long       256 x 32,768 tokens (2048 blocks per chain); a 64-token prefix
             shared by all requests, then uniform; 4096 principals uniform;
             BOUNDARY at token 64 (block 4).  Fresh seed per run.
  wide       131,072 x 128 tokens (8 blocks per chain), otherwise as long.

Seeds: tiny uses 1; sysprompt, template and probe use 2026 + their position
in the list above (2027, 2028, 2029), after the paper's `--seed 2026`
(section 7); long and wide take the seed of each run.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

VOCAB = 152064
UNSALTED, ROOT, BOUNDARY = 0, 1, 2

NAMES = ("tiny", "sysprompt", "template", "probe", "long", "wide")
DEFAULT_SEEDS = {"tiny": 1, "sysprompt": 2027, "template": 2028, "probe": 2029, "long": 2030, "wide": 2031}


@dataclass
class Batch:
    tokens: np.ndarray          # int32, flat, 16-byte-aligned start when copied to the device
    tok_off: np.ndarray         # int64 [n + 1]
    principal: np.ndarray       # int32 [n], row of the salt table
    boundary_tok: np.ndarray    # int32 [n], boundary token offset (BOUNDARY mode)

    @property
    def n(self) -> int:
        return len(self.tok_off) - 1

    def lengths(self) -> np.ndarray:
        return np.diff(self.tok_off)


@dataclass
class Workload:
    name: str
    seed: int
    secret: bytes
    ids: np.ndarray             # uint8 principal-id bytes (CSR)
    id_off: np.ndarray          # int64 [n_principals + 1]
    batch: Batch
    modes: tuple                # salt placements to run
    capacity: int               # table slots (power of two)
    fill: tuple                 # requests [fill[0], fill[1]) of `fill_from` whose chains pre-fill the table
    fill_from: str = "batch"    # "batch" or "prior"
    prior: Batch | None = None  # earlier requests whose chains fill the table (probe workload)
    random_keys: np.ndarray | None = None   # uint8 [m, 32] extra resident keys
    probe: tuple = (0, 0)       # requests [probe[0], probe[1]) of `batch` that are probed
    info: dict = field(default_factory=dict)

    @property
    def n_principals(self) -> int:
        return len(self.id_off) - 1


def principal_ids(n_p: int):
    """Principal p's id = 4-byte little-endian p."""
    ids = np.arange(n_p, dtype="<u4").view(np.uint8).copy()
    id_off = np.arange(n_p + 1, dtype=np.int64) * 4
    return ids, id_off


def _uniform(rng, shape):
    return rng.integers(0, VOCAB, size=shape, dtype=np.int32)


def _regular(tokens_2d: np.ndarray, principal, boundary=0) -> Batch:
    n, L = tokens_2d.shape
    return Batch(tokens=np.ascontiguousarray(tokens_2d.reshape(-1)),
                 tok_off=np.arange(n + 1, dtype=np.int64) * L,
                 principal=np.ascontiguousarray(principal, dtype=np.int32),
                 boundary_tok=np.full(n, boundary, dtype=np.int32))


def gini(counts) -> float:
    x = np.sort(np.asarray(counts, dtype=np.float64))
    n = len(x)
    if n == 0 or x.sum() == 0:
        return 0.0
    cum = np.cumsum(x)
    return float((n + 1 - 2 * (cum.sum() / cum[-1])) / n)


def tiny(seed: int = 1, n_req: int = 64) -> Workload:
    # draw order: secret, tokens [n, 256], template [128]
    rng = np.random.default_rng(seed)
    secret = rng.bytes(32)
    toks = _uniform(rng, (n_req, 256))
    template = _uniform(rng, 128)
    toks[: min(32, n_req), :128] = template
    ids, id_off = principal_ids(8)
    return Workload("tiny", seed, secret, ids, id_off, _regular(toks, np.arange(n_req) % 8),
                    modes=(ROOT,), capacity=1024, fill=(0, min(16, n_req)), probe=(0, n_req))


def sysprompt(seed: int = 2027, n_req: int = 1024, fill_n: int = 256) -> Workload:
    # draw order: secret, system prefix [1024], suffix tokens [n, 1095], principals
    rng = np.random.default_rng(seed)
    secret = rng.bytes(32)
    prefix = _uniform(rng, 1024)
    toks = np.empty((n_req, 2119), dtype=np.int32)
    toks[:, :1024] = prefix
    toks[:, 1024:] = _uniform(rng, (n_req, 2119 - 1024))
    ranks = np.arange(1, 65, dtype=np.float64)
    pz = ranks ** -1.1
    pz /= pz.sum()
    principal = rng.choice(64, size=n_req, p=pz)
    ids, id_off = principal_ids(64)
    w = Workload("sysprompt", seed, secret, ids, id_off, _regular(toks, principal),
                 modes=(ROOT,), capacity=65536, fill=(0, min(fill_n, n_req)), probe=(0, n_req))
    w.info["gini"] = gini(np.bincount(principal, minlength=64))
    return w


FIELD_OFFSETS = (96, 200, 304, 408)


def template(seed: int = 2028, n_req: int = 8192, capacity: int = 262144) -> Workload:
    # draw order: secret, template [512], 4 dictionaries [1000, 8] each,
    # field choices [n, 4], principals [n]
    rng = np.random.default_rng(seed)
    secret = rng.bytes(32)
    tmpl = _uniform(rng, 512)
    dicts = [_uniform(rng, (1000, 8)) for _ in FIELD_OFFSETS]
    choice = rng.integers(0, 1000, size=(n_req, len(FIELD_OFFSETS)))
    principal = rng.integers(0, 256, size=n_req)
    toks = np.broadcast_to(tmpl, (n_req, 512)).copy()
    for f, off in enumerate(FIELD_OFFSETS):
        toks[:, off:off + 8] = dicts[f][choice[:, f]]
    ids, id_off = principal_ids(256)
    half = n_req // 2
    return Workload("template", seed, secret, ids, id_off, _regular(toks, principal, boundary=96),
                    modes=(UNSALTED, ROOT, BOUNDARY), capacity=capacity, fill=(0, half), probe=(half, n_req))


def probe(seed: int = 2029, n_req: int = 65536, n_prior: int = 8192, capacity: int = 1 << 24,
          n_random: int | None = None) -> Workload:
    # draw order: secret, prior tokens [n_prior, 512], prior principals,
    # fresh tokens [n, 512], reuse flags, prior choice, cut c, fresh principals,
    # random keys [n_random, 32]
    rng = np.random.default_rng(seed)
    secret = rng.bytes(32)
    prior_toks = _uniform(rng, (n_prior, 512))
    prior_principal = rng.integers(0, 1024, size=n_prior)
    toks = _uniform(rng, (n_req, 512))
    reuse = rng.random(n_req) < 0.3
    src = rng.integers(0, n_prior, size=n_req)
    cut = rng.integers(0, 32, size=n_req)
    principal = rng.integers(0, 1024, size=n_req)
    rows = np.nonzero(reuse)[0]
    keep = np.arange(512)[None, :] < 16 * cut[rows][:, None]
    toks[rows] = np.where(keep, prior_toks[src[rows]], toks[rows])
    principal = np.where(reuse, prior_principal[src], principal)
    if n_random is None:
        n_random = capacity // 2 - n_prior * 32
    keys = rng.integers(0, 256, size=(max(n_random, 0), 32), dtype=np.uint8)
    ids, id_off = principal_ids(1024)
    w = Workload("probe", seed, secret, ids, id_off, _regular(toks, principal),
                 modes=(ROOT,), capacity=capacity, fill=(0, n_prior), fill_from="prior",
                 prior=_regular(prior_toks, prior_principal), random_keys=keys, probe=(0, n_req))
    w.info.update(reuse=reuse, src=src, cut=np.where(reuse, cut, 0))
    return w


def _sweep(name: str, seed: int, n_req: int, length: int) -> Workload:
    # draw order: secret, shared prefix [64], tokens [n, length - 64], principals
    rng = np.random.default_rng(seed)
    secret = rng.bytes(32)
    prefix = _uniform(rng, 64)
    toks = np.empty((n_req, length), dtype=np.int32)
    toks[:, :64] = prefix
    toks[:, 64:] = _uniform(rng, (n_req, length - 64))
    principal = rng.integers(0, 4096, size=n_req)
    ids, id_off = principal_ids(4096)
    return Workload(name, seed, secret, ids, id_off, _regular(toks, principal, boundary=64),
                    modes=(BOUNDARY,), capacity=0, fill=(0, 0), probe=(0, 0))


def long(seed: int = 2030, n_req: int = 256) -> Workload:
    return _sweep("long", seed, n_req, 32768)


def wide(seed: int = 2031, n_req: int = 131072) -> Workload:
    return _sweep("wide", seed, n_req, 128)


def make(name: str, seed: int | None = None, **kw) -> Workload:
    fn = {"tiny": tiny, "sysprompt": sysprompt, "template": template, "probe": probe, "long": long,
          "wide": wide}[name]
    return fn(DEFAULT_SEEDS[name] if seed is None else seed, **kw)


def ragged(seed: int, lengths) -> Batch:
    """Requests of the given token lengths, uniform tokens, principals 0..7,
    boundary offsets cycling over 0, 15, 16, 17, 31, 32, 64, 10**6."""
    rng = np.random.default_rng(seed)
    lengths = np.asarray(lengths, dtype=np.int64)
    tok_off = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    tokens = _uniform(rng, int(tok_off[-1]))
    n = len(lengths)
    principal = rng.integers(0, 8, size=n).astype(np.int32)
    cyc = np.array([0, 15, 16, 17, 31, 32, 64, 10 ** 6], dtype=np.int32)
    boundary = cyc[np.arange(n) % len(cyc)]
    return Batch(tokens=tokens, tok_off=tok_off, principal=principal, boundary_tok=boundary)


@dataclass
class AuditBatch:
    """ORIGAMI audit problems (paper section 4.3): tenant values at risk in
    CSR form and one budget per problem."""
    values: np.ndarray          # float32 [total tenants]
    off: np.ndarray             # int64 [n_prob + 1]
    budget: np.ndarray          # float32 [n_prob]

    @property
    def n(self) -> int:
        return len(self.off) - 1


def audit(seed: int = 2032, n_prob: int = 1 << 20, n_tenants: int = 50, budget: float = 10.0,
          alpha: float = 1.29) -> AuditBatch:
    """The adversarial-load setting of section 5.5, batched: n_prob problems
    of n_tenants tenants whose values are Pareto(alpha) (x_m = 1; alpha = 1.29
    gives Gini about 0.63), budget K each."""
    rng = np.random.default_rng(seed)
    values = (1.0 + rng.pareto(alpha, n_prob * n_tenants)).astype(np.float32)
    off = np.arange(0, n_prob * n_tenants + 1, n_tenants, dtype=np.int64)
    return AuditBatch(values=values, off=off, budget=np.full(n_prob, budget, np.float32))


def audit_ragged(seed: int, n_prob: int, max_tenants: int = 300) -> AuditBatch:
    """Audit problems of 0..max_tenants tenants, Pareto or uniform values (a
    fifth of the problems all-equal), budgets in [0, n + 2] (some above n)."""
    rng = np.random.default_rng(seed)
    sizes = rng.integers(0, max_tenants + 1, n_prob)
    vals = []
    for n in sizes:
        if rng.random() < 0.2:
            vals.append(np.full(n, float(rng.uniform(0.5, 5.0)), np.float32))
        else:
            vals.append((1.0 + rng.pareto(float(rng.uniform(0.8, 3.0)), n)).astype(np.float32))
    off = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    budget = (rng.random(n_prob) * (sizes + 2)).astype(np.float32)
    return AuditBatch(values=np.concatenate(vals + [np.zeros(0, np.float32)]).astype(np.float32), off=off,
                      budget=budget)
