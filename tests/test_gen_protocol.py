"""The table's lock-free protocols inside one launch, checked on the CPU over
random interleavings: the one-launch serving step (kvgov_chain_hash_serve: a
batch's lookups and its own inserts in one launch, told apart by per-slot
generations) and the lookups of the insert-in-chain step (lower bounds while
another batch's insert runs).

Model: the main slots as 8-byte words, and a generation per slot; every
access of a thread is one step, and a random scheduler picks the thread that
steps next.  The kernels' weak and read-only loads (ld.global, ld.global.nc)
may return any value a word held since the launch began -- its value at the
launch's start or any later one -- chosen independently per 8-byte word (a
torn 16-byte read); the 128-bit compare-and-swap and the relaxed loads of the
insert's wait read the current value.  Writes to different words may be seen
in any order.  The threads follow csrc/kvgov_insert.cuh (insert_one, with the
start offset a lookup hands it) and csrc/kvgov_lookup.cuh (lookup_serve,
lookup) step by step, and chain_body's kFuseServe branch for the order of a
request's lookups and inserts.  A model of the protocol, not of the hashing:
the GPU tests check the results."""
import random

import pytest

CAP = 8                        # main slots (a power of two); the probe window is the whole table here
WINDOW = CAP


class Words:
    """Each word's values since the launch began (the first is its value at the start)."""

    def __init__(self, start):
        self.hist = [[v] for v in start]

    def cur(self, i):
        return self.hist[i][-1]

    def write(self, i, v):
        self.hist[i].append(v)

    def weak(self, i, rng):
        return rng.choice(self.hist[i])


def home(key):
    return key[0] & (CAP - 1)


def insert_one(mem, gen, key, g, rng, start=0):
    """insert_one: look first (a weak read), claim an empty-looking slot by a
    compare-and-swap of the first half, write the second half, then the
    generation; wait (coherent reads) for a half-written slot whose first
    half is the key's."""
    for n in range(start, WINDOW):
        pos = (home(key) + n) & (CAP - 1)
        o0 = mem.weak(4 * pos, rng)
        yield
        o1 = mem.weak(4 * pos + 1, rng)
        yield
        if o0 == 0 or o1 == 0:
            c0, c1 = mem.cur(4 * pos), mem.cur(4 * pos + 1)
            claimed = c0 == 0 and c1 == 0
            if claimed:
                mem.write(4 * pos, key[0])
                mem.write(4 * pos + 1, key[1])
            else:
                o0, o1 = c0, c1
            yield
            if claimed:
                mem.write(4 * pos + 2, key[2])
                mem.write(4 * pos + 3, key[3])
                yield
                gen.write(pos, g)
                yield
                return "new", pos
        if (o0, o1) != (key[0], key[1]):
            continue
        w2 = mem.weak(4 * pos + 2, rng)
        yield
        w3 = mem.weak(4 * pos + 3, rng)
        yield
        while w2 == 0 or w3 == 0:                       # the claimer's second half is on its way
            w2 = mem.cur(4 * pos + 2)
            yield
            w3 = mem.cur(4 * pos + 3)
            yield
        if (w2, w3) == (key[2], key[3]):
            return "dup", pos
    return "full", None


def lookup_serve(mem, gen, key, floor, g, rng, careless_start=False):
    """lookup_serve: (1 cached, 0 in the table with another generation, -1 not
    found) and the offset where an insert may begin its walk.  careless_start
    (a planted mistake): the walk's start moves past every non-empty slot,
    the key's own half-written first half included."""
    h = home(key)
    gv_home = gen.weak(h, rng)                          # read with the home slot
    yield
    start, open_ = 0, True
    for n in range(WINDOW):
        pos = (h + n) & (CAP - 1)
        a0 = mem.weak(4 * pos, rng)
        yield
        a1 = mem.weak(4 * pos + 1, rng)
        yield
        if a0 == 0 and a1 == 0:
            return -1, (n if open_ else start)
        mine = (a0, a1) == (key[0], key[1])
        if mine:
            b0 = mem.weak(4 * pos + 2, rng)
            yield
            b1 = mem.weak(4 * pos + 3, rng)
            yield
            if (b0, b1) == (key[2], key[3]):
                if n == 0:
                    gv = gv_home
                else:
                    gv = gen.weak(pos, rng)
                    yield
                return (1 if floor <= gv < g else 0), start
        if open_ and (mine or a0 == 0 or a1 == 0) and not careless_start:
            start, open_ = n, False
    return -1, (WINDOW if open_ else start)


def lookup(mem, key, rng):
    """lookup (the read-only walk of the insert-in-chain launch's lookups)."""
    h = home(key)
    for n in range(WINDOW):
        pos = (h + n) & (CAP - 1)
        a0 = mem.weak(4 * pos, rng)
        yield
        a1 = mem.weak(4 * pos + 1, rng)
        yield
        if a0 == 0 and a1 == 0:
            return False
        if (a0, a1) == (key[0], key[1]):
            b0 = mem.weak(4 * pos + 2, rng)
            yield
            b1 = mem.weak(4 * pos + 3, rng)
            yield
            if (b0, b1) == (key[2], key[3]):
                return True
    return False


def serve_request(mem, gen, keys, floor, g, rng, log, careless_start=False):
    """One thread of kFuseServe: block j looked up while blocks 0..j-1 were all
    cached, inserted unless cached or already added by this batch."""
    hits = 0
    for j, key in enumerate(keys):
        res, start = -1, 0
        if hits == j:
            res, start = yield from lookup_serve(mem, gen, key, floor, g, rng, careless_start)
            log["lookups"].append((key, res))
        if res == 1:
            hits = j + 1
        elif res < 0:
            r, pos = yield from insert_one(mem, gen, key, g, rng, start)
            log["inserts"].append((key, r, pos))
    log["prefix"].append((tuple(keys), hits))


def run(threads, rng, max_steps=200000):
    live = list(threads)
    steps = 0
    while live:
        t = rng.choice(live)
        try:
            next(t)
        except StopIteration:
            live.remove(t)
        steps += 1
        assert steps < max_steps, "no progress"


def make_key(rng, pool_home):
    k0 = rng.choice(pool_home)
    k1 = rng.choice([0, rng.randrange(1, 50)]) if k0 != 0 else rng.randrange(1, 50)   # one zero word at most
    return (k0, k1, rng.randrange(1, 1000), rng.randrange(1, 1000))


def fill(keys_with_gen, floor, rng):
    """The table at the launch's start: the old keys, inserted one after
    another, with generations in [floor, g); every other slot's generation a
    stale value below floor."""
    words = [0] * (4 * CAP)
    gens = [rng.randrange(0, floor) for _ in range(CAP)]
    for key, gv in keys_with_gen:
        for n in range(WINDOW):
            pos = (home(key) + n) & (CAP - 1)
            if words[4 * pos] == 0 and words[4 * pos + 1] == 0:
                words[4 * pos:4 * pos + 4] = key
                gens[pos] = gv
                break
    return Words(words), Words(gens)


def table_keys(mem):
    got = []
    for pos in range(CAP):
        w = tuple(mem.cur(4 * pos + i) for i in range(4))
        if w[0] or w[1]:
            got.append(w)
    return got


@pytest.mark.parametrize("seed", range(300))
def test_serve_lookups_never_count_the_batch_s_own_keys(seed):
    """Whatever the interleaving and whatever older values the weak reads
    return: a lookup counts a key as cached exactly when it was in the table
    before the launch; every request's prefix is that of the oracle's probe
    before the batch's insert; afterwards each key is in the table once, the
    new ones with the batch's generation, and the inserts report each new key
    as new exactly once."""
    rng = random.Random(seed)
    floor = rng.randrange(1, 4)
    g = floor + rng.randrange(1, 4)
    pool_home = [rng.randrange(0, CAP) for _ in range(3)]           # few homes: long walks, collisions
    old = list({make_key(rng, pool_home) for _ in range(rng.randrange(0, 3))})
    mem, gen = fill([(k, rng.randrange(floor, g)) for k in old], floor, rng)
    fresh = list({make_key(rng, pool_home) for _ in range(4)} - set(old))
    requests = []
    for _ in range(rng.randrange(2, 5)):                            # requests share keys: in-batch duplicates
        keys = [rng.choice(old)] if old and rng.random() < 0.6 else []
        keys += [rng.choice(fresh) for _ in range(rng.randrange(1, 3))]
        requests.append(keys)
    log = {"lookups": [], "inserts": [], "prefix": []}
    run([serve_request(mem, gen, keys, floor, g, rng, log) for keys in requests], rng)
    oldset = set(old)
    for key, res in log["lookups"]:
        assert (res == 1) == (key in oldset), (key, res)
    for keys, hits in log["prefix"]:
        want = next((j for j, k in enumerate(keys) if k not in oldset), len(keys))
        assert hits == want
    inserted = {k for keys, hits in log["prefix"] for k in keys[hits:]}
    assert all(r != "full" for _, r, _ in log["inserts"])
    final = table_keys(mem)
    assert sorted(final) == sorted(oldset | inserted), "every key once, none lost"
    new = [k for k, r, _ in log["inserts"] if r == "new"]
    assert sorted(new) == sorted(inserted - oldset), "each new key claimed once"
    for k, r, pos in log["inserts"]:
        if r == "new":
            assert gen.cur(pos) == g


@pytest.mark.parametrize("seed", range(200))
def test_lookups_racing_another_batch_s_insert_give_lower_bounds(seed):
    """The insert-in-chain launch: lookups of this batch's keys while threads
    insert the previous batch's.  A lookup never finds a key that is not in
    the table at the launch's end, and always finds one that was there at its
    start -- so a prefix from these lookups is at most the prefix on the
    table after the insert, and the probe that resumes from it is exact."""
    rng = random.Random(10_000 + seed)
    pool_home = [rng.randrange(0, CAP) for _ in range(3)]
    old = list({make_key(rng, pool_home) for _ in range(rng.randrange(0, 3))})
    mem, gen = fill([(k, 1) for k in old], 1, rng)
    prev = list({make_key(rng, pool_home) for _ in range(3)} - set(old))
    probes = [rng.choice(old + prev + [make_key(rng, pool_home)]) for _ in range(4)]
    found = []

    def inserter(key):
        yield from insert_one(mem, gen, key, 2, rng)

    def looker(key):
        f = yield from lookup(mem, key, rng)
        found.append((key, f))

    run([inserter(k) for k in prev] + [looker(k) for k in probes], rng)
    final = set(table_keys(mem))
    assert final == set(old) | set(prev)
    for key, f in found:
        if f:
            assert key in final, "a lookup found a key that is not in the table"
        if key in old:
            assert f, "a lookup missed a key that was in the table before the launch"


def test_a_planted_mistake_fails_the_model():
    """The model catches the mistake it is for: a lookup that counts any
    generation below the batch's as cached (no floor), with stale
    generations below the floor left in empty slots, finds this batch's own
    keys cached in some interleaving."""
    caught = False
    for seed in range(300):
        rng = random.Random(seed)
        floor, g = 3, 4
        pool_home = [rng.randrange(0, CAP) for _ in range(2)]
        mem, gen = fill([], floor, rng)
        keys = list({make_key(rng, pool_home) for _ in range(3)})
        log = {"lookups": [], "inserts": [], "prefix": []}
        run([serve_request(mem, gen, [k], 0, g, rng, log) for k in keys for _ in range(2)], rng)
        if any(res == 1 for _, res in log["lookups"]):
            caught = True
            break
    assert caught


def test_a_careless_insert_start_fails_the_model():
    """And the other one: a lookup that hands the insert a start past a slot
    holding the key's own first half (claimed by another thread, second half
    not yet written) lets the key be stored twice in some interleaving."""
    caught = False
    for seed in range(2000):
        rng = random.Random(seed)
        pool_home = [rng.randrange(0, CAP)]
        mem, gen = fill([], 1, rng)
        keys = list({make_key(rng, pool_home) for _ in range(2)})
        log = {"lookups": [], "inserts": [], "prefix": []}
        run([serve_request(mem, gen, [k], 1, 2, rng, log, careless_start=True) for k in keys for _ in range(3)],
            rng)
        final = table_keys(mem)
        if len(final) != len(set(final)):
            caught = True
            break
    assert caught
