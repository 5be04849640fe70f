"""The named-barrier hand-offs of the small-batch kernels (the chain hash in
csrc/kvgov_chain_split.cu, the exact-response keys in csrc/kvgov_response.cu),
checked on the CPU over random interleavings.

Per 32 chains a round warp and a schedule warp meet on barriers of 64
threads: a barrier completes when both warps have reached it (bar.arrive or
bar.sync), releasing the waiter.  Each warp's sequence of barrier operations
and buffer accesses below is the kernel's, block by block.  The model checks
that no interleaving deadlocks, that no barrier completes a phase with one
warp's two arrivals, and that every shared-memory buffer is read after the
write of the same block and rewritten only after that read.  A model of the
protocol, not of the arithmetic: the digests are checked on the GPU."""
import random

import pytest

H, B, E = 0, 1, 4          # barrier ids relative to the pair's base: H, B..D = 1..3, E0/E1 = 4/5


def round_warp(jmax):
    for j in range(jmax):
        yield ("sync", E + (j & 1))                     # the block's second compression and pre-message
        yield ("read", ("pm", j & 1), j)
        for q in range(1, 4):                           # first compression, values 16..63
            yield ("sync", B + q - 1)
            yield ("read", ("kw1", q), j)
        for q in range(4):
            yield ("read", ("kw2", j & 1, q), j)
        yield ("write", ("h",), j)                      # the digest
        yield ("arrive", H)


def schedule_warp(jmax):
    for j in range(jmax):
        if j > 0:
            yield ("sync", H)
            yield ("read", ("h",), j - 1)
        if j == 0:
            for q in range(4):
                yield ("write", ("kw2", 0, q), 0)
            yield ("write", ("pm", 0), 0)
            yield ("arrive", E + 0)
        for q in range(1, 4):
            yield ("write", ("kw1", q), j)
            yield ("arrive", B + q - 1)
        if j + 1 < jmax:
            for q in range(4):
                yield ("write", ("kw2", (j + 1) & 1, q), j + 1)
            yield ("write", ("pm", (j + 1) & 1), j + 1)
            yield ("arrive", E + ((j + 1) & 1))
    if jmax > 0:
        yield ("sync", H)
        yield ("read", ("h",), jmax - 1)


class ProtocolError(AssertionError):
    pass


def run(jmax, rng, warps=(round_warp, schedule_warp)):
    progs = {w.__name__: w(jmax) for w in warps}
    cur = {w: next(p, None) for w, p in progs.items()}
    count, phase, opener, waiting, last_write, reads = {}, {}, {}, {}, {}, {}

    def arrive(b, w):
        if count.get(b, 0) == 32 and opener[b] == w:
            raise ProtocolError(f"barrier {b} completed by {w}'s two arrivals")
        if count.get(b, 0) == 0:
            opener[b] = w
        count[b] = count.get(b, 0) + 32
        if count[b] == 64:
            count[b] = 0
            phase[b] = phase.get(b, 0) + 1

    def step(w):
        cur[w] = next(progs[w], None)

    while any(op is not None for op in cur.values()):
        ready = [w for w, op in cur.items() if op is not None and
                 (w not in waiting or phase.get(waiting[w][0], 0) > waiting[w][1])]
        if not ready:
            raise ProtocolError(f"deadlock at {cur}")
        w = rng.choice(ready)
        op = cur[w]
        if w in waiting:                                # released
            del waiting[w]
            step(w)
            continue
        kind = op[0]
        if kind == "arrive":
            arrive(op[1], w)
            step(w)
        elif kind == "sync":
            ph = phase.get(op[1], 0)
            arrive(op[1], w)
            waiting[w] = (op[1], ph)
        elif kind == "write":
            buf, blk = op[1], op[2]
            prev = last_write.get(buf)
            if prev is not None and reads.get((buf, prev), 0) != 1:
                raise ProtocolError(f"{buf}: block {blk} overwrites block {prev} before it was read")
            last_write[buf] = blk
            step(w)
        else:
            buf, blk = op[1], op[2]
            if last_write.get(buf) != blk:
                raise ProtocolError(f"{buf}: block {blk} read while it holds block {last_write.get(buf)}")
            reads[(buf, blk)] = reads.get((buf, blk), 0) + 1
            step(w)
    if any(count.values()):
        raise ProtocolError(f"a barrier phase left open: {count}")


# The exact-response key kernel's two warps (csrc/kvgov_response.cu,
# response_split_kernel): message m's K_t + W_t go through a ring of two
# buffers; the schedule warp waits for a buffer to be emptied before reusing
# it (EMPTY), the round warp for it to be filled (FULL).  Barrier ids relative
# to the pair's base: FULL0/1 = 0/1, EMPTY0/1 = 2/3.
FULL, EMPTY = 0, 2


def response_round_warp(mmax):
    for m in range(mmax):
        yield ("sync", FULL + (m & 1))
        for q in range(4):
            yield ("read", ("kw", m & 1, q), m)
        if m + 2 < mmax:                                # the schedule warp reuses the buffer
            yield ("arrive", EMPTY + (m & 1))


def response_schedule_warp(mmax):
    for m in range(mmax):
        if m >= 2:
            yield ("sync", EMPTY + (m & 1))
        for q in range(4):
            yield ("write", ("kw", m & 1, q), m)
        yield ("arrive", FULL + (m & 1))


@pytest.mark.parametrize("mmax", [0, 1, 2, 3, 4, 7])
def test_response_ring_is_deadlock_and_race_free(mmax):
    rng = random.Random(100 + mmax)
    warps = (response_round_warp, response_schedule_warp)
    for _ in range(1500):
        run(mmax, rng, warps)


def test_model_catches_a_ring_without_the_empty_wait():
    """A planted mistake: the schedule warp refills a buffer without waiting
    for the round warp to empty it."""
    def sw(mmax):
        for op in response_schedule_warp(mmax):
            if op[0] != "sync":
                yield op

    def rw(mmax):
        for op in response_round_warp(mmax):
            if op[0] != "arrive":
                yield op

    sw.__name__, rw.__name__ = "response_schedule_warp", "response_round_warp"
    with pytest.raises(ProtocolError):
        for seed in range(200):
            run(5, random.Random(seed), (rw, sw))


@pytest.mark.parametrize("jmax", [0, 1, 2, 3, 5, 8])
def test_hand_off_is_deadlock_and_race_free(jmax):
    rng = random.Random(jmax)
    for _ in range(1500):
        run(jmax, rng)


def test_model_catches_a_single_second_compression_buffer():
    """A planted mistake in the model: one buffer for the second compression
    instead of two by block parity."""
    def rw(jmax):
        for op in round_warp(jmax):
            yield (op[0], ("kw2", 0, op[1][2]), op[2]) if op[0] == "read" and op[1][0] == "kw2" else op

    def sw(jmax):
        for op in schedule_warp(jmax):
            yield (op[0], ("kw2", 0, op[1][2]), op[2]) if op[0] == "write" and op[1][0] == "kw2" else op

    rw.__name__, sw.__name__ = "round_warp", "schedule_warp"
    rng = random.Random(0)
    with pytest.raises(ProtocolError):
        for _ in range(500):
            run(4, rng, (rw, sw))


def test_model_catches_a_duplicate_arrival():
    """A planted mistake: the schedule warp announces block 0's second
    compression twice, which lets one warp complete a barrier alone (or, if
    the round warp waited in between, opens a phase that a later block's
    wait would complete before its data is written)."""
    def sw(jmax):
        for op in schedule_warp(jmax):
            yield op
            if op == ("arrive", E + 0):
                yield ("arrive", E + 0)

    sw.__name__ = "schedule_warp"
    with pytest.raises(ProtocolError):
        for seed in range(50):
            run(4, random.Random(seed), (round_warp, sw))


def test_model_catches_a_missing_final_wait():
    """A planted mistake: the schedule warp skips its last wait on H, so the
    round warp's last arrival opens a phase nobody closes."""
    def sw(jmax):
        ops = list(schedule_warp(jmax))
        yield from ops[:-2]

    sw.__name__ = "schedule_warp"
    with pytest.raises(ProtocolError):
        run(3, random.Random(0), (round_warp, sw))
