"""Reading a table tensor back on the host, for the tests: the set of keys it
holds, from the layout the C header documents (main slots, then the side
store of KVGOV_STASH_SLOTS slots).  Test infrastructure only."""
import numpy as np

STASH_SLOTS = 64
STASH_KEYS = 56
STASH_HEADER_SLOTS = 8
STASH_LIVE = 1


def stash_entries(s: np.ndarray) -> list:
    """The live side-store keys of a table read back as a [rows, 32] u8 array."""
    cap = s.shape[0] - STASH_SLOTS
    hdr = s[cap:cap + STASH_HEADER_SLOTS].reshape(-1)
    count = int(hdr[:4].view("<u4")[0])
    state = hdr[32:32 + 4 * STASH_KEYS].view("<u4")
    return [s[cap + STASH_HEADER_SLOTS + e].tobytes() for e in range(min(count, STASH_KEYS)) if state[e] == STASH_LIVE]


def table_keys(slots) -> set:
    """Every key a table tensor holds: the non-empty main slots (first 16
    bytes not all zero) and the live side-store entries."""
    s = slots.cpu().numpy() if hasattr(slots, "cpu") else np.asarray(slots)
    cap = s.shape[0] - STASH_SLOTS
    main = s[:cap]
    keys = {r.tobytes() for r in main[main[:, :16].any(axis=1)]}
    side = stash_entries(s)
    assert len(side) == len(set(side)), "a key is live in two side-store entries"
    assert not keys & set(side), "a key is in a main slot and in the side store"
    return keys | set(side)


def main_slot_storable(k: bytes) -> bool:
    """Keys a main slot can hold: first half not all zero, no all-zero 8-byte
    word in the second half (the others live in the side store)."""
    return any(k[:16]) and any(k[16:24]) and any(k[24:])
