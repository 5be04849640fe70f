"""The CPU oracle against its pins (no GPU), and evidence that the pins bite:
copies of oracle.c with a planted mistake must fail at least one pin."""
import os
import shutil
import subprocess

import pytest

import oracle
from tests import pins

ORACLE_C = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")


@pytest.mark.parametrize("pin", pins.PINS, ids=[p.__name__ for p in pins.PINS])
def test_pin(pin):
    pin()


def test_constants_are_derived_not_typed():
    """K and H(0) come from exact integer roots of the first primes (FIPS 180-4
    section 4.2.2 / 5.3.3); spot-check the definition with Python integers."""
    k, iv = oracle.sha256_constants()

    def iroot(n, e):
        x = int(round(n ** (1.0 / e)))
        while x ** e > n:
            x -= 1
        while (x + 1) ** e <= n:
            x += 1
        return x

    primes = [p for p in range(2, 400) if all(p % d for d in range(2, int(p ** 0.5) + 1))][:64]
    for t, p in enumerate(primes):
        assert int(k[t]) == iroot(p << 96, 3) & 0xFFFFFFFF
    for i, p in enumerate(primes[:8]):
        assert int(iv[i]) == iroot(p << 64, 2) & 0xFFFFFFFF


# Each entry: (name, exact text in oracle.c, replacement).  A plausible slip
# in every part of the oracle: SHA rounds and schedule, HMAC, serialisation,
# salt placement, boundary index, concatenation order, lookup stop rule.
MUTATIONS = [
    ("bsig1_rotation", "ROTR(x, 6) ^ ROTR(x, 11) ^ ROTR(x, 25)", "ROTR(x, 6) ^ ROTR(x, 11) ^ ROTR(x, 24)"),
    ("maj_is_ch", "return (x & y) ^ (x & z) ^ (y & z);", "return (x & y) ^ (~x & z);"),
    ("schedule_drops_w7", "SSIG1(W[t - 2]) + W[t - 7] + SSIG0(W[t - 15])", "SSIG1(W[t - 2]) + SSIG0(W[t - 15])"),
    ("length_in_bytes", "uint64_t bits = (uint64_t)len * 8u;", "uint64_t bits = (uint64_t)len;"),
    ("hmac_ipad_is_opad", "inner_msg[i] = K0[i] ^ 0x36;", "inner_msg[i] = K0[i] ^ 0x5c;"),
    ("hmac_long_key_not_hashed", "if (key_len > 64) oracle_sha256(key, key_len, K0);",
     "if (key_len > 64) memcpy(K0, key, 64);"),
    ("tokens_big_endian", "out[4 * i] = (uint8_t)v;\n        out[4 * i + 1] = (uint8_t)(v >> 8);",
     "out[4 * i + 1] = (uint8_t)v;\n        out[4 * i] = (uint8_t)(v >> 8);"),
    ("root_salt_dropped", "if (mode == ORACLE_ROOT) k = 0;", "if (mode == ORACLE_ROOT) k = -1;"),
    ("boundary_ceil", "k = boundary_tok[r] / ORACLE_B;", "k = (boundary_tok[r] + ORACLE_B - 1) / ORACLE_B;"),
    ("boundary_parent_dropped", "if (j > 0) { memcpy(msg + m, prev, 32); m += 32; }", "if (0) { }"),
    ("salt_after_parent",
     "memcpy(msg + m, sigma, 32); m += 32;\n                if (j > 0) { memcpy(msg + m, prev, 32); m += 32; }",
     "if (j > 0) { memcpy(msg + m, prev, 32); m += 32; }\n                memcpy(msg + m, sigma, 32); m += 32;"),
    ("lookup_counts_all_hits",
     "while (j < nb && oracle_set_contains(set_keys, n_set, digests + 32 * (size_t)(blk_off[r] + j)))\n            j++;",
     "for (int64_t q = 0; q < nb; q++) j += oracle_set_contains(set_keys, n_set, digests + 32 * (size_t)(blk_off[r] + q));"),
    ("arrival_caches_before_lookup",
     "        while (j < nb && chain_set_contains(&s, req + 32 * (size_t)j))\n            j++;\n"
     "        prefix_blocks[r] = (int32_t)j;\n"
     "        for (int64_t q = 0; q < nb; q++)\n"
     "            if (!oracle_key_is_zero(req + 32 * (size_t)q)) chain_set_add(&s, req + 32 * (size_t)q);",
     "        for (int64_t q = 0; q < nb; q++)\n"
     "            if (!oracle_key_is_zero(req + 32 * (size_t)q)) chain_set_add(&s, req + 32 * (size_t)q);\n"
     "        while (j < nb && chain_set_contains(&s, req + 32 * (size_t)j))\n            j++;\n"
     "        prefix_blocks[r] = (int32_t)j;"),
    ("arrival_initial_set_dropped",
     "for (int64_t i = 0; i < n_set; i++) chain_set_add(&s, set_keys + 32 * (size_t)i);", ""),
    ("arrival_counts_all_hits",
     "        while (j < nb && chain_set_contains(&s, req + 32 * (size_t)j))\n            j++;",
     "        for (int64_t q = 0; q < nb; q++) j += chain_set_contains(&s, req + 32 * (size_t)q);"),
    ("boundary_off_by_one",
     "while (i < len_r && i < len_t && tokens[tok_off[r] + i] == tpl_tokens[tpl_off[t] + i])\n                i++;",
     "while (i < len_r && i < len_t && tokens[tok_off[r] + i] == tpl_tokens[tpl_off[t] + i])\n                i++;\n"
     "            if (i < len_r && i < len_t) i++;"),
    ("boundary_any_takes_first", "if (i > best) best = i;", "if (best == 0) best = i;"),
    ("boundary_none_compares", "        if (id == -1) continue;\n", ""),
    ("response_salt_after_prompt", "oracle_sha256(msg, salt_len + 4 * (size_t)len, keys + 32 * (size_t)r);",
     "oracle_sha256(msg + salt_len, 4 * (size_t)len, keys + 32 * (size_t)r);"),
    ("response_token_bytes_swapped",
     "msg[salt_len + 4 * i] = (uint8_t)v;\n            msg[salt_len + 4 * i + 1] = (uint8_t)(v >> 8);",
     "msg[salt_len + 4 * i + 1] = (uint8_t)v;\n            msg[salt_len + 4 * i] = (uint8_t)(v >> 8);"),
    ("origami_ascending_order", "return (x < y) - (x > y);", "return (x > y) - (x < y);"),
    ("origami_budget_sign", "const double lm = ((double)m - K) / inv_sum;", "const double lm = ((double)m + K) / inv_sum;"),
    ("origami_no_clamp", "(1.0 - lam / x > 0.0 ? 1.0 - lam / x : 0.0)", "(1.0 - lam / x)"),
    ("arrival_zero_key_stored",
     "            if (!oracle_key_is_zero(req + 32 * (size_t)q)) chain_set_add(&s, req + 32 * (size_t)q);",
     "            chain_set_add(&s, req + 32 * (size_t)q);"),
    ("set_zero_key_stored", "        if (oracle_key_is_zero(key)) { flags |= ORACLE_FLAG_ZERO_KEY; continue; }", ""),
    ("set_refuses_zero_first_half",
     "    for (int i = 0; i < 32; i++)\n        if (key[i] != 0) return 0;",
     "    for (int i = 0; i < 16; i++)\n        if (key[i] != 0) return 0;"),
    ("set_refuses_zero_last_word",
     "    for (int i = 0; i < 32; i++)\n        if (key[i] != 0) return 0;\n    return 1;",
     "    { int z = 1; for (int i = 24; i < 32; i++) if (key[i] != 0) z = 0; if (z) return 1; }\n"
     "    for (int i = 0; i < 32; i++)\n        if (key[i] != 0) return 0;\n    return 1;"),
]


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(tmp_path, name, old, new):
    src = open(ORACLE_C).read()
    assert src.count(old) == 1, f"mutation {name} no longer matches oracle.c"
    mutated = tmp_path / "oracle_mut.c"
    mutated.write_text(src.replace(old, new))
    so = tmp_path / "liboracle_mut.so"
    subprocess.run([shutil.which("gcc") or "gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", str(so),
                    str(mutated)], check=True)
    failed = []
    with oracle.using_library(oracle.load_library(str(so))):
        for pin in pins.PINS:
            try:
                pin()
            except AssertionError:
                failed.append(pin.__name__)
    assert failed, f"planted mistake {name} passed every pin"
