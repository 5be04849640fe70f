/*
 * oracle.c -- plain, slow CPU oracle for KVGov's salted block-hash chain and
 * block prefix-cache lookup (arxiv 2608.09225).
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the package smoke check and the
 * benchmark's CPU-baseline leg load this library.  The CUDA library never
 * links, includes or calls it, and it shares no header, table or helper with
 * the CUDA sources.  Every function follows a published definition step by
 * step, with no blocking, midstate reuse or fusion:
 *
 *   SHA-256 ............ FIPS 180-4, sections 4.1.2, 4.2.2, 5.1.1, 5.2.1,
 *                        5.3.3 and 6.2.2.  The round constants and initial
 *                        hash value are derived here from their definition
 *                        (first 32 fractional bits of cube / square roots of
 *                        the first primes) with exact integer roots, not typed.
 *   HMAC-SHA-256 ....... RFC 2104, section 2 (block size 64 bytes).
 *   salt derivation .... paper section 4.1, equation for sigma_p.
 *   chained block hash . paper section 2.1 equation (unsalted chain),
 *                        section 4.1 equation (salt at the root),
 *                        section 4.2 equation (salt at the divergence block).
 *   prefix lookup ...... paper section 2.1 (longest common prefix from
 *                        position 0 truncated to a block boundary), Table 1
 *                        row 1 (the oracle returns the first k matched
 *                        blocks) and section 5.7 (a divergence at token i
 *                        invalidates blocks floor(i/B) onward).
 *   arrival-order ...... the same lookup applied request by request, each
 *   serving              request then caching its blocks (sections 2.1 and
 *                        4.2): a sequential replay over a chained hash set.
 *   divergence ......... section 4.2 / 5.7: a request's boundary token is its
 *   boundary             longest common prefix with its registered preamble.
 *   exact-response key . Table 1 / section 4.1: SHA-256(sigma_p || prompt).
 *   ORIGAMI ............ section 4.3, Theorem: the water-filling audit
 *                        allocation, from its closed form over the sorted
 *                        values (fp64).
 *
 * Byte conventions (readings where the paper is silent): a token is its
 * int32 value serialised as 4 little-endian bytes; a block is B = 16 tokens
 * = 64 bytes; "h, tokens" and "sigma || h, tokens" are byte concatenations in
 * the order written; a digest is the 32-byte SHA-256 output.  Only full
 * blocks are hashed: a request of len tokens has floor(len/16) blocks.
 *
 * The cache index is modelled as a mathematical set of 32-byte keys, kept as
 * a sorted array searched with bsearch; it has nothing in common with the
 * GPU's open-addressing table except the keys it holds.  Every 32-byte key
 * but one can be a member: the all-zero key is refused, as the library's
 * boundary refuses it (it is the value of an empty slot).  A SHA-256 digest
 * equals it with probability 2^-256.
 *
 * Parity pins (tests/test_oracle_pins.py): SHA-256 against Python hashlib on
 * every message length 0..300 and random messages; HMAC against Python hmac;
 * each chain equation against hashlib compositions; the paper's worked
 * examples of section 4.2 and section 5.7; brute force on tiny inputs; the
 * arrival-order replay against a Python-set replay and closed forms
 * (repeated requests, multi-turn prefix extensions, per-principal salts).
 */
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <math.h>
#include <string.h>

/* --------------------------------------------------------------------- */
/* FIPS 180-4 section 4.2.2 / 5.3.3: constants derived from their definition */
/* --------------------------------------------------------------------- */

static uint32_t K256[64];
static uint32_t IV256[8];

/* Largest x with x*x*x <= n (exact, by bisection). */
static uint64_t icbrt_u128(unsigned __int128 n)
{
    uint64_t lo = 0, hi = (uint64_t)1 << 42;
    while (lo < hi) {
        uint64_t mid = lo + (hi - lo + 1) / 2;
        unsigned __int128 c = (unsigned __int128)mid * mid * mid;
        if (c <= n) lo = mid; else hi = mid - 1;
    }
    return lo;
}

/* Largest x with x*x <= n (exact, by bisection). */
static uint64_t isqrt_u128(unsigned __int128 n)
{
    uint64_t lo = 0, hi = (uint64_t)1 << 40;
    while (lo < hi) {
        uint64_t mid = lo + (hi - lo + 1) / 2;
        unsigned __int128 s = (unsigned __int128)mid * mid;
        if (s <= n) lo = mid; else hi = mid - 1;
    }
    return lo;
}

static int is_prime(uint32_t p)
{
    if (p < 2) return 0;
    for (uint32_t d = 2; d * d <= p; d++)
        if (p % d == 0) return 0;
    return 1;
}

/* K_t = first 32 bits of the fractional part of cbrt(p_t), p_t the t-th prime:
 * floor(cbrt(p) * 2^32) mod 2^32 = floor(cbrt(p * 2^96)) mod 2^32.
 * H(0)_i = first 32 bits of the fractional part of sqrt(p_i), i < 8:
 * floor(sqrt(p * 2^64)) mod 2^32. */
__attribute__((constructor)) static void derive_constants(void)
{
    uint32_t p = 2;
    for (int t = 0; t < 64; p++) {
        if (!is_prime(p)) continue;
        unsigned __int128 n = (unsigned __int128)p << 96;
        K256[t] = (uint32_t)(icbrt_u128(n) & 0xffffffffu);
        if (t < 8) {
            unsigned __int128 m = (unsigned __int128)p << 64;
            IV256[t] = (uint32_t)(isqrt_u128(m) & 0xffffffffu);
        }
        t++;
    }
}

void oracle_sha256_constants(uint32_t k_out[64], uint32_t iv_out[8])
{
    memcpy(k_out, K256, sizeof(K256));
    memcpy(iv_out, IV256, sizeof(IV256));
}

/* --------------------------------------------------------------------- */
/* FIPS 180-4 section 4.1.2: the six logical functions                    */
/* --------------------------------------------------------------------- */

static uint32_t ROTR(uint32_t x, unsigned n) { return (x >> n) | (x << (32u - n)); }
static uint32_t SHR(uint32_t x, unsigned n) { return x >> n; }
static uint32_t Ch(uint32_t x, uint32_t y, uint32_t z) { return (x & y) ^ (~x & z); }
static uint32_t Maj(uint32_t x, uint32_t y, uint32_t z) { return (x & y) ^ (x & z) ^ (y & z); }
static uint32_t BSIG0(uint32_t x) { return ROTR(x, 2) ^ ROTR(x, 13) ^ ROTR(x, 22); }
static uint32_t BSIG1(uint32_t x) { return ROTR(x, 6) ^ ROTR(x, 11) ^ ROTR(x, 25); }
static uint32_t SSIG0(uint32_t x) { return ROTR(x, 7) ^ ROTR(x, 18) ^ SHR(x, 3); }
static uint32_t SSIG1(uint32_t x) { return ROTR(x, 17) ^ ROTR(x, 19) ^ SHR(x, 10); }

/* FIPS 180-4 section 6.2.2: process one 512-bit block M (64 bytes) into H. */
static void sha256_process_block(uint32_t H[8], const uint8_t M[64])
{
    uint32_t W[64];
    /* step 1: message schedule; words are big-endian (section 3.1 / 5.2.1) */
    for (int t = 0; t < 16; t++)
        W[t] = ((uint32_t)M[4 * t] << 24) | ((uint32_t)M[4 * t + 1] << 16) |
               ((uint32_t)M[4 * t + 2] << 8) | (uint32_t)M[4 * t + 3];
    for (int t = 16; t < 64; t++)
        W[t] = SSIG1(W[t - 2]) + W[t - 7] + SSIG0(W[t - 15]) + W[t - 16];
    /* step 2: initialise the working variables */
    uint32_t a = H[0], b = H[1], c = H[2], d = H[3];
    uint32_t e = H[4], f = H[5], g = H[6], h = H[7];
    /* step 3: 64 rounds */
    for (int t = 0; t < 64; t++) {
        uint32_t T1 = h + BSIG1(e) + Ch(e, f, g) + K256[t] + W[t];
        uint32_t T2 = BSIG0(a) + Maj(a, b, c);
        h = g; g = f; f = e; e = d + T1;
        d = c; c = b; b = a; a = T1 + T2;
    }
    /* step 4: intermediate hash value */
    H[0] += a; H[1] += b; H[2] += c; H[3] += d;
    H[4] += e; H[5] += f; H[6] += g; H[7] += h;
}

/* SHA-256 of an arbitrary byte string.  Section 5.1.1 padding is built
 * explicitly: the message, one 0x80 byte, zeros, then the 64-bit big-endian
 * bit length, for a total that is a multiple of 64 bytes. */
void oracle_sha256(const uint8_t *msg, size_t len, uint8_t out[32])
{
    size_t padded = ((len + 1 + 8 + 63) / 64) * 64;
    uint8_t small[512];
    uint8_t *buf = padded <= sizeof(small) ? small : (uint8_t *)malloc(padded);
    if (len) memcpy(buf, msg, len);
    buf[len] = 0x80;
    memset(buf + len + 1, 0, padded - len - 1);
    uint64_t bits = (uint64_t)len * 8u;
    for (int i = 0; i < 8; i++)
        buf[padded - 1 - i] = (uint8_t)(bits >> (8 * i));

    uint32_t H[8];
    memcpy(H, IV256, sizeof(H));
    for (size_t off = 0; off < padded; off += 64)
        sha256_process_block(H, buf + off);
    for (int i = 0; i < 8; i++) {
        out[4 * i] = (uint8_t)(H[i] >> 24);
        out[4 * i + 1] = (uint8_t)(H[i] >> 16);
        out[4 * i + 2] = (uint8_t)(H[i] >> 8);
        out[4 * i + 3] = (uint8_t)H[i];
    }
    if (buf != small) free(buf);
}

/* --------------------------------------------------------------------- */
/* RFC 2104 section 2: HMAC with H = SHA-256, B = 64, L = 32               */
/* --------------------------------------------------------------------- */

void oracle_hmac_sha256(const uint8_t *key, size_t key_len,
                        const uint8_t *msg, size_t msg_len, uint8_t out[32])
{
    uint8_t K0[64];
    memset(K0, 0, sizeof(K0));
    if (key_len > 64) oracle_sha256(key, key_len, K0);     /* keys longer than B are hashed */
    else if (key_len) memcpy(K0, key, key_len);           /* then zero-padded to B bytes */

    /* inner = H((K0 xor ipad) || text) */
    uint8_t *inner_msg = (uint8_t *)malloc(64 + msg_len);
    for (int i = 0; i < 64; i++) inner_msg[i] = K0[i] ^ 0x36;
    if (msg_len) memcpy(inner_msg + 64, msg, msg_len);
    uint8_t inner[32];
    oracle_sha256(inner_msg, 64 + msg_len, inner);
    free(inner_msg);

    /* out = H((K0 xor opad) || inner) */
    uint8_t outer_msg[64 + 32];
    for (int i = 0; i < 64; i++) outer_msg[i] = K0[i] ^ 0x5c;
    memcpy(outer_msg + 64, inner, 32);
    oracle_sha256(outer_msg, sizeof(outer_msg), out);
}

/* --------------------------------------------------------------------- */
/* Paper section 4.1: sigma_p = HMAC_K(secret, principal_id)             */
/* --------------------------------------------------------------------- */

/* ids: concatenated principal-id byte strings; id_off[n+1] their offsets.
 * Returns 0, or -1 on a malformed offset array. */
int oracle_derive_salts(const uint8_t *secret, size_t secret_len,
                        const uint8_t *ids, const int64_t *id_off,
                        int32_t n_principals, uint8_t *salts)
{
    for (int32_t p = 0; p < n_principals; p++) {
        int64_t a = id_off[p], b = id_off[p + 1];
        if (a < 0 || b < a) return -1;
        oracle_hmac_sha256(secret, secret_len, ids + a, (size_t)(b - a), salts + 32 * (size_t)p);
    }
    return 0;
}

/* --------------------------------------------------------------------- */
/* Paper section 2.1: blocking, B = 16                                    */
/* --------------------------------------------------------------------- */

#define ORACLE_B 16

/* blk_off[r] = sum over requests q < r of floor(len_q / B). */
int oracle_block_offsets(const int64_t *tok_off, int32_t n_req, int64_t *blk_off)
{
    blk_off[0] = 0;
    for (int32_t r = 0; r < n_req; r++) {
        int64_t len = tok_off[r + 1] - tok_off[r];
        if (len < 0) return -1;
        blk_off[r + 1] = blk_off[r] + len / ORACLE_B;
    }
    return 0;
}

/* Serialise tokens[0..15] of one block as 64 little-endian bytes. */
static void block_bytes(const int32_t *tok, uint8_t out[64])
{
    for (int i = 0; i < ORACLE_B; i++) {
        uint32_t v = (uint32_t)tok[i];
        out[4 * i] = (uint8_t)v;
        out[4 * i + 1] = (uint8_t)(v >> 8);
        out[4 * i + 2] = (uint8_t)(v >> 16);
        out[4 * i + 3] = (uint8_t)(v >> 24);
    }
}

#define ORACLE_UNSALTED 0
#define ORACLE_ROOT 1
#define ORACLE_BOUNDARY 2

/*
 * Chained block digests of every request, written in request order: request
 * r's block j goes to digests[(blk_off[r] + j) * 32], blk_off as above.
 *
 *   UNSALTED (section 2.1):  h_0 = H(T_0),          h_j = H(h_{j-1} || T_j)
 *   ROOT     (section 4.1):  h_0 = H(sigma || T_0), h_j = H(h_{j-1} || T_j)
 *   BOUNDARY (section 4.2), k = floor(b / B) for the request's boundary token
 *   offset b:  j < k: the UNSALTED rule;  j = k: H(sigma || h_{k-1} || T_k)
 *   (k = 0 has no h_{-1}: H(sigma || T_0));  j > k: H(h_{j-1} || T_j).
 *   A boundary at or past the last full block leaves the chain unsalted.
 *
 * principal[r] selects row principal[r] of salts (ignored for UNSALTED);
 * boundary_tok[r] is used only for BOUNDARY.  Returns 0, or -1 on a bad
 * mode, principal index, boundary offset or token offset.
 */
int oracle_chain_hash(int mode, const int32_t *tokens, const int64_t *tok_off,
                      int32_t n_req, const int32_t *principal,
                      const uint8_t *salts, int32_t n_principals,
                      const int32_t *boundary_tok, uint8_t *digests)
{
    if (mode != ORACLE_UNSALTED && mode != ORACLE_ROOT && mode != ORACLE_BOUNDARY) return -1;
    int64_t out_blk = 0;
    for (int32_t r = 0; r < n_req; r++) {
        int64_t len = tok_off[r + 1] - tok_off[r];
        if (len < 0) return -1;
        int64_t nb = len / ORACLE_B;
        const int32_t *t = tokens + tok_off[r];
        const uint8_t *sigma = NULL;
        if (mode != ORACLE_UNSALTED) {
            if (principal[r] < 0 || principal[r] >= n_principals) return -1;
            sigma = salts + 32 * (size_t)principal[r];
        }
        int64_t k = -1;                         /* -1: no salted block */
        if (mode == ORACLE_ROOT) k = 0;
        if (mode == ORACLE_BOUNDARY) {
            if (boundary_tok[r] < 0) return -1;
            k = boundary_tok[r] / ORACLE_B;
        }

        uint8_t prev[32];
        for (int64_t j = 0; j < nb; j++) {
            uint8_t msg[32 + 32 + 64];
            size_t m = 0;
            if (j == k) {                       /* the salted block */
                memcpy(msg + m, sigma, 32); m += 32;
                if (j > 0) { memcpy(msg + m, prev, 32); m += 32; }
            } else if (j > 0) {                 /* ordinary chained block */
                memcpy(msg + m, prev, 32); m += 32;
            }
            block_bytes(t + ORACLE_B * j, msg + m); m += 64;
            uint8_t *hj = digests + 32 * (size_t)(out_blk + j);
            oracle_sha256(msg, m, hj);
            memcpy(prev, hj, 32);
        }
        out_blk += nb;
    }
    return 0;
}

/* --------------------------------------------------------------------- */
/* The cache index as a set; paper section 2.1 / Table 1 row 1 lookup     */
/* --------------------------------------------------------------------- */

#define ORACLE_FLAG_ZERO_KEY 1u

static int key_cmp(const void *a, const void *b) { return memcmp(a, b, 32); }

/* The one key the set refuses (see header): all 32 bytes zero. */
int oracle_key_is_zero(const uint8_t *key)
{
    for (int i = 0; i < 32; i++)
        if (key[i] != 0) return 0;
    return 1;
}

int oracle_set_contains(const uint8_t *set_keys, int64_t n_set, const uint8_t *key)
{
    return n_set > 0 && bsearch(key, set_keys, (size_t)n_set, 32, key_cmp) != NULL;
}

/*
 * Add keys to the set held sorted and duplicate-free in set_keys[0..*n_set)
 * (room for set_cap keys): append every key but the all-zero one, sort,
 * drop repeats.  Duplicates, within the batch or with the set, are therefore
 * no-ops, and the result does not depend on the order of keys.  *n_new
 * receives how many keys the set gained.  Returns ORACLE_FLAG_ZERO_KEY if an
 * all-zero key was given (it is skipped), 0 otherwise, or -1 if set_cap is
 * too small for the appended keys.
 */
int64_t oracle_set_insert(uint8_t *set_keys, int64_t *n_set, int64_t set_cap,
                          const uint8_t *keys, int64_t n_keys, int64_t *n_new)
{
    int64_t flags = 0, n = *n_set;
    for (int64_t i = 0; i < n_keys; i++) {
        const uint8_t *key = keys + 32 * (size_t)i;
        if (oracle_key_is_zero(key)) { flags |= ORACLE_FLAG_ZERO_KEY; continue; }
        if (n >= set_cap) return -1;
        memcpy(set_keys + 32 * (size_t)n, key, 32);
        n++;
    }
    qsort(set_keys, (size_t)n, 32, key_cmp);
    int64_t u = 0;
    for (int64_t i = 0; i < n; i++) {
        if (u > 0 && memcmp(set_keys + 32 * (size_t)(u - 1), set_keys + 32 * (size_t)i, 32) == 0)
            continue;
        if (u != i) memcpy(set_keys + 32 * (size_t)u, set_keys + 32 * (size_t)i, 32);
        u++;
    }
    *n_new = u - *n_set;
    *n_set = u;
    return flags;
}

/*
 * prefix_blocks[r] = the number of leading blocks of request r whose digests
 * are all in the set: the smallest j with h_j not in the set, or n_b(r) if
 * every block is present.  A later hit after a miss does not count.
 */
int oracle_prefix_blocks(const uint8_t *set_keys, int64_t n_set,
                         const uint8_t *digests, const int64_t *blk_off,
                         int32_t n_req, int32_t *prefix_blocks)
{
    for (int32_t r = 0; r < n_req; r++) {
        int64_t nb = blk_off[r + 1] - blk_off[r];
        if (nb < 0) return -1;
        int64_t j = 0;
        while (j < nb && oracle_set_contains(set_keys, n_set, digests + 32 * (size_t)(blk_off[r] + j)))
            j++;
        prefix_blocks[r] = (int32_t)j;
    }
    return 0;
}

/* --------------------------------------------------------------------- */
/*
 * Arrival-order serving of one batch (paper section 2.1: a lookup matches
 * the longest cached prefix of blocks from position 0; section 4.2: the
 * uncached blocks are prefilled, after which they are cached), written as its
 * definition: the requests are taken one at a time, in order.  Request r's
 * prefix length is its number of leading blocks present in the set as it
 * stands -- the keys given (cached before the batch) plus every block of
 * requests 0..r-1 -- and then all of r's blocks join the set (the all-zero
 * key excepted).
 *
 * The set is a chained hash set: bucket heads indexed by bytes 8..15 of the
 * key, a node array with next links, keys compared whole.
 */
typedef struct {
    int64_t *head;            /* [n_buckets] first node or -1 */
    int64_t *next;            /* [cap] next node or -1 */
    const uint8_t **key;      /* [cap] the node's key (points into the inputs) */
    int64_t n, cap;
    uint64_t mask;
} chain_set;

static uint64_t chain_set_bucket(const chain_set *s, const uint8_t *k)
{
    uint64_t h = 0;
    for (int i = 15; i >= 8; i--) h = (h << 8) | k[i];
    return h & s->mask;
}

static int chain_set_contains(const chain_set *s, const uint8_t *k)
{
    for (int64_t i = s->head[chain_set_bucket(s, k)]; i >= 0; i = s->next[i])
        if (memcmp(s->key[i], k, 32) == 0) return 1;
    return 0;
}

/* Adds k if absent; returns 1 if it was added. */
static int chain_set_add(chain_set *s, const uint8_t *k)
{
    if (chain_set_contains(s, k)) return 0;
    const uint64_t b = chain_set_bucket(s, k);
    s->key[s->n] = k;
    s->next[s->n] = s->head[b];
    s->head[b] = s->n;
    s->n++;
    return 1;
}

/*
 * set_keys[0..n_set): the keys cached before the batch.  digests, blk_off,
 * n_req: the batch (request-major digests, block offsets).  prefix_blocks
 * [n_req] receives the prefix lengths, *n_new how many keys the batch added
 * to the set.  The all-zero key is never added, as in oracle_set_insert.  Returns 0, or -1 for malformed offsets or no memory.
 */
int oracle_arrival_prefix(const uint8_t *set_keys, int64_t n_set, const uint8_t *digests,
                          const int64_t *blk_off, int32_t n_req, int32_t *prefix_blocks,
                          int64_t *n_new)
{
    if (n_set < 0 || n_req < 0 || blk_off[0] != 0) return -1;
    for (int32_t r = 0; r < n_req; r++)
        if (blk_off[r + 1] < blk_off[r]) return -1;
    const int64_t cap = n_set + blk_off[n_req] + 1;
    uint64_t n_buckets = 1;
    while (n_buckets < (uint64_t)(2 * cap)) n_buckets <<= 1;
    chain_set s;
    s.head = malloc(n_buckets * sizeof(int64_t));
    s.next = malloc((size_t)cap * sizeof(int64_t));
    s.key = malloc((size_t)cap * sizeof(const uint8_t *));
    s.n = 0;
    s.cap = cap;
    s.mask = n_buckets - 1;
    if (!s.head || !s.next || !s.key) {
        free(s.head); free(s.next); free(s.key);
        return -1;
    }
    for (uint64_t b = 0; b < n_buckets; b++) s.head[b] = -1;
    for (int64_t i = 0; i < n_set; i++) chain_set_add(&s, set_keys + 32 * (size_t)i);
    const int64_t before = s.n;
    for (int32_t r = 0; r < n_req; r++) {
        const uint8_t *req = digests + 32 * (size_t)blk_off[r];
        const int64_t nb = blk_off[r + 1] - blk_off[r];
        int64_t j = 0;
        while (j < nb && chain_set_contains(&s, req + 32 * (size_t)j))
            j++;
        prefix_blocks[r] = (int32_t)j;
        for (int64_t q = 0; q < nb; q++)
            if (!oracle_key_is_zero(req + 32 * (size_t)q)) chain_set_add(&s, req + 32 * (size_t)q);
    }
    *n_new = s.n - before;
    free(s.head); free(s.next); free(s.key);
    return 0;
}

/* --------------------------------------------------------------------- */
/*
 * Divergence boundary (paper section 4.2: the salt goes in at the block
 * where a request diverges from the shared preamble; section 5.7: a
 * divergence at token i invalidates blocks floor(i/B) onward).  For request
 * r, boundary_tok[r] is the number of leading tokens it has in common with
 * its registered preamble: compare token by token from position 0 and stop
 * at the first difference or at the end of the shorter sequence.
 * template_id[r] names the preamble (an index below n_tpl), -1 (none:
 * boundary 0) or -2 (the longest such prefix over all preambles).  An id out
 * of range gives boundary 0.  Returns 1 if some id or offset was out of
 * range, else 0.
 */
int oracle_divergence_boundary(const int32_t *tokens, const int64_t *tok_off, int32_t n_req,
                               const int32_t *template_id, const int32_t *tpl_tokens,
                               const int64_t *tpl_off, int32_t n_tpl, int32_t *boundary_tok)
{
    int flag = 0;
    for (int32_t r = 0; r < n_req; r++) {
        const int32_t id = template_id[r];
        const int64_t len_r = tok_off[r + 1] - tok_off[r];
        boundary_tok[r] = 0;
        if (id < -2 || id >= n_tpl || len_r < 0) { flag = 1; continue; }
        if (id == -1) continue;
        int64_t best = 0;
        for (int32_t t = 0; t < n_tpl; t++) {
            if (id >= 0 && t != id) continue;
            const int64_t len_t = tpl_off[t + 1] - tpl_off[t];
            int64_t i = 0;
            while (i < len_r && i < len_t && tokens[tok_off[r] + i] == tpl_tokens[tpl_off[t] + i])
                i++;
            if (i > best) best = i;
        }
        boundary_tok[r] = (int32_t)best;
    }
    return flag;
}

/* --------------------------------------------------------------------- */
/*
 * Exact-response cache key (paper Table 1: the key is the whole prompt;
 * section 4.1: sigma_p is prepended to it): SHA-256 over the byte string
 * sigma_p || LE32(t_0) || LE32(t_1) || ... with every token of the request,
 * or over the token bytes alone in mode UNSALTED.  The message is built in
 * full and hashed with oracle_sha256.  Returns -1 for a bad mode, range or
 * principal, or no memory; 0 otherwise.
 */
int oracle_response_key(int mode, const int32_t *tokens, const int64_t *tok_off, int32_t n_req,
                        const int32_t *principal, const uint8_t *salts, int32_t n_principals,
                        uint8_t *keys)
{
    if (mode != ORACLE_UNSALTED && mode != ORACLE_ROOT) return -1;
    for (int32_t r = 0; r < n_req; r++) {
        const int64_t len = tok_off[r + 1] - tok_off[r];
        if (len < 0) return -1;
        const size_t salt_len = mode == ORACLE_ROOT ? 32 : 0;
        uint8_t *msg = malloc(salt_len + 4 * (size_t)len + 1);
        if (!msg) return -1;
        if (mode == ORACLE_ROOT) {
            if (principal[r] < 0 || principal[r] >= n_principals) { free(msg); return -1; }
            memcpy(msg, salts + 32 * (size_t)principal[r], 32);
        }
        for (int64_t i = 0; i < len; i++) {
            const uint32_t v = (uint32_t)tokens[tok_off[r] + i];
            msg[salt_len + 4 * i] = (uint8_t)v;
            msg[salt_len + 4 * i + 1] = (uint8_t)(v >> 8);
            msg[salt_len + 4 * i + 2] = (uint8_t)(v >> 16);
            msg[salt_len + 4 * i + 3] = (uint8_t)(v >> 24);
        }
        oracle_sha256(msg, salt_len + 4 * (size_t)len, keys + 32 * (size_t)r);
        free(msg);
    }
    return 0;
}

/* --------------------------------------------------------------------- */
/*
 * ORIGAMI audit allocation (paper section 4.3, Theorem): minimise
 * max_i v_i (1 - p_i) subject to sum_i p_i = K and p_i in [0, 1]; the
 * optimum is p_i = max(0, 1 - lambda / v_i) with the water level lambda that
 * meets the budget.  Written out from that statement, in fp64: take the
 * tenants with positive value in decreasing order of value; if the top m of
 * them are the audited ones, sum_{i <= m} (1 - lambda / v_(i)) = K gives
 * lambda_m = (m - K) / sum_{i <= m} 1 / v_(i); the water level is the
 * lambda_m that lies in [v_(m+1), v_(m)) (v_(n+1) = 0), i.e. exactly the top
 * m tenants are above it.  K is capped at the number of positive values
 * (all audited, lambda = 0); K = 0 gives lambda = the largest value.  Values
 * <= 0 get p = 0.  utility[q] = max_i v_i (1 - p_i).  Returns 1 if some
 * value was not a finite number or some budget was negative (read as 0),
 * -1 for no memory, 0 otherwise.
 */
static int cmp_desc(const void *a, const void *b)
{
    const double x = *(const double *)a, y = *(const double *)b;
    return (x < y) - (x > y);
}

int oracle_origami(const float *values, const int64_t *off, int32_t n_prob, const float *budget,
                   double *p, double *lambda, double *utility)
{
    int flag = 0;
    for (int32_t q = 0; q < n_prob; q++) {
        const int64_t b0 = off[q], n = off[q + 1] - off[q];
        double *pos = malloc((size_t)(n > 0 ? n : 1) * sizeof(double));
        if (!pos) return -1;
        int64_t npos = 0;
        for (int64_t i = 0; i < n; i++) {
            const double x = values[b0 + i];
            if (x > 0.0 && x <= 3.0e38) pos[npos++] = x;
            else if (!(x <= 0.0)) flag = 1;
        }
        qsort(pos, (size_t)npos, sizeof(double), cmp_desc);
        double K = budget[q];
        if (!(K >= 0.0)) { flag = 1; K = 0.0; }
        if (K > (double)npos) K = (double)npos;
        double lam;
        if (npos == 0 || K <= 0.0) {
            lam = npos > 0 ? pos[0] : 0.0;
        } else if (K >= (double)npos) {
            lam = 0.0;
        } else {
            double inv_sum = 0.0;
            lam = 0.0;
            for (int64_t m = 1; m <= npos; m++) {
                inv_sum += 1.0 / pos[m - 1];
                const double lm = ((double)m - K) / inv_sum;
                const double below = m < npos ? pos[m] : 0.0;
                if (lm >= below && lm < pos[m - 1]) { lam = lm; break; }
            }
        }
        double u = -HUGE_VAL;
        for (int64_t i = 0; i < n; i++) {
            const double x = values[b0 + i];
            const double pi = (x > 0.0 && x <= 3.0e38) ? (1.0 - lam / x > 0.0 ? 1.0 - lam / x : 0.0) : 0.0;
            p[b0 + i] = pi;
            if (x == x && x * (1.0 - pi) > u) u = x * (1.0 - pi);
        }
        lambda[q] = lam;
        utility[q] = n > 0 ? u : 0.0;
        free(pos);
    }
    return flag;
}
