/*
 * kvgov.h -- C ABI of libkvgov: the salted block-hash chain and block
 * prefix-cache probe of KVGov (arxiv 2608.09225), on one GB300 (sm_103a).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Pointers named d_* are DEVICE pointers owned by the caller.  Nothing
 *    here allocates device or host memory, synchronises, or keeps a pointer
 *    after returning.  Every call only enqueues kernels on `stream` (a
 *    cudaStream_t; NULL is the legacy default stream) and returns.
 *  - Return value: KVGOV_OK, or a host-detected error (KVGOV_EINVAL for a bad
 *    argument, KVGOV_ECUDA when a launch fails).  On a host-detected error
 *    nothing is enqueued.
 *  - Errors that only the device can see (a bad per-request index, the
 *    all-zero key, a full table, a wait that ran out) are OR-ed as
 *    KVGOV_F_* bits into the u32 at d_status.  The caller zeroes it before
 *    the call and reads it after synchronising.  Where d_status may be NULL
 *    the flags are dropped.
 *  - A token is an int32; the hashed bytes of a token are its 4 bytes in
 *    little-endian order.  A block is KVGOV_BLOCK = 16 consecutive tokens of
 *    one request; only full blocks are hashed (a request of len tokens has
 *    n_b = floor(len / 16) blocks; the tail is not hashed).  A digest is the
 *    32-byte SHA-256 output.
 *  - Requests are given in CSR form: request r is tokens
 *    d_tokens[d_tok_off[r] .. d_tok_off[r+1]), d_tok_off non-decreasing,
 *    int64.  Block-level outputs are request-major: block j of request r is
 *    row d_blk_off[r] + j, with d_blk_off the exclusive prefix sum of n_b
 *    (see kvgov_block_offsets).
 */
#ifndef KVGOV_H
#define KVGOV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t / CUstream. */
typedef struct CUstream_st *kvgov_stream_t;

#define KVGOV_BLOCK 16             /* tokens per block, B in the paper        */
#define KVGOV_DIGEST_BYTES 32      /* SHA-256 digest and table key size       */
#define KVGOV_MAX_SECRET 1024      /* longest HMAC key kvgov_derive_salts takes */
#define KVGOV_MIN_CAPACITY 32      /* smallest table capacity (slots)         */
#define KVGOV_PROBE_WINDOW 1024    /* a key lives within this many slots of its
                                      home slot (fewer if the table is smaller) */
#define KVGOV_STASH_SLOTS 64       /* slots after the `capacity` main ones: the
                                      table's side store (see the table section) */
#define KVGOV_STASH_KEYS 56        /* keys the side store holds               */
#define KVGOV_TEMPLATE_NONE (-1)   /* kvgov_divergence_boundary: no preamble   */
#define KVGOV_TEMPLATE_ANY (-2)    /* ... the longest match over all preambles */

/* Return codes (host-detected). */
#define KVGOV_OK 0
#define KVGOV_EINVAL 1             /* bad argument; nothing was enqueued      */
#define KVGOV_ECUDA 2              /* a kernel launch failed                  */

/* Device-detected flags, OR-ed into *d_status. */
#define KVGOV_F_BADINDEX 0x10u     /* a principal index, boundary offset or
                                      offset array entry was out of range; the
                                      affected request produced no output     */
#define KVGOV_F_SENTINEL 0x20u     /* the all-zero key (the value of an empty
                                      slot) was given to an insert; it is
                                      skipped                                  */
#define KVGOV_F_TABLE_FULL 0x40u   /* an insert found no free slot in a key's
                                      probe window, or the side store was
                                      full; the key is not stored             */
#define KVGOV_F_TIMEOUT 0x80u      /* an insert gave up waiting for another
                                      thread to finish writing a slot's key,
                                      or a bulk copy of kvgov_origami did not
                                      complete within its bounded wait        */

/* Salt placement (paper section 2.1 equation, section 4.1, section 4.2). */
#define KVGOV_UNSALTED 0           /* h_0 = H(T_0), h_j = H(h_{j-1} || T_j)   */
#define KVGOV_ROOT 1               /* h_0 = H(sigma_p || T_0), then chained   */
#define KVGOV_BOUNDARY 2           /* salt injected at block k = floor(b/16)  */

/*
 * kvgov_status_string -- a static, human-readable name for a return code or
 * for a single KVGOV_F_* flag.  Never NULL.
 */
const char *kvgov_status_string(int status);

/*
 * kvgov_block_offsets -- blocking, paper section 2.1 (keys are per B-token
 * block; only full blocks are keyed).
 *
 *   d_tok_off [n_req + 1] int64, non-decreasing token offsets (CSR).
 *   d_blk_off [n_req + 1] int64 output: d_blk_off[0] = 0 and
 *             d_blk_off[r+1] = d_blk_off[r] + floor(len_r / 16).
 *   d_status  nullable; KVGOV_F_BADINDEX if some len_r < 0 (that request
 *             then counts 0 blocks).
 * n_req = 0 writes d_blk_off[0] = 0.  EINVAL: n_req < 0 or a NULL array.
 * Two ordinary (non-cooperative) launches on `stream`, so the scan may run
 * beside other kernels; between them d_blk_off holds per-chunk partial
 * totals (it is its own scratch space), so nothing may read d_blk_off until
 * the call's work on `stream` has completed.
 */
int kvgov_block_offsets(const int64_t *d_tok_off, int32_t n_req, int64_t *d_blk_off,
                        uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_count_blocks -- the blocking of kvgov_block_offsets computed on the
 * host, for sizing buffers before any launch: *n_blocks = the sum over
 * requests of floor(len_r / 16) (paper section 2.1), a negative len_r
 * counting 0, so it equals the d_blk_off[n_req] that kvgov_block_offsets
 * writes for the same offsets.
 *   h_tok_off [n_req + 1] int64 HOST token offsets (CSR).
 *   h_blk_off [n_req + 1] int64 HOST output, nullable: the same exclusive
 *             prefix sum kvgov_block_offsets writes.
 *   n_blocks  HOST output, required.
 * Runs on the calling thread; touches no device.  EINVAL: n_req < 0, a NULL
 * h_tok_off or n_blocks.
 */
int kvgov_count_blocks(const int64_t *h_tok_off, int32_t n_req, int64_t *h_blk_off, int64_t *n_blocks);

/*
 * kvgov_divergence_boundary -- where each request's salt goes in, paper
 * section 4.2 (salt at the divergence boundary k: the blocks before it hold
 * the shared preamble, which tells no principal apart) and section 5.7 (a
 * divergence at token i invalidates every block from floor(i/B) on).
 * d_boundary_tok[r] = the length of the longest common prefix of request r's
 * tokens and its registered preamble: the index of the first token where
 * they differ, or the shorter length if one is a prefix of the other.  It is
 * the d_boundary_tok input of kvgov_chain_hash in BOUNDARY mode (k = b / 16).
 *   d_tokens, d_tok_off, n_req  the batch (CSR int32 tokens, int64 offsets).
 *   d_template_id  [n_req] int32: the preamble of request r, an index into
 *               the registered preambles, KVGOV_TEMPLATE_NONE (b = 0: salt at
 *               the root) or KVGOV_TEMPLATE_ANY (the longest match over all
 *               preambles).
 *   d_tpl_tokens, d_tpl_off, n_tpl  the registered preambles (CSR int32
 *               tokens, int64 offsets [n_tpl + 1]); may be NULL if n_tpl = 0.
 *   d_boundary_tok [n_req] int32 output.
 *   d_status    nullable; KVGOV_F_BADINDEX for an id outside
 *               [KVGOV_TEMPLATE_ANY, n_tpl) or malformed offsets (that
 *               request gets b = 0).
 * One warp per request.  n_req = 0 is a no-op.  EINVAL: negative counts,
 * NULL arrays.
 */
int kvgov_divergence_boundary(const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                              const int32_t *d_template_id, const int32_t *d_tpl_tokens,
                              const int64_t *d_tpl_off, int32_t n_tpl, int32_t *d_boundary_tok,
                              uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_response_key -- exact-response cache keys, paper Table 1 (an
 * exact-response cache keys on byte equality of the whole prompt) and
 * section 4.1 (sigma_p is prepended to that key):
 *   ROOT      key_r = SHA-256(sigma_p || bytes(tokens of r))
 *   UNSALTED  key_r = SHA-256(bytes(tokens of r))
 * with every token of the request (no block truncation), tokens as int32
 * little-endian.  The keys go into the same table as block digests
 * (kvgov_insert; kvgov_probe with one "block" per request gives 1 for a
 * cached response, 0 otherwise).
 *   d_tokens, d_tok_off, n_req  the batch (CSR; tokens 16-byte aligned).
 *   d_principal, d_salts, n_principals  as for kvgov_chain_hash (ROOT only).
 *   d_keys     [n_req][32] u8 output (16-byte aligned).
 *   d_status   nullable; KVGOV_F_BADINDEX for a malformed range or principal
 *              (that request's key is undefined).
 * One thread per request.  n_req = 0 is a no-op.  EINVAL: mode BOUNDARY or
 * unknown, NULL or misaligned arrays, ROOT without salts.
 */
int kvgov_response_key(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                       const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals, uint8_t *d_keys,
                       uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_origami -- ORIGAMI audit allocation for a batch of problems, paper
 * section 4.3, Theorem (ORIGAMI water-filling solution): for each problem,
 * tenants with values at risk v_i and an audit budget K, the audit
 * probabilities minimising the adversary's best payoff max_i v_i (1 - p_i)
 * subject to sum p_i = K, p_i in [0, 1]:
 *     p_i = max(0, 1 - lambda / v_i),  lambda the unique level with sum = K.
 *   d_values   float32, the problems' tenant values back to back (CSR).
 *   d_off      [n_prob + 1] int64 offsets into d_values.
 *   d_budget   [n_prob] float32 K.  K is capped at the number of usable
 *              tenants (all audited, lambda = 0); K = 0 gives p = 0 and
 *              lambda = the largest value.
 *   d_p        float32 output beside d_values.
 *   d_lambda   [n_prob] float32 output (nullable): the water level.
 *   d_utility  [n_prob] float32 output (nullable): the adversary's best
 *              payoff max_i v_i (1 - p_i) under the allocation.
 *   d_status   nullable; KVGOV_F_BADINDEX for a NaN or infinite value, a
 *              negative or NaN budget (read as 0) or malformed offsets.
 * Tenants with v_i <= 0 get p_i = 0.  fp32 arithmetic.  A problem of at
 * most 64 tenants with every value positive and finite (and at most 2^126)
 * is solved by one thread in registers, any other by a warp.  With d_values
 * and d_p on 16-byte boundaries the values stream through shared memory by
 * bulk copies (a persistent grid, each warp on its own tiles of 32
 * problems); otherwise each CTA of 128 problems stages its values with
 * plain loads.  The results are the same either way.
 * n_prob = 0 is a no-op.  EINVAL: negative n_prob, NULL arrays.
 * KVGOV_F_TIMEOUT: a bulk copy did not complete within its bounded wait
 * (the results are then incomplete).
 */
int kvgov_origami(const float *d_values, const int64_t *d_off, int32_t n_prob, const float *d_budget, float *d_p,
                  float *d_lambda, float *d_utility, uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_derive_salts -- per-principal salt, paper section 4.1:
 * sigma_p = HMAC_K(secret, principal_id), HMAC per RFC 2104 with SHA-256.
 *
 *   secret, secret_len  HOST bytes of the server secret K, the HMAC key
 *                       (0 <= secret_len <= KVGOV_MAX_SECRET; keys longer
 *                       than 64 bytes are first hashed, as RFC 2104 says).
 *                       Copied into the launch; the host buffer may be
 *                       reused as soon as the call returns.
 *   d_ids, d_id_off     the principal ids as byte strings in CSR form:
 *                       principal p is d_ids[d_id_off[p] .. d_id_off[p+1]).
 *   d_salts             [n_principals][32] u8 output.
 *   d_status            nullable; KVGOV_F_BADINDEX for a negative or
 *                       decreasing id offset (that salt is left untouched).
 * n_principals = 0 is a no-op.  EINVAL: secret_len too large, secret NULL
 * with secret_len > 0, n_principals < 0, a NULL device array.
 */
int kvgov_derive_salts(const uint8_t *secret, size_t secret_len, const uint8_t *d_ids,
                       const int64_t *d_id_off, int32_t n_principals, uint8_t *d_salts,
                       uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_chain_hash -- the chained block digests of every request:
 *   UNSALTED (paper section 2.1):  h_0 = H(T_0), h_j = H(h_{j-1} || T_j);
 *   ROOT     (section 4.1):        h_0 = H(sigma_p || T_0), h_j as above;
 *   BOUNDARY (section 4.2): with k = floor(b_r / 16) for the request's
 *     boundary token offset b_r, blocks j < k follow UNSALTED, block k is
 *     H(sigma_p || h_{k-1} || T_k) (H(sigma_p || T_0) when k = 0), and
 *     blocks j > k are chained as usual.  k >= n_b leaves the chain unsalted.
 * H is SHA-256, T_j the 64 bytes of block j, || byte concatenation.
 *
 *   mode            KVGOV_UNSALTED, KVGOV_ROOT or KVGOV_BOUNDARY.
 *   d_tokens        int32 tokens; must be 16-byte aligned (blocks are staged
 *                   with aligned 16-byte copies; no byte outside
 *                   [d_tokens, d_tokens + d_tok_off[n_req]) is read).
 *   d_tok_off       [n_req + 1] int64 token offsets.
 *   d_principal     [n_req] int32 row of d_salts per request; unused (may be
 *                   NULL) for UNSALTED.
 *   d_salts         [n_principals][32] u8 salts (kvgov_derive_salts); unused
 *                   for UNSALTED.
 *   d_boundary_tok  [n_req] int32 boundary token offset b_r >= 0; used (and
 *                   required) only for BOUNDARY.
 *   d_blk_off       [n_req + 1] int64 from kvgov_block_offsets.
 *   d_digests       [d_blk_off[n_req]][32] u8 output, 16-byte aligned.
 *   d_status        nullable; KVGOV_F_BADINDEX for a principal outside
 *                   [0, n_principals), a negative b_r, or a malformed token
 *                   offset (that request's digests are not written).
 * n_req = 0 is a no-op (d_principal, d_salts and d_boundary_tok may then be
 * NULL).  EINVAL: bad mode, misaligned or NULL array.
 */
int kvgov_chain_hash(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                     const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                     const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                     uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_chain_hash_probe -- kvgov_chain_hash and kvgov_probe in one launch:
 * writes the same d_digests as kvgov_chain_hash and the same
 * d_prefix_blocks as kvgov_probe on the table (d_slots, capacity) would
 * (paper section 2.1: the block keys of a request and its longest cached
 * prefix).  Each thread looks up a block's digest as soon as it has computed
 * it, while other warps go on hashing; the table must not change during the
 * call (run inserts after it).  A batch too small to give each SM
 * sub-partition two warps (n_req < 2 * 32 * 4 * SMs) runs the lookups as a
 * second kernel after the chain instead, since a warp alone on its scheduler
 * would stall on each lookup; the results are the same.  Arguments as for those two calls;
 * d_prefix_blocks [n_req] int32 output, required.  EINVAL: as for
 * kvgov_chain_hash, plus a NULL or misaligned d_slots or a bad capacity.
 */
int kvgov_chain_hash_probe(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                           const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                           const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                           const uint8_t *d_slots, uint64_t capacity, int32_t *d_prefix_blocks,
                           uint32_t *d_status, kvgov_stream_t stream);

/*
 * The prefix-cache index (paper section 2.1 and Table 1, row 1: a block
 * prefix cache keyed by chained block hashes): the set of 32-byte keys of
 * cached blocks.  Every key but the all-zero one (KVGOV_F_SENTINEL) can be
 * stored.  The caller owns the table's memory: capacity + KVGOV_STASH_SLOTS
 * slots of 32 bytes (capacity a power of two >= KVGOV_MIN_CAPACITY, d_slots
 * 16-byte aligned), and passes `capacity`.
 *
 * Main slots 0 .. capacity-1: a slot is empty when its first 16 bytes are
 * zero; a key's home slot is its first 8 bytes read as a little-endian u64,
 * modulo capacity, with linear probing inside a window of
 * min(capacity, KVGOV_PROBE_WINDOW) slots: an insert that finds no free slot
 * in its window reports KVGOV_F_TABLE_FULL (at load factor 0.5 a walk longer
 * than a few dozen slots practically never happens), and lookups stop at the
 * end of the window.  Keys are stored verbatim, claimed with a 128-bit
 * compare-and-swap of their first 16 bytes, the second half written after.
 *
 * Side store, slots capacity .. capacity+63: the keys a main slot cannot
 * hold -- those whose bytes 0-15 are all zero (they would read as empty) or
 * whose bytes 16-23 or 24-31 are all zero (they would read as still being
 * written) -- up to KVGOV_STASH_KEYS of them (KVGOV_F_TABLE_FULL past that).
 * For SHA-256 digests that is a key with probability about 2^-63.  Its
 * layout: bytes 0-3 of slot `capacity` count the entries handed out, the
 * u32 at byte 32 + 4e of that slot onwards is entry e's state (1 = live),
 * and entry e's key is slot capacity + 8 + e.
 */

/* kvgov_table_init -- mark every slot empty, main slots and side store
 * (capacity + KVGOV_STASH_SLOTS slots).  EINVAL: bad capacity/pointer. */
int kvgov_table_init(uint8_t *d_slots, uint64_t capacity, kvgov_stream_t stream);

/*
 * kvgov_insert -- add d_keys[n_keys][32] (16-byte aligned) to the set.
 * Duplicates, within the batch or with the table, are no-ops, so the
 * resulting set does not depend on order.  Calls on the same table must not
 * overlap in time with each other or with kvgov_probe (stream order them).
 *   d_n_new   nullable; the number of keys newly stored is ADDED to it.
 *   d_status  required; KVGOV_F_SENTINEL, KVGOV_F_TABLE_FULL and
 *             KVGOV_F_TIMEOUT as above.  A wait for another thread to finish
 *             writing a slot with the same first 16 bytes is bounded
 *             (kvgov_set_spin_limit); on timeout the key is not inserted.
 * n_keys = 0 is a no-op.  EINVAL: bad capacity, NULL or misaligned pointer,
 * n_keys < 0.
 */
int kvgov_insert(uint8_t *d_slots, uint64_t capacity, const uint8_t *d_keys, int64_t n_keys,
                 unsigned long long *d_n_new, uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_probe -- block prefix-cache lookup, paper section 2.1 (a lookup
 * matches the longest common prefix from position 0, truncated to a block
 * boundary), Table 1 row 1 (the probe learns the first k matched blocks) and
 * section 5.7 (a divergence at token i invalidates blocks floor(i/B) on):
 *   d_prefix_blocks[r] = min { j : h_j(r) not in table }, or n_b(r) if every
 *   block of request r is present.  Tokens served from cache = 16 * that.
 *
 *   d_digests       [d_blk_off[n_req]][32] u8 (kvgov_chain_hash output).
 *   d_blk_off       [n_req + 1] int64.
 *   d_prefix_blocks [n_req] int32 output.
 *   d_status        nullable; KVGOV_F_BADINDEX for a request whose rows are
 *                   not inside [d_blk_off[r], d_blk_off[n_req]) (it gets 0).
 * n_req = 0 is a no-op.  EINVAL: bad capacity, NULL or misaligned pointer.
 */
int kvgov_probe(const uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests,
                const int64_t *d_blk_off, int32_t n_req, int32_t *d_prefix_blocks,
                uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_probe_resume -- kvgov_probe when a lower bound of every prefix is
 * known: request r's walk starts at block d_prefix_blocks[r] (clamped to
 * [0, n_b(r)]) instead of block 0, and the blocks before it are taken as
 * cached.  Same definition and output as kvgov_probe (paper section 2.1)
 * as long as each input entry is at most the request's prefix length on the
 * table as it is now; a larger entry is not checked and is returned as if
 * its blocks were cached.  The serving step uses it after a chain launch
 * whose own lookups ran while the table was still growing
 * (kvgov_chain_hash_insert_prev).
 *   d_prefix_blocks [n_req] int32: in, the lower bounds (< 0 reads as 0);
 *                   out, the prefix lengths.
 *   other arguments, flags and EINVAL as for kvgov_probe.
 */
int kvgov_probe_resume(const uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests,
                       const int64_t *d_blk_off, int32_t n_req, int32_t *d_prefix_blocks, uint32_t *d_status,
                       kvgov_stream_t stream);

/*
 * kvgov_insert_uncached -- insert a probed batch: for every request r, its
 * blocks j >= d_prefix_blocks[r] (the output of kvgov_probe on the same
 * table, digests and offsets).  The blocks before that were found in the
 * table, and a table only grows, so the resulting set and *d_n_new are those
 * of inserting every digest with kvgov_insert.  In the serving step of the
 * paper's block prefix cache (section 2.1: lookup, then the uncached blocks
 * are computed and cached) this is the insert after the probe.
 *   d_digests, d_blk_off, n_req  as for kvgov_probe.
 *   d_prefix_blocks  [n_req] int32 from kvgov_probe (values < 0 read as 0).
 *   d_n_new, d_status  as for kvgov_insert (d_status required); also
 *                    KVGOV_F_BADINDEX for rows outside [d_blk_off[r], d_blk_off[n_req]).
 * Must not overlap in time with other calls on the same table.
 * n_req = 0 is a no-op.  EINVAL: bad capacity, NULL or misaligned pointer.
 */
int kvgov_insert_uncached(uint8_t *d_slots, uint64_t capacity, const uint8_t *d_digests,
                          const int64_t *d_blk_off, int32_t n_req, const int32_t *d_prefix_blocks,
                          unsigned long long *d_n_new, uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_chain_hash_insert_prev -- kvgov_chain_hash of one batch with, in the
 * same launch, kvgov_insert_uncached of the previous batch, and (if
 * d_prefix_blocks is given) kvgov_probe of this batch after that insert
 * (paper section 2.1: a served request's uncached blocks are computed and
 * cached; the next lookups see them).  In a stream of batches, batch i+1's
 * chain hash does not touch the table, so batch i's insert can run inside
 * it: each thread inserts uncached blocks of the previous batch between its
 * own compressions, and the inserts' memory latency is covered by the other
 * warps' hashing.  Results: the digests of kvgov_chain_hash; the table,
 * *d_n_new and the insert flags of kvgov_insert_uncached on the previous
 * batch; the prefix lengths of kvgov_probe of this batch on the table after
 * that insert.  With d_prefix_blocks the chain launch also looks each block
 * up as it is computed, while the insert runs: such a lookup can miss a key
 * still being inserted but never finds an absent one, so it leaves a lower
 * bound of each prefix, and a second launch resumes every request's walk
 * from there to the exact prefix length.
 *   mode .. d_digests  as for kvgov_chain_hash (this batch).
 *   d_slots, capacity  the table (as for kvgov_insert).
 *   d_prev_digests, d_prev_blk_off, prev_n_req, d_prev_prefix_blocks
 *              the previous batch, as for kvgov_insert_uncached; its arrays
 *              must not overlap this batch's d_digests.  prev_n_req = 0: no
 *              insert.
 *   d_prefix_blocks  [n_req] int32 output, or NULL for no probe.
 *   d_n_new, d_status  as for kvgov_insert_uncached (d_status required).
 * The table must not be read or written by other calls while this one runs.
 * A batch too small to give every SM sub-partition two warps (n_req < 2 * 32
 * * 4 * SMs) runs the chain hash and the insert as separate launches
 * instead; the results are the same.  EINVAL: as for kvgov_chain_hash and
 * kvgov_insert_uncached, prev_n_req < 0.
 */
int kvgov_chain_hash_insert_prev(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                 const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                                 const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                                 uint8_t *d_slots, uint64_t capacity, const uint8_t *d_prev_digests,
                                 const int64_t *d_prev_blk_off, int32_t prev_n_req,
                                 const int32_t *d_prev_prefix_blocks, int32_t *d_prefix_blocks,
                                 unsigned long long *d_n_new, uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_table_gen_stamp -- the table's generations (the per-key counter that
 * kvgov_chain_hash_serve keeps beside it): d_gen[h] = value for every handle h
 * that holds a key -- main slot h, or capacity + 8 + e for live side-store
 * entry e (the handles of kvgov_insert_arrival) -- and 0 for every other.
 *   d_gen  [capacity + KVGOV_STASH_SLOTS] u32, owned by the caller.
 * EINVAL: bad capacity, NULL or misaligned pointer.
 */
int kvgov_table_gen_stamp(const uint8_t *d_slots, uint64_t capacity, uint32_t *d_gen, uint32_t value,
                          kvgov_stream_t stream);

/*
 * kvgov_chain_hash_serve -- one batch through the whole serving step in one
 * launch (paper section 2.1: the batch's requests look up their cached
 * prefixes, then their uncached blocks are cached): kvgov_chain_hash, the
 * prefix lengths of kvgov_probe against the table as it was before this
 * call, and kvgov_insert_uncached of the batch after that, with its new keys
 * given generation `gen`.  The lookups and the insert run in the same
 * launch: a key counts as cached for this batch only if its generation is in
 * [gen_floor, gen), and every key this call adds gets generation gen, so the
 * batch's own keys never count as cached for it, whichever thread gets to a
 * key first.  A slot this call claims held no key when it began, so its
 * generation then is below gen_floor whenever the caller keeps the contract:
 *   - every key in the table has a generation in [gen_floor, gen) (stamp
 *     the keys of a table filled otherwise with kvgov_table_gen_stamp);
 *   - every handle that holds no key has a generation below gen_floor
 *     (zero the array with the table, or raise gen_floor to the first gen
 *     after each kvgov_table_init);
 *   - gen grows from one call to the next.
 *   mode .. d_digests  as for kvgov_chain_hash.
 *   d_slots, capacity  the table (as for kvgov_insert).
 *   d_gen  [capacity + KVGOV_STASH_SLOTS] u32 generations (above).
 *   d_prefix_blocks  [n_req] int32 output, as for kvgov_probe.
 *   d_n_new, d_status  as for kvgov_insert_uncached (d_status required).
 * The table must not be read or written by other calls while this one runs.
 * A batch too small to give every SM sub-partition two warps (n_req < 2 * 32
 * * 4 * SMs) runs the chain hash, the probe and the insert as separate
 * launches instead; the results are the same.  EINVAL: as for
 * kvgov_chain_hash and kvgov_insert_uncached, d_gen NULL, gen_floor > gen.
 */
int kvgov_chain_hash_serve(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                           const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                           const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                           uint8_t *d_slots, uint64_t capacity, uint32_t *d_gen, uint32_t gen, uint32_t gen_floor,
                           int32_t *d_prefix_blocks, unsigned long long *d_n_new, uint32_t *d_status,
                           kvgov_stream_t stream);

/*
 * Arrival-order serving of one batch -- paper section 2.1 (a lookup matches
 * the longest cached prefix of blocks from position 0) and section 4.2
 * (prefill cost is proportional to the uncached tokens), applied request by
 * request: the requests of the batch arrive in order; request r's cached
 * prefix is its longest run of leading blocks that were cached when it
 * arrived (in the table before the batch, or blocks of a request that
 * arrived before it), and then all its blocks are cached.  The result equals
 * serving the requests one at a time with kvgov_probe and kvgov_insert, in
 * one pass over the batch:
 *
 *   kvgov_insert_arrival(...)   every block's key into the table, recording
 *                               its slot and, per slot, the first arrival;
 *   kvgov_probe_arrival(...)    the prefix lengths.
 *
 * Arrival positions: block j of request r has position
 * seq_base + blk_off[r] + j, so a batch covers blk_off[n_req] positions from
 * seq_base.  The owner array d_owner [capacity + KVGOV_STASH_SLOTS] u64,
 * beside the table, holds per slot (a main slot, or a side-store entry at its
 * handle capacity + 8 + e) the smallest position whose block inserted the
 * slot's key through
 * kvgov_insert_arrival (0 for keys inserted any other way, which count as
 * cached before every arrival).  Zero it once with kvgov_owner_init when the
 * table is created; it stays valid across kvgov_table_init as long as
 * positions only grow: every call's seq_base must be at least the previous
 * call's seq_base + blk_off[n_req] (on the same owner array).  seq_base lies
 * in [1, 2^62].  capacity: a power of two in [32, 2^30].
 */

/*
 * kvgov_owner_init -- zero d_owner [capacity + KVGOV_STASH_SLOTS] u64
 * (16-byte aligned).
 * EINVAL: NULL or misaligned pointer, bad capacity.
 */
int kvgov_owner_init(uint64_t *d_owner, uint64_t capacity, kvgov_stream_t stream);

/*
 * kvgov_insert_arrival -- insert every block of the batch (the set semantics
 * and protocol of kvgov_insert) and settle the owners of the keys it adds.
 *   d_slots, capacity, d_digests, d_blk_off, n_req  as for kvgov_probe.
 *   d_owner    [capacity + KVGOV_STASH_SLOTS] u64, see above.
 *   seq_base   arrival position of the batch's first block.
 *   d_slot_of  [d_blk_off[n_req]] u32 output: the handle of each block's
 *              key (its main slot, or capacity + 8 + its side-store entry),
 *              or 0xFFFFFFFF if it could not be stored (the all-zero key, a
 *              full window or side store, a timeout -- flagged in
 *              *d_status).  This is the
 *              block's handle in the cache and the input of
 *              kvgov_probe_arrival.
 *   d_n_new, d_status  as for kvgov_insert (d_status required); also
 *              KVGOV_F_BADINDEX if d_blk_off[n_req] < 0.
 * Two launches on `stream`, one thread per block.  Must not overlap in time
 * with other calls on the same table or owner array.  n_req = 0 is a no-op.
 * EINVAL: bad capacity, NULL or misaligned pointer, seq_base out of range.
 */
int kvgov_insert_arrival(uint8_t *d_slots, uint64_t *d_owner, uint64_t capacity, const uint8_t *d_digests,
                         const int64_t *d_blk_off, int32_t n_req, uint64_t seq_base, uint32_t *d_slot_of,
                         unsigned long long *d_n_new, uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_probe_arrival -- d_prefix_blocks[r] = the smallest j such that block
 * j of request r was not cached when r arrived (its d_slot_of is 0xFFFFFFFF,
 * or its slot's owner is >= seq_base + d_blk_off[r]), or n_b(r) if every
 * block was.  Run after kvgov_insert_arrival of the same batch (same
 * d_blk_off, n_req and seq_base) and before the next call on the owner array.
 *   d_owner, capacity  as for kvgov_insert_arrival; d_slot_of its output.
 *   d_status  nullable; KVGOV_F_BADINDEX for malformed offsets.
 * n_req = 0 is a no-op.  EINVAL: bad capacity, NULL pointer, seq_base out of
 * range.
 */
int kvgov_probe_arrival(const uint64_t *d_owner, uint64_t capacity, const uint32_t *d_slot_of,
                        const int64_t *d_blk_off, int32_t n_req, uint64_t seq_base, int32_t *d_prefix_blocks,
                        uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_serve_arrival_static -- kvgov_insert_arrival followed by
 * kvgov_probe_arrival on one batch, allocating nothing: the slot of each
 * block lives in a device array of 2^21 entries (8 MiB) inside the library
 * rather than in caller memory.  The paper has no counterpart; it is an
 * allocation-free form of the same computation (same table, owners, key
 * count and prefix lengths; the slot handles are not returned).
 *   Arguments as for kvgov_insert_arrival and kvgov_probe_arrival;
 *   n_blocks   the batch's block count, d_blk_off[n_req]; d_digests must
 *              hold at least n_blocks rows.  Every kernel of the call bounds
 *              the rows it reads by n_blocks.
 * EINVAL also when n_blocks exceeds 2^21.  If d_blk_off[n_req] differs from
 * n_blocks by being larger, no block is inserted, no digest row past
 * n_blocks is read, and every request is flagged KVGOV_F_BADINDEX with
 * prefix 0.  The array is shared by every call on the device: calls that
 * overlap in time (other streams, other host threads) race on it and give
 * wrong results.  Its device address is looked up (cudaGetSymbolAddress) on
 * the first call made with each device current and kept for the process, so
 * that first call should come before any stream capture, and the library
 * does not survive a cudaDeviceReset of that device.  Three launches on
 * `stream`, four for batches of 4096 requests or more (their first 32
 * requests' blocks are inserted first, as in kvgov_insert_arrival).
 */
int kvgov_serve_arrival_static(uint8_t *d_slots, uint64_t *d_owner, uint64_t capacity, const uint8_t *d_digests,
                               const int64_t *d_blk_off, int32_t n_req, int64_t n_blocks, uint64_t seq_base,
                               int32_t *d_prefix_blocks, unsigned long long *d_n_new, uint32_t *d_status,
                               kvgov_stream_t stream);

/*
 * kvgov_chain_hash_arrival -- a batch's chain hash and its arrival-order
 * serving in one call: the digests of kvgov_chain_hash, then the table,
 * owners, slot handles, prefix lengths and key count of kvgov_insert_arrival
 * followed by kvgov_probe_arrival, bit for bit.
 *   mode .. d_digests  as for kvgov_chain_hash.
 *   d_slots, d_owner, capacity, seq_base, d_slot_of, d_n_new  as for
 *              kvgov_insert_arrival (d_slot_of [d_blk_off[n_req]]).
 *   d_prefix_blocks  [n_req] int32 output, as for kvgov_probe_arrival.
 *   d_status   required: KVGOV_F_BADINDEX as for kvgov_chain_hash, and the
 *              insert flags.
 * Batches that give every SM sub-partition at least two warps
 * (n_req >= 2 x 32 x 4 x SMs) insert each digest from the chain kernel as
 * soon as it is computed -- the lanes of a warp hold block j of 32
 * consecutive requests, so a key their prefixes share is inserted once per
 * warp -- then settle the owners and probe (three launches); smaller batches
 * run the chain, the insert and the probe as separate launches.  Same
 * results either way.  Must not overlap in time with other calls on the same
 * table or owner array.  n_req = 0 is a no-op.  EINVAL: as for
 * kvgov_chain_hash and kvgov_insert_arrival.
 */
int kvgov_chain_hash_arrival(int mode, const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                             const int32_t *d_principal, const uint8_t *d_salts, int32_t n_principals,
                             const int32_t *d_boundary_tok, const int64_t *d_blk_off, uint8_t *d_digests,
                             uint8_t *d_slots, uint64_t *d_owner, uint64_t capacity, uint64_t seq_base,
                             uint32_t *d_slot_of, int32_t *d_prefix_blocks, unsigned long long *d_n_new,
                             uint32_t *d_status, kvgov_stream_t stream);

/*
 * kvgov_set_spin_limit -- bound on how many times an inserting thread
 * re-reads a slot whose key another thread is still writing before it gives
 * up with KVGOV_F_TIMEOUT (about 100 ns per re-read).
 * Process-wide; applies to launches made after the call.  0 restores the
 * default (2^23, about a second).  Returns the previous value.
 */
uint32_t kvgov_set_spin_limit(uint32_t limit);

#ifdef __cplusplus
}
#endif

#endif /* KVGOV_H */
