/*
 * kvgov_pipeline.h -- C ABI of libkvgov's serving engine: a stream of
 * batches served back to back through the hot path of kvgov.h (salts,
 * blocking, chain hash, probe, insert of the uncached blocks), with the
 * stream schedule kept on the host side of the library rather than in the
 * caller's language.  Paper section 2.1: every request looks up its longest
 * cached block prefix, then its uncached blocks are computed and cached; a
 * batch sees every block of the batches before it.
 *
 * Unlike kvgov.h, an engine is stateful: kvgov_pipeline_create copies the
 * caller's description (device buffers, events, streams -- all owned by the
 * caller, which keeps them alive until kvgov_pipeline_destroy) into a small
 * host-side object, the only memory the library allocates; the engine keeps
 * those pointers between calls.  Every call only enqueues work and returns;
 * none synchronises.  Return values as in kvgov.h (KVGOV_OK, KVGOV_EINVAL,
 * KVGOV_ECUDA for a failed launch or event call); device-detected flags go to
 * the description's d_status.
 *
 * Schedule of kvgov_pipeline_submit for batch i (slot s = i mod n_slots):
 *   prep stream     waits for `after` (the batch's inputs are ready), for
 *                   batch i-1's chain launch to have started, and for slot s
 *                   to be free; then kvgov_derive_salts (unless UNSALTED)
 *                   and kvgov_block_offsets into slot s; records prepared[s].
 *   compute stream  waits for prepared[s]; with `flush`, first runs the
 *                   pending insert (below) and kvgov_table_init; records
 *                   chain_start[s] as the last command before the chain
 *                   launch, so that batch i+1's prep runs beside it; then
 *     insert_in_chain = 1: kvgov_chain_hash_insert_prev (batch i's chain
 *                   hash carrying the insert of the pending batch i-1, its
 *                   own lookups of batch i leaving in d_prefix[s] a lower
 *                   bound of each prefix), then the probe of batch i resuming
 *                   each walk from there (the prefix lengths of kvgov_probe
 *                   on the table after the insert); batch i's insert is left pending
 *                   for the next submit (or kvgov_pipeline_drain); slot s-1
 *                   is free once the chain launch is done.  With no pending
 *                   batch: kvgov_chain_hash_probe.
 *     insert_in_chain = 0: kvgov_chain_hash_probe, then kvgov_insert_uncached.
 *     insert_in_chain = 2 (KVGOV_SCHEDULE_ONE_LAUNCH): kvgov_chain_hash_serve,
 *                   batch i's lookups and insert in one launch, with
 *                   generation g_i in d_gen: the engine stamps the keys
 *                   already in the table with generation 1 before its first
 *                   batch (kvgov_table_gen_stamp), gives batch i generation
 *                   g_i = i + 2, and after a flush raises the floor to the
 *                   flushing batch's generation; no insert is left pending.
 *                   records probed[s] after the probe (batch i's prefix
 *                   lengths are then valid in d_prefix[s]).
 * The results equal serving the batches one at a time in order.
 */
#ifndef KVGOV_PIPELINE_H
#define KVGOV_PIPELINE_H

#include <stddef.h>
#include <stdint.h>

#include "kvgov.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaEvent_t / CUevent. */
typedef struct CUevent_st *kvgov_event_t;

#define KVGOV_PIPELINE_MAX_SLOTS 3
#define KVGOV_SCHEDULE_ONE_LAUNCH 2   /* kvgov_pipeline_desc.insert_in_chain: see above */

/* What an engine serves with; every pointer and handle is the caller's. */
typedef struct kvgov_pipeline_desc {
    int mode;                     /* KVGOV_UNSALTED / KVGOV_ROOT / KVGOV_BOUNDARY        */
    int insert_in_chain;          /* the schedule above: 1 (3 slots), 0 or 2 (2 slots)   */
    int n_slots;                  /* 3 if insert_in_chain is 1, else 2                   */
    int32_t max_req;              /* capacity of each slot: requests ...                 */
    int64_t max_blocks;           /* ... and blocks                                      */
    /* the cache */
    uint8_t *d_slots;             /* [capacity + KVGOV_STASH_SLOTS][32] table             */
    uint64_t capacity;
    uint32_t *d_status;           /* flags (required)                                    */
    unsigned long long *d_n_new;  /* keys inserted (nullable)                            */
    /* principals (salted modes): the ids as for kvgov_derive_salts */
    const uint8_t *d_ids;
    const int64_t *d_id_off;      /* [n_principals + 1]                                  */
    int32_t n_principals;
    /* per slot: salts [n_principals][32], block offsets [max_req + 1],
       digests [max_blocks][32] (16-byte aligned), prefix lengths [max_req] */
    uint8_t *d_salts[KVGOV_PIPELINE_MAX_SLOTS];
    int64_t *d_blk_off[KVGOV_PIPELINE_MAX_SLOTS];
    uint8_t *d_digests[KVGOV_PIPELINE_MAX_SLOTS];
    int32_t *d_prefix[KVGOV_PIPELINE_MAX_SLOTS];
    /* per slot events, created by the caller, recorded by the engine */
    kvgov_event_t prepared[KVGOV_PIPELINE_MAX_SLOTS];
    kvgov_event_t chain_start[KVGOV_PIPELINE_MAX_SLOTS];
    kvgov_event_t probed[KVGOV_PIPELINE_MAX_SLOTS];
    kvgov_event_t free_ev[KVGOV_PIPELINE_MAX_SLOTS];
    kvgov_stream_t prep_stream;
    kvgov_stream_t compute_stream;
    /* insert_in_chain = 2 only: the table's generations, [capacity +
       KVGOV_STASH_SLOTS] u32, zeroed by the caller with the table (or left
       as an earlier engine of this schedule left them), and used by no
       other engine while this one is alive.  From the engine's first submit
       on, the table must change only through it: a key added otherwise has
       no generation of this engine's and would not count as cached. */
    uint32_t *d_gen;
} kvgov_pipeline_desc;

typedef struct kvgov_pipeline kvgov_pipeline;   /* opaque */

/*
 * kvgov_pipeline_create -- check the description and make an engine.
 * EINVAL: bad mode, insert_in_chain not 0, 1 or 2, slot count not 3 (insert_in_chain = 1) or 2, a NULL buffer,
 * event or stream, max_req < 0 or max_blocks < 0, a bad capacity, salted
 * mode without ids, misaligned digests or table.
 */
int kvgov_pipeline_create(const kvgov_pipeline_desc *desc, kvgov_pipeline **out);

/*
 * kvgov_pipeline_submit -- queue one batch (the schedule in the header
 * comment).  The batch: d_tokens, d_tok_off [n_req + 1], d_principal and
 * d_boundary_tok as for kvgov_chain_hash (device, caller-owned, read by the
 * engine's streams until *slot_out's probed event; with insert_in_chain the
 * batch's digests are read again by the next submit's chain launch, from
 * the engine's slot); n_blocks = d_blk_off[n_req] as the caller knows it (it
 * sizes the slot; EINVAL above max_blocks); n_req above max_req is EINVAL.
 * secret: host bytes for kvgov_derive_salts, copied before returning.
 * after: nullable; waited on before the batch's inputs are read.
 * flush: nonzero empties the cache before this batch (after the pending
 * insert, so that the previous batch is cached and then dropped like every
 * other).  chain_ev, table_ev: nullable pairs of timing events recorded
 * around the chain-hash launch and around the table kernel after it (the
 * probe; the insert when insert_in_chain = 0); not recorded when the batch
 * runs no such kernel of its own.  *slot_out: the slot holding the batch's
 * prefix lengths (d_prefix[slot]), valid once probed[slot] has completed
 * and overwritten by a later submit into the same slot.
 */
int kvgov_pipeline_submit(kvgov_pipeline *pl, const uint8_t *secret, size_t secret_len, const int32_t *d_tokens,
                          const int64_t *d_tok_off, int32_t n_req, const int32_t *d_principal,
                          const int32_t *d_boundary_tok, int64_t n_blocks, kvgov_event_t after, int flush,
                          kvgov_event_t chain_ev0, kvgov_event_t chain_ev1, kvgov_event_t table_ev0,
                          kvgov_event_t table_ev1, int32_t *slot_out);

/*
 * kvgov_pipeline_drain -- run the pending insert, if any, on the compute
 * stream; afterwards the table holds every submitted batch.
 */
int kvgov_pipeline_drain(kvgov_pipeline *pl);

/* kvgov_pipeline_pending -- 1 if a batch's insert is pending, else 0. */
int kvgov_pipeline_pending(const kvgov_pipeline *pl);

/* kvgov_pipeline_destroy -- free the engine (not the caller's buffers); NULL is a no-op. */
void kvgov_pipeline_destroy(kvgov_pipeline *pl);

#ifdef __cplusplus
}
#endif

#endif /* KVGOV_PIPELINE_H */
