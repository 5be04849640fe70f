// kvgov_pipeline.cu -- the serving engine of kvgov_pipeline.h: the stream
// schedule of a stream of batches through the hot path (paper section 2.1:
// every request looks up its longest cached block prefix, then its uncached
// blocks are cached; each batch sees every block of the batches before it).
//
// Host code only: it orders the entry points of kvgov.h on the caller's
// streams with the caller's events, one call per batch, so that a caller
// in any language pays one foreign call per batch rather than one per
// launch, wait and record.  The schedule is written out in the header.
#include <cuda_runtime.h>

#include <new>

#include "../../include/kvgov.h"
#include "../../include/kvgov_pipeline.h"
#include "kvgov_internal.cuh"

struct kvgov_pipeline {
    kvgov_pipeline_desc d;
    long long submitted = 0;                       // batches queued so far
    int pending = -1;                              // slot whose batch's insert has not run yet
    int last = -1;                                 // slot of the last batch whose chain launch was queued
    bool used[KVGOV_PIPELINE_MAX_SLOTS] = {};
    int32_t n_req[KVGOV_PIPELINE_MAX_SLOTS] = {};  // the batch in each slot
    // KVGOV_SCHEDULE_ONE_LAUNCH: the last generation given, the floor, and
    // whether the table's keys have been stamped with generation 1
    uint32_t gen = 1;
    uint32_t gen_floor = 1;
    bool stamped = false;
};

namespace {

cudaStream_t stream_of(kvgov_stream_t s) { return reinterpret_cast<cudaStream_t>(s); }
cudaEvent_t event_of(kvgov_event_t e) { return reinterpret_cast<cudaEvent_t>(e); }

int record(kvgov_event_t e, kvgov_stream_t s) {
    return cudaEventRecord(event_of(e), stream_of(s)) == cudaSuccess ? KVGOV_OK : KVGOV_ECUDA;
}
int wait(kvgov_stream_t s, kvgov_event_t e) {
    return cudaStreamWaitEvent(stream_of(s), event_of(e), 0) == cudaSuccess ? KVGOV_OK : KVGOV_ECUDA;
}

// The pending batch's insert as its own launch on the compute stream; its
// slot is free after it.
int insert_pending(kvgov_pipeline *pl) {
    const int q = pl->pending;
    if (q < 0) return KVGOV_OK;
    const kvgov_pipeline_desc &d = pl->d;
    int rc = kvgov_insert_uncached(d.d_slots, d.capacity, d.d_digests[q], d.d_blk_off[q], pl->n_req[q],
                                   d.d_prefix[q], d.d_n_new, d.d_status, d.compute_stream);
    if (rc == KVGOV_OK) rc = record(d.free_ev[q], d.compute_stream);
    pl->pending = -1;
    return rc;
}

bool desc_ok(const kvgov_pipeline_desc &d) {
    using kvgov_host::aligned16;
    if (d.mode != KVGOV_UNSALTED && d.mode != KVGOV_ROOT && d.mode != KVGOV_BOUNDARY) return false;
    if (d.insert_in_chain < 0 || d.insert_in_chain > KVGOV_SCHEDULE_ONE_LAUNCH) return false;
    if (d.n_slots != (d.insert_in_chain == 1 ? 3 : 2)) return false;
    if (d.insert_in_chain == KVGOV_SCHEDULE_ONE_LAUNCH && !d.d_gen) return false;
    if (d.max_req < 0 || d.max_blocks < 0) return false;
    if (!d.d_slots || !aligned16(d.d_slots) || !kvgov_host::pow2_capacity(d.capacity) || !d.d_status) return false;
    if (d.mode != KVGOV_UNSALTED && (!d.d_ids || !d.d_id_off || d.n_principals <= 0)) return false;
    if (!d.prep_stream || !d.compute_stream) return false;
    for (int s = 0; s < d.n_slots; ++s) {
        if (!d.d_blk_off[s] || !d.d_digests[s] || !aligned16(d.d_digests[s]) || !d.d_prefix[s]) return false;
        if (d.mode != KVGOV_UNSALTED && (!d.d_salts[s] || !aligned16(d.d_salts[s]))) return false;
        if (!d.prepared[s] || !d.chain_start[s] || !d.probed[s] || !d.free_ev[s]) return false;
    }
    return true;
}

}  // namespace

extern "C" int kvgov_pipeline_create(const kvgov_pipeline_desc *desc, kvgov_pipeline **out) {
    if (!desc || !out || !desc_ok(*desc)) return KVGOV_EINVAL;
    kvgov_pipeline *pl = new (std::nothrow) kvgov_pipeline;
    if (!pl) return KVGOV_ECUDA;
    pl->d = *desc;
    *out = pl;
    return KVGOV_OK;
}

extern "C" int kvgov_pipeline_submit(kvgov_pipeline *pl, const uint8_t *secret, size_t secret_len,
                                     const int32_t *d_tokens, const int64_t *d_tok_off, int32_t n_req,
                                     const int32_t *d_principal, const int32_t *d_boundary_tok, int64_t n_blocks,
                                     kvgov_event_t after, int flush, kvgov_event_t chain_ev0,
                                     kvgov_event_t chain_ev1, kvgov_event_t table_ev0, kvgov_event_t table_ev1,
                                     int32_t *slot_out) {
    if (!pl || !slot_out) return KVGOV_EINVAL;
    const kvgov_pipeline_desc &d = pl->d;
    // every argument is checked before anything is queued
    if (n_req < 0 || n_req > d.max_req || n_blocks < 0 || n_blocks > d.max_blocks || !d_tok_off) return KVGOV_EINVAL;
    if (n_req > 0 && !d_tokens) return KVGOV_EINVAL;
    if (d.mode != KVGOV_UNSALTED && n_req > 0 && !d_principal) return KVGOV_EINVAL;
    if (d.mode == KVGOV_BOUNDARY && n_req > 0 && !d_boundary_tok) return KVGOV_EINVAL;
    if (d.mode != KVGOV_UNSALTED && (secret_len > KVGOV_MAX_SECRET || (secret_len > 0 && !secret)))
        return KVGOV_EINVAL;
    if ((chain_ev0 == nullptr) != (chain_ev1 == nullptr) || (table_ev0 == nullptr) != (table_ev1 == nullptr))
        return KVGOV_EINVAL;

    if (d.insert_in_chain == KVGOV_SCHEDULE_ONE_LAUNCH && pl->gen == 0xffffffffu) return KVGOV_EINVAL;   // spent
    const int s = (int)(pl->submitted % d.n_slots);
    const kvgov_stream_t ps = d.prep_stream, cs = d.compute_stream;
    const bool salted = d.mode != KVGOV_UNSALTED;
    int rc = KVGOV_OK;
#define KV_TRY(call)                     \
    do {                                 \
        rc = (call);                     \
        if (rc != KVGOV_OK) return rc;   \
    } while (0)

    // prep stream: salts and block offsets of this batch, beside the previous chain launch
    if (after) KV_TRY(wait(ps, after));
    if (pl->last >= 0) KV_TRY(wait(ps, d.chain_start[pl->last]));
    if (pl->used[s]) KV_TRY(wait(ps, d.free_ev[s]));
    if (salted)
        KV_TRY(kvgov_derive_salts(secret, secret_len, d.d_ids, d.d_id_off, d.n_principals, d.d_salts[s], d.d_status,
                                  ps));
    KV_TRY(kvgov_block_offsets(d_tok_off, n_req, d.d_blk_off[s], d.d_status, ps));
    KV_TRY(record(d.prepared[s], ps));

    // compute stream
    if (after) KV_TRY(wait(cs, after));
    KV_TRY(wait(cs, d.prepared[s]));
    const bool one_launch = d.insert_in_chain == KVGOV_SCHEDULE_ONE_LAUNCH;
    if (flush) {
        KV_TRY(insert_pending(pl));
        KV_TRY(kvgov_table_init(d.d_slots, d.capacity, cs));
        pl->gen_floor = pl->gen + 1;                  // every generation given so far is below it
        pl->stamped = true;                           // the table is empty: nothing to stamp
    }
    if (one_launch && !pl->stamped) {                 // keys already in the table: generation 1
        KV_TRY(kvgov_table_gen_stamp(d.d_slots, d.capacity, d.d_gen, 1u, cs));
        pl->stamped = true;
    }
    if (chain_ev0) KV_TRY(record(chain_ev0, cs));
    // the last command before the chain launch: the next batch's prep starts
    // only once this chain kernel is being placed
    KV_TRY(record(d.chain_start[s], cs));
    pl->last = s;
    const int q = d.insert_in_chain == 1 ? pl->pending : -1;
    const int32_t *pr = salted ? d_principal : nullptr;
    const uint8_t *sl = salted ? d.d_salts[s] : nullptr;
    const int32_t *bt = d.mode == KVGOV_BOUNDARY ? d_boundary_tok : nullptr;
    // one launch: the batch's lookups and insert in its chain launch.  Else,
    // with the previous batch's insert in the chain launch, that launch also
    // looks this batch's blocks up (a lower bound of each prefix) and the
    // probe below resumes the walks from there
    if (one_launch) {
        const uint32_t g = ++pl->gen;
        KV_TRY(kvgov_chain_hash_serve(d.mode, d_tokens, d_tok_off, n_req, pr, sl, d.n_principals, bt, d.d_blk_off[s],
                                      d.d_digests[s], d.d_slots, d.capacity, d.d_gen, g, pl->gen_floor,
                                      d.d_prefix[s], d.d_n_new, d.d_status, cs));
    } else if (q >= 0)
        KV_TRY(kvgov_host::chain_insert_prev_lower(d.mode, d_tokens, d_tok_off, n_req, pr, sl, d.n_principals, bt,
                                                   d.d_blk_off[s], d.d_digests[s], d.d_slots, d.capacity,
                                                   d.d_digests[q], d.d_blk_off[q], pl->n_req[q], d.d_prefix[q],
                                                   d.d_prefix[s], d.d_n_new, d.d_status, cs));
    else
        KV_TRY(kvgov_chain_hash_probe(d.mode, d_tokens, d_tok_off, n_req, pr, sl, d.n_principals, bt, d.d_blk_off[s],
                                      d.d_digests[s], d.d_slots, d.capacity, d.d_prefix[s], d.d_status, cs));
    if (chain_ev1) KV_TRY(record(chain_ev1, cs));
    if (q >= 0) {
        KV_TRY(record(d.free_ev[q], cs));             // the previous batch is cached: its slot is free
        pl->pending = -1;
    }
    if (one_launch) {
        KV_TRY(record(d.probed[s], cs));
        KV_TRY(record(d.free_ev[s], cs));            // the batch is cached: its slot is free
    } else if (d.insert_in_chain) {
        if (q >= 0) {                                 // the probe after the insert
            if (table_ev0) KV_TRY(record(table_ev0, cs));
            KV_TRY(kvgov_host::probe_resume(d.d_slots, d.capacity, d.d_digests[s], d.d_blk_off[s], n_req,
                                            d.d_prefix[s], d.d_status, cs));
            if (table_ev1) KV_TRY(record(table_ev1, cs));
        }
        KV_TRY(record(d.probed[s], cs));
        pl->pending = s;
    } else {
        KV_TRY(record(d.probed[s], cs));
        if (table_ev0) KV_TRY(record(table_ev0, cs));
        KV_TRY(kvgov_insert_uncached(d.d_slots, d.capacity, d.d_digests[s], d.d_blk_off[s], n_req, d.d_prefix[s],
                                     d.d_n_new, d.d_status, cs));
        if (table_ev1) KV_TRY(record(table_ev1, cs));
        KV_TRY(record(d.free_ev[s], cs));
    }
#undef KV_TRY
    pl->used[s] = true;
    pl->n_req[s] = n_req;
    ++pl->submitted;
    *slot_out = s;
    return KVGOV_OK;
}

extern "C" int kvgov_pipeline_drain(kvgov_pipeline *pl) {
    if (!pl) return KVGOV_EINVAL;
    return insert_pending(pl);
}

extern "C" int kvgov_pipeline_pending(const kvgov_pipeline *pl) { return pl && pl->pending >= 0 ? 1 : 0; }

extern "C" void kvgov_pipeline_destroy(kvgov_pipeline *pl) { delete pl; }
