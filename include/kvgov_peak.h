/*
 * kvgov_peak.h -- C ABI of libkvgov_peak: the integer issue-rate
 * microbenchmark that sets the roofline denominator for the hashing kernels,
 * and the random-slot read microbenchmark that sets the ceiling for the
 * table kernels.  They are measurement tools beside libkvgov, not part of
 * the method.
 *
 * The hashing path of the paper (SHA-256 block keys and HMAC salts, section
 * 4.1; Table 9) is integer work: rotates, three-input booleans and adds.
 * Its roofline is the rate at which an SM can issue those instructions.
 */
#ifndef KVGOV_PEAK_H
#define KVGOV_PEAK_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *kvgov_stream_t;

/*
 * kvgov_peak_int -- launch `blocks` CTAs of `threads` threads, each running
 * `iters` iterations of the instruction body of `kind`:
 *   0 LOP3, 1 SHF (funnel shift), 2 IADD3, 3 SHA-256 compression (FIPS 180-4)
 *   with ALU adds, 4 the same with every add as IMAD (FMA pipe), 5 IMAD,
 *   6 SHA-256 rounds alone with K_t + W_t in registers (T1/T2 grouping),
 *   7 the same rounds with the shorter e-to-e grouping, and two-kind mixes
 *   (half the streams each, interleaved) that show whether two kinds share
 *   a pipe: 8 LOP3 + IADD3, 9 LOP3 + IMAD, 10 SHF + IADD3; 11 the chain
 *   kernel's steady block (a 96-byte message, two compact compressions,
 *   2 x 1384 nominal ops) with every add on the ALU, 12 the same with the
 *   adds off the rounds' dependency chain on the FMA pipe.
 * d_clocks [blocks][3] u64 receives, per CTA, its SM id and its clock64()
 * at start and end.  d_sink [1] u32 is written only in a case that never
 * happens (keeps results live).  Asynchronous on `stream`.
 * Returns 0, 1 for a bad argument (nothing launched), 2 for a launch error.
 */
int kvgov_peak_int(int kind, int iters, int blocks, int threads, uint32_t *d_sink,
                   unsigned long long *d_clocks, kvgov_stream_t stream);

/*
 * kvgov_peak_gather -- the bandwidth ceiling of the table kernels: `n_reads`
 * reads of `slot_bytes` (16: the first half of a slot, as the fused lookup
 * reads; 32: a whole slot, as the probe and insert read) at pseudo-random
 * slots of a table of `n_slots` 32-byte slots (slot of read i =
 * splitmix64(seed + i) mod n_slots).
 *   d_table  [n_slots][32] bytes, device, 16-byte aligned, only read.
 *   n_slots  a power of two.
 *   d_sink   [1] u32, written only in a case that never happens.
 * Asynchronous on `stream`.  Returns 0, 1 for a bad argument (nothing
 * launched), 2 for a launch error.  Algorithmic bytes = n_reads x slot_bytes.
 */
int kvgov_peak_gather(const void *d_table, uint64_t n_slots, int slot_bytes, int64_t n_reads, uint64_t seed,
                      uint32_t *d_sink, kvgov_stream_t stream);

/*
 * kvgov_peak_slot_ops -- the write side of that ceiling: `n_ops` operations
 * on pseudo-random 32-byte slots (slot of op i = splitmix64(seed + i) mod
 * n_slots) of a table that must be zero: kind 0 a 128-bit compare-and-swap
 * of the slot's first 16 bytes from zero; kind 1 that CAS and a 16-byte
 * store of the second half (an insert's claim of a new key); kind 2 a
 * 16-byte read of the first half before them (the insert's look first).
 *   d_table  [n_slots][32] bytes, device, 16-byte aligned, zeroed; modified.
 * Asynchronous on `stream`.  Returns 0, 1 for a bad argument (nothing
 * launched), 2 for a launch error.
 */
int kvgov_peak_slot_ops(void *d_table, uint64_t n_slots, int kind, int64_t n_ops, uint64_t seed, uint32_t *d_sink,
                        kvgov_stream_t stream);

/* Thread-operations one thread executes per iteration of `kind` (nominal
 * SHA-256 count of 1384 per compression for kinds 3 and 4), or 0 for a bad
 * kind. */
int kvgov_peak_ops_per_iter(int kind);

#ifdef __cplusplus
}
#endif

#endif /* KVGOV_PEAK_H */
