/*
 * opattn.h -- C ABI of libopattn: causal grouped-query prefill attention over
 * a ragged, packed batch of prompts, on one NVIDIA GB300 (sm_103a).
 *
 * The operation is the attention operator that OpScale (§2.1, "Compute
 * Sensitivity") identifies as the prompt-length-sensitive, O(L^2 b) operator
 * that sets time-to-first-token; it is exact softmax attention computed
 * without materialising the L x L score matrix (§2.1, "Memory Sensitivity",
 * FlashAttention).  Query heads are grouped over key/value heads
 * (grouped-query attention, §5.6) and the causal mask is aligned to the
 * bottom-right corner of each sequence so that a chunk of a prompt attends to
 * its already-cached prefix (chunked prefill, §6).
 *
 * For sequence s with Lq = cu_seqlens_q[s+1] - cu_seqlens_q[s] queries and
 * Lk = cu_seqlens_k[s+1] - cu_seqlens_k[s] keys, query row i (0-based within
 * the sequence) sees key j iff j <= i + (Lk - Lq) and j < Lk.  With
 * G = Hq / Hkv, query head h reads key/value head h / G.  For every query
 * row i and head h:
 *     x_j = scale * <q[i,h,:], k[j,h/G,:]>
 *     O[i,h,:]  = sum_j softmax(x)_j * v[j,h/G,:]
 *     LSE[i,h]  = ln sum_j exp(x_j)          (natural log, scaled logits)
 * A row that sees no key gets O = 0 and LSE = -infinity.
 *
 * Layouts (all packed, contiguous, row-major):
 *     q   bf16 [total_q, Hq,  d]     total_q = cu_seqlens_q[n_seq]
 *     k,v bf16 [total_k, Hkv, d]     total_k = cu_seqlens_k[n_seq]
 *     o   bf16 [total_q, Hq,  d]
 *     lse fp32 [total_q, Hq]
 * q, k, v, o and lse are device pointers; q, k, v and o must be 16-byte
 * aligned and lse 4-byte aligned.  cu_seqlens_q / cu_seqlens_k are HOST
 * arrays of n_seq + 1 int32 offsets, starting at 0 and non-decreasing.
 * Sequences may be empty and may have Lq > Lk.
 *
 * Ownership: the caller owns every buffer and the stream.  The library keeps
 * no pointer to caller memory after a call returns.
 *
 * Asynchrony: every call except opattn_prefill_checked and the plan
 * create/destroy calls is asynchronous with respect to the host and ordered
 * on `stream` (a cudaStream_t; NULL means the legacy default stream).
 * Outputs are valid once the stream has reached the call.
 *
 * Errors: every function returns an opattn_status.  Argument errors are
 * detected on the host before any device work and leave outputs untouched.
 * The kernel bounds every wait; if one expires it stops early and records
 * the error in a device status word, which opattn_prefill_checked reads back.
 */
#ifndef OPATTN_H
#define OPATTN_H

#include <stdint.h>

#if defined(__GNUC__)
#define OPATTN_API __attribute__((visibility("default")))
#else
#define OPATTN_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum opattn_status {
    OPATTN_OK = 0,
    OPATTN_ERR_INVALID_ARG = 1,  /* null pointer, bad count, non-monotone offsets, scale <= 0 */
    OPATTN_ERR_UNSUPPORTED = 2,  /* d not in {64, 128}, or Hq / Hkv > 128 */
    OPATTN_ERR_MISALIGNED = 3,   /* q/k/v/o not 16-byte or lse not 4-byte aligned */
    OPATTN_ERR_CUDA = 4,         /* a CUDA runtime call or the launch failed */
    OPATTN_ERR_TIMEOUT = 5,      /* a bounded device wait expired (checked entry point only) */
    OPATTN_ERR_CAPACITY = 6      /* an output array given to opattn_schedule is too small */
} opattn_status;

/* Library version as major * 10000 + minor * 100 + patch. */
OPATTN_API int32_t opattn_version(void);

/* Static, NUL-terminated description of a status code. */
OPATTN_API const char *opattn_status_string(int32_t status);

/*
 * One-shot prefill attention (the definition above).  Builds the work
 * list on the host (L2-sized groups of (sequence, kv head) pairs, longest
 * unit first within a group) in mapped pinned memory, then launches on
 * `stream` a small upload kernel that reads it into stream-ordered device
 * scratch and one persistent kernel over min(#SMs, #units) CTAs (or, for a
 * batch split into pieces, one CTA per SM); no copy-engine transfer.  The
 * scratch (the work list, and the pieces' partial results when key ranges
 * are split: 129 fp32 per row of a piece at d = 128) is allocated with
 * cudaMallocFromPoolAsync from a memory pool the library creates per device
 * and freed on `stream`; the pool keeps up to 64 MB of freed scratch mapped
 * between calls.  The scheduler's host working arrays are kept per calling
 * thread and reused by its next call (they grow to the largest batch the
 * thread has scheduled, about 120 bytes per work unit), so that a call
 * allocates no host memory once the thread has seen a batch as large.
 * The call does not wait for the GPU, except when the host runs 32 calls
 * ahead of it: the work lists are staged in a pool of at most 32 pinned
 * buffers, and a call that finds all of them still queued for upload waits
 * for the oldest upload instead of pinning more memory.
 * Returns OPATTN_OK with no device work when total_q == 0.  `scale` must be finite and > 0 (usually
 * 1 / sqrt(d)).  Device-side wait timeouts are not reported here; use
 * opattn_prefill_checked to observe them.
 */
OPATTN_API opattn_status opattn_prefill(const void *q, const void *k, const void *v, void *o, float *lse,
                             const int32_t *cu_seqlens_q, const int32_t *cu_seqlens_k,
                             int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, float scale,
                             void *stream);

/*
 * Allocation-free variant of opattn_prefill (the paper has no counterpart;
 * this is a library convenience).  For callers that cannot have the library
 * allocate device memory: a serving engine that reserves almost all of HBM
 * for its KV cache and hands out memory only from its own pool, a process
 * whose device memory is capped by a quota, or a device without the
 * stream-ordered allocator.  Same arguments and computation as
 * opattn_prefill; the caller still provides q, k, v, o and lse.  The work
 * list and status word go to a fixed device array inside the library
 * (OPATTN_NOALLOC_MAX_UNITS work units of 52 bytes plus 8 KiB, about
 * 1.7 MB), which every GPU that loads the library keeps until the process
 * exits.  Key ranges are never split here (the array has no room for the
 * pieces' partial results), so a batch that opattn_prefill would split runs
 * as the list schedule and agrees with it within the tolerance only.  It
 * calls no cudaMalloc, cudaMallocAsync or cudaFree, and no cudaHostAlloc
 * either: the host side builds the list in ordinary heap memory and copies
 * it with cudaMemcpyAsync.
 *   - That copy from pageable memory may block the calling thread until the
 *     runtime has staged the bytes (it can wait for work already queued on
 *     `stream`); opattn_prefill, whose list sits in pinned memory, never
 *     blocks.
 *   - Not for stream capture: the copy reads heap memory that is freed when
 *     the call returns, so a captured call could not be replayed.  A call on
 *     a capturing stream returns OPATTN_ERR_INVALID_ARG before any device
 *     work; use the opattn_plan_* calls for CUDA graphs.
 *   - The first call on a device looks up the array's device address with
 *     that device current and keeps it for later calls, so cudaDeviceReset
 *     while the library is loaded is not supported.
 *   - All calls share the one array and each overwrites it: calls that
 *     overlap on the GPU (unordered streams, or several host threads) race,
 *     so order them on one stream or serialize them.
 *   - Returns OPATTN_ERR_CAPACITY, before touching the GPU, when the batch
 *     needs more than OPATTN_NOALLOC_MAX_UNITS work units (a unit is one kv
 *     head x 2 * (128 / G) query tokens of one sequence); use
 *     opattn_prefill for such batches.
 */
#define OPATTN_NOALLOC_MAX_UNITS 32768
OPATTN_API opattn_status opattn_prefill_noalloc(const void *q, const void *k, const void *v, void *o, float *lse,
                                                const int32_t *cu_seqlens_q, const int32_t *cu_seqlens_k,
                                                int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, float scale,
                                                void *stream);

/*
 * Diagnostic variant: the same computation, then it synchronizes `stream`
 * and reads back the kernel's status word; returns OPATTN_ERR_TIMEOUT if a
 * bounded wait expired.  `flags` must be 0 except in the library's own
 * failure-path tests, where OPATTN_FLAG_TEST_FORCE_TIMEOUT makes one wait of
 * every CTA run out on purpose (after ~20 ms), and
 * OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA only the one of CTA 0 (the other
 * CTAs finish their work), so that the error path is exercised without
 * hanging the GPU; outputs are then unspecified.
 */
#define OPATTN_FLAG_TEST_FORCE_TIMEOUT 1u
#define OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA 2u
OPATTN_API opattn_status opattn_prefill_checked(const void *q, const void *k, const void *v, void *o, float *lse,
                                     const int32_t *cu_seqlens_q, const int32_t *cu_seqlens_k,
                                     int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, float scale,
                                     void *stream, uint32_t flags);

/*
 * Reusable plan.  All layers of a model share the same cu_seqlens within a
 * batch, so the work list can be built and uploaded once and then run per
 * layer.  opattn_plan_create validates the geometry, builds the list for at
 * most `max_ctas` CTAs (0 = one per SM of the current device), allocates
 * device memory with cudaMalloc on the current device and copies the list
 * synchronously.  opattn_plan_run launches the kernel only (no host work
 * beyond tensor-map encoding, no allocation); it must run on the device the
 * plan was created on.  opattn_plan_destroy frees the plan after
 * synchronizing that device.  *plan is set to NULL on failure.
 */
typedef struct opattn_plan opattn_plan;
OPATTN_API opattn_status opattn_plan_create(opattn_plan **plan, const int32_t *cu_seqlens_q,
                                 const int32_t *cu_seqlens_k, int32_t n_seq, int32_t Hq,
                                 int32_t Hkv, int32_t d, int32_t max_ctas);
OPATTN_API opattn_status opattn_plan_run(const opattn_plan *plan, const void *q, const void *k, const void *v,
                              void *o, float *lse, float scale, void *stream);
OPATTN_API opattn_status opattn_plan_destroy(opattn_plan *plan);
/*
 * Diagnostic run of a packed-K/V plan (prefill or decode): zeroes the plan's
 * device status word, launches like opattn_plan_run with the test `flags` of
 * opattn_prefill_checked, synchronizes `stream` and returns
 * OPATTN_ERR_TIMEOUT if a bounded device wait expired.  Paged plans return
 * OPATTN_ERR_INVALID_ARG.
 */
OPATTN_API opattn_status opattn_plan_run_checked(const opattn_plan *plan, const void *q, const void *k,
                                                 const void *v, void *o, float *lse, float scale, void *stream,
                                                 uint32_t flags);
/* Number of work units and CTAs of a plan (either pointer may be NULL). */
OPATTN_API opattn_status opattn_plan_info(const opattn_plan *plan, int64_t *n_units, int32_t *n_ctas);

/*
 * Host-only scheduler (no GPU needed), exposed for testing and capacity
 * planning: the work list opattn_prefill and opattn_plan_create build.  A
 * work unit is (sequence, kv head, block of 2 * (128 / G) query tokens).
 * Its cost is the number of 128-key tiles it visits after whole tiles above
 * the causal diagonal are skipped, plus one.  The (sequence, kv head) pairs
 * are gathered in order into groups of at most 48 MB of K/V (so that a
 * group's K/V stays in L2); units are taken group by group, longest first
 * within a group, and each is given to the CTA with the least assigned cost
 * so far (greedy list scheduling: makespan within the mean load plus the
 * largest unit).  A CTA runs its units in that order.
 * Split-KV: when the largest units set that makespan (few units over long
 * key ranges, e.g. one prompt chunk over a long cached prefix), the key
 * tiles of all units, in pair order, are instead cut into one equal stretch
 * per CTA; a unit cut by stretch boundaries becomes pieces on consecutive
 * CTAs, each over its own run of key tiles, whose partial results the last
 * piece to finish merges in the same launch.  The cut is taken when a
 * CTA's stretch is at least 4 key tiles and its makespan, counting two more
 * per piece, is below 0.85 of the list schedule's.
 * Writes `units` as 13 int32 per unit (or piece):
 *     {first packed query row, tokens in unit, first packed key row of the
 *      sequence, Lk, last visible key of the unit's first token, kv head,
 *      key tiles visited, sequence index, first key tile visited, partial
 *      slot (-1: not split), merge group (-1: not split), piece index,
 *      pieces of the unit}
 * grouped by CTA, and cta_offsets[0..n_ctas] (unit index ranges).  n_ctas
 * used = min(n_ctas, #units) for the list schedule and min(n_ctas, key
 * tiles) for the cut, returned in *n_ctas_used.  Fails with
 * OPATTN_ERR_CAPACITY (and *n_units_out set) if unit_capacity is too small.
 */
OPATTN_API opattn_status opattn_schedule(const int32_t *cu_seqlens_q, const int32_t *cu_seqlens_k,
                              int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, int32_t n_ctas,
                              int32_t *units, int64_t unit_capacity, int32_t *cta_offsets,
                              int64_t *n_units_out, int32_t *n_ctas_used);

/*
 * Decode-shaped batches.  A decode iteration (§3.1: each iteration after
 * prefill produces one token per request, and its latency is held to the
 * TBT objective) runs the same operator with one query token per sequence
 * (a few with speculative tokens) over the sequence's whole cached key
 * range.  opattn_decode computes exactly what opattn_prefill computes, with
 * the same arguments, layouts, mask and outputs, with a kernel built for
 * that shape: it is bound by reading K and V from HBM, cuts the key ranges
 * into chunks processed in parallel (split-KV, balanced over the SMs) and
 * merges the chunks' partial results with their log-sum-exp weights inside
 * the same launch.
 *
 * Supported shapes: d = 128, G = Hq / Hkv dividing 32 (1, 2, 4, 8, 16, 32),
 * and Lq * G <= 32 for every sequence (e.g. G = 8: up to 4 query tokens per
 * sequence); anything else returns OPATTN_ERR_UNSUPPORTED before any device
 * work.  Lk may be anything, including 0 and Lk < Lq.
 *
 * Scratch: the one-shot call allocates its work list and the chunks'
 * partial results (kDecCols x d fp32 per chunk, 16 KB) on `stream` from the
 * library's memory pool (as opattn_prefill) and frees them there.  opattn_decode_checked additionally
 * waits for the stream and reports a device timeout (flags as for
 * opattn_prefill_checked).
 */
OPATTN_API opattn_status opattn_decode(const void *q, const void *k, const void *v, void *o, float *lse,
                                       const int32_t *cu_seqlens_q, const int32_t *cu_seqlens_k, int32_t n_seq,
                                       int32_t Hq, int32_t Hkv, int32_t d, float scale, void *stream);
OPATTN_API opattn_status opattn_decode_checked(const void *q, const void *k, const void *v, void *o, float *lse,
                                               const int32_t *cu_seqlens_q, const int32_t *cu_seqlens_k,
                                               int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, float scale,
                                               void *stream, uint32_t flags);
/*
 * A plan for the decode kernel: same contract as opattn_plan_create, and the
 * plan is run, queried and destroyed with opattn_plan_run / _info / _destroy.
 * The plan owns the chunk partials, so two runs of one plan must not overlap
 * (run them on one stream).  A run is one kernel launch and nothing else: the
 * plan's merge counters are zeroed when it is created and tagged with a
 * launch epoch that the kernel itself advances when the launch's last CTA
 * exits, so runs can also be captured in a CUDA graph and replayed.  A run
 * that stopped early (a device wait timed out) leaves counts under its own
 * epoch only, which later runs of the plan ignore: the plan stays usable.
 * Plan runs do not read the device status word; opattn_plan_run_checked
 * does.
 */
OPATTN_API opattn_status opattn_decode_plan_create(opattn_plan **plan, const int32_t *cu_seqlens_q,
                                                   const int32_t *cu_seqlens_k, int32_t n_seq, int32_t Hq,
                                                   int32_t Hkv, int32_t d, int32_t max_ctas);
/*
 * Paged K/V caches (the layout of paged-attention serving engines).  k_cache
 * and v_cache are device arrays [num_blocks, block_size, Hkv, d] bf16;
 * sequence s owns Lk_s = seqlens_k[s] keys (HOST array of n_seq int32), and
 * key j of s is row j % block_size of page block_table[s * max_blocks +
 * j / block_size] (block_table: DEVICE int32 [n_seq, max_blocks], read by
 * the kernel).  Everything else (q, o, lse, cu_seqlens_q, mask, outputs) is
 * as for opattn_decode.  block_size must be 8, 16, 32, 64 or 128, and every
 * sequence needs ceil(Lk_s / block_size) <= max_blocks; otherwise
 * OPATTN_ERR_UNSUPPORTED / OPATTN_ERR_INVALID_ARG before any device work.
 * Page ids are not checked on the host: an id outside [0, num_blocks)
 * makes the kernel read zeros for that page, never memory outside the
 * caches.  The rows of a sequence's last page past its last key are read
 * and weighted by zero, so they must hold finite values (any data a reused
 * page held before is fine; NaN or infinity there would reach O).
 */
OPATTN_API opattn_status opattn_decode_paged(const void *q, const void *k_cache, const void *v_cache,
                                             const int32_t *block_table, int64_t num_blocks, int32_t block_size,
                                             int32_t max_blocks, void *o, float *lse,
                                             const int32_t *cu_seqlens_q, const int32_t *seqlens_k, int32_t n_seq,
                                             int32_t Hq, int32_t Hkv, int32_t d, float scale, void *stream);
/* The prefill kernel over the same paged caches (e.g. a chunk of a prompt
 * attending to its prefix in the cache): arguments as opattn_decode_paged,
 * shapes as opattn_prefill (d = 64 or 128, G <= 128, any Lq). */
OPATTN_API opattn_status opattn_prefill_paged(const void *q, const void *k_cache, const void *v_cache,
                                              const int32_t *block_table, int64_t num_blocks, int32_t block_size,
                                              int32_t max_blocks, void *o, float *lse,
                                              const int32_t *cu_seqlens_q, const int32_t *seqlens_k, int32_t n_seq,
                                              int32_t Hq, int32_t Hkv, int32_t d, float scale, void *stream);
/* Paged plans (prefill or decode kernel): built from the host key counts,
 * run with opattn_plan_run_paged (opattn_plan_run rejects them with
 * OPATTN_ERR_INVALID_ARG, and opattn_plan_run_paged rejects other plans). */
OPATTN_API opattn_status opattn_prefill_paged_plan_create(opattn_plan **plan, const int32_t *cu_seqlens_q,
                                                          const int32_t *seqlens_k, int32_t n_seq, int32_t Hq,
                                                          int32_t Hkv, int32_t d, int32_t block_size,
                                                          int32_t max_blocks, int32_t max_ctas);
OPATTN_API opattn_status opattn_decode_paged_plan_create(opattn_plan **plan, const int32_t *cu_seqlens_q,
                                                         const int32_t *seqlens_k, int32_t n_seq, int32_t Hq,
                                                         int32_t Hkv, int32_t d, int32_t block_size,
                                                         int32_t max_blocks, int32_t max_ctas);
OPATTN_API opattn_status opattn_plan_run_paged(const opattn_plan *plan, const void *q, const void *k_cache,
                                               const void *v_cache, const int32_t *block_table,
                                               int64_t num_blocks, void *o, float *lse, float scale,
                                               void *stream);
/*
 * Host-only decode scheduler (no GPU needed).  A unit is (sequence, kv head,
 * range of 128-key tiles).  The tiles of all (sequence, kv head) pairs, in
 * order, are cut into min(n_ctas, tiles) equal stretches, one per CTA, so
 * every CTA streams the same number of tiles to within one; a pair cut by
 * stretch boundaries becomes several chunks on consecutive CTAs.  Pairs
 * without keys become zero-tile units spread over the CTAs.  Writes
 * `units` as 12 int32 per unit:
 *     {first packed query row, query tokens of the sequence, first packed key
 *      row, Lk, kv head, first key tile of the chunk, tiles in the chunk,
 *      partial slot (-1: the chunk is the whole sequence), merge group (-1),
 *      chunk index, chunks of the (sequence, kv head), sequence index}
 * and cta_offsets as opattn_schedule does.  Sequences with Lq = 0 get no unit.
 */
OPATTN_API opattn_status opattn_decode_schedule(const int32_t *cu_seqlens_q, const int32_t *cu_seqlens_k,
                                                int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d,
                                                int32_t n_ctas, int32_t *units, int64_t unit_capacity,
                                                int32_t *cta_offsets, int64_t *n_units_out,
                                                int32_t *n_ctas_used);
/*
 * The decode schedule that the one-shot decode calls and decode plans without
 * an SM budget (max_ctas = 0) build on a device with `sms` SMs.  A batch whose
 * (sequence, kv head) pairs all have the same number of key tiles takes the
 * largest grid down to 4/5 of `sms` that splits no pair, or splits every pair
 * into equal chunks.  A batch with at most `sms` pairs may instead be cut
 * pair by pair: every pair into ceil(tiles / M) nearly equal chunks, one CTA
 * each, for the smallest M that fits; that cut is taken when a cost model
 * (a CTA's key tiles, plus five tiles' time per unit in its chain, plus two
 * when a pair is split, with HBM saturated by about 96 streaming CTAs) rates
 * it no slower than the stream-K cut.  Same outputs and errors as
 * opattn_decode_schedule; `sms` must be positive.
 */
OPATTN_API opattn_status opattn_decode_schedule_default(const int32_t *cu_seqlens_q, const int32_t *cu_seqlens_k,
                                                        int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d,
                                                        int32_t sms, int32_t *units, int64_t unit_capacity,
                                                        int32_t *cta_offsets, int64_t *n_units_out,
                                                        int32_t *n_ctas_used);

#ifdef __cplusplus
}
#endif

#endif /* OPATTN_H */
