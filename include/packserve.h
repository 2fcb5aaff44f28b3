/*
 * packserve.h -- C ABI of the GB300 scheduler hot path of PackServe (KVC-first, SLO-aware request
 * packing for agentic LLM serving, arXiv 2609.33224).
 *
 * For a window of requests against every serving instance the library computes, on one GPU:
 *   1. the KV-cache prefix-hit length of each (request, instance) pair (Section 7: the scheduler's
 *      prefix tree of cached prefixes, here per-instance hash tables of chained block hashes);
 *   2. predicted TTFT and TPOT from the white-box prefill/decode model (Eq. 4-7, Eq. 9);
 *   3. the capacity guard, the normalised recompute filter (Eq. 8) and the SLO admission test
 *      (Algorithm 1), and the decode-batch-size-centric packing key or the cache-aware fallback;
 *   4. the greedy in-window assignment: requests in arrival order, each decided on the state left
 *      by the earlier decisions of the window (Section 4: state tracked along request paths).
 *
 * Conventions (all calls):
 *   - Every call returns a ps_status; on failure ps_last_error() describes the first error.
 *   - Calls are ordered on the context's CUDA stream and return after their results are in the
 *     caller's buffers (they synchronise the stream), so device-side errors surface in the same call.
 *   - Caller buffers are host memory unless the call's *_on_device flag says device memory of the
 *     context's device.  The caller owns them; the library never keeps a pointer to a host buffer.
 *     Host buffers that are page-locked (cudaHostAlloc / torch pin_memory) copy fastest.
 *   - The library owns its tables, instance state and scratch, all allocated in ps_create and
 *     released in ps_destroy.  One context must not be used from two threads at once.
 *   - Block hashes are 64-bit chained hashes: block k's hash covers the request's first 16(k+1)
 *     tokens, so a cached block hash means its whole prefix is cached.  The values 0 and
 *     0xFFFFFFFFFFFFFFFF are reserved (empty / deleted slot): ps_insert_* rejects them and a request
 *     block with either value never counts as cached.
 *   - Instance ids are 0..num_instances-1; ties are broken towards the lowest id.
 */
#ifndef PACKSERVE_H
#define PACKSERVE_H

#include <stdint.h>

#if defined(__GNUC__)
#define PS_API __attribute__((visibility("default")))
#else
#define PS_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct ps_ctx ps_ctx; /* opaque, owned by the library */

typedef enum {
  PS_OK = 0,
  PS_ERR_INVALID = 1,    /* bad argument, size or layout; nothing was changed */
  PS_ERR_CUDA = 2,       /* a CUDA runtime call failed (message in ps_last_error) */
  PS_ERR_OOM = 3,        /* device or pinned allocation failed in ps_create */
  PS_ERR_TABLE_FULL = 4, /* a hash table has no free slot left for an insert */
  PS_ERR_TIMEOUT = 5,    /* a bounded device-side wait of the greedy pass gave up (ps_set_wait_limit) */
  PS_ERR_CAPACITY = 6,   /* an instance holds more blocks than its cache capacity */
  PS_ERR_STATE = 7       /* call out of order (e.g. commit with no pending window) */
} ps_status;

enum { PS_MAX_EMA_SEGMENTS = 16, PS_BLOCK_TOKENS = 16 };

/* Performance model (Section 5; all times in ms, fp32).
 * Prefill, Eq. 6 plus the Section 5.3 empirical C and C^2 terms, evaluated in exactly this order:
 *   T_pf(N, C) = ((((a0 + a1*N) + a2*(N*C)) + a3*(N*N)) + a4*C) + a5*(C*C)
 * Decode iteration, Eq. 7:  T_iter(B, S) = (b0 + b1*B) + b2*S, scaled by the online EMA factor of
 * B's decode-batch segment (Section 5.3): segment s covers B >= seg_lo[s] (ascending, seg_lo[0] <= 1).
 * TPOT (Eq. 5), with B = b + qr + 1 and S = S_tokens + L after admission:
 *   interference_mode 0:  T_iter * f + g_q * (q_tokens + n)           (queued-prefill form)
 *   interference_mode 1:  T_iter * f + [b + qr > 0] T_pf(n, c) / max(1, lout_median)   (Eq. 9)
 * TTFT (Eq. 4, overhead neglected): T_pf(n, c) + (a0*qr + a1*q_tokens).
 * eta: recompute budget of Eq. 8 (>= 0; the paper's default is 0.5).
 * ttft_filter: 1 adds "TTFT <= max(ttft_target, T_pf(L, 0))" to the TPOT admission test of
 * Algorithm 1 (the TTFT SLO of Section 8.1 Metrics); 0 applies Algorithm 1 exactly.
 * All coefficients must be finite with magnitude <= 1e9; EMA factors finite and > 0.
 *
 * Policy variants of the evaluation (Section 8.3; all zero = Algorithm 1 as above):
 *   cache_filter_off  1: no KVC-first filter, C = A (Table 3 configurations G and T).
 *   slo_filter_off    1: no SLO admission, T = C (Table 3 G and C; the TTFT test goes with it).
 *   fallback_dcq      1: with T empty, pick over C by the D-C-Q order instead of the LMetric product
 *                     (Table 3 T and CT; path 1 as for the LMetric fallback).
 *   selector          order inside T (Table 4): PS_SELECT_DCQ (0, Section 6.2: more decoding
 *                     requests, then more cached blocks, then fewer queued requests), PS_SELECT_D,
 *                     PS_SELECT_DQ, PS_SELECT_DC, PS_SELECT_DQC, PS_SELECT_HCQ (smallest predicted
 *                     TPOT headroom tpot_target - TPOT in fp32 first, then more cached blocks, then
 *                     fewer queued requests).  Every order ends with the lowest instance id. */
enum { PS_SELECT_DCQ = 0, PS_SELECT_D = 1, PS_SELECT_DQ = 2, PS_SELECT_DC = 3, PS_SELECT_DQC = 4,
       PS_SELECT_HCQ = 5 };

typedef struct {
  float a0, a1, a2, a3, a4, a5;
  float b0, b1, b2;
  float g_q;
  float eta;
  float lout_median;
  int32_t interference_mode;
  int32_t ttft_filter;
  int32_t nseg;
  int32_t seg_lo[PS_MAX_EMA_SEGMENTS];
  float ema_factor[PS_MAX_EMA_SEGMENTS];
  int32_t cache_filter_off;
  int32_t slo_filter_off;
  int32_t fallback_dcq;
  int32_t selector;
} ps_model;

/* Context configuration (ps_create).
 *   device, cuda_stream   CUDA device ordinal and the cudaStream_t to launch on (NULL: the
 *                         library creates and owns a non-blocking stream).
 *   num_instances         1..2048 (the greedy pass keeps every instance's state in the shared memory
 *                         of one SM, about 100 bytes per instance).
 *   max_window_requests   largest R a window may have (1..131072).
 *   max_window_chain_blocks  largest total chain length (sum over requests) of a window.
 *   block_tokens          must be 16 (PS_BLOCK_TOKENS).
 *   cap_blocks            host array [num_instances]: cache capacity of each instance in blocks.
 *   table_load_factor     slots of instance i = ceil(cap_blocks[i] / table_load_factor), rounded
 *                         up to whole 8-slot (64-byte) buckets; (0, 0.95].
 *   model                 the performance model above.
 *   probe_mode            how hit lengths are found (both give the same hits on the caches they
 *                         accept):
 *     PS_PROBE_LINEAR  (0) walk the chain 32 blocks per warp step until the first block that is
 *                          not cached; exact for any cache contents.
 *     PS_PROBE_SEARCH  (1) the caches must be prefix-closed (every cached block's parent is
 *                          cached, as in the paper's Section 7 prefix tree).  Then "block k is
 *                          cached" is monotone along a chain, so the first miss is found by search:
 *                          each lane binary-searches one instance (about log2(chain length)
 *                          lookups per pair), and the continuation of a chain past an earlier
 *                          request's end is found by a warp's 32-ary search (32 evenly spaced
 *                          lookups per step).  ps_insert_* checks the closure: a chain whose
 *                          parent_hash is neither 0 nor cached after the call fails with
 *                          PS_ERR_INVALID.
 *   track_lru             1: keep per-block (last_use, child count, parent) metadata so that
 *                         ps_advance_window can evict leaf-first LRU (the tables must then hold fewer
 *                         than 2^32 - 2 slots in total); 0: no eviction.
 *   max_active_requests   0: no request tracking.  > 0: each instance keeps up to this many queued
 *                         and this many decoding requests for ps_advance_window (streaming windows);
 *                         committed windows then need ps_window.out_tokens. */
enum { PS_PROBE_LINEAR = 0, PS_PROBE_SEARCH = 1 };

typedef struct {
  int32_t device;
  void* cuda_stream;
  uint32_t num_instances;
  uint32_t max_window_requests;
  uint64_t max_window_chain_blocks;
  uint32_t block_tokens;
  const uint64_t* cap_blocks;
  float table_load_factor;
  ps_model model;
  int32_t probe_mode;
  int32_t track_lru;
  uint32_t max_active_requests;
} ps_config;

/* Scheduler-tracked state of one instance (Section 4 Metadata service; Section 6.2):
 * b decoding requests, qr queued (not yet decoding) requests, q_tokens queued uncached prefill
 * tokens, S_tokens KV tokens held by the active requests, M_KV_tokens KV capacity, B_max decode-slot
 * limit.  Capacity guard of Algorithm 1: b + qr + 1 <= B_max and S_tokens + L <= M_KV_tokens.
 * Limits: 0 <= b, qr < 2^17; 0 <= q_tokens < 2^40; 0 <= S_tokens, M_KV_tokens < 2^50. */
typedef struct {
  int32_t b, qr;
  int64_t q_tokens, S_tokens, M_KV_tokens;
  int32_t B_max;
} ps_instance_state;

/* One window of requests in arrival order (Algorithm 1's request r: a session's token prefix as a
 * chain of block hashes, plus its SLO targets).
 *   chain_off      [R+1], chain_off[0] = 0, non-decreasing; request r's chain is
 *                  chain_hash[chain_off[r] .. chain_off[r+1]) (with parent: its own blocks, below).
 *   chain_hash     [chain_off[R]] block hashes.
 *   prompt_tokens  [R] input length L_r in tokens; its chain must have exactly L_r / 16 blocks
 *                  (full blocks only).  L_r < 2^30.
 *   ttft_target, tpot_target  [R] per-request SLO targets in ms.
 *   out_tokens     [R] output length of each request (only read by ps_commit_window on a context
 *                  with request tracking, to queue the admitted requests; may be NULL otherwise).
 *   inputs_on_device  0: all arrays are host memory, 1: all are device memory.
 *   parent         [R] or NULL.  The shared-prefix (prefix-tree) form of the window: an agentic
 *                  session resends its whole history with every step (Section 3), so a request's
 *                  prompt usually extends an earlier request's.  parent[r] = p (0 <= p < r) says that
 *                  request r's chain starts with request p's whole chain, and chain_hash[chain_off[r]
 *                  .. chain_off[r+1]) then holds only the blocks after it (L_r/16 - L_p/16 of them);
 *                  parent[r] = -1 gives the whole chain as usual.  The library rebuilds every chain on
 *                  the device (one pass over the window), so the host sends each shared prefix once.
 *                  Host inputs only (inputs_on_device 0); NULL: every chain is given whole.
 * A window with device inputs is read in place; its buffers must stay unchanged until the window is
 * committed or discarded (ps_commit_window / the next ps_schedule_window). */
typedef struct {
  uint32_t R;
  const uint64_t* chain_off;
  const uint64_t* chain_hash;
  const uint32_t* prompt_tokens;
  const float* ttft_target;
  const float* tpot_target;
  const uint32_t* out_tokens;
  int32_t inputs_on_device;
  const int32_t* parent;
} ps_window;

/* Per-pair and per-request scoring outputs.  Any pointer may be NULL (not wanted).
 *   hits  [R*I] row-major (request-major) prefix-hit length in blocks.
 *   tpot, ttft  [R*I] predicted latencies in ms (computed for every pair).
 *   cls   [R*I] 0: in T (capacity, recompute and SLO tests pass), 1: in C but not T,
 *               2: in A but filtered by Eq. 8, 3: not capacity-eligible (not in A).
 *   best  [R] Algorithm 1's pick against the current state, -1 = Reject.
 *   path  [R] 0: packed (from T), 1: fallback (CacheAwareLB over C), 2: Reject.
 *   outputs_on_device  0: host buffers, 1: device buffers. */
typedef struct {
  uint32_t* hits;
  float* tpot;
  float* ttft;
  uint8_t* cls;
  int32_t* best;
  uint8_t* path;
  int32_t outputs_on_device;
} ps_scores;

/* Greedy decisions of a window (ps_schedule_window).
 *   assign      [R] chosen instance, -1 = Reject.
 *   path        [R] 0 packed, 1 fallback, 2 reject.
 *   hit_chosen  [R] prefix-hit length (blocks) on the chosen instance at decision time (0 on reject).
 * Any pointer may be NULL.  outputs_on_device as in ps_scores. */
typedef struct {
  int32_t* assign;
  uint8_t* path;
  uint32_t* hit_chosen;
  int32_t outputs_on_device;
} ps_decisions;

/* Create a context: the scheduler of Section 4 (System overview) with the per-instance prefix caches
 * of Section 7 (Implementation: the scheduler's prefix tree of cached prefixes, here one hash table of
 * chained block hashes per instance) and the performance model of Section 5.  Allocates every table
 * and buffer up front (instance hash tables sized by cap_blocks / table_load_factor, a window-scoped
 * delta table of 2 * max_window_chain_blocks slots, window staging and score scratch).  Instances
 * start empty with zero state.  cfg is read during the call only.
 * Errors: PS_ERR_INVALID (config), PS_ERR_CUDA, PS_ERR_OOM.  *out is NULL on failure. */
PS_API ps_status ps_create(const ps_config* cfg, ps_ctx** out);

/* Replace the committed state of all instances (host array of n = num_instances entries): the
 * per-instance records the paper's metadata service keeps (Section 4, "Metadata service": running
 * decode batch, queued requests and prefill tokens, KV usage and capacity).  Discards any pending
 * window.  Errors: PS_ERR_INVALID (n or a field out of range); the state is unchanged then. */
PS_API ps_status ps_load_instances(ps_ctx* ctx, const ps_instance_state* s, uint32_t n);

/* Read the committed state (host array of n = num_instances entries): the Section 4 metadata-service
 * records as the library holds them after the last commit or load. */
PS_API ps_status ps_get_instances(ps_ctx* ctx, ps_instance_state* out, uint32_t n);

/* Online calibration of the decode model (Section 5.3, "Online calibration"): feed n pure-decode
 * feedback samples, in order (host arrays): batch[k] the measured decode batch size, ctx_tokens[k]
 * the total context tokens of the batch, measured_ms[k] the forward's duration.  For each, the base
 * prediction (b0 + b1 B) + b2 S at the same B and S gives the measured-to-predicted ratio, clipped
 * to [0.5, 2]; the EMA factor of B's decode-batch segment (ps_model.seg_lo) moves towards it by
 * `weight` (the paper uses 0.02), f <- f + weight (ratio - f), and is clipped to [1, 2].  The
 * factors scale the decode term of every later TPOT prediction of the context.  Host-side only (no
 * device work, no synchronisation).  PS_ERR_INVALID for n > 0 with a NULL array, a batch size below
 * 0, a context below 0, a non-finite or non-positive duration, or a weight outside (0, 1]. */
PS_API ps_status ps_calibrate(ps_ctx* ctx, uint32_t n, const int32_t* batch, const int64_t* ctx_tokens,
                              const float* measured_ms, float weight);

/* The current EMA factors of Section 5.3's online calibration, one per decode-batch segment (host
 * array of n >= ps_model.nseg entries; entries past nseg are left untouched). */
PS_API ps_status ps_get_ema_factors(ps_ctx* ctx, float* out, uint32_t n);

/* Replace the performance model (Section 5 coefficients, eta of Eq. 8, the TTFT filter, the EMA
 * segments and factors) with the same checks as ps_create.  The new model's EMA factors replace
 * what ps_calibrate has learned.  Takes effect at the next ps_score_window, ps_schedule_window or
 * ps_advance_window; a pending window keeps the decisions it was made with.  Host-side only (no
 * device work).  Used, for instance, to sweep the recompute budget eta over one window (the
 * sensitivity study of Section 8) without rebuilding the tables.
 * Errors: PS_ERR_INVALID (NULL model or a field out of range; the previous model stays). */
PS_API ps_status ps_set_model(ps_ctx* ctx, const ps_model* model);

/* Bound on every cross-block wait of the greedy pass (ns; 0 restores the default of 1 s; at most
 * 60 s).  The greedy's thread blocks hand decisions, inserts and probed hits to one another through
 * flags in device memory (Section 4's per-request state tracking, run as a pipeline); a block that
 * waits longer than this records the failure and returns, so a launch always ends, and the call
 * returns PS_ERR_TIMEOUT with the window's outputs undefined and no pending window.  The context
 * stays usable: the next call starts from the committed state.  Host-side only.
 * Errors: PS_ERR_INVALID (ns above 60 s). */
PS_API ps_status ps_set_wait_limit(ps_ctx* ctx, uint64_t ns);

/* Read the state a pending window would commit (the committed state updated by each of the
 * window's admitted requests: qr += 1, q_tokens += n, S_tokens += L, the per-decision state update
 * of Section 4's request-path tracking).  PS_ERR_STATE if none. */
PS_API ps_status ps_get_pending_instances(ps_ctx* ctx, ps_instance_state* out, uint32_t n);

/* Cache a chain of n blocks on instance inst (host array): a path of the instance's prefix tree
 * (Section 7, Implementation), block 0 continuing parent_hash (0 = the chain starts at the root) and
 * block k continuing block k-1.  Blocks already cached are skipped.
 * last_use stamps the blocks for LRU bookkeeping.
 * Errors: PS_ERR_INVALID (inst, reserved hash, or in PS_PROBE_SEARCH mode a parent_hash that is not
 * cached once the call's blocks are in), PS_ERR_TABLE_FULL (no slot left), PS_ERR_CAPACITY (the
 * instance now holds more than cap_blocks blocks).  On any of these errors the blocks that could be
 * inserted stay cached. */
PS_API ps_status ps_insert_blocks(ps_ctx* ctx, uint32_t inst, const uint64_t* chain, uint64_t n,
                           uint64_t parent_hash, uint32_t last_use);

/* Bulk form of ps_insert_blocks (Section 7 prefix-tree paths) over nchains chains in CSR form: chain c goes to instance inst[c],
 * its blocks are hash[off[c] .. off[c+1]) and its first block continues parent[c].  on_device
 * selects host (0) or device (1) arrays.  Same errors as ps_insert_blocks. */
PS_API ps_status ps_insert_chains(ps_ctx* ctx, uint64_t nchains, const uint32_t* inst, const uint64_t* off,
                           const uint64_t* hash, const uint64_t* parent, uint32_t last_use,
                           int32_t on_device);

/* Number of blocks cached on each instance's prefix cache (Section 7; host array
 * [n = num_instances]). */
PS_API ps_status ps_cached_blocks(ps_ctx* ctx, uint64_t* out, uint32_t n);

/* Score a window: Algorithm 1 (Section 6) for every request independently against the committed
 * state (no state change), with the hit lengths of Section 7's prefix caches and the latencies of
 * Eq. 4-9.
 * Runs the probe kernel (hit lengths of all R x I pairs) and the fused score kernel (latencies,
 * filters, packing key and per-request argmin).  Errors: PS_ERR_INVALID (window layout, R too
 * large, chain length != L/16, total blocks too large), PS_ERR_CUDA. */
PS_API ps_status ps_score_window(ps_ctx* ctx, const ps_window* w, ps_scores* out);

/* Greedy in-window assignment (Algorithm 1 per request in arrival order, each admitted request
 * updating its instance's state and caching its blocks there before the next decision).
 * The result is a pending window: the committed state and caches are unchanged until
 * ps_commit_window; the next ps_schedule_window or ps_load_instances discards it.
 * opt_scores (may be NULL) receives the window's independent scores against the committed state
 * (hits = the hit lengths before the window; best/path as ps_score_window).
 * Errors: as ps_score_window, plus PS_ERR_TABLE_FULL if the delta table overflowed (cannot happen
 * within max_window_chain_blocks). */
PS_API ps_status ps_schedule_window(ps_ctx* ctx, const ps_window* w, ps_decisions* out,
                             ps_scores* opt_scores);

/* ---- Column-block scoring (one instance pool split over several contexts) ---------------------
 * Algorithm 1 (Section 6) maps every instance to a pair evaluation and then reduces each request's
 * row twice: W_min over the capacity-eligible set A (the KVC-first filter's reference, Eq. 8), then
 * the smallest packing key over C (Section 6.2's order inside T, the LMetric fallback over C when T
 * is empty).  Both reductions are minima, so a pool whose instances are split into column blocks,
 * one context each (for instance one per GPU), scores a window in two exchanges:
 *   1. every block calls ps_shard_wmin; the caller takes the minimum of wmin_ord over the blocks
 *      (an all-reduce MIN of u32 words);
 *   2. every block calls ps_shard_pick with that minimum; the caller takes, per request, the
 *      smallest key over the blocks and, among the blocks holding it, the smallest tie word (two
 *      all-reduce MINs).  The request's pick is then the tie word's instance id (its low 12 bits
 *      under PS_SELECT_HCQ, the whole word otherwise), Reject when the key is all ones or the pool's
 *      W_min is all ones; its path is key >> 62.
 * The result equals ps_score_window over the whole pool.  The greedy assignment does not split this
 * way (each decision needs the previous one): ps_schedule_window runs on a context holding the whole
 * pool.
 *
 * ps_shard_wmin: runs the probe phase of ps_score_window on this context's instances and writes, per
 * request, W_min over this block's A as order-preserving bits (float bits b with the sign bit set ->
 * ~b, else b | 0x80000000, so unsigned order = float order), 0xFFFFFFFF when the block's A is empty.
 * wmin_ord [R] is host (on_device 0) or device (1) memory.  The window's hit lengths stay in the
 * context for the ps_shard_pick that follows; a window with device inputs must stay unchanged until
 * then.  Errors: as ps_score_window, PS_ERR_INVALID for a NULL wmin_ord. */
PS_API ps_status ps_shard_wmin(ps_ctx* ctx, const ps_window* w, uint32_t* wmin_ord, int32_t on_device);

/* ps_shard_pick: the second half of the last ps_shard_wmin's window.  wmin_ord [R] is the pool's
 * W_min (the minimum over the blocks, same encoding); key [R] receives this block's smallest packed
 * key over C under that W_min (all ones if none): class in the top two bits (0 in T, 1 in C \ T),
 * then the order's fields, so the unsigned order of keys is Algorithm 1's order; tie [R] receives its
 * tie word with the pool instance id id_base + local id (all ones if none).  wmin_ord, key and tie are
 * host (on_device 0) or device (1) memory.  opt (may be NULL) receives this block's columns of
 * ps_score_window's outputs under the pool's W_min (hits, tpot, ttft, cls; best is this block's own
 * pick in local ids, path its path).  Must follow ps_shard_wmin with no call in between that scores
 * or schedules a window or changes the context's state, caches or model (PS_ERR_STATE otherwise).  Errors: PS_ERR_INVALID (NULL arrays,
 * id_base + num_instances above 2^31 - 1, or above 4096 under PS_SELECT_HCQ), PS_ERR_STATE. */
PS_API ps_status ps_shard_pick(ps_ctx* ctx, const uint32_t* wmin_ord, uint32_t id_base, uint64_t* key, uint32_t* tie,
                               int32_t on_device, ps_scores* opt);

/* Commit the pending window (Section 4: the gateway updates the instance records along the
 * request path): the pending state becomes the committed state and each admitted
 * request's uncached blocks are cached on its instance.  With track_lru every block of an admitted
 * request's chain on its instance (cached prefix and new blocks) gets last_use; with request
 * tracking each admitted request joins its instance's FIFO queue (remaining prefill = its uncached
 * tokens, output length from out_tokens).  The window's buffers are read again here.  An instance
 * may end above its cache capacity (ps_cached_blocks shows it) until ps_advance_window evicts.
 * Errors: PS_ERR_STATE (no pending window), PS_ERR_TABLE_FULL (no free slot left),
 * PS_ERR_CAPACITY (an instance's request queue is full); the state is committed in every case. */
PS_API ps_status ps_commit_window(ps_ctx* ctx, uint32_t last_use);

/* ---- Streaming windows (between-window progress) ----------------------------------------------
 * The paper's gateway tracks requests along their request and response paths (Section 4); the
 * engine's progress between two windows is simulated with these rules (the serving engine's
 * behaviour, which the paper leaves to the engine):
 *   1. every decoding request emits k = max(1, floor(window_ms / ((b0 + b1 b) + b2 S))) tokens
 *      (fp32, b and S at the window start); S grows by the tokens emitted; a request whose output
 *      is exhausted leaves (b -= 1, S -= L + out);
 *   2. each instance's queue drains prefill_tokens tokens in FIFO order; a request whose prefill
 *      completes starts decoding (qr -= 1, b += 1, q falls by the tokens drained);
 *   3. with evict = 1 (needs track_lru): while an instance holds more blocks than its capacity,
 *      its leaf block (no cached child) with the smallest (last_use, hash) is evicted. */

/* Requests in flight at the start of a stream (Section 4's request-path tracking; context created
 * with max_active_requests > 0),
 * host arrays of n entries: instance, state (0 queued, in FIFO order per instance; 1 decoding),
 * prompt tokens L, output tokens out, rem (queued: remaining prefill tokens; decoding: remaining
 * output tokens, 1..out).  Replaces all tracked requests; the committed state's b, qr, q_tokens
 * and S_tokens are recomputed from them (S = queued L + decoding L + tokens already emitted).
 * Errors: PS_ERR_INVALID (bad instance, state or rem), PS_ERR_CAPACITY (more than
 * max_active_requests of one kind on an instance), PS_ERR_STATE (no request tracking). */
PS_API ps_status ps_load_requests(ps_ctx* ctx, uint64_t n, const uint32_t* inst, const uint32_t* state,
                                  const uint32_t* L, const uint32_t* out, const uint64_t* rem);

typedef struct {
  float window_ms;          /* engine time between two windows (ms), > 0 */
  uint64_t prefill_tokens;  /* prefill tokens each instance processes in that time */
  int32_t evict;            /* 1: evict to capacity (needs track_lru) */
} ps_advance_params;

/* Advance every instance by one window (rules above: Section 4's response-path updates, with the
 * engine's progress simulated).  Errors: PS_ERR_STATE (a scheduled window
 * is still pending, or no request tracking), PS_ERR_INVALID (params), PS_ERR_CAPACITY (a decoding
 * list is full), PS_ERR_TABLE_FULL (an instance has more leaves than the eviction buffer holds,
 * 4096; its eviction stops), PS_ERR_TIMEOUT (an eviction block's metadata-prefetch warp found no
 * work for 1 s, which a round of at most 1536 evictions never takes; the evictions already made
 * stand, with counts and parent links consistent, and no further round runs). */
PS_API ps_status ps_advance_window(ps_ctx* ctx, const ps_advance_params* p);

/* Scheduling overhead, the quantity Section 8.3.3 reports as arrival-to-decision latency: device
 * time in ms (CUDA events recorded on the context's stream around each kernel) of the last
 * ps_score_window / ps_schedule_window call and of the commit after it: ms[0] probe phase (relations
 * + both probe kernels), ms[1] fused score, ms[2] greedy, ms[3] commit; with n >= 7 also the probe
 * phase's parts: ms[4] relations kernel, ms[5] probe of the rows searched from scratch, ms[6] probe
 * of the derived rows.  -1 where that kernel did not run.  n must be >= 4; entries past 7 are left
 * untouched. */
PS_API ps_status ps_last_timings(ps_ctx* ctx, float* ms, uint32_t n);

/* Counters of the last probe phase (the Section 7 prefix-cache lookups of ps_score_window /
 * ps_schedule_window), for roofline accounting
 * (host array of n >= 6 entries):
 *   out[0] rows searched from scratch        out[1] rows derived from an earlier request's row
 *   out[2] table lookups in scratch rows     out[3] table lookups in derived rows
 *   out[4] chain blocks read from global memory (a lookup's key, or a block staged in shared memory)
 *   out[5] (row, instance) pairs searched past the earlier request's chain (derived rows)
 * Of the last ps_schedule_window in PS_PROBE_SEARCH mode (else 0), where n reaches them:
 *   out[6] decisions taken from a row summary corrected for the recent picks
 *   out[7] decisions that needed a full pass over the row
 *   out[8..15] SM clock cycles, summed over the thread blocks of each role of the greedy pass: the
 *          deciding warp waiting for staged rows, the deciding warp in all, its feeder waiting for a
 *          free staging slot, the feeder waiting for published row summaries, the summary blocks
 *          waiting for published decisions, waiting for probed rows, and evaluating rows, the probe
 *          blocks waiting for the inserts of earlier decisions
 * A table lookup reads the key's two candidate buckets (2 x 64 bytes) and one overflow word.
 * All zero if no probe phase ran.  Synchronises the context's stream. */
PS_API ps_status ps_last_probe_stats(ps_ctx* ctx, uint64_t* out, uint32_t n);

/* ---- Scoring without device allocation ------------------------------------------------------
 * The paper has no counterpart to this call; it exists for callers that cannot allocate device
 * memory: a serving process whose memory manager reserves the GPU at start-up (leaving the rest to
 * the KV cache) and forbids later allocations, or a scheduler loop that must not call cudaMalloc
 * because an allocation can synchronise the device and stall the serving streams.  Such callers
 * cannot create a context (ps_create allocates), so this call takes every buffer from the caller
 * and needs no context.
 *
 * It computes what ps_score_window computes (probe kernel + fused score kernel, same results) for
 * caches laid out the way the library lays them out:
 *   slots    device u64 array holding every instance's table, 16-byte aligned; value 0 = empty
 *            slot.  0 and 0xFFFFFFFFFFFFFFFF are reserved key values: a request block with either
 *            value never counts as cached (its hit ends there), so a block hash must avoid both.
 *   overflow_bits  device u64 array of overflow bitmaps, one bit per bucket (8-byte aligned).
 *   tables   device array [num_instances] of ps_table_desc (8-byte aligned): instance i's table is
 *            num_buckets >= 1 buckets of 8 slots starting at slot `base`, a multiple of 8 (whole
 *            buckets), and its overflow bitmap starts at word `overflow_base` of overflow_bits (bit b
 *            of the bitmap = word b / 64, bit b % 64).  Every table and bitmap must lie inside the
 *            caller's arrays (the library cannot see their sizes); a descriptor with num_buckets 0 or
 *            a base that is not a multiple of 8 is rejected (PS_ERR_INVALID) before any lookup.
 *            A block hash h has two candidate buckets, b1 = (h * num_buckets) >> 64 and
 *            b2 = (g * num_buckets) >> 64 with g = (h ^ (h >> 31)) * 0x7FB5D329728EA185 mod 2^64
 *            (high 64 bits of the 128-bit products), and is stored in one of them; if both were
 *            full when it was inserted, it is stored in the first bucket after b1 (wrapping) that
 *            had a free slot, and b1 and every bucket passed on the way carry overflow bit 1.
 *   state    device arrays of the instance state (ps_instance_state fields, structure of arrays).
 *   window   inputs_on_device must be 1 and parent NULL; out->outputs_on_device must be 1 (all
 *            device buffers).
 *   probe_mode  as ps_config.probe_mode (PS_PROBE_SEARCH only for prefix-closed caches).
 *   cuda_stream  the stream to run on; the call synchronises it before returning.
 * The hit matrix it needs in between is kept in a fixed device array inside the library
 * (PS_NOALLOC_MAX_PAIRS u32 entries, 8 MiB, held on every GPU that loads the library until the
 * process exits), so R * num_instances may not exceed PS_NOALLOC_MAX_PAIRS (split larger windows).
 * The first call on each device resolves that array's device address; make that first call before
 * any stream capture.  All calls share the one array: calls that overlap on the GPU (other threads
 * or streams) race and must be serialised by the caller.  The call allocates nothing (no
 * cudaMalloc, cudaFree or allocating library routine).
 * Errors: PS_ERR_INVALID (NULL or host buffers, misaligned arrays, a bad table descriptor, sizes
 * beyond the limit, bad window layout or model), PS_ERR_CUDA.  No context exists, so there is no
 * message for ps_last_error. */
#define PS_NOALLOC_MAX_PAIRS 2097152u

typedef struct {
  uint64_t base;
  uint64_t overflow_base;
  uint32_t num_buckets;
  uint32_t reserved;
} ps_table_desc;

typedef struct {
  const int32_t* b;
  const int32_t* qr;
  const int64_t* q_tokens;
  const int64_t* S_tokens;
  const int64_t* M_KV_tokens;
  const int32_t* B_max;
} ps_state_arrays;

PS_API ps_status ps_score_window_noalloc(const uint64_t* slots, const uint64_t* overflow_bits,
                                         const ps_table_desc* tables, uint32_t num_instances,
                                         const ps_state_arrays* state,
                                         const ps_window* window, const ps_model* model,
                                         int32_t probe_mode, ps_scores* out, void* cuda_stream);

/* Text of the last error on this context ("" if none).  Valid until the next call.  Error
 * reporting only: the paper has no counterpart. */
PS_API const char* ps_last_error(const ps_ctx* ctx);

/* Release every resource of the context (its prefix-cache tables of Section 7 and the scheduler
 * state of Section 4): waits for the context's stream, then frees every allocation.  NULL is
 * accepted.  The context pointer is invalid afterwards. */
PS_API void ps_destroy(ps_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* PACKSERVE_H */
