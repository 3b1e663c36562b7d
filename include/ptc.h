/*
 * ptc.h — prefix-cache curves on one GPU (GB300, sm_103a).
 *
 * Turns a request trace into block-level LRU prefix-cache hit curves and
 * compute-saved curves for every capacity at once, after "When Fancy Eviction
 * Fails: Rethinking Cache Replacement For LLM Prefix Reuse":
 *
 *   trace (session, timestamp, tokens)       Sec. 3.1 (traces), Sec. 2.3 (sessions)
 *     -> ptc_hash_blocks     chained per-block prefix keys     Sec. 2.2 (block identity)
 *     -> ptc_assign_ids      dense block ids                   Sec. 4 ("each KV block is a distinct cache object")
 *     -> ptc_reuse_indices   previous / next use of each block Sec. 3.2, 5.2 (Belady's next access)
 *     -> ptc_stack_distance  LRU stack distance of each access App. B ("reuses reachable within C")
 *     -> ptc_curves          hits and compute saved per C      Sec. 3.2 (hit ratio), Sec. 5.2 (compute savings)
 *   with Belady's offline optimum from the same reuse indices,
 *        ptc_belady_curves                                     Sec. 3.2 (offline ceiling)
 *   and session-level instead of block-level eviction,
 *        ptc_session_lru_curves                                Sec. 5.3 (eviction granularity)
 *   with, for the semantics variants (touch order, whole-request residency),
 *        ptc_stack_distance_variant                           Sec. 3.1 (simulator)
 *   and, over the same arrays,
 *        ptc_trace_stats     lifetimes, reuse intervals, frequency, block categories,
 *                            session lengths, reuses reachable within C
 *                                                              Sec. 4.1-4.3, App. B
 *
 * Conventions shared by every call
 *   - Pointers are caller-owned DEVICE memory unless the name ends in _host.
 *     The library allocates no device memory: each call takes a device
 *     workspace `ws` of at least ptc_<call>_workspace_bytes(...) bytes,
 *     256-byte aligned.  The workspace holds no state between calls.
 *   - Host staging: the first call made by a host thread allocates one small
 *     page-locked, device-mapped block for that thread (cudaHostAlloc, about
 *     110 KB), through which status words and results reach the host without
 *     a copy-engine transfer.  It lives until ptc_release_host_staging() is
 *     called on that thread (the next call allocates it again).  Like any
 *     cudaHostAlloc, that first allocation may synchronize the device, so a
 *     serving loop should make one call before it starts.  If page-locked
 *     memory cannot be had, ordinary thread-local memory is used instead.
 *     ptc_curves_noalloc never allocates it.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Work is
 *     enqueued on it.  Every call returns after reading its device status
 *     word, so it synchronizes `stream` once before returning; outputs are
 *     ready when it returns PTC_OK.
 *   - Errors are returned, never thrown or aborted.  Device-side checks
 *     (ordering, ranges, bounded waits) set a status word that the call reads
 *     before returning.  A CUDA runtime error maps to PTC_ERR_CUDA.  On any
 *     error the contents of the outputs are unspecified.
 *   - Sizes: the number of block accesses N and of distinct blocks D must be
 *     below 2^32 - 1 (0xFFFFFFFF is the "none / infinite" marker, PTC_NONE);
 *     token counts and offsets are 64-bit.
 *   - Indices are 0-based.  The access stream is requests in trace order and,
 *     within a request, blocks root-first (depth k = 0, 1, ...).
 */
#ifndef PTC_H
#define PTC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define PTC_NONE 0xFFFFFFFFu
#define PTC_MAX_BLOCK_SIZE 512u
#define PTC_MAX_CAPACITIES 1024u

typedef enum {
  PTC_OK = 0,
  PTC_ERR_INVALID_ARG = 1,    /* a host-checked argument is out of range, or device data is malformed */
  PTC_ERR_UNSORTED = 2,       /* request timestamps decrease */
  PTC_ERR_OVERFLOW = 3,       /* N or D would reach 2^32 - 1, or a cost constant overflows 64 bits */
  PTC_ERR_WORKSPACE = 4,      /* ws is NULL, misaligned or smaller than the size query returned */
  PTC_ERR_CUDA = 5,           /* a CUDA runtime call failed */
  PTC_ERR_TIMEOUT = 6,        /* a device-side wait gave up (bounded spin); no result */
  PTC_ERR_HASH_COLLISION = 7, /* ptc_verify_ids found two different prefixes under one id */
  PTC_ERR_NOT_IMPLEMENTED = 8,
  PTC_ERR_BOUNDS = 9          /* checked build only: an index read from data fell outside its array */
} ptc_status;

/* Unsigned 128-bit integer, little-endian halves. */
typedef struct {
  uint64_t lo, hi;
} ptc_u128;

/*
 * Per-block recompute cost (Sec. 5.2 "compute-savings ratio"; App. C linear
 * model).  Block k (0-based depth) of a request with block size B costs
 *   PTC_COST_UNIFORM   1                                   (compute saved = hits)
 *   PTC_COST_MEASURED  B*f_lin + f_attn * sum_{t=Bk}^{Bk+B-1} (t+1)
 *   PTC_COST_LINEAR    f_attn * sum_{t=Bk}^{Bk+B-1} (t+1)  (attention term only)
 * The sum counts, for each token of the block, the positions it attends to.
 * The measured-shape constants for a 48-layer, 32-head, head-dim-128 MoE with
 * ~3.3B active parameters are f_lin = 2*3.3e9 and f_attn = 4*48*32*128.
 */
enum { PTC_COST_UNIFORM = 0, PTC_COST_MEASURED = 1, PTC_COST_LINEAR = 2 };
typedef struct {
  uint64_t f_lin;
  uint64_t f_attn;
  int32_t kind;
} ptc_cost_model;

/* Human-readable name of a status code (static storage). */
const char* ptc_strerror(ptc_status s);
/* Library version string (static storage). */
const char* ptc_version(void);

/*
 * ptc_hash_blocks — chained block keys (Sec. 2.2: KV state is kept in blocks of
 * B tokens, 16 in the paper's setup, and a cached block is reusable iff its
 * entire preceding sequence matches).
 *
 * Request r owns tokens[req_tok_off[r] : req_tok_off[r+1]] and has
 * n_r = floor(len_r / B) full blocks; a trailing partial block is not a cache
 * object.  Block k of request r gets the key of its whole prefix
 * [0, B(k+1)):  sum over t < B(k+1) of (tok_t + 1) * u^(t+1)  mod 2^61 - 1,
 * at two bases u_0, u_1 drawn from `seed` with SplitMix64
 * (u_b = 2 + (output b) mod (2^61 - 4)).  keys_out[i].lo / .hi are the values
 * at u_0 / u_1.  Every coefficient tok + 1 is nonzero, so two different
 * prefixes of at most m tokens (of equal or different length) share a key
 * with probability at most (m / (2^61 - 1))^2 (the Schwartz-Zippel bound for
 * each base); ptc_verify_ids checks exactly.
 *
 *   tokens          u32[n_tok]; any alignment (16-byte aligned is fastest)
 *   req_tok_off     u64[n_req + 1], non-decreasing, req_tok_off[n_req] <= n_tok
 *   req_ts_us       i64[n_req] arrival times, must be non-decreasing
 *                   (PTC_ERR_UNSORTED otherwise); may be NULL to skip the check
 *   block_size      B in [1, PTC_MAX_BLOCK_SIZE]
 *   keys_out        ptc_u128[keys_cap]; keys_cap >= N is required, and
 *                   floor(n_tok / B) always suffices
 *   req_blk_off_out u64[n_req + 1]: first access index of each request; [n_req] = N
 *   n_access_host_out  receives N on the host
 */
size_t ptc_hash_blocks_workspace_bytes(uint32_t n_req, uint64_t n_tok, uint32_t block_size);
ptc_status ptc_hash_blocks(const uint32_t* tokens, uint64_t n_tok, const uint64_t* req_tok_off,
                           const int64_t* req_ts_us, uint32_t n_req, uint32_t block_size, uint64_t seed,
                           ptc_u128* keys_out, uint64_t keys_cap, uint64_t* req_blk_off_out,
                           uint64_t* n_access_host_out, void* ws, size_t ws_bytes, void* stream);

/*
 * ptc_assign_ids — dense block ids (Sec. 4: each KV block is a distinct cache
 * object).  ids_out[i] in [0, D), numbered by first occurrence in the access
 * stream: the first access with a given key gets the next unused id.  Equal
 * keys get equal ids.  D is returned in n_distinct_host_out.
 *
 *   keys      ptc_u128[n] from ptc_hash_blocks (values below 2^61 - 1 in both halves)
 *   ids_out   u32[n]
 */
size_t ptc_assign_ids_workspace_bytes(uint64_t n);
ptc_status ptc_assign_ids(const ptc_u128* keys, uint64_t n, uint32_t* ids_out, uint64_t* n_distinct_host_out,
                          void* ws, size_t ws_bytes, void* stream);

/*
 * ptc_assign_ids_prior — the ids of ptc_assign_ids, with a prior-request hint
 * that saves work: fewer keys to settle in the table or the partitions.  Sec. 2.3: a turn of a multi-turn session sends
 * the whole context again, so request r usually repeats every block of an
 * earlier request of its session and appends to it.  req_prior[r] names such
 * an earlier request (or PTC_NONE).  The leading depths of r whose keys
 * equal those of the same depths of req_prior[r] are repeats: they are not
 * settled (inserted into the table, or moved into the partitions of the
 * partitioned dedup) and take their ids from the prior request's chain;
 * only the other accesses are settled.  The keys must be prefix keys as
 * ptc_hash_blocks writes them (equal keys at depth k imply equal keys at
 * every depth below k), so the end of that leading run is found by a binary
 * search over the depths, reading about 2 log2(n_r) keys per request rather
 * than the prior request's key of every access.  The ids are then exactly
 * those of ptc_assign_ids for ANY hint with req_prior[r] < r or PTC_NONE (a
 * poor hint only costs time); req_prior[r] >= r is PTC_ERR_INVALID_ARG.
 * A key that is not a field element is reported when it is settled; the
 * keys of repeated depths are only compared.
 *   keys         ptc_u128[n] as for ptc_assign_ids, prefix keys
 *   req_blk_off  u64[n_req + 1] from ptc_hash_blocks (req_blk_off[n_req] == n)
 *   req_prior    u32[n_req]
 */
size_t ptc_assign_ids_prior_workspace_bytes(uint64_t n, uint32_t n_req);
ptc_status ptc_assign_ids_prior(const ptc_u128* keys, uint64_t n, const uint64_t* req_blk_off, const uint32_t* req_prior,
                                uint32_t n_req, uint32_t* ids_out, uint64_t* n_distinct_host_out, void* ws,
                                size_t ws_bytes, void* stream);

/*
 * ptc_assign_ids_ex — ptc_assign_ids (n_req = 0) or ptc_assign_ids_prior
 * (n_req > 0, same hint rules) with the way keys are deduplicated named.
 * Every method gives the same ids and D:
 *   PTC_IDS_TABLE        one open-addressing table of 16-byte slots: a first
 *                        attempt with n / 3 slots (3 n / 4 once that is larger
 *                        than 64 MB), the whole stage again with 1.5 n slots
 *                        if a probe sequence outruns it
 *   PTC_IDS_PARTITIONED  the keys to settle are moved, in streaming passes,
 *                        into 65,536 partitions by 16 key bits, and each
 *                        partition is deduplicated in a table in shared
 *                        memory; a partition with more than 6,144 distinct
 *                        keys sends the stage to the full table as above
 *   PTC_IDS_AUTO         PTC_IDS_PARTITIONED when the first table would exceed
 *                        64 MB (n above about 12.6M), else PTC_IDS_TABLE; what
 *                        ptc_assign_ids and ptc_assign_ids_prior do
 * Workspace: ptc_assign_ids_ex_workspace_bytes(n, n_req, method).  An
 * unknown method is PTC_ERR_INVALID_ARG.
 */
enum { PTC_IDS_AUTO = 0, PTC_IDS_TABLE = 1, PTC_IDS_PARTITIONED = 2 };
size_t ptc_assign_ids_ex_workspace_bytes(uint64_t n, uint32_t n_req, int method);
ptc_status ptc_assign_ids_ex(const ptc_u128* keys, uint64_t n, const uint64_t* req_blk_off, const uint32_t* req_prior,
                             uint32_t n_req, uint32_t* ids_out, uint64_t* n_distinct_host_out, int method, void* ws,
                             size_t ws_bytes, void* stream);

/*
 * ptc_session_prior — the hint above from session labels (Sec. 2.3,
 * sessions): prior_out[r] = the latest request before r with the same label,
 * or PTC_NONE for a session's first request.  req_session u32[n_req], labels
 * below n_session (PTC_ERR_INVALID_ARG otherwise); prior_out u32[n_req].
 * A stable radix sort of the requests by label, then one pass.
 */
size_t ptc_session_prior_workspace_bytes(uint32_t n_req);
ptc_status ptc_session_prior(const uint32_t* req_session, uint32_t n_req, uint32_t n_session, uint32_t* prior_out,
                             void* ws, size_t ws_bytes, void* stream);

/*
 * ptc_verify_ids — exact check of the ids (Sec. 2.2 identity, without hashing):
 * every access must carry the same B tokens as the first access of its id,
 * and its parent (the previous block of its request, or "none" at depth 0)
 * must have the same id as that first access's parent.  By induction over
 * depth this makes equal ids equivalent to equal prefixes.  Returns
 * PTC_ERR_HASH_COLLISION if any access fails the check.
 *
 *   tokens, n_tok, req_tok_off, n_req, block_size  as given to ptc_hash_blocks
 *   req_blk_off  u64[n_req + 1] from ptc_hash_blocks
 *   ids          u32[n] from ptc_assign_ids, n = req_blk_off[n_req]
 */
size_t ptc_verify_ids_workspace_bytes(uint64_t n, uint64_t n_distinct);
ptc_status ptc_verify_ids(const uint32_t* tokens, uint64_t n_tok, const uint64_t* req_tok_off, const uint64_t* req_blk_off,
                          uint32_t n_req, uint32_t block_size, const uint32_t* ids, uint64_t n,
                          uint64_t n_distinct, void* ws, size_t ws_bytes, void* stream);

/*
 * ptc_reuse_indices — previous and next use of each block (Sec. 3.2 and 5.2:
 * Belady's policy needs the time until each block's next access).
 *   prev_out[i] = max{ j < i : ids[j] == ids[i] }, or PTC_NONE
 *   next_out[i] = min{ j > i : ids[j] == ids[i] }, or PTC_NONE
 * Computed from a stable radix sort: of the runs of consecutive ids, cut
 * into pieces that every run holds whole or not at all (one piece per
 * (interval of id-space, run)), or, when those pieces exceed a quarter of
 * the accesses, of every (id, i) pair.
 *
 *   ids        u32[n], every value < n_distinct (PTC_ERR_INVALID_ARG otherwise)
 *   prev_out, next_out  u32[n]
 */
size_t ptc_reuse_indices_workspace_bytes(uint64_t n, uint64_t n_distinct);
ptc_status ptc_reuse_indices(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out,
                             uint32_t* next_out, void* ws, size_t ws_bytes, void* stream);

/*
 * ptc_reuse_indices_ex — the same outputs with the sort chosen by the caller:
 * PTC_REUSE_SORT sorts every (id, i); PTC_REUSE_RUNS sorts the pieces of the
 * id-runs whatever their number; PTC_REUSE_AUTO is ptc_reuse_indices.
 * Workspace: ptc_reuse_indices_ex_workspace_bytes(n, n_distinct, method).
 */
enum { PTC_REUSE_AUTO = 0, PTC_REUSE_SORT = 1, PTC_REUSE_RUNS = 2 };
size_t ptc_reuse_indices_ex_workspace_bytes(uint64_t n, uint64_t n_distinct, int method);
ptc_status ptc_reuse_indices_ex(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out,
                                uint32_t* next_out, int method, void* ws, size_t ws_bytes, void* stream);

/*
 * ptc_stack_distance — LRU stack distance of every access (App. B: the stack
 * distance between reuses decides whether a reuse is reachable within a
 * cache of C blocks).  With p = prev[i]:
 *   dist_out[i] = 1 + #{distinct blocks accessed in positions p+1 .. i-1}
 *               = 1 + #{ j : p < j < i, prev[j] < p or prev[j] == PTC_NONE }
 * and PTC_NONE (never seen) when p == PTC_NONE.  An access hits in an LRU
 * cache of C >= 1 blocks iff dist <= C (Mattson et al. 1970).  The count is a
 * 2-D dominance count answered by N range-rank queries on a wavelet matrix
 * (Claude, Navarro, Ordonez 2015) built over v_j = prev[j] + 1.
 *
 *   prev      u32[n] from ptc_reuse_indices (prev[i] < i or PTC_NONE)
 *   dist_out  u32[n], 1-based; PTC_NONE for a first access
 */
size_t ptc_stack_distance_workspace_bytes(uint64_t n);
ptc_status ptc_stack_distance(const uint32_t* prev, uint64_t n, uint32_t* dist_out, void* ws, size_t ws_bytes,
                              void* stream);

/*
 * ptc_stack_distance_ex — the same distances with the matrix chosen by the
 * caller.  PTC_SD_POINTS builds the wavelet matrix over every access.
 * PTC_SD_RUNS builds it over runs: maximal stretches where prev grows by one
 * from access to access, or that are all first accesses.  A run is either
 * wholly counted or wholly left out of every window (an access has at most
 * one next use), so a matrix over runs weighted by their lengths gives the
 * same counts with R points instead of n.  PTC_SD_AUTO (what
 * ptc_stack_distance does) finds the runs first and takes the matrix over
 * runs when R <= n / 3 and the workspace holds it, else the one over accesses.
 *   prev must come from ptc_reuse_indices, or at least satisfy prev[i] < i and
 *   take each value other than PTC_NONE at most once; the matrix over runs
 *   relies on the latter, and neither checks it.
 * Workspace: ptc_stack_distance_ex_workspace_bytes(n, method);
 * PTC_ERR_WORKSPACE when PTC_SD_RUNS finds more runs than the workspace holds.
 */
enum { PTC_SD_AUTO = 0, PTC_SD_POINTS = 1, PTC_SD_RUNS = 2 };
size_t ptc_stack_distance_ex_workspace_bytes(uint64_t n, int method);
ptc_status ptc_stack_distance_ex(const uint32_t* prev, uint64_t n, uint32_t* dist_out, int method, void* ws,
                                 size_t ws_bytes, void* stream);

/*
 * ptc_stack_distance_variant — stack distances under the semantics variants
 * of Sec. 3.1 (the paper's simulator keeps a whole request resident, making
 * room for it before its prefill) and of the order a request's blocks are
 * touched in.  The result feeds ptc_curves unchanged: block k of a request
 * counts at capacity C iff the largest distance over its depths 0..k is <= C.
 *   touch_order  PTC_TOUCH_ROOT_FIRST: depth 0, 1, ... (the hot path's order)
 *                PTC_TOUCH_LEAF_FIRST: the deepest block first, the root last
 *   residency    PTC_RESIDENCY_BLOCK:   each block is looked up when touched;
 *                                       its distance is its LRU stack depth then
 *                PTC_RESIDENCY_REQUEST: every block of a request is looked up at
 *                                       the request's arrival, before any is
 *                                       touched; its distance is its stack depth
 *                                       at arrival (1 + distinct blocks touched
 *                                       since its last touch and before the
 *                                       request)
 * Every request's blocks are then touched in touch_order.  (ROOT_FIRST, BLOCK)
 * is ptc_stack_distance.
 *   prev         u32[n] from ptc_reuse_indices (root-first access order)
 *   req_blk_off  u64[n_req + 1] from ptc_hash_blocks, req_blk_off[n_req] == n
 *   dist_out     u32[n] in root-first access order; PTC_NONE for a first access
 * PTC_ERR_INVALID_ARG for other touch_order / residency values, malformed
 * offsets, or prev[i] >= i.  Workspace:
 * ptc_stack_distance_variant_workspace_bytes(n, n_req, touch_order, residency).
 */
enum { PTC_TOUCH_ROOT_FIRST = 0, PTC_TOUCH_LEAF_FIRST = 1 };
enum { PTC_RESIDENCY_BLOCK = 0, PTC_RESIDENCY_REQUEST = 1 };
size_t ptc_stack_distance_variant_workspace_bytes(uint64_t n, uint32_t n_req, int touch_order, int residency);
ptc_status ptc_stack_distance_variant(const uint32_t* prev, uint64_t n, const uint64_t* req_blk_off, uint32_t n_req,
                                      int touch_order, int residency, uint32_t* dist_out, void* ws, size_t ws_bytes,
                                      void* stream);
/*
 * ptc_stack_distance_variant_ex — the same, with the route for per-request
 * residency chosen by the caller.  Per request, dist = the per-block distance
 * on the touch stream minus the number of the request's own earlier touches
 * whose previous touch precedes this block's (a block touched after the
 * request began is new to the shorter window iff that holds).  PTC_SD_RUNS
 * counts them over the request's runs (prev growing by one, or first
 * accesses), O(runs of the request) per access; PTC_SD_POINTS answers the
 * window ending at the request's start on the matrix over every access;
 * PTC_SD_AUTO takes the runs when they are at most a third of the accesses.
 * Per-block residency ignores the method.  Same workspace size.
 */
ptc_status ptc_stack_distance_variant_ex(const uint32_t* prev, uint64_t n, const uint64_t* req_blk_off,
                                         uint32_t n_req, int touch_order, int residency, uint32_t* dist_out,
                                         int method, void* ws, size_t ws_bytes, void* stream);

/*
 * ptc_curves — hit and compute-saved curves for every capacity at once
 * (Sec. 3.2 block hit ratio; Sec. 5.2 compute-savings ratio; prefix reuse
 * from Sec. 2.2).  Block k of a request is counted as a hit at capacity C iff
 * every block 0..k of that request is resident, i.e. iff
 *   e_i = max(dist[j] : j in the request, depth(j) <= k) <= C.
 *   hits_host_out[g]      = #{ i : e_i <= cap_host[g] }
 *   saved_host_out[g]     = sum of cost(k_i) over those i   (128-bit)
 *   total_cost_host_out   = sum of cost(k_i) over all i     (128-bit)
 * Block hit ratio = hits / N; compute-savings ratio = saved / total.
 *
 *   dist          u32[n] from ptc_stack_distance
 *   req_blk_off   u64[n_req + 1] from ptc_hash_blocks, req_blk_off[n_req] == n
 *   cm            cost model (host pointer); PTC_ERR_OVERFLOW if a per-block
 *                 cost could exceed 64 bits
 *   cap_host      u64[n_cap] capacities in blocks, strictly ascending, >= 1,
 *                 1 <= n_cap <= PTC_MAX_CAPACITIES (host memory)
 *   hits_host_out u64[n_cap], saved_host_out ptc_u128[n_cap], total_cost_host_out
 *                 ptc_u128[1] (host memory)
 */
size_t ptc_curves_workspace_bytes(uint64_t n, uint32_t n_req, uint32_t n_cap);
ptc_status ptc_curves(const uint32_t* dist, uint64_t n, const uint64_t* req_blk_off, uint32_t n_req,
                      uint32_t block_size, const ptc_cost_model* cm, const uint64_t* cap_host, uint32_t n_cap,
                      uint64_t* hits_host_out, ptc_u128* saved_host_out, ptc_u128* total_cost_host_out, void* ws,
                      size_t ws_bytes, void* stream);

/*
 * ptc_belady_curves — Belady's offline optimum (Sec. 3.2: the offline ceiling
 * the paper sets every eviction policy against) at every capacity of the
 * grid: the block hit and compute-saved curves of Belady's MIN, which on a
 * miss with a full cache evicts the resident block, other than the one just
 * brought in, whose next access lies farthest (never again counts as
 * farthest); every accessed block is admitted.  Block k of a request counts
 * as a hit iff blocks 0..k of that request were all resident (the prefix rule
 * of ptc_curves), and compute saved sums the cost model over those hits.
 * MIN's hits are computed from the reuse intervals (prev[i], i): they are the
 * intervals an earliest-end-first greedy with best-fit tracks keeps with at
 * most C - 1 of them spanning any access.
 *   prev            u32[n] from ptc_reuse_indices (prev[i] < i or PTC_NONE,
 *                   PTC_ERR_INVALID_ARG otherwise)
 *   req_blk_off, n_req, block_size, cm, cap_host, n_cap   as for ptc_curves
 *   hits_host_out   u64[n_cap], saved_host_out ptc_u128[n_cap] (host)
 *   raw_hits_host_out  u64[n_cap] (host) or NULL: resident accesses at each
 *                   capacity without the prefix rule
 * One warp per capacity replays the runs of consecutive re-reads in order;
 * the time grows with the number of runs, not of accesses.
 */
size_t ptc_belady_curves_workspace_bytes(uint64_t n, uint32_t n_req, uint32_t n_cap);
ptc_status ptc_belady_curves(const uint32_t* prev, uint64_t n, const uint64_t* req_blk_off, uint32_t n_req,
                             uint32_t block_size, const ptc_cost_model* cm, const uint64_t* cap_host, uint32_t n_cap,
                             uint64_t* hits_host_out, ptc_u128* saved_host_out, uint64_t* raw_hits_host_out, void* ws,
                             size_t ws_bytes, void* stream);

/*
 * ptc_session_lru_curves — session-level LRU eviction (Sec. 5.3: evicting
 * whole sessions instead of blocks, the eviction-granularity study) at every
 * capacity of the grid, with the prefix rule and cost model of ptc_curves.
 * Rules (the paper states none; these are this library's reading):
 *   - a block belongs to the session whose request brought it into the cache
 *     until it is evicted; hits by other sessions do not change that, so
 *     evicting a session also drops shared prompts it brought in;
 *   - sessions are ordered by the arrival of their latest request (a session
 *     is touched when its request arrives, before its blocks);
 *   - while more than C blocks are resident, every block of the least
 *     recently touched session other than the current one is evicted;
 *   - a session that alone holds more than C blocks keeps only the block
 *     just brought in.
 * Not a stack algorithm: each capacity is replayed on its own (one warp per
 * capacity), so the time grows with n, not with the number of runs.
 *   ids          u32[n] from ptc_assign_ids, each below n_distinct
 *   req_session  u32[n_req] labels below n_session
 *   req_blk_off, n_req, block_size, cm, cap_host, n_cap, hits/saved  as ptc_curves
 * Workspace: ptc_session_lru_curves_workspace_bytes (n_cap x n_distinct x 8
 * bytes for block ownership, plus per-session state).
 */
size_t ptc_session_lru_curves_workspace_bytes(uint64_t n_distinct, uint32_t n_session, uint32_t n_cap);
ptc_status ptc_session_lru_curves(const uint32_t* ids, uint64_t n, uint64_t n_distinct, const uint64_t* req_blk_off,
                                  const uint32_t* req_session, uint32_t n_req, uint32_t n_session,
                                  uint32_t block_size, const ptc_cost_model* cm, const uint64_t* cap_host,
                                  uint32_t n_cap, uint64_t* hits_host_out, ptc_u128* saved_host_out, void* ws,
                                  size_t ws_bytes, void* stream);

/*
 * ptc_pipeline — the five calls in order (hash, ids, reuse, stack distance,
 * curves) in one call, for a trace already on the device.  Semantics, limits
 * and errors are those of the individual calls; the first error stops the
 * pipeline and is returned.
 *   keys_out, req_blk_off_out, ids_out, prev_out, next_out, dist_out
 *       optional device outputs (NULL: kept in the workspace and discarded);
 *       sizes as for the individual calls, keys_out at least
 *       floor(n_tok / block_size) entries
 *   cap_host, n_cap, cm, hits/saved/total outputs  as for ptc_curves
 *   n_access_host_out, n_distinct_host_out        N and D on the host
 *   req_session, n_session   optional (NULL, 0): u32[n_req] session label of
 *       each request, below n_session (PTC_ERR_INVALID_ARG otherwise).  With
 *       them, stage a2 takes the previous request of each request's session
 *       as its prior-request hint (ptc_session_prior, ptc_assign_ids_prior):
 *       a turn of a session re-sends that request's context (Sec. 2.3), so
 *       most of its blocks need not be settled.  The hint is taken only
 *       when the id table would exceed L2 (then stage a2 deduplicates by
 *       partitions, ptc_assign_ids_ex).  The results do not depend on the
 *       sessions; only the time does.
 * The workspace holds the intermediate arrays not supplied plus the largest
 * scratch of any stage (ptc_pipeline_workspace_bytes).  Stages b and c do not
 * wait for their own status; an error they raise is returned with stage d's.
 */
size_t ptc_pipeline_workspace_bytes(uint32_t n_req, uint64_t n_tok, uint32_t block_size, uint32_t n_cap);
ptc_status ptc_pipeline(const uint32_t* tokens, uint64_t n_tok, const uint64_t* req_tok_off, const int64_t* req_ts_us,
                        const uint32_t* req_session, uint32_t n_session, uint32_t n_req, uint32_t block_size, uint64_t seed, const ptc_cost_model* cm,
                        const uint64_t* cap_host, uint32_t n_cap, ptc_u128* keys_out, uint64_t* req_blk_off_out,
                        uint32_t* ids_out, uint32_t* prev_out, uint32_t* next_out, uint32_t* dist_out,
                        uint64_t* n_access_host_out, uint64_t* n_distinct_host_out, uint64_t* hits_host_out,
                        ptc_u128* saved_host_out, ptc_u128* total_cost_host_out, void* ws, size_t ws_bytes,
                        void* stream);

/*
 * ptc_pipeline_host — ptc_pipeline for a trace held in HOST memory: the call
 * a user with a trace on the host makes.  tokens_host (u32[n_tok]),
 * req_tok_off_host (u64[n_req + 1]), req_ts_us_host (i64[n_req], or NULL
 * to skip the order check) and req_session_host (u32[n_req] labels below
 * n_session, or NULL) are host pointers; they are copied on `stream`
 * into the front of the workspace (page-locked host memory copies
 * asynchronously at full link speed, pageable memory is staged by the
 * driver), then the whole path runs on the copy exactly as ptc_pipeline.
 * On a machine with several CPU sockets, keep the page-locked buffers on
 * the NUMA node nearest the GPU: the same 40 GB trace copied in 189 ms from
 * the near node and took up to 2.5x longer from pages on the far one.
 * The curves, N and D come back in host memory as for ptc_pipeline; the
 * per-access arrays stay in the workspace and are not returned.
 * Workspace: ptc_pipeline_host_workspace_bytes, which is
 * ptc_pipeline_workspace_bytes plus room for the copied trace.  The caller
 * keeps the host buffers unchanged until the call returns.
 */
size_t ptc_pipeline_host_workspace_bytes(uint32_t n_req, uint64_t n_tok, uint32_t block_size, uint32_t n_cap);
ptc_status ptc_pipeline_host(const uint32_t* tokens_host, uint64_t n_tok, const uint64_t* req_tok_off_host,
                             const int64_t* req_ts_us_host, const uint32_t* req_session_host, uint32_t n_session,
                             uint32_t n_req, uint32_t block_size, uint64_t seed,
                             const ptc_cost_model* cm, const uint64_t* cap_host, uint32_t n_cap,
                             uint64_t* n_access_host_out, uint64_t* n_distinct_host_out, uint64_t* hits_host_out,
                             ptc_u128* saved_host_out, ptc_u128* total_cost_host_out, void* ws, size_t ws_bytes,
                             void* stream);

/*
 * ptc_trace_stats — trace characterization over the arrays of the path
 * (Sec. 4.1 block lifetimes, categories and the one-hit share; Sec. 4.2 reuse
 * intervals; Sec. 4.3 frequency, reuse interval and lifetime against
 * frequency, requests per session; App. B reuses reachable within a cache of
 * C blocks).  Access i of request r happens at req_ts_us[r] in session
 * req_session[r].  For a block d:
 *   frequency f_d    its number of accesses
 *   lifetime         time of its last access minus time of its first (0 if used once)
 *   category c_d     0 shared across sessions: d appears in two or more sessions,
 *                      at least one of which has two or more requests
 *                    1 session history: d appears in exactly one session, and
 *                      that session has two or more requests
 *                    2 single-turn: every session d appears in has one request
 *                    (the paper's three categories are by message role, which a
 *                    token trace does not carry; sessions stand in for roles)
 * and for a reuse (an access with a previous access of its block) the reuse
 * interval, its time minus the time of that previous access.  bin(x) is the
 * bit length of x: 0 for x = 0, else floor(log2 x) + 1, in [0, 64].
 * Every field of ptc_trace_summary counts:
 *   blocks[c], accesses[c]   blocks of category c and their accesses
 *   freq[c][k]               blocks of category c used exactly k times, 1 <= k < 256;
 *                            freq[c][0]: those used 256 times or more
 *   freq_log2[c][b]          blocks of category c with bin(f) = b
 *   lifetime_us[c][b]        blocks of category c with bin(lifetime) = b
 *   reuse_us[c][b]           reuses of category-c blocks with bin(interval) = b
 *   reuse_by_freq[bf][b]     reuses whose block has bin(f) = bf, with bin(interval) = b
 *   lifetime_by_freq[bf][b]  blocks with bin(f) = bf and bin(lifetime) = b
 *   dist_log2[b]             reuses with bin(stack distance) = b (zero without dist)
 *   sess_requests[b]         sessions with at least one request, by bin(request count)
 *   sess_duration_us[b]      the same sessions by bin(last minus first request time)
 *   n_access = n, n_distinct, n_reuse = n - n_distinct, n_sessions (with at least
 *   one request), n_multi_sessions (with two or more)
 *
 *   ids, prev, next  u32[n] from ptc_assign_ids and ptc_reuse_indices; every id
 *                    below n_distinct and every id used (PTC_ERR_INVALID_ARG
 *                    otherwise, as for prev[i] >= i or next[i] <= i)
 *   dist             u32[n] from ptc_stack_distance, or NULL
 *   req_blk_off      u64[n_req + 1] from ptc_hash_blocks, req_blk_off[n_req] == n
 *   req_ts_us        i64[n_req], non-decreasing (PTC_ERR_UNSORTED otherwise)
 *   req_session      u32[n_req], labels below n_session (PTC_ERR_INVALID_ARG otherwise)
 *   cap_host         u64[n_cap] capacities, strictly ascending and >= 1, host
 *                    memory; n_cap <= PTC_MAX_CAPACITIES, 0 allowed (then NULL)
 *   reach_host_out   u64[n_cap] (host): reuses with stack distance <= cap_host[g];
 *                    needs dist when n > 0 and n_cap > 0
 *   stats_host_out   host memory
 */
#define PTC_STAT_CATEGORIES 3
#define PTC_STAT_BINS 65
#define PTC_STAT_FREQ_EXACT 256
typedef struct {
  uint64_t blocks[PTC_STAT_CATEGORIES];
  uint64_t accesses[PTC_STAT_CATEGORIES];
  uint64_t freq[PTC_STAT_CATEGORIES][PTC_STAT_FREQ_EXACT];
  uint64_t freq_log2[PTC_STAT_CATEGORIES][PTC_STAT_BINS];
  uint64_t reuse_us[PTC_STAT_CATEGORIES][PTC_STAT_BINS];
  uint64_t lifetime_us[PTC_STAT_CATEGORIES][PTC_STAT_BINS];
  uint64_t reuse_by_freq[PTC_STAT_BINS][PTC_STAT_BINS];
  uint64_t lifetime_by_freq[PTC_STAT_BINS][PTC_STAT_BINS];
  uint64_t dist_log2[PTC_STAT_BINS];
  uint64_t sess_requests[PTC_STAT_BINS];
  uint64_t sess_duration_us[PTC_STAT_BINS];
  uint64_t n_access, n_distinct, n_reuse, n_sessions, n_multi_sessions;
} ptc_trace_summary;
size_t ptc_trace_stats_workspace_bytes(uint64_t n, uint64_t n_distinct, uint32_t n_req, uint32_t n_session);
ptc_status ptc_trace_stats(const uint32_t* ids, const uint32_t* prev, const uint32_t* next, const uint32_t* dist,
                           uint64_t n, uint64_t n_distinct, const uint64_t* req_blk_off, const int64_t* req_ts_us,
                           const uint32_t* req_session, uint32_t n_req, uint32_t n_session, const uint64_t* cap_host,
                           uint32_t n_cap, uint64_t* reach_host_out, ptc_trace_summary* stats_host_out, void* ws,
                           size_t ws_bytes, void* stream);

/*
 * ptc_curves_noalloc — ptc_curves for callers that cannot allocate device
 * memory.  The paper has no counterpart; this entry point exists for callers
 * with no way to supply `ws`: code running inside a runtime that owns all
 * device memory and offers no allocator, hosts that forbid cudaMalloc (which
 * may synchronize the device), or loops that must never enter an allocator.
 * Its scratch is one fixed 4 MiB array in the library's device image, which
 * every GPU that loads the library holds until the process exits.  Same
 * arguments and results as ptc_curves without ws / ws_bytes.
 *   - n at most 2^24 accesses (PTC_ERR_WORKSPACE beyond that), n_cap at most
 *     PTC_MAX_CAPACITIES.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current; make that first call
 *     before any stream capture.  The address is kept for the life of the
 *     process: after cudaDeviceReset on a device (which unloads the
 *     library's device code there) do not call this entry point on that
 *     device again in the same process.
 *   - Every call on a device shares the one array, and each call leaves its
 *     contents behind (the next call re-zeroes what must start at zero).
 *     Calls whose work overlaps on the GPU (for example on two streams) race
 *     on it and give wrong results: serialize them.
 *   - Allocates nothing: no cudaMalloc or cudaFree.
 */
ptc_status ptc_curves_noalloc(const uint32_t* dist, uint64_t n, const uint64_t* req_blk_off, uint32_t n_req,
                              uint32_t block_size, const ptc_cost_model* cm, const uint64_t* cap_host,
                              uint32_t n_cap, uint64_t* hits_host_out, ptc_u128* saved_host_out,
                              ptc_u128* total_cost_host_out, void* stream);

/* Frees the calling thread's page-locked staging block (see the
 * conventions above); safe to call at any time between calls. */
void ptc_release_host_staging(void);

/*
 * ptc_test_wait_polls — test hook for the bounded waits (no counterpart in
 * the paper: failure detection).  Kernels that wait on other CTAs (the
 * decoupled look-back of stage a1's block offsets) poll a bounded number of
 * times and then give up with PTC_ERR_TIMEOUT instead of hanging.  With
 * polls > 0, every later ptc_hash_blocks / ptc_pipeline call in the process
 * makes those waits see no predecessor as ready (a flag that nothing sets)
 * and give up after `polls` polls, so a test can drive the give-up path: the
 * call must return PTC_ERR_TIMEOUT and leave the device usable.  polls = 0
 * restores normal waits.  Process-wide; not for production use.
 */
void ptc_test_wait_polls(uint32_t polls);

/*
 * Measurement hooks (no counterpart in the paper: instrumentation for the
 * roofline figures).  ptc_launch_count() counts every kernel this library has
 * launched in the process.  While ptc_timer_enable(1) is in force, every
 * launch is bracketed by two CUDA events on its stream; each call resolves
 * them when it synchronizes and adds the duration to a per-kernel total.
 * ptc_timer_read() copies up to `cap` totals into `out` (host memory) and
 * returns how many kernels have totals.  Not thread-safe across concurrent
 * calls on different streams while enabled.
 */
typedef struct {
  char name[48];
  uint64_t launches;
  double total_ms;
} ptc_kernel_time;
void ptc_timer_enable(int on);
void ptc_timer_reset(void);
uint32_t ptc_timer_read(ptc_kernel_time* out, uint32_t cap);
uint64_t ptc_launch_count(void);

/*
 * ptc_probe_random_rmw — measurement hook (no counterpart in the paper:
 * instrumentation for the roofline figures).  Launches on `stream`, without
 * waiting, `probes` random read-modify-write probes of a table of `slots`
 * 16-byte slots at `table` (device memory, 16-byte aligned, `slots` a power of
 * two, every slot set to all ones by the caller beforehand): each probe reads
 * the slot at a seeded pseudo-random index (SplitMix64) and, if it is still
 * all ones, claims it with a 128-bit compare-and-swap, as the id table's
 * insert does for a key it has not seen.  `sink` is 8 bytes of device memory
 * the kernel may write.  The caller times the launch: probes over seconds is
 * the random read-modify-write rate that bounds the table method's insert
 * on a table of that size (the bench sets it beside the partitioned dedup).  Allocates
 * nothing.  PTC_ERR_INVALID_ARG for a null, misaligned or non-power-of-two
 * table.
 */
ptc_status ptc_probe_random_rmw(void* table, uint64_t slots, uint64_t probes, uint64_t seed, void* sink, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* PTC_H */
