// Host-side helpers shared by the C-ABI entry points.
#pragma once

#include <cuda_runtime.h>

#include <utility>

#include "../../include/ptc.h"
#include "ptc_common.cuh"

namespace ptc {

// Launch accounting and optional per-kernel CUDA-event timing (ptc_timer_*).
// Every kernel launch goes through PTC_LAUNCH, which counts it and, while
// timing is enabled, brackets it with two events on the launch stream.  The
// events are resolved when the call synchronizes (end_call).
void timer_launch_begin(const char* name, cudaStream_t s);
void timer_launch_end(cudaStream_t s);
void timer_resolve();

#define PTC_LAUNCH(name, stream, ...)           \
  do {                                          \
    ::ptc::timer_launch_begin(name, stream);    \
    __VA_ARGS__;                                \
    ::ptc::timer_launch_end(stream);            \
  } while (0)

// Launch with programmatic stream serialization: the kernel's CTAs may be
// scheduled before the previous kernel on `s` has finished, and wait for it
// in grid_dep_sync() (every kernel of this library starts with it).  After a
// copy or memset the launch is ordered as usual.  A launch error is left for
// end_call's cudaGetLastError.
template <typename... KArgs, typename... Args>
inline void launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  (void)cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// PTC_KERNEL(name, stream, kernel, grid, block, smem, args...): a counted
// (and, while timing, bracketed) launch_pdl.  A template kernel whose
// arguments hold a comma goes in parentheses.
#define PTC_KERNEL(name, stream, kernel, grid, block, smem, ...) \
  PTC_LAUNCH(name, stream, ::ptc::launch_pdl(kernel, grid, block, smem, stream, __VA_ARGS__))

// Fill `bytes` at `p` with the 32-bit `pattern` (0 or all ones) on `s`.  A
// kernel (k_fill, ptc_abi.cu) rather than cudaMemsetAsync, so that it joins
// the programmatic launch chain instead of draining the stream around it;
// sizes or addresses that are not whole 32-bit words go to cudaMemsetAsync.
ptc_status fill_async(void* p, uint32_t pattern, size_t bytes, cudaStream_t s);

// Several fills in one launch (one kernel, one grid row per range), for the
// regions a call clears before its first kernel; a range that is not whole
// 32-bit words goes to fill_async on its own.
struct FillRange {
  void* p;
  size_t bytes;
  uint32_t pattern;
};
constexpr int kFillRanges = 4;
ptc_status fill_many_async(const FillRange* r, int n, cudaStream_t s);

// Zero the status block (and any extra prefix of the workspace) on `stream`.
inline ptc_status begin_call(void* ws, size_t zero_bytes, cudaStream_t stream) {
  return fill_async(ws, 0u, zero_bytes, stream);
}

// The poll count set by ptc_test_wait_polls (0: normal waits), read by the
// calls whose kernels wait on each other (stage a1's look-back).
uint32_t test_wait_polls();

// Words of ptc_trace_stats's results: the summary and the reach bins.
constexpr size_t kStatsHostWords = sizeof(ptc_trace_summary) / 8 + PTC_MAX_CAPACITIES + 1;
// Page-locked host buffers for the small copies around a call's wait, one
// set per host thread (ptc_abi.cu).  A copy from or to pageable memory goes
// through a driver bounce buffer and costs the wait tens of microseconds.
// Falls back to ordinary thread-local memory if page-locked memory cannot be
// had.  Valid until the thread's next call.
struct HostStage {
  DevStatus st;
  uint64_t out[3 * PTC_MAX_CAPACITIES + 2];
  alignas(16) uint64_t stats[kStatsHostWords];
  HostStage* dev;  // the same memory as seen by kernels (mapped), or null
};
HostStage* host_stage();
void release_host_stage();  // frees the calling thread's page-locked block
// Copy `bytes` from device memory to `host_dst`.  When `host_dst` lies in
// the thread's host stage and that stage is mapped, a one-CTA kernel
// (k_copy_words) writes it straight into host memory, which joins the launch
// chain; otherwise cudaMemcpyAsync.
ptc_status copy_to_host_async(void* host_dst, const void* dev_src, size_t bytes, cudaStream_t s);
// While one is alive on a thread, host_stage() allocates nothing (the
// allocation-free entry points): it hands out the thread-local fallback
// unless the page-locked set already exists.
struct NoHostAlloc {
  NoHostAlloc();
  ~NoHostAlloc();
  bool prev;
};

// Wait for the call's work and translate the device status block.
// The status a device error word stands for.
inline ptc_status status_of(uint32_t e) {
  if (e & kErrBounds) return PTC_ERR_BOUNDS;
  if (e & kErrTimeout) return PTC_ERR_TIMEOUT;
  if (e & kErrUnsorted) return PTC_ERR_UNSORTED;
  if (e & kErrOverflow) return PTC_ERR_OVERFLOW;
  if (e & kErrCollision) return PTC_ERR_HASH_COLLISION;
  if (e & (kErrInvalid | kErrTableFull)) return PTC_ERR_INVALID_ARG;
  return PTC_OK;
}

inline ptc_status end_call(const DevStatus* dev, cudaStream_t stream, DevStatus* host_copy) {
  if (cudaGetLastError() != cudaSuccess) return PTC_ERR_CUDA;
  DevStatus* pin = &host_stage()->st;
  if (copy_to_host_async(pin, dev, sizeof(DevStatus), stream) != PTC_OK) return PTC_ERR_CUDA;
  if (cudaStreamSynchronize(stream) != cudaSuccess) return PTC_ERR_CUDA;
  *host_copy = *pin;
  timer_resolve();
  return status_of(host_copy->err);
}

// Instead of waiting for a call's status, queue a copy of its error word to
// `slot`, for a later call that does wait to fold in (ptc_pipeline).
// Ranks over a bitmap (ptc_abi.cu): pre[w] = set bits in words [0, w) for
// w < nwords, by a count per tile of kRankTile words, the last CTA's prefix
// over the tiles, then a pass per word.  Scratch: tcnt and tpre of
// rank_tiles(nwords) + 1 entries, and a zeroed counter *done.  With `total`
// the number of set bits is stored there (device memory).
constexpr uint32_t kRankTile = 2048;
inline uint32_t rank_tiles(uint32_t nwords) { return (nwords + kRankTile - 1) / kRankTile; }
ptc_status bitmap_ranks(const uint32_t* bits, uint32_t nwords, uint32_t* pre, uint32_t* tcnt, uint32_t* tpre,
                        uint32_t* done, uint64_t* total, cudaStream_t s);

// OR the n (at most 32) deferred error words at `err` into st->err.
ptc_status carry_errors(const uint32_t* err, uint32_t n, DevStatus* st, cudaStream_t s);
// With `value_slot`, value[value_index .. value_index + value_count) of the
// status block is copied there too.
ptc_status defer_status(const DevStatus* dev, uint32_t* slot, cudaStream_t stream, uint64_t* value_slot = nullptr,
                        uint32_t value_index = 0, uint32_t value_count = 1);

// Streaming multiprocessors of the current device (persistent grids).
inline int num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 148;
  return n;
}

inline bool ws_ok(const void* ws, size_t ws_bytes, size_t need) {
  return ws != nullptr && ((uintptr_t)ws & 255) == 0 && ws_bytes >= need;
}

// The runs stage c leaves in its workspace when it used the matrix over runs
// (ptc_runs.cu); the pipeline hands them to stage d.
struct RunsView {
  bool used = false;
  uint32_t R = 0;
  const uint32_t* rec_s = nullptr;  // R + 1 run starts (rec_s[R] = n)
  const uint32_t* sd = nullptr;     // distance of every run
  const uint32_t* bits = nullptr;   // run-start bitmap, one word per 32 accesses
  const uint32_t* wpre = nullptr;   // runs starting before each word
};
// Keys left without the carry from earlier tiles (stage a1 skips its
// chain pass): block i of tile t = i / tile_blocks still needs carry[t] added
// (mod p, per word) when i - t tile_blocks < lead[t]; tile_blocks is a power
// of two.  Device arrays of
// hash_carry_tiles() entries, owned by the caller.
struct KeyCarry {
  ulonglong2* carry;
  uint32_t* lead;
  uint32_t tile_blocks;
};
uint64_t hash_carry_tiles(uint64_t n_tok, uint32_t block_size);

// Stage a1 (ptc_hash.cu).  With `n_slot` and `err_slot` (device memory) the
// final wait is replaced by defer_status: N goes to *n_slot, the error word
// to *err_slot, and *n_access_host_out is left 0.  With `carry` the keys are
// left without the cross-tile carry, which goes to carry's arrays instead.
ptc_status hash_impl(const uint32_t* tokens, uint64_t n_tok, const uint64_t* req_tok_off, const int64_t* req_ts_us,
                     uint32_t n_req, uint32_t block_size, uint64_t seed, ptc_u128* keys_out, uint64_t keys_cap,
                     uint64_t* req_blk_off_out, uint64_t* n_access_host_out, void* ws, size_t ws_bytes,
                     cudaStream_t s, uint64_t* n_slot, uint32_t* err_slot, KeyCarry* carry = nullptr);
// Stage a2 (ptc_ids.cu) over n_ub keys, of which the first min(*n_dev, n_ub)
// are used when `n_dev` (device memory) is given.  Error words at
// `carry_err` join the call's own.  Reports the number used and D.  With
// `kc` each key gets its tile's carry as it is read.
// With `nd_slot` and `err_slot` (device memory) the call does not wait: it
// makes one attempt (the partitioned dedup, or the table's small first
// size) and leaves D in nd_slot[0], the number of keys used in nd_slot[1]
// and its error word in *err_slot (an attempt that outran its table shows as
// exactly kErrTableFull; redo the stage then with `full_table`).
// The prior-request hint of stage a2 (ptc_assign_ids_prior): prior[r] is an
// earlier request whose blocks request r is likely to repeat, or PTC_NONE.
struct IdsHint {
  const uint64_t* blk_off;  // n_req + 1 (device)
  const uint32_t* prior;    // n_req (device)
  uint32_t n_req;
  const uint32_t* order;    // optional (device): the requests in session order, prior[r] = the place before r
  const uint32_t* pos;      //   and the place of every request in it
};
size_t ids_ws_bytes(uint64_t n, uint32_t n_req_hint);
// Whether the id table for n keys is larger than the part of L2 it may take:
// only then do the table probes the prior-request hint saves cost DRAM
// traffic (an L2-resident table probes faster than the hint's extra reads),
// and only then does stage a2 deduplicate by partitions instead.
bool ids_table_in_dram(uint64_t n);
// The previous request of each request's session (ptc_session_prior),
// queued on `s` without waiting; scratch of session_prior_bytes(n_req).
size_t session_prior_bytes(uint32_t n_req);
void session_prior(const uint32_t* req_session, uint32_t n_req, uint32_t n_session, uint32_t* prior, void* ws,
                   cudaStream_t s, uint32_t* err, uint32_t* order = nullptr,
                   uint32_t* pos = nullptr);
ptc_status ids_impl(const ptc_u128* keys, uint64_t n_ub, const uint64_t* n_dev, uint32_t* ids_out,
                    uint64_t* n_used_host_out, uint64_t* n_distinct_host_out, void* ws, size_t ws_bytes,
                    cudaStream_t s, const uint32_t* carry_err, uint32_t n_carry, const KeyCarry* kc = nullptr,
                    uint64_t* nd_slot = nullptr, uint32_t* err_slot = nullptr, bool full_table = false,
                    const IdsHint* hint = nullptr, int method = PTC_IDS_AUTO);
ptc_status stack_distance_view(const uint32_t* prev, uint64_t n, uint32_t* dist_out, int method, void* ws,
                               size_t ws_bytes, cudaStream_t s, RunsView* view, uint32_t* defer_err);
// Stage b as ptc_reuse_indices does it (ptc_reuse.cu); with `defer_err` the
// final wait is replaced by defer_status.  With `din`, stage a2 has not
// waited: n and n_distinct are upper bounds, the kernels before this stage's
// own wait read the real ones from din->nd (nd[0] = D, nd[1] = accesses),
// and that wait reports them, with stage a2's error word, in *hout.  If that
// word is not 0 the call returns PTC_OK at once and its results are void.
struct ReuseDevIn {
  const uint64_t* nd;
  const uint32_t* ids_err;
};
struct ReuseHostOut {
  uint64_t n = 0, D = 0;
  uint32_t ids_err = 0;
};
ptc_status reuse_view(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out, uint32_t* next_out,
                      void* ws, size_t ws_bytes, cudaStream_t s, uint32_t* defer_err, const ReuseDevIn* din = nullptr,
                      ReuseHostOut* hout = nullptr);
// The per-block cost as cost(k) = alpha + beta k for block size B (R7: every
// cost kind is affine in the depth k); PTC_ERR_OVERFLOW if a coefficient
// exceeds 64 bits, PTC_ERR_INVALID_ARG for an unknown kind (ptc_curves.cu).
ptc_status cost_coeffs(const ptc_cost_model* cm, uint32_t block_size, uint64_t* alpha, uint64_t* beta);
// Stage d (ptc_curves.cu); with `runs` (from stack_distance_view) the curves
// come from the runs instead of a pass over every distance.
ptc_status curves_impl(const uint32_t* dist, uint64_t n, const uint64_t* req_blk_off, uint32_t n_req,
                       uint32_t block_size, const ptc_cost_model* cm, const uint64_t* cap_host, uint32_t n_cap,
                       uint64_t* hits_host_out, ptc_u128* saved_host_out, ptc_u128* total_cost_host_out, void* ws,
                       size_t ws_bytes, cudaStream_t s, const RunsView* runs, const uint32_t* carry_err = nullptr,
                       uint32_t n_carry = 0);

// Stage c on the matrix over every access (ptc_wavelet.cu); the C entry
// points in ptc_runs.cu choose between it and the matrix over runs.  With
// `wend` (device, one entry per access) the window of access i ends at
// wend[i] <= i instead of at i: dist = 1 + distinct values in (prev[i], wend[i]).
size_t stack_distance_points_bytes(uint64_t n);
ptc_status stack_distance_points(const uint32_t* prev, uint64_t n, uint32_t* dist_out, void* ws, size_t ws_bytes,
                                 cudaStream_t s, const uint32_t* wend = nullptr);

// Stage b by a radix sort of every access (ptc_sort.cu), and the same sort
// for any (key, value) pairs; the C entry point in ptc_reuse.cu chooses.
size_t reuse_by_sort_bytes(uint64_t n);
ptc_status reuse_by_sort(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out,
                         uint32_t* next_out, void* ws, size_t ws_bytes, cudaStream_t s);
size_t sort_pairs_bytes(uint64_t n);
void sort_pairs(const uint32_t* keys, const uint32_t* vals, uint32_t n, uint32_t bits, void* ws, cudaStream_t s,
                DevStatus* st, const uint32_t** keys_sorted, const uint32_t** vals_sorted);

}  // namespace ptc
