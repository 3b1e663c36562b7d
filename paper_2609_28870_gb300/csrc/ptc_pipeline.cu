// ptc_pipeline: the five calls in order inside the library, so a whole trace
// needs one crossing of the C boundary.  Intermediate arrays live in caller
// buffers when given, otherwise in the workspace; the stages' own scratch
// reuses one region of the workspace because they run one after another on
// the same stream.  Stage d has a region of its own: when stage c used the
// matrix over runs, the curves come from those runs (still in stage c's
// scratch) instead of a pass over every distance.
#include <algorithm>

#include "ptc_internal.h"

namespace {

struct PipeLayout {
  ptc_u128* keys;
  uint64_t* blk_off;
  uint32_t *ids, *prev, *next, *dist;
  void* scratch;
  size_t scratch_bytes;
  void* curves;
  size_t curves_bytes;
  uint32_t* defer;  // error words of stages a1, prior, b, c and a2, read with a later stage's
  uint32_t* prior;  // previous request of each request's session (sessions given)
  uint32_t* order;  // the requests in session order, and the place of each in it (sessions given)
  uint32_t* pos;
  uint64_t* n_slot;  // N as stage a1 left it, for stage a2
  uint64_t* nd_slot;  // D and N as stage a2 left them, for stage b
  ulonglong2* carry;  // per hash tile: the carry stage a2 adds to the keys (when they are not returned)
  uint32_t* lead;
  size_t total;
};

size_t stage_scratch_bytes(uint32_t n_req, uint64_t n_tok, uint32_t B, uint32_t n_cap) {
  const uint64_t n = n_tok / B;
  size_t m = ptc_hash_blocks_workspace_bytes(n_req, n_tok, B);
  const size_t c[] = {ptc::ids_ws_bytes(n, n_req ? n_req : 1), ptc_reuse_indices_workspace_bytes(n, n),
                      ptc_stack_distance_workspace_bytes(n), ptc::session_prior_bytes(n_req)};
  for (size_t x : c) m = x > m ? x : m;
  return m;
}

PipeLayout pipe_layout(void* ws, uint32_t n_req, uint64_t n_tok, uint32_t B, uint32_t n_cap, bool keys, bool blk,
                       bool ids, bool prev, bool next, bool dist) {
  PipeLayout L;
  ptc::Carver cv(ws);
  const uint64_t n = n_tok / B ? n_tok / B : 1;
  L.keys = keys ? nullptr : cv.take<ptc_u128>(n);
  L.blk_off = blk ? nullptr : cv.take<uint64_t>((uint64_t)n_req + 1);
  L.ids = ids ? nullptr : cv.take<uint32_t>(n);
  L.prev = prev ? nullptr : cv.take<uint32_t>(n);
  L.next = next ? nullptr : cv.take<uint32_t>(n);
  L.dist = dist ? nullptr : cv.take<uint32_t>(n);
  L.scratch_bytes = stage_scratch_bytes(n_req, n_tok, B, n_cap);
  L.scratch = cv.take<unsigned char>(L.scratch_bytes);
  L.curves_bytes = ptc_curves_workspace_bytes(n_tok / B, n_req, n_cap);
  L.curves = cv.take<unsigned char>(L.curves_bytes);
  L.defer = cv.take<uint32_t>(5);
  L.prior = cv.take<uint32_t>(n_req ? n_req : 1);
  L.order = cv.take<uint32_t>(n_req ? n_req : 1);
  L.pos = cv.take<uint32_t>(n_req ? n_req : 1);
  L.n_slot = cv.take<uint64_t>(1);
  L.nd_slot = cv.take<uint64_t>(2);
  const uint64_t ct = keys ? 1 : ptc::hash_carry_tiles(n_tok, B);
  L.carry = cv.take<ulonglong2>(ct);
  L.lead = cv.take<uint32_t>(ct);
  L.total = cv.bytes();
  return L;
}

}  // namespace

extern "C" size_t ptc_pipeline_workspace_bytes(uint32_t n_req, uint64_t n_tok, uint32_t block_size, uint32_t n_cap) {
  if (block_size == 0) block_size = 1;
  return pipe_layout(nullptr, n_req, n_tok, block_size, n_cap, false, false, false, false, false, false).total;
}

extern "C" ptc_status ptc_pipeline(const uint32_t* tokens, uint64_t n_tok, const uint64_t* req_tok_off,
                                   const int64_t* req_ts_us, const uint32_t* req_session, uint32_t n_session,
                                   uint32_t n_req, uint32_t block_size, uint64_t seed,
                                   const ptc_cost_model* cm, const uint64_t* cap_host, uint32_t n_cap,
                                   ptc_u128* keys_out, uint64_t* req_blk_off_out, uint32_t* ids_out,
                                   uint32_t* prev_out, uint32_t* next_out, uint32_t* dist_out,
                                   uint64_t* n_access_host_out, uint64_t* n_distinct_host_out,
                                   uint64_t* hits_host_out, ptc_u128* saved_host_out,
                                   ptc_u128* total_cost_host_out, void* ws, size_t ws_bytes, void* stream) {
  if (block_size < 1 || block_size > PTC_MAX_BLOCK_SIZE) return PTC_ERR_INVALID_ARG;
  if (!n_access_host_out || !n_distinct_host_out) return PTC_ERR_INVALID_ARG;
  if (req_session && n_session == 0 && n_req > 0) return PTC_ERR_INVALID_ARG;
  const PipeLayout need = pipe_layout(nullptr, n_req, n_tok, block_size, n_cap, keys_out, req_blk_off_out, ids_out,
                                      prev_out, next_out, dist_out);
  if (!ptc::ws_ok(ws, ws_bytes, need.total)) return PTC_ERR_WORKSPACE;
  const PipeLayout L = pipe_layout(ws, n_req, n_tok, block_size, n_cap, keys_out, req_blk_off_out, ids_out, prev_out,
                                   next_out, dist_out);
  ptc_u128* keys = keys_out ? keys_out : L.keys;
  uint64_t* blk = req_blk_off_out ? req_blk_off_out : L.blk_off;
  uint32_t* ids = ids_out ? ids_out : L.ids;
  uint32_t* prev = prev_out ? prev_out : L.prev;
  uint32_t* next = next_out ? next_out : L.next;
  uint32_t* dist = dist_out ? dist_out : L.dist;
  const uint64_t cap = n_tok / block_size ? n_tok / block_size : 1;
  uint64_t n = 0, d = 0, unused = 0;
  *n_access_host_out = 0;
  *n_distinct_host_out = 0;
  cudaStream_t s = (cudaStream_t)stream;
  // Stages a1, a2, b and c do not wait for their own status.  a1's error
  // word and N go to device slots that stage a2 reads (its grids cover N's
  // upper bound, n_tok / B); a2's error word, N and D go to slots that stage
  // b's first kernels read, and reach the host with stage b's own wait; b's
  // and c's error words are read with stage d's.
  if (ptc::fill_async(L.defer, 0u, 5 * sizeof(uint32_t), s) != PTC_OK) return PTC_ERR_CUDA;
  // with sessions, stage a2 is told the previous request of each request's
  // session, whose blocks the request mostly repeats (computed here, in the
  // scratch region, before stage a1 takes it over); only a DRAM-sized id
  // table gains from it
  // (the labels are checked whenever they are given)
  const bool hinted = req_session != nullptr && n_req > 0 && ptc::ids_table_in_dram(cap);
  if (req_session && n_req > 0)
    ptc::session_prior(req_session, n_req, n_session, L.prior, L.scratch, s, &L.defer[1], L.order, L.pos);
  const ptc::IdsHint hint{blk, L.prior, n_req, L.order, L.pos};
  const ptc::IdsHint* hp = hinted ? &hint : nullptr;
  // keys the caller does not take skip their carry pass: stage a2 adds the
  // carry as it reads them
  ptc::KeyCarry kc{L.carry, L.lead, 1};
  ptc::KeyCarry* kcp = keys_out ? nullptr : &kc;
  ptc_status rc = ptc::hash_impl(tokens, n_tok, req_tok_off, req_ts_us, n_req, block_size, seed, keys, cap, blk,
                                 &unused, L.scratch, L.scratch_bytes, s, L.n_slot, &L.defer[0], kcp);
  if (rc != PTC_OK) return rc;
  rc = ptc::ids_impl(keys, cap, L.n_slot, ids, &n, &d, L.scratch, L.scratch_bytes, s, &L.defer[0], 2, kcp,
                     L.nd_slot, &L.defer[4], false, hp);
  if (rc != PTC_OK) return rc;
  const ptc::ReuseDevIn din{L.nd_slot, &L.defer[4]};
  ptc::ReuseHostOut hout;
  rc = ptc::reuse_view(ids, cap, cap, prev, next, L.scratch, L.scratch_bytes, s, &L.defer[2], &din, &hout);
  *n_access_host_out = n = hout.n;
  *n_distinct_host_out = d = hout.D;
  if (rc != PTC_OK) return rc;
  if (hout.ids_err) {
    // stage a2's first attempt outran its table (or a1 / a2 failed): redo a2
    // with the full table, waiting for it, then stage b with the host's N
    // and D
    if (hout.ids_err != ptc::kErrTableFull) return ptc::status_of(hout.ids_err);
    rc = ptc::ids_impl(keys, cap, L.n_slot, ids, &n, &d, L.scratch, L.scratch_bytes, s, &L.defer[0], 2, kcp, nullptr,
                       nullptr, true, hp);
    *n_access_host_out = n;
    *n_distinct_host_out = d;
    if (rc != PTC_OK) return rc;
    if (n > 0) rc = ptc::reuse_view(ids, n, d, prev, next, L.scratch, L.scratch_bytes, s, &L.defer[2]);
    if (rc != PTC_OK) return rc;
  }
  ptc::RunsView runs;
  if (n > 0) {
    rc = ptc::stack_distance_view(prev, n, dist, PTC_SD_AUTO, L.scratch, L.scratch_bytes, s, &runs, &L.defer[3]);
    if (rc != PTC_OK) return rc;
  }
  return ptc::curves_impl(dist, n, blk, n_req, block_size, cm, cap_host, n_cap, hits_host_out, saved_host_out,
                          total_cost_host_out, L.curves, L.curves_bytes, s, &runs, &L.defer[2], 2);
}

// ptc_pipeline_host: the same path for a trace in host memory.  The trace is
// copied into the front of the workspace on `stream` (offsets, times and
// sessions first, then the tokens in one copy), and ptc_pipeline runs on the
// copy.
namespace {

struct HostLayout {
  uint32_t* tok;
  uint64_t* off;
  int64_t* ts;
  uint32_t* ses;
  void* pws;
  size_t pws_bytes;
  size_t total;
};

HostLayout host_layout(void* ws, uint32_t n_req, uint64_t n_tok, uint32_t B, uint32_t n_cap) {
  HostLayout L;
  ptc::Carver cv(ws);
  L.tok = cv.take<uint32_t>(n_tok ? n_tok : 1);
  L.off = cv.take<uint64_t>((uint64_t)n_req + 1);
  L.ts = cv.take<int64_t>(n_req ? n_req : 1);
  L.ses = cv.take<uint32_t>(n_req ? n_req : 1);
  L.pws_bytes = ptc_pipeline_workspace_bytes(n_req, n_tok, B, n_cap);
  L.pws = cv.take<unsigned char>(L.pws_bytes);
  L.total = cv.bytes();
  return L;
}

}  // namespace

extern "C" size_t ptc_pipeline_host_workspace_bytes(uint32_t n_req, uint64_t n_tok, uint32_t block_size,
                                                    uint32_t n_cap) {
  if (block_size == 0) block_size = 1;
  return host_layout(nullptr, n_req, n_tok, block_size, n_cap).total;
}

extern "C" ptc_status ptc_pipeline_host(const uint32_t* tokens_host, uint64_t n_tok, const uint64_t* req_tok_off_host,
                                        const int64_t* req_ts_us_host, const uint32_t* req_session_host,
                                        uint32_t n_session, uint32_t n_req, uint32_t block_size,
                                        uint64_t seed, const ptc_cost_model* cm, const uint64_t* cap_host,
                                        uint32_t n_cap, uint64_t* n_access_host_out, uint64_t* n_distinct_host_out,
                                        uint64_t* hits_host_out, ptc_u128* saved_host_out,
                                        ptc_u128* total_cost_host_out, void* ws, size_t ws_bytes, void* stream) {
  if (block_size < 1 || block_size > PTC_MAX_BLOCK_SIZE) return PTC_ERR_INVALID_ARG;
  if (!n_access_host_out || !n_distinct_host_out || !req_tok_off_host) return PTC_ERR_INVALID_ARG;
  if (n_tok > 0 && !tokens_host) return PTC_ERR_INVALID_ARG;
  *n_access_host_out = 0;
  *n_distinct_host_out = 0;
  if (!ptc::ws_ok(ws, ws_bytes, host_layout(nullptr, n_req, n_tok, block_size, n_cap).total))
    return PTC_ERR_WORKSPACE;
  const HostLayout L = host_layout(ws, n_req, n_tok, block_size, n_cap);
  cudaStream_t s = (cudaStream_t)stream;
  if (cudaMemcpyAsync(L.off, req_tok_off_host, sizeof(uint64_t) * ((uint64_t)n_req + 1), cudaMemcpyHostToDevice, s) !=
      cudaSuccess)
    return PTC_ERR_CUDA;
  if (req_ts_us_host && n_req > 0 &&
      cudaMemcpyAsync(L.ts, req_ts_us_host, sizeof(int64_t) * n_req, cudaMemcpyHostToDevice, s) != cudaSuccess)
    return PTC_ERR_CUDA;
  if (req_session_host && n_req > 0 &&
      cudaMemcpyAsync(L.ses, req_session_host, sizeof(uint32_t) * n_req, cudaMemcpyHostToDevice, s) != cudaSuccess)
    return PTC_ERR_CUDA;
  if (n_tok > 0 &&
      cudaMemcpyAsync(L.tok, tokens_host, sizeof(uint32_t) * n_tok, cudaMemcpyHostToDevice, s) != cudaSuccess)
    return PTC_ERR_CUDA;
  return ptc_pipeline(L.tok, n_tok, L.off, req_ts_us_host ? L.ts : nullptr, req_session_host ? L.ses : nullptr,
                      n_session, n_req, block_size, seed, cm, cap_host,
                      n_cap, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, n_access_host_out,
                      n_distinct_host_out, hits_host_out, saved_host_out, total_cost_host_out, L.pws, L.pws_bytes,
                      stream);
}
