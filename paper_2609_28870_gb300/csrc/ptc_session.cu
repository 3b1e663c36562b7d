// Session-level LRU eviction at every capacity of a grid (Sec. 5.3: block-
// level vs session-level eviction).  Session-level eviction is not a stack
// algorithm (a cache of C + 1 blocks can hold a session that a cache of C
// blocks dropped whole), so each capacity is its own replay: one warp per
// capacity walks the trace in order.
//
// Readings: a block belongs to the session whose request brought it in,
// until evicted (hits by other sessions do not move it); sessions are ordered
// by their latest request, touched when it arrives; while more than C blocks
// are resident the least recently touched other session loses all its
// blocks; a session that alone holds more than C keeps only the block just
// brought in.  Blocks count with the prefix rule (Sec. 2.2).
//
// State per capacity, all O(1) per step:
//   owner[id]  (session << 32 | epoch) of the session that brought block id
//              in, all ones if never; the block is resident iff that epoch is
//              still its session's current one;
//   epoch[s]   bumped when session s is evicted, which drops all its blocks
//              at once; count[s] its resident blocks;
//   last[s]    its latest request; the requests themselves are the recency
//              queue: the next victim is the oldest request r at the front
//              that is still its session's latest and whose session holds
//              blocks (a passed entry never becomes valid again, so the front
//              only moves forward).
// A request's blocks go 32 at a time, one per lane.  The lanes of a chunk
// settle together up to the first miss that would take the cache past C (or
// the second copy of a repeated block); lane 0 brings that block in and
// evicts, and the lanes after it are tested again, since an eviction can drop
// a later block of the same chunk.  Session epochs sit in shared memory when
// there are at most 16,384 sessions.
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr uint64_t kNoOwner = ~0ULL;

struct SesCaps {
  uint64_t c[PTC_MAX_CAPACITIES];
};

struct SesArgs {
  const uint32_t* ids;
  const uint64_t* blk_off;
  const uint32_t* ses;
  uint32_t n_req, n_session;
  uint64_t n_distinct;
  uint64_t* owner;  // G slices of n_distinct
  uint32_t *epoch, *count, *last;  // G slices of n_session each
  uint64_t sD, sS;
  uint32_t G;
  uint64_t alpha, beta;
  uint64_t* out;  // hits[G] | saved[G] (lo, hi)
  DevStatus* st;
};

__device__ __forceinline__ void add_mul128(uint64_t& lo, uint64_t& hi, uint64_t a, uint64_t b) {
  const uint64_t plo = a * b, phi = __umul64hi(a, b);
  lo += plo;
  hi += phi + (lo < plo ? 1 : 0);
}

// Request offsets checked once (the replay trusts them afterwards).
__global__ void k_ses_check(const uint64_t* __restrict__ blk_off, uint32_t R, uint64_t n,
                            const uint32_t* __restrict__ ses, uint32_t S, DevStatus* st) {
  grid_dep_sync();
  const uint64_t r = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= R) return;
  const uint64_t a = blk_off[r], b = blk_off[r + 1];
  if (b < a || b > n || (r == 0 && a != 0) || (r + 1 == R && b != n) || ses[r] >= S) raise_err(st, kErrInvalid);
}

constexpr uint32_t kSesSmemSessions = 16384;  // session epochs kept in shared memory up to this many (64 KB)

__global__ void __launch_bounds__(32) k_ses_sim(SesArgs a, SesCaps caps) {
  extern __shared__ uint32_t s_epoch[];
  grid_dep_sync();
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t g = blockIdx.x;
  if (g >= a.G || a.st->err) return;  // malformed offsets or labels: nothing to replay
  uint64_t* owner = a.owner + g * a.sD;
  uint32_t* count = a.count + g * a.sS;
  uint32_t* last = a.last + g * a.sS;
  const bool in_smem = a.n_session <= kSesSmemSessions;
  volatile uint32_t* ep = in_smem ? s_epoch : a.epoch + g * a.sS;  // one warp owns it: plain accesses
  if (in_smem)
    for (uint32_t t = lane; t < a.n_session; t += 32) s_epoch[t] = 0;
  __syncwarp();
  const uint64_t C = caps.c[g];
  uint64_t total = 0, hits = 0, sv_lo = 0, sv_hi = 0;
  uint32_t front = 0;
  for (uint32_t r = 0; r < a.n_req; ++r) {
    const uint32_t s = a.ses[r];
    const uint64_t b = a.blk_off[r], e = a.blk_off[r + 1];
    if (lane == 0) __stcg(&last[s], r);
    uint32_t es = ep[s];
    bool missed = false;
    uint32_t id_next = b + lane < e ? a.ids[b + lane] : 0u;
    for (uint64_t c = b; c < e; c += 32) {
      const bool valid = c + lane < e;
      uint32_t id = id_next;
      id_next = c + 32 + lane < e ? a.ids[c + 32 + lane] : 0u;  // in flight while this chunk settles
      if (valid && id >= a.n_distinct) {
        raise_err(a.st, kErrInvalid);
        id = 0;
      }
      uint32_t pending = __ballot_sync(kFull, valid);
      while (pending) {
        const bool mine = (pending >> lane) & 1u;
        bool res = false;
        if (mine) {
          const uint64_t o = __ldcg(&owner[id]);
          res = o != kNoOwner && in_bounds(a.st, o >> 32, a.n_session) && ep[(uint32_t)(o >> 32)] == (uint32_t)o;
        }
        // a block repeated inside the chunk is settled after its first copy
        uint32_t same = 0;
        if (mine) same = __match_any_sync(pending, id);
        const uint32_t later_copy = __ballot_sync(kFull, mine && (same & ((1u << lane) - 1u)) != 0);
        const uint32_t miss = __ballot_sync(kFull, mine && !res);
        // the first miss that would push the cache past C
        const uint64_t room = C - total;
        uint32_t over = 32;
        if ((uint64_t)__popc(miss) > room) {
          uint32_t m = miss;
          for (uint64_t k = 0; k < room; ++k) m &= m - 1u;
          over = (uint32_t)(__ffs(m) - 1);
        }
        const uint32_t rep = later_copy ? (uint32_t)(__ffs(later_copy) - 1) : 32u;
        const uint32_t stop = over < rep ? over : rep;
        const uint32_t batch = pending & (stop == 32 ? kFull : ((1u << stop) - 1u));
        // lanes before `stop` settle together: no eviction among them
        const uint32_t bmiss = miss & batch;
        if (((batch >> lane) & 1u) && !res) __stcg(&owner[id], ((uint64_t)s << 32) | es);
        total += __popc(bmiss);
        if (lane == 0 && bmiss) __stcg(&count[s], __ldcg(&count[s]) + __popc(bmiss));
        if (!missed && batch) {
          const uint32_t lo = __ffs(batch) - 1;
          const uint32_t f = (bmiss ? (uint32_t)(__ffs(bmiss) - 1) : 32u - __clz(batch)) - lo;
          const uint64_t d0 = c + lo - b;
          hits += f;
          add_mul128(sv_lo, sv_hi, a.alpha, f);
          add_mul128(sv_lo, sv_hi, a.beta, (uint64_t)f * d0 + (uint64_t)f * (f ? f - 1 : 0) / 2);
          missed = bmiss != 0;
        }
        pending &= ~batch;
        if (stop == 32 || stop == rep) continue;  // done, or a repeated block: test it again
        // lane `stop` misses and overflows: lane 0 brings it in and evicts
        __syncwarp();
        const uint32_t x = __shfl_sync(kFull, id, stop);
        if (lane == 0) {
          __stcg(&owner[x], ((uint64_t)s << 32) | es);
          __stcg(&count[s], __ldcg(&count[s]) + 1u);
          total += 1;
          while (total > C) {
            uint32_t v = kNone;
            while (front < r) {
              const uint32_t t = a.ses[front];
              if (in_bounds(a.st, t, a.n_session) && __ldcg(&last[t]) == front && __ldcg(&count[t]) > 0) {
                v = t;
                break;
              }
              ++front;
            }
            if (v != kNone) {  // the least recently touched other session goes whole
              ep[v] = ep[v] + 1u;
              total -= __ldcg(&count[v]);
              __stcg(&count[v], 0u);
              ++front;
            } else {  // the current session alone is above C: it keeps the block just brought in
              es += 1;
              ep[s] = es;
              __stcg(&owner[x], ((uint64_t)s << 32) | es);
              __stcg(&count[s], 1u);
              total = 1;
            }
          }
        }
        missed = true;
        pending &= ~(1u << stop);
        __syncwarp();
        total = __shfl_sync(kFull, total, 0);
        es = __shfl_sync(kFull, es, 0);
      }
      __syncwarp();
    }
  }
  if (lane == 0) {
    a.out[g] = hits;
    a.out[a.G + 2 * g] = sv_lo;
    a.out[a.G + 2 * g + 1] = sv_hi;
  }
}

struct SesLayout {
  DevStatus* st;
  uint64_t* owner;
  uint32_t *epoch, *count, *last;
  uint64_t sD, sS;
  uint64_t* out;
  size_t total;
};

SesLayout ses_layout(void* ws, uint64_t n_distinct, uint32_t n_session, uint32_t n_cap) {
  SesLayout L;
  Carver cv(ws);
  const uint64_t G = n_cap ? n_cap : 1;
  L.sD = n_distinct ? n_distinct : 1;
  L.sS = n_session ? n_session : 1;
  L.st = cv.take<DevStatus>(1);
  L.owner = cv.take<uint64_t>(L.sD * G);
  L.epoch = cv.take<uint32_t>(2 * L.sS * G);  // epochs, then counts: cleared together
  L.count = L.epoch + L.sS * G;
  L.last = cv.take<uint32_t>(L.sS * G);
  L.out = cv.take<uint64_t>(3 * G);
  L.total = cv.bytes();
  return L;
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_session_lru_curves_workspace_bytes(uint64_t n_distinct, uint32_t n_session, uint32_t n_cap) {
  return ses_layout(nullptr, n_distinct, n_session, n_cap).total;
}

extern "C" ptc_status ptc_session_lru_curves(const uint32_t* ids, uint64_t n, uint64_t n_distinct,
                                             const uint64_t* req_blk_off, const uint32_t* req_session,
                                             uint32_t n_req, uint32_t n_session, uint32_t block_size,
                                             const ptc_cost_model* cm, const uint64_t* cap_host, uint32_t n_cap,
                                             uint64_t* hits_host_out, ptc_u128* saved_host_out, void* ws,
                                             size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone || n_distinct > n) return PTC_ERR_INVALID_ARG;
  if (!cm || !cap_host || !hits_host_out || !saved_host_out) return PTC_ERR_INVALID_ARG;
  if (n_cap < 1 || n_cap > PTC_MAX_CAPACITIES) return PTC_ERR_INVALID_ARG;
  if (block_size < 1 || block_size > PTC_MAX_BLOCK_SIZE) return PTC_ERR_INVALID_ARG;
  if (n > 0 && (!ids || !req_blk_off || !req_session || n_req == 0 || n_session == 0 || n_distinct == 0))
    return PTC_ERR_INVALID_ARG;
  for (uint32_t g = 0; g < n_cap; ++g)
    if (cap_host[g] < 1 || (g && cap_host[g] <= cap_host[g - 1])) return PTC_ERR_INVALID_ARG;
  uint64_t alpha = 0, beta = 0;
  const ptc_status crc = cost_coeffs(cm, block_size, &alpha, &beta);
  if (crc != PTC_OK) return crc;
  if (n == 0) {
    for (uint32_t g = 0; g < n_cap; ++g) {
      hits_host_out[g] = 0;
      saved_host_out[g] = ptc_u128{0, 0};
    }
    return PTC_OK;
  }
  if (!ws_ok(ws, ws_bytes, ses_layout(nullptr, n_distinct, n_session, n_cap).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const SesLayout L = ses_layout(ws, n_distinct, n_session, n_cap);
  const FillRange zf[4] = {{ws, kStatusBytes, 0u},
                           {L.owner, sizeof(uint64_t) * L.sD * n_cap, ~0u},
                           {L.epoch, sizeof(uint32_t) * L.sS * n_cap * 2, 0u},  // epoch and count
                           {L.last, sizeof(uint32_t) * L.sS * n_cap, ~0u}};
  if (fill_many_async(zf, 4, s) != PTC_OK) return PTC_ERR_CUDA;
  PTC_KERNEL("k_ses_check", s, k_ses_check, ceil_div_u32(n_req, 256), 256, 0, req_blk_off, n_req, n, req_session,
             n_session, L.st);
  SesArgs a;
  a.ids = ids;
  a.blk_off = req_blk_off;
  a.ses = req_session;
  a.n_req = n_req;
  a.n_session = n_session;
  a.n_distinct = n_distinct;
  a.owner = L.owner;
  a.epoch = L.epoch;
  a.count = L.count;
  a.last = L.last;
  a.sD = L.sD;
  a.sS = L.sS;
  a.G = n_cap;
  a.alpha = alpha;
  a.beta = beta;
  a.out = L.out;
  a.st = L.st;
  SesCaps caps;
  for (uint32_t g = 0; g < n_cap; ++g) caps.c[g] = cap_host[g];
  const size_t smem = n_session <= kSesSmemSessions ? sizeof(uint32_t) * n_session : 0;
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(k_ses_sim, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return PTC_ERR_CUDA;
  PTC_KERNEL("k_ses_sim", s, k_ses_sim, n_cap, 32, smem, a, caps);
  HostStage* hs = host_stage();
  if (copy_to_host_async(hs->out, L.out, sizeof(uint64_t) * 3 * n_cap, s) != PTC_OK) return PTC_ERR_CUDA;
  DevStatus h;
  const ptc_status rc = end_call(L.st, s, &h);
  if (rc != PTC_OK) return rc;
  for (uint32_t g = 0; g < n_cap; ++g) {
    hits_host_out[g] = hs->out[g];
    saved_host_out[g].lo = hs->out[n_cap + 2 * g];
    saved_host_out[g].hi = hs->out[n_cap + 2 * g + 1];
  }
  return PTC_OK;
}
