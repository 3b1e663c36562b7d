// ptc_trace_stats — trace characterization over the arrays of the path
// (Sec. 4.1 lifetimes, block categories, one-hit share; Sec. 4.2 reuse
// intervals; Sec. 4.3 frequency against reuse interval and lifetime, requests
// per session; App. B reuses reachable within a capacity).
//
//   k_st_req     one thread per request: timestamp order, offsets, session
//                labels; per session its request count and first / last request
//   k_st_access  tiles of accesses: the request of every access (req_of), the
//                per-block word (frequency; "in a session with two or more
//                requests"; "in two or more sessions", decided against the
//                first session that claims the block's tag), the first and
//                last request of every block, and the stack-distance and
//                reach bins
//   k_st_blocks  one thread per block: category, frequency and lifetime bins
//   k_st_reuse   tiles of accesses: the interval of every reuse, binned by the
//                category and frequency of its block
//   k_st_sess    one thread per session: request-count and duration bins
//
// Every histogram is counted in shared memory, one update per distinct bin of
// a warp (__match_any_sync), and added to the u64 totals once per CTA.
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kStThreads = 256;
constexpr int kStPer = 8;
constexpr uint32_t kStTile = kStThreads * kStPer;
constexpr uint32_t kBins = PTC_STAT_BINS;
constexpr uint32_t kCats = PTC_STAT_CATEGORIES;
constexpr uint32_t kFreqExact = PTC_STAT_FREQ_EXACT;
// The per-block word: frequency in the low 32 bits, then two flags.
constexpr unsigned long long kMulti = 1ull << 32;  // appears in a session with >= 2 requests
constexpr unsigned long long kCross = 1ull << 33;  // appears in >= 2 sessions

typedef unsigned long long ull;

__device__ __forceinline__ uint32_t bit_len(uint64_t x) { return 64u - (uint32_t)__clzll((long long)x); }
__device__ __forceinline__ uint32_t category_of(ull w) { return (w & kMulti) ? ((w & kCross) ? 0u : 1u) : 2u; }
__host__ __device__ __forceinline__ ull* U(uint64_t* p) { return reinterpret_cast<ull*>(p); }
__device__ __forceinline__ uint32_t cdiv(uint32_t a, uint32_t b) { return a / b + (a % b != 0); }

// One shared-memory update per distinct key of the warp: the lowest lane of
// each group of equal keys calls add(key, group size).  Every lane of the
// warp must call it; kNone adds nothing.
template <class F>
__device__ __forceinline__ void warp_bin(uint32_t key, F add) {
  const uint32_t peers = __match_any_sync(kFull, key);
  if (key != kNone && (threadIdx.x & 31) == (uint32_t)(__ffs(peers) - 1)) add(key, (uint32_t)__popc(peers));
}

// Adds the nonzero entries of a shared histogram to its u64 totals.
__device__ __forceinline__ void flush(const uint32_t* s, ull* g, uint32_t len) {
  for (uint32_t j = threadIdx.x; j < len; j += blockDim.x)
    if (s[j]) atomicAdd(g + j, (ull)s[j]);
}

// Largest r in [lo, hi] with off[r] <= i.
__device__ __forceinline__ uint32_t req_search(const uint64_t* __restrict__ off, uint32_t lo, uint32_t hi,
                                               uint64_t i) {
  while (lo < hi) {
    const uint32_t mid = lo + (hi - lo + 1) / 2;
    if (__ldg(off + mid) <= i) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

struct ReqArgs {
  const uint64_t* off;
  const int64_t* ts;
  const uint32_t* sess;
  uint64_t n;
  uint32_t n_req;
  uint32_t n_session;
  uint32_t* s_cnt;
  uint32_t* s_first;
  uint32_t* s_last;
  DevStatus* st;
};

__global__ void __launch_bounds__(kStThreads) k_st_req(ReqArgs a) {
  grid_dep_sync();
  const uint32_t r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= a.n_req) return;
  const uint64_t lo = a.off[r], hi = a.off[r + 1];
  if (hi < lo || hi > a.n || (r == 0 && lo != 0) || (r + 1 == a.n_req && hi != a.n)) raise_err(a.st, kErrInvalid);
  if (r > 0 && a.ts[r] < a.ts[r - 1]) raise_err(a.st, kErrUnsorted);
  const uint32_t s = a.sess[r];
  if (s >= a.n_session) {
    raise_err(a.st, kErrInvalid);
    return;
  }
  atomicAdd(&a.s_cnt[s], 1u);
  atomicMin(&a.s_first[s], r);
  atomicMax(&a.s_last[s], r);
}

struct AccArgs {
  const uint32_t* ids;
  const uint32_t* prev;
  const uint32_t* next;
  const uint32_t* dist;  // or null
  uint32_t n;
  uint32_t D;
  const uint64_t* off;
  const uint32_t* sess;
  const uint32_t* s_cnt;
  uint32_t n_req;
  uint32_t n_session;
  uint32_t* req_of;
  ull* blk;
  uint32_t* tag;  // first session seen for each block, kNone before
  uint2* fl;      // (first request, last request) of each block
  ull* dist_bins;   // kBins
  ull* reach_bins;  // G + 1: reuses first reachable at grid point g (G: at none)
  ull* n_reuse;
  DevStatus* st;
  uint32_t G;
  uint32_t caps[PTC_MAX_CAPACITIES];  // clamped below kNone
};

__global__ void __launch_bounds__(kStThreads) k_st_access(const __grid_constant__ AccArgs a) {
  __shared__ uint32_t s_caps[PTC_MAX_CAPACITIES];
  __shared__ uint32_t s_reach[PTC_MAX_CAPACITIES + 1];
  __shared__ uint32_t s_dist[kBins];
  __shared__ uint32_t s_r[2];
  grid_dep_sync();
  for (uint32_t j = threadIdx.x; j < a.G; j += blockDim.x) s_caps[j] = a.caps[j];
  for (uint32_t j = threadIdx.x; j <= a.G; j += blockDim.x) s_reach[j] = 0;
  for (uint32_t j = threadIdx.x; j < kBins; j += blockDim.x) s_dist[j] = 0;
  const bool with_dist = a.dist != nullptr;
  uint32_t reuses = 0;
  const uint32_t tiles = cdiv(a.n, kStTile);
  for (uint32_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    const uint32_t i0 = t * kStTile;
    const uint32_t iend = a.n - i0 < kStTile ? a.n : i0 + kStTile;
    __syncthreads();
    if (threadIdx.x == 0) {
      const uint32_t r0 = req_search(a.off, 0, a.n_req - 1, i0);
      s_r[0] = r0;
      s_r[1] = req_search(a.off, r0, a.n_req - 1, iend - 1);
    }
    __syncthreads();
    const uint32_t r0 = s_r[0], r1 = s_r[1];
    uint32_t id[kStPer], pv[kStPer], nx[kStPer], dv[kStPer];
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      const uint32_t i = i0 + k * kStThreads + threadIdx.x;
      const bool in = (uint64_t)i0 + k * kStThreads + threadIdx.x < iend;
      id[k] = in ? __ldg(a.ids + i) : 0u;
      pv[k] = in ? __ldg(a.prev + i) : kNone;
      nx[k] = in ? __ldg(a.next + i) : 0u;
      dv[k] = in && with_dist ? __ldg(a.dist + i) : kNone;
    }
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      const uint32_t i = i0 + k * kStThreads + threadIdx.x;
      bool ok = (uint64_t)i0 + k * kStThreads + threadIdx.x < iend;
      uint32_t key = kNone;
      if (ok) {
        const uint32_t r = req_search(a.off, r0, r1, i);
        a.req_of[i] = r;
        const uint32_t d = id[k], p = pv[k], x = nx[k];
        if (d >= a.D || (p != kNone && p >= i) || (x != kNone && (x <= i || x >= a.n))) {
          raise_err(a.st, kErrInvalid);
          ok = false;
        }
        const uint32_t s = ok ? __ldg(a.sess + r) : kNone;
        if (ok && s < a.n_session) {
          const ull w = atomicAdd(&a.blk[d], 1ull);
          ull set = 0;
          if (!(w & kMulti) && __ldg(a.s_cnt + s) >= 2u) set |= kMulti;
          if (!(w & kCross)) {
            // The tag only ever changes from kNone to one session, so any
            // other value read (even a stale one) is final.
            uint32_t v = a.tag[d];
            if (v == kNone) v = atomicCAS(&a.tag[d], kNone, s);
            if (v != kNone && v != s) set |= kCross;
          }
          if (set) atomicOr(&a.blk[d], set);
        }
        if (ok) {
          if (p == kNone) a.fl[d].x = r;
          if (x == kNone) a.fl[d].y = r;
          if (p != kNone) {
            ++reuses;
            if (with_dist) {
              const uint32_t dd = dv[k];
              uint32_t lo = 0, hi = a.G;  // first grid point with cap >= dd
              while (lo < hi) {
                const uint32_t mid = (lo + hi) >> 1;
                if (s_caps[mid] < dd) lo = mid + 1;
                else hi = mid;
              }
              key = bit_len(dd) | (lo << 7);
            }
          }
        }
      }
      warp_bin(key, [&](uint32_t kk, uint32_t c) {
        atomicAdd(&s_dist[kk & 127u], c);
        atomicAdd(&s_reach[kk >> 7], c);
      });
    }
  }
  __syncthreads();
  flush(s_dist, a.dist_bins, kBins);
  flush(s_reach, a.reach_bins, a.G + 1);
  const uint32_t wsum = __reduce_add_sync(kFull, reuses);
  if ((threadIdx.x & 31) == 0 && wsum) atomicAdd(a.n_reuse, (ull)wsum);
}

struct BlkArgs {
  const ull* blk;
  const uint2* fl;
  const int64_t* ts;
  uint32_t D;
  uint32_t n_req;
  ptc_trace_summary* out;
  DevStatus* st;
};

__global__ void __launch_bounds__(kStThreads) k_st_blocks(const __grid_constant__ BlkArgs a) {
  __shared__ uint32_t s_freq[kCats * kFreqExact];
  __shared__ uint32_t s_flog[kCats * kBins];
  __shared__ uint32_t s_life[kCats * kBins];
  __shared__ uint32_t s_lbf[kBins * kBins];
  grid_dep_sync();
  for (uint32_t j = threadIdx.x; j < kCats * kFreqExact; j += blockDim.x) s_freq[j] = 0;
  for (uint32_t j = threadIdx.x; j < kCats * kBins; j += blockDim.x) s_flog[j] = s_life[j] = 0;
  for (uint32_t j = threadIdx.x; j < kBins * kBins; j += blockDim.x) s_lbf[j] = 0;
  __syncthreads();
  uint32_t nblk[kCats] = {0, 0, 0};
  ull nacc[kCats] = {0, 0, 0};
  const uint32_t stride = gridDim.x * blockDim.x;
  const uint32_t rounds = cdiv(a.D, stride);
  for (uint32_t round = 0; round < rounds; ++round) {
    const uint32_t d = round * stride + blockIdx.x * blockDim.x + threadIdx.x;
    uint32_t key = kNone;
    if (d < a.D) {
      const ull w = a.blk[d];
      const uint2 fl = a.fl[d];
      const uint32_t f = (uint32_t)w;
      if (f == 0 || fl.x >= a.n_req || fl.y >= a.n_req) {
        raise_err(a.st, kErrInvalid);
      } else {
        const uint32_t c = category_of(w);
        const uint64_t life = (uint64_t)(__ldg(a.ts + fl.y) - __ldg(a.ts + fl.x));
        const uint32_t fe = f < kFreqExact ? f : 0u;
        key = c | (fe << 2) | (bit_len(life) << 10) | (bit_len(f) << 17);
#pragma unroll
        for (uint32_t cc = 0; cc < kCats; ++cc) {
          nblk[cc] += cc == c;
          nacc[cc] += cc == c ? f : 0u;
        }
      }
    }
    warp_bin(key, [&](uint32_t kk, uint32_t cnt) {
      const uint32_t c = kk & 3u, fe = (kk >> 2) & 255u, bl = (kk >> 10) & 127u, bf = kk >> 17;
      atomicAdd(&s_freq[c * kFreqExact + fe], cnt);
      atomicAdd(&s_flog[c * kBins + bf], cnt);
      atomicAdd(&s_life[c * kBins + bl], cnt);
      atomicAdd(&s_lbf[bf * kBins + bl], cnt);
    });
  }
  __syncthreads();
  ptc_trace_summary* o = a.out;
  flush(s_freq, U(&o->freq[0][0]), kCats * kFreqExact);
  flush(s_flog, U(&o->freq_log2[0][0]), kCats * kBins);
  flush(s_life, U(&o->lifetime_us[0][0]), kCats * kBins);
  flush(s_lbf, U(&o->lifetime_by_freq[0][0]), kBins * kBins);
#pragma unroll
  for (uint32_t c = 0; c < kCats; ++c) {
    const uint32_t b = __reduce_add_sync(kFull, nblk[c]);
    ull s = nacc[c];
    for (int o2 = 16; o2 > 0; o2 >>= 1) s += __shfl_xor_sync(kFull, s, o2);
    if ((threadIdx.x & 31) == 0) {
      if (b) atomicAdd(U(&o->blocks[c]), (ull)b);
      if (s) atomicAdd(U(&o->accesses[c]), s);
    }
  }
}

struct ReuseArgs {
  const uint32_t* ids;
  const uint32_t* prev;
  const uint32_t* req_of;
  const ull* blk;
  const int64_t* ts;
  uint32_t n;
  uint32_t D;
  ptc_trace_summary* out;
};

__global__ void __launch_bounds__(kStThreads) k_st_reuse(const __grid_constant__ ReuseArgs a) {
  __shared__ uint32_t s_ru[kCats * kBins];
  __shared__ uint32_t s_rbf[kBins * kBins];
  grid_dep_sync();
  for (uint32_t j = threadIdx.x; j < kCats * kBins; j += blockDim.x) s_ru[j] = 0;
  for (uint32_t j = threadIdx.x; j < kBins * kBins; j += blockDim.x) s_rbf[j] = 0;
  __syncthreads();
  const uint32_t tiles = cdiv(a.n, kStTile);
  for (uint32_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    const uint32_t i0 = t * kStTile;
    uint32_t pv[kStPer];
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      const uint64_t i = (uint64_t)i0 + k * kStThreads + threadIdx.x;
      pv[k] = i < a.n ? __ldg(a.prev + i) : kNone;
    }
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      const uint64_t i = (uint64_t)i0 + k * kStThreads + threadIdx.x;
      const uint32_t p = pv[k];
      uint32_t key = kNone;
      // out-of-range ids or prev were reported by k_st_access; skip them here
      if (p < i && i < a.n) {
        const uint32_t d = __ldg(a.ids + i);
        if (d < a.D) {
          const ull w = a.blk[d];
          const uint64_t gap = (uint64_t)(__ldg(a.ts + __ldg(a.req_of + i)) - __ldg(a.ts + __ldg(a.req_of + p)));
          key = category_of(w) | (bit_len(gap) << 2) | (bit_len((uint32_t)w) << 9);
        }
      }
      warp_bin(key, [&](uint32_t kk, uint32_t cnt) {
        const uint32_t c = kk & 3u, bg = (kk >> 2) & 127u, bf = kk >> 9;
        atomicAdd(&s_ru[c * kBins + bg], cnt);
        atomicAdd(&s_rbf[bf * kBins + bg], cnt);
      });
    }
  }
  __syncthreads();
  flush(s_ru, U(&a.out->reuse_us[0][0]), kCats * kBins);
  flush(s_rbf, U(&a.out->reuse_by_freq[0][0]), kBins * kBins);
}

struct SessArgs {
  const uint32_t* s_cnt;
  const uint32_t* s_first;
  const uint32_t* s_last;
  const int64_t* ts;
  uint32_t n_session;
  uint32_t n_req;
  ptc_trace_summary* out;
};

__global__ void __launch_bounds__(kStThreads) k_st_sess(SessArgs a) {
  __shared__ uint32_t s_req[kBins];
  __shared__ uint32_t s_dur[kBins];
  grid_dep_sync();
  for (uint32_t j = threadIdx.x; j < kBins; j += blockDim.x) s_req[j] = s_dur[j] = 0;
  __syncthreads();
  uint32_t used = 0, multi = 0;
  const uint32_t stride = gridDim.x * blockDim.x;
  const uint32_t rounds = cdiv(a.n_session, stride);
  for (uint32_t round = 0; round < rounds; ++round) {
    const uint32_t s = round * stride + blockIdx.x * blockDim.x + threadIdx.x;
    uint32_t key = kNone;
    if (s < a.n_session) {
      const uint32_t c = a.s_cnt[s];
      const uint32_t f = a.s_first[s], l = a.s_last[s];
      if (c > 0 && f < a.n_req && l < a.n_req) {
        ++used;
        multi += c >= 2u;
        key = bit_len(c) | (bit_len((uint64_t)(__ldg(a.ts + l) - __ldg(a.ts + f))) << 7);
      }
    }
    warp_bin(key, [&](uint32_t kk, uint32_t cnt) {
      atomicAdd(&s_req[kk & 127u], cnt);
      atomicAdd(&s_dur[kk >> 7], cnt);
    });
  }
  __syncthreads();
  flush(s_req, U(&a.out->sess_requests[0]), kBins);
  flush(s_dur, U(&a.out->sess_duration_us[0]), kBins);
  const uint32_t u = __reduce_add_sync(kFull, used), m = __reduce_add_sync(kFull, multi);
  if ((threadIdx.x & 31) == 0) {
    if (u) atomicAdd(U(&a.out->n_sessions), (ull)u);
    if (m) atomicAdd(U(&a.out->n_multi_sessions), (ull)m);
  }
}

struct StatsLayout {
  DevStatus* st;
  ptc_trace_summary* out;
  ull* reach_bins;
  uint32_t* s_cnt;
  uint32_t* s_last;
  ull* blk;
  size_t zero_bytes;   // [0, zero_bytes) starts at zero
  uint32_t* s_first;   // these three start at all ones
  uint32_t* tag;
  uint2* fl;
  size_t ones_from, ones_bytes;
  uint32_t* req_of;
  size_t total;
};

StatsLayout stats_layout(void* ws, uint64_t n, uint64_t D, uint32_t n_session) {
  StatsLayout L;
  Carver cv(ws);
  L.st = cv.take<DevStatus>(1);
  L.out = cv.take<ptc_trace_summary>(1);
  L.reach_bins = cv.take<ull>(PTC_MAX_CAPACITIES + 1);
  L.s_cnt = cv.take<uint32_t>(n_session);
  L.s_last = cv.take<uint32_t>(n_session);
  L.blk = cv.take<ull>(D);
  L.zero_bytes = cv.off;
  L.ones_from = cv.bytes();
  L.s_first = cv.take<uint32_t>(n_session);
  L.tag = cv.take<uint32_t>(D);
  L.fl = cv.take<uint2>(D);
  L.ones_bytes = cv.off - L.ones_from;
  L.req_of = cv.take<uint32_t>(n);
  L.total = cv.bytes();
  return L;
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_trace_stats_workspace_bytes(uint64_t n, uint64_t n_distinct, uint32_t n_req,
                                                  uint32_t n_session) {
  (void)n_req;
  return stats_layout(nullptr, n, n_distinct, n_session).total;
}

extern "C" ptc_status ptc_trace_stats(const uint32_t* ids, const uint32_t* prev, const uint32_t* next,
                                      const uint32_t* dist, uint64_t n, uint64_t n_distinct,
                                      const uint64_t* req_blk_off, const int64_t* req_ts_us,
                                      const uint32_t* req_session, uint32_t n_req, uint32_t n_session,
                                      const uint64_t* cap_host, uint32_t n_cap, uint64_t* reach_host_out,
                                      ptc_trace_summary* stats_host_out, void* ws, size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone || n_distinct >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (!stats_host_out || n_distinct > n || (n > 0 && n_distinct == 0)) return PTC_ERR_INVALID_ARG;
  if (n_cap > PTC_MAX_CAPACITIES || (n_cap > 0 && (!cap_host || !reach_host_out || (n > 0 && !dist))))
    return PTC_ERR_INVALID_ARG;
  for (uint32_t g = 0; g < n_cap; ++g)
    if (cap_host[g] < 1 || (g && cap_host[g] <= cap_host[g - 1])) return PTC_ERR_INVALID_ARG;
  if (n > 0 && (!ids || !prev || !next || n_req == 0)) return PTC_ERR_INVALID_ARG;
  if (n_req > 0 && (!req_blk_off || !req_ts_us || !req_session || n_session == 0)) return PTC_ERR_INVALID_ARG;
  if (!ws_ok(ws, ws_bytes, stats_layout(nullptr, n, n_distinct, n_session).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const StatsLayout L = stats_layout(ws, n, n_distinct, n_session);
  if (begin_call(ws, L.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  if (fill_async((char*)ws + L.ones_from, 0xFFFFFFFFu, L.ones_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  const int sms = num_sms();
  if (n_req > 0) {
    const ReqArgs ra{req_blk_off, req_ts_us, req_session, n, n_req, n_session, L.s_cnt, L.s_first, L.s_last, L.st};
    PTC_KERNEL("k_st_req", s, k_st_req, ceil_div_u32(n_req, kStThreads), kStThreads, 0, ra);
  }
  if (n > 0) {
    const uint32_t tiles = ceil_div_u32(n, kStTile);
    const uint32_t grid = tiles < (uint32_t)(4 * sms) ? tiles : (uint32_t)(4 * sms);
    AccArgs aa;
    aa.ids = ids;
    aa.prev = prev;
    aa.next = next;
    aa.dist = dist;
    aa.n = (uint32_t)n;
    aa.D = (uint32_t)n_distinct;
    aa.off = req_blk_off;
    aa.sess = req_session;
    aa.s_cnt = L.s_cnt;
    aa.n_req = n_req;
    aa.n_session = n_session;
    aa.req_of = L.req_of;
    aa.blk = L.blk;
    aa.tag = L.tag;
    aa.fl = L.fl;
    aa.dist_bins = U(&L.out->dist_log2[0]);
    aa.reach_bins = L.reach_bins;
    aa.n_reuse = U(&L.out->n_reuse);
    aa.st = L.st;
    aa.G = n_cap;
    for (uint32_t g = 0; g < n_cap; ++g) aa.caps[g] = cap_host[g] >= (uint64_t)kNone ? kNone - 1 : (uint32_t)cap_host[g];
    PTC_KERNEL("k_st_access", s, k_st_access, grid, kStThreads, 0, aa);
    const BlkArgs ba{L.blk, L.fl, req_ts_us, (uint32_t)n_distinct, n_req, L.out, L.st};
    const uint32_t bgrid0 = ceil_div_u32(n_distinct, kStThreads);
    const uint32_t bgrid = bgrid0 < (uint32_t)(4 * sms) ? bgrid0 : (uint32_t)(4 * sms);
    PTC_KERNEL("k_st_blocks", s, k_st_blocks, bgrid, kStThreads, 0, ba);
    const ReuseArgs rua{ids, prev, L.req_of, L.blk, req_ts_us, (uint32_t)n, (uint32_t)n_distinct, L.out};
    PTC_KERNEL("k_st_reuse", s, k_st_reuse, grid, kStThreads, 0, rua);
  }
  if (n_session > 0 && n_req > 0) {
    const uint32_t sgrid0 = ceil_div_u32(n_session, kStThreads);
    const uint32_t sgrid = sgrid0 < (uint32_t)(2 * sms) ? sgrid0 : (uint32_t)(2 * sms);
    const SessArgs sa{L.s_cnt, L.s_first, L.s_last, req_ts_us, n_session, n_req, L.out};
    PTC_KERNEL("k_st_sess", s, k_st_sess, sgrid, kStThreads, 0, sa);
  }
  if (cudaMemcpyAsync(stats_host_out, L.out, sizeof(ptc_trace_summary), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return PTC_ERR_CUDA;
  uint64_t* bins = nullptr;
  if (n_cap > 0) {
    bins = host_stage()->out;  // PTC_MAX_CAPACITIES + 1 <= 3 * PTC_MAX_CAPACITIES + 2 entries
    if (copy_to_host_async(bins, L.reach_bins, sizeof(uint64_t) * (n_cap + 1), s) != PTC_OK) return PTC_ERR_CUDA;
  }
  DevStatus h;
  const ptc_status rc = end_call(L.st, s, &h);
  if (rc != PTC_OK) return rc;
  stats_host_out->n_access = n;
  stats_host_out->n_distinct = n_distinct;
  uint64_t run = 0;
  for (uint32_t g = 0; g < n_cap; ++g) reach_host_out[g] = (run += bins[g]);
  return PTC_OK;
}
