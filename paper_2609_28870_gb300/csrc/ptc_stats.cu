// ptc_trace_stats — trace characterization over the arrays of the path
// (Sec. 4.1 lifetimes, block categories, one-hit share; Sec. 4.2 reuse
// intervals; Sec. 4.3 frequency against reuse interval and lifetime, requests
// per session; App. B reuses reachable within a capacity).
//
//   k_st_req     one thread per request: timestamp order, offsets, session
//                labels; per session its request count and first / last request
//   k_st_access  tiles of accesses: the request of every access (req_of), the
//                frequency and flags of every block ("in two or more
//                sessions", decided against the first session that claims
//                the block's tag; "in a session with two or more requests"),
//                the first and last request of every block, and the
//                stack-distance and reach bins
//   k_st_blocks  one thread per block: category, frequency and lifetime bins,
//                and a class byte (category, frequency bin) per block; then
//                one thread per session: request-count and duration bins
//   k_st_reuse   tiles of accesses: the interval of every reuse, binned by the
//                category and frequency of its block (its class byte)
//
// Every histogram is counted in shared memory, one update per distinct bin of
// a warp (__match_any_sync), and added to the u64 totals once per CTA.
#include <cstring>

#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kStThreads = 256;
constexpr int kStPer = 4;
constexpr uint32_t kStTile = kStThreads * kStPer;
constexpr uint32_t kBins = PTC_STAT_BINS;
constexpr uint32_t kCats = PTC_STAT_CATEGORIES;
constexpr uint32_t kFreqExact = PTC_STAT_FREQ_EXACT;
// Per-block flags.
constexpr uint32_t kFlagMulti = 1u;  // appears in a session with >= 2 requests
constexpr uint32_t kFlagCross = 2u;  // appears in >= 2 sessions

typedef unsigned long long ull;

__device__ __forceinline__ uint32_t bit_len(uint64_t x) { return 64u - (uint32_t)__clzll((long long)x); }
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
  uint32_t* tile_req;  // request holding the first access of each access tile; [tiles] = n_req - 1
  uint32_t tiles;
  DevStatus* st;
};

__global__ void __launch_bounds__(kStThreads) k_st_req(ReqArgs a) {
  grid_dep_sync();
  const uint32_t r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= a.n_req) return;
  const uint64_t lo = a.off[r], hi = a.off[r + 1];
  if (hi < lo || hi > a.n || (r == 0 && lo != 0) || (r + 1 == a.n_req && hi != a.n)) raise_err(a.st, kErrInvalid);
  if (r > 0 && a.ts[r] < a.ts[r - 1]) raise_err(a.st, kErrUnsorted);
  if (hi > lo && hi <= a.n)
    for (uint64_t t = (lo + kStTile - 1) / kStTile; t * kStTile < hi; ++t) a.tile_req[t] = r;
  if (r + 1 == a.n_req) a.tile_req[a.tiles] = r;
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
  const uint32_t* tile_req;
  uint32_t* req_of;
  uint32_t* cnt;    // accesses of each block
  uint32_t* flg;    // kFlagMulti / kFlagCross of each block
  uint32_t* tag;    // 1 + the first session that claimed the block, 0 before
  uint2* fl;        // (first request, last request) of each block
  ull* dist_bins;   // kBins
  ull* reach_bins;  // G + 1: reuses first reachable at grid point g (G: at none)
  ull* n_reuse;
  DevStatus* st;
  uint32_t G;
  uint32_t caps[PTC_MAX_CAPACITIES];  // clamped below kNone
};

// Access pass.  The two-sessions test: a block's tag is claimed once, by the
// first session whose access gets to it; an access of any other session sees
// a different tag and marks the block as crossing sessions (and, if its own
// session has two or more requests, as appearing in such a session; the
// claiming session's request count is looked up in the block pass).  The tag
// only ever changes from 0 to its final value, so any nonzero value read,
// even a stale one, is final.  Loads are issued for all of a thread's
// accesses before any result is used.
__global__ void __launch_bounds__(kStThreads, 6) k_st_access(const __grid_constant__ AccArgs a) {
  __shared__ uint32_t s_caps[PTC_MAX_CAPACITIES];
  __shared__ uint32_t s_reach[PTC_MAX_CAPACITIES + 1];
  __shared__ uint32_t s_dist[kBins];
  __shared__ uint32_t s_oct[34];  // s_oct[b]: first grid point with cap >= 2^(b-1) (b >= 1)
  grid_dep_sync();
  for (uint32_t j = threadIdx.x; j < a.G; j += blockDim.x) s_caps[j] = a.caps[j];
  for (uint32_t j = threadIdx.x; j <= a.G; j += blockDim.x) s_reach[j] = 0;
  for (uint32_t j = threadIdx.x; j < kBins; j += blockDim.x) s_dist[j] = 0;
  if (threadIdx.x < 34) {
    const uint64_t x = threadIdx.x == 0 ? 0 : 1ull << (threadIdx.x - 1);
    uint32_t lo = 0, hi = a.G;
    while (lo < hi) {
      const uint32_t mid = (lo + hi) >> 1;
      if ((uint64_t)a.caps[mid] < x) lo = mid + 1;
      else hi = mid;
    }
    s_oct[threadIdx.x] = lo;
  }
  __syncthreads();
  const bool with_dist = a.dist != nullptr;
  uint32_t reuses = 0;
  const uint32_t tiles = cdiv(a.n, kStTile);
  for (uint32_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    const uint32_t i0 = t * kStTile;
    const uint32_t iend = a.n - i0 < kStTile ? a.n : i0 + kStTile;
    // requests of the tile: from the one holding its first access to the one
    // holding the next tile's first access (clamped: malformed offsets have
    // raised an error already)
    uint32_t r0 = __ldg(a.tile_req + t), r1 = __ldg(a.tile_req + t + 1);
    r0 = r0 < a.n_req ? r0 : a.n_req - 1;
    r1 = r1 < a.n_req ? (r1 > r0 ? r1 : r0) : a.n_req - 1;
    uint32_t id[kStPer], pv[kStPer], nx[kStPer], dv[kStPer], rq[kStPer], ss[kStPer], tg[kStPer];
    bool ok[kStPer];
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      const uint32_t i = i0 + k * kStThreads + threadIdx.x;
      const bool in = (uint64_t)i0 + k * kStThreads + threadIdx.x < iend;
      id[k] = in ? __ldg(a.ids + i) : 0u;
      pv[k] = in ? __ldg(a.prev + i) : kNone;
      nx[k] = in ? __ldg(a.next + i) : 0u;
      dv[k] = in && with_dist ? __ldg(a.dist + i) : kNone;
      ok[k] = in;
    }
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      const uint32_t i = i0 + k * kStThreads + threadIdx.x;
      rq[k] = 0;
      ss[k] = kNone;
      if (ok[k]) {
        rq[k] = req_search(a.off, r0, r1, i);
        a.req_of[i] = rq[k];
        const uint32_t d = id[k], p = pv[k], x = nx[k];
        if (d >= a.D || (p != kNone && p >= i) || (x != kNone && (x <= i || x >= a.n))) {
          raise_err(a.st, kErrInvalid);
          ok[k] = false;
        } else {
          ss[k] = __ldg(a.sess + rq[k]);
        }
      }
    }
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      tg[k] = 0;
      if (ok[k] && ss[k] < a.n_session) {
        atomicAdd(&a.cnt[id[k]], 1u);
        tg[k] = a.tag[id[k]];
      }
    }
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      if (ok[k] && ss[k] < a.n_session) {
        const uint32_t mine = ss[k] + 1;
        uint32_t v = tg[k];
        if (v == 0) v = atomicCAS(&a.tag[id[k]], 0u, mine);
        if (v != 0 && v != mine)
          atomicOr(&a.flg[id[k]], kFlagCross | (__ldg(a.s_cnt + ss[k]) >= 2u ? kFlagMulti : 0u));
      }
    }
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      uint32_t key = kNone;
      if (ok[k]) {
        const uint32_t d = id[k], p = pv[k];
        if (p == kNone) a.fl[d].x = rq[k];
        if (nx[k] == kNone) a.fl[d].y = rq[k];
        if (p != kNone) {
          ++reuses;
          if (with_dist) {
            // first grid point with cap >= dd: between those of the powers
            // of two around dd (2^(b-1) <= dd < 2^b, b = bit length of dd)
            const uint32_t dd = dv[k], b = bit_len(dd);
            uint32_t lo = s_oct[b], hi = s_oct[b < 33 ? b + 1 : 33];
            while (lo < hi) {
              const uint32_t mid = (lo + hi) >> 1;
              if (s_caps[mid] < dd) lo = mid + 1;
              else hi = mid;
            }
            key = b | (lo << 7);
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
  const uint32_t* cnt;
  const uint32_t* flg;
  const uint32_t* tag;
  const uint2* fl;
  const int64_t* ts;
  const uint32_t* s_cnt;
  const uint32_t* s_first;
  const uint32_t* s_last;
  uint8_t* cls;  // category | bit_len(frequency) << 2, for the reuse pass
  uint32_t D;
  uint32_t n_req;
  uint32_t n_session;
  ptc_trace_summary* out;
  DevStatus* st;
};

constexpr int kBlkPer = 4;

// Block pass (categories, frequency and lifetime bins, the class byte of
// every block), then the session bins.
__global__ void __launch_bounds__(kStThreads) k_st_blocks(const __grid_constant__ BlkArgs a) {
  __shared__ uint32_t s_freq[kCats * kFreqExact];
  __shared__ uint32_t s_flog[kCats * kBins];
  __shared__ uint32_t s_life[kCats * kBins];
  __shared__ uint32_t s_lbf[kBins * kBins];
  __shared__ uint32_t s_req[kBins];
  __shared__ uint32_t s_dur[kBins];
  grid_dep_sync();
  for (uint32_t j = threadIdx.x; j < kCats * kFreqExact; j += blockDim.x) s_freq[j] = 0;
  for (uint32_t j = threadIdx.x; j < kCats * kBins; j += blockDim.x) s_flog[j] = s_life[j] = 0;
  for (uint32_t j = threadIdx.x; j < kBins * kBins; j += blockDim.x) s_lbf[j] = 0;
  for (uint32_t j = threadIdx.x; j < kBins; j += blockDim.x) s_req[j] = s_dur[j] = 0;
  __syncthreads();
  uint32_t nblk[kCats] = {0, 0, 0};
  ull nacc[kCats] = {0, 0, 0};
  const uint32_t chunk = gridDim.x * blockDim.x * kBlkPer;
  const uint32_t rounds = cdiv(a.D, chunk);
  for (uint32_t round = 0; round < rounds; ++round) {
    const uint64_t base = (uint64_t)round * chunk + (uint64_t)blockIdx.x * blockDim.x * kBlkPer + threadIdx.x;
    uint32_t f[kBlkPer], fg[kBlkPer], tg[kBlkPer];
    uint2 fl[kBlkPer];
#pragma unroll
    for (int k = 0; k < kBlkPer; ++k) {
      const uint64_t d = base + (uint64_t)k * blockDim.x;
      const bool in = d < a.D;
      f[k] = in ? a.cnt[d] : 0u;
      fg[k] = in ? a.flg[d] : 0u;
      tg[k] = in ? a.tag[d] : 0u;
      fl[k] = in ? a.fl[d] : make_uint2(kNone, kNone);
    }
#pragma unroll
    for (int k = 0; k < kBlkPer; ++k) {
      const uint64_t d = base + (uint64_t)k * blockDim.x;
      uint32_t key = kNone;
      if (d < a.D) {
        if (f[k] == 0 || fl[k].x >= a.n_req || fl[k].y >= a.n_req || tg[k] == 0 || tg[k] > a.n_session) {
          raise_err(a.st, kErrInvalid);
        } else {
          const bool multi = (fg[k] & kFlagMulti) || __ldg(a.s_cnt + tg[k] - 1) >= 2u;
          const uint32_t c = multi ? ((fg[k] & kFlagCross) ? 0u : 1u) : 2u;
          const uint64_t life = (uint64_t)(__ldg(a.ts + fl[k].y) - __ldg(a.ts + fl[k].x));
          const uint32_t fe = f[k] < kFreqExact ? f[k] : 0u, bf = bit_len(f[k]);
          a.cls[d] = (uint8_t)(c | (bf << 2));
          key = c | (fe << 2) | (bit_len(life) << 10) | (bf << 17);
#pragma unroll
          for (uint32_t cc = 0; cc < kCats; ++cc) {
            nblk[cc] += cc == c;
            nacc[cc] += cc == c ? f[k] : 0u;
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
  }
  // sessions
  uint32_t used = 0, multi_s = 0;
  const uint32_t stride = gridDim.x * blockDim.x;
  const uint32_t srounds = cdiv(a.n_session, stride);
  for (uint32_t round = 0; round < srounds; ++round) {
    const uint32_t s = round * stride + blockIdx.x * blockDim.x + threadIdx.x;
    uint32_t key = kNone;
    if (s < a.n_session) {
      const uint32_t c = a.s_cnt[s];
      const uint32_t fr = a.s_first[s], lr = a.s_last[s];
      if (c > 0 && fr < a.n_req && lr < a.n_req) {
        ++used;
        multi_s += c >= 2u;
        key = bit_len(c) | (bit_len((uint64_t)(__ldg(a.ts + lr) - __ldg(a.ts + fr))) << 7);
      }
    }
    warp_bin(key, [&](uint32_t kk, uint32_t cnt) {
      atomicAdd(&s_req[kk & 127u], cnt);
      atomicAdd(&s_dur[kk >> 7], cnt);
    });
  }
  __syncthreads();
  ptc_trace_summary* o = a.out;
  flush(s_freq, U(&o->freq[0][0]), kCats * kFreqExact);
  flush(s_flog, U(&o->freq_log2[0][0]), kCats * kBins);
  flush(s_life, U(&o->lifetime_us[0][0]), kCats * kBins);
  flush(s_lbf, U(&o->lifetime_by_freq[0][0]), kBins * kBins);
  flush(s_req, U(&o->sess_requests[0]), kBins);
  flush(s_dur, U(&o->sess_duration_us[0]), kBins);
#pragma unroll
  for (uint32_t c = 0; c < kCats; ++c) {
    const uint32_t b = __reduce_add_sync(kFull, nblk[c]);
    ull sum = nacc[c];
    for (int o2 = 16; o2 > 0; o2 >>= 1) sum += __shfl_xor_sync(kFull, sum, o2);
    if ((threadIdx.x & 31) == 0) {
      if (b) atomicAdd(U(&o->blocks[c]), (ull)b);
      if (sum) atomicAdd(U(&o->accesses[c]), sum);
    }
  }
  const uint32_t u = __reduce_add_sync(kFull, used), m = __reduce_add_sync(kFull, multi_s);
  if ((threadIdx.x & 31) == 0) {
    if (u) atomicAdd(U(&o->n_sessions), (ull)u);
    if (m) atomicAdd(U(&o->n_multi_sessions), (ull)m);
  }
}

struct ReuseArgs {
  const uint32_t* ids;
  const uint32_t* prev;
  const uint32_t* req_of;
  const uint8_t* cls;
  const int64_t* ts;
  uint32_t n;
  uint32_t D;
  ptc_trace_summary* out;
};

// Reuse pass: the interval of every reuse, binned by its block's category
// and frequency (the class byte).  The random loads (the previous access's
// request, the class byte, two arrival times) are issued for all of a
// thread's accesses before any is used.
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
    uint32_t pv[kStPer], id[kStPer], ri[kStPer], rp[kStPer], cl[kStPer];
    bool use[kStPer];
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      const uint64_t i = (uint64_t)i0 + k * kStThreads + threadIdx.x;
      const bool in = i < a.n;
      pv[k] = in ? __ldg(a.prev + i) : kNone;
      id[k] = in ? __ldg(a.ids + i) : 0u;
      ri[k] = in ? __ldg(a.req_of + i) : 0u;
      // out-of-range ids or prev were reported by the access pass; skip them
      use[k] = in && pv[k] < i && id[k] < a.D;
    }
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      rp[k] = use[k] ? __ldg(a.req_of + pv[k]) : 0u;
      cl[k] = use[k] ? (uint32_t)__ldg(a.cls + id[k]) : 0u;
    }
#pragma unroll
    for (int k = 0; k < kStPer; ++k) {
      uint32_t key = kNone;
      if (use[k]) {
        const uint64_t gap = (uint64_t)(__ldg(a.ts + ri[k]) - __ldg(a.ts + rp[k]));
        key = (cl[k] & 3u) | (bit_len(gap) << 2) | ((cl[k] >> 2) << 9);
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

struct StatsLayout {
  DevStatus* st;
  ptc_trace_summary* out;  // the summary, then the reach bins right after it
  ull* reach_bins;
  uint32_t* s_cnt;
  uint32_t* s_last;
  uint32_t* cnt;
  uint32_t* flg;
  uint32_t* tag;
  size_t zero_bytes;   // [0, zero_bytes) starts at zero
  uint32_t* s_first;   // these two start at all ones
  uint2* fl;
  size_t ones_from, ones_bytes;
  uint8_t* cls;
  uint32_t* req_of;
  uint32_t* tile_req;
  size_t total;
};

// One wave of CTAs (as many as fit on every SM at once), or fewer if there
// is less work: the kernels above loop over their tiles.
template <class K>
uint32_t persistent_grid(K kernel, int threads, int sms, uint32_t work) {
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, 0) != cudaSuccess || per_sm < 1)
    per_sm = 1;
  const uint32_t wave = (uint32_t)(per_sm * sms);
  return work < wave ? (work ? work : 1u) : wave;
}

StatsLayout stats_layout(void* ws, uint64_t n, uint64_t D, uint32_t n_session) {
  StatsLayout L;
  Carver cv(ws);
  L.st = cv.take<DevStatus>(1);
  L.out = cv.take<ptc_trace_summary>(1);
  L.reach_bins = cv.take<ull>(PTC_MAX_CAPACITIES + 1, 8);
  L.s_cnt = cv.take<uint32_t>(n_session);
  L.s_last = cv.take<uint32_t>(n_session);
  L.cnt = cv.take<uint32_t>(D);
  L.flg = cv.take<uint32_t>(D);
  L.tag = cv.take<uint32_t>(D);
  L.zero_bytes = cv.off;
  L.ones_from = cv.bytes();
  L.s_first = cv.take<uint32_t>(n_session);
  L.fl = cv.take<uint2>(D);
  L.ones_bytes = cv.off - L.ones_from;
  L.cls = cv.take<uint8_t>(D);
  L.req_of = cv.take<uint32_t>(n);
  L.tile_req = cv.take<uint32_t>((n + kStTile - 1) / kStTile + 1);
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
    const ReqArgs ra{req_blk_off, req_ts_us, req_session, n, n_req, n_session, L.s_cnt, L.s_first, L.s_last,
                     L.tile_req, ceil_div_u32(n, kStTile), L.st};
    PTC_KERNEL("k_st_req", s, k_st_req, ceil_div_u32(n_req, kStThreads), kStThreads, 0, ra);
  }
  const uint32_t tiles = ceil_div_u32(n, kStTile);
  const uint32_t grid_acc = persistent_grid(k_st_access, kStThreads, sms, tiles);
  const uint32_t grid_reuse = persistent_grid(k_st_reuse, kStThreads, sms, tiles);
  if (n > 0) {
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
    aa.tile_req = L.tile_req;
    aa.req_of = L.req_of;
    aa.cnt = L.cnt;
    aa.flg = L.flg;
    aa.tag = L.tag;
    aa.fl = L.fl;
    aa.dist_bins = U(&L.out->dist_log2[0]);
    aa.reach_bins = L.reach_bins;
    aa.n_reuse = U(&L.out->n_reuse);
    aa.st = L.st;
    aa.G = n_cap;
    for (uint32_t g = 0; g < n_cap; ++g) aa.caps[g] = cap_host[g] >= (uint64_t)kNone ? kNone - 1 : (uint32_t)cap_host[g];
    PTC_KERNEL("k_st_access", s, k_st_access, grid_acc, kStThreads, 0, aa);
  }
  if (n_req > 0) {  // blocks (if any), then sessions
    const BlkArgs ba{L.cnt, L.flg, L.tag, L.fl, req_ts_us, L.s_cnt, L.s_first, L.s_last, L.cls,
                     (uint32_t)n_distinct, n_req, n_session, L.out, L.st};
    const uint64_t want = n_distinct / kBlkPer > n_session ? n_distinct / kBlkPer : n_session;
    const uint32_t bgrid = persistent_grid(k_st_blocks, kStThreads, sms, ceil_div_u32(want ? want : 1, kStThreads));
    PTC_KERNEL("k_st_blocks", s, k_st_blocks, bgrid, kStThreads, 0, ba);
  }
  if (n > 0) {
    const ReuseArgs rua{ids, prev, L.req_of, L.cls, req_ts_us, (uint32_t)n, (uint32_t)n_distinct, L.out};
    PTC_KERNEL("k_st_reuse", s, k_st_reuse, grid_reuse, kStThreads, 0, rua);
  }
  // the summary and the reach bins (contiguous in the workspace) in one copy
  HostStage* hs = host_stage();
  const size_t words = sizeof(ptc_trace_summary) / 8 + (n_cap ? n_cap + 1 : 0);
  static_assert(sizeof(ptc_trace_summary) % 8 == 0, "summary of u64 fields");
  if ((const char*)L.reach_bins != (const char*)L.out + sizeof(ptc_trace_summary)) return PTC_ERR_CUDA;
  if (copy_to_host_async(hs->stats, L.out, 8 * words, s) != PTC_OK) return PTC_ERR_CUDA;
  DevStatus h;
  const ptc_status rc = end_call(L.st, s, &h);
  if (rc != PTC_OK) return rc;
  std::memcpy(stats_host_out, hs->stats, sizeof(ptc_trace_summary));
  stats_host_out->n_access = n;
  stats_host_out->n_distinct = n_distinct;
  const uint64_t* bins = hs->stats + sizeof(ptc_trace_summary) / 8;
  uint64_t run = 0;
  for (uint32_t g = 0; g < n_cap; ++g) reach_host_out[g] = (run += bins[g]);
  return PTC_OK;
}
