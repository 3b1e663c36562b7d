// Stage d: hit and compute-saved curves for every capacity at once
// (paper Sec. 3.2 block hit ratio, Sec. 5.2 compute-savings ratio, prefix
// reuse from Sec. 2.2).
//
// Block k of a request is a prefix hit at capacity C iff blocks 0..k of the
// request are all resident, i.e. iff e_i = max(dist over the request's blocks
// up to k) <= C (an access hits alone iff dist <= C: Mattson inclusion).  So
// one pass computes e_i (a per-request running max: segmented scan with
// decoupled look-back), finds the first capacity >= e_i, and histograms
// count and depth per capacity bin.  Every cost model is affine in depth,
// cost(k) = alpha + beta k, so compute saved = alpha * hits + beta * (sum of k),
// formed exactly in 128 bits by the finalize kernel.
//   k_heads     marks the first access of every non-empty request (bitmap)
//   k_curves_fast  when the distances never fall inside a request (the case
//               for any trace whose blocks are root-first: a longer prefix
//               is never more recently used than its parent), the running
//               max is the distance itself; bins and depths straight from
//               the distances, request starts from a per-tile table.  A
//               fall inside a request sets a flag, and then the scan
//               kernels below redo the curves from scratch.
//   k_curves    running max, bin search in shared memory, run-merged
//               shared histograms, one global atomic per non-empty bin
//   k_curves_runs  (ptc_pipeline) the same from stage c's runs: one thread
//               per request, one (count, depth sum) per piece of a run that
//               lies in the request; a fall between the runs of a request
//               sets the flag for the scan kernels
//   k_finalize  cumulative sums over bins (a block scan); 128-bit saved and
//               total cost
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kCvThreads = 512;
constexpr int kCvPer = 8;
constexpr int kCvTile = kCvThreads * kCvPer;

// Also records, for every tile of kCvTile accesses, the request holding its
// first access (each tile has exactly one such request).
__global__ void k_heads(const uint64_t* __restrict__ blk_off, uint32_t R, uint64_t n, uint32_t* __restrict__ bitmap,
                        uint32_t* __restrict__ tile_req, DevStatus* st) {
  grid_dep_sync();
  const uint64_t r = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= R) return;
  const uint64_t a = blk_off[r], b = blk_off[r + 1];
  if (b < a || b > n || (r == 0 && a != 0) || (r + 1 == R && b != n)) {
    raise_err(st, kErrInvalid);
    return;
  }
  if (b > a) {
    atomicOr(&bitmap[a >> 5], 1u << (a & 31));
    for (uint64_t t = (a + kCvTile - 1) / kCvTile; t * kCvTile < b; ++t) tile_req[t] = (uint32_t)r;
  }
}

struct RunMax {  // (segment-start flag, running max, start index of the segment); n < 2^32 - 1
  uint32_t m;
  uint32_t start;
  uint32_t f;
  uint32_t pad;
};
struct RunMaxOp {
  __device__ RunMax operator()(const RunMax& a, const RunMax& b) const {
    RunMax r;
    r.f = a.f | b.f;
    r.m = b.f ? b.m : (a.m > b.m ? a.m : b.m);
    r.start = b.f ? b.start : a.start;
    r.pad = 0;
    return r;
  }
};

struct CurveArgs {
  const uint32_t* dist;
  uint32_t n;
  const uint32_t* bitmap;
  uint32_t caps[PTC_MAX_CAPACITIES];  // the grid, clamped below kNone; by value, so no copy
  uint32_t G;
  unsigned long long* cnt;   // G + 1 bins (last: miss at every capacity)
  unsigned long long* ksum;  // G + 1 bins
  const RunMax* tile_agg;
  DevStatus* st;
  const uint64_t* blk_off;   // request block offsets (R + 1)
  const uint32_t* tile_req;  // request holding each tile's first access
  uint32_t R;
  uint32_t* slow;            // set when a distance falls inside a request
};

// Loads the kCvPer distances of this thread and the head bits of its range,
// and folds them into the thread's running max (with the segment start).
__device__ __forceinline__ void load_run(const uint32_t* __restrict__ dist, const uint32_t* __restrict__ bitmap,
                                         uint32_t n, uint32_t i0, uint32_t (&e)[kCvPer], uint32_t (&st_idx)[kCvPer],
                                         uint32_t& has_head, RunMax& loc) {
  uint32_t d[kCvPer];
  if (i0 + kCvPer <= n && ((reinterpret_cast<uintptr_t>(dist) & 15) == 0)) {
    const uint4 x = __ldg(reinterpret_cast<const uint4*>(dist + i0));
    const uint4 y = __ldg(reinterpret_cast<const uint4*>(dist + i0 + 4));
    d[0] = x.x; d[1] = x.y; d[2] = x.z; d[3] = x.w;
    d[4] = y.x; d[5] = y.y; d[6] = y.z; d[7] = y.w;
  } else {
#pragma unroll
    for (int j = 0; j < kCvPer; ++j) d[j] = i0 + j < n ? dist[i0 + j] : 0u;
  }
  const uint32_t heads = i0 < n ? (bitmap[i0 >> 5] >> (i0 & 31)) & 0xFFu : 0u;
  loc = RunMax{0, 0, 0, 0};
  has_head = 0;
#pragma unroll
  for (int j = 0; j < kCvPer; ++j) {
    const uint32_t dv = (i0 + j < n) ? d[j] : 0u;
    if ((heads >> j) & 1u) {
      loc.f = 1;
      loc.m = dv;
      loc.start = i0 + j;
    } else {
      loc.m = dv > loc.m ? dv : loc.m;
    }
    e[j] = loc.m;
    st_idx[j] = loc.start;
    if (loc.f) has_head |= 1u << j;
  }
}

__device__ __forceinline__ RunMax shfl_up_rm(const RunMax& x, int o) {
  RunMax y;
  y.m = __shfl_up_sync(kFull, x.m, o);
  y.start = __shfl_up_sync(kFull, x.start, o);
  y.f = __shfl_up_sync(kFull, x.f, o);
  y.pad = 0;
  return y;
}

// CTA-wide inclusive segmented scan of the thread aggregates: returns the
// thread's inclusive value within its warp in *x and leaves the inclusive value
// over warps in s_w (s_w[last] is the tile aggregate).
__device__ __forceinline__ void cta_runmax_scan(RunMax& x, RunMax* s_w) {
  RunMaxOp op;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const RunMax y = shfl_up_rm(x, o);
    if (lane >= (uint32_t)o) x = op(y, x);
  }
  if (lane == 31) s_w[w] = x;
  __syncthreads();
  if (w == 0) {
    RunMax z = lane < kCvThreads / 32 ? s_w[lane] : RunMax{0, 0, 0, 0};
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const RunMax y = shfl_up_rm(z, o);
      if (lane >= (uint32_t)o) z = op(y, z);
    }
    if (lane < kCvThreads / 32) s_w[lane] = z;
  }
  __syncthreads();
}

// Pass 1: every tile's aggregate (request start seen?, running max since the
// last start, index of that start).  Tiles are independent.
__global__ void __launch_bounds__(kCvThreads) k_curves_agg(const uint32_t* __restrict__ dist, uint32_t n,
                                                           const uint32_t* __restrict__ bitmap,
                                                           RunMax* __restrict__ tile_agg, const uint32_t* slow,
                                                           unsigned long long* cnt, unsigned long long* ksum,
                                                           uint32_t G) {
  grid_dep_sync();
  __shared__ RunMax s_w[kCvThreads / 32];
  if (!*slow) return;  // k_curves_fast's bins stand
  if (blockIdx.x == 0)  // the scan path starts the bins afresh
    for (uint32_t g = threadIdx.x; g <= G; g += kCvThreads) cnt[g] = ksum[g] = 0;
  const uint32_t i0 = blockIdx.x * kCvTile + threadIdx.x * kCvPer;
  uint32_t e[kCvPer], st_idx[kCvPer];
  uint32_t has_head;
  RunMax x;
  load_run(dist, bitmap, n, i0, e, st_idx, has_head, x);
  cta_runmax_scan(x, s_w);
  if (threadIdx.x == 0) tile_agg[blockIdx.x] = s_w[kCvThreads / 32 - 1];
}

// Persistent: each CTA walks tiles blockIdx.x, blockIdx.x + gridDim.x, ...
// and keeps its bin histograms in shared memory across them, so the global
// bins see one atomic per CTA and bin rather than per tile.
__global__ void __launch_bounds__(kCvThreads) k_curves(CurveArgs a) {
  grid_dep_sync();
  if (!*a.slow) return;
  __shared__ uint32_t s_cap[PTC_MAX_CAPACITIES];
  __shared__ uint32_t s_cnt[PTC_MAX_CAPACITIES + 1];
  __shared__ unsigned long long s_ks[PTC_MAX_CAPACITIES + 1];
  __shared__ RunMax s_w[kCvThreads / 32];
  __shared__ RunMax s_carry;
  const uint32_t G = a.G;
  for (uint32_t g = threadIdx.x; g < G; g += kCvThreads)
    s_cap[g] = a.caps[g];
  for (uint32_t g = threadIdx.x; g <= G; g += kCvThreads) {
    s_cnt[g] = 0;
    s_ks[g] = 0;
  }
  const uint32_t ntiles = (a.n + kCvTile - 1) / kCvTile;
  RunMaxOp op;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (uint32_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
    const uint32_t i0 = tile * kCvTile + threadIdx.x * kCvPer;
    uint32_t e[kCvPer], st_idx[kCvPer];
    uint32_t has_head;
    RunMax loc;
    load_run(a.dist, a.bitmap, a.n, i0, e, st_idx, has_head, loc);
    RunMax x = loc;
    cta_runmax_scan(x, s_w);
    // carry: fold of the aggregates of the tiles before this one, back to the
    // nearest tile where a request starts (all written by k_curves_agg)
    if (w == 0) {
      RunMax acc{0, 0, 0, 0};
      for (int64_t base = (int64_t)tile - 1; base >= 0; base -= 32) {
        const int64_t idx = base - (int64_t)lane;
        RunMax g{0, 0, 0, 0};
        if (idx >= 0) g = a.tile_agg[idx];
        const uint32_t heads = __ballot_sync(kFull, idx >= 0 && g.f);
        const uint32_t first = heads ? (uint32_t)(__ffs(heads) - 1) : 31u;
        if (lane > first) g = RunMax{0, 0, 0, 0};
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const RunMax y = shfl_down_payload(g, o);
          if (lane + o < 32) g = op(y, g);
        }
        acc = op(shfl_payload(g, 0), acc);
        if (heads) break;
      }
      if (lane == 0) s_carry = acc;
    }
    __syncthreads();
    // exclusive prefix of this thread = carry (+) warps before (+) lanes before
    RunMax pre = s_carry;
    if (w > 0) pre = op(pre, s_w[w - 1]);
    {
      const RunMax y = shfl_up_rm(x, 1);
      if (lane > 0) pre = op(pre, y);
    }

    // bin and accumulate; consecutive accesses mostly share e (runs), so the
    // bin is looked up only when e changes and counts merge until the bin does
    uint32_t cur_g = 0xFFFFFFFFu, run_c = 0, last_e = 0xFFFFFFFFu, last_g = G;
    unsigned long long run_k = 0;
#pragma unroll
    for (int j = 0; j < kCvPer; ++j) {
      if (i0 + j >= a.n) break;
      uint32_t ej = e[j], sj = st_idx[j];
      if (!((has_head >> j) & 1u)) {
        ej = pre.m > ej ? pre.m : ej;
        sj = pre.start;
      }
      uint32_t g = last_g;
      if (ej != last_e) {
        if (ej == kNone) {
          g = G;
        } else {  // first capacity >= ej
          uint32_t lo = 0, hi = G;
          while (lo < hi) {
            const uint32_t mid = (lo + hi) >> 1;
            if (s_cap[mid] >= ej)
              hi = mid;
            else
              lo = mid + 1;
          }
          g = lo;
        }
        last_e = ej;
        last_g = g;
      }
      const uint32_t k = (i0 + j) - sj;
      if (g != cur_g) {
        if (run_c) {
          atomicAdd(&s_cnt[cur_g], run_c);
          atomicAdd(&s_ks[cur_g], run_k);
        }
        cur_g = g;
        run_c = 0;
        run_k = 0;
      }
      ++run_c;
      run_k += k;
    }
    // the open run of every lane; inside long runs the whole warp shares one
    // bin, so it sums across lanes and adds once
    const uint32_t g0 = __shfl_sync(kFull, cur_g, 0);
    if (__all_sync(kFull, cur_g == g0 || run_c == 0)) {
      uint32_t c = run_c;
      unsigned long long kk = run_k;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        c += __shfl_xor_sync(kFull, c, o);
        kk += __shfl_xor_sync(kFull, kk, o);
      }
      if (lane == 0 && c) {
        atomicAdd(&s_cnt[g0], c);
        atomicAdd(&s_ks[g0], kk);
      }
    } else if (run_c) {
      atomicAdd(&s_cnt[cur_g], run_c);
      atomicAdd(&s_ks[cur_g], run_k);
    }
    __syncthreads();  // s_w and s_carry are reused by the next tile
  }
  for (uint32_t g = threadIdx.x; g <= G; g += kCvThreads) {
    if (s_cnt[g]) {
      atomicAdd(&a.cnt[g], (unsigned long long)s_cnt[g]);
      atomicAdd(&a.ksum[g], s_ks[g]);
    }
  }
}


// Bin of e among the capacities (first capacity >= e; G for a first access).
__device__ __forceinline__ uint32_t bin_of(const uint32_t* s_cap, uint32_t G, uint32_t e) {
  if (e == kNone) return G;
  uint32_t lo = 0, hi = G;
  while (lo < hi) {
    const uint32_t mid = (lo + hi) >> 1;
    if (s_cap[mid] >= e)
      hi = mid;
    else
      lo = mid + 1;
  }
  return lo;
}

constexpr int kFtReq = 128;  // requests a tile's table holds

__global__ void __launch_bounds__(kCvThreads) k_curves_fast(CurveArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_cap[PTC_MAX_CAPACITIES];
  __shared__ uint32_t s_cnt[PTC_MAX_CAPACITIES + 1];
  __shared__ unsigned long long s_ks[PTC_MAX_CAPACITIES + 1];
  __shared__ uint32_t s_off[kFtReq + 2];
  const uint32_t G = a.G;
  for (uint32_t g = threadIdx.x; g < G; g += kCvThreads)
    s_cap[g] = a.caps[g];
  for (uint32_t g = threadIdx.x; g <= G; g += kCvThreads) {
    s_cnt[g] = 0;
    s_ks[g] = 0;
  }
  const uint32_t ntiles = (a.n + kCvTile - 1) / kCvTile;
  const uint32_t lane = threadIdx.x & 31;
  bool fell = false;
  for (uint32_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
    const uint32_t t0 = tile * kCvTile, t1 = min(t0 + kCvTile, a.n) - 1;  // first / last access of the tile
    const uint32_t i0 = t0 + threadIdx.x * kCvPer;
    uint32_t d[kCvPer];
    if (i0 + kCvPer <= a.n && ((reinterpret_cast<uintptr_t>(a.dist) & 15) == 0)) {
      const uint4 x = __ldg(reinterpret_cast<const uint4*>(a.dist + i0));
      const uint4 y = __ldg(reinterpret_cast<const uint4*>(a.dist + i0 + 4));
      d[0] = x.x; d[1] = x.y; d[2] = x.z; d[3] = x.w;
      d[4] = y.x; d[5] = y.y; d[6] = y.z; d[7] = y.w;
    } else {
#pragma unroll
      for (int j = 0; j < kCvPer; ++j) d[j] = i0 + j < a.n ? a.dist[i0 + j] : 0u;
    }
    (void)t1;
    // the requests meeting the tile: from the one holding its first access to
    // the one holding the next tile's first access
    const uint32_t r0 = a.tile_req[tile];
    const uint32_t r1 = tile + 1 < ntiles ? a.tile_req[tile + 1] : a.R - 1;
    const bool cached = r1 - r0 + 1 <= kFtReq;
    if (cached)
      for (uint32_t k = threadIdx.x; k <= r1 - r0 + 1; k += kCvThreads) s_off[k] = (uint32_t)a.blk_off[r0 + k];
    __syncthreads();
    uint32_t before = __shfl_up_sync(kFull, d[kCvPer - 1], 1);  // distance of access i0 - 1
    if (lane == 0) before = i0 > 0 && i0 - 1 < a.n ? a.dist[i0 - 1] : 0u;
    uint32_t cur_g = 0xFFFFFFFFu, run_c = 0;
    unsigned long long run_k = 0;
    if (i0 < a.n) {
      // request of access i0, then walk forward
      uint32_t idx, start, nxt;
      if (cached) {
        uint32_t lo = 0, hi = r1 - r0;
        while (lo < hi) {
          const uint32_t mid = (lo + hi + 1) >> 1;
          if (s_off[mid] <= i0)
            lo = mid;
          else
            hi = mid - 1;
        }
        idx = lo;
        start = s_off[idx];
        nxt = s_off[idx + 1];
      } else {
        uint32_t lo = r0, hi = r1;
        while (lo < hi) {
          const uint32_t mid = (lo + hi + 1) >> 1;
          if (a.blk_off[mid] <= i0)
            lo = mid;
          else
            hi = mid - 1;
        }
        idx = lo;
        start = (uint32_t)a.blk_off[idx];
        nxt = (uint32_t)a.blk_off[idx + 1];
      }
      uint32_t last_e = 0xFFFFFFFEu, last_g = G;
      uint32_t prev_d = before;
#pragma unroll
      for (int j = 0; j < kCvPer; ++j) {
        const uint32_t i = i0 + j;
        if (i >= a.n) break;
        while (i >= nxt) {  // the next non-empty request
          ++idx;
          start = nxt;
          nxt = cached ? s_off[idx + 1] : (uint32_t)a.blk_off[idx + 1];
        }
        const uint32_t e = d[j];
        if (i != start && e < prev_d) fell = true;
        prev_d = e;
        if (e != last_e) {
          last_g = bin_of(s_cap, G, e);
          last_e = e;
        }
        const uint32_t g = last_g;
        if (g != cur_g) {
          if (run_c) {
            atomicAdd(&s_cnt[cur_g], run_c);
            atomicAdd(&s_ks[cur_g], run_k);
          }
          cur_g = g;
          run_c = 0;
          run_k = 0;
        }
        ++run_c;
        run_k += i - start;
      }
    }
    // the open run of every lane; inside long runs the whole warp shares one
    // bin, so it sums across lanes and adds once
    const uint32_t g0 = __shfl_sync(kFull, cur_g, 0);
    if (__all_sync(kFull, cur_g == g0 || run_c == 0)) {
      uint32_t c = run_c;
      unsigned long long kk = run_k;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        c += __shfl_xor_sync(kFull, c, o);
        kk += __shfl_xor_sync(kFull, kk, o);
      }
      if (lane == 0 && c) {
        atomicAdd(&s_cnt[g0], c);
        atomicAdd(&s_ks[g0], kk);
      }
    } else if (run_c) {
      atomicAdd(&s_cnt[cur_g], run_c);
      atomicAdd(&s_ks[cur_g], run_k);
    }
    __syncthreads();  // s_r / s_off are reused by the next tile
  }
  if (__syncthreads_or(fell) && threadIdx.x == 0) atomicOr(a.slow, 1u);
  for (uint32_t g = threadIdx.x; g <= G; g += kCvThreads) {
    if (s_cnt[g]) {
      atomicAdd(&a.cnt[g], (unsigned long long)s_cnt[g]);
      atomicAdd(&a.ksum[g], s_ks[g]);
    }
  }
}


// Index of the run holding access j (stage c's run-start bitmap and the runs
// starting before each 32-access word).
__device__ __forceinline__ uint32_t run_at(const uint32_t* bits, const uint32_t* wpre, uint32_t j) {
  const uint32_t wi = j >> 5, b = j & 31;
  const uint32_t mask_le = b == 31 ? kFull : ((2u << b) - 1u);
  return wpre[wi] + __popc(bits[wi] & mask_le) - 1u;
}

struct RunsArgs {
  const uint32_t* rec_s;
  const uint32_t* sd;
  const uint32_t* bits;
  const uint32_t* wpre;
};

__global__ void __launch_bounds__(256) k_curves_runs(CurveArgs a, RunsArgs ra) {
  grid_dep_sync();
  __shared__ uint32_t s_cap[PTC_MAX_CAPACITIES];
  __shared__ uint32_t s_cnt[PTC_MAX_CAPACITIES + 1];
  __shared__ unsigned long long s_ks[PTC_MAX_CAPACITIES + 1];
  const uint32_t G = a.G;
  for (uint32_t g = threadIdx.x; g < G; g += blockDim.x)
    s_cap[g] = a.caps[g];
  for (uint32_t g = threadIdx.x; g <= G; g += blockDim.x) {
    s_cnt[g] = 0;
    s_ks[g] = 0;
  }
  __syncthreads();
  bool fell = false;
  for (uint32_t q = blockIdx.x * blockDim.x + threadIdx.x; q < a.R; q += gridDim.x * blockDim.x) {
    const uint32_t start = (uint32_t)a.blk_off[q], end = (uint32_t)a.blk_off[q + 1];
    if (end <= start || end > a.n) continue;  // empty (bad offsets are reported by k_heads)
    const uint32_t r0 = run_at(ra.bits, ra.wpre, start), r1 = run_at(ra.bits, ra.wpre, end - 1);
    uint32_t prev_v = 0, last_v = 0xFFFFFFFEu, g = G;
    for (uint32_t r = r0; r <= r1; ++r) {
      const uint32_t s0 = max(ra.rec_s[r], start), e0 = min(ra.rec_s[r + 1], end), v = ra.sd[r];
      if (v < prev_v) fell = true;  // the running max would bind
      prev_v = v;
      if (v != last_v) {
        g = bin_of(s_cap, G, v);
        last_v = v;
      }
      const uint32_t c = e0 - s0;
      const unsigned long long k0 = s0 - start;
      atomicAdd(&s_cnt[g], c);
      atomicAdd(&s_ks[g], (unsigned long long)c * k0 + (unsigned long long)c * (c - 1) / 2);
    }
  }
  if (__syncthreads_or(fell) && threadIdx.x == 0) atomicOr(a.slow, 1u);
  for (uint32_t g = threadIdx.x; g <= G; g += blockDim.x) {
    if (s_cnt[g]) {
      atomicAdd(&a.cnt[g], (unsigned long long)s_cnt[g]);
      atomicAdd(&a.ksum[g], s_ks[g]);
    }
  }
}


struct U128 {
  uint64_t lo, hi;
};
__device__ __forceinline__ U128 mul_u64(uint64_t a, uint64_t b) { return U128{a * b, __umul64hi(a, b)}; }
__device__ __forceinline__ U128 add_u128(U128 a, U128 b) {
  U128 r;
  r.lo = a.lo + b.lo;
  r.hi = a.hi + b.hi + (r.lo < a.lo ? 1 : 0);
  return r;
}

// out layout: hits[G] | saved[G] (lo, hi) | total (lo, hi).  One CTA of
// 1,024 threads: an inclusive block scan of (count, depth sum) over the bins.
__global__ void __launch_bounds__(1024) k_finalize(const unsigned long long* __restrict__ cnt,
                                                   const unsigned long long* __restrict__ ksum, uint32_t G,
                                                   uint64_t alpha, uint64_t beta, uint64_t* __restrict__ out) {
  grid_dep_sync();
  __shared__ unsigned long long s_h[32], s_k[32];
  const uint32_t t = threadIdx.x, lane = t & 31, w = t >> 5;
  unsigned long long h = t < G ? cnt[t] : 0ull, k = t < G ? ksum[t] : 0ull;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long yh = __shfl_up_sync(kFull, h, o), yk = __shfl_up_sync(kFull, k, o);
    if (lane >= (uint32_t)o) {
      h += yh;
      k += yk;
    }
  }
  if (lane == 31) {
    s_h[w] = h;
    s_k[w] = k;
  }
  __syncthreads();
  for (uint32_t ww = 0; ww < w; ++ww) {
    h += s_h[ww];
    k += s_k[ww];
  }
  if (t < G) {
    const U128 sv = add_u128(mul_u64(alpha, h), mul_u64(beta, k));
    out[t] = h;
    out[G + 2 * t] = sv.lo;
    out[G + 2 * t + 1] = sv.hi;
  }
  if (t == G - 1) {  // G >= 1; the miss bin G joins the total
    const uint64_t hn = h + cnt[G], kn = k + ksum[G];
    const U128 tc = add_u128(mul_u64(alpha, hn), mul_u64(beta, kn));
    out[3 * G] = tc.lo;
    out[3 * G + 1] = tc.hi;
  }
}

struct CurvesLayout {
  DevStatus* st;
  unsigned long long* cnt;
  unsigned long long* ksum;
  uint32_t* bitmap;
  uint32_t* slow;
  uint32_t* tile_req;
  RunMax* lb_agg;
  uint64_t* out;
  size_t zero_bytes;
  size_t total;
};

CurvesLayout curves_layout(void* ws, uint64_t n, uint32_t G) {
  CurvesLayout L;
  Carver cv(ws);
  const uint32_t tiles = ceil_div_u32(n, kCvTile) + 1;
  L.st = cv.take<DevStatus>(1);
  L.cnt = cv.take<unsigned long long>(PTC_MAX_CAPACITIES + 1);
  L.ksum = cv.take<unsigned long long>(PTC_MAX_CAPACITIES + 1);
  L.bitmap = cv.take<uint32_t>(n / 32 + 2);
  L.slow = cv.take<uint32_t>(1);
  L.tile_req = cv.take<uint32_t>(tiles + 1);
  L.zero_bytes = cv.off;
  L.lb_agg = cv.take<RunMax>(tiles);
  L.out = cv.take<uint64_t>(3 * PTC_MAX_CAPACITIES + 2);
  L.total = cv.bytes();
  (void)G;
  return L;
}

bool mul_ok(uint64_t a, uint64_t b, uint64_t* r) {
  unsigned __int128 t = (unsigned __int128)a * b;
  *r = (uint64_t)t;
  return (t >> 64) == 0;
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_curves_workspace_bytes(uint64_t n, uint32_t n_req, uint32_t n_cap) {
  (void)n_req;
  return curves_layout(nullptr, n, n_cap).total;
}

ptc_status ptc::cost_coeffs(const ptc_cost_model* cm, uint32_t block_size, uint64_t* alpha_out, uint64_t* beta_out) {
  const uint64_t B = block_size;
  uint64_t alpha = 0, beta = 0, lin = 0, attn0 = 0;
  if (cm->kind == PTC_COST_UNIFORM) {
    alpha = 1;
  } else if (cm->kind == PTC_COST_MEASURED || cm->kind == PTC_COST_LINEAR) {
    if (!mul_ok(cm->f_attn, B * (B + 1) / 2, &attn0) || !mul_ok(cm->f_attn, B * B, &beta)) return PTC_ERR_OVERFLOW;
    if (cm->kind == PTC_COST_MEASURED && !mul_ok(cm->f_lin, B, &lin)) return PTC_ERR_OVERFLOW;
    alpha = lin + attn0;
    if (alpha < lin) return PTC_ERR_OVERFLOW;
  } else {
    return PTC_ERR_INVALID_ARG;
  }
  *alpha_out = alpha;
  *beta_out = beta;
  return PTC_OK;
}

ptc_status ptc::curves_impl(const uint32_t* dist, uint64_t n, const uint64_t* req_blk_off, uint32_t n_req,
                            uint32_t block_size, const ptc_cost_model* cm, const uint64_t* cap_host, uint32_t n_cap,
                            uint64_t* hits_host_out, ptc_u128* saved_host_out, ptc_u128* total_cost_host_out,
                            void* ws, size_t ws_bytes, cudaStream_t stream, const RunsView* runs,
                            const uint32_t* carry_err, uint32_t n_carry) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (!cm || !cap_host || !hits_host_out || !saved_host_out || !total_cost_host_out) return PTC_ERR_INVALID_ARG;
  if (n_cap < 1 || n_cap > PTC_MAX_CAPACITIES) return PTC_ERR_INVALID_ARG;
  if (block_size < 1 || block_size > PTC_MAX_BLOCK_SIZE) return PTC_ERR_INVALID_ARG;
  if (n > 0 && (!dist || !req_blk_off || n_req == 0)) return PTC_ERR_INVALID_ARG;
  for (uint32_t g = 0; g < n_cap; ++g)
    if (cap_host[g] < 1 || (g && cap_host[g] <= cap_host[g - 1])) return PTC_ERR_INVALID_ARG;
  // cost(k) = alpha + beta k
  uint64_t alpha = 0, beta = 0;
  const ptc_status crc = cost_coeffs(cm, block_size, &alpha, &beta);
  if (crc != PTC_OK) return crc;
  if (!ws_ok(ws, ws_bytes, curves_layout(nullptr, n, n_cap).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = stream;
  const CurvesLayout L = curves_layout(ws, n, n_cap);
  if (begin_call(ws, L.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  HostStage* hs = host_stage();
  if (n_carry && carry_errors(carry_err, n_carry, L.st, s) != PTC_OK) return PTC_ERR_CUDA;
  if (n > 0) {
    PTC_KERNEL("k_heads", s, k_heads, ceil_div_u32(n_req, 256), 256, 0, req_blk_off, n_req, n, L.bitmap, L.tile_req, L.st);
    CurveArgs a;
    a.dist = dist;
    a.n = (uint32_t)n;
    a.bitmap = L.bitmap;
    for (uint32_t g = 0; g < n_cap; ++g)
      a.caps[g] = cap_host[g] >= (uint64_t)kNone ? kNone - 1 : (uint32_t)cap_host[g];
    a.G = n_cap;
    a.cnt = L.cnt;
    a.ksum = L.ksum;
    a.tile_agg = L.lb_agg;
    a.st = L.st;
    a.blk_off = req_blk_off;
    a.tile_req = L.tile_req;
    a.R = n_req;
    a.slow = L.slow;
    if (runs && runs->used) {
      const RunsArgs ra{runs->rec_s, runs->sd, runs->bits, runs->wpre};
      const uint32_t g_r = ceil_div_u32(n_req, 256) < (uint32_t)(2 * num_sms()) ? ceil_div_u32(n_req, 256)
                                                                                  : (uint32_t)(2 * num_sms());
      PTC_KERNEL("k_curves_runs", s, k_curves_runs, g_r, 256, 0, a, ra);
    } else {
      const uint32_t tiles0 = ceil_div_u32(n, kCvTile);
      const uint32_t grid0 = tiles0 < (uint32_t)(3 * num_sms()) ? tiles0 : (uint32_t)(3 * num_sms());
      PTC_KERNEL("k_curves_fast", s, k_curves_fast, grid0, kCvThreads, 0, a);
    }
    PTC_KERNEL("k_curves_agg", s, k_curves_agg, ceil_div_u32(n, kCvTile), kCvThreads, 0, dist, (uint32_t)n, L.bitmap, L.lb_agg, L.slow, L.cnt, L.ksum, n_cap);
    const uint32_t tiles = ceil_div_u32(n, kCvTile);
    const uint32_t grid = tiles < (uint32_t)(3 * num_sms()) ? tiles : (uint32_t)(3 * num_sms());
    PTC_KERNEL("k_curves", s, k_curves, grid, kCvThreads, 0, a);
  }
  PTC_KERNEL("k_finalize", s, k_finalize, 1, 1024, 0, L.cnt, L.ksum, n_cap, alpha, beta, L.out);
  const uint64_t* host_out = hs->out;
  if (copy_to_host_async(hs->out, L.out, sizeof(uint64_t) * (3 * n_cap + 2), s) != PTC_OK) return PTC_ERR_CUDA;
  DevStatus h;
  const ptc_status rc = end_call(L.st, s, &h);
  if (rc != PTC_OK) return rc;
  for (uint32_t g = 0; g < n_cap; ++g) {
    hits_host_out[g] = host_out[g];
    saved_host_out[g].lo = host_out[n_cap + 2 * g];
    saved_host_out[g].hi = host_out[n_cap + 2 * g + 1];
  }
  total_cost_host_out->lo = host_out[3 * n_cap];
  total_cost_host_out->hi = host_out[3 * n_cap + 1];
  return PTC_OK;
}

extern "C" ptc_status ptc_curves(const uint32_t* dist, uint64_t n, const uint64_t* req_blk_off, uint32_t n_req,
                                 uint32_t block_size, const ptc_cost_model* cm, const uint64_t* cap_host, uint32_t n_cap,
                                 uint64_t* hits_host_out, ptc_u128* saved_host_out, ptc_u128* total_cost_host_out,
                                 void* ws, size_t ws_bytes, void* stream) {
  return ptc::curves_impl(dist, n, req_blk_off, n_req, block_size, cm, cap_host, n_cap, hits_host_out, saved_host_out,
                          total_cost_host_out, ws, ws_bytes, (cudaStream_t)stream, nullptr);
}

// ---------------------------------------------------------------------------
// ptc_curves_noalloc: the curves for callers that cannot allocate device
// memory.  Some callers have no way to hand this library a workspace: code
// that runs inside another runtime which owns every byte of device memory
// and exposes no allocator, plugin hosts that forbid cudaMalloc (it can
// synchronize the device and stall unrelated work), or latency-critical
// loops that must not enter the allocator at all.  For them the scratch that
// ptc_curves takes from `ws` lives in one fixed array in this library's
// device image instead, reserved when the library is loaded and held by every
// GPU that loads it until the process exits.
// ---------------------------------------------------------------------------
#include <mutex>

namespace {
constexpr uint64_t kNoAllocMaxAccesses = 1ULL << 24;
constexpr size_t kNoAllocScratchBytes = 4u << 20;
static __device__ __align__(256) unsigned char g_curves_scratch[kNoAllocScratchBytes];
constexpr int kNoAllocMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kNoAllocMaxDevices] = {};

// Device address of g_curves_scratch on the current device, looked up once per
// device (the host-side symbol is only a stand-in, not a device address).
ptc_status scratch_for_current_device(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return PTC_ERR_CUDA;
  if (dev < 0 || dev >= kNoAllocMaxDevices) return PTC_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> g(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_curves_scratch) != cudaSuccess || p == nullptr) return PTC_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return PTC_OK;
}
}  // namespace

extern "C" ptc_status ptc_curves_noalloc(const uint32_t* dist, uint64_t n, const uint64_t* req_blk_off,
                                         uint32_t n_req, uint32_t block_size, const ptc_cost_model* cm,
                                         const uint64_t* cap_host, uint32_t n_cap, uint64_t* hits_host_out,
                                         ptc_u128* saved_host_out, ptc_u128* total_cost_host_out, void* stream) {
  if (n > kNoAllocMaxAccesses) return PTC_ERR_WORKSPACE;
  if (n_cap > PTC_MAX_CAPACITIES) return PTC_ERR_INVALID_ARG;
  if (curves_layout(nullptr, n, n_cap).total > kNoAllocScratchBytes) return PTC_ERR_WORKSPACE;
  void* scratch = nullptr;
  const ptc_status rc = scratch_for_current_device(&scratch);
  if (rc != PTC_OK) return rc;
  // ptc_curves zeroes every part of the scratch that must start at zero.
  const NoHostAlloc no_alloc;
  return ptc_curves(dist, n, req_blk_off, n_req, block_size, cm, cap_host, n_cap, hits_host_out, saved_host_out,
                    total_cost_host_out, scratch, kNoAllocScratchBytes, stream);
}
