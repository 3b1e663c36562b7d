// Stage c over runs: the dominance count of App. B on a weighted wavelet
// matrix whose points are the runs of the access stream, not its accesses.
//
// With v_j = prev[j] + 1 (none -> 0), the stack distance of access i with
// p = prev[i] is
//   SD_i = 1 + #{ j : p < j < i, v_j <= p }.
// A run is a maximal stretch of accesses that either re-read a context block
// by block (v_{j+1} = v_j + 1, v_j > 0) or are all first accesses (v = 0).
// Re-reads of long shared prefixes make runs long: the conversational traces
// hold a few hundred accesses per run.
//
// Every run meets the window (p, i) either entirely inside or not at all in
// the count.  Inside the window no access has v_j = p + 1, because that value
// belongs to i alone (an access has at most one next use).  The values along
// a context run are consecutive, so those of a run that fall in the window
// lie all at or below p or all above it; a first-access run is all zeros.
// Hence
//   SD_i = 1 + [the run holding p+1, when it starts before p+1: its part in
//               the window if its value at p+1 is <= p]
//            + sum of the lengths of the runs wholly inside (p, i) whose
//              largest value is <= p,
// a weighted 2-D dominance count over runs (index, largest value; weight =
// length).  The matrix over runs answers it exactly as the matrix over
// accesses would, and a run head's distance is that of its whole run (a
// context run's accesses all share it, the run identity of App. B's
// stack-distance recurrence).
//
// Weighted wavelet matrix (Claude, Navarro, Ordonez 2015): level l orders the
// runs by the stable partition on bit L-1-l of the previous level's order and
// stores, for every position, the zeros before it and their total weight
// (Z, W).  A count of keys < x over [lo, hi) walks the L levels; where x has a
// one bit, the zeros of the current range (all smaller) add their weight.
//
//   k_runs_count   run starts per tile; the last CTA scans the tile counts
//   k_runs_mark    run starts again: bitmap, run index per 32-position word,
//                  run (start, first value) records
//                  (both with 16-byte loads, four accesses per lane and
//                  round, when prev is 16-byte aligned: k_runs_count4,
//                  k_runs_mark4)
//   bitmap_ranks   the runs' keys (marked by k_runs_mark in a bitmap over
//                  [0, n]) counted per word: the matrix holds each key's rank
//                  among the distinct keys, so it has ceil(log2(R + 2))
//                  levels instead of ceil(log2(n + 1)), and a query's
//                  threshold x becomes the number of keys below x
//   k_runs_init    level-0 keys and weights, per-tile zero counts / weights
//   k_runs_level   one level: (Z, W), stable partition, the next level's
//                  per-tile zero counts (four atomics per tile)
//   k_runs_query   one thread per run: the distance of its head
//   k_runs_expand  every access takes its run's distance
#include <cooperative_groups.h>

#include <utility>

#include <atomic>

#include "ptc_internal.h"

namespace cg = cooperative_groups;

namespace ptc {
namespace {

constexpr int kMT = 256;           // run marking: threads per tile
constexpr int kMR = 16;            // rounds of 32 positions per warp
constexpr int kMTile = kMT * kMR;  // 4096 positions; warp w owns [512 w, 512 w + 512)
constexpr int kRT = 256;           // level tiles: threads
constexpr int kRPer = 8;           // runs per thread (consecutive)
constexpr int kRTile = kRT * kRPer;

__device__ __forceinline__ uint32_t vval(uint32_t p) { return p == kNone ? 0u : p + 1u; }

struct MarkArgs {
  const uint32_t* prev;
  uint32_t n;
  uint32_t ntiles;
  uint32_t* bits;     // run-start bitmap, one word per 32 positions
  uint32_t* wpre;     // runs starting before each word
  uint32_t* rec_s;    // start of each run (rec_s[R] = n)
  uint32_t* rec_a;    // value at the start of each run
  uint32_t* tcnt;     // run starts in each tile
  uint32_t* tpre;     // runs starting before each tile; tpre[ntiles] = R
  uint32_t* done;
  uint32_t* kbits;    // bitmap of the runs' keys (largest values) over [0, n]
  DevStatus* st;      // value[1] <- R
};

// Run-start bits of the warp's 8 x 32 positions from `base` (the previous
// access decides whether one continues a run).
__device__ __forceinline__ void start_words(const MarkArgs& a, uint32_t base, uint32_t lane, uint32_t (&pv)[kMR],
                                            uint32_t (&words)[kMR], bool& bad, uint32_t* left = nullptr) {
#pragma unroll
  for (int k = 0; k < kMR; ++k) {
    const uint32_t j = base + k * 32 + lane;
    pv[k] = j < a.n ? a.prev[j] : kNone;
  }
  const uint32_t left0 = (lane == 0 && base > 0 && base - 1 < a.n) ? a.prev[base - 1] : kNone;
  uint32_t carry = vval(left0);  // value left of lane 0 (meaningful in lane 0 only)
#pragma unroll
  for (int k = 0; k < kMR; ++k) {
    const uint32_t j = base + k * 32 + lane;
    const bool valid = j < a.n;
    if (valid && pv[k] != kNone && pv[k] >= j) bad = true;
    const uint32_t v = vval(pv[k]);
    const uint32_t up = __shfl_up_sync(kFull, v, 1);
    const uint32_t vl = lane ? up : carry;
    carry = __shfl_sync(kFull, v, 31);
    const bool cont = j > 0 && ((v == vl + 1 && vl != 0) || (v == 0 && vl == 0));
    words[k] = __ballot_sync(kFull, valid && !cont);
    if (left) left[k] = vl;
  }
}

// The calling CTA learns whether it is the last of the grid to get here.
__device__ __forceinline__ bool last_cta(uint32_t* done) {
  __shared__ uint32_t s_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(done, 1u) == gridDim.x - 1;
  __syncthreads();
  if (s_last) __threadfence();
  return s_last;
}

// Pass 1: run starts per tile; the last CTA turns them into tile prefixes.
__global__ void __launch_bounds__(kMT) k_runs_count(MarkArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_wcnt[kMT / 32];
  const uint32_t tile = blockIdx.x;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint32_t pv[kMR], words[kMR];
  bool bad = false;
  start_words(a, tile * kMTile + w * (32 * kMR), lane, pv, words, bad);
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kMR; ++k) cnt += __popc(words[k]);
  if (lane == 0) s_wcnt[w] = cnt;
  if (bad) raise_err(a.st, kErrInvalid);
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t t = 0;
    for (int ww = 0; ww < kMT / 32; ++ww) t += s_wcnt[ww];
    a.tcnt[tile] = t;
  }
  if (!last_cta(a.done)) return;
  const uint32_t total = cta_tiles_prefix(a.tcnt, a.tpre, a.ntiles);  // exclusive prefix of the tile counts
  if (threadIdx.x == 0) a.st->value[1] = total;
}

// Pass 2: bitmap, run index per word, and the (start, first value) records.
__global__ void __launch_bounds__(kMT) k_runs_mark(MarkArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_wcnt[kMT / 32];
  const uint32_t tile = blockIdx.x;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t base = tile * kMTile + w * (32 * kMR);
  uint32_t pv[kMR], words[kMR], left[kMR];
  bool bad = false;
  start_words(a, base, lane, pv, words, bad, left);
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kMR; ++k) cnt += __popc(words[k]);
  if (lane == 0) s_wcnt[w] = cnt;
  // The runs' keys for rank compression: a run's largest value is its last
  // one (values along a context run rise by one; a first-access run is all
  // zeros), i.e. the value left of the next run's start, or the last
  // access's.  Nonzero keys are distinct (each access is the previous use of
  // at most one other); 0 is always entered, once.
#pragma unroll
  for (int k = 0; k < kMR; ++k) {
    const uint32_t j = base + k * 32 + lane;
    if (j < a.n) {
      if (((words[k] >> lane) & 1u) && j > 0 && left[k] != 0) atomicOr(&a.kbits[left[k] >> 5], 1u << (left[k] & 31));
      const uint32_t v = vval(pv[k]);
      if (j + 1 == a.n && v != 0) atomicOr(&a.kbits[v >> 5], 1u << (v & 31));
    }
  }
  if (tile == 0 && threadIdx.x == 0) atomicOr(&a.kbits[0], 1u);
  __syncthreads();
  uint32_t run = a.tpre[tile];
  for (int ww = 0; ww < (int)w; ++ww) run += s_wcnt[ww];
#pragma unroll
  for (int k = 0; k < kMR; ++k) {
    const uint32_t j = base + k * 32 + lane;
    if (base + k * 32 < a.n && lane == 0) {
      a.bits[(base + k * 32) >> 5] = words[k];
      a.wpre[(base + k * 32) >> 5] = run;
    }
    if ((words[k] >> lane) & 1u) {
      const uint32_t r = run + __popc(words[k] & lanemask_lt());
      a.rec_s[r] = j;
      a.rec_a[r] = vval(pv[k]);
    }
    run += __popc(words[k]);
  }
  if (tile == a.ntiles - 1 && threadIdx.x == 0) a.rec_s[a.tpre[a.ntiles]] = a.n;
}

// ---- the same two passes with 16-byte loads (prev 16-byte aligned): lane l
// of warp w reads positions base + 128 k + 4 l .. + 3 (k < 4, base = the
// warp's 512 positions), one load per four accesses.
constexpr int kMR4 = kMR / 4;

// Four values from position p (a multiple of 4), kNone past n.
__device__ __forceinline__ uint4 load4(const uint32_t* __restrict__ v, uint32_t p, uint32_t n) {
  if (p + 4 <= n) return __ldcs(reinterpret_cast<const uint4*>(v + p));
  return make_uint4(p < n ? v[p] : kNone, p + 1 < n ? v[p + 1] : kNone, p + 2 < n ? v[p + 2] : kNone,
                    p + 3 < n ? v[p + 3] : kNone);
}

// Run starts among positions p .. p + 3 as bits 0..3, from their previous
// uses v and the previous use `pl` at p - 1.  A run continues at j when
// prev[j] = prev[j - 1] + 1 with prev[j - 1] a use, or both are first
// accesses (as start_words, with prev values instead of v = prev + 1).
__device__ __forceinline__ uint32_t starts4(const uint4 v, uint32_t pl, uint32_t p, uint32_t n, bool& bad) {
  const uint32_t pv[4] = {v.x, v.y, v.z, v.w};
  uint32_t x = 0, left = pl;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const uint32_t j = p + e, P = pv[e];
    if (j < n) {
      if (P != kNone && P >= j) bad = true;
      const bool cont = j > 0 && ((P == left + 1u && left != kNone) || (P == kNone && left == kNone));
      x |= (cont ? 0u : 1u) << e;
    }
    left = P;
  }
  return x;
}

// The warp's four loads and their run-start nibbles.
__device__ __forceinline__ uint32_t warp_starts4(const MarkArgs& a, uint32_t base, uint32_t lane, uint4 (&v)[kMR4],
                                                 uint32_t (&x)[kMR4], uint32_t (&pl)[kMR4], bool& bad) {
#pragma unroll
  for (int k = 0; k < kMR4; ++k) v[k] = load4(a.prev, base + 128 * k + 4 * lane, a.n);
  uint32_t carry = (base > 0 && base - 1 < a.n) ? a.prev[base - 1] : kNone;  // lane 0 of the first round
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kMR4; ++k) {
    const uint32_t up = __shfl_up_sync(kFull, v[k].w, 1);
    pl[k] = lane ? up : carry;
    carry = __shfl_sync(kFull, v[k].w, 31);
    x[k] = starts4(v[k], pl[k], base + 128 * k + 4 * lane, a.n, bad);
    cnt += __popc(x[k]);
  }
  return cnt;
}

__global__ void __launch_bounds__(kMT) k_runs_count4(MarkArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_wcnt[kMT / 32];
  const uint32_t tile = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint4 v[kMR4];
  uint32_t x[kMR4], pl[kMR4];
  bool bad = false;
  const uint32_t cnt = __reduce_add_sync(kFull, warp_starts4(a, tile * kMTile + w * (32 * kMR), lane, v, x, pl, bad));
  if (lane == 0) s_wcnt[w] = cnt;
  if (bad) raise_err(a.st, kErrInvalid);
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t t = 0;
    for (int ww = 0; ww < kMT / 32; ++ww) t += s_wcnt[ww];
    a.tcnt[tile] = t;
  }
  if (!last_cta(a.done)) return;
  const uint32_t total = cta_tiles_prefix(a.tcnt, a.tpre, a.ntiles);
  if (threadIdx.x == 0) a.st->value[1] = total;
}

__global__ void __launch_bounds__(kMT) k_runs_mark4(MarkArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_wcnt[kMT / 32];
  const uint32_t tile = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t base = tile * kMTile + w * (32 * kMR);
  uint4 v[kMR4];
  uint32_t x[kMR4], pl[kMR4];
  bool bad = false;
  const uint32_t cnt = __reduce_add_sync(kFull, warp_starts4(a, base, lane, v, x, pl, bad));
  if (lane == 0) s_wcnt[w] = cnt;
  if (tile == 0 && threadIdx.x == 0) atomicOr(&a.kbits[0], 1u);
  __syncthreads();
  uint32_t run = a.tpre[tile];
  for (int ww = 0; ww < (int)w; ++ww) run += s_wcnt[ww];
  const uint32_t g = lane >> 3, sh = 4 * (lane & 7);
#pragma unroll
  for (int k = 0; k < kMR4; ++k) {
    const uint32_t p = base + 128 * k + 4 * lane;
    // the 32-position word of lane group g (lanes 8g .. 8g + 7)
    uint32_t word = x[k] << sh;
    word |= __shfl_xor_sync(kFull, word, 1);
    word |= __shfl_xor_sync(kFull, word, 2);
    word |= __shfl_xor_sync(kFull, word, 4);
    const uint32_t c0 = __popc(__shfl_sync(kFull, word, 0)), c1 = __popc(__shfl_sync(kFull, word, 8)),
                   c2 = __popc(__shfl_sync(kFull, word, 16)), c3 = __popc(__shfl_sync(kFull, word, 24));
    const uint32_t before = (g > 0 ? c0 : 0u) + (g > 1 ? c1 : 0u) + (g > 2 ? c2 : 0u);
    if ((lane & 7) == 0 && base + 128 * k + 32 * g < a.n) {
      a.bits[(base + 128 * k + 32 * g) >> 5] = word;
      a.wpre[(base + 128 * k + 32 * g) >> 5] = run + before;
    }
    // The runs' keys for rank compression: a run's largest value is its last
    // one, i.e. the value left of the next run's start, or the last access's.
    // Nonzero keys are distinct; 0 is always entered, once.
    uint32_t r = run + before + __popc(word & ((1u << sh) - 1u));
    const uint32_t pv[4] = {v[k].x, v[k].y, v[k].z, v[k].w};
    uint32_t left = pl[k];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t j = p + e, vl = left + 1u, vj = pv[e] + 1u;  // v = prev + 1, none -> 0
      if ((x[k] >> e) & 1u) {
        a.rec_s[r] = j;
        a.rec_a[r] = vj;
        if (j > 0 && vl != 0) atomicOr(&a.kbits[vl >> 5], 1u << (vl & 31));
        ++r;
      }
      if (j + 1 == a.n && vj != 0) atomicOr(&a.kbits[vj >> 5], 1u << (vj & 31));
      left = pv[e];
    }
    run += c0 + c1 + c2 + c3;
  }
  if (tile == a.ntiles - 1 && threadIdx.x == 0) a.rec_s[a.tpre[a.ntiles]] = a.n;
}

// Keys in the bitmap below v: the rank of v when v is a key.
__device__ __forceinline__ uint32_t key_rank(const uint32_t* __restrict__ kbits, const uint32_t* __restrict__ kpre,
                                             uint32_t v) {
  return __ldg(&kpre[v >> 5]) + __popc(__ldg(&kbits[v >> 5]) & ((1u << (v & 31)) - 1u));
}

// Exclusive scan over the threads of a 256-thread CTA.
__device__ __forceinline__ unsigned long long cta_excl_scan(unsigned long long x, unsigned long long* s_warp,
                                                            unsigned long long& total) {
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  unsigned long long incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long y = __shfl_up_sync(kFull, incl, o);
    if (lane >= (uint32_t)o) incl += y;
  }
  if (lane == 31) s_warp[w] = incl;
  __syncthreads();
  unsigned long long pre = 0, tot = 0;
#pragma unroll
  for (int ww = 0; ww < kRT / 32; ++ww) {
    const unsigned long long v = s_warp[ww];
    if (ww < (int)w) pre += v;
    tot += v;
  }
  __syncthreads();
  total = tot;
  return pre + incl - x;
}

// (zeros, zero weight) packed as weight << 32 | count; a tile holds at most
// 2048 runs and all weights sum to N < 2^32, so neither half overflows.
__device__ __forceinline__ unsigned long long pack_zw(uint32_t z, uint32_t w) {
  return ((unsigned long long)w << 32) | z;
}

// Run by the last CTA of a level: exclusive prefix of the per-tile (zeros,
// zero weight) of the next level over its tiles; pre[ntiles] = totals.
__device__ void tile_prefix(const uint2* acc, uint2* pre, uint32_t ntiles, unsigned long long* s_warp) {
  const uint32_t per = (ntiles + kRT - 1) / kRT;
  const uint32_t t0 = threadIdx.x * per, t1 = min(t0 + per, ntiles);
  unsigned long long s = 0;
  for (uint32_t t = t0; t < t1; ++t) {
    const uint2 v = __ldcg(&acc[t]);
    s += pack_zw(v.x, v.y);
  }
  unsigned long long total;
  unsigned long long run = cta_excl_scan(s, s_warp, total);
  for (uint32_t t = t0; t < t1; ++t) {
    const uint2 v = __ldcg(&acc[t]);
    pre[t] = make_uint2((uint32_t)run, (uint32_t)(run >> 32));
    run += pack_zw(v.x, v.y);
  }
  if (threadIdx.x == 0) pre[ntiles] = make_uint2((uint32_t)total, (uint32_t)(total >> 32));
}

struct LevelArgs {
  const uint32_t* key_in;   // this level's order
  const uint32_t* wt_in;
  uint32_t* key_out;        // the next level's order (null at the last level)
  uint32_t* wt_out;
  uint2* zw;                // (Z, W) of this level, R + 1 entries
  const uint2* pre;         // (zeros, zero weight) before each tile of this level
  uint2* acc_next;          // per-tile (zeros, zero weight) of the next level
  uint2* pre_next;
  uint32_t* done;
  uint32_t R, ntiles, shift;
};

// Level-0 keys (largest value of each run) and weights (lengths) and the
// per-tile zero counts of level 0.
__global__ void __launch_bounds__(kRT) k_runs_init(const uint32_t* __restrict__ rec_s, const uint32_t* __restrict__ rec_a,
                                                  const uint32_t* __restrict__ kbits, const uint32_t* __restrict__ kpre,
                                                  uint32_t* __restrict__ key, uint32_t* __restrict__ wt,
                                                  uint2* __restrict__ acc, uint2* __restrict__ pre, uint32_t* done,
                                                  uint32_t R, uint32_t ntiles, uint32_t shift) {
  grid_dep_sync();
  __shared__ unsigned long long s_warp[kRT / 32];
  const uint32_t r0 = blockIdx.x * kRTile + threadIdx.x * kRPer;
  uint32_t cz = 0, cw = 0;
#pragma unroll
  for (int k = 0; k < kRPer; ++k) {
    const uint32_t r = r0 + k;
    if (r < R) {
      const uint32_t s = rec_s[r], e = rec_s[r + 1], a0 = rec_a[r];
      const uint32_t len = e - s;
      const uint32_t kv = key_rank(kbits, kpre, a0 ? a0 + len - 1 : 0u);
      key[r] = kv;
      wt[r] = len;
      if (!((kv >> shift) & 1u)) {
        ++cz;
        cw += len;
      }
    }
  }
  unsigned long long total;
  cta_excl_scan(pack_zw(cz, cw), s_warp, total);
  if (threadIdx.x == 0) acc[blockIdx.x] = make_uint2((uint32_t)total, (uint32_t)(total >> 32));
  if (last_cta(done)) tile_prefix(acc, pre, ntiles, s_warp);
}

__global__ void __launch_bounds__(kRT) k_runs_level(LevelArgs a) {
  grid_dep_sync();
  __shared__ unsigned long long s_warp[kRT / 32];
  __shared__ uint32_t s_red[4][2][kRT / 32];
  const uint32_t t = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t r0 = t * kRTile + threadIdx.x * kRPer;
  uint32_t kv[kRPer], wv[kRPer];
  if (r0 + kRPer <= a.R) {
    const uint4* k4 = reinterpret_cast<const uint4*>(a.key_in + r0);
    const uint4* w4 = reinterpret_cast<const uint4*>(a.wt_in + r0);
    const uint4 ka = k4[0], kb = k4[1], wa = w4[0], wb = w4[1];
    kv[0] = ka.x; kv[1] = ka.y; kv[2] = ka.z; kv[3] = ka.w;
    kv[4] = kb.x; kv[5] = kb.y; kv[6] = kb.z; kv[7] = kb.w;
    wv[0] = wa.x; wv[1] = wa.y; wv[2] = wa.z; wv[3] = wa.w;
    wv[4] = wb.x; wv[5] = wb.y; wv[6] = wb.z; wv[7] = wb.w;
  } else {
#pragma unroll
    for (int k = 0; k < kRPer; ++k) {
      kv[k] = r0 + k < a.R ? a.key_in[r0 + k] : 0u;
      wv[k] = r0 + k < a.R ? a.wt_in[r0 + k] : 0u;
    }
  }
  uint32_t cz = 0, cw = 0;
#pragma unroll
  for (int k = 0; k < kRPer; ++k) {
    if (r0 + k < a.R && !((kv[k] >> a.shift) & 1u)) {
      ++cz;
      cw += wv[k];
    }
  }
  unsigned long long tile_tot;
  const unsigned long long ex = cta_excl_scan(pack_zw(cz, cw), s_warp, tile_tot);
  const uint2 tp = a.pre[t];
  const uint32_t Zc = a.pre[a.ntiles].x;
  uint32_t z = tp.x + (uint32_t)ex, wsum = tp.y + (uint32_t)(ex >> 32);
  // destinations: this tile's zeros fill [tp.x, tp.x + tz), its ones
  // [Zc + t * kRTile - tp.x, ...); each range meets at most two next-level tiles
  const uint32_t zfirst = tp.x / kRTile, ofirst = (Zc + t * kRTile - tp.x) / kRTile;
  uint32_t nz[4] = {0, 0, 0, 0}, nw[4] = {0, 0, 0, 0};
#pragma unroll
  for (int k = 0; k < kRPer; ++k) {
    const uint32_t r = r0 + k;
    if (r < a.R) {
      a.zw[r] = make_uint2(z, wsum);
      const bool zero = !((kv[k] >> a.shift) & 1u);
      const uint32_t dst = zero ? z : Zc + (r - z);
      if (zero) {
        ++z;
        wsum += wv[k];
      }
      if (a.key_out && dst < a.R) {
        a.key_out[dst] = kv[k];
        a.wt_out[dst] = wv[k];
        if (!((kv[k] >> (a.shift - 1)) & 1u)) {
          const uint32_t slot = (zero ? 0u : 2u) + ((dst / kRTile) != (zero ? zfirst : ofirst) ? 1u : 0u);
          ++nz[slot];
          nw[slot] += wv[k];
        }
      }
    }
  }
  if (a.key_out) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        nz[q] += __shfl_xor_sync(kFull, nz[q], o);
        nw[q] += __shfl_xor_sync(kFull, nw[q], o);
      }
      if (lane == 0) {
        s_red[q][0][w] = nz[q];
        s_red[q][1][w] = nw[q];
      }
    }
    __syncthreads();
    if (threadIdx.x < 4) {
      const uint32_t q = threadIdx.x;
      uint32_t c = 0, s = 0;
#pragma unroll
      for (int ww = 0; ww < kRT / 32; ++ww) {
        c += s_red[q][0][ww];
        s += s_red[q][1][ww];
      }
      const uint32_t tile_next = (q < 2 ? zfirst : ofirst) + (q & 1u);
      if (c && tile_next < a.ntiles) {
        atomicAdd(&a.acc_next[tile_next].x, c);
        atomicAdd(&a.acc_next[tile_next].y, s);
      }
    }
  }
  if (last_cta(a.done)) {
    if (threadIdx.x == 0) a.zw[a.R] = a.pre[a.ntiles];
    if (a.key_out) tile_prefix(a.acc_next, a.pre_next, a.ntiles, s_warp);
  }
}

// All L levels in one launch of one thread-block cluster when the runs fit in
// its shared memory.  CTA c owns positions [c S, c S + S) of every level's
// order.  A level: read the slice, stable-partition it locally (zeros, then
// ones) into the same buffer, publish the CTA's (zeros, zero weight), and
// after a cluster barrier copy the two partitioned segments, which are
// contiguous in the next level's order, into their owners' other buffer with
// coalesced distributed-shared-memory stores; a second barrier ends the level.
// Same (Z, W) arrays as k_runs_level.
constexpr int kCT = 1024;           // threads per CTA of the cluster
constexpr int kCPer = 8;            // most elements a thread holds (one per round)
constexpr int kCSlice = kCT * kCPer;
constexpr int kCMax = 16;           // largest cluster (above 8 needs the non-portable attribute)

struct BuildArgs {
  const uint32_t* rec_s;
  const uint32_t* rec_a;
  const uint32_t* kbits;  // keys enter the matrix as their ranks (key_rank)
  const uint32_t* kpre;
  uint2* zw;
  uint32_t R, L, slice;
};

__global__ void __launch_bounds__(kCT) k_runs_build_cluster(BuildArgs a) {
  grid_dep_sync();
  extern __shared__ uint2 s_dyn[];  // two buffers of `slice` (key, weight)
  __shared__ unsigned long long s_rw[kCPer * 32];  // per (round, warp) (zeros, zero weight)
  __shared__ unsigned long long s_tot, s_pre, s_all;
  cg::cluster_group cl = cg::this_cluster();
  const uint32_t rank = cl.block_rank(), C = cl.num_blocks();
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t S = a.slice, base = rank * S;
  const uint32_t cnt = base < a.R ? min(S, a.R - base) : 0u;
  const uint32_t q = (S + kCT - 1) / kCT;  // rounds (the same in every CTA)
  const float invS = 1.0f / (float)S;
  for (uint32_t i = threadIdx.x; i < cnt; i += kCT) {
    const uint32_t r = base + i;
    const uint32_t st = a.rec_s[r], e = a.rec_s[r + 1], a0 = a.rec_a[r];
    const uint32_t len = e - st;
    s_dyn[i] = make_uint2(key_rank(a.kbits, a.kpre, a0 ? a0 + len - 1 : 0u), len);
  }
  cl.sync();
  for (uint32_t l = 0; l < a.L; ++l) {
    uint2* cur = s_dyn + (l & 1) * S;
    uint2* nxt = s_dyn + ((l + 1) & 1) * S;
    const uint32_t shift = a.L - 1 - l;
    // round k holds positions [k * kCT, k * kCT + kCT): lane order is index order
    uint2 el[kCPer];
    uint32_t lz[kCPer], lw[kCPer];
#pragma unroll
    for (int k = 0; k < kCPer; ++k) {
      if (k >= (int)q) break;  // q is the same for the whole CTA
      const uint32_t i = k * kCT + threadIdx.x;
      const bool valid = i < cnt;
      el[k] = valid ? cur[i] : make_uint2(0u, 0u);
      const bool zero = valid && !((el[k].x >> shift) & 1u);
      const uint32_t m = __ballot_sync(kFull, zero);
      uint32_t wi = zero ? el[k].y : 0u;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, wi, o);
        if (lane >= (uint32_t)o) wi += y;
      }
      lz[k] = __popc(m & lanemask_lt());
      lw[k] = wi - (zero ? el[k].y : 0u);
      if (lane == 31 && k < (int)q) s_rw[k * 32 + w] = pack_zw(__popc(m), wi);
    }
    __syncthreads();
    // exclusive scan of the q x 32 (round, warp) totals in index order, by
    // warp 0: lane l sums the q consecutive entries [l q, l q + q)
    if (w == 0) {
      unsigned long long part[kCPer];
      unsigned long long sum = 0;
#pragma unroll
      for (int k = 0; k < kCPer; ++k) {
        part[k] = 0;
        if (k < (int)q) {
          part[k] = s_rw[lane * q + k];
          sum += part[k];
        }
      }
      unsigned long long incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(kFull, incl, o);
        if (lane >= (uint32_t)o) incl += y;
      }
      unsigned long long run = incl - sum;
#pragma unroll
      for (int k = 0; k < kCPer; ++k) {
        if (k < (int)q) {
          s_rw[lane * q + k] = run;
          run += part[k];
        }
      }
      if (lane == 31) s_tot = incl;
    }
    __syncthreads();
    const uint32_t nz = (uint32_t)s_tot;
    // local stable partition into `cur` (every element is in registers)
#pragma unroll
    for (int k = 0; k < kCPer; ++k) {
      if (k >= (int)q) break;
      const uint32_t i = k * kCT + threadIdx.x;
      if (i < cnt) {
        const unsigned long long rw = s_rw[k * 32 + w];
        lz[k] += (uint32_t)rw;
        lw[k] += (uint32_t)(rw >> 32);
        const bool zero = !((el[k].x >> shift) & 1u);
        cur[zero ? lz[k] : nz + (i - lz[k])] = el[k];
      }
    }
    cl.sync();  // every CTA's total is published and every slice partitioned
    if (w == 0) {
      const unsigned long long v = lane < C ? *cl.map_shared_rank(&s_tot, lane) : 0ull;
      unsigned long long in = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(kFull, in, o);
        if (lane >= (uint32_t)o) in += y;
      }
      if (lane == rank) s_pre = in - v;
      if (lane == 31) s_all = in;
    }
    __syncthreads();
    const uint32_t Zpre = (uint32_t)s_pre, Wpre = (uint32_t)(s_pre >> 32), Zc = (uint32_t)s_all;
    if (l + 1 < a.L) {
      // zeros go to [Zpre, Zpre + nz), ones to [Zc + base - Zpre, ...)
      const uint32_t one0 = Zc + (base - Zpre);
      for (uint32_t j = threadIdx.x; j < cnt; j += kCT) {
        const uint32_t dst = j < nz ? Zpre + j : one0 + (j - nz);
        // dst / S through a float reciprocal (dst < 2^24, so dst is exact in
        // a float and the estimate is off by at most one)
        int32_t owner = (int32_t)((float)dst * invS);
        int32_t off = (int32_t)dst - owner * (int32_t)S;
        if (off < 0) {
          --owner;
          off += (int32_t)S;
        } else if (off >= (int32_t)S) {
          ++owner;
          off -= (int32_t)S;
        }
        if (dst < a.R) *cl.map_shared_rank(&nxt[off], owner) = cur[j];
      }
    }
    // the barrier orders the copies above; the (Z, W) stores, read only by
    // the next kernel, go out while the other CTAs arrive
    auto token = cl.barrier_arrive();
    uint2* zl = a.zw + (size_t)l * (a.R + 1);
#pragma unroll
    for (int k = 0; k < kCPer; ++k) {
      if (k >= (int)q) break;
      const uint32_t i = k * kCT + threadIdx.x;
      if (i < cnt) zl[base + i] = make_uint2(Zpre + lz[k], Wpre + lw[k]);
    }
    if (rank == 0 && threadIdx.x == 0) zl[a.R] = make_uint2(Zc, (uint32_t)(s_all >> 32));
    cl.barrier_wait(std::move(token));  // the next level's order is in place
  }
}

struct QueryArgs {
  const uint32_t* rec_s;
  const uint32_t* rec_a;
  const uint32_t* bits;
  const uint32_t* wpre;
  const uint32_t* kbits;  // the matrix holds key ranks: thresholds go through key_rank too
  const uint32_t* kpre;
  const uint2* zw;      // level l at zw + l * (R + 1)
  uint32_t* sd;         // distance of each run
  uint32_t R, L;
};

// Index of the run holding position j.
__device__ __forceinline__ uint32_t run_of(const uint32_t* bits, const uint32_t* wpre, uint32_t j) {
  const uint32_t wi = j >> 5, b = j & 31;
  const uint32_t mask_le = b == 31 ? kFull : ((2u << b) - 1u);
  return wpre[wi] + __popc(bits[wi] & mask_le) - 1u;
}

__global__ void __launch_bounds__(256) k_runs_query(QueryArgs a) {
  grid_dep_sync();
  const uint32_t r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= a.R) return;
  const uint32_t x = a.rec_a[r];  // p + 1
  if (x == 0) {
    a.sd[r] = kNone;
    return;
  }
  const uint32_t s = a.rec_s[r];
  const uint32_t rho = run_of(a.bits, a.wpre, x);
  uint32_t lo = rho, partial = 0;
  const uint32_t s1 = a.rec_s[rho];
  if (s1 < x) {  // the run holding p + 1 starts before the window
    const uint32_t e1 = a.rec_s[rho + 1], a1 = a.rec_a[rho];
    const uint32_t vfirst = a1 ? a1 + (x - s1) : 0u;
    if (vfirst < x) partial = min(e1, s) - x;
    lo = rho + 1;
  }
  uint32_t hi = r, cnt = 0;
  const uint32_t stride = a.R + 1;
  // keys below x are the keys whose rank is below the number of keys below x
  const uint32_t xr = key_rank(a.kbits, a.kpre, x);
  for (uint32_t l = 0; l < a.L && lo < hi; ++l) {
    const uint2* zl = a.zw + (size_t)l * stride;
    const uint2 zlo = zl[lo], zhi = zl[hi];
    if ((xr >> (a.L - 1 - l)) & 1u) {
      const uint32_t Zc = zl[a.R].x;
      cnt += zhi.y - zlo.y;
      lo = Zc + (lo - zlo.x);
      hi = Zc + (hi - zhi.x);
    } else {
      lo = zlo.x;
      hi = zhi.x;
    }
  }
  a.sd[r] = 1u + partial + cnt;
}

// kExpPer accesses per thread, kExpThreads apart: each thread's dependent
// loads (word, then distance) for all of them are in flight together.
constexpr int kExpThreads = 256;
constexpr int kExpPer = 8;
__global__ void __launch_bounds__(kExpThreads) k_runs_expand(const uint32_t* __restrict__ bits,
                                                            const uint32_t* __restrict__ wpre,
                                                            const uint32_t* __restrict__ sd, uint32_t n,
                                                            uint32_t* __restrict__ dist, uint32_t nruns,
                                                            const DevStatus* st) {
  grid_dep_sync();
  const uint32_t j0 = blockIdx.x * (kExpThreads * kExpPer) + threadIdx.x;
  uint32_t r[kExpPer];
#pragma unroll
  for (int k = 0; k < kExpPer; ++k) {
    const uint32_t j = j0 + k * kExpThreads;
    r[k] = j < n ? run_of(bits, wpre, j) : 0u;
  }
#pragma unroll
  for (int k = 0; k < kExpPer; ++k) {
    const uint32_t j = j0 + k * kExpThreads;
    if (j < n && in_bounds(st, r[k], nruns)) __stcs(&dist[j], __ldg(&sd[r[k]]));
  }
}

uint32_t key_bits_n(uint64_t n) {  // keys and thresholds lie in [0, n]
  uint32_t L = 1;
  while (L < 33 && (1ULL << L) <= n) ++L;
  return L;
}

// Arrays the marking pass writes (sized by N) come first; those sized by the
// number of runs R follow.
struct RunsLayout {
  DevStatus* st;
  uint32_t* done;
  uint32_t* kbits;  // key bitmap over [0, n] (zeroed with the status)
  uint32_t *tcnt, *tpre;
  uint32_t *kpre, *ktcnt, *ktpre;
  uint32_t kwords, ktiles;
  size_t zero_bytes;
  uint32_t *bits, *wpre, *rec_s, *rec_a;
  uint32_t *sd, *k0, *k1, *w0, *w1;
  uint2 *acc, *pre, *zw;
  uint32_t L, mtiles, rtiles;
  size_t acc_bytes;
  size_t total;
};

RunsLayout runs_layout(void* ws, uint64_t n, uint64_t R) {
  RunsLayout W;
  Carver cv(ws);
  const uint64_t nn = n ? n : 1, rr = R ? R : 1;
  W.L = key_bits_n(rr + 1);  // key ranks and thresholds lie in [0, R + 1]
  W.mtiles = ceil_div_u32(nn, kMTile);
  W.rtiles = ceil_div_u32(rr, kRTile);
  W.kwords = (uint32_t)(nn / 32 + 2);  // keys and thresholds lie in [0, n]
  W.ktiles = rank_tiles(W.kwords);
  W.st = cv.take<DevStatus>(1);
  W.done = cv.take<uint32_t>(64);
  W.kbits = cv.take<uint32_t>(W.kwords);
  W.zero_bytes = cv.off;
  W.tcnt = cv.take<uint32_t>(W.mtiles + 1);
  W.tpre = cv.take<uint32_t>(W.mtiles + 1);
  W.kpre = cv.take<uint32_t>(W.kwords);
  W.ktcnt = cv.take<uint32_t>(W.ktiles + 1);
  W.ktpre = cv.take<uint32_t>(W.ktiles + 1);
  W.bits = cv.take<uint32_t>(nn / 32 + 2);
  W.wpre = cv.take<uint32_t>(nn / 32 + 2);
  W.rec_s = cv.take<uint32_t>(nn + 1);
  W.rec_a = cv.take<uint32_t>(nn);
  const size_t acc_off = cv.off;
  W.acc = cv.take<uint2>((uint64_t)(W.L + 1) * (W.rtiles + 1));
  W.acc_bytes = cv.off - acc_off;
  W.pre = cv.take<uint2>((uint64_t)(W.L + 1) * (W.rtiles + 1));
  W.sd = cv.take<uint32_t>(rr);
  W.k0 = cv.take<uint32_t>(rr);
  W.k1 = cv.take<uint32_t>(rr);
  W.w0 = cv.take<uint32_t>(rr);
  W.w1 = cv.take<uint32_t>(rr);
  W.zw = cv.take<uint2>((uint64_t)W.L * (rr + 1));
  W.total = cv.bytes();
  return W;
}

// Runs the automatic choice reserves room for: a third of the accesses, at
// most 2^24 (the matrix over runs then costs less than the one over accesses).
uint64_t runs_reserve(uint64_t n) {
  const uint64_t r = n / 3 + 1;
  return r < (1ULL << 24) ? r : (1ULL << 24);
}

// Whether a cluster of C CTAs of k_runs_build_cluster can be resident, asked
// once per device and cluster size with the largest shared-memory request (a
// smaller one fits whenever that does); the occupancy query is slow next to
// the kernels around it.
bool cluster_fits(uint32_t C, const cudaLaunchConfig_t& cfg) {
  constexpr int kDevs = 64;
  static std::atomic<int8_t> known[kDevs][kCMax + 1];  // 0 unknown, 1 yes, 2 no
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kDevs || C > (uint32_t)kCMax) {
    (void)cudaGetLastError();
    return false;
  }
  const int8_t k = known[dev][C].load(std::memory_order_relaxed);
  if (k) return k == 1;
  cudaLaunchConfig_t q = cfg;
  q.dynamicSmemBytes = 2 * kCSlice * sizeof(uint2);
  int clusters = 0;
  const bool ok = cudaOccupancyMaxActiveClusters(&clusters, k_runs_build_cluster, &q) == cudaSuccess && clusters >= 1;
  if (!ok) (void)cudaGetLastError();
  known[dev][C].store(ok ? 1 : 2, std::memory_order_relaxed);
  return ok;
}

ptc_status stack_distance_runs(const uint32_t* prev, uint64_t n, uint32_t* dist_out, void* ws, size_t ws_bytes,
                               cudaStream_t s, int method, RunsView* view, uint32_t* defer_err = nullptr) {
  const RunsLayout M = runs_layout(ws, n, 1);
  if (!ws_ok(ws, ws_bytes, M.total)) return PTC_ERR_WORKSPACE;
  if (begin_call(ws, M.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  MarkArgs m;
  m.prev = prev;
  m.n = (uint32_t)n;
  m.ntiles = M.mtiles;
  m.bits = M.bits;
  m.wpre = M.wpre;
  m.rec_s = M.rec_s;
  m.rec_a = M.rec_a;
  m.tcnt = M.tcnt;
  m.tpre = M.tpre;
  m.done = &M.done[63];
  m.kbits = M.kbits;
  m.st = M.st;
  if ((reinterpret_cast<uintptr_t>(prev) & 15) == 0) {
    PTC_KERNEL("k_runs_count", s, k_runs_count4, M.mtiles, kMT, 0, m);
    PTC_KERNEL("k_runs_mark", s, k_runs_mark4, M.mtiles, kMT, 0, m);
  } else {
    PTC_KERNEL("k_runs_count", s, k_runs_count, M.mtiles, kMT, 0, m);
    PTC_KERNEL("k_runs_mark", s, k_runs_mark, M.mtiles, kMT, 0, m);
  }
  if (bitmap_ranks(M.kbits, M.kwords, M.kpre, M.ktcnt, M.ktpre, &M.done[62], nullptr, s) != PTC_OK) return PTC_ERR_CUDA;
  DevStatus h;
  ptc_status rc = end_call(M.st, s, &h);
  if (rc != PTC_OK) return rc;
  const uint64_t R = h.value[1];
  const RunsLayout W = runs_layout(ws, n, R);
  const bool fits = R >= 1 && R <= n && ws_bytes >= W.total;
  if (method == PTC_SD_AUTO && (!fits || R > n / 3)) return stack_distance_points(prev, n, dist_out, ws, ws_bytes, s);
  if (!fits) return PTC_ERR_WORKSPACE;
  const FillRange zf[2] = {{W.acc, W.acc_bytes, 0u}, {W.done, 64 * sizeof(uint32_t), 0u}};
  if (fill_many_async(zf, 2, s) != PTC_OK) return PTC_ERR_CUDA;
  const uint32_t R32 = (uint32_t)R, T = W.rtiles, L = W.L;
  const size_t tstride = (size_t)T + 1;
  // one cluster when the runs fit in its shared memory, else one launch per level
  bool built = false;
  static int attrs_set = -1;  // per process: the attributes belong to the device function
  if (attrs_set < 0)
    attrs_set = cudaFuncSetAttribute(k_runs_build_cluster, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)(2 * kCSlice * sizeof(uint2))) == cudaSuccess &&
                cudaFuncSetAttribute(k_runs_build_cluster, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) ==
                    cudaSuccess;
  for (uint32_t cmax = kCMax; attrs_set == 1 && !built && cmax >= 8; cmax /= 2) {
    uint32_t C = ceil_div_u32(R, 2048);  // about two runs per thread
    if (C > cmax) C = cmax;
    if ((uint64_t)C * kCSlice < R) continue;
    BuildArgs b;
    b.rec_s = W.rec_s;
    b.rec_a = W.rec_a;
    b.kbits = W.kbits;
    b.kpre = W.kpre;
    b.zw = W.zw;
    b.R = R32;
    b.L = L;
    b.slice = ceil_div_u32(R, C);
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(C);
    cfg.blockDim = dim3(kCT);
    cfg.dynamicSmemBytes = 2 * (size_t)b.slice * sizeof(uint2);
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (!cluster_fits(C, cfg)) continue;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // as launch_pdl
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.numAttrs = 2;
    cudaError_t e = cudaSuccess;
    PTC_LAUNCH("k_runs_build_cluster", s, e = cudaLaunchKernelEx(&cfg, k_runs_build_cluster, b));
    if (e == cudaSuccess)
      built = true;
    else
      (void)cudaGetLastError();
  }
  if (!built) {
    PTC_KERNEL("k_runs_init", s, k_runs_init, T, kRT, 0, W.rec_s, W.rec_a, W.kbits, W.kpre, W.k0, W.w0, W.acc, W.pre,
               &W.done[0], R32, T, L - 1);
    uint32_t* keys[2] = {W.k0, W.k1};
    uint32_t* wts[2] = {W.w0, W.w1};
    for (uint32_t l = 0; l < L; ++l) {
      const bool last = l + 1 == L;
      LevelArgs a;
      a.key_in = keys[l & 1];
      a.wt_in = wts[l & 1];
      a.key_out = last ? nullptr : keys[(l + 1) & 1];
      a.wt_out = last ? nullptr : wts[(l + 1) & 1];
      a.zw = W.zw + (size_t)l * (R + 1);
      a.pre = W.pre + (size_t)l * tstride;
      a.acc_next = last ? nullptr : W.acc + (size_t)(l + 1) * tstride;
      a.pre_next = last ? nullptr : W.pre + (size_t)(l + 1) * tstride;
      a.done = &W.done[1 + l];
      a.R = R32;
      a.ntiles = T;
      a.shift = L - 1 - l;
      PTC_KERNEL("k_runs_level", s, k_runs_level, T, kRT, 0, a);
    }
  }
  QueryArgs q;
  q.rec_s = W.rec_s;
  q.rec_a = W.rec_a;
  q.bits = W.bits;
  q.wpre = W.wpre;
  q.kbits = W.kbits;
  q.kpre = W.kpre;
  q.zw = W.zw;
  q.sd = W.sd;
  q.R = R32;
  q.L = L;
  PTC_KERNEL("k_runs_query", s, k_runs_query, ceil_div_u32(R, 256), 256, 0, q);
  PTC_KERNEL("k_runs_expand", s, k_runs_expand, ceil_div_u32(n, kExpThreads * kExpPer), kExpThreads, 0, W.bits, W.wpre, W.sd, (uint32_t)n, dist_out, R32, W.st);
  const ptc_status done = defer_err ? defer_status(W.st, defer_err, s) : end_call(W.st, s, &h);
  if (done == PTC_OK && view) {
    view->used = true;
    view->R = R32;
    view->rec_s = W.rec_s;
    view->sd = W.sd;
    view->bits = W.bits;
    view->wpre = W.wpre;
  }
  return done;
}

}  // namespace

ptc_status stack_distance_view(const uint32_t* prev, uint64_t n, uint32_t* dist_out, int method, void* ws,
                               size_t ws_bytes, cudaStream_t s, RunsView* view, uint32_t* defer_err) {
  *view = RunsView{};
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (n == 0) return PTC_OK;
  if (!prev || !dist_out) return PTC_ERR_INVALID_ARG;
  if (method == PTC_SD_POINTS) return stack_distance_points(prev, n, dist_out, ws, ws_bytes, s);
  return stack_distance_runs(prev, n, dist_out, ws, ws_bytes, s, method, view, defer_err);
}

}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_stack_distance_ex_workspace_bytes(uint64_t n, int method) {
  const size_t pts = stack_distance_points_bytes(n);
  if (method == PTC_SD_POINTS) return pts;
  if (method == PTC_SD_RUNS) return runs_layout(nullptr, n, n).total;
  const size_t runs = runs_layout(nullptr, n, runs_reserve(n)).total;
  return pts > runs ? pts : runs;
}

extern "C" size_t ptc_stack_distance_workspace_bytes(uint64_t n) {
  return ptc_stack_distance_ex_workspace_bytes(n, PTC_SD_AUTO);
}

extern "C" ptc_status ptc_stack_distance_ex(const uint32_t* prev, uint64_t n, uint32_t* dist_out, int method,
                                            void* ws, size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (method != PTC_SD_AUTO && method != PTC_SD_POINTS && method != PTC_SD_RUNS) return PTC_ERR_INVALID_ARG;
  if (n == 0) return PTC_OK;
  if (!prev || !dist_out) return PTC_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  if (method == PTC_SD_POINTS) return stack_distance_points(prev, n, dist_out, ws, ws_bytes, s);
  return stack_distance_runs(prev, n, dist_out, ws, ws_bytes, s, method, nullptr);
}

extern "C" ptc_status ptc_stack_distance(const uint32_t* prev, uint64_t n, uint32_t* dist_out, void* ws,
                                         size_t ws_bytes, void* stream) {
  return ptc_stack_distance_ex(prev, n, dist_out, PTC_SD_AUTO, ws, ws_bytes, stream);
}
