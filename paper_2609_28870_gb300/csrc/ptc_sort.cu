// Stage b: previous / next use of every block (Belady's next access).
//
// A stable LSD radix sort of (id, i) pairs by id groups the accesses of each
// block in index order; neighbours in the sorted order with equal ids are
// (prev, next) pairs.  Each digit pass is reduce-then-scan, so no tile ever
// waits on another:
//   k_sort_count    digit counts of every tile, stored digit-major
//   k_sort_rowscan  one CTA per digit: exclusive prefix of its counts over
//                   tiles, and the digit's total
//   k_sort_scatter  stable rank of every element inside its tile (warp
//                   match_any + per-warp counters), reorder in shared memory,
//                   coalesced writes to (digit base + tile prefix + rank).
//                   The last pass writes prev / next instead of the sorted
//                   pairs: neighbours inside a tile's digit run are linked on
//                   the spot, and the first / last pair of every run is kept
//                   for k_sort_links
//   k_sort_links    one CTA per digit of the last pass: links the runs of
//                   consecutive non-empty tiles
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kSortThreads = 256;
constexpr int kSortPer = 16;
constexpr int kSortTile = kSortThreads * kSortPer;  // 4096
constexpr int kSortWarps = kSortThreads / 32;
constexpr int kRadix = 256;                          // largest digit range

// Digit counts of one tile for one pass: cnt[d * T + tile].  Per-warp
// shared-memory histograms keep same-address atomics inside one warp.
__global__ void __launch_bounds__(kSortThreads) k_sort_count(const uint32_t* __restrict__ keys, uint32_t n,
                                                             uint32_t shift, uint32_t R, uint32_t T,
                                                             uint32_t key_limit, bool vec,
                                                             uint32_t* __restrict__ cnt, DevStatus* st) {
  grid_dep_sync();
  __shared__ uint32_t h[kSortWarps][kRadix];
  for (uint32_t x = threadIdx.x; x < kSortWarps * kRadix; x += kSortThreads) (&h[0][0])[x] = 0;
  __syncthreads();
  const uint32_t tile = blockIdx.x, w = threadIdx.x >> 5;
  const uint32_t base = tile * kSortTile;
  bool bad = false;
  if (vec && base + kSortTile <= n) {  // 16-byte aligned keys, whole tile
    const uint4* k4 = reinterpret_cast<const uint4*>(keys + base);
    uint4 v[kSortPer / 4];
#pragma unroll
    for (int j = 0; j < kSortPer / 4; ++j) v[j] = k4[j * kSortThreads + threadIdx.x];
#pragma unroll
    for (int j = 0; j < kSortPer / 4; ++j) {
      const uint32_t e[4] = {v[j].x, v[j].y, v[j].z, v[j].w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        bad |= e[q] >= key_limit;
        atomicAdd(&h[w][(e[q] >> shift) & (R - 1)], 1u);
      }
    }
  } else {
    for (uint32_t i = base + threadIdx.x; i < n; i += kSortThreads) {
      const uint32_t k = keys[i];
      bad |= k >= key_limit;
      atomicAdd(&h[w][(k >> shift) & (R - 1)], 1u);
    }
  }
  if (bad) raise_err(st, kErrInvalid);
  __syncthreads();
  for (uint32_t x = threadIdx.x; x < R; x += kSortThreads) {
    uint32_t c = 0;
#pragma unroll
    for (int ww = 0; ww < kSortWarps; ++ww) c += h[ww][x];
    cnt[(size_t)x * T + tile] = c;
  }
}

// Lanes of the warp holding the same digit (ballot per digit bit: warp-level
// multisplit), restricted to the lanes in `valid`.
__device__ __forceinline__ uint32_t digit_peers(uint32_t d, uint32_t width, uint32_t valid) {
  uint32_t peers = valid;
#pragma unroll
  for (uint32_t b = 0; b < 8; ++b) {
    if (b < width) {
      const uint32_t bit = (d >> b) & 1u;
      const uint32_t bal = __ballot_sync(kFull, bit);
      peers &= bit ? bal : ~bal;
    }
  }
  return peers;
}

// Exclusive block scan of one value per thread (256 threads); returns the
// exclusive prefix, `total` receives the block sum.
template <class V>
__device__ __forceinline__ V block_excl_scan(V x, V* s_warp, V& total) {
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  V incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const V y = __shfl_up_sync(kFull, incl, o);
    if (lane >= (uint32_t)o) incl += y;
  }
  if (lane == 31) s_warp[w] = incl;
  __syncthreads();
  V pre = 0, tot = 0;
#pragma unroll
  for (int ww = 0; ww < kSortWarps; ++ww) {
    const V v = s_warp[ww];
    if (ww < (int)w) pre += v;
    tot += v;
  }
  __syncthreads();
  total = tot;
  return pre + incl - x;
}

// One CTA per digit: off[d * T + t] = sum of cnt[d * T + t'] over t' < t,
// tot[d] = the row's sum.
__global__ void __launch_bounds__(kSortThreads) k_sort_rowscan(const uint32_t* __restrict__ cnt, uint32_t T,
                                                               uint32_t* __restrict__ off, uint32_t* __restrict__ tot) {
  grid_dep_sync();
  __shared__ uint32_t s_warp[kSortWarps];
  const uint32_t d = blockIdx.x;
  const uint32_t per = (T + kSortThreads - 1) / kSortThreads;
  const uint32_t t0 = threadIdx.x * per, t1 = min(t0 + per, T);
  const uint32_t* row = cnt + (size_t)d * T;
  uint32_t s = 0;
  for (uint32_t t = t0; t < t1; ++t) s += row[t];
  uint32_t total;
  uint32_t run = block_excl_scan<uint32_t>(s, s_warp, total);
  uint32_t* orow = off + (size_t)d * T;
  for (uint32_t t = t0; t < t1; ++t) {
    const uint32_t c = row[t];
    orow[t] = run;
    run += c;
  }
  if (threadIdx.x == 0) tot[d] = total;
}

struct ScatterArgs {
  const uint32_t* keys_in;
  const uint32_t* vals_in;  // null: values are the element indices
  uint32_t* keys_out;       // sorted pairs (all passes but the last)
  uint32_t* vals_out;
  uint32_t* prev;           // last pass: prev / next by element index
  uint32_t* next;
  uint2* head_kv;           // last pass: first / last (key, value) of each (digit, tile) run
  uint2* tail_kv;
  const uint32_t* off;      // this pass's tile prefixes, digit-major
  const uint32_t* tot;      // this pass's digit totals
  uint32_t n, T, shift, R, width;
  const DevStatus* st;      // for the checked build's bounds checks
};

template <bool LAST>
__global__ void __launch_bounds__(kSortThreads, 3) k_sort_scatter(ScatterArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_keys[kSortTile];
  __shared__ uint32_t s_vals[kSortTile];
  __shared__ uint32_t s_whist[kSortWarps][kRadix];
  __shared__ uint32_t s_start[kRadix + 1];
  __shared__ uint32_t s_gbase[kRadix];
  __shared__ unsigned long long s_warp[kSortWarps];

  const uint32_t tile = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t R = a.R, dmask = R - 1;
  for (uint32_t x = lane; x < R; x += 32) s_whist[w][x] = 0;
  __syncwarp();

  // stable rank of each element among the equal digits of its warp slice
  const uint32_t wbase = tile * kSortTile + w * (32 * kSortPer);
  uint32_t key[kSortPer], rank2[kSortPer / 2];  // ranks < 512, two per register
#pragma unroll
  for (int j = 0; j < kSortPer; ++j) {
    const uint32_t i = wbase + j * 32 + lane;
    key[j] = i < a.n ? a.keys_in[i] : 0u;
  }
#pragma unroll
  for (int j = 0; j < kSortPer; ++j) {
    const uint32_t i = wbase + j * 32 + lane;
    const bool valid = i < a.n;
    const uint32_t d = (key[j] >> a.shift) & dmask;
    const uint32_t peers = digit_peers(d, a.width, __ballot_sync(kFull, valid));
    const uint32_t leader = valid ? __ffs(peers) - 1 : lane;
    uint32_t before = 0;
    if (valid && lane == leader) {
      before = s_whist[w][d];
      s_whist[w][d] = before + __popc(peers);
    }
    before = __shfl_sync(kFull, before, leader);
    const uint32_t r = before + __popc(peers & lanemask_lt());
    if (j & 1) rank2[j >> 1] |= r << 16; else rank2[j >> 1] = r;
    __syncwarp();
  }
  __syncthreads();

  // per digit: offsets of the warps inside the tile, the tile's count, the
  // digit's start in the tile and its global base
  const uint32_t d = threadIdx.x;
  uint32_t c = 0;
  if (d < R) {
#pragma unroll
    for (int ww = 0; ww < kSortWarps; ++ww) {
      const uint32_t v = s_whist[ww][d];
      s_whist[ww][d] = c;
      c += v;
    }
  }
  const unsigned long long packed = d < R ? ((unsigned long long)a.tot[d] << 32) | c : 0ull;
  unsigned long long all;
  const unsigned long long ex = block_excl_scan<unsigned long long>(packed, s_warp, all);
  if (d < R) {
    s_start[d] = (uint32_t)ex;
    s_gbase[d] = (uint32_t)(ex >> 32) + a.off[(size_t)d * a.T + tile];
  }
  if (d == 0) s_start[R] = (uint32_t)all;
  __syncthreads();

  // reorder the tile by digit in shared memory
#pragma unroll
  for (int j = 0; j < kSortPer; ++j) {
    const uint32_t i = wbase + j * 32 + lane;
    if (i < a.n) {
      const uint32_t dd = (key[j] >> a.shift) & dmask;
      const uint32_t p = s_start[dd] + s_whist[w][dd] + ((rank2[j >> 1] >> (16 * (j & 1))) & 0xFFFFu);
      s_keys[p] = key[j];
      s_vals[p] = a.vals_in ? a.vals_in[i] : i;
    }
  }
  __syncthreads();

  const uint32_t tile_n = s_start[R];
  if (!LAST) {
    for (uint32_t p = threadIdx.x; p < tile_n; p += kSortThreads) {
      const uint32_t k = s_keys[p];
      const uint32_t dd = (k >> a.shift) & dmask;
      const uint32_t dst = s_gbase[dd] + (p - s_start[dd]);
      if (in_bounds(a.st, dst, a.n)) {
        a.keys_out[dst] = k;
        a.vals_out[dst] = s_vals[p];
      }
    }
  } else {
    for (uint32_t p = threadIdx.x; p < tile_n; p += kSortThreads) {
      const uint32_t k = s_keys[p], v = s_vals[p];
      const uint32_t dd = (k >> a.shift) & dmask;
      const uint32_t lo = s_start[dd], hi = s_start[dd + 1];
      if (in_bounds(a.st, v, a.n)) {
        if (p > lo) a.prev[v] = s_keys[p - 1] == k ? s_vals[p - 1] : kNone;
        if (p + 1 < hi) a.next[v] = s_keys[p + 1] == k ? s_vals[p + 1] : kNone;
      }
      const size_t cell = (size_t)dd * a.T + tile;
      if (p == lo) a.head_kv[cell] = make_uint2(k, v);
      if (p + 1 == hi) a.tail_kv[cell] = make_uint2(k, v);
    }
  }
}

__device__ __forceinline__ void link_runs(const uint2* __restrict__ head_kv, const uint2* __restrict__ tail_kv,
                                          size_t row, int32_t prev_cell, uint32_t cell, uint32_t n,
                                          uint32_t* __restrict__ prev, uint32_t* __restrict__ next) {
  const uint2 h = head_kv[row + cell];
  if (prev_cell < 0) {
    if (h.y < n) prev[h.y] = kNone;
    return;
  }
  const uint2 t = tail_kv[row + (uint32_t)prev_cell];
  const bool same = t.x == h.x;
  if (h.y < n) prev[h.y] = same ? t.y : kNone;
  if (t.y < n) next[t.y] = same ? h.y : kNone;
}

// One CTA per digit of the last pass: joins each non-empty (digit, tile) run
// to the previous non-empty run of the same digit.
__global__ void __launch_bounds__(kSortThreads) k_sort_links(const uint32_t* __restrict__ cnt, uint32_t T,
                                                             const uint2* __restrict__ head_kv,
                                                             const uint2* __restrict__ tail_kv, uint32_t n,
                                                             uint32_t* __restrict__ prev, uint32_t* __restrict__ next) {
  grid_dep_sync();
  __shared__ int32_t s_last[kSortThreads];
  const uint32_t d = blockIdx.x;
  const size_t row = (size_t)d * T;
  const uint32_t per = (T + kSortThreads - 1) / kSortThreads;
  const uint32_t t0 = threadIdx.x * per, t1 = min(t0 + per, T);
  int32_t last = -1;
  for (uint32_t t = t0; t < t1; ++t)
    if (cnt[row + t]) last = (int32_t)t;
  s_last[threadIdx.x] = last;
  __syncthreads();
  // last non-empty tile before this thread's chunk, and of the whole row
  int32_t before = -1, row_last = -1;
  for (uint32_t x = 0; x < kSortThreads; ++x) {
    const int32_t v = s_last[x];
    if (x < threadIdx.x && v > before) before = v;
    if (v > row_last) row_last = v;
  }
  for (uint32_t t = t0; t < t1; ++t) {
    if (!cnt[row + t]) continue;
    link_runs(head_kv, tail_kv, row, before, t, n, prev, next);
    before = (int32_t)t;
  }
  if (row_last >= 0 && (uint32_t)row_last >= t0 && (uint32_t)row_last < t1) {
    const uint2 t = tail_kv[row + (uint32_t)row_last];
    if (t.y < n) next[t.y] = kNone;
  }
}

uint32_t key_bits(uint64_t D) {
  uint32_t b = 1;
  while (b < 32 && (1ULL << b) < D) ++b;
  return b;
}

struct SortLayout {
  DevStatus* st;
  uint32_t *cnt, *off, *tot;
  uint2 *head_kv, *tail_kv;
  uint32_t *k0, *v0, *k1, *v1;
  size_t zero_bytes;
  size_t total;
};

SortLayout sort_layout(void* ws, uint64_t n) {
  SortLayout L;
  Carver cv(ws);
  const uint64_t nn = n ? n : 1;
  const uint64_t cells = (uint64_t)kRadix * (ceil_div_u32(nn, kSortTile));
  L.st = cv.take<DevStatus>(1);
  L.zero_bytes = cv.off;
  L.cnt = cv.take<uint32_t>(cells);
  L.off = cv.take<uint32_t>(cells);
  L.tot = cv.take<uint32_t>(kRadix);
  L.head_kv = cv.take<uint2>(cells);
  L.tail_kv = cv.take<uint2>(cells);
  L.k0 = cv.take<uint32_t>(nn);
  L.v0 = cv.take<uint32_t>(nn);
  L.k1 = cv.take<uint32_t>(nn);
  L.v1 = cv.take<uint32_t>(nn);
  L.total = cv.bytes();
  return L;
}

}  // namespace
}  // namespace ptc

using namespace ptc;

size_t ptc::reuse_by_sort_bytes(uint64_t n) { return sort_layout(nullptr, n).total; }

// prev / next from a stable radix sort of every (id, i) (argument checks are
// the caller's).
ptc_status ptc::reuse_by_sort(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out,
                              uint32_t* next_out, void* ws, size_t ws_bytes, cudaStream_t s) {
  if (!ws_ok(ws, ws_bytes, sort_layout(nullptr, n).total)) return PTC_ERR_WORKSPACE;
  const SortLayout L = sort_layout(ws, n);
  if (begin_call(ws, L.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  const uint32_t bits = key_bits(n_distinct);
  const uint32_t passes = (bits + 7) / 8;
  const uint32_t T = ceil_div_u32(n, kSortTile);
  const uint32_t n32 = (uint32_t)n;
  const uint32_t* kin = ids;
  const uint32_t* vin = nullptr;
  uint32_t *kout = L.k0, *vout = L.v0;
  uint32_t shift = 0;
  for (uint32_t p = 0; p < passes; ++p) {
    const uint32_t width = (bits - shift + (passes - p) - 1) / (passes - p);  // spread bits evenly
    const uint32_t R = 1u << width;
    const bool last = p + 1 == passes;
    PTC_KERNEL("k_sort_count", s, k_sort_count, T, kSortThreads, 0, kin, n32, shift, R, T, p == 0 ? (uint32_t)n_distinct : kNone, ((uintptr_t)kin & 15) == 0, L.cnt, L.st);
    PTC_KERNEL("k_sort_rowscan", s, k_sort_rowscan, R, kSortThreads, 0, L.cnt, T, L.off, L.tot);
    ScatterArgs a;
    a.keys_in = kin;
    a.vals_in = vin;
    a.keys_out = kout;
    a.vals_out = vout;
    a.prev = prev_out;
    a.next = next_out;
    a.head_kv = L.head_kv;
    a.tail_kv = L.tail_kv;
    a.off = L.off;
    a.tot = L.tot;
    a.n = n32;
    a.T = T;
    a.shift = shift;
    a.R = R;
    a.width = width;
    a.st = L.st;
    if (last) {
      PTC_KERNEL("k_sort_scatter", s, k_sort_scatter<true>, T, kSortThreads, 0, a);
      PTC_KERNEL("k_sort_links", s, k_sort_links, R, kSortThreads, 0, L.cnt, T, L.head_kv, L.tail_kv, n32, prev_out, next_out);
    } else {
      PTC_KERNEL("k_sort_scatter", s, k_sort_scatter<false>, T, kSortThreads, 0, a);
    }
    kin = kout;
    vin = vout;
    kout = (kout == L.k0) ? L.k1 : L.k0;
    vout = (vout == L.v0) ? L.v1 : L.v0;
    shift += width;
  }
  DevStatus h;
  return end_call(L.st, s, &h);
}

size_t ptc::sort_pairs_bytes(uint64_t n) { return sort_layout(nullptr, n).total; }

// Stable LSD sort of (keys, vals) by the low `bits` bits of the keys, queued
// on `s` without waiting; *keys_sorted / *vals_sorted point into `ws` (which
// must hold sort_pairs_bytes(n)).  Errors go to `st`.
void ptc::sort_pairs(const uint32_t* keys, const uint32_t* vals, uint32_t n, uint32_t bits, void* ws,
                     cudaStream_t s, DevStatus* st, const uint32_t** keys_sorted, const uint32_t** vals_sorted) {
  const SortLayout L = sort_layout(ws, n);
  if (bits < 1) bits = 1;
  const uint32_t passes = (bits + 7) / 8;
  const uint32_t T = ceil_div_u32(n ? n : 1, kSortTile);
  const uint32_t* kin = keys;
  const uint32_t* vin = vals;
  uint32_t *kout = L.k0, *vout = L.v0;
  uint32_t shift = 0;
  for (uint32_t p = 0; p < passes; ++p) {
    const uint32_t width = (bits - shift + (passes - p) - 1) / (passes - p);
    const uint32_t R = 1u << width;
    PTC_KERNEL("k_sort_count", s, k_sort_count, T, kSortThreads, 0, kin, n, shift, R, T, kNone, ((uintptr_t)kin & 15) == 0, L.cnt, st);
    PTC_KERNEL("k_sort_rowscan", s, k_sort_rowscan, R, kSortThreads, 0, L.cnt, T, L.off, L.tot);
    ScatterArgs a = {};
    a.keys_in = kin;
    a.vals_in = vin;
    a.keys_out = kout;
    a.vals_out = vout;
    a.off = L.off;
    a.tot = L.tot;
    a.n = n;
    a.T = T;
    a.shift = shift;
    a.R = R;
    a.width = width;
    a.st = st;
    PTC_KERNEL("k_sort_scatter", s, k_sort_scatter<false>, T, kSortThreads, 0, a);
    kin = kout;
    vin = vout;
    kout = (kout == L.k0) ? L.k1 : L.k0;
    vout = (vout == L.v0) ? L.v1 : L.v0;
    shift += width;
  }
  *keys_sorted = kin;
  *vals_sorted = vin;
}
