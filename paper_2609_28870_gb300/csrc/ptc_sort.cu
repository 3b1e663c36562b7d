// Stage b: previous / next use of every block (Belady's next access).
//
// A stable LSD radix sort of (id, i) pairs by id groups the accesses of each
// block in index order; neighbours in the sorted order with equal ids are
// (prev, next) pairs.
//   k_sort_hist      digit histograms of every pass in one read of ids
//   k_sort_pass      one 8-bit digit pass, single-pass ("onesweep" style,
//                    Adinets & Merrill 2022): warp-level ranking with
//                    match_any, per-digit decoupled look-back across tiles,
//                    reorder in shared memory, coalesced writes
//   k_adjacent       prev/next from the sorted pairs
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kSortThreads = 256;
constexpr int kSortPer = 16;
constexpr int kSortTile = kSortThreads * kSortPer;  // 4096
constexpr int kSortWarps = kSortThreads / 32;
constexpr int kRadix = 256;

__global__ void __launch_bounds__(256) k_sort_hist(const uint32_t* __restrict__ ids, uint64_t n, uint64_t D,
                                                   uint32_t passes, uint32_t bits,
                                                   unsigned long long* __restrict__ hist, DevStatus* st) {
  __shared__ uint32_t sh[4][kRadix];
  for (uint32_t x = threadIdx.x; x < 4 * kRadix; x += blockDim.x) (&sh[0][0])[x] = 0;
  __syncthreads();
  bool bad = false;
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x) {
    const uint32_t k = ids[i];
    if (k >= D) bad = true;
    for (uint32_t p = 0; p < passes; ++p) {
      const uint32_t sh_bits = 8 * p;
      const uint32_t w = bits - sh_bits < 8 ? bits - sh_bits : 8;
      atomicAdd(&sh[p][(k >> sh_bits) & ((1u << w) - 1)], 1u);
    }
  }
  if (bad) raise_err(st, kErrInvalid);
  __syncthreads();
  for (uint32_t x = threadIdx.x; x < passes * kRadix; x += blockDim.x) {
    const uint32_t v = (&sh[0][0])[x];
    if (v) atomicAdd(&hist[x], (unsigned long long)v);
  }
}

// Exclusive offsets of every digit of every pass from the histograms.
__global__ void __launch_bounds__(kRadix) k_sort_offsets(const unsigned long long* __restrict__ hist, uint32_t passes,
                                                         unsigned long long* __restrict__ offs) {
  __shared__ unsigned long long s_w[kRadix / 32];
  const uint32_t d = threadIdx.x, lane = d & 31, w = d >> 5;
  for (uint32_t p = 0; p < passes; ++p) {
    const unsigned long long c = hist[p * kRadix + d];
    unsigned long long x = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long y = __shfl_up_sync(kFull, x, o);
      if (lane >= (uint32_t)o) x += y;
    }
    if (lane == 31) s_w[w] = x;
    __syncthreads();
    unsigned long long pre = 0;
    for (uint32_t ww = 0; ww < w; ++ww) pre += s_w[ww];
    offs[p * kRadix + d] = pre + x - c;
    __syncthreads();
  }
}

struct PassArgs {
  const uint32_t* keys_in;
  const uint32_t* vals_in;  // null: values are the element indices
  uint32_t* keys_out;
  uint32_t* vals_out;
  uint64_t n;
  uint32_t shift, width;
  const unsigned long long* digit_base;  // this pass's exclusive digit offsets
  uint64_t* lb;                    // tiles x 256 packed look-back words
  DevStatus* st;
  int epoch;
};

__global__ void __launch_bounds__(kSortThreads) k_sort_pass(PassArgs a) {
  __shared__ uint32_t s_keys[kSortTile];
  __shared__ uint32_t s_vals[kSortTile];
  __shared__ uint32_t s_whist[kSortWarps][kRadix];
  __shared__ uint32_t s_local_start[kRadix];
  __shared__ uint64_t s_gbase[kRadix];
  __shared__ uint32_t s_scan[kSortThreads / 32];

  const uint32_t tile = next_tile(a.st, a.epoch);
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint64_t tile0 = (uint64_t)tile * kSortTile;
  const uint32_t dmask = (1u << a.width) - 1;

  for (uint32_t x = threadIdx.x; x < kSortWarps * kRadix; x += kSortThreads) (&s_whist[0][0])[x] = 0;
  __syncthreads();

  uint32_t key[kSortPer], val[kSortPer], rank[kSortPer];
  const uint64_t wbase = tile0 + (uint64_t)w * (32 * kSortPer);
#pragma unroll
  for (int j = 0; j < kSortPer; ++j) {
    const uint64_t i = wbase + (uint64_t)j * 32 + lane;
    const bool valid = i < a.n;
    key[j] = valid ? a.keys_in[i] : 0u;
    val[j] = valid ? (a.vals_in ? a.vals_in[i] : (uint32_t)i) : 0u;
    const uint32_t d = (key[j] >> a.shift) & dmask;
    const uint32_t peers = __match_any_sync(kFull, valid ? d : 0x10000u + lane);
    const uint32_t leader = __ffs(peers) - 1;
    uint32_t before = 0;
    if (valid && lane == leader) {
      before = s_whist[w][d];
      s_whist[w][d] = before + __popc(peers);
    }
    before = __shfl_sync(kFull, before, leader);
    rank[j] = before + __popc(peers & lanemask_lt());
    __syncwarp();
  }
  __syncthreads();

  // per digit (thread d): offsets of each warp inside the tile, tile count
  const uint32_t d = threadIdx.x;  // kSortThreads == kRadix
  uint32_t cnt = 0;
#pragma unroll
  for (int ww = 0; ww < kSortWarps; ++ww) {
    const uint32_t c = s_whist[ww][d];
    s_whist[ww][d] = cnt;
    cnt += c;
  }
  // exclusive scan of tile counts over digits -> local start in the reorder buffer
  {
    uint32_t x = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(kFull, x, o);
      if (lane >= (uint32_t)o) x += y;
    }
    if (lane == 31) s_scan[w] = x;
    __syncthreads();
    uint32_t wpre = 0;
    for (uint32_t ww = 0; ww < w; ++ww) wpre += s_scan[ww];
    s_local_start[d] = wpre + x - cnt;
  }
  // per-digit look-back over earlier tiles
  uint64_t* words = a.lb + (uint64_t)tile * kRadix;
  if (tile == 0) {
    st_relaxed_u64(&words[d], lb_pack(a.epoch, 2, cnt));
  } else {
    st_relaxed_u64(&words[d], lb_pack(a.epoch, 1, cnt));
  }
  __syncthreads();
  uint64_t prev_cnt = 0;
  if (tile > 0) {
    int64_t j = (int64_t)tile - 1;
    uint32_t spins = 0, ns = 20;
    while (j >= 0) {
      const uint64_t wv = ld_relaxed_u64(&a.lb[(uint64_t)j * kRadix + d]);
      const uint32_t f = ((uint32_t)(wv >> 58) == (uint32_t)a.epoch) ? (uint32_t)((wv >> 56) & 3) : 0u;
      if (f == 0) {
        if (++spins > kSpinCap) {
          raise_err(a.st, kErrTimeout);
          break;
        }
        __nanosleep(ns);
        if (ns < 1000) ns += ns;
        continue;
      }
      prev_cnt += wv & kLbValMask;
      if (f == 2) break;
      --j;
    }
    st_relaxed_u64(&words[d], lb_pack(a.epoch, 2, prev_cnt + cnt));
  }
  s_gbase[d] = a.digit_base[d] + prev_cnt;
  __syncthreads();

  // reorder into shared memory by digit
#pragma unroll
  for (int j = 0; j < kSortPer; ++j) {
    const uint64_t i = wbase + (uint64_t)j * 32 + lane;
    if (i < a.n) {
      const uint32_t dd = (key[j] >> a.shift) & dmask;
      const uint32_t p = s_local_start[dd] + s_whist[w][dd] + rank[j];
      s_keys[p] = key[j];
      s_vals[p] = val[j];
    }
  }
  __syncthreads();
  const uint32_t tile_n = (uint32_t)(a.n - tile0 < (uint64_t)kSortTile ? a.n - tile0 : kSortTile);
  for (uint32_t p = threadIdx.x; p < tile_n; p += kSortThreads) {
    const uint32_t k = s_keys[p];
    const uint32_t dd = (k >> a.shift) & dmask;
    const uint64_t dst = s_gbase[dd] + (p - s_local_start[dd]);
    if (dst < a.n) {  // always true unless a bounded wait gave up (reported as a timeout)
      a.keys_out[dst] = k;
      a.vals_out[dst] = s_vals[p];
    }
  }
}

__global__ void k_adjacent(const uint32_t* __restrict__ sk, const uint32_t* __restrict__ sv, uint64_t n,
                           uint32_t* __restrict__ prev, uint32_t* __restrict__ next) {
  const uint64_t q = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= n) return;
  const uint32_t k = sk[q], v = sv[q];
  prev[v] = (q > 0 && sk[q - 1] == k) ? sv[q - 1] : kNone;
  next[v] = (q + 1 < n && sk[q + 1] == k) ? sv[q + 1] : kNone;
}

uint32_t key_bits(uint64_t D) {
  uint32_t b = 1;
  while (b < 32 && (1ULL << b) < D) ++b;
  return b;
}

struct SortLayout {
  DevStatus* st;
  unsigned long long* hist;
  unsigned long long* offs;
  uint64_t* lb;
  uint32_t *k0, *v0, *k1, *v1;
  size_t zero_bytes;
  size_t total;
};

SortLayout sort_layout(void* ws, uint64_t n) {
  SortLayout L;
  Carver cv(ws);
  const uint64_t nn = n ? n : 1;
  L.st = cv.take<DevStatus>(1);
  L.hist = cv.take<unsigned long long>(4 * kRadix);
  L.offs = cv.take<unsigned long long>(4 * kRadix);
  L.lb = cv.take<uint64_t>((uint64_t)(ceil_div_u32(n, kSortTile) + 1) * kRadix);
  L.zero_bytes = cv.off;
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

extern "C" size_t ptc_reuse_indices_workspace_bytes(uint64_t n, uint64_t n_distinct) {
  (void)n_distinct;
  return sort_layout(nullptr, n).total;
}

extern "C" ptc_status ptc_reuse_indices(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out,
                                        uint32_t* next_out, void* ws, size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (n == 0) return PTC_OK;
  if (!ids || !prev_out || !next_out || n_distinct == 0 || n_distinct > n) return PTC_ERR_INVALID_ARG;
  if (!ws_ok(ws, ws_bytes, sort_layout(nullptr, n).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const SortLayout L = sort_layout(ws, n);
  if (begin_call(ws, L.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  const uint32_t bits = key_bits(n_distinct);
  const uint32_t passes = (bits + 7) / 8;
  PTC_LAUNCH("k_sort_hist", s, k_sort_hist<<<1216, 256, 0, s>>>(ids, n, n_distinct, passes, bits, L.hist, L.st));
  PTC_LAUNCH("k_sort_offsets", s, k_sort_offsets<<<1, kRadix, 0, s>>>(L.hist, passes, L.offs));
  const uint32_t tiles = ceil_div_u32(n, kSortTile);
  const uint32_t* kin = ids;
  const uint32_t* vin = nullptr;
  uint32_t *kout = L.k0, *vout = L.v0;
  for (uint32_t p = 0; p < passes; ++p) {
    PassArgs a;
    a.keys_in = kin;
    a.vals_in = vin;
    a.keys_out = kout;
    a.vals_out = vout;
    a.n = n;
    a.shift = 8 * p;
    a.width = bits - 8 * p < 8 ? bits - 8 * p : 8;
    a.digit_base = L.offs + p * kRadix;
    a.lb = L.lb;
    a.st = L.st;
    a.epoch = 1 + (int)p;
    PTC_LAUNCH("k_sort_pass", s, k_sort_pass<<<tiles, kSortThreads, 0, s>>>(a));
    kin = kout;
    vin = vout;
    kout = (kout == L.k0) ? L.k1 : L.k0;
    vout = (vout == L.v0) ? L.v1 : L.v0;
  }
  PTC_LAUNCH("k_adjacent", s, k_adjacent<<<ceil_div_u32(n, 256), 256, 0, s>>>(kin, vin, n, prev_out, next_out));
  DevStatus h;
  return end_call(L.st, s, &h);
}
