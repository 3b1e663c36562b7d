// Shared device/host helpers of the ptc kernels (sm_103a).
//
//  * Device status block: every call's workspace starts with one.  Kernels
//    report malformed input and give-ups of bounded waits by OR-ing flags into
//    it; the C-ABI entry reads it back before returning.  No kernel traps.
//  * Decoupled look-back (Merrill & Garland 2016) for single-pass scans: tiles
//    take dynamic ids from a counter so that every predecessor of a running
//    tile has started, publish their aggregate, then their inclusive prefix.
//    Status words carry a 6-bit epoch (one per launch inside a call), so one
//    zeroing per call serves every launch.  Every wait is bounded.
//  * Arithmetic in GF(p), p = 2^61 - 1.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace ptc {

constexpr uint32_t kNone = 0xFFFFFFFFu;
constexpr uint64_t kP61 = (1ULL << 61) - 1;
constexpr uint32_t kFull = 0xFFFFFFFFu;

// error flags in DevStatus::err
enum : uint32_t {
  kErrTimeout = 1u,
  kErrUnsorted = 2u,
  kErrInvalid = 4u,
  kErrOverflow = 8u,
  kErrCollision = 16u,
  kErrTableFull = 32u,
  kErrBounds = 64u,  // the checked build caught an index outside its array
};

constexpr int kMaxEpochs = 64;

struct DevStatus {
  uint32_t err;
  // 0 normally.  Otherwise a test has asked the look-back waits of this call
  // to see no predecessor as ready (a flag nothing sets) and to give up after
  // this many polls: the bounded-wait path, forced (ptc_test_wait_polls).
  uint32_t wait_test;
  uint64_t value[8];              // per-call results (N, D, max depth ...)
  uint32_t tile_ctr[kMaxEpochs];  // dynamic tile counter of each launch
};
static_assert(sizeof(DevStatus) <= 512, "status block");
constexpr size_t kStatusBytes = 512;

// Bounded spin: about 2^20 polls with capped exponential back-off (~1 s).
constexpr uint32_t kSpinCap = 1u << 20;

__device__ __forceinline__ void raise_err(DevStatus* st, uint32_t f) { atomicOr(&st->err, f); }

// The checked build (compiled with -DPTC_CHECKED; paper_2609_28870_gb300
// build(checked=True)): an index that comes from data another stage or the
// caller wrote is checked before it is used; a failed check raises
// kErrBounds in the call's status word (PTC_ERR_BOUNDS) and the access is
// skipped, never trapped.  In the normal build the check compiles away.
__device__ __forceinline__ bool in_bounds(const DevStatus* st, uint64_t i, uint64_t bound) {
#ifdef PTC_CHECKED
  if (i < bound) return true;
  atomicOr(const_cast<uint32_t*>(&st->err), kErrBounds);
  return false;
#else
  (void)st;
  (void)i;
  (void)bound;
  return true;
#endif
}

// Programmatic dependent launch.  Kernels are launched so that the next one
// on the stream is set up while the previous one is still running; every
// kernel calls this first, before it touches global memory: it waits until
// the previous kernel has completed and its writes are visible (a no-op for a
// launch without the attribute).  No kernel signals early completion
// (griddepcontrol.launch_dependents): measured over the whole pipeline,
// letting the next grid's CTAs in while the last wave of many short CTAs
// still runs cost more than it saved.  Each kernel waits for its predecessor,
// so the chain stays ordered end to end.
__device__ __forceinline__ void grid_dep_sync() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// The request of access i: the largest r in [lo, hi] with off[r] <= i
// (request block offsets, non-decreasing).
__device__ __forceinline__ uint32_t req_search(const uint64_t* __restrict__ off, uint32_t lo, uint32_t hi,
                                               uint64_t i) {
  while (lo < hi) {
    const uint32_t mid = lo + (hi - lo + 1) / 2;
    if (__ldg(off + mid) <= i) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

__device__ __forceinline__ uint32_t next_tile(DevStatus* st, int epoch) {
  __shared__ uint32_t s_tile;
  if (threadIdx.x == 0) s_tile = atomicAdd(&st->tile_ctr[epoch], 1u);
  __syncthreads();
  return s_tile;
}

__device__ __forceinline__ uint64_t ld_relaxed_u64(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_relaxed_u64(uint64_t* p, uint64_t v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_relaxed_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_relaxed_u32(uint32_t* p, uint32_t v) {
  asm volatile("st.relaxed.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint64_t ld_cg_u64(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ uint64_t warp_sum_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// ---------------------------------------------------------------------------
// Exclusive prefix of the per-tile counts cnt[0, T) into pre[0, T), with
// pre[T] = the total, which it also returns.  Run by every thread of ONE CTA
// (the last of a grid to finish, after last-CTA fencing; blockDim.x a
// multiple of 32).  Warp w owns a contiguous range of rows of 32 tiles and
// reads kTpRows rows per round with coalesced loads that are all in flight
// together, so the scan costs a few memory round trips rather than one per
// tile and thread.
// ---------------------------------------------------------------------------
constexpr int kTpRows = 8;
__device__ inline uint32_t cta_tiles_prefix(const uint32_t* cnt, uint32_t* pre, uint32_t T) {
  __shared__ uint32_t s_tp[32];
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const uint32_t rows = (T + 31) / 32, rpw = (rows + nw - 1) / nw;
  const uint32_t r0 = w * rpw < rows ? w * rpw : rows, r1 = r0 + rpw < rows ? r0 + rpw : rows;
  uint32_t sum = 0;
  for (uint32_t r = r0; r < r1; r += kTpRows) {
    uint32_t v[kTpRows];
#pragma unroll
    for (int u = 0; u < kTpRows; ++u) {
      const uint32_t t = (r + u) * 32 + lane;
      v[u] = (r + u < r1 && t < T) ? __ldcg(&cnt[t]) : 0u;
    }
#pragma unroll
    for (int u = 0; u < kTpRows; ++u) sum += v[u];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(kFull, sum, o);
  if (lane == 0) s_tp[w] = sum;
  __syncthreads();
  uint32_t base = 0, total = 0;
  for (uint32_t i = 0; i < nw; ++i) {
    const uint32_t x = s_tp[i];
    if (i < w) base += x;
    total += x;
  }
  for (uint32_t r = r0; r < r1; r += kTpRows) {
    uint32_t v[kTpRows];
#pragma unroll
    for (int u = 0; u < kTpRows; ++u) {
      const uint32_t t = (r + u) * 32 + lane;
      v[u] = (r + u < r1 && t < T) ? __ldcg(&cnt[t]) : 0u;
    }
#pragma unroll
    for (int u = 0; u < kTpRows; ++u) {
      uint32_t incl = v[u];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, incl, o);
        if (lane >= (uint32_t)o) incl += y;
      }
      const uint32_t t = (r + u) * 32 + lane;
      if (r + u < r1 && t < T) pre[t] = base + incl - v[u];
      base += __shfl_sync(kFull, incl, 31);
    }
  }
  if (threadIdx.x == 0) pre[T] = total;
  return total;
}

// ---------------------------------------------------------------------------
// Packed look-back words for sums below 2^56: epoch(6) | flag(2) | value(56);
// flag 1 = aggregate, 2 = inclusive prefix.
// ---------------------------------------------------------------------------
constexpr uint64_t kLbValMask = (1ULL << 56) - 1;
__device__ __forceinline__ uint64_t lb_pack(uint32_t epoch, uint32_t flag, uint64_t v) {
  return ((uint64_t)epoch << 58) | ((uint64_t)flag << 56) | (v & kLbValMask);
}

// Shuffles of a payload of 8-byte words across a warp.
template <class T>
__device__ __forceinline__ T shfl_down_payload(const T& v, int o) {
  T r;
  const uint64_t* s = reinterpret_cast<const uint64_t*>(&v);
  uint64_t* d = reinterpret_cast<uint64_t*>(&r);
#pragma unroll
  for (int i = 0; i < (int)(sizeof(T) / 8); ++i) d[i] = __shfl_down_sync(kFull, s[i], o);
  return r;
}
template <class T>
__device__ __forceinline__ T shfl_payload(const T& v, int src) {
  T r;
  const uint64_t* s = reinterpret_cast<const uint64_t*>(&v);
  uint64_t* d = reinterpret_cast<uint64_t*>(&r);
#pragma unroll
  for (int i = 0; i < (int)(sizeof(T) / 8); ++i) d[i] = __shfl_sync(kFull, s[i], src);
  return r;
}

// ---------------------------------------------------------------------------
// CTA-wide look-back: every thread of the CTA calls it, and each round
// inspects blockDim.x predecessors at once, so the inclusive-prefix frontier
// advances a whole CTA width per round trip.  blockDim.x must be a multiple of
// 32 (at most 1024).  Returns the exclusive prefix in every thread.
// ---------------------------------------------------------------------------
__device__ inline uint64_t lookback_sum_cta(uint64_t* words, uint32_t tile, uint64_t agg, uint32_t epoch,
                                            DevStatus* st) {
  __shared__ uint64_t s_part[32];
  __shared__ uint32_t s_first;
  __shared__ uint64_t s_excl;
  const uint32_t t = threadIdx.x, lane = t & 31, wid = t >> 5, nw = blockDim.x >> 5;
  if (tile == 0) {
    if (t == 0) st_relaxed_u64(&words[0], lb_pack(epoch, 2, agg));
    return 0;
  }
  if (t == 0) {
    st_relaxed_u64(&words[tile], lb_pack(epoch, 1, agg));
    s_excl = 0;
  }
  int64_t base = (int64_t)tile - 1;
  uint32_t spins = 0, ns = 20;
  const uint32_t wait_test = ld_relaxed_u32(&st->wait_test);
  const uint32_t cap = wait_test ? wait_test : kSpinCap;
  for (;;) {
    const int64_t idx = base - (int64_t)t;
    uint32_t f = 2;
    uint64_t v = 0;
    if (idx >= 0) {
      const uint64_t wv = ld_relaxed_u64(&words[idx]);
      f = ((uint32_t)(wv >> 58) == epoch) ? (uint32_t)((wv >> 56) & 3) : 0u;
      v = wv & kLbValMask;
      if (wait_test) f = 0;
    }
    // the nearest published prefix; only the tiles after it must be ready
    if (t == 0) s_first = 0xFFFFFFFFu;
    __syncthreads();
    if (f == 2) atomicMin(&s_first, t);
    __syncthreads();
    const uint32_t first = s_first;
    if (__syncthreads_or(f == 0 && t < first)) {
      if (++spins > cap) {
        if (t == 0) {
          raise_err(st, kErrTimeout);
          s_excl = 0;
        }
        break;
      }
      __nanosleep(ns);
      if (ns < 500) ns += ns;
      continue;
    }
    if (t > first) v = 0;
    v = warp_sum_u64(v);
    if (lane == 0) s_part[wid] = v;
    __syncthreads();
    if (t == 0) {
      uint64_t sum = 0;
      for (uint32_t k = 0; k < nw; ++k) sum += s_part[k];
      s_excl += sum;
    }
    __syncthreads();
    if (first != 0xFFFFFFFFu) break;
    base -= (int64_t)blockDim.x;
  }
  if (t == 0) st_relaxed_u64(&words[tile], lb_pack(epoch, 2, s_excl + agg));
  __syncthreads();
  return s_excl;
}

// ---------------------------------------------------------------------------
// GF(2^61 - 1)
// ---------------------------------------------------------------------------
__host__ __device__ __forceinline__ uint64_t p61_fold(uint64_t x) {  // x < 2^64 -> [0, p)
  x = (x & kP61) + (x >> 61);
  x = (x & kP61) + (x >> 61);
  return x >= kP61 ? x - kP61 : x;
}
__host__ __device__ __forceinline__ uint64_t p61_add(uint64_t a, uint64_t b) {  // a, b < p
  uint64_t r = a + b;
  return r >= kP61 ? r - kP61 : r;
}
__host__ __device__ __forceinline__ uint64_t p61_mul(uint64_t a, uint64_t b) {  // a, b < p
#ifdef __CUDA_ARCH__
  uint64_t lo = a * b, hi = __umul64hi(a, b);
#else
  unsigned __int128 t = (unsigned __int128)a * b;
  uint64_t lo = (uint64_t)t, hi = (uint64_t)(t >> 64);
#endif
  // a*b < 2^122, so hi < 2^58 and hi << 3 does not overflow
  uint64_t r = (lo & kP61) + (lo >> 61) + (hi << 3);
  r = (r & kP61) + (r >> 61);
  return r >= kP61 ? r - kP61 : r;
}
__host__ __device__ inline uint64_t p61_pow(uint64_t b, uint64_t e) {
  uint64_t r = 1;
  while (e) {
    if (e & 1) r = p61_mul(r, b);
    b = p61_mul(b, b);
    e >>= 1;
  }
  return r;
}

__host__ __device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t n) {
  uint64_t z = seed + (n + 1) * 0x9E3779B97F4A7C15ULL;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

}  // namespace ptc

// ---------------------------------------------------------------------------
// Host side: workspace carving and status read-back
// ---------------------------------------------------------------------------
#include <cstddef>

namespace ptc {

struct Carver {
  char* base;
  size_t off = 0;
  explicit Carver(void* b) : base((char*)b) {}
  template <class T>
  T* take(size_t count, size_t align = 256) {
    off = (off + align - 1) / align * align;
    T* p = base ? (T*)(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
  size_t bytes() const { return (off + 255) / 256 * 256; }
};

inline uint32_t ceil_div_u32(uint64_t a, uint64_t b) { return (uint32_t)((a + b - 1) / b); }

}  // namespace ptc
