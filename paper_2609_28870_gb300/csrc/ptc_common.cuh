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
};

constexpr int kMaxEpochs = 64;

struct DevStatus {
  uint32_t err;
  uint32_t pad0;
  uint64_t value[8];              // per-call results (N, D, max depth ...)
  uint32_t tile_ctr[kMaxEpochs];  // dynamic tile counter of each launch
};
static_assert(sizeof(DevStatus) <= 512, "status block");
constexpr size_t kStatusBytes = 512;

// Bounded spin: about 2^20 polls with capped exponential back-off (~1 s).
constexpr uint32_t kSpinCap = 1u << 20;

__device__ __forceinline__ void raise_err(DevStatus* st, uint32_t f) { atomicOr(&st->err, f); }

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
// Packed look-back for sums below 2^56: word = epoch(6) | flag(2) | value(56).
// flag 1 = aggregate, 2 = inclusive prefix.  Called by all 32 lanes of ONE
// warp; returns the exclusive prefix of `tile` (0 if the wait gave up, with
// kErrTimeout raised).
// ---------------------------------------------------------------------------
constexpr uint64_t kLbValMask = (1ULL << 56) - 1;
__device__ __forceinline__ uint64_t lb_pack(uint32_t epoch, uint32_t flag, uint64_t v) {
  return ((uint64_t)epoch << 58) | ((uint64_t)flag << 56) | (v & kLbValMask);
}

__device__ inline uint64_t lookback_sum(uint64_t* words, uint32_t tile, uint64_t agg, uint32_t epoch,
                                        DevStatus* st) {
  const uint32_t lane = threadIdx.x & 31;
  if (tile == 0) {
    if (lane == 0) st_relaxed_u64(&words[0], lb_pack(epoch, 2, agg));
    return 0;
  }
  if (lane == 0) st_relaxed_u64(&words[tile], lb_pack(epoch, 1, agg));
  uint64_t excl = 0;
  int64_t base = (int64_t)tile - 1;
  uint32_t spins = 0, ns = 20;
  for (;;) {
    int64_t idx = base - (int64_t)lane;
    uint32_t f = 2;
    uint64_t v = 0;
    if (idx >= 0) {
      uint64_t w = ld_relaxed_u64(&words[idx]);
      f = ((uint32_t)(w >> 58) == epoch) ? (uint32_t)((w >> 56) & 3) : 0u;
      v = w & kLbValMask;
    }
    // only the tiles after the nearest published prefix must be ready
    const uint32_t incl = __ballot_sync(kFull, f == 2);
    const uint32_t first = incl ? (uint32_t)(__ffs(incl) - 1) : 31u;
    const uint32_t upto = first == 31u ? kFull : ((2u << first) - 1u);
    if (__ballot_sync(kFull, f == 0) & upto) {
      if (++spins > kSpinCap) {
        if (lane == 0) raise_err(st, kErrTimeout);
        return 0;
      }
      __nanosleep(ns);
      if (ns < 1000) ns += ns;
      continue;
    }
    if (incl) {
      if (lane > first) v = 0;
      excl += warp_sum_u64(v);
      break;
    }
    excl += warp_sum_u64(v);
    base -= 32;
  }
  if (lane == 0) st_relaxed_u64(&words[tile], lb_pack(epoch, 2, excl + agg));
  return excl;
}

// ---------------------------------------------------------------------------
// Generic look-back for a payload T with an associative operator `op` and a
// two-sided identity.  Status word per tile: epoch << 2 | flag.  Payloads go
// to separate aggregate / inclusive arrays, published before the flag with a
// fence.  Called by ONE thread.
// ---------------------------------------------------------------------------
template <class T>
struct LbArrays {
  uint32_t* status;
  T* agg;
  T* incl;
};

template <class T>
__device__ __forceinline__ void lb_store(T* dst, const T& v) {
  volatile uint64_t* d = reinterpret_cast<volatile uint64_t*>(dst);
  const uint64_t* s = reinterpret_cast<const uint64_t*>(&v);
#pragma unroll
  for (int i = 0; i < (int)(sizeof(T) / 8); ++i) d[i] = s[i];
}
template <class T>
__device__ __forceinline__ T lb_load(const T* src) {
  T v;
  const volatile uint64_t* s = reinterpret_cast<const volatile uint64_t*>(src);
  uint64_t* d = reinterpret_cast<uint64_t*>(&v);
#pragma unroll
  for (int i = 0; i < (int)(sizeof(T) / 8); ++i) d[i] = s[i];
  return v;
}

template <class T, class Op>
__device__ inline T lookback_generic(LbArrays<T> a, uint32_t tile, const T& agg, const T& identity, Op op,
                                     uint32_t epoch, DevStatus* st) {
  static_assert(sizeof(T) % 8 == 0, "payload must be a multiple of 8 bytes");
  if (tile == 0) {
    lb_store(&a.incl[0], agg);
    __threadfence();
    st_relaxed_u32(&a.status[0], (epoch << 2) | 2u);
    return identity;
  }
  lb_store(&a.agg[tile], agg);
  __threadfence();
  st_relaxed_u32(&a.status[tile], (epoch << 2) | 1u);
  T acc = identity;
  int64_t j = (int64_t)tile - 1;
  uint32_t spins = 0, ns = 20;
  while (j >= 0) {
    uint32_t s = ld_relaxed_u32(&a.status[j]);
    uint32_t f = ((s >> 2) == epoch) ? (s & 3u) : 0u;
    if (f == 0) {
      if (++spins > kSpinCap) {
        raise_err(st, kErrTimeout);
        return identity;
      }
      __nanosleep(ns);
      if (ns < 1000) ns += ns;
      continue;
    }
    __threadfence();
    if (f == 2) {
      acc = op(lb_load(&a.incl[j]), acc);
      break;
    }
    acc = op(lb_load(&a.agg[j]), acc);
    --j;
  }
  T inc = op(acc, agg);
  lb_store(&a.incl[tile], inc);
  __threadfence();
  st_relaxed_u32(&a.status[tile], (epoch << 2) | 2u);
  return acc;
}

// Warp-parallel variant of lookback_generic: called by all 32 lanes of ONE
// warp; each round inspects 32 predecessors at once and folds them in order
// (a higher lane holds an earlier tile, so it is the left operand).  Returns
// the exclusive prefix in every lane.
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

template <class T, class Op>
__device__ inline T lookback_warp(LbArrays<T> a, uint32_t tile, const T& agg, const T& identity, Op op,
                                  uint32_t epoch, DevStatus* st) {
  static_assert(sizeof(T) % 8 == 0, "payload must be a multiple of 8 bytes");
  const uint32_t lane = threadIdx.x & 31;
  if (tile == 0) {
    if (lane == 0) {
      lb_store(&a.incl[0], agg);
      __threadfence();
      st_relaxed_u32(&a.status[0], (epoch << 2) | 2u);
    }
    return identity;
  }
  if (lane == 0) {
    lb_store(&a.agg[tile], agg);
    __threadfence();
    st_relaxed_u32(&a.status[tile], (epoch << 2) | 1u);
  }
  T acc = identity;
  int64_t base = (int64_t)tile - 1;
  uint32_t spins = 0, ns = 20;
  for (;;) {
    const int64_t idx = base - (int64_t)lane;
    uint32_t f = 2;
    if (idx >= 0) {
      const uint32_t s = ld_relaxed_u32(&a.status[idx]);
      f = ((s >> 2) == epoch) ? (s & 3u) : 0u;
    }
    if (__any_sync(kFull, f == 0)) {
      if (++spins > kSpinCap) {
        if (lane == 0) raise_err(st, kErrTimeout);
        return identity;
      }
      __nanosleep(ns);
      if (ns < 1000) ns += ns;
      continue;
    }
    __threadfence();
    const uint32_t incl = __ballot_sync(kFull, f == 2);
    const uint32_t first = incl ? (uint32_t)(__ffs(incl) - 1) : 31u;
    T x = identity;
    if (idx >= 0 && lane <= first) x = (f == 2) ? lb_load(&a.incl[idx]) : lb_load(&a.agg[idx]);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const T y = shfl_down_payload(x, o);
      if (lane + o < 32) x = op(y, x);
    }
    acc = op(shfl_payload(x, 0), acc);
    if (incl) break;
    base -= 32;
  }
  if (lane == 0) {
    const T inc = op(acc, agg);
    lb_store(&a.incl[tile], inc);
    __threadfence();
    st_relaxed_u32(&a.status[tile], (epoch << 2) | 2u);
  }
  return acc;
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
  for (;;) {
    const int64_t idx = base - (int64_t)t;
    uint32_t f = 2;
    uint64_t v = 0;
    if (idx >= 0) {
      const uint64_t wv = ld_relaxed_u64(&words[idx]);
      f = ((uint32_t)(wv >> 58) == epoch) ? (uint32_t)((wv >> 56) & 3) : 0u;
      v = wv & kLbValMask;
    }
    // the nearest published prefix; only the tiles after it must be ready
    if (t == 0) s_first = 0xFFFFFFFFu;
    __syncthreads();
    if (f == 2) atomicMin(&s_first, t);
    __syncthreads();
    const uint32_t first = s_first;
    if (__syncthreads_or(f == 0 && t < first)) {
      if (++spins > kSpinCap) {
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

template <class T, class Op>
__device__ inline T lookback_cta(LbArrays<T> a, uint32_t tile, const T& agg, const T& identity, Op op,
                                 uint32_t epoch, DevStatus* st) {
  static_assert(sizeof(T) % 8 == 0, "payload must be a multiple of 8 bytes");
  __shared__ T s_wres[32];
  __shared__ T s_acc;
  __shared__ uint32_t s_first;
  const uint32_t t = threadIdx.x, lane = t & 31, wid = t >> 5, nw = blockDim.x >> 5;
  if (tile == 0) {
    if (t == 0) {
      lb_store(&a.incl[0], agg);
      __threadfence();
      st_relaxed_u32(&a.status[0], (epoch << 2) | 2u);
    }
    return identity;
  }
  if (t == 0) {
    lb_store(&a.agg[tile], agg);
    __threadfence();
    st_relaxed_u32(&a.status[tile], (epoch << 2) | 1u);
    s_acc = identity;
  }
  int64_t base = (int64_t)tile - 1;
  uint32_t spins = 0, ns = 20;
  for (;;) {
    const int64_t idx = base - (int64_t)t;
    uint32_t f = 2;
    if (idx >= 0) {
      const uint32_t sv = ld_relaxed_u32(&a.status[idx]);
      f = ((sv >> 2) == epoch) ? (sv & 3u) : 0u;
    }
    if (__syncthreads_or(f == 0)) {
      if (++spins > kSpinCap) {
        if (t == 0) {
          raise_err(st, kErrTimeout);
          s_acc = identity;
        }
        break;
      }
      __nanosleep(ns);
      if (ns < 500) ns += ns;
      continue;
    }
    __threadfence();
    if (t == 0) s_first = 0xFFFFFFFFu;
    __syncthreads();
    if (f == 2 && idx >= 0) atomicMin(&s_first, t);
    __syncthreads();
    const uint32_t first = s_first;
    T x = identity;
    if (idx >= 0 && t <= first) x = (f == 2) ? lb_load(&a.incl[idx]) : lb_load(&a.agg[idx]);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const T y = shfl_down_payload(x, o);
      if (lane + o < 32) x = op(y, x);
    }
    if (lane == 0) s_wres[wid] = x;
    __syncthreads();
    if (t == 0) {
      T r = identity;
      for (int k = (int)nw - 1; k >= 0; --k) r = op(r, s_wres[k]);
      s_acc = op(r, s_acc);
    }
    __syncthreads();
    // a window reaching past tile 0 counts as complete (idx < 0 reads as inclusive)
    if (first != 0xFFFFFFFFu || base < (int64_t)blockDim.x) break;
    base -= (int64_t)blockDim.x;
  }
  if (t == 0) {
    const T inc = op(s_acc, agg);
    lb_store(&a.incl[tile], inc);
    __threadfence();
    st_relaxed_u32(&a.status[tile], (epoch << 2) | 2u);
  }
  __syncthreads();
  return s_acc;
}

// ---------------------------------------------------------------------------
// Bulk (TMA) copies global -> shared with mbarrier completion (sm_90+).
// The source and destination must be 16-byte aligned and the size a multiple
// of 16 bytes.  Waits are bounded: on give-up the caller raises kErrTimeout.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_init_fence() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_addr(dst)),
               "l"(src), "r"(bytes), "r"(smem_addr(bar))
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t phase) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(phase)
      : "memory");
  return ok != 0;
}
// Wait for phase `phase` of `bar`; false if the bounded wait gave up.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t phase) {
  for (uint32_t i = 0; i < (1u << 22); ++i)
    if (mbar_try_wait(bar, phase)) return true;
  return false;
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
