// Stage a2: dense block ids in first-occurrence order (each distinct prefix
// key is one cache object), and the exact check of those ids against tokens.
//
// ptc_assign_ids
//   k_ids_insert   open-addressing table, 16-byte slots claimed with one
//                  128-bit CAS: 96 key bits + the smallest access index seen
//                  (lowered with a 32-bit atomicMin); linear probing.
//   k_ids_rank     access i is a first occurrence iff its slot's index == i;
//                  an exclusive scan of those flags (decoupled look-back)
//                  numbers the keys in access order; first occurrences
//                  publish their rank into the slot's id word.
//   k_ids_gather   ids[i] = id word of i's slot.
// ptc_verify_ids
//   k_verify_first first access of every id (atomicMin)
//   k_verify       compares every access's B tokens and parent id with those
//                  of the first access of its id.
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kInsThreads = 256;
constexpr int kRankThreads = 512;
constexpr int kRankPer = 8;
constexpr int kRankTile = kRankThreads * kRankPer;
constexpr int kEpochRank = 1;

__device__ __forceinline__ ulonglong2 cas128(ulonglong2* addr, ulonglong2 cmp, ulonglong2 val) {
  ulonglong2 old;
  asm volatile(
      "{\n\t.reg .b128 c, v, d;\n\t"
      "mov.b128 c, {%2, %3};\n\t"
      "mov.b128 v, {%4, %5};\n\t"
      "atom.global.cas.b128 d, [%6], c, v;\n\t"
      "mov.b128 {%0, %1}, d;\n\t}"
      : "=l"(old.x), "=l"(old.y)
      : "l"(cmp.x), "l"(cmp.y), "l"(val.x), "l"(val.y), "l"(addr)
      : "memory");
  return old;
}

__device__ __forceinline__ uint64_t home_slot(uint64_t h0, uint64_t h1, uint32_t log2m) {
  uint64_t z = (h0 ^ (h1 * 0x9E3779B97F4A7C15ULL)) * 0xD6E8FEB86659FD93ULL;
  z ^= z >> 32;
  z *= 0xD6E8FEB86659FD93ULL;
  return log2m ? z >> (64 - log2m) : 0;
}

__global__ void __launch_bounds__(kInsThreads) k_ids_insert(const ulonglong2* __restrict__ keys, uint64_t n,
                                                            ulonglong2* table, uint32_t log2m, uint64_t probe_cap,
                                                            uint32_t* __restrict__ slot_of, DevStatus* st) {
  const uint64_t i = (uint64_t)blockIdx.x * kInsThreads + threadIdx.x;
  if (i >= n) return;
  const ulonglong2 k = keys[i];
  if (k.x >= kP61 || k.y >= kP61) {
    raise_err(st, kErrInvalid);
    slot_of[i] = 0;
    return;
  }
  // 96 key bits: all of h0 (61) + 35 bits of h1.  Word 0 is never all-ones
  // because h0 < 2^61 - 1, so all-ones marks an empty slot.
  const uint64_t w0 = k.x | ((k.y & 7ULL) << 61);
  const uint32_t w1lo = (uint32_t)(k.y >> 3);
  const ulonglong2 mine = make_ulonglong2(w0, (uint64_t)w1lo | ((uint64_t)(uint32_t)i << 32));
  const ulonglong2 empty = make_ulonglong2(~0ULL, ~0ULL);
  const uint64_t mask = (1ULL << log2m) - 1;
  uint64_t pos = home_slot(k.x, k.y, log2m);
  for (uint64_t probe = 0; probe <= mask && probe < probe_cap; ++probe) {
    const ulonglong2 old = cas128(&table[pos], empty, mine);
    if (old.x == ~0ULL && old.y == ~0ULL) {
      slot_of[i] = (uint32_t)pos;
      return;
    }
    if (old.x == w0 && (uint32_t)old.y == w1lo) {
      if ((uint32_t)(old.y >> 32) > (uint32_t)i) atomicMin(reinterpret_cast<uint32_t*>(&table[pos]) + 3, (uint32_t)i);
      slot_of[i] = (uint32_t)pos;
      return;
    }
    pos = (pos + 1) & mask;
  }
  raise_err(st, kErrTableFull);
  slot_of[i] = 0;
}

__device__ __forceinline__ uint64_t cta_exclusive_sum512(uint64_t v, uint64_t* total) {
  __shared__ uint64_t s_w[kRankThreads / 32];
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint64_t x = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    uint64_t y = __shfl_up_sync(kFull, x, d);
    if (lane >= (uint32_t)d) x += y;
  }
  if (lane == 31) s_w[w] = x;
  __syncthreads();
  if (w == 0) {
    uint64_t t = lane < kRankThreads / 32 ? s_w[lane] : 0;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      uint64_t y = __shfl_up_sync(kFull, t, d);
      if (lane >= (uint32_t)d) t += y;
    }
    if (lane < kRankThreads / 32) s_w[lane] = t;
  }
  __syncthreads();
  *total = s_w[kRankThreads / 32 - 1];
  return (w ? s_w[w - 1] : 0) + x - v;
}

__global__ void __launch_bounds__(kRankThreads) k_ids_rank(const ulonglong2* __restrict__ table,
                                                           const uint32_t* __restrict__ slot_of, uint64_t n,
                                                           uint32_t* __restrict__ slot_id, uint64_t* lb,
                                                           DevStatus* st) {
  const uint32_t tile = next_tile(st, kEpochRank);
  const uint64_t i0 = (uint64_t)tile * kRankTile + (uint64_t)threadIdx.x * kRankPer;
  uint32_t slots[kRankPer];
  uint32_t flags = 0, cnt = 0;
#pragma unroll
  for (int j = 0; j < kRankPer; ++j) {
    const uint64_t i = i0 + j;
    slots[j] = 0;
    if (i < n) {
      slots[j] = slot_of[i];
      const uint32_t first = reinterpret_cast<const uint32_t*>(&table[slots[j]])[3];
      if (first == (uint32_t)i) {
        flags |= 1u << j;
        ++cnt;
      }
    }
  }
  uint64_t total;
  const uint64_t excl = cta_exclusive_sum512(cnt, &total);
  uint64_t rank = lookback_sum_cta(lb, tile, total, kEpochRank, st) + excl;
#pragma unroll
  for (int j = 0; j < kRankPer; ++j) {
    if (flags & (1u << j)) slot_id[slots[j]] = (uint32_t)rank++;
    if (i0 + j + 1 == n) {
      st->value[0] = rank;
      if (rank >= (uint64_t)kNone) raise_err(st, kErrOverflow);
    }
  }
}

__global__ void k_ids_gather(const uint32_t* __restrict__ slot_of, const uint32_t* __restrict__ slot_id, uint64_t n,
                             uint32_t* __restrict__ ids) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) ids[i] = slot_id[slot_of[i]];
}

// Slots for n keys at most: the full table holds 1.5 n; the first attempt
// holds n / 3 (real traces repeat most blocks, so it is rarely more than 40%
// full and, at this size, stays in L2).  If a probe sequence of the first
// attempt runs past kSmallProbeCap slots, the call redoes the stage with the
// full table.
constexpr uint64_t kSmallProbeCap = 4096;
uint32_t table_log2(uint64_t want) {
  uint32_t l = 10;
  while ((1ULL << l) < want) ++l;
  return l;
}
uint32_t full_table_log2(uint64_t n) { return table_log2(n + n / 2 + 64); }
uint32_t small_table_log2(uint64_t n) { return table_log2(n / 3 + 64); }

struct IdsLayout {
  DevStatus* st;
  uint64_t* lb;
  ulonglong2* table;
  uint32_t* slot_id;
  uint32_t* slot_of;
  size_t zero_bytes;
  size_t total;
  uint32_t log2m;
};

IdsLayout ids_layout(void* ws, uint64_t n) {
  IdsLayout L;
  Carver cv(ws);
  L.log2m = full_table_log2(n);
  const uint64_t m = 1ULL << L.log2m;
  L.st = cv.take<DevStatus>(1);
  L.lb = cv.take<uint64_t>(ceil_div_u32(n, kRankTile) + 1);
  L.zero_bytes = cv.off;
  L.table = cv.take<ulonglong2>(m);
  L.slot_id = cv.take<uint32_t>(m);
  L.slot_of = cv.take<uint32_t>(n ? n : 1);
  L.total = cv.bytes();
  return L;
}

// ---------------------------------------------------------------- verify
__global__ void k_verify_first(const uint32_t* __restrict__ ids, uint64_t n, uint64_t D, uint32_t* first,
                               DevStatus* st) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint32_t id = ids[i];
  if (id >= D) {
    raise_err(st, kErrInvalid);
    return;
  }
  atomicMin(&first[id], (uint32_t)i);
}

__device__ __forceinline__ uint32_t request_of(const uint64_t* __restrict__ blk_off, uint32_t R, uint64_t b) {
  uint32_t lo = 0, hi = R - 1;
  while (lo < hi) {
    const uint32_t mid = (lo + hi + 1) >> 1;
    if (__ldg(&blk_off[mid]) <= b)
      lo = mid;
    else
      hi = mid - 1;
  }
  return lo;
}

__global__ void k_verify(const uint32_t* __restrict__ tokens, uint64_t n_tok, const uint64_t* __restrict__ tok_off,
                         const uint64_t* __restrict__ blk_off, uint32_t R, uint32_t B,
                         const uint32_t* __restrict__ ids, uint64_t n, uint64_t D,
                         const uint32_t* __restrict__ first, DevStatus* st) {
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint32_t id = ids[i];
  if (id >= D) return;  // reported by k_verify_first
  const uint32_t f = first[id];
  if (f == kNone) {
    raise_err(st, kErrInvalid);
    return;
  }
  if (f == (uint32_t)i) return;
  const uint32_t ri = request_of(blk_off, R, i), rf = request_of(blk_off, R, f);
  const uint64_t ki = i - blk_off[ri], kf = f - blk_off[rf];
  // the block offsets must describe these token offsets (no read past a request)
  if (ki >= (tok_off[ri + 1] - tok_off[ri]) / B || kf >= (tok_off[rf + 1] - tok_off[rf]) / B ||
      tok_off[ri + 1] < tok_off[ri] || tok_off[rf + 1] < tok_off[rf] || tok_off[ri + 1] > n_tok ||
      tok_off[rf + 1] > n_tok) {
    raise_err(st, kErrInvalid);
    return;
  }
  const uint32_t pi = ki ? ids[i - 1] : kNone, pf = kf ? ids[f - 1] : kNone;
  bool same = pi == pf;
  const uint32_t* ti = tokens + tok_off[ri] + (uint64_t)B * ki;
  const uint32_t* tf = tokens + tok_off[rf] + (uint64_t)B * kf;
  for (uint32_t t = 0; same && t < B; ++t) same = ti[t] == tf[t];
  if (!same) raise_err(st, kErrCollision);
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_assign_ids_workspace_bytes(uint64_t n) { return ids_layout(nullptr, n).total; }

extern "C" ptc_status ptc_assign_ids(const ptc_u128* keys, uint64_t n, uint32_t* ids_out, uint64_t* n_distinct_host_out,
                                     void* ws, size_t ws_bytes, void* stream) {
  if (n_distinct_host_out == nullptr) return PTC_ERR_INVALID_ARG;
  *n_distinct_host_out = 0;
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (n > 0 && (keys == nullptr || ids_out == nullptr)) return PTC_ERR_INVALID_ARG;
  if (!ws_ok(ws, ws_bytes, ids_layout(nullptr, n).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const IdsLayout L = ids_layout(ws, n);
  if (begin_call(ws, L.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  auto run = [&](uint32_t log2m, uint64_t probe_cap) -> bool {
    if (cudaMemsetAsync(L.table, 0xFF, sizeof(ulonglong2) << log2m, s) != cudaSuccess) return false;
    const ulonglong2* k = reinterpret_cast<const ulonglong2*>(keys);
    PTC_LAUNCH("k_ids_insert", s, k_ids_insert<<<ceil_div_u32(n, kInsThreads), kInsThreads, 0, s>>>(
                                      k, n, L.table, log2m, probe_cap, L.slot_of, L.st));
    PTC_LAUNCH("k_ids_rank", s, k_ids_rank<<<ceil_div_u32(n, kRankTile), kRankThreads, 0, s>>>(
                                    L.table, L.slot_of, n, L.slot_id, L.lb, L.st));
    PTC_LAUNCH("k_ids_gather", s, k_ids_gather<<<ceil_div_u32(n, 256), 256, 0, s>>>(L.slot_of, L.slot_id, n, ids_out));
    return true;
  };
  if (n > 0) {
    const uint32_t small = small_table_log2(n);
    if (!run(small, small < L.log2m ? kSmallProbeCap : ~0ULL)) return PTC_ERR_CUDA;
    if (small < L.log2m) {
      DevStatus h1;
      const ptc_status rc1 = end_call(L.st, s, &h1);
      if (rc1 == PTC_OK) {
        *n_distinct_host_out = h1.value[0];
        return PTC_OK;
      }
      if (!(h1.err & kErrTableFull)) return rc1;
      // the small table overflowed: redo with the full one
      if (begin_call(ws, L.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
      if (!run(L.log2m, ~0ULL)) return PTC_ERR_CUDA;
    }
  }
  DevStatus h;
  const ptc_status rc = end_call(L.st, s, &h);
  *n_distinct_host_out = n ? h.value[0] : 0;
  return rc;
}

extern "C" size_t ptc_verify_ids_workspace_bytes(uint64_t n, uint64_t n_distinct) {
  (void)n;
  Carver cv(nullptr);
  cv.take<DevStatus>(1);
  cv.take<uint32_t>(n_distinct ? n_distinct : 1);
  return cv.bytes();
}

extern "C" ptc_status ptc_verify_ids(const uint32_t* tokens, uint64_t n_tok, const uint64_t* req_tok_off,
                                     const uint64_t* req_blk_off,
                                     uint32_t n_req, uint32_t block_size, const uint32_t* ids, uint64_t n,
                                     uint64_t n_distinct, void* ws, size_t ws_bytes, void* stream) {
  if (block_size < 1 || block_size > PTC_MAX_BLOCK_SIZE) return PTC_ERR_INVALID_ARG;
  if (n >= (uint64_t)kNone || n_distinct > n) return PTC_ERR_INVALID_ARG;
  if (n == 0) return PTC_OK;
  if (!tokens || !req_tok_off || !req_blk_off || !ids || n_req == 0) return PTC_ERR_INVALID_ARG;
  if (!ws_ok(ws, ws_bytes, ptc_verify_ids_workspace_bytes(n, n_distinct))) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  Carver cv(ws);
  DevStatus* st = cv.take<DevStatus>(1);
  uint32_t* first = cv.take<uint32_t>(n_distinct ? n_distinct : 1);
  if (begin_call(ws, kStatusBytes, s) != PTC_OK) return PTC_ERR_CUDA;
  if (cudaMemsetAsync(first, 0xFF, sizeof(uint32_t) * (n_distinct ? n_distinct : 1), s) != cudaSuccess)
    return PTC_ERR_CUDA;
  PTC_LAUNCH("k_verify_first", s, k_verify_first<<<ceil_div_u32(n, 256), 256, 0, s>>>(ids, n, n_distinct, first, st));
  PTC_LAUNCH("k_verify", s, k_verify<<<ceil_div_u32(n, 256), 256, 0, s>>>(tokens, n_tok, req_tok_off, req_blk_off, n_req, block_size, ids, n,
                                               n_distinct, first, st));
  DevStatus h;
  return end_call(st, s, &h);
}
