// Stage a2: dense block ids in first-occurrence order (each distinct prefix
// key is one cache object), and the exact check of those ids against tokens.
//
// ptc_assign_ids
//   k_ids_insert   open-addressing table, 16-byte slots: 96 key bits + the
//                  smallest access index seen.  A slot is read first; only an
//                  empty (or half-written) slot is claimed with one 128-bit
//                  CAS, and a stored index above i is lowered with atomicMin.
//                  Linear probing.  Each claim and each lowering toggles bits
//                  of the first-occurrence bitmap over positions, which ends
//                  with exactly the smallest index of every key set.
//   bitmap_ranks   first occurrences before every 32-position word, and D
//   k_ids_gather   ids[i] = rank, among the first occurrences, of i itself
//                  if its bit is set, else of the index stored in i's slot.
// With a prior-request hint (ptc_assign_ids_prior), k_ids_lam finds the
// leading depths of each request that repeat the hinted request, which skip
// the table (k_ids_insert_prior) and take their ids along the hint chain
// (k_ids_follow).
// ptc_verify_ids
//   k_verify_first first access of every id (atomicMin)
//   k_verify       compares every access's B tokens and parent id with those
//                  of the first access of its id.
#include <algorithm>

#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kInsThreads = 256;

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

// The keys are polynomial hashes of their prefixes, spread evenly over
// [0, 2^61 - 1), so their low bits index the table directly.
__device__ __forceinline__ uint64_t home_slot(uint64_t h0, uint64_t h1, uint32_t log2m) {
  return (h0 ^ (h1 >> 17)) & ((1ULL << log2m) - 1);
}

__device__ __forceinline__ ulonglong2 ld_slot(const ulonglong2* p) {
  ulonglong2 v;
  asm volatile("ld.relaxed.gpu.global.v2.u64 {%0, %1}, [%2];" : "=l"(v.x), "=l"(v.y) : "l"(p) : "memory");
  return v;
}

// The number of keys: n, or min(*n_dev, n) when the count is only known on
// the device (the pipeline does not wait for stage a1).
__device__ __forceinline__ uint32_t keys_used(uint32_t n, const uint64_t* n_dev) {
  if (!n_dev) return n;
  const uint64_t v = *n_dev;
  return v < n ? (uint32_t)v : n;
}

// Block 0 reports the number of keys used (value[1]); a count above the
// keys buffer is malformed input.
__device__ __forceinline__ void report_keys_used(uint32_t n_ub, const uint64_t* n_dev, DevStatus* st) {
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    st->value[1] = n_dev ? *n_dev : n_ub;
    if (n_dev && *n_dev > n_ub) raise_err(st, kErrInvalid);
  }
}

constexpr int kInsK = 1;  // keys per thread: their key and slot loads are in flight together

// Settle the key k of access i, whose home slot `pos` was read as `cur`:
// claim an empty (or half-written) slot with one 128-bit CAS, or find the
// key's slot and lower its stored index to i if it is above; linear probing.
// The slot goes to *slot_out.
// The first-occurrence bitmap is kept as the table changes: every index that
// becomes a slot's stored index toggles its bit, and so does every index that
// an atomicMin replaces (the atomicMin's return value names it, to one thread
// only).  An index that is stored and later replaced is toggled twice, the
// final one once, and XOR does not depend on the order in which the toggles
// land, so once all keys are settled the set bits are exactly the smallest
// index of every key.
// 96 key bits: all of h0 (61) + 35 bits of h1.  Word 0 is never all-ones
// because h0 < 2^61 - 1, and word 1 of a filled slot holds an index below
// 2^32 - 1, so an all-ones word marks an empty or half-written slot.
__device__ __forceinline__ void toggle(uint32_t* bits, uint32_t i) { atomicXor(&bits[i >> 5], 1u << (i & 31)); }

__device__ __forceinline__ void settle(ulonglong2* table, uint64_t mask, uint64_t probe_cap, uint32_t i,
                                       ulonglong2 k, uint64_t pos, ulonglong2 cur, uint32_t* __restrict__ slot_out,
                                       uint32_t* bits, DevStatus* st) {
  const uint64_t w0 = k.x | ((k.y & 7ULL) << 61);
  const uint32_t w1lo = (uint32_t)(k.y >> 3);
  const ulonglong2 mine = make_ulonglong2(w0, (uint64_t)w1lo | ((uint64_t)i << 32));
  const ulonglong2 empty = make_ulonglong2(~0ULL, ~0ULL);
  for (uint64_t probe = 0;;) {
    if (cur.x == ~0ULL || cur.y == ~0ULL) {  // empty, or being filled: settle it with the CAS
      cur = cas128(&table[pos], empty, mine);
      if (cur.x == ~0ULL && cur.y == ~0ULL) {
        toggle(bits, i);
        __stcs(slot_out, (uint32_t)pos);
        return;
      }
    }
    if (cur.x == w0 && (uint32_t)cur.y == w1lo) {
      if ((uint32_t)(cur.y >> 32) > i) {
        const uint32_t old = atomicMin(reinterpret_cast<uint32_t*>(&table[pos]) + 3, i);
        if (old > i) {
          toggle(bits, i);
          toggle(bits, old);
        }
      }
      __stcs(slot_out, (uint32_t)pos);
      return;
    }
    if (++probe > mask || probe >= probe_cap) break;
    pos = (pos + 1) & mask;
    cur = ld_slot(&table[pos]);
  }
  raise_err(st, kErrTableFull);
  *slot_out = 0;
}

// kInsK keys per thread, kInsThreads apart: all their key loads, then all
// their home-slot loads, go out before any is settled.
// Keys read by the insert; with kc.carry set they still lack the carry from
// earlier tiles, which is added here (both words are below p, so p61_add).
struct InsCarry {
  const ulonglong2* carry;
  const uint32_t* lead;
  uint32_t tile_shift;  // log2 of the blocks per hash tile (a power of two)
};

__global__ void __launch_bounds__(kInsThreads) k_ids_insert(const ulonglong2* __restrict__ keys, uint32_t n_ub,
                                                            const uint64_t* n_dev, ulonglong2* table, uint32_t log2m,
                                                            uint64_t probe_cap, uint32_t* __restrict__ slot_of,
                                                            uint32_t* bits, DevStatus* st, InsCarry kc) {
  grid_dep_sync();
  report_keys_used(n_ub, n_dev, st);
  const uint32_t i0 = blockIdx.x * (kInsThreads * kInsK) + threadIdx.x;
  const uint64_t mask = (1ULL << log2m) - 1;
  ulonglong2 k[kInsK], cur[kInsK], cy[kInsK];
  uint32_t lead[kInsK];
  uint64_t pos[kInsK];
  // Every load that does not depend on a key goes out first, together: the
  // keys (the buffer holds n_ub of them, so reading up to n_ub stays inside
  // it), their tiles' carries, and the key count.
#pragma unroll
  for (int j = 0; j < kInsK; ++j) {
    const uint32_t i = i0 + j * kInsThreads;
    k[j] = i < n_ub ? __ldcs(&keys[i]) : make_ulonglong2(~0ULL, ~0ULL);  // streamed once: keep L2 for the table
    lead[j] = 0;
    cy[j] = make_ulonglong2(0, 0);
    if (kc.carry && i < n_ub) {
      const uint32_t t = i >> kc.tile_shift;
      lead[j] = __ldg(&kc.lead[t]);
      cy[j] = __ldg(&kc.carry[t]);
    }
  }
  const uint32_t n = keys_used(n_ub, n_dev);
#pragma unroll
  for (int j = 0; j < kInsK; ++j) {
    const uint32_t i = i0 + j * kInsThreads;
    if (i >= n) {
      k[j] = make_ulonglong2(~0ULL, ~0ULL);
    } else if ((i & ((1u << kc.tile_shift) - 1u)) < lead[j] && k[j].x < kP61 && k[j].y < kP61) {
      k[j] = make_ulonglong2(p61_add(k[j].x, cy[j].x), p61_add(k[j].y, cy[j].y));
    }
  }
#pragma unroll
  for (int j = 0; j < kInsK; ++j) {
    pos[j] = home_slot(k[j].x, k[j].y, log2m);
    cur[j] = k[j].x < kP61 && k[j].y < kP61 ? ld_slot(&table[pos[j]]) : make_ulonglong2(0, 0);
  }
#pragma unroll
  for (int j = 0; j < kInsK; ++j) {
    const uint32_t i = i0 + j * kInsThreads;
    if (i >= n) continue;
    if (k[j].x >= kP61 || k[j].y >= kP61) {
      raise_err(st, kErrInvalid);
      slot_of[i] = 0;
      continue;
    }
    settle(table, mask, probe_cap, i, k[j], pos[j], cur[j], &slot_of[i], bits, st);
  }
}

// ids[i] = rank of the first occurrence of i's key among all first
// occurrences, the bitmap's word prefixes giving ranks.  A first occurrence
// finds its own bit set and is its own first occurrence, with no table read
// (its bitmap word is shared with its neighbours, so the read is coalesced);
// a later occurrence reads its slot's stored index, or, after the
// partitioned dedup (table null), finds the index in slot_of itself.  kGaPer accesses per
// thread, kGaThreads apart, their dependent loads in flight together.
constexpr int kGaThreads = 256;
constexpr int kGaPer = 8;
// slot_of of an access that the prior-request hint matched (no slot)
constexpr uint32_t kMatchedSlot = 0xFFFFFFFFu;
__global__ void __launch_bounds__(kGaThreads) k_ids_gather(const uint32_t* __restrict__ slot_of,
                                                          const ulonglong2* __restrict__ table, uint64_t m,
                                                          const uint32_t* __restrict__ bits,
                                                          const uint32_t* __restrict__ wpre, uint32_t n_ub,
                                                          const uint64_t* n_dev, uint32_t* __restrict__ ids,
                                                          const DevStatus* st) {
  grid_dep_sync();
  const uint32_t n = keys_used(n_ub, n_dev);
  const uint32_t i0 = blockIdx.x * (kGaThreads * kGaPer) + threadIdx.x;
  uint32_t f[kGaPer], own[kGaPer];
#pragma unroll
  for (int k = 0; k < kGaPer; ++k) {
    const uint32_t i = i0 + k * kGaThreads;
    f[k] = i < n ? __ldcs(&slot_of[i]) : kMatchedSlot;
    own[k] = i < n ? bits[i >> 5] : 0u;
  }
#pragma unroll
  for (int k = 0; k < kGaPer; ++k) {
    const uint32_t i = i0 + k * kGaThreads;
    if (f[k] == kMatchedSlot) continue;
    if ((own[k] >> (i & 31)) & 1u)
      f[k] = i;
    else if (table)
      f[k] = in_bounds(st, f[k], m) ? __ldg(reinterpret_cast<const uint32_t*>(&table[f[k]]) + 3) : kNone;
    // else (partitioned dedup): slot_of already holds the first occurrence
  }
  uint32_t wp[kGaPer], bw[kGaPer];
#pragma unroll
  for (int k = 0; k < kGaPer; ++k) {
    const uint32_t i = i0 + k * kGaThreads;
    const bool ok = f[k] < n;
    wp[k] = ok ? wpre[f[k] >> 5] : 0u;
    bw[k] = f[k] == i ? own[k] : ok ? bits[f[k] >> 5] : 0u;
  }
  // a matched access (prior-request hint) gets its id from k_ids_follow
#pragma unroll
  for (int k = 0; k < kGaPer; ++k) {
    const uint32_t i = i0 + k * kGaThreads;
    if (i < n && f[k] != kMatchedSlot) ids[i] = f[k] < n ? wp[k] + __popc(bw[k] & ((1u << (f[k] & 31)) - 1u)) : kNone;
  }
}

// Key i with the carry of its hash tile added (as k_ids_insert does), or
// all-ones past the buffer.
__device__ __forceinline__ ulonglong2 carried_key(const ulonglong2* __restrict__ keys, uint32_t i, uint32_t n_ub,
                                                  const InsCarry& kc) {
  if (i >= n_ub) return make_ulonglong2(~0ULL, ~0ULL);
  ulonglong2 k = __ldcs(&keys[i]);
  if (kc.carry) {
    const uint32_t t = i >> kc.tile_shift;
    if ((i & ((1u << kc.tile_shift) - 1u)) < __ldg(&kc.lead[t]) && k.x < kP61 && k.y < kP61) {
      const ulonglong2 c = __ldg(&kc.carry[t]);
      k = make_ulonglong2(p61_add(k.x, c.x), p61_add(k.y, c.y));
    }
  }
  return k;
}

// ---------------------------------------------------------------- prior-request hint
// A request usually re-sends the whole context of an earlier request of its
// session and appends to it (Sec. 2.3: the turns of a multi-turn session
// extend one context).  Given a hint prior[r] (an earlier request, or none),
// access (r, k) is "matched" when its key equals that of block k of request
// prior[r]: its prefix occurred earlier, so it is not a first occurrence and
// is not inserted.  Equal keys mean equal prefixes, so the matched blocks of
// r are its depths k < lam[r] (k_ids_lam).  A first occurrence is never matched, so the
// table of the unmatched keys still holds every key with its smallest access
// index.  A matched access takes the id of block k of the nearest request on
// its prior chain whose depth k is unmatched (k_ids_follow).  The ids do not
// depend on the hint: any prior[r] < r gives the same ids, only the number of
// table probes changes.
constexpr uint32_t kMatched = kMatchedSlot;  // slot_of of a matched access

struct PriorHint {
  const uint64_t* blk_off;  // n_req + 1 access offsets of the requests
  const uint32_t* prior;    // n_req: an earlier request, or kNone
  const uint32_t* order;    // with sessions: the requests in session order (prior = the place before), or null
  const uint32_t* pos;      //   and the place of every request in it
  uint32_t n_req;
  uint32_t* lam;            // n_req: first unmatched depth (written by k_ids_lam)
  uint32_t* tile_req;       // request of the first access of every kReqTile accesses, and n_req - 1 last
};
constexpr uint32_t kReqTileLog2 = 11;  // 2048 accesses per entry of tile_req

// The last request r in [lo, hi] with off[r] <= i (requests without blocks
// are skipped because a later offset equals theirs).
__device__ __forceinline__ uint32_t req_at(const uint64_t* __restrict__ off, uint32_t lo, uint32_t hi, uint64_t i) {
  while (lo < hi) {
    const uint32_t mid = (lo + hi + 1) >> 1;
    if (__ldg(&off[mid]) <= i)
      lo = mid;
    else
      hi = mid - 1;
  }
  return lo;
}

// tile_req[t] = the request of access t * 2048 (one binary search per entry),
// and tile_req[T] = n_req - 1, so accesses of tile t lie in requests
// [tile_req[t], tile_req[t + 1]].
__global__ void k_tile_req(PriorHint ph, uint32_t n_ub, const uint64_t* n_dev) {
  grid_dep_sync();
  const uint32_t n = keys_used(n_ub, n_dev);
  const uint32_t T = (n + (1u << kReqTileLog2) - 1) >> kReqTileLog2;
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t < T) ph.tile_req[t] = req_at(ph.blk_off, 0, ph.n_req - 1, (uint64_t)t << kReqTileLog2);
  if (t == T) ph.tile_req[t] = ph.n_req - 1;
}

// lam[r], one thread per request: the number of leading depths at which r's
// key equals that of prior[r] (the keys of both requests, as far as the
// shorter one goes).  The keys are prefix keys: equal keys at depth k mean
// equal prefixes through block k, hence equal keys at every depth below k,
// so the equal depths are a leading run and a binary search over the depths
// finds its end in about log2(n_r) pairs of key reads instead of one pair
// per access.  A request with no hint, or none of whose blocks the hint
// repeats, gets 0.  A hint that does not point to an earlier request, or
// offsets that do not fit the keys, raise kErrInvalid.
constexpr int kLamThreads = 256;
__global__ void __launch_bounds__(kLamThreads) k_ids_lam(const ulonglong2* __restrict__ keys, uint32_t n_ub,
                                                         const uint64_t* n_dev, InsCarry kc, PriorHint ph,
                                                         DevStatus* st) {
  grid_dep_sync();
  const uint32_t r = blockIdx.x * kLamThreads + threadIdx.x;
  if (r >= ph.n_req) return;
  const uint32_t n = keys_used(n_ub, n_dev);
  const uint32_t p = __ldg(&ph.prior[r]);
  uint64_t lam = 0;
  if (p != kNone && p >= r) {
    raise_err(st, kErrInvalid);  // a hint must point to an earlier request
  } else if (p != kNone) {
    const uint64_t b = __ldg(&ph.blk_off[r]), e = __ldg(&ph.blk_off[r + 1]);
    const uint64_t pb = __ldg(&ph.blk_off[p]), pe = __ldg(&ph.blk_off[p + 1]);
    if (b > e || pb > pe || e > n || pe > n) {
      raise_err(st, kErrInvalid);
    } else {
      uint64_t hi = e - b < pe - pb ? e - b : pe - pb;  // depths below lam are equal, depth hi is not (or the end)
      while (lam < hi) {
        const uint64_t mid = (lam + hi) >> 1;
        const ulonglong2 x = carried_key(keys, (uint32_t)(b + mid), n, kc);
        const ulonglong2 y = carried_key(keys, (uint32_t)(pb + mid), n, kc);
        if (x.x == y.x && x.y == y.y && x.x < kP61 && x.y < kP61)  // a key that is not a field element is never equal
          lam = mid + 1;
        else
          hi = mid;
      }
    }
  }
  ph.lam[r] = (uint32_t)lam;
}

// kPriorK accesses per thread, kInsThreads apart.  Each access finds its
// request by binary search among the few requests its 2048-access tile
// spans (tile_req); a depth below its request's lam repeats the hint and
// writes kMatched without reading its key; any other access settles its key
// in the table as k_ids_insert does.  The request searches, then the keys and
// slot loads of the unmatched accesses go out together.
constexpr int kPriorK = 1;
template <int K>
__global__ void __launch_bounds__(kInsThreads) k_ids_insert_prior(const ulonglong2* __restrict__ keys, uint32_t n_ub,
                                                                  const uint64_t* n_dev, ulonglong2* table,
                                                                  uint32_t log2m, uint64_t probe_cap,
                                                                  uint32_t* __restrict__ slot_of, uint32_t* bits,
                                                                  DevStatus* st, InsCarry kc, PriorHint ph) {
  grid_dep_sync();
  report_keys_used(n_ub, n_dev, st);
  const uint32_t n = keys_used(n_ub, n_dev);
  const uint32_t base = blockIdx.x * (kInsThreads * K) + threadIdx.x;
  if (blockIdx.x * (kInsThreads * K) >= n) return;  // the whole CTA
  bool unm[K];
#pragma unroll
  for (int j = 0; j < K; ++j) {
    const uint32_t i = base + j * kInsThreads;
    unm[j] = false;
    if (i >= n) continue;
    const uint32_t t = i >> kReqTileLog2;
    const uint32_t r = req_at(ph.blk_off, __ldg(&ph.tile_req[t]), __ldg(&ph.tile_req[t + 1]), i);
    unm[j] = i - __ldg(&ph.blk_off[r]) >= __ldg(&ph.lam[r]);
    if (!unm[j]) __stcs(&slot_of[i], kMatched);
  }
  ulonglong2 k[K], cur[K];
  uint64_t pos[K];
#pragma unroll
  for (int j = 0; j < K; ++j) {
    const uint32_t i = base + j * kInsThreads;
    k[j] = unm[j] ? carried_key(keys, i, n, kc) : make_ulonglong2(0, 0);
    if (unm[j] && (k[j].x >= kP61 || k[j].y >= kP61)) {
      raise_err(st, kErrInvalid);
      slot_of[i] = 0;
      unm[j] = false;
    }
    pos[j] = home_slot(k[j].x, k[j].y, log2m);
    cur[j] = unm[j] ? ld_slot(&table[pos[j]]) : make_ulonglong2(0, 0);
  }
#pragma unroll
  for (int j = 0; j < K; ++j) {
    if (!unm[j]) continue;
    settle(table, (1ULL << log2m) - 1, probe_cap, base + j * kInsThreads, k[j], pos[j], cur[j],
           &slot_of[base + j * kInsThreads], bits, st);
  }
}

// ids of the matched accesses, one warp per request r: its depths below
// lam[r] equal those of prior[r]; walking the prior chain t = prior[r],
// prior[t], ..., the depths in [lam[t], hi) are unmatched in t (their ids
// come from the table) and are copied, and hi drops to lam[t], until no
// depth is left.  A chain that does not strictly descend, or that ends while
// depths are left, is malformed input.
constexpr int kFoThreads = 256;
__global__ void __launch_bounds__(kFoThreads) k_ids_follow(PriorHint ph, uint32_t* __restrict__ ids, DevStatus* st) {
  grid_dep_sync();
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t r = blockIdx.x * (kFoThreads / 32) + (threadIdx.x >> 5);
  if (r >= ph.n_req) return;
  const uint64_t b = ph.blk_off[r], nr = ph.blk_off[r + 1] - b;
  const uint32_t lr = ph.lam[r];
  uint64_t hi = lr < nr ? lr : nr;
  uint32_t cur = r, t = ph.prior[r];
  while (hi > 0) {
    if (t == kNone || t >= cur) {
      if (lane == 0) raise_err(st, kErrInvalid);
      return;
    }
    const uint64_t tb = ph.blk_off[t];
    const uint64_t lo = ph.lam[t];  // depths [lo, n_t) of t are unmatched
    if (lo < hi) {
      if (!in_bounds(st, tb + hi - 1, b) || !in_bounds(st, b + hi - 1, ph.blk_off[ph.n_req])) return;
      for (uint64_t d = lo + lane; d < hi; d += 32) ids[b + d] = ids[tb + d];
      hi = lo;
    }
    cur = t;
    t = ph.prior[t];
  }
}

// The same with the session order (the pipeline's hint: prior[r] is the
// request just before r in its session): the warp of request r reads 32
// ancestors at once, places pos[r] - 1, pos[r] - 2, ... of the order, down
// to the session's first request (whose prior is none).  Ancestor i of the
// window copies depths [lam, hi_i) when lam < hi_i, hi_i being the smallest
// of hi and the lam of the ancestors before it (a prefix minimum over the
// lanes), exactly as the walk one ancestor at a time would.  Two dependent
// load rounds per 32 ancestors instead of one per ancestor.
__global__ void __launch_bounds__(kFoThreads) k_ids_follow_win(PriorHint ph, uint32_t* __restrict__ ids,
                                                               DevStatus* st) {
  grid_dep_sync();
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t r = blockIdx.x * (kFoThreads / 32) + (threadIdx.x >> 5);
  if (r >= ph.n_req) return;
  const uint64_t b = ph.blk_off[r], nr = ph.blk_off[r + 1] - b;
  const uint32_t lr = ph.lam[r];
  uint64_t hi = lr < nr ? lr : nr;
  if (hi == 0) return;
  const uint32_t j = ph.pos[r];
  if (j >= ph.n_req || ph.order[j] != r || ph.prior[r] == kNone || j == 0 || ph.order[j - 1] != ph.prior[r]) {
    if (lane == 0) raise_err(st, kErrInvalid);  // the order does not match the hint
    return;
  }
  uint32_t carry_p = ph.prior[r];  // the prior of the nearest ancestor not yet read
  for (uint32_t dist = 1;; dist += 32) {
    const int64_t q = (int64_t)j - dist - lane;
    const uint32_t a = q >= 0 ? __ldg(&ph.order[q]) : kNone;
    uint32_t la = kNone, pa = kNone;
    uint64_t ta = 0;
    if (a != kNone) {
      la = __ldg(&ph.lam[a]);
      pa = __ldg(&ph.prior[a]);
      ta = __ldg(&ph.blk_off[a]);
    }
    // the chain: the lane's ancestor is the prior of the lane before's, until
    // a session's first request (prior none) ends it
    uint32_t prev_p = __shfl_up_sync(kFull, pa, 1);
    if (lane == 0) prev_p = carry_p;
    const bool linked = prev_p == a && a != kNone;
    const uint32_t ends = __ballot_sync(kFull, a != kNone && pa == kNone);
    const uint32_t first_end = ends ? __ffs(ends) - 1 : 32u;
    const bool valid = lane <= first_end && a != kNone;
    if (__any_sync(kFull, lane <= first_end && !(valid && linked))) {
      if (lane == 0) raise_err(st, kErrInvalid);  // a broken chain, or one that runs out with depths left
      return;
    }
    // hi before this lane's ancestor: the prefix minimum of lam over the lanes before it
    uint64_t m = valid ? (uint64_t)la : ~0ULL;
    uint64_t incl = m;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t y = __shfl_up_sync(kFull, incl, o);
      if (lane >= (uint32_t)o) incl = y < incl ? y : incl;
    }
    uint64_t excl = __shfl_up_sync(kFull, incl, 1);
    if (lane == 0) excl = ~0ULL;
    const uint64_t hl = excl < hi ? excl : hi;
    uint32_t todo = __ballot_sync(kFull, valid && (uint64_t)la < hl);
    while (todo) {
      const int src = __ffs(todo) - 1;
      todo &= todo - 1;
      const uint64_t lo = __shfl_sync(kFull, (uint64_t)la, src), top = __shfl_sync(kFull, hl, src);
      const uint64_t tb = __shfl_sync(kFull, ta, src);
      if (!in_bounds(st, tb + top - 1, b) || !in_bounds(st, b + top - 1, ph.blk_off[ph.n_req])) return;
      for (uint64_t d = lo + lane; d < top; d += 32) ids[b + d] = ids[tb + d];
    }
    const uint64_t wmin = __shfl_sync(kFull, incl, 31);
    hi = wmin < hi ? wmin : hi;
    carry_p = __shfl_sync(kFull, pa, 31);
    if (hi == 0) return;
    if (first_end < 32) {  // the session's first request was reached with depths left
      if (lane == 0) raise_err(st, kErrInvalid);
      return;
    }
  }
}

// prior[r] = the previous request of r's session, from the requests sorted
// stably by session label: neighbours in that order with the same label.
// With `order` and `pos` (or null), also the session order itself: order[j]
// = the request at place j, pos[r] = the place of request r.
__global__ void k_session_prior(const uint32_t* __restrict__ ses_sorted, const uint32_t* __restrict__ req_sorted,
                                const uint32_t* __restrict__ ses, uint32_t n_req, uint32_t n_session,
                                uint32_t* __restrict__ prior, uint32_t* err, uint32_t* __restrict__ order,
                                uint32_t* __restrict__ pos) {
  grid_dep_sync();
  const uint32_t j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= n_req) return;
  if (ses[j] >= n_session) atomicOr(err, kErrInvalid);  // the sort sees only the label's low bits
  const uint32_t sj = ses_sorted[j], rj = req_sorted[j];
  prior[rj] = (j > 0 && ses_sorted[j - 1] == sj) ? req_sorted[j - 1] : kNone;
  if (order) {
    order[j] = rj;
    pos[rj] = j;
  }
}

// ---------------------------------------------------------------- partitioned dedup
// With a table larger than L2 every settled key costs a random DRAM sector
// (read, then the claimed sector written back), about 20 G keys/s.  The
// partitioned method moves the keys to be settled (the unmatched accesses)
// instead, in streaming passes, into 2^16 partitions by 16 bits of h0, and
// settles every partition in a table of its own in shared memory:
//   k_pd_flags     the bitmap of the accesses to settle (ubits), and its
//                  copy that becomes the first-occurrence bitmap (bits):
//                  every access without a hint; with one, the depths of each
//                  request from its lam on (a warp per request)
//   k_pd_count     level 1: per CTA of a persistent grid, the keys of its
//                  range of accesses per bucket (h0 bits 53..60)
//   k_pd_rows1     one CTA per bucket: the prefix of its counts over the
//                  level-1 CTAs, and the bucket's total
//   k_pd_scatter1  the same pass again: a 16-byte record (96 key bits,
//                  access index) per access to settle, in bucket order
//   k_pd_count2    level 2: per tile of kPdTile2 records of one bucket, the
//                  records per partition (h0 bits 45..60); one atomic per
//                  tile and partition claims the tile's place in it
//   k_pd_rows2     one CTA per bucket: the bounds of its partitions
//   k_pd_scatter2  every tile's records moved to their partitions
//   k_pd_dedup     one partition at a time per CTA: every record settles its
//                  key in a shared-memory table (key + smallest index); an
//                  index that is never stored, or that a smaller one
//                  replaces, is a repeat and goes to a list, whose entries
//                  then take their key's smallest index into slot_of and
//                  clear their bit.
// bits then holds exactly the first occurrences, and k_ids_gather_pd reads a
// repeat's first occurrence from slot_of itself (slot_of is written for the
// repeats only; ubits tells the settled accesses from the matched ones).  A partition holding more
// distinct keys than its shared table raises kErrTableFull, as an overfull
// hash table does, and the call redoes the stage with the full table.
// Both scatters sort a round's records by destination in shared memory
// first, so that a warp's stores land in runs of consecutive records
// rather than one 16-byte store per destination.
constexpr int kPdThreads = 512;
constexpr int kPdPer = 8;
constexpr uint32_t kPdRound = kPdThreads * kPdPer;   // accesses per level-1 round (and staged records)
constexpr uint32_t kPdBuckets = 256;                 // level 1: h0 bits 53..60
constexpr uint32_t kPdParts = 65536;                 // level 2: h0 bits 45..60
constexpr uint32_t kPdMaxG1 = 2048;                  // largest level-1 grid
constexpr int kPd2Threads = 512;
constexpr int kPd2Per = 8;
constexpr uint32_t kPdTile2 = kPd2Threads * kPd2Per;  // 4096 records per level-2 tile
constexpr int kPdDedupThreads = 512;
constexpr int kPdDedupPer = 4;
constexpr uint32_t kPdSlots = 6144;  // shared table: 96 KB
constexpr uint32_t kPdList = 1536;   // repeats listed per partition: 12 KB
constexpr size_t kPdDedupSmem = sizeof(ulonglong2) * kPdSlots + sizeof(uint2) * kPdList;

constexpr size_t kPdStageSmem = sizeof(ulonglong2) * kPdRound;  // 64 KB
static_assert(kPdTile2 == kPdRound, "both scatters stage one round of records");

// The record of access i with key k: the same 96 key bits as a table slot.
__device__ __forceinline__ ulonglong2 pd_record(ulonglong2 k, uint32_t i) {
  return make_ulonglong2(k.x | ((k.y & 7ULL) << 61), (uint64_t)(uint32_t)(k.y >> 3) | ((uint64_t)i << 32));
}
__device__ __forceinline__ uint32_t pd_bucket(uint64_t w0) { return (uint32_t)(w0 >> 53) & (kPdBuckets - 1); }
__device__ __forceinline__ uint32_t pd_part(uint64_t w0) { return (uint32_t)(w0 >> 45) & (kPdParts - 1); }

// Exclusive prefix of v over threads 0..255 and the total, for a CTA of at
// least 256 threads (the others pass 0); every thread calls it.
__device__ __forceinline__ uint32_t scan256(uint32_t v, uint32_t* total) {
  __shared__ uint32_t s_w[8];
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint32_t inc = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint32_t t = __shfl_up_sync(kFull, inc, d);
    if (lane >= (uint32_t)d) inc += t;
  }
  if (w < 8 && lane == 31) s_w[w] = inc;
  __syncthreads();
  uint32_t before = 0, tot = 0;
#pragma unroll
  for (uint32_t k = 0; k < 8; ++k) {
    const uint32_t x = s_w[k];
    if (k < w) before += x;
    tot += x;
  }
  __syncthreads();
  *total = tot;
  return before + inc - v;
}

// s_bst[0..256]: the bucket bounds in the level-1 records (prefix of tot1).
__device__ __forceinline__ void pd_bucket_bounds(const uint32_t* tot1, uint32_t* s_bst) {
  uint32_t total;
  const uint32_t ex = scan256(threadIdx.x < kPdBuckets ? tot1[threadIdx.x] : 0u, &total);
  if (threadIdx.x < kPdBuckets) s_bst[threadIdx.x] = ex;
  if (threadIdx.x == 0) s_bst[kPdBuckets] = total;
  __syncthreads();
}

// s_tp[0..256]: the first level-2 tile of every bucket, and the tile count.
__device__ __forceinline__ void pd_tile_starts(const uint32_t* s_bst, uint32_t* s_tp) {
  uint32_t total;
  const uint32_t nt = threadIdx.x < kPdBuckets
                          ? (uint32_t)(((uint64_t)s_bst[threadIdx.x + 1] - s_bst[threadIdx.x] + kPdTile2 - 1) / kPdTile2)
                          : 0u;
  const uint32_t ex = scan256(nt, &total);
  if (threadIdx.x < kPdBuckets) s_tp[threadIdx.x] = ex;
  if (threadIdx.x == 0) s_tp[kPdBuckets] = total;
  __syncthreads();
}

struct PdArgs {
  const ulonglong2* keys;
  uint32_t n_ub;
  const uint64_t* n_dev;
  InsCarry kc;
  PriorHint ph;        // ph.lam null: no hint
  uint32_t per;        // accesses per level-1 CTA, a multiple of kPdRound
  uint32_t* cnt1;      // [bucket * grid + cta]
  uint32_t* off1;      // its prefix along each bucket's row
  uint32_t* tot1;      // kPdBuckets totals
  const uint32_t* ubits;  // the accesses to settle (k_pd_flags)
  ulonglong2* rec1;    // n_ub records
  DevStatus* st;
};

// The accesses to settle, as the bitmap `ubits`, and its copy `bits`, which
// the dedup turns into the first occurrences (both zeroed before): without a
// hint all of [0, n), one thread per word; with one, a warp per request sets
// the bits of its depths from lam on (whole words by plain stores, the two
// partial words at its ends by atomicOr, as neighbouring requests share
// them).
__global__ void __launch_bounds__(256) k_pd_flags(PriorHint ph, uint32_t n_ub, const uint64_t* n_dev,
                                                  uint32_t* __restrict__ ubits, uint32_t* __restrict__ bits,
                                                  uint32_t nwords) {
  grid_dep_sync();
  const uint32_t n = keys_used(n_ub, n_dev);
  if (!ph.lam) {
    const uint32_t w = blockIdx.x * 256 + threadIdx.x;
    if (w < nwords) {
      const uint64_t lo = 32ULL * w;
      const uint32_t m = lo + 32 <= n ? ~0u : lo < n ? (1u << (n - lo)) - 1u : 0u;
      ubits[w] = m;
      bits[w] = m;
    }
    return;
  }
  const uint32_t r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= ph.n_req) return;
  const uint64_t b = __ldg(&ph.blk_off[r]);
  uint64_t e = __ldg(&ph.blk_off[r + 1]);
  if (e > n) e = n;
  if (e <= b) return;
  const uint64_t l = __ldg(&ph.lam[r]);
  const uint64_t u0 = l < e - b ? b + l : e;
  if (u0 >= e) return;
  const uint64_t w0 = u0 >> 5, w1 = (e - 1) >> 5;
  for (uint64_t w = w0 + lane; w <= w1; w += 32) {
    const uint32_t lo = w == w0 ? (uint32_t)(u0 & 31) : 0u;
    const uint32_t hi = w == w1 ? (uint32_t)((e - 1) & 31) + 1 : 32u;
    const uint32_t m = (hi == 32 ? ~0u : (1u << hi) - 1u) & ~((1u << lo) - 1u);
    if (m == ~0u) {
      ubits[w] = m;
      bits[w] = m;
    } else {
      atomicOr(&ubits[w], m);
      atomicOr(&bits[w], m);
    }
  }
}

// The carries of the hash tiles that a round of kPdRound accesses from
// `base` spans (base a multiple of kPdRound, hence of every tile size; a
// hash tile holds 8 to 256 blocks), read once per round into shared memory:
// entry t is tile (base >> tile_shift) + t, up to hi.
constexpr uint32_t kPdRoundTiles = kPdRound / 8;
__device__ __forceinline__ void pd_round_carry(const InsCarry& kc, uint64_t base, uint64_t hi, uint32_t* s_lead,
                                               ulonglong2* s_cy) {
  if (!kc.carry) return;
  const uint32_t nt = kPdRound >> kc.tile_shift;
  const uint64_t t0 = base >> kc.tile_shift;
  for (uint32_t t = threadIdx.x; t < nt; t += blockDim.x)
    if (((t0 + t) << kc.tile_shift) < hi) {
      s_lead[t] = __ldg(&kc.lead[t0 + t]);
      s_cy[t] = __ldg(&kc.carry[t0 + t]);
    }
}

// Key i of the round from `base`, with its tile's carry added (as
// carried_key does) from the round's shared copy.
__device__ __forceinline__ ulonglong2 pd_key(const ulonglong2* __restrict__ keys, uint32_t i, uint64_t base,
                                             const InsCarry& kc, const uint32_t* s_lead, const ulonglong2* s_cy) {
  ulonglong2 k = __ldcs(&keys[i]);
  if (kc.carry) {
    const uint32_t t = (uint32_t)(i - base) >> kc.tile_shift;
    if ((i & ((1u << kc.tile_shift) - 1u)) < s_lead[t] && k.x < kP61 && k.y < kP61) {
      const ulonglong2 c = s_cy[t];
      k = make_ulonglong2(p61_add(k.x, c.x), p61_add(k.y, c.y));
    }
  }
  return k;
}

// h0 of key i with the carry of its hash tile added (the first word of
// carried_key, for a key whose second word is a field element).
__device__ __forceinline__ uint64_t carried_h0(const ulonglong2* __restrict__ keys, uint32_t i, const InsCarry& kc) {
  uint64_t x = __ldcs(reinterpret_cast<const unsigned long long*>(&keys[i]));
  if (kc.carry) {
    const uint32_t t = i >> kc.tile_shift;
    if ((i & ((1u << kc.tile_shift) - 1u)) < __ldg(&kc.lead[t]) && x < kP61)
      x = p61_add(x, __ldg(reinterpret_cast<const unsigned long long*>(&kc.carry[t])));
  }
  return x;
}

// Level 1, counting: the keys of CTA g's accesses [g per, (g + 1) per) per
// bucket.  Only h0 is read (the bucket is in it).  The scatter below skips a
// key whose h1 is not a field element as well, and raises kErrInvalid, so
// the counts can only differ from it on input the call rejects.
__global__ void __launch_bounds__(kPdThreads, 4) k_pd_count(PdArgs a) {
  grid_dep_sync();
  report_keys_used(a.n_ub, a.n_dev, a.st);
  __shared__ uint32_t h[kPdBuckets];
  for (uint32_t x = threadIdx.x; x < kPdBuckets; x += kPdThreads) h[x] = 0;
  const uint32_t n = keys_used(a.n_ub, a.n_dev);
  const uint64_t lo = (uint64_t)blockIdx.x * a.per;
  const uint64_t hi = lo + a.per < n ? lo + a.per : n;
  __syncthreads();
  for (uint64_t base = lo; base < hi; base += kPdRound) {
    bool u[kPdPer];
    uint64_t x[kPdPer];
#pragma unroll
    for (int j = 0; j < kPdPer; ++j) {
      const uint64_t i = base + j * kPdThreads + threadIdx.x;
      u[j] = i < hi && ((__ldg(&a.ubits[i >> 5]) >> (i & 31)) & 1u);
    }
#pragma unroll
    for (int j = 0; j < kPdPer; ++j)
      x[j] = u[j] ? carried_h0(a.keys, (uint32_t)(base + j * kPdThreads + threadIdx.x), a.kc) : ~0ULL;
#pragma unroll
    for (int j = 0; j < kPdPer; ++j)
      if (u[j] && x[j] < kP61) atomicAdd(&h[pd_bucket(x[j])], 1u);
  }
  __syncthreads();
  for (uint32_t x = threadIdx.x; x < kPdBuckets; x += kPdThreads) a.cnt1[x * gridDim.x + blockIdx.x] = h[x];
}

// Level 1, scattering: the same accesses and keys as k_pd_count.  Each round
// ranks its records per bucket, sorts them into shared memory by bucket, and
// writes each bucket's run at the CTA's running place in the bucket.
__global__ void __launch_bounds__(kPdThreads, 2) k_pd_scatter1(PdArgs a) {
  grid_dep_sync();
  extern __shared__ ulonglong2 stage[];  // kPdRound records
  __shared__ uint32_t h[kPdBuckets];     // the next place in each bucket
  __shared__ uint32_t c[kPdBuckets], so[kPdBuckets];  // the round's records per bucket, their offsets
  __shared__ uint32_t s_bst[kPdBuckets + 1];
  __shared__ uint32_t s_lead[kPdRoundTiles];
  __shared__ ulonglong2 s_cy[kPdRoundTiles];
  pd_bucket_bounds(a.tot1, s_bst);
  for (uint32_t x = threadIdx.x; x < kPdBuckets; x += kPdThreads) {
    h[x] = s_bst[x] + a.off1[x * gridDim.x + blockIdx.x];
    c[x] = 0;
  }
  const uint32_t n = keys_used(a.n_ub, a.n_dev);
  const uint64_t lo = (uint64_t)blockIdx.x * a.per;
  const uint64_t hi = lo + a.per < n ? lo + a.per : n;
  pd_round_carry(a.kc, lo, hi, s_lead, s_cy);
  __syncthreads();
  for (uint64_t base = lo; base < hi; base += kPdRound) {
    bool u[kPdPer];
    ulonglong2 k[kPdPer];
    uint32_t rk[kPdPer];
#pragma unroll
    for (int j = 0; j < kPdPer; ++j) {
      const uint64_t i = base + j * kPdThreads + threadIdx.x;
      u[j] = i < hi && ((__ldg(&a.ubits[i >> 5]) >> (i & 31)) & 1u);
    }
#pragma unroll
    for (int j = 0; j < kPdPer; ++j) {
      const uint32_t i = (uint32_t)(base + j * kPdThreads + threadIdx.x);
      k[j] = u[j] ? pd_key(a.keys, i, base, a.kc, s_lead, s_cy) : make_ulonglong2(0, 0);
      if (u[j] && (k[j].x >= kP61 || k[j].y >= kP61)) {  // not a field element: never settled
        raise_err(a.st, kErrInvalid);
        u[j] = false;
      }
    }
#pragma unroll
    for (int j = 0; j < kPdPer; ++j) rk[j] = u[j] ? atomicAdd(&c[pd_bucket(k[j].x)], 1u) : 0u;
    __syncthreads();
    uint32_t nrec;
    const uint32_t ex = scan256(threadIdx.x < kPdBuckets ? c[threadIdx.x] : 0u, &nrec);
    if (threadIdx.x < kPdBuckets) so[threadIdx.x] = ex;
    __syncthreads();
#pragma unroll
    for (int j = 0; j < kPdPer; ++j)
      if (u[j])
        stage[so[pd_bucket(k[j].x)] + rk[j]] = pd_record(k[j], (uint32_t)(base + j * kPdThreads + threadIdx.x));
    __syncthreads();
    for (uint32_t x = threadIdx.x; x < nrec; x += kPdThreads) {
      const ulonglong2 r = stage[x];
      const uint32_t d = pd_bucket(r.x);
      const uint32_t at = h[d] + (x - so[d]);
      if (at < a.n_ub)
        __stcg(&a.rec1[at], r);
      else
        raise_err(a.st, kErrInvalid);
    }
    __syncthreads();
    for (uint32_t x = threadIdx.x; x < kPdBuckets; x += kPdThreads) {
      h[x] += c[x];
      c[x] = 0;
    }
    pd_round_carry(a.kc, base + kPdRound, hi, s_lead, s_cy);  // the next round's (its reads of these are done)
    __syncthreads();
  }
}

// One CTA per bucket: the exclusive prefix of the bucket's counts along the
// level-1 CTAs (its place in the bucket for each), and the bucket's total.
__global__ void __launch_bounds__(256) k_pd_rows1(const uint32_t* __restrict__ cnt1, uint32_t g1,
                                                  uint32_t* __restrict__ off1, uint32_t* __restrict__ tot1) {
  grid_dep_sync();
  const uint32_t* row = cnt1 + (size_t)blockIdx.x * g1;
  uint32_t* out = off1 + (size_t)blockIdx.x * g1;
  const uint32_t per = (g1 + 255) / 256;
  const uint32_t a0 = threadIdx.x * per < g1 ? threadIdx.x * per : g1;
  const uint32_t a1 = a0 + per < g1 ? a0 + per : g1;
  uint32_t sum = 0;
  for (uint32_t e = a0; e < a1; ++e) sum += row[e];
  uint32_t total;
  uint32_t run = scan256(sum, &total);
  for (uint32_t e = a0; e < a1; ++e) {
    const uint32_t v = row[e];
    out[e] = run;
    run += v;
  }
  if (threadIdx.x == 0) tot1[blockIdx.x] = total;
}

struct PdLevel2 {
  const ulonglong2* rec1;
  const uint32_t* tot1;
  uint32_t* tot2;     // kPdParts totals (zeroed by the call)
  uint32_t* rel2;     // [tile * 256 + partition of the bucket]: the tile's place in the partition
  const uint32_t* base2;
  ulonglong2* rec2;
  uint32_t cap;       // records rec1 and rec2 hold
  uint32_t max_tiles; // entries of rel2 / 256
  DevStatus* st;
};

// Level 2 over tiles of kPdTile2 records of one bucket (a persistent grid
// walks the tiles).  The count pass claims the tile's range of every
// partition (the atomic's old value); the scatter pass writes the tile's
// records there, ranked per partition inside the tile, so they fill the
// claimed ranges exactly (both passes read the same records).
template <bool SCATTER>
__global__ void __launch_bounds__(kPd2Threads, 2) k_pd_level2(PdLevel2 a) {
  grid_dep_sync();
  extern __shared__ ulonglong2 stage[];  // scatter: kPdTile2 records
  __shared__ uint32_t h[256], s_at[256], so[256];
  __shared__ uint32_t s_bst[kPdBuckets + 1], s_tp[kPdBuckets + 1];
  pd_bucket_bounds(a.tot1, s_bst);
  pd_tile_starts(s_bst, s_tp);
  const uint32_t T = s_tp[kPdBuckets];
  if (T > a.max_tiles) {
    if (threadIdx.x == 0 && blockIdx.x == 0) raise_err(a.st, kErrInvalid);
    return;
  }
  for (uint32_t tile = blockIdx.x; tile < T; tile += gridDim.x) {
    uint32_t lo = 0, hi = kPdBuckets - 1;  // the bucket: the last d with s_tp[d] <= tile
    while (lo < hi) {
      const uint32_t mid = (lo + hi + 1) >> 1;
      if (s_tp[mid] <= tile)
        lo = mid;
      else
        hi = mid - 1;
    }
    const uint64_t start = s_bst[lo] + (uint64_t)(tile - s_tp[lo]) * kPdTile2;
    const uint64_t end = start + kPdTile2 < s_bst[lo + 1] ? start + kPdTile2 : s_bst[lo + 1];
    const uint32_t pbase = lo << 8;
    for (uint32_t x = threadIdx.x; x < 256; x += kPd2Threads) {
      h[x] = 0;
      if (SCATTER) s_at[x] = a.base2[pbase + x] + a.rel2[(size_t)tile * 256 + x];
    }
    __syncthreads();
    ulonglong2 v[kPd2Per];
    uint32_t rk[kPd2Per];
#pragma unroll
    for (int q = 0; q < kPd2Per; ++q) {
      const uint64_t x = start + q * kPd2Threads + threadIdx.x;
      v[q] = x < end && x < a.cap ? __ldcs(&a.rec1[x]) : make_ulonglong2(~0ULL, ~0ULL);
    }
#pragma unroll
    for (int q = 0; q < kPd2Per; ++q)
      rk[q] = v[q].x != ~0ULL ? atomicAdd(&h[pd_part(v[q].x) & 255], 1u) : 0u;
    __syncthreads();
    if (!SCATTER) {
      for (uint32_t x = threadIdx.x; x < 256; x += kPd2Threads)
        a.rel2[(size_t)tile * 256 + x] = h[x] ? atomicAdd(&a.tot2[pbase + x], h[x]) : 0u;
    } else {  // sort the tile by partition in shared memory, then write the runs
      uint32_t nrec;
      const uint32_t ex = scan256(threadIdx.x < 256 ? h[threadIdx.x] : 0u, &nrec);
      if (threadIdx.x < 256) so[threadIdx.x] = ex;
      __syncthreads();
#pragma unroll
      for (int q = 0; q < kPd2Per; ++q)
        if (v[q].x != ~0ULL) stage[so[pd_part(v[q].x) & 255] + rk[q]] = v[q];
      __syncthreads();
      for (uint32_t x = threadIdx.x; x < nrec; x += kPd2Threads) {
        const ulonglong2 r = stage[x];
        const uint32_t p2 = pd_part(r.x) & 255;
        const uint32_t pos = s_at[p2] + (x - so[p2]);
        if (pd_bucket(r.x) == lo && pos < a.cap)
          __stcg(&a.rec2[pos], r);
        else
          raise_err(a.st, kErrInvalid);
      }
    }
    __syncthreads();
  }
}

// One CTA per bucket: the bounds of its 256 partitions (the bucket's bound
// plus the prefix of their totals); base2[kPdParts] = the record count.
__global__ void __launch_bounds__(256) k_pd_rows2(const uint32_t* __restrict__ tot1, const uint32_t* __restrict__ tot2,
                                                  uint32_t* __restrict__ base2, DevStatus* st) {
  grid_dep_sync();
  __shared__ uint32_t s_bst[kPdBuckets + 1];
  pd_bucket_bounds(tot1, s_bst);
  const uint32_t d = blockIdx.x;
  uint32_t total;
  const uint32_t ex = scan256(tot2[d * 256 + threadIdx.x], &total);
  base2[d * 256 + threadIdx.x] = s_bst[d] + ex;
  if (threadIdx.x == 0 && total != s_bst[d + 1] - s_bst[d]) raise_err(st, kErrInvalid);
  if (d == kPdBuckets - 1 && threadIdx.x == 0) base2[kPdParts] = s_bst[kPdBuckets];
}

__device__ __forceinline__ ulonglong2 ld_shared_v2(const ulonglong2* p) {
  ulonglong2 v;
  asm volatile("ld.volatile.shared.v2.u64 {%0, %1}, [%2];"
               : "=l"(v.x), "=l"(v.y)
               : "r"((uint32_t)__cvta_generic_to_shared(p))
               : "memory");
  return v;
}

__device__ __forceinline__ ulonglong2 cas128_shared(ulonglong2* addr, ulonglong2 cmp, ulonglong2 val) {
  ulonglong2 old;
  asm volatile(
      "{\n\t.reg .b128 c, v, d;\n\t"
      "mov.b128 c, {%2, %3};\n\t"
      "mov.b128 v, {%4, %5};\n\t"
      "atom.shared.cas.b128 d, [%6], c, v;\n\t"
      "mov.b128 {%0, %1}, d;\n\t}"
      : "=l"(old.x), "=l"(old.y)
      : "l"(cmp.x), "l"(cmp.y), "l"(val.x), "l"(val.y), "r"((uint32_t)__cvta_generic_to_shared(addr))
      : "memory");
  return old;
}

// Home slot of a record in a partition's table of ts slots: h0's low 32 bits
// (the partition fixes bits 45..60 only).
__device__ __forceinline__ uint32_t pd_home(uint64_t w0, uint32_t ts) { return __umulhi((uint32_t)w0, ts); }

// One probe for record r at slot sl of the shared table (linear probing from
// pd_home): claim the slot if it is empty, with one 128-bit CAS, or meet r's
// key there, where the smaller of the two indices stays.  The index that
// does not stay (r's own, or the one r's atomicMin replaced) is a repeat: it
// comes back in *rep with the slot in *rs.  True when r is settled here;
// false when the slot holds another key (probe the next one).
__device__ __forceinline__ bool pd_probe(ulonglong2* tab, uint32_t ts, ulonglong2 r, uint32_t sl, uint32_t* rep,
                                         uint32_t* rs) {
  const ulonglong2 empty = make_ulonglong2(~0ULL, ~0ULL);
  const uint32_t idx = (uint32_t)(r.y >> 32);
  ulonglong2 cur = ld_shared_v2(&tab[sl]);
  if (cur.x == ~0ULL || cur.y == ~0ULL) {  // empty (or read while being claimed): the CAS settles it
    cur = cas128_shared(&tab[sl], empty, r);
    if (cur.x == ~0ULL && cur.y == ~0ULL) return true;
  }
  if (cur.x == r.x && (uint32_t)cur.y == (uint32_t)r.y) {
    uint32_t out = idx;
    if ((uint32_t)(cur.y >> 32) > idx) {
      const uint32_t old = atomicMin(reinterpret_cast<uint32_t*>(&tab[sl]) + 3, idx);
      out = old > idx ? old : idx;
    }
    *rep = out;
    *rs = sl;
    return true;
  }
  return false;
}

// Appends (rep, rs) to the shared repeat list for the lanes that have one
// (rep != kNone), one atomic per warp; past kPdList entries only the count
// grows.  Every lane of the warp calls it.
__device__ __forceinline__ void pd_list_push(uint32_t rep, uint32_t rs, uint2* list, uint32_t* nlist) {
  const uint32_t m = __ballot_sync(kFull, rep != kNone);
  if (!m) return;
  const uint32_t lane = threadIdx.x & 31;
  uint32_t base = 0;
  if (lane == __ffs(m) - 1) base = atomicAdd(nlist, (uint32_t)__popc(m));
  base = __shfl_sync(kFull, base, __ffs(m) - 1);
  if (rep != kNone) {
    const uint32_t k = base + __popc(m & ((1u << lane) - 1u));
    if (k < kPdList) list[k] = make_uint2(rep, rs);
  }
}

// The smallest index stored for r's key, or kNone if the key is not there.
__device__ __forceinline__ uint32_t pd_find(const ulonglong2* tab, uint32_t ts, ulonglong2 r) {
  uint32_t s = pd_home(r.x, ts);
  for (uint32_t probe = 0; probe < ts; ++probe) {
    const ulonglong2 cur = tab[s];
    if (cur.x == r.x && (uint32_t)cur.y == (uint32_t)r.y) return (uint32_t)(cur.y >> 32);
    if (cur.x == ~0ULL) return kNone;
    s = s + 1 == ts ? 0 : s + 1;
  }
  return kNone;
}

__device__ __forceinline__ void pd_repeat(uint32_t* slot_of, uint32_t* bits, uint32_t i, uint32_t m) {
  slot_of[i] = m;
  atomicAnd(&bits[i >> 5], ~(1u << (i & 31)));
}

struct PdDedup {
  const ulonglong2* rec2;
  const uint32_t* base2;  // kPdParts + 1 partition bounds
  uint32_t cap;
  uint32_t* slot_of;
  uint32_t* bits;
  uint32_t n_ub;
  DevStatus* st;
};

// A partition's table takes twice its records in slots (at most kPdSlots),
// so small partitions clear little shared memory.  The loads of the next
// chunk of records (or of the next partition's first chunk) are issued
// before the current chunk is inserted, so they overlap its inserts.
__global__ void __launch_bounds__(kPdDedupThreads, 2) k_pd_dedup(PdDedup a) {
  grid_dep_sync();
  extern __shared__ ulonglong2 tab[];  // kPdSlots, then the repeat list
  uint2* list = reinterpret_cast<uint2*>(tab + kPdSlots);
  __shared__ uint32_t s_nlist;
  constexpr uint32_t kChunk = kPdDedupThreads * kPdDedupPer;
  const ulonglong2 empty = make_ulonglong2(~0ULL, ~0ULL);
  auto load = [&](ulonglong2(&dst)[kPdDedupPer], uint32_t c, uint32_t end) {
#pragma unroll
    for (int q = 0; q < kPdDedupPer; ++q) {
      const uint32_t x = c + q * kPdDedupThreads + threadIdx.x;
      dst[q] = x < end && x < a.cap ? __ldcs(&a.rec2[x]) : empty;
    }
  };
  uint32_t p = blockIdx.x, b = 0, e = 0;
  if (p < kPdParts) {
    b = a.base2[p];
    e = a.base2[p + 1];
  }
  ulonglong2 v[kPdDedupPer];
  load(v, b, e);
  while (p < kPdParts) {
    const uint32_t pn = p + gridDim.x;
    uint32_t bn = 0, en = 0;
    if (pn < kPdParts) {
      bn = a.base2[pn];
      en = a.base2[pn + 1];
    }
    if (b >= e || e > a.cap) {  // nothing to settle (or bounds past the records: malformed)
      if (b < e && threadIdx.x == 0) raise_err(a.st, kErrInvalid);
      load(v, bn, en);
    } else {
      const uint32_t ts = e - b < kPdSlots / 2 ? ((2 * (e - b) + 31) & ~31u) : kPdSlots;
      for (uint32_t x = threadIdx.x; x < ts; x += kPdDedupThreads) tab[x] = empty;
      if (threadIdx.x == 0) s_nlist = 0;
      __syncthreads();
      bool full = false;
      for (uint32_t c = b;; c += kChunk) {
        const bool more = c + kChunk < e;
        ulonglong2 w[kPdDedupPer];
        if (more)
          load(w, c + kChunk, e);
        else
          load(w, bn, en);
        // one probe per lane per round: a lane that settles its record takes
        // its next one at once, so a long probe run holds back only its own
        // lane's queue rather than the whole warp at every record
        uint32_t nv = 0;
#pragma unroll
        for (int q = 0; q < kPdDedupPer; ++q) nv += v[q].x != ~0ULL;
        uint32_t sl = pd_home(v[0].x, ts), probes = 0;
        while (__any_sync(kFull, nv > 0)) {
          uint32_t rep = kNone, rs = 0;
          if (nv > 0) {
            bool done = pd_probe(tab, ts, v[0], sl, &rep, &rs);
            if (!done && ++probes >= ts) {  // every slot probed: no room
              full = true;
              done = true;
            }
            if (done) {
              --nv;
#pragma unroll
              for (int q = 0; q + 1 < kPdDedupPer; ++q) v[q] = v[q + 1];
              sl = pd_home(v[0].x, ts);
              probes = 0;
            } else {
              sl = sl + 1 == ts ? 0 : sl + 1;
            }
          }
          pd_list_push(rep, rs, list, &s_nlist);
        }
#pragma unroll
        for (int q = 0; q < kPdDedupPer; ++q) v[q] = w[q];
        if (!more) break;
      }
      if (full) raise_err(a.st, kErrTableFull);
      __syncthreads();
      const uint32_t nl = s_nlist;
      if (nl <= kPdList) {
        for (uint32_t x = threadIdx.x; x < nl; x += kPdDedupThreads) {
          const uint2 rp = list[x];
          const uint32_t m = reinterpret_cast<const uint32_t*>(&tab[rp.y])[3];
          if (m < rp.x && rp.x < a.n_ub) pd_repeat(a.slot_of, a.bits, rp.x, m);
        }
      } else {  // more repeats than the list holds: look every record up again
        for (uint32_t c = b; c < e; c += kChunk) {
          ulonglong2 r[kPdDedupPer];
#pragma unroll
          for (int q = 0; q < kPdDedupPer; ++q) {
            const uint32_t x = c + q * kPdDedupThreads + threadIdx.x;
            r[q] = x < e ? __ldcg(&a.rec2[x]) : empty;
          }
#pragma unroll
          for (int q = 0; q < kPdDedupPer; ++q) {
            if (r[q].x == ~0ULL) continue;
            const uint32_t i = (uint32_t)(r[q].y >> 32), m = pd_find(tab, ts, r[q]);
            if (m < i && i < a.n_ub) pd_repeat(a.slot_of, a.bits, i, m);
          }
        }
      }
      __syncthreads();
    }
    p = pn;
    b = bn;
    e = en;
  }
}

// ids after the partitioned dedup: ubits marks the settled accesses, bits
// their first occurrences; a settled access that is not a first occurrence
// (a repeat) finds its first occurrence in slot_of.  Matched accesses are
// left to k_ids_follow.
__global__ void __launch_bounds__(kGaThreads) k_ids_gather_pd(const uint32_t* __restrict__ slot_of,
                                                             const uint32_t* __restrict__ ubits,
                                                             const uint32_t* __restrict__ bits,
                                                             const uint32_t* __restrict__ wpre, uint32_t n_ub,
                                                             const uint64_t* n_dev, uint32_t* __restrict__ ids) {
  grid_dep_sync();
  const uint32_t n = keys_used(n_ub, n_dev);
  const uint32_t i0 = blockIdx.x * (kGaThreads * kGaPer) + threadIdx.x;
  uint32_t f[kGaPer], own[kGaPer], uw[kGaPer];
  // the three words of every access are read together (slot_of whether or
  // not the access turns out to be a repeat: one coalesced stream)
#pragma unroll
  for (int k = 0; k < kGaPer; ++k) {
    const uint32_t i = i0 + k * kGaThreads;
    uw[k] = i < n ? __ldg(&ubits[i >> 5]) : 0u;
    own[k] = i < n ? bits[i >> 5] : 0u;
    f[k] = i < n ? __ldcs(&slot_of[i]) : 0u;
  }
#pragma unroll
  for (int k = 0; k < kGaPer; ++k) {
    const uint32_t i = i0 + k * kGaThreads;
    if (!((uw[k] >> (i & 31)) & 1u))
      f[k] = kMatchedSlot;
    else if ((own[k] >> (i & 31)) & 1u)
      f[k] = i;
  }
  uint32_t wp[kGaPer], bw[kGaPer];
#pragma unroll
  for (int k = 0; k < kGaPer; ++k) {
    const uint32_t i = i0 + k * kGaThreads;
    const bool ok = f[k] < n;
    wp[k] = ok ? wpre[f[k] >> 5] : 0u;
    bw[k] = f[k] == i ? own[k] : ok ? bits[f[k] >> 5] : 0u;
  }
#pragma unroll
  for (int k = 0; k < kGaPer; ++k) {
    const uint32_t i = i0 + k * kGaThreads;
    if (i < n && f[k] != kMatchedSlot) ids[i] = f[k] < n ? wp[k] + __popc(bw[k] & ((1u << (f[k] & 31)) - 1u)) : kNone;
  }
}

// Slots for n keys at most: the full table holds 1.5 n.  The first attempt
// holds n / 3 while that is at most 2^22 slots (64 MB, half of L2): traces
// that repeat most blocks fill it well below half, and it stays in L2.  A
// larger table lives in DRAM whatever its size, so there the first attempt
// takes 3n / 4 slots instead: a trace that repeats few blocks (an agentic
// trace, D near n / 2) then probes a table at most about half full rather
// than one near 90% full, whose linear probe runs are tens of slots long.  If
// a probe sequence of the first attempt runs past kSmallProbeCap slots, the
// call redoes the stage with the full table.
constexpr uint64_t kSmallProbeCap = 4096;
constexpr uint32_t kL2TableLog2 = 22;
uint32_t table_log2(uint64_t want) {
  uint32_t l = 10;
  while ((1ULL << l) < want) ++l;
  return l;
}
uint32_t full_table_log2(uint64_t n) { return table_log2(n + n / 2 + 64); }
uint32_t small_table_log2(uint64_t n) {
  const uint32_t l = table_log2(n / 3 + 64);
  return l <= kL2TableLog2 ? l : table_log2(n / 4 * 3 + 64);
}

struct IdsLayout {
  DevStatus* st;
  uint32_t* done;
  ulonglong2* table;
  uint32_t* slot_of;  // per access: its slot, or kMatched (partitioned: a repeat's first occurrence)
  uint32_t *bits, *wpre, *tcnt, *tpre;  // first-occurrence bitmap and its ranks
  uint32_t* lam;               // prior hint: first unmatched depth of each request
  uint32_t* tile_req;          // prior hint: request of every 2048th access
  // partitioned dedup (null without it): level-1 counts and their prefix,
  // bucket bounds and level-2 tiles, partition totals, bounds and cursors,
  // and the records of both levels (in the table's region)
  uint32_t *pd_ubits, *pd_cnt1, *pd_off1, *pd_tot1, *pd_tot2, *pd_rel2, *pd_base2;
  ulonglong2 *pd_rec1, *pd_rec2;
  uint32_t pd_max_tiles;
  uint32_t nwords;
  size_t zero_bytes;
  size_t total;
  uint32_t log2m;
};

IdsLayout ids_layout(void* ws, uint64_t n, uint32_t n_req_hint, bool pd) {
  IdsLayout L;
  Carver cv(ws);
  L.log2m = full_table_log2(n);
  const uint64_t m = 1ULL << L.log2m;
  const uint64_t nn = n ? n : 1;
  L.nwords = ceil_div_u32(nn, 32);
  L.st = cv.take<DevStatus>(1);
  L.done = cv.take<uint32_t>(64);
  L.pd_tot2 = pd ? cv.take<uint32_t>(kPdParts) : nullptr;  // zeroed with the status block
  L.zero_bytes = cv.off;
  L.slot_of = cv.take<uint32_t>(nn);
  L.bits = cv.take<uint32_t>(L.nwords + 1);
  L.wpre = cv.take<uint32_t>(L.nwords + 1);
  L.tcnt = cv.take<uint32_t>(rank_tiles(L.nwords) + 1);
  L.tpre = cv.take<uint32_t>(rank_tiles(L.nwords) + 1);
  L.lam = n_req_hint ? cv.take<uint32_t>(n_req_hint) : nullptr;
  L.tile_req = n_req_hint ? cv.take<uint32_t>((nn >> kReqTileLog2) + 2) : nullptr;
  L.pd_max_tiles = ceil_div_u32(nn, kPdTile2) + kPdBuckets;
  L.pd_ubits = pd ? cv.take<uint32_t>(L.nwords + 1) : nullptr;
  L.pd_cnt1 = pd ? cv.take<uint32_t>(kPdBuckets * kPdMaxG1) : nullptr;
  L.pd_off1 = pd ? cv.take<uint32_t>(kPdBuckets * kPdMaxG1) : nullptr;
  L.pd_tot1 = pd ? cv.take<uint32_t>(kPdBuckets) : nullptr;
  L.pd_rel2 = pd ? cv.take<uint32_t>((size_t)L.pd_max_tiles * 256) : nullptr;
  L.pd_base2 = pd ? cv.take<uint32_t>(kPdParts + 1) : nullptr;
  // the table last: it starts past every other array of the stage (and past
  // stage a1's workspace, which the pipeline checks before it has stage a1
  // fill the table); the partitioned dedup keeps its records there
  L.table = cv.take<ulonglong2>(pd && 2 * nn > m ? 2 * nn : m);
  L.pd_rec1 = pd ? L.table : nullptr;
  L.pd_rec2 = pd && L.table ? L.table + nn : nullptr;
  L.total = cv.bytes();
  return L;
}

// Which dedup a first attempt takes: the partitioned one when asked, or (the
// default) when the table would not fit in L2.
bool ids_partitioned(uint64_t n, int method) {
  return method == PTC_IDS_PARTITIONED || (method == PTC_IDS_AUTO && ids_table_in_dram(n));
}

// ---------------------------------------------------------------- verify
__global__ void k_verify_first(const uint32_t* __restrict__ ids, uint64_t n, uint64_t D, uint32_t* first,
                               DevStatus* st) {
  grid_dep_sync();
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
  grid_dep_sync();
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

extern "C" size_t ptc_assign_ids_workspace_bytes(uint64_t n) {
  return ids_layout(nullptr, n, 0, ids_partitioned(n, PTC_IDS_AUTO)).total;
}

ptc_status ptc::ids_impl(const ptc_u128* keys, uint64_t n, const uint64_t* n_dev, uint32_t* ids_out,
                        uint64_t* n_used_host_out, uint64_t* n_distinct_host_out, void* ws, size_t ws_bytes,
                        cudaStream_t s, const uint32_t* carry_err, uint32_t n_carry, const KeyCarry* kc,
                        uint64_t* nd_slot, uint32_t* err_slot, bool full_table, const IdsHint* hint, int method) {
  if (hint && (hint->n_req == 0 || !hint->blk_off || !hint->prior)) return PTC_ERR_INVALID_ARG;
  if (kc && (kc->tile_blocks == 0 || (kc->tile_blocks & (kc->tile_blocks - 1)) != 0)) return PTC_ERR_INVALID_ARG;
  if (method != PTC_IDS_AUTO && method != PTC_IDS_TABLE && method != PTC_IDS_PARTITIONED) return PTC_ERR_INVALID_ARG;
  const InsCarry ic = kc ? InsCarry{kc->carry, kc->lead, (uint32_t)__builtin_ctz(kc->tile_blocks)}
                        : InsCarry{nullptr, nullptr, 0};
  if (n_distinct_host_out == nullptr) return PTC_ERR_INVALID_ARG;
  *n_distinct_host_out = 0;
  if (n_used_host_out) *n_used_host_out = 0;
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (n > 0 && (keys == nullptr || ids_out == nullptr)) return PTC_ERR_INVALID_ARG;
  const uint32_t hreq = hint ? hint->n_req : 0;
  const bool pd_layout = ids_partitioned(n, method);
  if (!ws_ok(ws, ws_bytes, ids_layout(nullptr, n, hreq, pd_layout).total)) return PTC_ERR_WORKSPACE;
  const IdsLayout L = ids_layout(ws, n, hreq, pd_layout);
  const PriorHint ph = hint ? PriorHint{hint->blk_off, hint->prior, hint->order, hint->pos, hint->n_req, L.lam, L.tile_req}
                            : PriorHint{nullptr, nullptr, nullptr, nullptr, 0, nullptr, nullptr};
  const bool pd = pd_layout && !full_table;  // the first attempt deduplicates by partitions
  // the status block, the table (all ones: empty; none for the partitioned
  // dedup) and the bitmaps are cleared by one launch
  auto start = [&](uint32_t log2m, bool table) -> bool {
    const bool fill_table = n > 0 && table;
    const FillRange zf[4] = {{ws, L.zero_bytes, 0u},
                            {L.table, fill_table ? sizeof(ulonglong2) << log2m : 0, ~0u},
                            {L.bits, n > 0 ? sizeof(uint32_t) * L.nwords : 0, 0u},
                            {L.pd_ubits, L.pd_ubits && n > 0 && !table ? sizeof(uint32_t) * L.nwords : 0, 0u}};
    return fill_many_async(zf, 4, s) == PTC_OK && carry_errors(carry_err, n_carry, L.st, s) == PTC_OK;
  };
  const ulonglong2* k = reinterpret_cast<const ulonglong2*>(keys);
  const uint32_t n32 = (uint32_t)n;
  auto hint_prep = [&]() {
    PTC_KERNEL("k_tile_req", s, k_tile_req, ceil_div_u32((n >> kReqTileLog2) + 2, 256), 256, 0, ph, n32, n_dev);
    PTC_KERNEL("k_ids_lam", s, k_ids_lam, ceil_div_u32(hint->n_req, kLamThreads), kLamThreads, 0, k, n32, n_dev, ic,
               ph, L.st);
  };
  // ranks of the first occurrences, the ids of the settled accesses, then
  // those of the matched ones
  auto finish = [&](const ulonglong2* table, uint64_t m) -> bool {
    if (bitmap_ranks(L.bits, L.nwords, L.wpre, L.tcnt, L.tpre, &L.done[0], &L.st->value[0], s) != PTC_OK)
      return false;
    if (table)
      PTC_KERNEL("k_ids_gather", s, k_ids_gather, ceil_div_u32(n, kGaThreads * kGaPer), kGaThreads, 0, L.slot_of,
                 table, m, L.bits, L.wpre, n32, n_dev, ids_out, L.st);
    else
      PTC_KERNEL("k_ids_gather", s, k_ids_gather_pd, ceil_div_u32(n, kGaThreads * kGaPer), kGaThreads, 0, L.slot_of,
                 L.pd_ubits, L.bits, L.wpre, n32, n_dev, ids_out);
    if (hint)
      if (ph.order)
        PTC_KERNEL("k_ids_follow", s, k_ids_follow_win, ceil_div_u32(hint->n_req, kFoThreads / 32), kFoThreads, 0,
                   ph, ids_out, L.st);
      else
        PTC_KERNEL("k_ids_follow", s, k_ids_follow, ceil_div_u32(hint->n_req, kFoThreads / 32), kFoThreads, 0, ph,
                   ids_out, L.st);
    return true;
  };
  auto run = [&](uint32_t log2m, uint64_t probe_cap) -> bool {
    if (hint) {
      hint_prep();
      PTC_KERNEL("k_ids_insert_prior", s, k_ids_insert_prior<kPriorK>, ceil_div_u32(n, kInsThreads * kPriorK),
                 kInsThreads, 0, k, n32, n_dev, L.table, log2m, probe_cap, L.slot_of, L.bits, L.st, ic, ph);
    } else {
      PTC_KERNEL("k_ids_insert", s, k_ids_insert, ceil_div_u32(n, kInsThreads * kInsK), kInsThreads, 0, k, n32, n_dev,
                 L.table, log2m, probe_cap, L.slot_of, L.bits, L.st, ic);
    }
    return finish(L.table, 1ULL << log2m);
  };
  auto run_pd = [&]() -> bool {
    if (hint) hint_prep();
    const uint32_t sms = (uint32_t)num_sms();
    uint32_t g1 = std::min(ceil_div_u32(n, kPdRound), std::min(4 * sms, kPdMaxG1));
    const uint32_t per = ceil_div_u32(ceil_div_u32(n, g1), kPdRound) * kPdRound;
    g1 = ceil_div_u32(n, per);
    if (cudaFuncSetAttribute(k_pd_scatter1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPdStageSmem) !=
            cudaSuccess ||
        cudaFuncSetAttribute(k_pd_level2<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPdStageSmem) !=
            cudaSuccess ||
        cudaFuncSetAttribute(k_pd_dedup, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPdDedupSmem) !=
            cudaSuccess)
      return false;
    PTC_KERNEL("k_pd_flags", s, k_pd_flags, hint ? ceil_div_u32(hint->n_req, 8) : ceil_div_u32(L.nwords, 256), 256,
               0, ph, n32, n_dev, L.pd_ubits, L.bits, L.nwords);
    const PdArgs pa{k, n32, n_dev, ic, ph, per, L.pd_cnt1, L.pd_off1, L.pd_tot1, L.pd_ubits, L.pd_rec1, L.st};
    PTC_KERNEL("k_pd_count", s, k_pd_count, g1, kPdThreads, 0, pa);
    PTC_KERNEL("k_pd_rows1", s, k_pd_rows1, kPdBuckets, 256, 0, L.pd_cnt1, g1, L.pd_off1, L.pd_tot1);
    PTC_KERNEL("k_pd_scatter1", s, k_pd_scatter1, g1, kPdThreads, kPdStageSmem, pa);
    const uint32_t g2 = std::min(L.pd_max_tiles, 4 * sms);
    const PdLevel2 p2{L.pd_rec1, L.pd_tot1, L.pd_tot2, L.pd_rel2, L.pd_base2, L.pd_rec2, n32, L.pd_max_tiles, L.st};
    PTC_KERNEL("k_pd_count2", s, k_pd_level2<false>, g2, kPd2Threads, 0, p2);
    PTC_KERNEL("k_pd_rows2", s, k_pd_rows2, kPdBuckets, 256, 0, L.pd_tot1, L.pd_tot2, L.pd_base2, L.st);
    PTC_KERNEL("k_pd_scatter2", s, k_pd_level2<true>, g2, kPd2Threads, kPdStageSmem, p2);
    PTC_KERNEL("k_pd_dedup", s, k_pd_dedup, std::min(kPdParts, 2 * sms), kPdDedupThreads, kPdDedupSmem,
               PdDedup{L.pd_rec2, L.pd_base2, n32, L.slot_of, L.bits, n32, L.st});
    return finish(nullptr, 0);
  };
  const uint32_t first_log2m = full_table ? L.log2m : small_table_log2(n);
  if (!start(first_log2m, !pd)) return PTC_ERR_CUDA;
  DevStatus h{};
  if (nd_slot && err_slot) {  // one attempt, nothing waits
    const uint32_t lg = first_log2m;
    if (n > 0 && !(pd ? run_pd() : run(lg, lg < L.log2m ? kSmallProbeCap : ~0ULL))) return PTC_ERR_CUDA;
    return defer_status(L.st, err_slot, s, nd_slot, 0, 2);
  }
  if (n > 0) {
    const uint32_t small = first_log2m;
    if (!(pd ? run_pd() : run(small, small < L.log2m ? kSmallProbeCap : ~0ULL))) return PTC_ERR_CUDA;
    if (pd || small < L.log2m) {
      const ptc_status rc1 = end_call(L.st, s, &h);
      // anything but a first attempt outrunning its table is final
      if (rc1 == PTC_OK || h.err != kErrTableFull) {
        *n_distinct_host_out = h.value[0];
        if (n_used_host_out) *n_used_host_out = h.value[1];
        return rc1;
      }
      // the first attempt's table overflowed: redo with the full one
      if (!start(L.log2m, true) || !run(L.log2m, ~0ULL)) return PTC_ERR_CUDA;
    }
  }
  const ptc_status rc = end_call(L.st, s, &h);
  *n_distinct_host_out = n ? h.value[0] : 0;
  if (n_used_host_out) *n_used_host_out = n ? h.value[1] : 0;
  return rc;
}

extern "C" ptc_status ptc_assign_ids(const ptc_u128* keys, uint64_t n, uint32_t* ids_out, uint64_t* n_distinct_host_out,
                                     void* ws, size_t ws_bytes, void* stream) {
  return ptc::ids_impl(keys, n, nullptr, ids_out, nullptr, n_distinct_host_out, ws, ws_bytes, (cudaStream_t)stream,
                       nullptr, 0);
}

bool ptc::ids_table_in_dram(uint64_t n) { return n / 3 + 64 > (1ULL << kL2TableLog2); }

size_t ptc::ids_ws_bytes(uint64_t n, uint32_t n_req_hint) {
  return ids_layout(nullptr, n, n_req_hint, ids_partitioned(n, PTC_IDS_AUTO)).total;
}

extern "C" size_t ptc_assign_ids_prior_workspace_bytes(uint64_t n, uint32_t n_req) {
  return ids_layout(nullptr, n, n_req ? n_req : 1, ids_partitioned(n, PTC_IDS_AUTO)).total;
}

extern "C" size_t ptc_assign_ids_ex_workspace_bytes(uint64_t n, uint32_t n_req, int method) {
  return ids_layout(nullptr, n, n_req, ids_partitioned(n, method)).total;
}

extern "C" ptc_status ptc_assign_ids_ex(const ptc_u128* keys, uint64_t n, const uint64_t* req_blk_off,
                                        const uint32_t* req_prior, uint32_t n_req, uint32_t* ids_out,
                                        uint64_t* n_distinct_host_out, int method, void* ws, size_t ws_bytes,
                                        void* stream) {
  if (n > 0 && n_req > 0 && (!req_blk_off || !req_prior)) return PTC_ERR_INVALID_ARG;
  const IdsHint h{req_blk_off, req_prior, n_req, nullptr, nullptr};
  return ptc::ids_impl(keys, n, nullptr, ids_out, nullptr, n_distinct_host_out, ws, ws_bytes, (cudaStream_t)stream,
                       nullptr, 0, nullptr, nullptr, nullptr, false, n > 0 && n_req > 0 ? &h : nullptr, method);
}

extern "C" ptc_status ptc_assign_ids_prior(const ptc_u128* keys, uint64_t n, const uint64_t* req_blk_off,
                                           const uint32_t* req_prior, uint32_t n_req, uint32_t* ids_out,
                                           uint64_t* n_distinct_host_out, void* ws, size_t ws_bytes, void* stream) {
  if (n > 0 && (n_req == 0 || !req_blk_off || !req_prior)) return PTC_ERR_INVALID_ARG;
  if (n == 0 || n_req == 0)
    return ptc::ids_impl(keys, n, nullptr, ids_out, nullptr, n_distinct_host_out, ws, ws_bytes,
                         (cudaStream_t)stream, nullptr, 0);
  const IdsHint h{req_blk_off, req_prior, n_req, nullptr, nullptr};
  return ptc::ids_impl(keys, n, nullptr, ids_out, nullptr, n_distinct_host_out, ws, ws_bytes, (cudaStream_t)stream,
                       nullptr, 0, nullptr, nullptr, nullptr, false, &h);
}

size_t ptc::session_prior_bytes(uint32_t n_req) {
  Carver cv(nullptr);
  cv.take<DevStatus>(1);
  cv.take<unsigned char>(sort_pairs_bytes(n_req ? n_req : 1));
  return cv.bytes();
}

// prior[r] = the previous request of r's session (kNone for a session's
// first request): a stable sort of the requests by session label, then one
// pass over neighbours.  Queued on `s`; a label >= n_session raises
// kErrInvalid into *err.
void ptc::session_prior(const uint32_t* req_session, uint32_t n_req, uint32_t n_session, uint32_t* prior, void* ws,
                        cudaStream_t s, uint32_t* err, uint32_t* order, uint32_t* pos) {
  Carver cv(ws);
  DevStatus* st = cv.take<DevStatus>(1);  // the sort has no bound to check and raises nothing
  void* sws = cv.take<unsigned char>(sort_pairs_bytes(n_req ? n_req : 1));
  uint32_t bits = 1;
  while (bits < 32 && (1ULL << bits) < n_session) ++bits;
  const uint32_t *ks = nullptr, *vs = nullptr;
  sort_pairs(req_session, nullptr, n_req, bits, sws, s, st, &ks, &vs);
  PTC_KERNEL("k_session_prior", s, k_session_prior, ceil_div_u32(n_req, 256), 256, 0, ks, vs, req_session, n_req,
             n_session, prior, err, order, pos);
}

extern "C" size_t ptc_session_prior_workspace_bytes(uint32_t n_req) {
  Carver cv(nullptr);
  cv.take<DevStatus>(1);
  cv.take<unsigned char>(session_prior_bytes(n_req));
  return cv.bytes();
}

extern "C" ptc_status ptc_session_prior(const uint32_t* req_session, uint32_t n_req, uint32_t n_session,
                                        uint32_t* prior_out, void* ws, size_t ws_bytes, void* stream) {
  if (n_req == 0) return PTC_OK;
  if (!req_session || !prior_out || n_session == 0) return PTC_ERR_INVALID_ARG;
  if (!ws_ok(ws, ws_bytes, ptc_session_prior_workspace_bytes(n_req))) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  Carver cv(ws);
  DevStatus* st = cv.take<DevStatus>(1);
  void* sws = cv.take<unsigned char>(session_prior_bytes(n_req));
  if (begin_call(ws, kStatusBytes, s) != PTC_OK) return PTC_ERR_CUDA;
  session_prior(req_session, n_req, n_session, prior_out, sws, s, &st->err, nullptr, nullptr);
  DevStatus h;
  return end_call(st, s, &h);
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
  if (fill_async(first, ~0u, sizeof(uint32_t) * (n_distinct ? n_distinct : 1), s) != PTC_OK)
    return PTC_ERR_CUDA;
  PTC_KERNEL("k_verify_first", s, k_verify_first, ceil_div_u32(n, 256), 256, 0, ids, n, n_distinct, first, st);
  PTC_KERNEL("k_verify", s, k_verify, ceil_div_u32(n, 256), 256, 0, tokens, n_tok, req_tok_off, req_blk_off, n_req, block_size, ids, n, n_distinct, first, st);
  DevStatus h;
  return end_call(st, s, &h);
}
