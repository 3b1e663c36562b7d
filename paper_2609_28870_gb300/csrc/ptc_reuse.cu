// Stage b over id-runs: previous / next use of every access, from a stable
// sort of runs of consecutive ids rather than of single accesses.
//
// An id-run is a maximal stretch of accesses whose ids go up by one from
// access to access (id-run r: positions [s_r, s_r + len_r) holding ids
// [x_r, x_r + len_r)).  Dense ids number blocks in order of first use, so a
// context read back block by block is a handful of id-runs: the conversational
// traces hold about a hundred accesses per id-run.
//
// Cut id-space at every run's first id and one past its last id: between two
// consecutive cuts (an elementary interval e) every id-run holds all of e or
// none of it.  For a fixed e, the runs holding it, in time order, are the
// successive uses of each id in e, so the previous use of id y in e by run r
// is y's place in the run just before r in that list (and the next use, in
// the run just after).  So one stable sort of the (e, r) incidences by e
// (run order is time order) gives prev and next of every access; on a trace
// without runs it is the sort of every (id, i).
//
//   k_ir_count     id-run starts per tile (ids < D checked); last CTA: prefixes
//                  (k_ir_count4: 16-byte loads when the ids are 16-byte aligned)
//   k_ir_mark      id-run records (start, first id) and the cuts, as a bitmap
//                  over [0, D]
//   k_bm_count / k_bm_words   ranks of the cuts (and the cut of each rank)
//   k_ir_inc1      elementary intervals per run; last CTA: prefixes and K
//   k_ir_inc2      the K incidences (e, r)
//   (sort_pairs)   stable radix sort of the incidences by e
//   k_ir_links     the first access of each incidence's neighbours on its e
//   k_ir_fill      prev / next of every access, written in position order
//
// When the incidences exceed a quarter of the accesses the stage falls back
// to sorting every access (ptc_sort.cu).
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kIT = 256;            // threads per tile
constexpr int kIR = 16;             // rounds of 32 positions per warp
constexpr int kITile = kIT * kIR;   // 4096 positions; warp w owns [512 w, 512 w + 512)
constexpr int kBmPer = 4;           // bitmap words per thread
constexpr int kBmTile = kIT * kBmPer;
constexpr int kRunPer = 8;          // runs per thread in the incidence kernels
constexpr int kRunTile = kIT * kRunPer;

struct IrArgs {
  const uint32_t* ids;
  uint32_t n, D, ntiles;  // with nd: n is an upper bound, and D and the used n come from nd
  const uint64_t* nd;     // device: nd[0] = D, nd[1] = accesses (stage a2 did not wait), or null
  const uint32_t* ext_err;  // device: stage a2's error word, reported in value[6], or null
  uint32_t* tcnt;
  uint32_t* tpre;     // runs before each tile; tpre[ntiles] = number of runs
  uint32_t* done;
  uint32_t* rec_s;    // start of each run (rec_s[R] = n)
  uint32_t* rec_x;    // first id of each run
  uint32_t* cut;      // bitmap over [0, D]: the cuts of id-space
  DevStatus* st;      // value[1] <- number of runs
};

// Exclusive prefix over the threads of a 256-thread CTA (total in *all).
__device__ __forceinline__ uint32_t cta_excl_u32(uint32_t x, uint32_t* s_w, uint32_t* all) {
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint32_t incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFull, incl, o);
    if (lane >= (uint32_t)o) incl += y;
  }
  __syncthreads();
  if (lane == 31) s_w[w] = incl;
  __syncthreads();
  uint32_t pre = 0, tot = 0;
#pragma unroll
  for (int ww = 0; ww < kIT / 32; ++ww) {
    const uint32_t v = s_w[ww];
    if (ww < (int)w) pre += v;
    tot += v;
  }
  *all = tot;
  return pre + incl - x;
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

// Run by the last CTA: exclusive prefix of cnt[0..T) into pre, pre[T] = total.
__device__ uint32_t tiles_prefix(const uint32_t* cnt, uint32_t* pre, uint32_t T, uint32_t* s_w) {
  (void)s_w;
  return cta_tiles_prefix(cnt, pre, T);
}

// Id-run starts of the warp's 8 x 32 positions from `base`, with the id left
// of each position.
__device__ __forceinline__ void id_starts(const IrArgs& a, uint32_t base, uint32_t lane, uint32_t (&id)[kIR],
                                          uint32_t (&left)[kIR], uint32_t (&words)[kIR], bool& bad) {
#pragma unroll
  for (int k = 0; k < kIR; ++k) {
    const uint32_t j = base + k * 32 + lane;
    id[k] = j < a.n ? a.ids[j] : 0u;
  }
  uint32_t carry = (lane == 0 && base > 0 && base - 1 < a.n) ? a.ids[base - 1] : 0u;
#pragma unroll
  for (int k = 0; k < kIR; ++k) {
    const uint32_t j = base + k * 32 + lane;
    const bool valid = j < a.n;
    if (valid && id[k] >= a.D) bad = true;
    const uint32_t up = __shfl_up_sync(kFull, id[k], 1);
    const uint32_t l = lane ? up : carry;
    carry = __shfl_sync(kFull, id[k], 31);
    left[k] = l;
    words[k] = __ballot_sync(kFull, valid && (j == 0 || id[k] != l + 1u));
  }
}

// n and D from the device when stage a2 did not wait for them.
__device__ __forceinline__ IrArgs resolved(const IrArgs& in) {
  IrArgs a = in;
  if (a.nd) {
    const uint64_t nn = a.nd[1], d = a.nd[0];
    a.n = nn < a.n ? (uint32_t)nn : a.n;
    a.D = d < a.n ? (uint32_t)d : a.n;
  }
  return a;
}

__global__ void __launch_bounds__(kIT) k_ir_count(IrArgs a0) {
  grid_dep_sync();
  __shared__ uint32_t s_w[kIT / 32];
  const IrArgs a = resolved(a0);
  if (a0.nd && blockIdx.x == 0 && threadIdx.x == 0) {
    a.st->value[4] = a0.nd[1];
    a.st->value[5] = a0.nd[0];
    a.st->value[6] = a0.ext_err ? *a0.ext_err : 0u;
  }
  const uint32_t tile = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint32_t id[kIR], left[kIR], words[kIR];
  bool bad = false;
  id_starts(a, tile * kITile + w * (32 * kIR), lane, id, left, words, bad);
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kIR; ++k) cnt += __popc(words[k]);
  if (bad) raise_err(a.st, kErrInvalid);
  uint32_t total;
  cta_excl_u32(lane == 0 ? cnt : 0u, s_w, &total);
  if (threadIdx.x == 0) a.tcnt[tile] = total;
  if (!last_cta(a.done)) return;
  const uint32_t R = tiles_prefix(a.tcnt, a.tpre, a.ntiles, s_w);
  if (threadIdx.x == 0) a.st->value[1] = R;
}

__global__ void __launch_bounds__(kIT) k_ir_mark(IrArgs a0) {
  grid_dep_sync();
  __shared__ uint32_t s_w[kIT / 32];
  const IrArgs a = resolved(a0);
  if (*(volatile uint32_t*)&a.st->err) return;  // ids >= D: reported, nothing is indexed by them
  const uint32_t tile = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t base = tile * kITile + w * (32 * kIR);
  uint32_t id[kIR], left[kIR], words[kIR];
  bool bad = false;
  id_starts(a, base, lane, id, left, words, bad);
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kIR; ++k) cnt += __popc(words[k]);
  uint32_t total;
  uint32_t run = a.tpre[tile] + cta_excl_u32(lane == 0 ? cnt : 0u, s_w, &total);
  run = __shfl_sync(kFull, run, 0);
#pragma unroll
  for (int k = 0; k < kIR; ++k) {
    const uint32_t j = base + k * 32 + lane;
    if ((words[k] >> lane) & 1u) {
      const uint32_t r = run + __popc(words[k] & lanemask_lt());
      a.rec_s[r] = j;
      a.rec_x[r] = id[k];
      atomicOr(&a.cut[id[k] >> 5], 1u << (id[k] & 31));
      if (j > 0) atomicOr(&a.cut[(left[k] + 1) >> 5], 1u << ((left[k] + 1) & 31));
    }
    if (j + 1 == a.n) {
      atomicOr(&a.cut[(id[k] + 1) >> 5], 1u << ((id[k] + 1) & 31));
      a.rec_s[a.tpre[a.ntiles]] = a.n;
    }
    run += __popc(words[k]);
  }
}

// ---- the counting pass with 16-byte loads (ids 16-byte aligned): lane l of
// warp w reads positions base + 128 k + 4 l .. + 3 (k < 4, base = the warp's
// 512 positions), one load per four accesses.
constexpr int kIR4 = kIR / 4;

__device__ __forceinline__ uint4 ir_load4(const uint32_t* __restrict__ v, uint32_t p, uint32_t n) {
  if (p + 4 <= n) return __ldcs(reinterpret_cast<const uint4*>(v + p));
  return make_uint4(p < n ? v[p] : 0u, p + 1 < n ? v[p + 1] : 0u, p + 2 < n ? v[p + 2] : 0u, p + 3 < n ? v[p + 3] : 0u);
}

// Id-run starts among positions p .. p + 3 as bits 0..3 (the id left of p is
// `il`), and whether an id is out of range.
__device__ __forceinline__ uint32_t id_starts4(const uint4 v, uint32_t il, uint32_t p, uint32_t n, uint32_t D,
                                               bool& bad) {
  const uint32_t iv[4] = {v.x, v.y, v.z, v.w};
  uint32_t x = 0, left = il;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const uint32_t j = p + e;
    if (j < n) {
      if (iv[e] >= D) bad = true;
      x |= (j == 0 || iv[e] != left + 1u ? 1u : 0u) << e;
    }
    left = iv[e];
  }
  return x;
}

__device__ __forceinline__ uint32_t warp_id_starts4(const IrArgs& a, uint32_t base, uint32_t lane, uint4 (&v)[kIR4],
                                                    uint32_t (&x)[kIR4], uint32_t (&il)[kIR4], bool& bad) {
#pragma unroll
  for (int k = 0; k < kIR4; ++k) v[k] = ir_load4(a.ids, base + 128 * k + 4 * lane, a.n);
  uint32_t carry = (base > 0 && base - 1 < a.n) ? a.ids[base - 1] : 0u;
  uint32_t cnt = 0;
#pragma unroll
  for (int k = 0; k < kIR4; ++k) {
    const uint32_t up = __shfl_up_sync(kFull, v[k].w, 1);
    il[k] = lane ? up : carry;
    carry = __shfl_sync(kFull, v[k].w, 31);
    x[k] = id_starts4(v[k], il[k], base + 128 * k + 4 * lane, a.n, a.D, bad);
    cnt += __popc(x[k]);
  }
  return cnt;
}

__global__ void __launch_bounds__(kIT) k_ir_count4(IrArgs a0) {
  grid_dep_sync();
  __shared__ uint32_t s_wcnt[kIT / 32];
  const IrArgs a = resolved(a0);
  if (a0.nd && blockIdx.x == 0 && threadIdx.x == 0) {
    a.st->value[4] = a0.nd[1];
    a.st->value[5] = a0.nd[0];
    a.st->value[6] = a0.ext_err ? *a0.ext_err : 0u;
  }
  const uint32_t tile = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint4 v[kIR4];
  uint32_t x[kIR4], il[kIR4];
  bool bad = false;
  const uint32_t cnt = __reduce_add_sync(kFull, warp_id_starts4(a, tile * kITile + w * (32 * kIR), lane, v, x, il, bad));
  if (lane == 0) s_wcnt[w] = cnt;
  if (bad) raise_err(a.st, kErrInvalid);
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t t = 0;
    for (int ww = 0; ww < kIT / 32; ++ww) t += s_wcnt[ww];
    a.tcnt[tile] = t;
  }
  if (!last_cta(a.done)) return;
  const uint32_t R = cta_tiles_prefix(a.tcnt, a.tpre, a.ntiles);
  if (threadIdx.x == 0) a.st->value[1] = R;
}

// Ranks of the cuts: per tile of kBmTile words the set bits, then (last CTA)
// tile prefixes; k_bm_words turns them into the cuts before every word and
// lists the cut of every rank.
__global__ void __launch_bounds__(kIT) k_bm_count(const uint32_t* __restrict__ bits, uint32_t nwords, uint32_t T,
                                                  uint32_t* tcnt, uint32_t* tpre, uint32_t* done, DevStatus* st) {
  grid_dep_sync();
  __shared__ uint32_t s_w[kIT / 32];
  const uint32_t w0 = blockIdx.x * kBmTile + threadIdx.x * kBmPer;
  uint32_t c = 0;
#pragma unroll
  for (int k = 0; k < kBmPer; ++k)
    if (w0 + k < nwords) c += __popc(bits[w0 + k]);
  uint32_t total;
  cta_excl_u32(c, s_w, &total);
  if (threadIdx.x == 0) tcnt[blockIdx.x] = total;
  if (!last_cta(done)) return;
  const uint32_t M = tiles_prefix(tcnt, tpre, T, s_w);
  if (threadIdx.x == 0) st->value[2] = M;
}

__global__ void __launch_bounds__(kIT) k_bm_words(const uint32_t* __restrict__ bits, uint32_t nwords,
                                                  const uint32_t* __restrict__ tpre, uint32_t* __restrict__ wpre,
                                                  uint32_t* __restrict__ cut_at) {
  grid_dep_sync();
  __shared__ uint32_t s_w[kIT / 32];
  const uint32_t w0 = blockIdx.x * kBmTile + threadIdx.x * kBmPer;
  uint32_t b[kBmPer], c = 0;
#pragma unroll
  for (int k = 0; k < kBmPer; ++k) {
    b[k] = w0 + k < nwords ? bits[w0 + k] : 0u;
    c += __popc(b[k]);
  }
  uint32_t total;
  uint32_t r = tpre[blockIdx.x] + cta_excl_u32(c, s_w, &total);
#pragma unroll
  for (int k = 0; k < kBmPer; ++k) {
    if (w0 + k < nwords) wpre[w0 + k] = r;
    for (uint32_t m = b[k]; m; m &= m - 1) cut_at[r++] = (w0 + k) * 32 + (__ffs(m) - 1);
  }
}

// Cuts at or below y, minus one: the elementary interval holding id y.
__device__ __forceinline__ uint32_t interval_of(const uint32_t* bits, const uint32_t* wpre, uint32_t y) {
  const uint32_t wi = y >> 5, b = y & 31;
  const uint32_t mask_le = b == 31 ? kFull : ((2u << b) - 1u);
  return wpre[wi] + __popc(bits[wi] & mask_le) - 1u;
}

struct IncArgs {
  const uint32_t* rec_s;
  const uint32_t* rec_x;
  const uint32_t* cut;
  const uint32_t* cwpre;
  const DevStatus* stc;     // value[1] = number of runs
  uint32_t* tcnt;
  uint32_t* tpre;
  uint32_t* done;
  const uint32_t* cut_at;   // id of every cut, by rank
  uint32_t* key;            // incidences: elementary interval
  uint32_t* val;            //             index in position order (the order written here)
  uint32_t* ipos;           // per incidence, in position order: its first access
  uint32_t* ilen;           //                                   and its accesses
  uint32_t max_tiles;       // tiles of tcnt / tpre
  DevStatus* st;            // value[3] <- K
};

// Intervals of run r: [first, end).
__device__ __forceinline__ void run_intervals(const IncArgs& a, uint32_t r, uint32_t& first, uint32_t& end) {
  const uint32_t x = a.rec_x[r], len = a.rec_s[r + 1] - a.rec_s[r];
  first = interval_of(a.cut, a.cwpre, x);
  end = interval_of(a.cut, a.cwpre, x + len - 1) + 1;
}

// Persistent over the run tiles (the number of runs is known on the device only).
__global__ void __launch_bounds__(kIT) k_ir_inc1(IncArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_w[kIT / 32];
  if (*(volatile const uint32_t*)&a.stc->err) return;  // the records are incomplete
  const uint32_t R = (uint32_t)a.stc->value[1];
  const uint32_t T = (R + kRunTile - 1) / kRunTile;
  for (uint32_t t = blockIdx.x; t < T; t += gridDim.x) {
    const uint32_t r0 = t * kRunTile + threadIdx.x * kRunPer;
    uint32_t c = 0;
#pragma unroll
    for (int k = 0; k < kRunPer; ++k) {
      if (r0 + k < R) {
        uint32_t f, e;
        run_intervals(a, r0 + k, f, e);
        c += e - f;
      }
    }
    uint32_t total;
    cta_excl_u32(c, s_w, &total);
    if (threadIdx.x == 0) a.tcnt[t] = total;
  }
  if (!last_cta(a.done)) return;
  const uint32_t K = tiles_prefix(a.tcnt, a.tpre, T < a.max_tiles ? T : a.max_tiles, s_w);
  if (threadIdx.x == 0) a.st->value[3] = K;
}

__global__ void __launch_bounds__(kIT) k_ir_inc2(IncArgs a, uint32_t R) {
  grid_dep_sync();
  __shared__ uint32_t s_w[kIT / 32];
  const uint32_t t = blockIdx.x;
  const uint32_t r0 = t * kRunTile + threadIdx.x * kRunPer;
  uint32_t f[kRunPer], e[kRunPer], c = 0;
#pragma unroll
  for (int k = 0; k < kRunPer; ++k) {
    f[k] = e[k] = 0;
    if (r0 + k < R) {
      run_intervals(a, r0 + k, f[k], e[k]);
      c += e[k] - f[k];
    }
  }
  uint32_t total;
  uint32_t o = a.tpre[t] + cta_excl_u32(c, s_w, &total);
#pragma unroll
  for (int k = 0; k < kRunPer; ++k) {
    if (f[k] == e[k]) continue;
    const uint32_t s0 = a.rec_s[r0 + k] - a.rec_x[r0 + k];  // the position of id y in the run is s0 + y
    uint32_t lo = a.cut_at[f[k]];
    for (uint32_t iv = f[k]; iv < e[k]; ++iv) {
      const uint32_t hi = a.cut_at[iv + 1];
      a.key[o] = iv;
      a.val[o] = o;
      a.ipos[o] = s0 + lo;
      a.ilen[o] = hi - lo;
      lo = hi;
      ++o;
    }
  }
}

struct FillArgs {
  const uint32_t* key;     // sorted incidences: elementary interval
  const uint32_t* val;     //                    index in position order
  uint32_t K, n;
  const uint32_t* ipos;    // per incidence in position order: first access, accesses
  const uint32_t* ilen;
  uint32_t* ip0;           // per incidence in position order: first access of the previous / next
  uint32_t* in0;           // incidence on the same interval, or none
  uint32_t* prev;
  uint32_t* next;
  const DevStatus* st;     // for the checked build's bounds checks
};

// For every incidence (e, r), the incidences on e before and after it in
// time are its neighbours in the order sorted by e (a stable sort of the
// incidences, written in run order, i.e. time order).  Their first accesses
// go to the incidence's place in position order.
__global__ void __launch_bounds__(256) k_ir_links(FillArgs a) {
  grid_dep_sync();
  const uint32_t q = blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= a.K) return;
  const uint32_t e = a.key[q], o = a.val[q];
  const uint32_t p = q > 0 && a.key[q - 1] == e ? a.ipos[a.val[q - 1]] : kNone;
  const uint32_t x = q + 1 < a.K && a.key[q + 1] == e ? a.ipos[a.val[q + 1]] : kNone;
  if (in_bounds(a.st, o, a.K)) {
    a.ip0[o] = p;
    a.in0[o] = x;
  }
}

// prev / next of every access, written in position order: the incidences in
// position order tile the accesses, so a warp takes 32 consecutive
// incidences (their records read with one coalesced load per array) and
// writes their accesses one incidence after another: each store of the warp
// covers consecutive accesses, and neighbouring incidences complete each
// other's sectors back to back.  The access at offset t of an incidence
// whose neighbours start at p0 / n0 has prev p0 + t and next n0 + t (ids and
// positions run in step inside an id-run).
__global__ void __launch_bounds__(256) k_ir_fill(FillArgs a) {
  grid_dep_sync();
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t warps = gridDim.x * (blockDim.x >> 5);
  for (uint32_t o0 = ((blockIdx.x * blockDim.x + threadIdx.x) >> 5) * 32; o0 < a.K; o0 += warps * 32) {
    const uint32_t o = o0 + lane;
    const bool live = o < a.K;
    const uint32_t S = live ? a.ipos[o] : 0u, Ln = live ? a.ilen[o] : 0u;
    const uint32_t P = live ? a.ip0[o] : kNone, X = live ? a.in0[o] : kNone;
    const uint32_t nq = a.K - o0 < 32u ? a.K - o0 : 32u;
    for (uint32_t i = 0; i < nq; ++i) {
      const uint32_t si = __shfl_sync(kFull, S, i), li = __shfl_sync(kFull, Ln, i);
      const uint32_t pi = __shfl_sync(kFull, P, i), xi = __shfl_sync(kFull, X, i);
      for (uint32_t t = lane; t < li; t += 32) {
        const uint32_t j = si + t;
        if (in_bounds(a.st, j, a.n)) {
          a.prev[j] = pi != kNone ? pi + t : kNone;
          a.next[j] = xi != kNone ? xi + t : kNone;
        }
      }
    }
  }
}

struct ReuseLayout {
  DevStatus* st;
  uint32_t* done;
  size_t zero_bytes;
  uint32_t *tcnt, *tpre, *rec_s, *rec_x;
  uint32_t *cut, *cwpre, *cut_at, *btcnt, *btpre;
  uint32_t *rtcnt, *rtpre;
  uint32_t *key, *val;
  uint32_t *ipos, *ilen, *ip0, *in0;  // per incidence in position order
  void* sort_ws;
  uint32_t ntiles, nwords, btiles, rtiles_max;
  uint64_t kcap;
  size_t total;
};

// Incidences the run path takes before it falls back to sorting every access
// (all of them when the run path is forced: there are at most n).
uint64_t incidence_cap(uint64_t n, bool forced) { return forced ? n + 64 : n / 4 + 64; }

ReuseLayout reuse_layout(void* ws, uint64_t n, uint64_t D, bool forced) {
  ReuseLayout L;
  Carver cv(ws);
  const uint64_t nn = n ? n : 1;
  L.ntiles = ceil_div_u32(nn, kITile);
  L.nwords = (uint32_t)((D + 1) / 32 + 1);
  L.btiles = ceil_div_u32(L.nwords, kBmTile);
  L.rtiles_max = ceil_div_u32(nn, kRunTile);
  L.kcap = incidence_cap(nn, forced);
  L.st = cv.take<DevStatus>(1);
  L.done = cv.take<uint32_t>(64);
  L.zero_bytes = cv.off;
  L.tcnt = cv.take<uint32_t>(L.ntiles + 1);
  L.tpre = cv.take<uint32_t>(L.ntiles + 1);
  L.rec_s = cv.take<uint32_t>(nn + 1);
  L.rec_x = cv.take<uint32_t>(nn);
  L.cut = cv.take<uint32_t>(L.nwords);
  L.cwpre = cv.take<uint32_t>(L.nwords);
  L.cut_at = cv.take<uint32_t>(D + 3);
  L.btcnt = cv.take<uint32_t>(L.btiles + 1);
  L.btpre = cv.take<uint32_t>(L.btiles + 1);
  L.rtcnt = cv.take<uint32_t>(L.rtiles_max + 1);
  L.rtpre = cv.take<uint32_t>(L.rtiles_max + 1);
  L.key = cv.take<uint32_t>(L.kcap);
  L.val = cv.take<uint32_t>(L.kcap);
  L.ipos = cv.take<uint32_t>(L.kcap);
  L.ilen = cv.take<uint32_t>(L.kcap);
  L.ip0 = cv.take<uint32_t>(L.kcap);
  L.in0 = cv.take<uint32_t>(L.kcap);
  L.sort_ws = cv.take<unsigned char>(sort_pairs_bytes(L.kcap));
  L.total = cv.bytes();
  return L;
}

uint32_t bits_for(uint64_t v) {  // bits to hold values below v
  uint32_t b = 1;
  while (b < 32 && (1ULL << b) < v) ++b;
  return b;
}

ptc_status reuse_by_runs(const uint32_t* ids, uint64_t n, uint64_t D, uint32_t* prev_out, uint32_t* next_out, void* ws,
                         size_t ws_bytes, cudaStream_t s, bool forced, uint32_t* defer_err = nullptr,
                         const ReuseDevIn* din = nullptr, ReuseHostOut* hout = nullptr) {
  const ReuseLayout L = reuse_layout(ws, n, D, forced);
  if (!ws_ok(ws, ws_bytes, L.total)) return PTC_ERR_WORKSPACE;
  const FillRange zf[2] = {{ws, L.zero_bytes, 0u}, {L.cut, sizeof(uint32_t) * L.nwords, 0u}};
  if (fill_many_async(zf, 2, s) != PTC_OK) return PTC_ERR_CUDA;
  IrArgs a;
  a.ids = ids;
  a.n = (uint32_t)n;
  a.D = (uint32_t)D;
  a.ntiles = L.ntiles;
  a.tcnt = L.tcnt;
  a.tpre = L.tpre;
  a.done = &L.done[0];
  a.rec_s = L.rec_s;
  a.rec_x = L.rec_x;
  a.cut = L.cut;
  a.st = L.st;
  a.nd = din ? din->nd : nullptr;
  a.ext_err = din ? din->ids_err : nullptr;
  // the count with 16-byte loads when the ids allow them (measured faster);
  // the marking pass stays one access per lane and round (the 16-byte form
  // of it measured slower: 0.77 against 0.70 ms on the mixed 10B-token trace)
  if ((reinterpret_cast<uintptr_t>(ids) & 15) == 0)
    PTC_KERNEL("k_ir_count", s, k_ir_count4, L.ntiles, kIT, 0, a);
  else
    PTC_KERNEL("k_ir_count", s, k_ir_count, L.ntiles, kIT, 0, a);
  PTC_KERNEL("k_ir_mark", s, k_ir_mark, L.ntiles, kIT, 0, a);
  PTC_KERNEL("k_bm_count", s, k_bm_count, L.btiles, kIT, 0, L.cut, L.nwords, L.btiles, L.btcnt, L.btpre, &L.done[1], L.st);
  PTC_KERNEL("k_bm_words", s, k_bm_words, L.btiles, kIT, 0, L.cut, L.nwords, L.btpre, L.cwpre, L.cut_at);
  IncArgs ia;
  ia.rec_s = L.rec_s;
  ia.rec_x = L.rec_x;
  ia.cut = L.cut;
  ia.cwpre = L.cwpre;
  ia.stc = L.st;
  ia.tcnt = L.rtcnt;
  ia.tpre = L.rtpre;
  ia.done = &L.done[2];
  ia.cut_at = L.cut_at;
  ia.key = L.key;
  ia.val = L.val;
  ia.ipos = L.ipos;
  ia.ilen = L.ilen;
  ia.max_tiles = L.rtiles_max;
  ia.st = L.st;
  const uint32_t g1 = L.rtiles_max < (uint32_t)(2 * num_sms()) ? L.rtiles_max : (uint32_t)(2 * num_sms());
  PTC_KERNEL("k_ir_inc1", s, k_ir_inc1, g1, kIT, 0, ia);
  DevStatus h{};
  ptc_status rc = end_call(L.st, s, &h);
  if (din) {  // n and D were bounds: the real ones, and stage a2's status, arrive with this wait
    hout->n = h.value[4];
    hout->D = h.value[5];
    hout->ids_err = (uint32_t)h.value[6];
    if (rc == PTC_ERR_CUDA) return rc;
    if (hout->ids_err) return PTC_OK;  // this stage's results are void; the caller redoes a2 and b
    n = hout->n;
    D = hout->D;
    if (rc == PTC_OK && (n == 0 || D == 0)) return PTC_OK;  // no accesses: nothing to link
  }
  if (rc != PTC_OK) return rc;
  const uint64_t R = h.value[1], M = h.value[2], K = h.value[3];
  if (K > L.kcap || R == 0 || M < 2) {
    if (forced) return PTC_ERR_WORKSPACE;  // cannot happen: K <= n
    return reuse_by_sort(ids, n, D, prev_out, next_out, ws, ws_bytes, s);
  }
  PTC_KERNEL("k_ir_inc2", s, k_ir_inc2, ceil_div_u32(R, kRunTile), kIT, 0, ia, (uint32_t)R);
  const uint32_t *skey = nullptr, *sval = nullptr;
  sort_pairs(L.key, L.val, (uint32_t)K, bits_for(M - 1), L.sort_ws, s, L.st, &skey, &sval);
  FillArgs f;
  f.key = skey;
  f.val = sval;
  f.K = (uint32_t)K;
  f.n = (uint32_t)n;
  f.ipos = L.ipos;
  f.ilen = L.ilen;
  f.ip0 = L.ip0;
  f.in0 = L.in0;
  f.prev = prev_out;
  f.next = next_out;
  f.st = L.st;
  PTC_KERNEL("k_ir_links", s, k_ir_links, ceil_div_u32(K, 256), 256, 0, f);
  const uint32_t fill_blocks = ceil_div_u32(K, 256) < (uint32_t)(8 * num_sms()) ? ceil_div_u32(K, 256)
                                                                                : (uint32_t)(8 * num_sms());
  PTC_KERNEL("k_ir_fill", s, k_ir_fill, fill_blocks, 256, 0, f);
  if (defer_err) return defer_status(L.st, defer_err, s);
  return end_call(L.st, s, &h);
}

}  // namespace

ptc_status reuse_view(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out, uint32_t* next_out,
                      void* ws, size_t ws_bytes, cudaStream_t s, uint32_t* defer_err, const ReuseDevIn* din,
                      ReuseHostOut* hout) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (n == 0) return PTC_OK;
  if (!ids || !prev_out || !next_out || n_distinct == 0 || n_distinct > n) return PTC_ERR_INVALID_ARG;
  if (din && !hout) return PTC_ERR_INVALID_ARG;
  return reuse_by_runs(ids, n, n_distinct, prev_out, next_out, ws, ws_bytes, s, false, defer_err, din, hout);
}

}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_reuse_indices_ex_workspace_bytes(uint64_t n, uint64_t n_distinct, int method) {
  const uint64_t D = n_distinct ? n_distinct : (n ? n : 1);
  const size_t by_sort = reuse_by_sort_bytes(n);
  if (method == PTC_REUSE_SORT) return by_sort;
  const size_t by_runs = reuse_layout(nullptr, n, D, method == PTC_REUSE_RUNS).total;
  if (method == PTC_REUSE_RUNS) return by_runs;
  return by_sort > by_runs ? by_sort : by_runs;
}

extern "C" size_t ptc_reuse_indices_workspace_bytes(uint64_t n, uint64_t n_distinct) {
  return ptc_reuse_indices_ex_workspace_bytes(n, n_distinct, PTC_REUSE_AUTO);
}

extern "C" ptc_status ptc_reuse_indices_ex(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out,
                                           uint32_t* next_out, int method, void* ws, size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (method != PTC_REUSE_AUTO && method != PTC_REUSE_SORT && method != PTC_REUSE_RUNS) return PTC_ERR_INVALID_ARG;
  if (n == 0) return PTC_OK;
  if (!ids || !prev_out || !next_out || n_distinct == 0 || n_distinct > n) return PTC_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  if (method == PTC_REUSE_SORT) return reuse_by_sort(ids, n, n_distinct, prev_out, next_out, ws, ws_bytes, s);
  return reuse_by_runs(ids, n, n_distinct, prev_out, next_out, ws, ws_bytes, s, method == PTC_REUSE_RUNS);
}

extern "C" ptc_status ptc_reuse_indices(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev_out,
                                        uint32_t* next_out, void* ws, size_t ws_bytes, void* stream) {
  return ptc_reuse_indices_ex(ids, n, n_distinct, prev_out, next_out, PTC_REUSE_AUTO, ws, ws_bytes, stream);
}
