// Belady's offline optimum at every capacity of a grid at once (Sec. 3.2: the
// offline ceiling every eviction policy is compared with; App. A-B).
//
// Belady's MIN brings every accessed block in and, when the cache then holds
// more than C blocks, evicts the resident block (not the one just brought
// in) whose next access is farthest.  Its hits are reuses (prev[i], i) kept
// resident, and they are exactly the set this interval greedy picks: take
// the reuses in order of their end i; a cache of C blocks holds the block
// being accessed plus C - 1 kept blocks, so think of C - 1 tracks, each free
// from the last position it is busy at; reuse (p, i) is busy at p+1 .. i-1,
// hits iff some track is free by p, and then takes the track freed latest
// among those (best fit), which is free again from i - 1.  A reuse with
// p = i - 1 is busy nowhere and always hits.  (By end time with best fit,
// the greedy keeps the largest set of reuses with at most C - 1 of them busy
// at any access time -- Carlisle and Lloyd 1995 -- and that set is MIN's;
// the oracle's direct MIN simulation is the check.)
//
// Runs.  Accesses i .. i+L-1 whose previous accesses are p .. p+L-1 (a
// request re-reading a context) form a run.  With gap = i - p >= L, step k of
// a run takes the track freed at p + k if there is one (the latest free time
// <= p + k, since the tracks freed in [p, p + k) went to the earlier steps),
// else the latest free time below p, else a never-used track, else it
// misses; its track is then free from i - 1 + k.  So a run needs the free
// bits of [p, p + L), its number of other steps, that many of the latest free
// times below p, and the new free times of its hits.  If p + L = i, step 0's
// new free time i - 1 is the one step L - 1 looks for, handled on its own.  A
// run with gap < L is cut into pieces of length gap, which meet that case.
//
// One warp simulates one capacity: the free times are a bitmap over access
// positions with three summary levels (a bit per nonzero word, kept exact as
// words fill and empty) and a lower bound on the smallest free time, so a run
// with nothing free below p learns it at once; runs go in order, up to
// 1024 steps at a time, one 32-step word per lane.  Hits count with the
// prefix rule (Sec. 2.2): a request's accesses before its first miss.
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr uint32_t kBelStep = 1024;  // steps of a run simulated together (32 lanes x 32)

__device__ __forceinline__ uint32_t hi_bit(uint32_t v) { return 31u - __clz(v); }
__device__ __forceinline__ uint32_t mask_le(uint32_t b) { return b == 31 ? kFull : ((2u << b) - 1u); }
__device__ __forceinline__ uint32_t mask_lt(uint32_t b) { return b == 0 ? 0u : (kFull >> (32 - b)); }
// Position of the j-th lowest set bit of v (j = 0 is the lowest); v has more than j set bits.
__device__ __forceinline__ uint32_t nth_set(uint32_t v, uint32_t j) {
  for (uint32_t t = 0; t < j; ++t) v &= v - 1u;
  return (uint32_t)(__ffs(v) - 1);
}

// Request starts: one bit per access in `heads` and `rs`; offsets checked.
__global__ void k_bel_reqs(const uint64_t* __restrict__ blk_off, uint32_t R, uint64_t n, uint32_t* __restrict__ heads,
                           uint32_t* __restrict__ rs, DevStatus* st) {
  grid_dep_sync();
  const uint64_t r = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= R) return;
  const uint64_t a = blk_off[r], b = blk_off[r + 1];
  if (b < a || b > n || (r == 0 && a != 0) || (r + 1 == R && b != n)) {
    raise_err(st, kErrInvalid);
    return;
  }
  if (b > a) {
    atomicOr(&heads[a >> 5], 1u << (a & 31));
    atomicOr(&rs[a >> 5], 1u << (a & 31));
  }
}

// Run heads from prev: an access starts a run unless it and the one before
// are both cold, or both reuses with previous accesses one apart.
__global__ void k_bel_heads(const uint32_t* __restrict__ prev, uint32_t n, uint32_t* __restrict__ heads,
                            DevStatus* st) {
  grid_dep_sync();
  const uint32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  bool head = false;
  if (i < n) {
    const uint32_t p = prev[i], q = i ? prev[i - 1] : kNone;
    if (p != kNone && p >= i) raise_err(st, kErrInvalid);  // a previous access lies before
    head = i == 0 || (p == kNone) != (q == kNone) || (p != kNone && p != q + 1);
  }
  const uint32_t b = __ballot_sync(kFull, head);
  if ((threadIdx.x & 31) == 0 && b && i < n) atomicOr(&heads[i >> 5], b);
}

// Run records at the heads' ranks: first access, its previous access (kNone
// for a run of cold accesses), whether it opens a request; rec_start[runs] = n.
__global__ void k_bel_records(const uint32_t* __restrict__ prev, uint32_t n, const uint32_t* __restrict__ heads,
                              const uint32_t* __restrict__ rs, const uint32_t* __restrict__ wpre,
                              const uint64_t* __restrict__ nruns, uint32_t* __restrict__ rec_start,
                              uint32_t* __restrict__ rec_p, uint8_t* __restrict__ rec_rs) {
  grid_dep_sync();
  const uint32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) rec_start[*nruns] = n;
  if (i >= n) return;
  const uint32_t w = heads[i >> 5], bit = 1u << (i & 31);
  if (!(w & bit)) return;
  const uint32_t r = wpre[i >> 5] + __popc(w & (bit - 1u));
  rec_start[r] = i;
  rec_p[r] = prev[i];
  rec_rs[r] = (rs[i >> 5] & bit) ? 1 : 0;
}

struct BelCaps {
  uint64_t c[PTC_MAX_CAPACITIES];
};

struct BelArgs {
  const uint32_t* rec_start;
  const uint32_t* rec_p;
  const uint8_t* rec_rs;
  const uint64_t* nruns;
  uint32_t *lv0, *lv1, *lv2, *lv3;  // free-time bitmap and its summaries, one slice per capacity
  uint64_t s0, s1, s2, s3;          // words per slice
  uint32_t G;
  uint64_t alpha, beta;
  uint64_t* out;  // hits[G] | saved[G] (lo, hi) | raw hits[G]
  const DevStatus* st;
};

// One capacity's free-time bitmap: level 0 one bit per access position,
// level k + 1 one bit per nonzero word of level k.  `low` is a lower bound on
// every set position (raised when a search finds nothing below a point).
struct FreeBits {
  uint32_t *l0, *l1, *l2, *l3;
  uint64_t low;
  uint64_t words;     // level-0 words of the slice
  const DevStatus* st;

  __device__ void set_word(uint64_t w, uint32_t m) {
    if (!m || !in_bounds(st, w, words)) return;
    atomicOr(&l0[w], m);
    atomicOr(&l1[w >> 5], 1u << (w & 31));
    atomicOr(&l2[w >> 10], 1u << ((w >> 5) & 31));
    atomicOr(&l3[w >> 15], 1u << ((w >> 10) & 31));
  }
  // Clear bits m of word w; a word that becomes empty clears its summary
  // bit, and an emptied summary word its bit above (sets and clears of one
  // warp never overlap, so exactly one lane sees each word empty out).
  __device__ void clear_word(uint64_t w, uint32_t m) {
    if (!m || !in_bounds(st, w, words)) return;
    const uint32_t old = atomicAnd(&l0[w], ~m);
    if (old == 0 || (old & ~m) != 0) return;
    const uint32_t b1 = 1u << (w & 31);
    const uint32_t o1 = atomicAnd(&l1[w >> 5], ~b1);
    if (o1 == 0 || (o1 & ~b1) != 0) return;
    const uint32_t b2 = 1u << ((w >> 5) & 31);
    const uint32_t o2 = atomicAnd(&l2[w >> 10], ~b2);
    if (o2 != 0 && (o2 & ~b2) == 0) atomicAnd(&l3[w >> 15], ~(1u << ((w >> 10) & 31)));
  }
  // The highest set bit in words below w0, or -1.  Summary bits of words
  // found empty are cleared on the way.
  __device__ int64_t below_word(uint64_t w0) {
    uint64_t w1 = w0 >> 5;
    uint32_t m1 = __ldcg(&l1[w1]) & mask_lt((uint32_t)(w0 & 31));
    for (;;) {
      while (m1) {
        const uint32_t b = hi_bit(m1);
        const uint64_t ww = w1 * 32 + b;
        const uint32_t v = __ldcg(&l0[ww]);
        if (v) return (int64_t)(ww * 32 + hi_bit(v));
        atomicAnd(&l1[w1], ~(1u << b));
        m1 &= ~(1u << b);
      }
      uint64_t w2 = w1 >> 5;
      uint32_t m2 = __ldcg(&l2[w2]) & mask_lt((uint32_t)(w1 & 31));
      for (;;) {
        while (!m2) {  // the next nonzero level-2 word below w2, through level 3
          uint64_t w3 = w2 >> 5;
          uint32_t m3 = __ldcg(&l3[w3]) & mask_lt((uint32_t)(w2 & 31));
          while (!m3) {
            if (w3 == 0) return -1;
            --w3;
            m3 = __ldcg(&l3[w3]);
          }
          w2 = w3 * 32 + hi_bit(m3);
          m2 = __ldcg(&l2[w2]);
          if (!m2) atomicAnd(&l3[w3], ~(1u << (w2 & 31)));
        }
        const uint32_t b2 = hi_bit(m2);
        const uint64_t c1 = w2 * 32 + b2;
        const uint32_t mm = __ldcg(&l1[c1]);
        if (mm) {
          w1 = c1;
          m1 = mm;
          break;
        }
        atomicAnd(&l2[w2], ~(1u << b2));
        m2 &= ~(1u << b2);
      }
    }
  }
  // Clear the `need` highest set bits below position `pos`; returns how many
  // there were (fewer if the bitmap runs out).
  __device__ uint32_t pop_below(uint64_t pos, uint32_t need) {
    uint32_t got = 0;
    while (got < need && pos > low) {
      const uint64_t w = (pos - 1) >> 5;
      uint32_t v = __ldcg(&l0[w]) & mask_le((uint32_t)((pos - 1) & 31));
      uint64_t ww = w;
      if (!v) {
        const int64_t b = below_word(w);
        if (b < 0) {  // nothing set below pos (and appends only go above p0)
          low = low > pos ? low : pos;
          break;
        }
        ww = (uint64_t)b >> 5;
        v = __ldcg(&l0[ww]);
      }
      const uint32_t cnt = __popc(v), take = cnt < need - got ? cnt : need - got;
      uint32_t m = v;
      if (take < cnt) {  // keep the lowest cnt - take bits
        m = v & ~mask_le(nth_set(v, cnt - take - 1));
      }
      clear_word(ww, m);
      got += take;
      pos = ww * 32;
    }
    return got;
  }
};

__device__ __forceinline__ void add128(uint64_t& lo, uint64_t& hi, uint64_t a_lo, uint64_t a_hi) {
  lo += a_lo;
  hi += a_hi + (lo < a_lo ? 1 : 0);
}
__device__ __forceinline__ void add_mul(uint64_t& lo, uint64_t& hi, uint64_t a, uint64_t b) {
  add128(lo, hi, a * b, __umul64hi(a, b));
}

// One warp per capacity (capacity g = global warp index).
__global__ void __launch_bounds__(32) k_bel_sim(BelArgs a, BelCaps caps) {
  grid_dep_sync();
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t g = blockIdx.x;
  if (g >= a.G) return;
  FreeBits fb{a.lv0 + g * a.s0, a.lv1 + g * a.s1, a.lv2 + g * a.s2, a.lv3 + g * a.s3, 0, a.s0, a.st};
  uint64_t free_inf = caps.c[g] - 1;  // never-used tracks (lane 0's copy is the one used)
  uint64_t hits = 0, raw = 0, sv_lo = 0, sv_hi = 0;
  uint32_t req_start = 0;
  bool missed = false;
  const uint64_t R = *a.nruns;
  for (uint64_t r0 = 0; r0 < R; r0 += 32) {
    const uint64_t rl = r0 + lane;
    const uint32_t my_s = rl <= R ? a.rec_start[rl] : 0u;
    const uint32_t my_p = rl < R ? a.rec_p[rl] : kNone;
    const uint32_t my_rs = rl < R ? a.rec_rs[rl] : 0u;
    const uint32_t end32 = r0 + 32 <= R ? a.rec_start[r0 + 32] : 0u;
    const uint32_t nr = R - r0 < 32 ? (uint32_t)(R - r0) : 32u;
    for (uint32_t t = 0; t < nr; ++t) {
      uint32_t s = __shfl_sync(kFull, my_s, t);
      const uint32_t e = t + 1 < 32 ? __shfl_sync(kFull, my_s, (t + 1) & 31) : end32;
      uint32_t p = __shfl_sync(kFull, my_p, t);
      if (__shfl_sync(kFull, my_rs, t)) {
        req_start = s;
        missed = false;
      }
      uint32_t L = e - s;
      if (p == kNone || p >= s) {  // cold accesses: misses, no track (p >= s is malformed, reported)
        missed = true;
        continue;
      }
      if (s - p == 1) {  // every step re-reads the block just accessed: busy nowhere, hits
        raw += L;
        if (!missed) {
          const uint64_t d0 = s - req_start;
          hits += L;
          add_mul(sv_lo, sv_hi, a.alpha, L);
          add_mul(sv_lo, sv_hi, a.beta, (uint64_t)L * d0 + (uint64_t)L * (L - 1) / 2);
        }
        continue;
      }
      while (L > 0) {
        const uint32_t gap = s - p;
        const uint32_t Lj = L < gap ? (L < kBelStep ? L : kBelStep) : (gap < kBelStep ? gap : kBelStep);
        // this lane's 32 steps: k = 32 lane .. 32 lane + 31
        const uint32_t k0 = 32 * lane;
        const uint32_t valid = k0 >= Lj ? 0u : (Lj - k0 >= 32 ? kFull : ((1u << (Lj - k0)) - 1u));
        const uint64_t q = (uint64_t)p + k0, w = q >> 5;
        const uint32_t sh = (uint32_t)(q & 31);
        uint32_t Bk = 0;
        if (valid && in_bounds(a.st, w + (sh ? 1 : 0), a.s0)) {
          const uint32_t lo = __ldcg(&fb.l0[w]);
          const uint32_t hi = sh ? __ldcg(&fb.l0[w + 1]) : 0u;
          Bk = (sh ? (lo >> sh) | (hi << (32 - sh)) : lo) & valid;
        }
        const bool edge = Lj >= 2 && (uint64_t)p + Lj == s;
        const uint32_t elane = (Lj - 1) >> 5, ebit = 1u << ((Lj - 1) & 31);
        uint32_t zm = ~Bk & valid;
        if (edge && lane == elane) zm &= ~ebit;  // step Lj - 1: decided by step 0 below
        const uint32_t zc = __popc(zm);
        uint32_t zx = zc;  // exclusive prefix of the zero counts
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(kFull, zx, o);
          if (lane >= (uint32_t)o) zx += y;
        }
        const uint32_t z = __shfl_sync(kFull, zx, 31);
        zx -= zc;
        // the non-B steps take the latest free times below p, then never-used tracks
        uint32_t acc = 0;
        if (lane == 0 && z > 0) {
          const uint32_t got = fb.pop_below(p, z);
          const uint64_t rest = z - got;
          const uint64_t inf = rest < free_inf ? rest : free_inf;
          free_inf -= inf;
          acc = got + (uint32_t)inf;
        }
        __syncwarp();
        acc = __shfl_sync(kFull, acc, 0);
        const bool acc0 = (__shfl_sync(kFull, Bk, 0) & 1u) || acc >= 1;
        uint32_t A;
        if (acc >= zx + zc) {
          A = valid;
        } else if (acc <= zx) {
          A = valid & ~zm;
        } else {
          const uint32_t first_rej = nth_set(zm, acc - zx);
          A = (valid & ~zm) | (zm & mask_lt(first_rej));
        }
        if (edge && lane == elane) A = acc0 ? (A | ebit) : (A & ~ebit);
        const uint32_t rej = valid & ~A;
        const uint32_t my_f = rej ? k0 + (uint32_t)(__ffs(rej) - 1) : Lj;
        uint32_t f = my_f, nh = __popc(A);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const uint32_t of = __shfl_xor_sync(kFull, f, o);
          f = of < f ? of : f;
          nh += __shfl_xor_sync(kFull, nh, o);
        }
        // new free times s - 1 + k of the hits, then the free times of [p, p + Lj) are used up
        if (A) {
          const uint64_t q2 = (uint64_t)s - 1 + k0, w2 = q2 >> 5;
          const uint32_t sh2 = (uint32_t)(q2 & 31);
          fb.set_word(w2, A << sh2);
          if (sh2) fb.set_word(w2 + 1, A >> (32 - sh2));
        }
        __syncwarp();
        if (valid) {
          fb.clear_word(w, valid << sh);
          if (sh) fb.clear_word(w + 1, valid >> (32 - sh));
        }
        __syncwarp();
        raw += nh;
        if (!missed) {
          const uint64_t d0 = s - req_start;
          hits += f;
          add_mul(sv_lo, sv_hi, a.alpha, f);
          add_mul(sv_lo, sv_hi, a.beta, (uint64_t)f * d0 + (uint64_t)f * (f ? f - 1 : 0) / 2);
          if (f < Lj) missed = true;
        }
        s += Lj;
        p += Lj;
        L -= Lj;
      }
    }
  }
  if (lane == 0) {
    a.out[g] = hits;
    a.out[a.G + 2 * g] = sv_lo;
    a.out[a.G + 2 * g + 1] = sv_hi;
    a.out[3 * a.G + g] = raw;
  }
}

struct BelLayout {
  DevStatus* st;
  uint32_t* done;
  uint32_t *heads, *rs;  // zeroed with the status block
  uint32_t *wpre, *tcnt, *tpre;
  uint64_t* nruns;
  uint32_t *rec_start, *rec_p;
  uint8_t* rec_rs;
  uint32_t *lv0, *lv1, *lv2, *lv3;
  uint64_t s0, s1, s2, s3;
  uint64_t* out;
  size_t zero_bytes, bits_bytes;
  uint32_t nwords;
  size_t total;
};

BelLayout bel_layout(void* ws, uint64_t n, uint32_t n_cap) {
  BelLayout L;
  Carver cv(ws);
  const uint64_t nn = n ? n : 1;
  L.nwords = ceil_div_u32(nn, 32);
  L.st = cv.take<DevStatus>(1);
  L.done = cv.take<uint32_t>(64);
  L.heads = cv.take<uint32_t>(L.nwords + 1);
  L.rs = cv.take<uint32_t>(L.nwords + 1);
  L.zero_bytes = cv.off;
  L.wpre = cv.take<uint32_t>(L.nwords + 1);
  L.tcnt = cv.take<uint32_t>(rank_tiles(L.nwords) + 1);
  L.tpre = cv.take<uint32_t>(rank_tiles(L.nwords) + 1);
  L.nruns = cv.take<uint64_t>(1);
  L.rec_start = cv.take<uint32_t>(nn + 1);
  L.rec_p = cv.take<uint32_t>(nn);
  L.rec_rs = cv.take<uint8_t>(nn);
  const uint64_t G = n_cap ? n_cap : 1;
  L.s0 = (uint64_t)L.nwords + 2;
  L.s1 = (L.s0 + 31) / 32 + 1;
  L.s2 = (L.s1 + 31) / 32 + 1;
  L.s3 = (L.s2 + 31) / 32 + 1;
  L.lv0 = cv.take<uint32_t>((L.s0 + L.s1 + L.s2 + L.s3) * G);
  L.lv1 = L.lv0 + L.s0 * G;
  L.lv2 = L.lv1 + L.s1 * G;
  L.lv3 = L.lv2 + L.s2 * G;
  L.bits_bytes = sizeof(uint32_t) * (L.s0 + L.s1 + L.s2 + L.s3) * G;
  L.out = cv.take<uint64_t>(4 * G);
  L.total = cv.bytes();
  return L;
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_belady_curves_workspace_bytes(uint64_t n, uint32_t n_req, uint32_t n_cap) {
  (void)n_req;
  return bel_layout(nullptr, n, n_cap).total;
}

extern "C" ptc_status ptc_belady_curves(const uint32_t* prev, uint64_t n, const uint64_t* req_blk_off,
                                        uint32_t n_req, uint32_t block_size, const ptc_cost_model* cm,
                                        const uint64_t* cap_host, uint32_t n_cap, uint64_t* hits_host_out,
                                        ptc_u128* saved_host_out, uint64_t* raw_hits_host_out, void* ws,
                                        size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (!cm || !cap_host || !hits_host_out || !saved_host_out) return PTC_ERR_INVALID_ARG;
  if (n_cap < 1 || n_cap > PTC_MAX_CAPACITIES) return PTC_ERR_INVALID_ARG;
  if (block_size < 1 || block_size > PTC_MAX_BLOCK_SIZE) return PTC_ERR_INVALID_ARG;
  if (n > 0 && (!prev || !req_blk_off || n_req == 0)) return PTC_ERR_INVALID_ARG;
  for (uint32_t g = 0; g < n_cap; ++g)
    if (cap_host[g] < 1 || (g && cap_host[g] <= cap_host[g - 1])) return PTC_ERR_INVALID_ARG;
  uint64_t alpha = 0, beta = 0;
  const ptc_status crc = cost_coeffs(cm, block_size, &alpha, &beta);
  if (crc != PTC_OK) return crc;
  if (!ws_ok(ws, ws_bytes, bel_layout(nullptr, n, n_cap).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const BelLayout L = bel_layout(ws, n, n_cap);
  if (n == 0) {
    for (uint32_t g = 0; g < n_cap; ++g) {
      hits_host_out[g] = 0;
      saved_host_out[g] = ptc_u128{0, 0};
      if (raw_hits_host_out) raw_hits_host_out[g] = 0;
    }
    return PTC_OK;
  }
  const FillRange zf[2] = {{ws, L.zero_bytes, 0u}, {L.lv0, L.bits_bytes, 0u}};
  if (fill_many_async(zf, 2, s) != PTC_OK) return PTC_ERR_CUDA;
  const uint32_t n32 = (uint32_t)n;
  PTC_KERNEL("k_bel_reqs", s, k_bel_reqs, ceil_div_u32(n_req, 256), 256, 0, req_blk_off, n_req, n, L.heads, L.rs,
             L.st);
  PTC_KERNEL("k_bel_heads", s, k_bel_heads, ceil_div_u32(n, 256), 256, 0, prev, n32, L.heads, L.st);
  if (bitmap_ranks(L.heads, L.nwords, L.wpre, L.tcnt, L.tpre, L.done, L.nruns, s) != PTC_OK) return PTC_ERR_CUDA;
  PTC_KERNEL("k_bel_records", s, k_bel_records, ceil_div_u32(n, 256), 256, 0, prev, n32, L.heads, L.rs, L.wpre,
             L.nruns, L.rec_start, L.rec_p, L.rec_rs);
  BelArgs a;
  a.rec_start = L.rec_start;
  a.rec_p = L.rec_p;
  a.rec_rs = L.rec_rs;
  a.nruns = L.nruns;
  a.lv0 = L.lv0;
  a.lv1 = L.lv1;
  a.lv2 = L.lv2;
  a.lv3 = L.lv3;
  a.s0 = L.s0;
  a.s1 = L.s1;
  a.s2 = L.s2;
  a.s3 = L.s3;
  a.G = n_cap;
  a.alpha = alpha;
  a.beta = beta;
  a.out = L.out;
  a.st = L.st;
  BelCaps caps;
  for (uint32_t g = 0; g < n_cap; ++g) caps.c[g] = cap_host[g];
  PTC_KERNEL("k_bel_sim", s, k_bel_sim, n_cap, 32, 0, a, caps);
  HostStage* hs = host_stage();
  if (copy_to_host_async(hs->out, L.out, sizeof(uint64_t) * 3 * n_cap, s) != PTC_OK) return PTC_ERR_CUDA;
  if (raw_hits_host_out &&
      cudaMemcpyAsync(raw_hits_host_out, L.out + 3 * n_cap, sizeof(uint64_t) * n_cap, cudaMemcpyDeviceToHost, s) !=
          cudaSuccess)
    return PTC_ERR_CUDA;
  DevStatus h;
  const ptc_status rc = end_call(L.st, s, &h);
  if (rc != PTC_OK) return rc;
  for (uint32_t g = 0; g < n_cap; ++g) {
    hits_host_out[g] = hs->out[g];
    saved_host_out[g].lo = hs->out[n_cap + 2 * g];
    saved_host_out[g].hi = hs->out[n_cap + 2 * g + 1];
  }
  return PTC_OK;
}
