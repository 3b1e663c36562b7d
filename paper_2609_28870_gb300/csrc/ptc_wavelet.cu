// Stage c: LRU stack distance of every access (paper App. B, stack distance
// between reuses), as a 2-D dominance count on a wavelet matrix.
//
// For access i with previous use p = prev[i]:
//   SD_i - 1 = #distinct blocks in (p, i) = #{ j in (p, i) : prev[j] < p or prev[j] = none }
// because every block touched in (p, i) has exactly one access in that window
// whose previous use lies before p (its first access inside the window), and
// p's own block is not touched in (p, i).  With v_j = prev[j] + 1 (none -> 0)
// this is "count v_j < p + 1 for j in [p+1, i)": a range-rank query.
//
// Runs.  Adding the p + 1 positions j <= p (all have v_j < p + 1) turns the
// count into SD_i = #{ j < i : v_j < v_i } - p.  If prev[i] = prev[i-1] + 1
// then v_i = v_{i-1} + 1, the count grows by exactly one (the access i-1) and
// so does p: SD_i = SD_{i-1}.  Re-reads of a context copy it block by block,
// so such runs are long; only the first access of a run (a "head") runs a
// query and the rest of the run takes the head's value.
//
// Wavelet matrix (Claude, Navarro, Ordonez 2015) over v[0..N): L levels for
// values < 2^L.  Level l keeps one bit per position — bit (L-1-l) of the value
// at that position in level l's order — and level l+1's order is the stable
// partition of level l's order by that bit: its Z_l zeros, then its ones.
// Level l's order is therefore the stable sort of v by its top l bits read
// in reverse (the top bit least significant), so four levels are built per
// pass from one LSD radix-16 step on the reversed 4-bit digit.
//
// Layout of one level: a plain bitvector (LSB first) plus a rank directory of
// ones per 256-bit superblock (relative to its chunk of 256 superblocks) and
// per chunk; a rank reads the superblock's 32-byte sector and two counts.
//   k_wm_hist    per pass: tile histograms of the 4-bit key
//   k_wm_scan    per pass: tile prefixes and totals of every key
//   k_wm_pass    per pass: bits of 4 levels and the order after them
//   k_wm_dir     rank directories of all levels
//   k_wm_heads   run heads walk the L levels (early exit on an empty range)
//                and write their distances; tiles record their last head.
//   k_wm_propagate  every access takes the distance of the last head at or
//                before it (segmented scan; the carry comes from the tile
//                records, all written by the previous kernel).
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kWT = 256;                    // threads per tile
constexpr int kWR = 8;                      // elements per thread
constexpr int kWTile = kWT * kWR;           // 2048 positions per tile
constexpr int kWW = kWT / 32;               // warps per tile
constexpr int kWB = 4;                      // levels per pass
constexpr int kOwners = 30;                 // (k, key) for k = 1..4: 2 + 4 + 8 + 16
constexpr int kRegions = 14;                // (k, key) for k = 1..3
constexpr int kRegionWords = kWTile / 32 + 1;
constexpr int kSbBits = 256;                // rank-directory superblock
constexpr int kSbPerChunk = 256;
constexpr int kQThreads = 256;
constexpr int kQPer = 8;
constexpr int kQTile = kQThreads * kQPer;

// (k, key) pairs with k >= 1 numbered 2^k - 2 + key
__device__ __forceinline__ uint32_t owner_of(uint32_t k, uint32_t key) { return (1u << k) - 2u + key; }

struct PassArgs {
  const uint32_t* src;        // this pass's input order (prev itself on pass 0)
  int from_prev;              // values are prev + 1 (none -> 0)
  uint32_t* dst;              // the order after this pass (null on the last pass)
  uint32_t* bits;             // bitvectors, level l at bits + l * lw
  uint64_t lw;
  uint64_t n;
  uint32_t ntiles;
  uint32_t lvl0, r, sh;       // first level, levels in the pass, shift of the digit
  uint32_t* H;                // histogram of the pass key per tile, column-major [key][tile]
  uint32_t* T;                // exclusive prefix of H over tiles, same layout
  uint32_t* G;                // totals of the pass digit (16)
  uint32_t* done;             // CTAs finished (histogram kernel)
  unsigned long long* zcount; // Z_l for every level
  DevStatus* st;
};

__device__ __forceinline__ uint32_t load_v(const PassArgs& a, uint64_t j) {
  uint32_t x = a.src[j];
  if (a.from_prev) x = x == kNone ? 0u : x + 1u;
  return x;
}
// the r bits of levels lvl0 .. lvl0 + r - 1, reversed: bit k of the key is the
// bit of level lvl0 + k
__device__ __forceinline__ uint32_t key_of(uint32_t v, uint32_t sh, uint32_t r) {
  return __brev((v >> sh) & ((1u << r) - 1u)) >> (32 - r);
}

// Histogram of the pass keys per tile, stored column-major: H[key * ntiles + tile].
__global__ void __launch_bounds__(kWT) k_wm_hist(PassArgs a) {
  __shared__ uint32_t s_h[16];
  const uint32_t t = threadIdx.x, lane = t & 31;
  const uint64_t base = (uint64_t)blockIdx.x * kWTile;
  if (t < 16) s_h[t] = 0;
  __syncthreads();
  bool bad = false;
#pragma unroll
  for (int rd = 0; rd < kWR; ++rd) {
    const uint64_t j = base + (uint64_t)rd * kWT + t;
    const bool valid = j < a.n;
    uint32_t key = 0xFFFFu;
    if (valid) {
      if (a.from_prev) {
        const uint32_t p = a.src[j];
        if (p != kNone && (uint64_t)p >= j) bad = true;
      }
      key = key_of(load_v(a, j), a.sh, a.r);
    }
    const uint32_t peers = __match_any_sync(kFull, key);
    if (valid && lane == (uint32_t)(__ffs(peers) - 1)) atomicAdd(&s_h[key], (uint32_t)__popc(peers));
  }
  if (bad) raise_err(a.st, kErrInvalid);
  __syncthreads();
  if (t < 16) a.H[(uint64_t)t * a.ntiles + blockIdx.x] = s_h[t];
}

// One CTA per key: exclusive prefix of its histogram column over tiles, and
// the key's total.  Each thread takes a contiguous run of tiles.
constexpr int kScanThreads = 1024;
__global__ void __launch_bounds__(kScanThreads) k_wm_scan(PassArgs a) {
  __shared__ uint32_t s_w[kScanThreads / 32];
  const uint32_t key = blockIdx.x, t = threadIdx.x, lane = t & 31, w = t >> 5;
  if (key >= (1u << a.r)) {
    if (t == 0) a.G[key] = 0;
    return;
  }
  const uint32_t* col = a.H + (uint64_t)key * a.ntiles;
  uint32_t* out = a.T + (uint64_t)key * a.ntiles;
  const uint32_t per = (a.ntiles + kScanThreads - 1) / kScanThreads;
  const uint32_t lo = t * per < a.ntiles ? t * per : a.ntiles, hi = lo + per < a.ntiles ? lo + per : a.ntiles;
  uint32_t sum = 0;
  for (uint32_t i = lo; i < hi; ++i) sum += col[i];
  uint32_t x = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFull, x, o);
    if (lane >= (uint32_t)o) x += y;
  }
  if (lane == 31) s_w[w] = x;
  __syncthreads();
  uint32_t wpre = 0, tot = 0;
#pragma unroll 4
  for (int k = 0; k < kScanThreads / 32; ++k) {
    wpre += k < (int)w ? s_w[k] : 0u;
    tot += s_w[k];
  }
  uint32_t run = wpre + x - sum;
  for (uint32_t i = lo; i < hi; ++i) {
    out[i] = run;
    run += col[i];
  }
  if (t == 0) a.G[key] = tot;
}

// One pass = r levels.  Positions at level lvl0 + k are the stable order by
// the low k bits of the key (the level lvl0 bit least significant), so a tile
// of this pass's order lands, at level lvl0 + k, in 2^k runs (one per key),
// each contiguous.  Level lvl0's bits are ballots in place; the bits of levels
// lvl0 + 1 .. lvl0 + r - 1 are assembled per run in shared memory and written
// at the runs' global bit offsets (whole words stored, words shared with a
// neighbouring run OR-ed); the order after the pass is an LSD radix-2^r
// scatter by the full key.
__global__ void __launch_bounds__(kWT) k_wm_pass(PassArgs a) {
  __shared__ uint32_t s_reg[kRegions][kRegionWords];
  __shared__ uint32_t s_vals[kWTile];
  __shared__ uint32_t s_cnt[kWW][32];
  __shared__ uint32_t s_tot[32];
  __shared__ uint32_t s_run[32];
  __shared__ uint32_t s_lst[16];
  __shared__ uint32_t s_G[16], s_T[16];
  const uint32_t t = threadIdx.x, lane = t & 31, w = t >> 5;
  const uint32_t r = a.r;
  const uint32_t nown = (2u << r) - 2u;       // owners with k = 1..r
  const uint32_t nreg = r > 1 ? (2u << (r - 1)) - 2u : 0u;  // regions with k = 1..r-1
  const uint32_t tile = blockIdx.x;
  const uint64_t base = (uint64_t)tile * kWTile;
  for (uint32_t i = t; i < kRegions * kRegionWords; i += kWT) (&s_reg[0][0])[i] = 0;
  if (t < 16) {
    s_G[t] = a.G[t];
    s_T[t] = t < (1u << r) ? a.T[(uint64_t)t * a.ntiles + tile] : 0u;
  }
  uint32_t v[kWR];
#pragma unroll
  for (int rd = 0; rd < kWR; ++rd) {
    const uint64_t j = base + (uint64_t)w * (32 * kWR) + (uint64_t)rd * 32 + lane;
    v[rd] = j < a.n ? load_v(a, j) : 0u;
  }
  // this lane's (k, key) when it is an owner
  const bool own = lane < nown;
  uint32_t ok = 1, oc = 0;
  if (own) {
    while ((2u << ok) - 2u <= lane) ++ok;
    oc = lane - ((1u << ok) - 2u);
  }
  // ---- phase A: per-warp counts of every (k, key)
  uint32_t cnt = 0;
  uint32_t* bits0 = a.bits + (uint64_t)a.lvl0 * a.lw;
#pragma unroll
  for (int rd = 0; rd < kWR; ++rd) {
    const uint64_t j = base + (uint64_t)w * (32 * kWR) + (uint64_t)rd * 32 + lane;
    const uint32_t vm = __ballot_sync(kFull, j < a.n);
    const uint32_t key = key_of(v[rd], a.sh, r);
    uint32_t B[kWB];
#pragma unroll
    for (int i = 0; i < kWB; ++i) B[i] = (uint32_t)i < r ? __ballot_sync(kFull, (key >> i) & 1u) : 0u;
    if (lane == 0 && (vm & 1u)) bits0[(base + (uint64_t)w * (32 * kWR) + (uint64_t)rd * 32) >> 5] = B[0] & vm;
    if (own) {
      uint32_t m = vm;
#pragma unroll
      for (int i = 0; i < kWB; ++i)
        if ((uint32_t)i < ok) m &= ((oc >> i) & 1u) ? B[i] : ~B[i];
      cnt += __popc(m);
    }
  }
  if (own) s_cnt[w][lane] = cnt;
  __syncthreads();
  if (tile == 0 && t < r) {  // zeros of level lvl0 + t: keys whose bit t is 0
    uint64_t z = 0;
    for (uint32_t key = 0; key < (1u << r); ++key)
      if (!((key >> t) & 1u)) z += s_G[key];
    a.zcount[a.lvl0 + t] = z;
  }
  if (t < nown) {  // warp prefixes and tile totals
    uint32_t acc = 0;
    for (int ww = 0; ww < kWW; ++ww) {
      const uint32_t x = s_cnt[ww][t];
      s_cnt[ww][t] = acc;
      acc += x;
    }
    s_tot[t] = acc;
  }
  __syncthreads();
  if (t < nown) {  // global start of every run at level lvl0 + k
    uint32_t k = 1;
    while ((2u << k) - 2u <= t) ++k;
    const uint32_t c = t - ((1u << k) - 2u), msk = (1u << k) - 1u;
    uint32_t off = 0, pre = 0;
    for (uint32_t key = 0; key < (1u << r); ++key) {
      if ((key & msk) < c) off += s_G[key];
      if ((key & msk) == c) pre += s_T[key];
    }
    s_run[t] = off + pre;
    if (k == r) {  // local start of the final key group
      uint32_t ls = 0;
      for (uint32_t c2 = 0; c2 < c; ++c2) ls += s_tot[owner_of(r, c2)];
      s_lst[c] = ls;
    }
  }
  __syncthreads();
  // ---- phase B: ranks; bits of the middle levels into shared runs; reorder
  cnt = 0;
  const uint32_t lt = lanemask_lt();
#pragma unroll
  for (int rd = 0; rd < kWR; ++rd) {
    const uint64_t j = base + (uint64_t)w * (32 * kWR) + (uint64_t)rd * 32 + lane;
    const bool valid = j < a.n;
    const uint32_t vm = __ballot_sync(kFull, valid);
    const uint32_t key = key_of(v[rd], a.sh, r);
    uint32_t B[kWB];
#pragma unroll
    for (int i = 0; i < kWB; ++i) B[i] = (uint32_t)i < r ? __ballot_sync(kFull, (key >> i) & 1u) : 0u;
    uint32_t eq = vm;
#pragma unroll
    for (int k = 1; k <= kWB; ++k) {
      if ((uint32_t)k > r) break;
      eq &= ((key >> (k - 1)) & 1u) ? B[k - 1] : ~B[k - 1];
      const uint32_t kk = key & ((1u << k) - 1u);
      const uint32_t o = owner_of(k, kk);
      const uint32_t before = __shfl_sync(kFull, cnt, o);
      const uint32_t rank = s_cnt[w][o] + before + __popc(eq & lt);
      if (valid) {
        if ((uint32_t)k < r) {
          if ((key >> k) & 1u) atomicOr(&s_reg[o][rank >> 5], 1u << (rank & 31));
        } else {
          s_vals[s_lst[kk] + rank] = v[rd];
        }
      }
    }
    if (own) {
      uint32_t m = vm;
#pragma unroll
      for (int i = 0; i < kWB; ++i)
        if ((uint32_t)i < ok) m &= ((oc >> i) & 1u) ? B[i] : ~B[i];
      cnt += __popc(m);
    }
  }
  __syncthreads();
  // ---- the order after this pass
  const uint32_t tile_n = (uint32_t)(a.n - base < (uint64_t)kWTile ? a.n - base : kWTile);
  if (a.dst != nullptr) {
    for (uint32_t p = t; p < tile_n; p += kWT) {
      const uint32_t x = s_vals[p];
      const uint32_t key = key_of(x, a.sh, r);
      const uint32_t d = s_run[owner_of(r, key)] + (p - s_lst[key]);
      if ((uint64_t)d < a.n) a.dst[d] = x;  // in range on a well-formed input
    }
  }
  // ---- bit runs of levels lvl0 + 1 .. lvl0 + r - 1
  for (uint32_t rg = 0; rg < nreg; ++rg) {
    const uint32_t C = s_tot[rg];
    if (C == 0) continue;
    uint32_t k = 1;
    while ((2u << k) - 2u <= rg) ++k;
    const uint64_t S = s_run[rg];
    const uint64_t g0 = S >> 5, g1 = (S + C - 1) >> 5;
    uint32_t* lvl = a.bits + (uint64_t)(a.lvl0 + k) * a.lw;
    for (uint64_t g = g0 + t; g <= g1; g += kWT) {
      const int64_t q = (int64_t)(g * 32) - (int64_t)S;  // run offset of this word's bit 0
      uint32_t x;
      if (q < 0) {
        x = s_reg[rg][0] << (uint32_t)(-q);
      } else {
        const uint32_t w0 = (uint32_t)(q >> 5), sft = (uint32_t)(q & 31);
        x = s_reg[rg][w0] >> sft;
        if (sft) x |= s_reg[rg][w0 + 1] << (32 - sft);
      }
      const int64_t blo = q < 0 ? -q : 0, bhi = (int64_t)C - q < 32 ? (int64_t)C - q : 32;
      const uint32_t mask = (bhi >= 32 ? 0xFFFFFFFFu : ((1u << bhi) - 1u)) & ~((1u << blo) - 1u);
      x &= mask;
      if (mask == 0xFFFFFFFFu) {
        if (x) lvl[g] = x;
      } else if (x) {
        atomicOr(&lvl[g], x);
      }
    }
  }
}

// Rank directory of every level: dir[l][sb] = ones in the superblocks of its
// chunk before sb, csum[l][c] = ones in chunk c; the CTA that finishes last
// turns csum into cpre[l][c] = ones in the chunks before c.
__global__ void __launch_bounds__(kSbPerChunk) k_wm_dir(const uint32_t* __restrict__ bits, uint64_t lw, uint32_t L,
                                                        uint32_t nsb, uint32_t nchunk, uint32_t* __restrict__ dir,
                                                        uint32_t* csum, uint32_t* __restrict__ cpre, uint32_t* done) {
  __shared__ uint32_t s_w[kSbPerChunk / 32];
  __shared__ bool s_last;
  const uint32_t t = threadIdx.x, lane = t & 31, w = t >> 5;
  const uint32_t l = blockIdx.x / nchunk, ch = blockIdx.x % nchunk;
  const uint32_t sb = ch * kSbPerChunk + t;
  uint32_t ones = 0;
  if (sb < nsb) {
    const uint4* p = reinterpret_cast<const uint4*>(bits + (uint64_t)l * lw + (uint64_t)sb * 8);
    const uint4 x = p[0], y = p[1];
    ones = __popc(x.x) + __popc(x.y) + __popc(x.z) + __popc(x.w) + __popc(y.x) + __popc(y.y) + __popc(y.z) + __popc(y.w);
  }
  uint32_t xs = ones;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFull, xs, o);
    if (lane >= (uint32_t)o) xs += y;
  }
  if (lane == 31) s_w[w] = xs;
  __syncthreads();
  uint32_t wpre = 0, tot = 0;
  for (int k = 0; k < kSbPerChunk / 32; ++k) {
    wpre += k < (int)w ? s_w[k] : 0u;
    tot += s_w[k];
  }
  if (sb < nsb) dir[(uint64_t)l * nsb + sb] = wpre + xs - ones;
  if (t == 0) {
    csum[(uint64_t)l * nchunk + ch] = tot;
    __threadfence();
    s_last = atomicAdd(done, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (uint32_t lv = w; lv < L; lv += kSbPerChunk / 32) {  // one warp per level
    uint32_t run = 0;
    for (uint32_t c0 = 0; c0 < nchunk; c0 += 32) {
      const uint32_t c = c0 + lane;
      const uint32_t v = c < nchunk ? ld_relaxed_u32(&csum[(uint64_t)lv * nchunk + c]) : 0u;
      uint32_t x = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, x, o);
        if (lane >= (uint32_t)o) x += y;
      }
      if (c < nchunk) cpre[(uint64_t)lv * nchunk + c] = run + x - v;
      run += __shfl_sync(kFull, x, 31);
    }
  }
}

struct RankView {
  const uint32_t* bits;
  uint64_t lw;
  const uint32_t* dir;
  const uint32_t* cpre;
  uint32_t nsb, nchunk;
};

// zeros of level l in positions [0, pos)
__device__ __forceinline__ uint32_t rank0(const RankView& rv, uint32_t l, uint32_t pos) {
  const uint32_t sb = pos >> 8;
  const uint4* p = reinterpret_cast<const uint4*>(rv.bits + (uint64_t)l * rv.lw + (uint64_t)sb * 8);
  const uint4 x = __ldg(p), y = __ldg(p + 1);
  const uint32_t wd[8] = {x.x, x.y, x.z, x.w, y.x, y.y, y.z, y.w};
  const uint32_t wi = (pos >> 5) & 7, m = (1u << (pos & 31)) - 1u;
  uint32_t ones = __ldg(&rv.cpre[(uint64_t)l * rv.nchunk + (sb >> 8)]) + __ldg(&rv.dir[(uint64_t)l * rv.nsb + sb]);
#pragma unroll
  for (int k = 0; k < 8; ++k) ones += __popc((uint32_t)k < wi ? wd[k] : ((uint32_t)k == wi ? (wd[k] & m) : 0u));
  return pos - ones;
}

// #{ j in [s, e) : v_j < x } by walking the L levels
__device__ __forceinline__ uint32_t range_count_less(const RankView& rv, const uint32_t* s_z, uint32_t L, uint32_t nmax,
                                                     uint32_t x, uint32_t s, uint32_t e) {
  uint32_t cnt = 0;
  for (uint32_t l = 0; l < L && s < e; ++l) {
    if (e > nmax) e = nmax;  // positions stay in [0, n] on a well-formed matrix
    if (s > e) s = e;
    const uint32_t zs = rank0(rv, l, s), ze = rank0(rv, l, e);
    if ((x >> (L - 1 - l)) & 1u) {
      cnt += ze - zs;
      s = s_z[l] + (s - zs);
      e = s_z[l] + (e - ze);
    } else {
      s = zs;
      e = ze;
    }
  }
  return cnt;
}

struct RunVal {  // (distance of the last run head seen, whether one was seen)
  uint64_t v;
  uint64_t f;
};
struct RunValOp {
  __device__ RunVal operator()(const RunVal& a, const RunVal& b) const { return b.f ? b : a; }
};

struct QueryArgs {
  const uint32_t* prev;
  uint64_t n;
  uint32_t L;
  RankView rv;
  const unsigned long long* zcount;
  uint32_t* dist;
  uint8_t* heads;        // per 8 accesses: bit j set if access i0 + j starts a run
  RunVal* tile_agg;      // per tile: (distance of its last head, head seen)
  DevStatus* st;
};

// Pass 1: run heads query the matrix and write their distances; every tile
// records its head bits and (last head's distance, any head).  No tile waits.
__global__ void __launch_bounds__(kQThreads) k_wm_heads(QueryArgs a) {
  __shared__ uint32_t s_z[33];
  __shared__ RunVal s_last[kQThreads / 32];
  if (threadIdx.x < a.L) s_z[threadIdx.x] = (uint32_t)a.zcount[threadIdx.x];
  __syncthreads();
  const uint64_t i0 = (uint64_t)blockIdx.x * kQTile + (uint64_t)threadIdx.x * kQPer;
  const uint32_t nmax = (uint32_t)a.n;
  uint32_t p[kQPer];
  if (i0 + kQPer <= a.n && ((reinterpret_cast<uintptr_t>(a.prev) & 15) == 0)) {
    const uint4 x = __ldg(reinterpret_cast<const uint4*>(a.prev + i0));
    const uint4 y = __ldg(reinterpret_cast<const uint4*>(a.prev + i0 + 4));
    p[0] = x.x; p[1] = x.y; p[2] = x.z; p[3] = x.w;
    p[4] = y.x; p[5] = y.y; p[6] = y.z; p[7] = y.w;
  } else {
#pragma unroll
    for (int j = 0; j < kQPer; ++j) p[j] = i0 + j < a.n ? a.prev[i0 + j] : kNone;
  }
  const uint32_t before = (i0 > 0 && i0 - 1 < a.n) ? a.prev[i0 - 1] : kNone;
  RunVal loc{0, 0};
  uint32_t hbits = 0;
  bool bad = false;
#pragma unroll
  for (int j = 0; j < kQPer; ++j) {
    const uint64_t i = i0 + j;
    const uint32_t pj = p[j];
    const uint32_t pb = j ? p[j - 1] : before;
    const bool member = pj != kNone && pb != kNone && pb + 1u == pj;
    if (i < a.n && !member) {
      uint32_t d = kNone;
      if (pj != kNone) {
        if ((uint64_t)pj >= i)
          bad = true;
        else
          d = 1 + range_count_less(a.rv, s_z, a.L, nmax, pj + 1, pj + 1, (uint32_t)i);
      }
      a.dist[i] = d;
      hbits |= 1u << j;
      loc = RunVal{d, 1};
    }
  }
  if (bad) raise_err(a.st, kErrInvalid);
  if (i0 < a.n) a.heads[i0 / kQPer] = (uint8_t)hbits;
  // the tile's last head: the highest thread with a head
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t m = __ballot_sync(kFull, loc.f != 0);
  const RunVal wl = m ? shfl_payload(loc, 31 - __clz(m)) : RunVal{0, 0};
  if (lane == 0) s_last[w] = wl;
  __syncthreads();
  if (threadIdx.x == 0) {
    RunVal r{0, 0};
    for (int k = kQThreads / 32 - 1; k >= 0; --k)
      if (s_last[k].f) {
        r = s_last[k];
        break;
      }
    a.tile_agg[blockIdx.x] = r;
  }
}

// Pass 2: every access takes the distance of the last head at or before it.
__global__ void __launch_bounds__(kQThreads) k_wm_propagate(QueryArgs a) {
  __shared__ RunVal s_w[kQThreads / 32];
  __shared__ RunVal s_carry;
  const uint32_t tile = blockIdx.x;
  const uint64_t i0 = (uint64_t)tile * kQTile + (uint64_t)threadIdx.x * kQPer;
  const bool vec = i0 + kQPer <= a.n && ((reinterpret_cast<uintptr_t>(a.dist) & 15) == 0);
  uint32_t d[kQPer];
  if (vec) {
    const uint4 x = reinterpret_cast<const uint4*>(a.dist + i0)[0];
    const uint4 y = reinterpret_cast<const uint4*>(a.dist + i0)[1];
    d[0] = x.x; d[1] = x.y; d[2] = x.z; d[3] = x.w;
    d[4] = y.x; d[5] = y.y; d[6] = y.z; d[7] = y.w;
  } else {
#pragma unroll
    for (int j = 0; j < kQPer; ++j) d[j] = i0 + j < a.n ? a.dist[i0 + j] : 0u;
  }
  const uint32_t hbits = i0 < a.n ? a.heads[i0 / kQPer] : 0u;
  RunVal loc{0, 0};
  uint32_t val[kQPer];
  uint32_t covered = 0;
#pragma unroll
  for (int j = 0; j < kQPer; ++j) {
    if ((hbits >> j) & 1u) loc = RunVal{d[j], 1};
    val[j] = (uint32_t)loc.v;
    if (loc.f) covered |= 1u << j;
  }
  RunValOp op;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  RunVal x = loc;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    RunVal y;
    y.v = __shfl_up_sync(kFull, x.v, o);
    y.f = __shfl_up_sync(kFull, x.f, o);
    if (lane >= (uint32_t)o) x = op(y, x);
  }
  if (lane == 31) s_w[w] = x;
  __syncthreads();
  if (w == 0) {
    RunVal z = lane < kQThreads / 32 ? s_w[lane] : RunVal{0, 0};
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      RunVal y;
      y.v = __shfl_up_sync(kFull, z.v, o);
      y.f = __shfl_up_sync(kFull, z.f, o);
      if (lane >= (uint32_t)o) z = op(y, z);
    }
    if (lane < kQThreads / 32) s_w[lane] = z;
    // carry: the last head of the nearest earlier tile that has one
    RunVal c{0, 0};
    for (int64_t base = (int64_t)tile - 1; base >= 0; base -= 32) {
      const int64_t idx = base - (int64_t)lane;
      RunVal g{0, 0};
      if (idx >= 0) g = a.tile_agg[idx];
      const uint32_t hm = __ballot_sync(kFull, idx >= 0 && g.f);
      if (hm) {
        c = shfl_payload(g, __ffs(hm) - 1);
        break;
      }
    }
    if (lane == 0) s_carry = c;
  }
  __syncthreads();
  RunVal pre = s_carry;
  if (w > 0) pre = op(pre, s_w[w - 1]);
  {
    RunVal y;
    y.v = __shfl_up_sync(kFull, x.v, 1);
    y.f = __shfl_up_sync(kFull, x.f, 1);
    if (lane > 0) pre = op(pre, y);
  }
  uint32_t out[kQPer];
#pragma unroll
  for (int j = 0; j < kQPer; ++j) out[j] = ((covered >> j) & 1u) ? val[j] : (uint32_t)pre.v;
  if (vec) {
    reinterpret_cast<uint4*>(a.dist + i0)[0] = make_uint4(out[0], out[1], out[2], out[3]);
    reinterpret_cast<uint4*>(a.dist + i0)[1] = make_uint4(out[4], out[5], out[6], out[7]);
  } else {
#pragma unroll
    for (int j = 0; j < kQPer; ++j)
      if (i0 + j < a.n) a.dist[i0 + j] = out[j];
  }
}

uint32_t value_bits(uint64_t n) {  // values lie in [0, n]
  uint32_t L = 1;
  while (L < 33 && (1ULL << L) <= n) ++L;
  return L;
}

struct WmLayout {
  DevStatus* st;
  unsigned long long* zcount;
  uint32_t* done;
  uint32_t* G;
  uint32_t* H;
  uint32_t* T;
  uint32_t* csum;
  uint32_t* cpre;
  uint32_t* dir;
  RunVal* qagg;
  uint8_t* heads;
  uint32_t *va, *vb;
  uint32_t* bits;
  uint64_t lw;
  uint32_t L, ntiles, nsb, nchunk, passes;
  size_t zero_bytes;
  size_t total;
};

WmLayout wm_layout(void* ws, uint64_t n) {
  WmLayout W;
  Carver cv(ws);
  W.L = value_bits(n);
  W.passes = (W.L + kWB - 1) / kWB;
  W.ntiles = ceil_div_u32(n, kWTile) + 1;
  W.nsb = (uint32_t)(n / kSbBits) + 1;
  W.nchunk = ceil_div_u32(W.nsb, kSbPerChunk);
  W.lw = (uint64_t)W.nsb * 8 + 8;
  const uint64_t nn = n ? n : 1;
  const uint32_t qtiles = ceil_div_u32(n, kQTile) + 1;
  W.st = cv.take<DevStatus>(1);
  W.zcount = cv.take<unsigned long long>(40);
  W.done = cv.take<uint32_t>(64);
  W.zero_bytes = cv.off;
  W.G = cv.take<uint32_t>((uint64_t)W.passes * 16);
  W.H = cv.take<uint32_t>((uint64_t)W.ntiles * 16);
  W.T = cv.take<uint32_t>((uint64_t)W.ntiles * 16);
  W.csum = cv.take<uint32_t>((uint64_t)W.L * W.nchunk);
  W.cpre = cv.take<uint32_t>((uint64_t)W.L * W.nchunk);
  W.dir = cv.take<uint32_t>((uint64_t)W.L * W.nsb);
  W.qagg = cv.take<RunVal>(qtiles);
  W.heads = cv.take<uint8_t>(n / kQPer + 2);
  W.va = cv.take<uint32_t>(nn);
  W.vb = cv.take<uint32_t>(nn);
  W.bits = cv.take<uint32_t>((uint64_t)W.L * W.lw);
  W.total = cv.bytes();
  return W;
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_stack_distance_workspace_bytes(uint64_t n) { return wm_layout(nullptr, n).total; }

extern "C" ptc_status ptc_stack_distance(const uint32_t* prev, uint64_t n, uint32_t* dist_out, void* ws,
                                         size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (n == 0) return PTC_OK;
  if (!prev || !dist_out) return PTC_ERR_INVALID_ARG;
  if (!ws_ok(ws, ws_bytes, wm_layout(nullptr, n).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const WmLayout W = wm_layout(ws, n);
  if (begin_call(ws, W.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  if (cudaMemsetAsync(W.bits, 0, sizeof(uint32_t) * (uint64_t)W.L * W.lw, s) != cudaSuccess) return PTC_ERR_CUDA;
  const uint32_t tiles = ceil_div_u32(n, kWTile);
  const uint32_t* src = prev;
  uint32_t* bufs[2] = {W.va, W.vb};
  for (uint32_t pi = 0; pi < W.passes; ++pi) {
    PassArgs a;
    a.r = W.L - kWB * pi < (uint32_t)kWB ? W.L - kWB * pi : (uint32_t)kWB;
    a.lvl0 = kWB * pi;
    a.sh = W.L - a.lvl0 - a.r;
    a.src = src;
    a.from_prev = pi == 0;
    a.dst = pi + 1 < W.passes ? bufs[pi & 1] : nullptr;
    a.bits = W.bits;
    a.lw = W.lw;
    a.n = n;
    a.ntiles = tiles;
    a.H = W.H;
    a.T = W.T;
    a.G = W.G + 16 * pi;
    a.done = &W.done[pi];
    a.zcount = W.zcount;
    a.st = W.st;
    PTC_LAUNCH("k_wm_hist", s, k_wm_hist<<<tiles, kWT, 0, s>>>(a));
    PTC_LAUNCH("k_wm_scan", s, k_wm_scan<<<16, kScanThreads, 0, s>>>(a));
    PTC_LAUNCH("k_wm_pass", s, k_wm_pass<<<tiles, kWT, 0, s>>>(a));
    src = a.dst;
  }
  PTC_LAUNCH("k_wm_dir", s,
             k_wm_dir<<<W.L * W.nchunk, kSbPerChunk, 0, s>>>(W.bits, W.lw, W.L, W.nsb, W.nchunk, W.dir, W.csum, W.cpre,
                                                            &W.done[63]));
  QueryArgs q;
  q.prev = prev;
  q.n = n;
  q.L = W.L;
  q.rv = RankView{W.bits, W.lw, W.dir, W.cpre, W.nsb, W.nchunk};
  q.zcount = W.zcount;
  q.dist = dist_out;
  q.heads = W.heads;
  q.tile_agg = W.qagg;
  q.st = W.st;
  PTC_LAUNCH("k_wm_heads", s, k_wm_heads<<<ceil_div_u32(n, kQTile), kQThreads, 0, s>>>(q));
  PTC_LAUNCH("k_wm_propagate", s, k_wm_propagate<<<ceil_div_u32(n, kQTile), kQThreads, 0, s>>>(q));
  DevStatus h;
  return end_call(W.st, s, &h);
}
