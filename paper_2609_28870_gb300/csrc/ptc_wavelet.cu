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
//
// Layout of one level: a plain bitvector (LSB first) plus a rank directory of
// ones per 256-bit superblock (relative to its chunk of 256 superblocks) and
// per chunk; a rank reads the superblock's 32-byte sector and two counts.
//   k_wm_count0  level-0 zero counts of every tile and their prefixes
//   k_wm_level   one level: ballot bits, stable partition by the bit (see
//                the kernel's comment for how tile prefixes avoid waiting)
//   k_wm_dir     rank directories of all levels
//   k_wm_heads   run heads walk the L levels (early exit on an empty range)
//                and write their distances; tiles record their last head.
//   k_wm_propagate  every access takes the distance of the last head at or
//                before it (segmented scan; the carry comes from the tile
//                records, all written by the previous kernel).
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kLT = 256;                    // threads per tile
constexpr int kLR = 8;                      // rounds (32 positions each) per warp
constexpr int kLW = kLT / 32;               // warps per tile
constexpr int kLTile = kLT * kLR;           // 2048 positions per tile; warp w owns [256 w, 256 w + 256)
constexpr int kSbBits = 256;                // rank-directory superblock
constexpr int kSbPerChunk = 256;
constexpr int kQThreads = 256;
constexpr int kQPer = 8;
constexpr int kQTile = kQThreads * kQPer;

struct LevelArgs {
  const uint32_t* src;             // this level's order (prev itself at level 0)
  int from_prev;                   // values are prev + 1 (none -> 0)
  uint32_t* dst;                   // the next level's order (null at the last level)
  uint32_t* bits;                  // this level's bitvector
  uint64_t n;
  uint32_t ntiles;
  uint32_t shift;                  // bit tested at this level
  const uint32_t* tp;              // zeros before every tile of this level
  const unsigned long long* zl;    // Z of this level
  uint32_t* tz_next;               // zeros of every tile of the next level (accumulated here)
  uint32_t* tp_next;               // ... their exclusive prefix (written by the last CTA)
  unsigned long long* z_next;      // ... and their total, Z of the next level
  uint32_t* done;                  // CTAs finished
  DevStatus* st;
};

__device__ __forceinline__ uint32_t level_value(const LevelArgs& a, uint32_t j) {
  uint32_t x = a.src[j];
  if (a.from_prev) x = x == kNone ? 0u : x + 1u;
  return x;
}

// Run by every thread of the CTA that finished last (threadfence-reduction
// pattern): tp[i] = tz[0] + ... + tz[i-1] for i < ntiles and *total = sum.
// Each thread takes a contiguous run; loads bypass L1 (other CTAs' atomics).
__device__ inline void finish_counts(uint32_t* done, const uint32_t* tz, uint32_t* tp, uint32_t ntiles,
                                     unsigned long long* total) {
  __shared__ bool s_last;
  __shared__ uint32_t s_w[kLT / 32];
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(done, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const uint32_t t = threadIdx.x, lane = t & 31, w = t >> 5;
  const uint32_t per = (ntiles + kLT - 1) / kLT;
  const uint32_t lo = t * per < ntiles ? t * per : ntiles, hi = lo + per < ntiles ? lo + per : ntiles;
  uint32_t sum = 0;
  for (uint32_t i = lo; i < hi; ++i) sum += __ldcg(&tz[i]);
  uint32_t x = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFull, x, o);
    if (lane >= (uint32_t)o) x += y;
  }
  if (lane == 31) s_w[w] = x;
  __syncthreads();
  uint32_t wpre = 0, tot = 0;
#pragma unroll
  for (int k = 0; k < kLT / 32; ++k) {
    wpre += k < (int)w ? s_w[k] : 0u;
    tot += s_w[k];
  }
  uint32_t run = wpre + x - sum;
  for (uint32_t i = lo; i < hi; ++i) {
    tp[i] = run;
    run += __ldcg(&tz[i]);
  }
  if (t == 0) *total = tot;
}

// Level-0 zero count of every tile (bit L-1 of v = prev + 1), Z_0 and the
// tile prefixes; also checks prev[j] < j.
__global__ void __launch_bounds__(kLT) k_wm_count0(LevelArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_wz[kLW];
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t n32 = (uint32_t)a.n;
  const uint32_t wbase = blockIdx.x * kLTile + w * 256;
  uint32_t zc = 0;
  bool bad = false;
#pragma unroll
  for (int rd = 0; rd < kLR; ++rd) {
    const uint32_t j = wbase + rd * 32 + lane;
    bool zero = false;
    if (j < n32) {
      const uint32_t p = a.src[j];
      if (p != kNone && p >= j) bad = true;
      const uint32_t v = p == kNone ? 0u : p + 1u;
      zero = !((v >> a.shift) & 1u);
    }
    zc += __popc(__ballot_sync(kFull, zero));
  }
  if (bad) raise_err(a.st, kErrInvalid);
  if (lane == 0) s_wz[w] = zc;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t z = 0;
    for (int k = 0; k < kLW; ++k) z += s_wz[k];
    a.tz_next[blockIdx.x] = z;
  }
  finish_counts(a.done, a.tz_next, a.tp_next, a.ntiles, a.z_next);
}

// One level.  Each warp owns 256 consecutive positions (8 rounds of 32):
// ballot of the level bit -> bitvector word; stable partition -> the zeros go
// to [zeros before, ...), the ones to Z + [ones before, ...).  The tile's
// prefix comes from the previous level (no waiting).  Every element counts
// itself, in a packed per-lane counter, into the next level's tile it lands
// in (the zeros and the ones of a tile each meet at most two such tiles); the
// CTA that finishes last turns those counts into the next level's prefixes.
__global__ void __launch_bounds__(kLT) k_wm_level(LevelArgs a) {
  grid_dep_sync();
  __shared__ uint32_t s_wz[kLW];
  __shared__ uint32_t s_cnt[kLW][4];
  const uint32_t t = threadIdx.x, lane = t & 31, w = t >> 5;
  const uint32_t n32 = (uint32_t)a.n;
  const uint32_t tile = blockIdx.x;
  const uint32_t wbase = tile * kLTile + w * 256;
  uint32_t v[kLR];
#pragma unroll
  for (int rd = 0; rd < kLR; ++rd) {
    const uint32_t j = wbase + rd * 32 + lane;
    v[rd] = j < n32 ? level_value(a, j) : 0u;
  }
  const bool tail = wbase + 256 > n32;
  uint32_t m[kLR];
  uint32_t zc = 0;
#pragma unroll
  for (int rd = 0; rd < kLR; ++rd) {
    const uint32_t vm = tail ? __ballot_sync(kFull, wbase + rd * 32 + lane < n32) : kFull;
    m[rd] = __ballot_sync(kFull, (v[rd] >> a.shift) & 1u) & vm;
    zc += __popc(vm & ~m[rd]);
    if (lane == 0 && (vm & 1u)) a.bits[(wbase + rd * 32) >> 5] = m[rd];
  }
  if (lane == 0) s_wz[w] = zc;
  __syncthreads();
  uint32_t wp = 0, tzt = 0;
#pragma unroll
  for (int k = 0; k < kLW; ++k) {
    const uint32_t z = s_wz[k];
    wp += k < (int)w ? z : 0u;
    tzt += z;
  }
  const uint32_t tile_base = a.tp[tile];
  const uint32_t Z = (uint32_t)*a.zl;
  if (t == 0) {  // the published count must match the data
    const uint32_t next = tile + 1 < a.ntiles ? a.tp[tile + 1] : Z;
    if (next - tile_base != tzt) raise_err(a.st, kErrInvalid);
  }
  if (a.dst == nullptr) return;
  uint32_t zb = tile_base + wp;     // zeros before this warp's first position
  uint32_t ob = wbase - zb;         // ones before it
  const uint32_t SZ = (tile_base / kLTile + 1) * kLTile;
  const uint32_t SO = ((Z + tile * kLTile - tile_base) / kLTile + 1) * kLTile;
  const uint32_t nshift = a.shift - 1;
  const uint32_t lt = lanemask_lt();
  uint32_t cz = 0, co = 0;  // (early count) | (late count) << 16, for landing zeros / ones
#pragma unroll
  for (int rd = 0; rd < kLR; ++rd) {
    const uint32_t vm = tail ? __ballot_sync(kFull, wbase + rd * 32 + lane < n32) : kFull;
    const uint32_t mz = vm & ~m[rd];
    const uint32_t r0 = __popc(mz & lt);
    const bool one = (m[rd] >> lane) & 1u;
    const uint32_t dst = one ? Z + ob + (lane - r0) : zb + r0;
    const bool valid = (vm >> lane) & 1u;
    if (valid && dst < n32) a.dst[dst] = v[rd];
    const uint32_t inc = (valid && !((v[rd] >> nshift) & 1u)) ? (dst < (one ? SO : SZ) ? 1u : 0x10000u) : 0u;
    if (one)
      co += inc;
    else
      cz += inc;
    zb += __popc(mz);
    ob += __popc(m[rd]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    cz += __shfl_xor_sync(kFull, cz, o);
    co += __shfl_xor_sync(kFull, co, o);
  }
  if (lane == 0) {
    s_cnt[w][0] = cz & 0xFFFFu;
    s_cnt[w][1] = cz >> 16;
    s_cnt[w][2] = co & 0xFFFFu;
    s_cnt[w][3] = co >> 16;
  }
  __syncthreads();
  if (t < 4) {
    uint32_t c = 0;
    for (int k = 0; k < kLW; ++k) c += s_cnt[k][t];
    if (c) {
      const uint32_t dt = t < 2 ? SZ / kLTile - (t == 0 ? 1u : 0u) : SO / kLTile - (t == 2 ? 1u : 0u);
      if (dt < a.ntiles) atomicAdd(&a.tz_next[dt], c);
    }
  }
  finish_counts(a.done, a.tz_next, a.tp_next, a.ntiles, a.z_next);
}

// Rank directory of every level: dir[l][sb] = ones in the superblocks of its
// chunk before sb, csum[l][c] = ones in chunk c; the CTA that finishes last
// turns csum into cpre[l][c] = ones in the chunks before c.
__global__ void __launch_bounds__(kSbPerChunk) k_wm_dir(const uint32_t* __restrict__ bits, uint64_t lw, uint32_t L,
                                                        uint32_t nsb, uint32_t nchunk, uint32_t* __restrict__ dir,
                                                        uint32_t* csum, uint32_t* __restrict__ cpre, uint32_t* done) {
  grid_dep_sync();
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
  const uint32_t* wend;  // window end of every access (null: the access itself)
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
  grid_dep_sync();
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
  // window ends: a run continues only within one window end (with window
  // ends the distance then falls by one per access, see k_wm_propagate)
  uint32_t we[kQPer + 1];
#pragma unroll
  for (int j = 0; j <= kQPer; ++j) {
    const uint64_t i = i0 + j - 1;
    we[j] = (a.wend && j + i0 > 0 && i < a.n) ? __ldg(a.wend + i) : 0u;
  }
  RunVal loc{0, 0};
  uint32_t hbits = 0;
  bool bad = false;
#pragma unroll
  for (int j = 0; j < kQPer; ++j) {
    const uint64_t i = i0 + j;
    const uint32_t pj = p[j];
    const uint32_t pb = j ? p[j - 1] : before;
    const bool member = pj != kNone && pb != kNone && pb + 1u == pj && we[j + 1] == we[j];
    if (i < a.n && !member) {
      uint32_t d = kNone;
      if (pj != kNone) {
        const uint64_t e = a.wend ? (uint64_t)we[j + 1] : i;
        if ((uint64_t)pj >= e || e > i)
          bad = true;
        else
          d = 1 + range_count_less(a.rv, s_z, a.L, nmax, pj + 1, pj + 1, (uint32_t)e);
      }
      a.dist[i] = d;
      hbits |= 1u << j;
      loc = RunVal{(uint64_t)d + (a.wend ? i : 0), 1};  // the form k_wm_propagate carries
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
  grid_dep_sync();
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
  // With window ends a run's distance falls by one per access (the window
  // keeps its end and loses its first position), so the carried value is the
  // head's distance plus the head's index, and access i takes it minus i.
  const bool shift = a.wend != nullptr;
  RunVal loc{0, 0};
  uint64_t val[kQPer];
  uint32_t covered = 0;
#pragma unroll
  for (int j = 0; j < kQPer; ++j) {
    if ((hbits >> j) & 1u) loc = RunVal{(uint64_t)d[j] + (shift ? i0 + j : 0), 1};
    val[j] = loc.v;
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
  for (int j = 0; j < kQPer; ++j)
    out[j] = (uint32_t)((((covered >> j) & 1u) ? val[j] : pre.v) - (shift ? i0 + j : 0));
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
  uint32_t* tz;   // L x ntiles
  uint32_t* tp;   // L x ntiles
  uint32_t* csum;
  uint32_t* cpre;
  uint32_t* dir;
  RunVal* qagg;
  uint8_t* heads;
  uint32_t *va, *vb;
  uint32_t* bits;
  uint64_t lw;
  uint32_t L, ntiles, nsb, nchunk;
  size_t zero_bytes;
  size_t total;
};

WmLayout wm_layout(void* ws, uint64_t n) {
  WmLayout W;
  Carver cv(ws);
  W.L = value_bits(n);
  W.ntiles = ceil_div_u32(n, kLTile);
  W.nsb = (uint32_t)(n / kSbBits) + 1;
  W.nchunk = ceil_div_u32(W.nsb, kSbPerChunk);
  W.lw = (uint64_t)W.nsb * 8 + 8;
  const uint64_t nn = n ? n : 1;
  const uint32_t qtiles = ceil_div_u32(n, kQTile) + 1;
  W.st = cv.take<DevStatus>(1);
  W.zcount = cv.take<unsigned long long>(40);
  W.done = cv.take<uint32_t>(64);
  W.tz = cv.take<uint32_t>((uint64_t)W.L * (W.ntiles + 1));
  W.zero_bytes = cv.off;
  W.tp = cv.take<uint32_t>((uint64_t)W.L * (W.ntiles + 1));
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

size_t ptc::stack_distance_points_bytes(uint64_t n) { return wm_layout(nullptr, n).total; }

// The matrix over every access (argument checks are the caller's).
ptc_status ptc::stack_distance_points(const uint32_t* prev, uint64_t n, uint32_t* dist_out, void* ws,
                                      size_t ws_bytes, cudaStream_t s, const uint32_t* wend) {
  if (!ws_ok(ws, ws_bytes, wm_layout(nullptr, n).total)) return PTC_ERR_WORKSPACE;
  const WmLayout W = wm_layout(ws, n);
  if (begin_call(ws, W.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  if (fill_async(W.bits, 0u, sizeof(uint32_t) * (uint64_t)W.L * W.lw, s) != PTC_OK) return PTC_ERR_CUDA;
  const uint32_t tiles = W.ntiles;
  LevelArgs a;
  a.src = prev;
  a.from_prev = 1;
  a.dst = nullptr;
  a.bits = nullptr;
  a.n = n;
  a.ntiles = tiles;
  a.shift = W.L - 1;
  a.tp = nullptr;
  a.zl = nullptr;
  a.tz_next = W.tz;
  a.tp_next = W.tp;
  a.z_next = &W.zcount[0];
  a.done = &W.done[62];
  a.st = W.st;
  PTC_KERNEL("k_wm_count0", s, k_wm_count0, tiles, kLT, 0, a);
  uint32_t* bufs[2] = {W.va, W.vb};
  for (uint32_t l = 0; l < W.L; ++l) {
    const bool last = l + 1 == W.L;
    a.src = l == 0 ? prev : bufs[(l + 1) & 1];
    a.from_prev = l == 0;
    a.dst = last ? nullptr : bufs[l & 1];
    a.bits = W.bits + (uint64_t)l * W.lw;
    a.shift = W.L - 1 - l;
    a.tp = W.tp + (uint64_t)l * (tiles + 1);
    a.zl = &W.zcount[l];
    a.tz_next = last ? nullptr : W.tz + (uint64_t)(l + 1) * (tiles + 1);
    a.tp_next = last ? nullptr : W.tp + (uint64_t)(l + 1) * (tiles + 1);
    a.z_next = last ? nullptr : &W.zcount[l + 1];
    a.done = &W.done[l];
    PTC_KERNEL("k_wm_level", s, k_wm_level, tiles, kLT, 0, a);
  }
  PTC_KERNEL("k_wm_dir", s, k_wm_dir, W.L * W.nchunk, kSbPerChunk, 0, W.bits, W.lw, W.L, W.nsb, W.nchunk, W.dir, W.csum, W.cpre, &W.done[63]);
  QueryArgs q;
  q.prev = prev;
  q.wend = wend;
  q.n = n;
  q.L = W.L;
  q.rv = RankView{W.bits, W.lw, W.dir, W.cpre, W.nsb, W.nchunk};
  q.zcount = W.zcount;
  q.dist = dist_out;
  q.heads = W.heads;
  q.tile_agg = W.qagg;
  q.st = W.st;
  PTC_KERNEL("k_wm_heads", s, k_wm_heads, ceil_div_u32(n, kQTile), kQThreads, 0, q);
  PTC_KERNEL("k_wm_propagate", s, k_wm_propagate, ceil_div_u32(n, kQTile), kQThreads, 0, q);
  DevStatus h;
  return end_call(W.st, s, &h);
}
