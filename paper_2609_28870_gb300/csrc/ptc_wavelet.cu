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
// Layout of one level: blocks of 224 positions in 32 bytes,
//   word 0 = zeros before the block, words 1..7 = 224 bits (LSB first)
// so a rank is one 32-byte sector.
//   k_wm_count0  zero counts of every level-0 tile, and Z_0
//   k_wm_level   one level: ballot bits -> rank blocks; stable partition by
//                the bit.  Tile prefixes come from a look-back over zero
//                counts that the previous level already published (each
//                element adds itself to the count of the tile it lands in),
//                so no tile ever waits for another.
//   k_wm_query   run heads walk the L levels (early exit on an empty range);
//                a segmented scan hands each head's value to its run.
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kLvThreads = 256;
constexpr int kLvWarps = kLvThreads / 32;
constexpr int kBlkBits = 224;                 // positions per rank block
constexpr int kLvTile = kLvWarps * kBlkBits;  // 1792 positions per tile
constexpr int kQThreads = 256;
constexpr int kQPer = 8;
constexpr int kQTile = kQThreads * kQPer;
constexpr int kEpochQuery = 40;
constexpr int kLvCtasPerSm = 4;

struct LevelArgs {
  const uint32_t* prev;        // level 0 input (values derived on the fly)
  const uint32_t* vin;         // levels >= 1: this level's order
  uint32_t* vout;              // next level's order (null on the last level)
  uint32_t* mat;               // this level's rank blocks
  uint64_t n;
  uint32_t shift;              // bit tested at this level
  uint32_t level;
  const uint32_t* tz;          // zeros of every tile of this level (complete)
  uint32_t* tz_next;           // zeros of every tile of the next level (accumulated here)
  unsigned long long* zsum;    // zsum[l] = Z_l; zsum[level + 1] is accumulated here
  uint64_t* incl;              // inclusive prefixes of this level's tiles (packed words)
  DevStatus* st;
  uint32_t ntiles;
  int src_aligned;             // the input is 16-byte aligned (bulk copies allowed)
};

// Exclusive prefix of `tile` over counts that are all known before the kernel
// starts: a predecessor with no published inclusive prefix contributes its
// count, so the look-back never waits.  CTA-wide; every thread calls it.
__device__ inline uint64_t prepub_prefix(uint64_t* incl, const uint32_t* tz, uint32_t tile, uint32_t epoch) {
  __shared__ uint64_t s_part[kLvWarps];
  __shared__ uint32_t s_first;
  __shared__ uint64_t s_excl;
  const uint32_t t = threadIdx.x, lane = t & 31, wid = t >> 5;
  if (t == 0) s_excl = 0;
  __syncthreads();
  int64_t base = (int64_t)tile - 1;
  while (base >= 0) {
    const int64_t idx = base - (int64_t)t;
    uint64_t v = 0;
    bool inc = false;
    if (idx >= 0) {
      const uint64_t w = ld_relaxed_u64(&incl[idx]);
      inc = ((uint32_t)(w >> 58) == epoch) && ((w >> 56) & 3) == 2;
      v = inc ? (w & kLbValMask) : tz[idx];
    }
    if (t == 0) s_first = 0xFFFFFFFFu;
    __syncthreads();
    if (inc) atomicMin(&s_first, t);
    __syncthreads();
    const uint32_t first = s_first;
    if (t > first) v = 0;
    v = warp_sum_u64(v);
    if (lane == 0) s_part[wid] = v;
    __syncthreads();
    if (t == 0) {
      uint64_t sum = 0;
      for (int k = 0; k < kLvWarps; ++k) sum += s_part[k];
      s_excl += sum;
    }
    __syncthreads();
    if (first != 0xFFFFFFFFu) break;
    base -= kLvThreads;
  }
  const uint64_t e = s_excl;
  if (t == 0) st_relaxed_u64(&incl[tile], lb_pack(epoch, 2, e + tz[tile]));
  return e;
}

// Level-0 tile zero counts (bit L-1 of v = prev + 1) and Z_0; checks prev.
__global__ void __launch_bounds__(kLvThreads) k_wm_count0(const uint32_t* __restrict__ prev, uint64_t n,
                                                          uint32_t shift, uint32_t* __restrict__ tz,
                                                          unsigned long long* zsum, DevStatus* st) {
  __shared__ uint32_t s_wz[kLvWarps];
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint64_t base = ((uint64_t)blockIdx.x * kLvWarps + w) * kBlkBits;
  uint32_t zeros = 0;
  bool bad = false;
#pragma unroll
  for (int k = 0; k < 7; ++k) {
    const uint64_t j = base + (uint64_t)k * 32 + lane;
    bool zero = false;
    if (j < n) {
      const uint32_t p = prev[j];
      if (p != kNone && (uint64_t)p >= j) bad = true;
      const uint32_t v = p == kNone ? 0u : p + 1u;
      zero = !((v >> shift) & 1u);
    }
    zeros += __popc(__ballot_sync(kFull, zero));
  }
  if (bad) raise_err(st, kErrInvalid);
  if (lane == 0) s_wz[w] = zeros;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t z = 0;
    for (int k = 0; k < kLvWarps; ++k) z += s_wz[k];
    tz[blockIdx.x] = z;
    if (z) atomicAdd(&zsum[0], (unsigned long long)z);
  }
}

// Persistent CTAs: each claims tiles in order from the launch's counter and
// keeps the next tile's input streaming into shared memory (bulk copy, two
// stages) while it works on the current one.
__global__ void __launch_bounds__(kLvThreads) k_wm_level(LevelArgs a) {
  __shared__ __align__(128) uint32_t s_buf[2][kLvTile];
  __shared__ __align__(8) uint64_t s_bar[2];
  __shared__ uint32_t s_tile[2], s_full[2];
  __shared__ uint32_t s_wz[kLvWarps];
  __shared__ uint32_t s_next_zeros;
  const uint32_t epoch = a.level + 1;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t* src = a.level == 0 ? a.prev : a.vin;
  // thread 0: claim the next tile and start its copy; returns the elements copied
  auto claim_and_issue = [&](int stg) {
    const uint32_t tile = atomicAdd(&a.st->tile_ctr[epoch], 1u);
    s_tile[stg] = tile;
    uint32_t full = 0;
    const uint64_t start = (uint64_t)tile * kLvTile;
    if (tile < a.ntiles && start < a.n && a.src_aligned) {
      const uint64_t cnt = a.n - start < (uint64_t)kLvTile ? a.n - start : (uint64_t)kLvTile;
      const uint32_t bytes = (uint32_t)(cnt * 4) & ~15u;
      if (bytes) {
        mbar_expect_tx(&s_bar[stg], bytes);
        bulk_load(s_buf[stg], src + start, bytes, &s_bar[stg]);
        full = bytes / 4;
      }
    }
    s_full[stg] = full;
  };
  if (threadIdx.x == 0) {
    mbar_init(&s_bar[0], 1);
    mbar_init(&s_bar[1], 1);
    mbar_init_fence();
    s_next_zeros = 0;
  }
  __syncthreads();
  if (threadIdx.x == 0) claim_and_issue(0);
  __syncthreads();
  uint32_t stage = 0, phase[2] = {0, 0};
  for (;;) {
    const uint32_t tile = s_tile[stage];
    if (tile >= a.ntiles) break;
    const uint32_t full = s_full[stage];
    if (threadIdx.x == 0) claim_and_issue(stage ^ 1);
    if (full) {
      if (!mbar_wait(&s_bar[stage], phase[stage])) {
        raise_err(a.st, kErrTimeout);
        mbar_wait(&s_bar[stage], phase[stage]);  // give the copy one more bounded chance to land
        return;
      }
      phase[stage] ^= 1;
    }
    const uint64_t blk = (uint64_t)tile * kLvWarps + w;
    const uint64_t base = blk * kBlkBits;
    uint32_t v[7];
#pragma unroll
    for (int k = 0; k < 7; ++k) {
      const uint32_t rel = w * kBlkBits + k * 32 + lane;
      const uint64_t j = base + (uint64_t)k * 32 + lane;
      uint32_t x = 0;
      if (j < a.n) x = rel < full ? s_buf[stage][rel] : src[j];
      if (a.level == 0) x = (j < a.n && x != kNone) ? x + 1u : 0u;
      v[k] = x;
    }
    const uint64_t tile_base = prepub_prefix(a.incl, a.tz, tile, epoch);  // zeros before this tile
    uint32_t word[7], vmask[7];
    uint32_t zeros = 0;
#pragma unroll
    for (int k = 0; k < 7; ++k) {
      const uint64_t j = base + (uint64_t)k * 32 + lane;
      const bool valid = j < a.n;
      word[k] = __ballot_sync(kFull, valid && ((v[k] >> a.shift) & 1u));
      vmask[k] = __ballot_sync(kFull, valid);
      zeros += __popc(vmask[k] & ~word[k]);
    }
    if (lane == 0) s_wz[w] = zeros;
    __syncthreads();
    if (w == 0) {
      const uint32_t z = lane < kLvWarps ? s_wz[lane] : 0u;
      uint32_t x = z;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, x, o);
        if (lane >= (uint32_t)o) x += y;
      }
      if (lane < kLvWarps) s_wz[lane] = x - z;  // exclusive over warps
      // the counts the previous level published must match the data
      if (lane == 31 && x != a.tz[tile]) raise_err(a.st, kErrInvalid);
    }
    __syncthreads();
    const uint64_t zb = tile_base + s_wz[w];  // zeros before this rank block
    if (base <= a.n && lane < 8) {
      uint32_t out = (uint32_t)zb;
#pragma unroll
      for (int k = 0; k < 7; ++k)
        if (lane == (uint32_t)k + 1) out = word[k];
      a.mat[blk * 8 + lane] = out;
    }
    if (a.vout != nullptr) {
      const uint64_t Z = a.zsum[a.level];
      uint64_t zrun = zb;
      uint32_t next_zeros = 0;
      const uint32_t lt = lanemask_lt();
#pragma unroll
      for (int k = 0; k < 7; ++k) {
        const uint64_t j = base + (uint64_t)k * 32 + lane;
        const uint32_t zmask = vmask[k] & ~word[k];
        const bool valid = j < a.n;
        uint64_t dst = 0;
        if (valid) {
          const uint64_t zb_elem = zrun + __popc(zmask & lt);
          dst = ((word[k] >> lane) & 1u) ? Z + (j - zb_elem) : zb_elem;
          if (dst < a.n) a.vout[dst] = v[k];  // in range on a well-formed input
        }
        // zeros of the next level, counted into the tile each element lands in
        const bool nz = valid && dst < a.n && !((v[k] >> (a.shift - 1)) & 1u);
        const uint32_t dt = nz ? (uint32_t)(dst / kLvTile) : 0xFFFFFFFFu - lane;
        const uint32_t peers = __match_any_sync(kFull, dt);
        if (nz && lane == (uint32_t)(__ffs(peers) - 1)) atomicAdd(&a.tz_next[dt], (uint32_t)__popc(peers));
        next_zeros += __popc(__ballot_sync(kFull, nz));
        zrun += __popc(zmask);
      }
      if (lane == 0 && next_zeros) atomicAdd(&s_next_zeros, next_zeros);
    }
    __syncthreads();  // this stage's buffer is free; the next claim is visible
    stage ^= 1;
  }
  __syncthreads();
  if (threadIdx.x == 0 && s_next_zeros) atomicAdd(&a.zsum[a.level + 1], (unsigned long long)s_next_zeros);
}

__device__ __forceinline__ uint32_t rank0(const uint32_t* __restrict__ lvl, uint32_t pos) {
  const uint32_t b = pos / kBlkBits;
  const uint32_t off = pos - b * kBlkBits;
  const uint4* p = reinterpret_cast<const uint4*>(lvl + (uint64_t)b * 8);
  const uint4 lo = __ldg(p), hi = __ldg(p + 1);
  const uint32_t wi = off >> 5;
  const uint32_t m = (1u << (off & 31)) - 1u;
  const uint32_t w[7] = {lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
  uint32_t ones = 0;
#pragma unroll
  for (int k = 0; k < 7; ++k) {
    const uint32_t x = (uint32_t)k < wi ? w[k] : ((uint32_t)k == wi ? (w[k] & m) : 0u);
    ones += __popc(x);
  }
  return lo.x + off - ones;
}

// #{ j in [s, e) : v_j < x } by walking the L levels
__device__ __forceinline__ uint32_t range_count_less(const uint32_t* __restrict__ mat, uint64_t level_words,
                                                     const uint32_t* s_z, uint32_t L, uint32_t nmax, uint32_t x,
                                                     uint32_t s, uint32_t e) {
  uint32_t cnt = 0;
  for (uint32_t l = 0; l < L && s < e; ++l) {
    if (e > nmax) e = nmax;  // positions stay in [0, n] on a well-formed matrix
    if (s > e) s = e;
    const uint32_t* lvl = mat + (uint64_t)l * level_words;
    const uint32_t zs = rank0(lvl, s), ze = rank0(lvl, e);
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
  const uint32_t* mat;
  uint64_t level_words;
  const unsigned long long* zcount;
  uint32_t* dist;
  LbArrays<RunVal> lb;
  DevStatus* st;
};

__global__ void __launch_bounds__(kQThreads) k_wm_query(QueryArgs a) {
  __shared__ uint32_t s_z[33];
  __shared__ RunVal s_w[kQThreads / 32];
  __shared__ RunVal s_carry;
  if (threadIdx.x < a.L) s_z[threadIdx.x] = (uint32_t)a.zcount[threadIdx.x];
  const uint32_t tile = next_tile(a.st, kEpochQuery);  // also orders the s_z writes
  const uint64_t i0 = (uint64_t)tile * kQTile + (uint64_t)threadIdx.x * kQPer;
  const uint32_t nmax = (uint32_t)a.n;
  uint32_t p[kQPer];
#pragma unroll
  for (int j = 0; j < kQPer; ++j) p[j] = i0 + j < a.n ? a.prev[i0 + j] : kNone;
  const uint32_t before = (i0 > 0 && i0 - 1 < a.n) ? a.prev[i0 - 1] : kNone;

  // run heads query the matrix; every other access copies its head
  RunVal loc{0, 0};
  uint32_t val[kQPer];
  uint32_t covered = 0;
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
          d = 1 + range_count_less(a.mat, a.level_words, s_z, a.L, nmax, pj + 1, pj + 1, (uint32_t)i);
      }
      loc = RunVal{d, 1};
    }
    val[j] = (uint32_t)loc.v;
    if (loc.f) covered |= 1u << j;
  }
  if (bad) raise_err(a.st, kErrInvalid);

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
    if (lane < kQThreads / 32) s_w[lane] = z;  // inclusive over warps
  }
  __syncthreads();
  {
    const RunVal cin = lookback_cta(a.lb, tile, s_w[kQThreads / 32 - 1], RunVal{0, 0}, op, kEpochQuery, a.st);
    if (threadIdx.x == 0) s_carry = cin;
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
  if (i0 + kQPer <= a.n && ((reinterpret_cast<uintptr_t>(a.dist) & 15) == 0)) {
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
  uint64_t* lb;
  uint32_t* tz;  // L x tiles
  uint32_t* lbq_status;
  RunVal* lbq_agg;
  RunVal* lbq_incl;
  uint32_t *va, *vb;
  uint32_t tiles;
  uint32_t* mat;
  uint64_t level_words;
  uint32_t L;
  size_t zero_bytes;
  size_t total;
};

WmLayout wm_layout(void* ws, uint64_t n) {
  WmLayout L;
  Carver cv(ws);
  L.L = value_bits(n);
  const uint64_t nblk = n / kBlkBits + 2;
  const uint64_t nn = n ? n : 1;
  const uint32_t qtiles = ceil_div_u32(n, kQTile) + 1;
  L.level_words = nblk * 8;
  L.st = cv.take<DevStatus>(1);
  L.zcount = cv.take<unsigned long long>(40);
  L.tiles = ceil_div_u32(n + 1, kLvTile);
  L.lb = cv.take<uint64_t>(L.tiles + 1);
  L.tz = cv.take<uint32_t>((uint64_t)L.L * (L.tiles + 1));
  L.lbq_status = cv.take<uint32_t>(qtiles);
  L.zero_bytes = cv.off;
  L.lbq_agg = cv.take<RunVal>(qtiles);
  L.lbq_incl = cv.take<RunVal>(qtiles);
  L.va = cv.take<uint32_t>(nn);
  L.vb = cv.take<uint32_t>(nn);
  L.mat = cv.take<uint32_t>(L.level_words * L.L);
  L.total = cv.bytes();
  return L;
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
  const uint32_t tiles = W.tiles;
  const uint32_t grid = tiles < (uint32_t)(num_sms() * kLvCtasPerSm) ? tiles : (uint32_t)(num_sms() * kLvCtasPerSm);
  PTC_LAUNCH("k_wm_count0", s, k_wm_count0<<<tiles, kLvThreads, 0, s>>>(prev, n, W.L - 1, W.tz, W.zcount, W.st));
  const uint32_t* vin = nullptr;
  uint32_t* vout = W.va;
  for (uint32_t l = 0; l < W.L; ++l) {
    LevelArgs a;
    a.prev = prev;
    a.vin = vin;
    a.vout = (l + 1 < W.L) ? vout : nullptr;
    a.mat = W.mat + (uint64_t)l * W.level_words;
    a.n = n;
    a.shift = W.L - 1 - l;
    a.level = l;
    a.tz = W.tz + (uint64_t)l * (tiles + 1);
    a.tz_next = (l + 1 < W.L) ? W.tz + (uint64_t)(l + 1) * (tiles + 1) : nullptr;
    a.zsum = W.zcount;
    a.incl = W.lb;
    a.st = W.st;
    a.ntiles = tiles;
    a.src_aligned = l == 0 ? ((((uintptr_t)prev) & 15) == 0) : 1;
    PTC_LAUNCH("k_wm_level", s, k_wm_level<<<grid, kLvThreads, 0, s>>>(a));
    vin = vout;
    vout = (vout == W.va) ? W.vb : W.va;
  }
  QueryArgs q;
  q.prev = prev;
  q.n = n;
  q.L = W.L;
  q.mat = W.mat;
  q.level_words = W.level_words;
  q.zcount = W.zcount;
  q.dist = dist_out;
  q.lb = LbArrays<RunVal>{W.lbq_status, W.lbq_agg, W.lbq_incl};
  q.st = W.st;
  PTC_LAUNCH("k_wm_query", s, k_wm_query<<<ceil_div_u32(n, kQTile), kQThreads, 0, s>>>(q));
  DevStatus h;
  return end_call(W.st, s, &h);
}
